"""The seeded input generators follow the stated recipe (host only).

Every GPU test, the oracle comparisons and the benchmark draw their inputs here, so the
recipe is checked against its statement: bf16 rounding to nearest even (as torch's
conversion), unit-norm q and k, alpha = exp(-0.1 softplus(x)) in (0, 1], beta = sigmoid(x)
in (0, 1), packed lengths log-uniform in [512, 16384] summing to 65536, determinism per
seed, and per-head parameters d, b shared by every seed offset (data-parallel ranks).
"""
import numpy as np
import torch

from paper_2506_02475_gb300 import inputs


def test_bf16_rounding_matches_torch_conversion():
    rng = np.random.default_rng(0)
    x = np.concatenate([rng.standard_normal(10000).astype(np.float32) * 10.0 ** rng.integers(-6, 6, 10000),
                        np.array([0.0, -0.0, 1.0, 1.00390625, 1.005859375, -1.00390625, 3.4e38], np.float32)])
    want = torch.from_numpy(x).to(torch.bfloat16).float().numpy()
    np.testing.assert_array_equal(inputs.round_bf16(x), want)


def test_varlen_lengths_follow_the_recipe():
    rng = np.random.Generator(np.random.PCG64(123))
    lens = inputs.varlen_lengths(rng)
    assert len(lens) == 12 and lens.sum() == 65536
    assert lens.min() >= 512 and lens.max() <= 16384
    assert len(set(lens.tolist())) > 6          # spread out, not one length repeated
    w = inputs.make("custom", T=4096, H=2, dk=64, dv=64, lengths=[100, 0, 3000, 996])
    np.testing.assert_array_equal(w.cu_seqlens, [0, 100, 100, 3100, 4096])


def test_token_and_gate_distributions():
    w = inputs.make("custom", B=2, T=300, H=3, dk=128, dv=64, dtype="bf16", with_b=True, with_h0=True)
    for x in (w.q, w.k):
        np.testing.assert_allclose(np.linalg.norm(x.astype(np.float64), axis=-1), 1.0, atol=1e-2)
        np.testing.assert_array_equal(inputs.round_bf16(x), x)           # already bf16 values
    np.testing.assert_array_equal(inputs.round_bf16(w.v), w.v)
    np.testing.assert_array_equal(inputs.round_bf16(w.dO), w.dO)
    assert np.all((w.alpha > 0) & (w.alpha <= 1)) and np.all(w.alpha > np.exp(-0.1 * 10))
    assert np.all((w.beta > 0) & (w.beta < 1))
    assert np.all((w.d >= 0) & (w.d <= 1)) and np.all((w.b >= 0) & (w.b <= 1))
    assert w.h0.shape == (2, 3, 128, 64) and w.dhT.shape == (2, 3, 128, 64)


def test_seeded_and_parameters_shared_across_seed_offsets():
    a = inputs.make("custom", B=1, T=128, H=4, dk=64, dv=64, with_b=True)
    b = inputs.make("custom", B=1, T=128, H=4, dk=64, dv=64, with_b=True)
    c = inputs.make("custom", B=1, T=128, H=4, dk=64, dv=64, with_b=True, seed_offset=1)
    for name in ("q", "k", "v", "alpha", "beta", "d", "b", "dO"):
        np.testing.assert_array_equal(getattr(a, name), getattr(b, name))
    np.testing.assert_array_equal(a.d, c.d)
    np.testing.assert_array_equal(a.b, c.b)
    assert not np.array_equal(a.q, c.q) and not np.array_equal(a.alpha, c.alpha)


def test_feedback_vectors_stay_close_to_the_keys():
    w = inputs.make("custom", B=1, T=512, H=2, dk=128, dv=64, dtype="bf16")
    p = inputs.feedback_vectors(w.k, "bf16")
    n = np.linalg.norm(p.astype(np.float64), axis=-1)
    assert np.all((n > 0.49) & (n < 1.01))                               # s in (0.5, 1) times a unit vector
    assert np.mean(np.sum(p * w.k, axis=-1) > 0) > 0.95                  # p . k > 0 mostly
