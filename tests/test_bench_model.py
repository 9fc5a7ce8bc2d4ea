"""The bench's algorithmic byte and FLOP model, checked against explicit tensor lists.

`bench.py` reports each kernel's roofline from `stage_model` (bytes and tile-product
FLOPs per launch) and `compulsory_bytes` (the step's own inputs and outputs).  Here
every kernel of the bf16 d = 128 tcgen05 path (and, for bytes, of head dim 256) is
listed tile by tile: the tensors one
(chunk, head) unit must read or write once and the products it must form, written out
from the chunk equations of section 3.2 and the affine chunk maps (H_{n+1} =
(gamma_L I + Atilde) H_n + B).  The model must agree with the lists.
"""
import bench

C, dk, dv = 64, 128, 128
BF, F4 = 2, 4


def tile(r, c, es=BF):
    return r * c * es


def mm(m, n, k):
    return 2 * m * n * k


# per (chunk, head) unit, vg = 1, the forward saving the backward's factors
PREP = {"K": tile(C, dk), "V": tile(C, dv), "alpha": C * F4, "beta": C * F4, "G (log-decays, out)": C * F4,
        "W^T (out)": tile(dk, C), "U^T (out)": tile(dv, C), "U_s^T (out)": tile(dv, C), "M (out)": tile(C, C),
        "Atilde (out)": tile(dk, dk)}
PREP_PRODUCTS = [mm(C, C, dk),        # Gram K K^T
                 mm(C, dk, C),        # W = Mw K
                 mm(C, dv, C),        # U = Mu V
                 mm(dk, dk, C)]       # Atilde = -Kbar^T W
SCAN_FWD = {"Atilde": tile(dk, dk), "gamma_L": F4, "U_s^T": tile(dv, C), "K": tile(C, dk), "H_n (out)": tile(dv, dk)}
SCAN_FWD_PRODUCTS = [mm(dv, dk, dk),  # state through the chunk map
                     mm(dv, dk, C)]   # B^T = U_s^T K
OUTPUT = {"Q": tile(C, dk), "K": tile(C, dk), "W^T": tile(dk, C), "G": C * F4, "H_n": tile(dv, dk), "U^T": tile(dv, C),
          "O (out)": tile(C, dv), "E (out)": tile(C, dv), "Z^T (out)": tile(dk, C)}
OUTPUT_PRODUCTS = [mm(C, C, dk),      # S = Q~ K^T
                   mm(C, dv, dk),     # W H
                   mm(C, dv, dk),     # Qhat H
                   mm(C, dv, C),      # P E
                   mm(C, dk, C)]      # P W (for Z)
SCAN_BWD = {"Atilde": tile(dk, dk), "gamma_L": F4, "Z^T": tile(dk, C), "dO": tile(C, dv), "dH' (out)": tile(dv, dk)}
SCAN_BWD_PRODUCTS = [mm(dv, dk, dk), mm(dv, dk, C)]   # adjoint through the map, C^T = dO^T Z
LOCAL = {"Q": tile(C, dk), "K": tile(C, dk), "M": tile(C, C), "alpha": C * F4, "beta": C * F4, "G": C * F4,
         "V": tile(C, dv), "dO": tile(C, dv), "E": tile(C, dv), "H_n": tile(dv, dk), "dH'": tile(dv, dk),
         "dq (out)": tile(C, dk), "dk (out)": tile(C, dk), "dv (out)": tile(C, dv), "dalpha (out)": C * F4,
         "dbeta (out)": C * F4}
LOCAL_PRODUCTS = [mm(C, C, dk), mm(C, C, dk),                       # S = Q~ K^T, K K^T
                  mm(C, C, dv),                                     # dP = dO E^T
                  mm(C, dk, dv), mm(C, dk, dv), mm(C, dk, dv),      # dO H^T, E dH'^T, K dH'
                  mm(C, dv, C),                                     # P^T dO
                  mm(C, dv, C),                                     # M^T dE
                  mm(C, dk, dv),                                    # (M^T dE) H^T
                  mm(C, dk, C), mm(C, dk, C),                       # dPhat K, dPhat^T Q~
                  mm(C, C, dv),                                     # (M^T dE) E^T = M^T dM M^T
                  mm(C, dk, C), mm(C, dk, C)]                       # dG K, dG^T K


def test_per_unit_bytes_of_every_kernel_match_the_tensor_lists():
    m = bench.stage_model(dk, dv, slots=1, H=1, N=1, save=True, tc=True)
    assert m["prep"]["bytes"] == sum(PREP.values()) == 123_648
    assert m["scan_fwd"]["bytes"] == sum(SCAN_FWD.values()) == 98_308
    assert m["output"]["bytes"] == sum(OUTPUT.values()) == 147_712
    assert m["scan_bwd"]["bytes"] == sum(SCAN_BWD.values()) == 98_308
    assert m["bwd_local"]["bytes"] == sum(LOCAL.values()) == 206_080
    assert m["bwd_prep"]["bytes"] == 0 and m["output_E"]["bytes"] == 0


def test_per_unit_flops_of_every_kernel_match_the_product_lists():
    m = bench.stage_model(dk, dv, slots=1, H=1, N=1, save=True, tc=True)
    assert m["prep"]["flops"] == sum(PREP_PRODUCTS)
    assert m["scan_fwd"]["flops"] == sum(SCAN_FWD_PRODUCTS)
    assert m["output"]["flops"] == sum(OUTPUT_PRODUCTS)
    assert m["scan_bwd"]["flops"] == sum(SCAN_BWD_PRODUCTS)
    assert m["bwd_local"]["flops"] == sum(LOCAL_PRODUCTS)


def test_model_scales_with_units():
    one = bench.stage_model(dk, dv, slots=1, H=1, N=1)
    many = bench.stage_model(dk, dv, slots=64, H=16, N=4)
    for k in ("prep", "scan_fwd", "output", "scan_bwd", "bwd_local"):
        assert many[k]["bytes"] == 64 * 16 * one[k]["bytes"], k
        assert many[k]["flops"] == 64 * 16 * one[k]["flops"], k


def test_value_head_groups_count_key_side_tensors_once():
    """dv = 256 as two value heads of 128 per key head: q, k, gates, W, M, Atilde and the
    key-side gradients once per (chunk, key head), the rest per value head."""
    m = bench.stage_model(dk, dv, slots=1, H=2, N=1, vg=2)
    key = {"prep": PREP["K"] + PREP["alpha"] + PREP["beta"] + PREP["G (log-decays, out)"] + PREP["W^T (out)"]
           + PREP["M (out)"] + PREP["Atilde (out)"],
           "local": sum(LOCAL[n] for n in ("Q", "K", "M", "alpha", "beta", "G", "dq (out)", "dk (out)",
                                           "dalpha (out)", "dbeta (out)"))}
    assert m["prep"]["bytes"] == key["prep"] + 2 * (sum(PREP.values()) - key["prep"])
    assert m["bwd_local"]["bytes"] == key["local"] + 2 * (sum(LOCAL.values()) - key["local"])


def test_pk_adds_the_feedback_vectors_and_their_gradient():
    base = bench.stage_model(dk, dv, slots=1, H=1, N=1)
    pk = bench.stage_model(dk, dv, slots=1, H=1, N=1, pk=True)
    assert pk["prep"]["bytes"] - base["prep"]["bytes"] == tile(C, dk)               # P in
    assert pk["bwd_local"]["bytes"] - base["bwd_local"]["bytes"] == 2 * tile(C, dk)  # P in, dP out


def test_compulsory_bytes_per_token_head():
    """Forward: q, k, v, alpha, beta in, o out.  Backward: q, k, v, alpha, beta, dO in,
    dq, dk, dv, dalpha, dbeta out.  States: h0 in, hT out (forward); h0, dhT in, dh0 out."""
    fwd_tok = 3 * dk * BF + 2 * F4 + dv * BF
    bwd_tok = (2 * dk + dv) * BF + 2 * F4 + dv * BF + (2 * dk + dv) * BF + 2 * F4
    assert (fwd_tok, bwd_tok) == (1032, 1808)
    th, st = 1000, 3 * dk * dv
    fwd, bwd, per = bench.compulsory_bytes(dk, dv, th, st)
    assert fwd == th * fwd_tok + 2 * st * F4
    assert bwd == th * bwd_tok + 3 * st * F4
    assert per["bwd_local"] == th * bwd_tok
    assert per["prep"] == th * ((dk + dv) * BF + 2 * F4)
    assert per["output"] == th * ((2 * dk + dv) * BF + F4)


def test_head_dim_256_per_key_head_bytes_match_the_tensor_lists():
    """dk = 256 with four value heads 64 wide: key-side tiles once per (chunk, key head), the
    value heads' own tiles four times; no chunk map, W and K (or Z) streamed by the scans."""
    K, v = 256, 64
    key = dict(
        prep=tile(C, K) + tile(C, K) + 3 * C * F4 + tile(C, C),                 # K in, W out, alpha/beta/G, M out
        scan_fwd=2 * tile(C, K) + C * F4,                                        # W, K, gamma
        scan_bwd=3 * tile(C, K) + C * F4,                                        # W, K, Z, gamma
        output=3 * tile(C, K) + C * F4 + tile(C, K),                             # Q, K, W, G in; Z out
        bwd_local=2 * tile(C, K) + tile(C, C) + 3 * C * F4 + 2 * tile(C, K) + 2 * C * F4)
    per_value = dict(
        prep=2 * tile(C, v),                                                     # V in, U out
        scan_fwd=tile(C, v) + tile(v, K),                                        # U in, H_n out
        scan_bwd=tile(C, v) + tile(v, K),                                        # dO in, dH' out
        output=tile(C, v) + tile(v, K) + 2 * tile(C, v),                         # U, H_n in; O, E out
        bwd_local=3 * tile(C, v) + 2 * tile(v, K) + tile(C, v))                  # V, dO, E, H_n, dH' in; dv out
    m = bench.stage_model(K, v, slots=1, H=4, N=1, vg=4)
    for stage in key:
        assert m[stage]["bytes"] == key[stage] + 4 * per_value[stage], stage
    assert m["bwd_prep"]["bytes"] == 0
