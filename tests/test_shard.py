"""Data-parallel sharding: host logic and a world_size-2 gloo run on the CPU.

The gloo run shards a packed varlen batch over two ranks, runs the oracle on
each rank's sequences, sums the per-head parameter gradients (db, dd) across
ranks, and checks that the gathered results equal one unsharded run.
"""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from paper_2506_02475_gb300 import inputs, shard


def test_shard_bounds_cover_disjoint_balanced():
    for n in (0, 1, 5, 64, 1000):
        for world in (1, 2, 3, 8):
            spans = [shard.shard_bounds(n, world, r) for r in range(world)]
            assert spans[0][0] == 0 and spans[-1][1] == n
            assert all(spans[r][1] == spans[r + 1][0] for r in range(world - 1))
            sizes = [hi - lo for lo, hi in spans]
            assert max(sizes) - min(sizes) <= 1
    with pytest.raises(ValueError):
        shard.shard_bounds(4, 2, 2)


def test_shard_packed_assigns_every_sequence_once():
    rng = np.random.default_rng(0)
    for trial in range(200):
        n = int(rng.integers(0, 12))
        lens = rng.integers(0, 300, n)
        cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
        world = int(rng.integers(1, 6))
        owned = []
        for r in range(world):
            s_lo, s_hi, t_lo, t_hi, lcu = shard.shard_packed(cu, world, r)
            assert t_lo == cu[s_lo] and t_hi == cu[s_hi]
            assert lcu[0] == 0 and lcu[-1] == t_hi - t_lo and len(lcu) == s_hi - s_lo + 1
            np.testing.assert_array_equal(np.diff(lcu), lens[s_lo:s_hi])
            owned += list(range(s_lo, s_hi))
            # the shard's tokens exceed an even share by less than one sequence
            if s_hi > s_lo and world > 1:
                assert (t_hi - t_lo) - cu[-1] / world < lens[s_lo:s_hi].max() + 1
        assert owned == list(range(n))


def test_rank_batches_share_parameters_not_data():
    a = inputs.make("custom", B=1, T=64, H=3, dk=8, dv=8, with_b=True, seed_offset=shard.rank_seed_offset(0))
    c = inputs.make("custom", B=1, T=64, H=3, dk=8, dv=8, with_b=True, seed_offset=shard.rank_seed_offset(1))
    np.testing.assert_array_equal(a.d, c.d)
    np.testing.assert_array_equal(a.b, c.b)
    assert not np.array_equal(a.q, c.q)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out_dir):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import oracle
        lens = [37, 64, 0, 130, 5, 90, 71]
        w = inputs.make("custom", T=sum(lens), H=2, dk=8, dv=6, dtype="f32", with_b=True, with_h0=True,
                        with_grads=True, lengths=lens, seed_offset=7)
        s_lo, s_hi, t_lo, t_hi, lcu = shard.shard_packed(w.cu_seqlens, world, rank)
        tk = slice(t_lo, t_hi)
        args = (w.q[tk], w.k[tk], w.v[tk], w.alpha[tk], w.beta[tk], w.b, w.d)
        o, hT = oracle.fwd(*args, h0=w.h0[s_lo:s_hi], cu_seqlens=lcu, threads=1)
        g = oracle.bwd(*args, w.dO[tk], h0=w.h0[s_lo:s_hi], dhT=w.dhT[s_lo:s_hi], cu_seqlens=lcu, threads=1)
        tg = {k: torch.from_numpy(g[k]) for k in ("db", "dd")}
        shard.reduce_param_grads(tg, dist)
        g["db"], g["dd"] = tg["db"].numpy(), tg["dd"].numpy()
        ms = shard.max_over_ranks(1.5 + rank, dist)
        parts = [None] * world
        dist.all_gather_object(parts, dict(o=o, hT=hT, g=g, ms=ms))
        if rank == 0:
            full_o, full_hT = oracle.fwd(w.q, w.k, w.v, w.alpha, w.beta, w.b, w.d, h0=w.h0, cu_seqlens=w.cu_seqlens,
                                         threads=1)
            full_g = oracle.bwd(w.q, w.k, w.v, w.alpha, w.beta, w.b, w.d, w.dO, h0=w.h0, dhT=w.dhT,
                                cu_seqlens=w.cu_seqlens, threads=1)
            assert all(p["ms"] == 1.5 + world - 1 for p in parts)
            np.testing.assert_allclose(np.concatenate([p["o"] for p in parts]), full_o, rtol=0, atol=1e-13)
            np.testing.assert_allclose(np.concatenate([p["hT"] for p in parts]), full_hT, rtol=0, atol=1e-13)
            for key in ("dq", "dk", "dv", "dalpha", "dbeta", "dh0"):
                np.testing.assert_allclose(np.concatenate([p["g"][key] for p in parts]), full_g[key],
                                           rtol=0, atol=1e-12, err_msg=key)
            for key in ("db", "dd"):
                for p in parts:
                    np.testing.assert_allclose(p["g"][key], full_g[key], rtol=1e-12, atol=1e-12, err_msg=key)
            with open(os.path.join(out_dir, "ok"), "w") as f:
                f.write("ok")
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_two_rank_gloo_sharded_equals_unsharded(tmp_path):
    import oracle
    oracle.build()
    mp.spawn(_rank_main, args=(2, _free_port(), str(tmp_path)), nprocs=2, join=True)
    assert (tmp_path / "ok").exists()
