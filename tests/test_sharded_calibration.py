"""Sharded PTF calibration (Eqs. 8-10 over a batch split by rows across ranks).

CPU tests pin the oracle's sharded definition against its unsplit one, check
the library's host combine against it, and run the exchange protocol of
``paper_2111_13824_gb300.dist`` on gloo ranks (CPU processes) with the
per-rank stages computed by the oracle.  GPU tests run the per-rank stages in
the CUDA library, one shard after another on the one GPU, and compare with
the oracle bit for bit.
"""
from __future__ import annotations

import os
import socket

import numpy as np
import pytest
import torch

import oracle
from paper_2111_13824_gb300 import fqvit


def _batch(seed, rows, C, outliers=0):
    rng = np.random.default_rng(seed)
    r = np.exp(rng.normal(0, 1, C)) * 2
    if outliers:
        r[rng.choice(C, outliers, replace=False)] *= 40
    m = 0.25 * r * rng.normal(size=C)
    return (m + r / 6 * rng.normal(size=(rows, C))).astype(np.float32)


def _splits(rows, n, seed):
    cuts = np.sort(np.random.default_rng(seed).choice(np.arange(1, rows), n - 1, replace=False))
    return np.split(np.arange(rows), cuts)


# ---------------------------------------------------------------- oracle pins (CPU)

@pytest.mark.parametrize("K", [0, 3, 7])
def test_one_shard_is_the_unsplit_calibration(K):
    x = _batch(1, 700, 48, outliers=3)
    s, zp, a, sse = oracle.calibrate_ptf(x, K)
    s1, zp1, a1, sse1 = oracle.calibrate_ptf_sharded([x], K)
    assert (s1, zp1) == (s, zp)
    assert np.array_equal(a1, a) and np.array_equal(sse1, sse)


@pytest.mark.parametrize("n", [2, 3, 7])
def test_any_split_keeps_the_range_and_the_sums(n):
    K = 3
    x = _batch(2, 900, 64, outliers=4)
    s, zp, a, sse = oracle.calibrate_ptf(x, K)
    shards = [x[i] for i in _splits(len(x), n, n)]
    s2, zp2, a2, sse2 = oracle.calibrate_ptf_sharded(shards, K)
    # min / max are exact, so s and zp cannot depend on the split
    assert (s2, zp2) == (s, zp)
    # the sums differ from the sequential ones by fp64 rounding only
    assert np.allclose(sse2, sse, rtol=1e-12, atol=0)
    # alpha can only move where two factors tie to within that rounding
    srt = np.sort(sse, axis=1)
    clear = (srt[:, 1] - srt[:, 0]) > 1e-9 * srt[:, 1]
    assert np.array_equal(a2[clear], a[clear])


def test_sharded_sums_are_brute_force_sums():
    # a tiny batch: every term by hand in fp32 / fp64 (Eq. 10 with Eq. 7's clip and zero point)
    x = _batch(3, 9, 3)
    K = 2
    mn, mx = float(x.min()), float(x.max())
    s0 = np.float32(np.float32(mx) - np.float32(mn)) / np.float32(255)
    zp = int(np.clip(np.rint(np.float32(-np.float32(mn)) / s0), 0, 255))
    want = np.zeros((3, K + 1))
    for c in range(3):
        for a in range(K + 1):
            sa = np.float32(s0 * np.float32(2.0 ** (a - K)))
            for r in range(9):
                q = np.clip(np.rint(np.float32(x[r, c] / sa)), -zp, 255 - zp).astype(np.float32)
                d = np.float32(x[r, c] - np.float32(q * sa))
                want[c, a] += float(d) * float(d)
    got = oracle.calibrate_ptf_sharded([x[:4], x[4:]], K)[3]
    assert np.allclose(got, want, rtol=1e-12, atol=0)


# ---------------------------------------------------------------- library host combine (CPU)

@pytest.mark.parametrize("K,n", [(0, 2), (3, 2), (3, 5), (7, 3)])
def test_host_combine_matches_the_oracle(K, n):
    x = _batch(10 + K + n, 800, 96, outliers=2)
    shards = [x[i] for i in _splits(len(x), n, K)]
    ranges = [oracle.calibrate_minmax(p) for p in shards]
    mn, mx = min(r[0] for r in ranges), max(r[1] for r in ranges)
    parts = np.stack([oracle.calibrate_sse(p, K, mn, mx) for p in shards])
    s, zp, a, tot = fqvit.calibrate_combine(torch.from_numpy(parts), mn, mx, K)
    s_o, zp_o, a_o, tot_o = oracle.calibrate_ptf_sharded(shards, K)
    assert np.float32(s) == np.float32(s_o) and zp == zp_o
    assert np.array_equal(a.numpy(), a_o) and np.array_equal(tot.numpy(), tot_o)


def test_host_combine_breaks_ties_toward_the_smallest_factor():
    parts = np.zeros((2, 4, 4))
    parts[0] = [[1, 1, 1, 1], [2, 1, 1, 3], [5, 4, 3, 3], [0, 0, 0, 0]]
    s, zp, a, _ = fqvit.calibrate_combine(torch.from_numpy(parts), -1.0, 1.0, 3)
    assert a.tolist() == [0, 1, 2, 0]


def test_host_combine_rejects_an_empty_range():
    parts = torch.zeros(1, 4, 4, dtype=torch.float64)
    with pytest.raises(fqvit.FqvitError) as e:
        fqvit.calibrate_combine(parts, 1.0, -1.0, 3)
    assert e.value.code == fqvit.ERR_INVALID_ARG


# ---------------------------------------------------------------- gloo ranks (CPU)

class OracleOps:
    """Per-rank stages computed by the oracle on the CPU (stand-in for the GPU)."""

    def minmax(self, x):
        return torch.tensor(oracle.calibrate_minmax(x.numpy()), dtype=torch.float32)

    def sse_partial(self, x, K, mnmx):
        return torch.from_numpy(oracle.calibrate_sse(x.numpy(), K, float(mnmx[0]), float(mnmx[1])))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, shards, K, out):
    import torch.distributed as dist
    from paper_2111_13824_gb300.dist import calibrate_ptf_sharded
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        s, zp, a, tot = calibrate_ptf_sharded(torch.from_numpy(shards[rank]), K, ops=OracleOps())
        out.put((rank, s, zp, a.numpy(), tot.numpy()))
    finally:
        dist.destroy_process_group()


def _run_ranks(shards, K):
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, len(shards), port, shards, K, q)) for r in range(len(shards))]
    for p in procs:
        p.start()
    res = [q.get(timeout=120) for _ in procs]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    return sorted(res, key=lambda t: t[0])


@pytest.mark.parametrize("sizes", [(300, 212), (0, 450, 61)])
def test_gloo_ranks_agree_with_the_oracle(sizes):
    K = 3
    x = _batch(20, sum(sizes), 40, outliers=2)
    shards = np.split(x, np.cumsum(sizes)[:-1])
    res = _run_ranks(shards, K)
    s_o, zp_o, a_o, tot_o = oracle.calibrate_ptf_sharded(shards, K)
    for _, s, zp, a, tot in res:
        assert np.float32(s) == np.float32(s_o) and zp == zp_o
        assert np.array_equal(a, a_o) and np.array_equal(tot, tot_o)


# ---------------------------------------------------------------- CUDA per-rank stages (GPU)

DEV = "cuda:0"


@pytest.mark.gpu
@pytest.mark.parametrize("n,K", [(1, 3), (2, 3), (4, 0), (3, 7)])
def test_device_stages_match_the_oracle(n, K):
    x = _batch(30 + n, 5000, 384, outliers=8)
    shards = [x[i] for i in _splits(len(x), n, n)]
    dshards = [torch.from_numpy(p).to(DEV) for p in shards]
    ranges = [fqvit.calibrate_minmax(p) for p in dshards]
    for p, r in zip(shards, ranges):
        assert tuple(r.cpu().tolist()) == oracle.calibrate_minmax(p)
    mn = min(float(r[0]) for r in ranges)
    mx = max(float(r[1]) for r in ranges)
    mnmx = torch.tensor([mn, mx], dtype=torch.float32, device=DEV)
    parts = torch.stack([fqvit.calibrate_sse_partial(p, K, mnmx).cpu() for p in dshards])
    for p, got in zip(shards, parts):
        assert np.array_equal(got.numpy(), oracle.calibrate_sse(p, K, mn, mx))
    s, zp, a, tot = fqvit.calibrate_combine(parts, mn, mx, K)
    s_o, zp_o, a_o, tot_o = oracle.calibrate_ptf_sharded(shards, K)
    assert np.float32(s) == np.float32(s_o) and zp == zp_o
    assert np.array_equal(a.numpy(), a_o) and np.array_equal(tot.numpy(), tot_o)
    if n == 1:  # one rank is exactly the unsplit device calibration
        sse1 = torch.empty(384, K + 1, dtype=torch.float64, device=DEV)
        s1, zp1, a1 = fqvit.calibrate_ptf(dshards[0], K=K, sse=sse1)
        assert float(s1.item()) == s and int(zp1.item()) == zp
        assert torch.equal(a1.cpu(), a) and torch.equal(sse1.cpu(), tot)
