"""MinMax Linear layers on the GPU (fqvit_linear_q on the tcgen05 tensor cores) against the
oracle, bit for bit: the uint8 output and the int32 accumulators, for ragged M, N and K, every
zero-point regime of the exact chunking, adversarial sums at the chunk bound, every branch of
the dyadic multiplier, the invalid-scale status, back-to-back dependent launches, and the
ViT-L/384 and DeiT-S layer shapes from the synthetic generator.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2111_13824_gb300 import build as fbuild
from paper_2111_13824_gb300 import fqvit, synth

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    fbuild.build()
    fqvit.load()
    oracle.build()


def _gpu(x, zp_x, s_x, w, s_w, bias, s_y, zp_y, with_acc=True):
    xd = torch.from_numpy(x).to(DEV)
    wh = fqvit.linear_pack_weight(torch.from_numpy(w).to(DEV))
    sw = torch.from_numpy(s_w).to(DEV)
    bd = None if bias is None else torch.from_numpy(bias).to(DEV)
    acc = torch.empty(x.shape[0], w.shape[0], dtype=torch.int32, device=DEV) if with_acc else None
    y = fqvit.linear_q(xd, zp_x, s_x, wh, sw, bd, s_y, zp_y, acc=acc)
    fqvit.sync_status()
    return y.cpu().numpy(), None if acc is None else acc.cpu().numpy()


def _random_case(seed, M, K, N, zp_x):
    rng = np.random.default_rng(seed)
    x = rng.integers(0, 256, size=(M, K)).astype(np.uint8)
    w = rng.integers(-128, 128, size=(N, K)).astype(np.int8)
    s_w = (rng.uniform(0.5, 2.0, size=N) * 1e-3).astype(np.float32)
    bias = rng.integers(-(1 << 20), 1 << 20, size=N).astype(np.int32)
    s_x = 0.02
    s_y = float(np.float32(s_x * 1e-3 * np.sqrt(K) * 60.0 / 255.0))
    zp_y = int(rng.integers(0, 256))
    return x, zp_x, s_x, w, s_w, bias, s_y, zp_y


# (M, K, N, zp_x): one row; ragged M, K below one 64-step, N = 256 + 32; three M tiles with K = 3 x 64 + 8;
# many chunks (kc = 2 steps for zp_x = 37) with a half N tile; fc2-like K with N below one tile
@pytest.mark.parametrize("M,K,N,zp_x", [(1, 8, 16, 0), (200, 96, 288, 128), (257, 200, 512, 255),
                                         (384, 1040, 1152, 37), (130, 4096, 96, 200), (129, 64, 4096, 128)])
def test_linear_matches_oracle(M, K, N, zp_x):
    case = _random_case(M * 7 + K + N, M, K, N, zp_x)
    want_y, want_acc = oracle.linear_q(*case)
    y, acc = _gpu(*case)
    assert np.array_equal(acc, want_acc)
    assert np.array_equal(y, want_y)
    # without the accumulator output and without a bias (the other kernel variant)
    c2 = list(case)
    c2[5] = None
    want_y2, _ = oracle.linear_q(*c2)
    y2, _ = _gpu(*c2, with_acc=False)
    assert np.array_equal(y2, want_y2)


@pytest.mark.parametrize("zp_x", [0, 128, 255])
def test_exact_at_the_chunk_bound(zp_x):
    """Partial sums as large as the chunking allows (every large product of one sign) with unit
    products interleaved: a lost low bit anywhere in the tensor cores' fp32 sums shows."""
    M, K, N = 128, 4096, 64
    big = 255 if zp_x == 0 else 0          # x - zp_x = +-255 or -128
    x = np.full((M, K), big, np.uint8)
    x[:, 1::2] = zp_x + (1 if zp_x < 255 else -1)  # x - zp_x = +-1 at odd k
    w = np.zeros((N, K), np.int8)
    w[:, 0::2] = np.where(np.arange(N)[:, None] % 2 == 0, 127, -128)
    w[:, 1::2] = 1
    rng = np.random.default_rng(zp_x)
    flip = rng.random((M, K)) < 0.01       # a few products of the other sign and size
    x[flip] = rng.integers(0, 256, size=int(flip.sum()))
    s_w = np.full(N, 1e-3, np.float32)
    case = (x, zp_x, 0.01, w, s_w, None, 0.5, 128)
    want_y, want_acc = oracle.linear_q(*case)
    y, acc = _gpu(*case)
    assert np.array_equal(acc, want_acc)
    assert np.array_equal(y, want_y)


def test_multiplier_branches():
    """Per channel M_n = 1, 2^-3, 2^-30 (the N1 cap), 300 and 4096 (N1 <= 0), and typical values."""
    rng = np.random.default_rng(5)
    M, K, N = 64, 64, 32
    x = rng.integers(120, 137, size=(M, K)).astype(np.uint8)
    w = rng.integers(-3, 4, size=(N, K)).astype(np.int8)
    s_x, s_y = 0.5, 2.0
    Ms = [1.0, 2.0 ** -3, 2.0 ** -30, 300.0, 4096.0] + list(rng.uniform(1e-4, 0.5, size=N - 5))
    s_w = np.array([m * s_y / s_x for m in Ms], np.float32)
    case = (x, 128, s_x, w, s_w, rng.integers(-50, 50, size=N).astype(np.int32), s_y, 100)
    want_y, want_acc = oracle.linear_q(*case)
    y, acc = _gpu(*case)
    assert np.array_equal(acc, want_acc)
    assert np.array_equal(y, want_y)


def test_invalid_weight_scale_is_reported():
    case = list(_random_case(9, 64, 128, 64, 100))
    s_w = case[4].copy()
    s_w[3] = 0.0
    s_w[40] = np.nan
    case[4] = s_w
    with pytest.raises(fqvit.FqvitError) as e:
        _gpu(*case)
    assert e.value.code == fqvit.ERR_INVALID_ARG
    fqvit.sync_status()  # the status word was cleared
    # the other channels are computed; the invalid ones hold zp_y
    xd = torch.from_numpy(case[0]).to(DEV)
    wh = fqvit.linear_pack_weight(torch.from_numpy(case[3]).to(DEV))
    y = fqvit.linear_q(xd, case[1], case[2], wh, torch.from_numpy(s_w).to(DEV), torch.from_numpy(case[5]).to(DEV),
                       case[6], case[7])
    with pytest.raises(fqvit.FqvitError):
        fqvit.sync_status()
    ok_sw = s_w.copy()
    ok_sw[3] = ok_sw[40] = 1e-3
    want_y, _ = oracle.linear_q(case[0], case[1], case[2], case[3], ok_sw, case[5], case[6], case[7])
    got = y.cpu().numpy()
    keep = np.ones(64, bool)
    keep[[3, 40]] = False
    assert np.array_equal(got[:, keep], want_y[:, keep])
    assert np.all(got[:, 3] == case[7]) and np.all(got[:, 40] == case[7])


def test_pack_weight_is_the_fp16_of_the_codes():
    w = torch.randint(-128, 128, (300, 136), dtype=torch.int16).to(torch.int8)
    wh = fqvit.linear_pack_weight(w.to(DEV))
    assert torch.equal(wh.cpu(), w.to(torch.float16))


def test_chained_layers_back_to_back():
    """fc1 then fc2 of a small MLP, launched back to back (four dependent launches), against
    the oracle chain."""
    rng = np.random.default_rng(11)
    M, C = 300, 192
    x = rng.integers(0, 256, size=(M, C)).astype(np.uint8)
    w1 = rng.integers(-128, 128, size=(4 * C, C)).astype(np.int8)
    w2 = rng.integers(-128, 128, size=(C, 4 * C)).astype(np.int8)
    s1 = (rng.uniform(0.5, 2, size=4 * C) * 1e-3).astype(np.float32)
    s2 = (rng.uniform(0.5, 2, size=C) * 1e-3).astype(np.float32)
    s_h = float(np.float32(0.02 * 1e-3 * np.sqrt(C) * 60 / 255))
    s_o = float(np.float32(s_h * 1e-3 * np.sqrt(4 * C) * 60 / 255))
    h_want, _ = oracle.linear_q(x, 128, 0.02, w1, s1, None, s_h, 90)
    y_want, _ = oracle.linear_q(h_want, 90, s_h, w2, s2, None, s_o, 130)
    w1h = fqvit.linear_pack_weight(torch.from_numpy(w1).to(DEV))
    w2h = fqvit.linear_pack_weight(torch.from_numpy(w2).to(DEV))
    s1d, s2d = torch.from_numpy(s1).to(DEV), torch.from_numpy(s2).to(DEV)
    xd = torch.from_numpy(x).to(DEV)
    torch.cuda.synchronize()
    h = fqvit.linear_q(xd, 128, 0.02, w1h, s1d, None, s_h, 90)
    y = fqvit.linear_q(h, 90, s_h, w2h, s2d, None, s_o, 130)
    fqvit.sync_status()
    assert np.array_equal(h.cpu().numpy(), h_want)
    assert np.array_equal(y.cpu().numpy(), y_want)


@pytest.mark.parametrize("kind", ["fc1", "fc2"])
def test_vit_l384_layer_sampled(kind):
    """A ViT-L/384 MLP layer at full size (18464 tokens) in one call; rows sampled across the
    M tiles (first, tile edges, the ragged last tile) against the oracle."""
    a = synth.linear_inputs(synth.CONFIGS["vit_l384"], 0, kind)
    wh = fqvit.linear_pack_weight(a["w"].to(DEV))
    y = fqvit.linear_q(a["x"].to(DEV), a["zp_x"], a["s_x"], wh, a["s_w"].to(DEV), a["bias"].to(DEV), a["s_y"],
                       a["zp_y"])
    fqvit.sync_status()
    rows = [0, 1, 127, 128, 4096, 9231, 18431, 18432, 18463]
    got = y.cpu().numpy()[rows]
    want, _ = oracle.linear_q(a["x"].numpy()[rows], a["zp_x"], a["s_x"], a["w"].numpy(), a["s_w"].numpy(),
                              a["bias"].numpy(), a["s_y"], a["zp_y"])
    assert np.array_equal(got, want)


def test_deit_s_projection_full():
    a = synth.linear_inputs(synth.CONFIGS["deit_s"], 3, "proj")
    wh = fqvit.linear_pack_weight(a["w"].to(DEV))
    y = fqvit.linear_q(a["x"].to(DEV), a["zp_x"], a["s_x"], wh, a["s_w"].to(DEV), a["bias"].to(DEV), a["s_y"],
                       a["zp_y"])
    fqvit.sync_status()
    want, _ = oracle.linear_q(a["x"].numpy(), a["zp_x"], a["s_x"], a["w"].numpy(), a["s_w"].numpy(),
                              a["bias"].numpy(), a["s_y"], a["zp_y"])
    assert np.array_equal(y.cpu().numpy(), want)
