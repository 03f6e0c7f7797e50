"""Q_eps fused with the band digests (the BandHash of Algorithm 1) against the
oracle: codes and digests bit-exact, every band width the paper sweeps,
forced and narrowest widths, digests-only calls, unaligned rows, the AUTO
second pass, and the candidate structure planted duplicates must produce."""
import hashlib

import numpy as np
import pytest
import torch

import oracle
import paper_2609_32256_gb300 as lam
from paper_2609_32256_gb300 import inputs

pytestmark = pytest.mark.gpu
NP_DT = {1: np.int8, 2: np.int16, 4: np.int32}


def run(dev, x_np, eps, width, r, with_codes=True, offset=0):
    N, D = x_np.shape
    buf = torch.empty(N * D + offset, dtype=torch.float32, device=dev)
    buf[offset:] = torch.from_numpy(x_np.reshape(-1)).to(dev)
    x = buf[offset:].view(N, D)
    codes = torch.zeros(N * D * 4, dtype=torch.uint8, device=dev) if with_codes else None
    dig = torch.zeros((N, D // r), dtype=torch.int64, device=dev)
    ws = torch.zeros(lam.lam_quantize_workspace_size(), dtype=torch.uint8, device=dev)
    st, w, s, cmin, cmax = lam.lam_quantize_bands(x, eps, width, r, codes, dig, ws)
    c = codes[:N * D * w].cpu().numpy().view(NP_DT[w]).reshape(N, D) if with_codes else None
    return w, cmin, cmax, c, dig.cpu().numpy().view(np.uint64)


@pytest.mark.parametrize("r", [1, 2, 4, 8, 16, 32])
@pytest.mark.parametrize("eps,width", [(1e-2, 0), (1e-3, 2), (1e-4, 0), (1e-6, 4)])
def test_codes_and_digests_bit_exact(dev, r, eps, width):
    x = inputs.unit_rows(1000, 768, seed=r)
    oc, rmin, rmax, _ = oracle.quantize(x, eps)
    oc = oc.reshape(x.shape)
    w_exp = oracle.width(rmin, rmax) if width == 0 else width
    w, cmin, cmax, c, d = run(dev, x, eps, width, r)
    assert w == w_exp and (cmin, cmax) == (int(rmin), int(rmax))
    np.testing.assert_array_equal(c, oc.astype(NP_DT[w]))
    np.testing.assert_array_equal(d, oracle.band_digests(oc, r, w))


@pytest.mark.parametrize("eps", [1e-3, 0.0123457, 1e-13])
def test_codes_at_rounding_midpoints(dev, eps):
    """The fused band kernel's codes next to every quotient midpoint equal the
    oracle's (int32 codes, so every value is in range)."""
    from tests.test_gpu_quantize import midpoint_values
    x = midpoint_values(eps, n_random=100000)
    n = x.size // 768 * 768
    x = x[:n].reshape(-1, 768)
    oc, rmin, rmax, _ = oracle.quantize(x, eps)
    oc = oc.reshape(x.shape)
    w, cmin, cmax, c, d = run(dev, x, eps, 4, 8)
    assert w == 4 and (cmin, cmax) == (int(rmin), int(rmax))
    np.testing.assert_array_equal(c, oc.astype(np.int32))
    np.testing.assert_array_equal(d, oracle.band_digests(oc, 8, 4))


@pytest.mark.parametrize("r", [4, 32])
def test_digests_only_and_unaligned_rows(dev, r):
    x = inputs.unit_rows(333, 64, seed=9)
    oc, rmin, rmax, _ = oracle.quantize(x, 1e-3)
    w_exp = oracle.width(rmin, rmax)
    for offset in (0, 1, 2):  # 16-, 4- and 8-byte aligned starts
        w, _, _, _, d = run(dev, x, 1e-3, 0, r, with_codes=False, offset=offset)
        assert w == w_exp
        np.testing.assert_array_equal(d, oracle.band_digests(oc.reshape(x.shape), r, w))


def test_auto_second_pass_when_the_sample_misses_an_outlier(dev):
    x = inputs.unit_rows(4096, 256, seed=3)
    x[1000, 17] = np.float32(300 * 2 * 1e-3)  # code 300: int16, away from every sampled value
    oc, rmin, rmax, _ = oracle.quantize(x, 1e-3)
    assert oracle.width(rmin, rmax) == 2
    w, cmin, cmax, c, d = run(dev, x, 1e-3, 0, 8)
    assert w == 2 and cmax == 300
    np.testing.assert_array_equal(c, oc.reshape(x.shape).astype(np.int16))
    np.testing.assert_array_equal(d, oracle.band_digests(oc.reshape(x.shape), 8, 2))


def test_planted_duplicates_share_their_band_digests(dev):
    # rows that quantize to the same codes share every digest, so each one is
    # a candidate of the other under every band width
    x = inputs.planted_rows(2000, 768, seed=4)
    x[1500] = x[20]
    x[1999] = x[20]
    for r in (4, 8, 32):
        _, _, _, _, d = run(dev, x, 1e-2, 0, r)
        np.testing.assert_array_equal(d[1500], d[20])
        np.testing.assert_array_equal(d[1999], d[20])
        assert len(set(d[:, 0].tolist())) > 1


def test_range_and_nonfinite_errors(dev):
    x = inputs.unit_rows(64, 32, seed=1)
    x[3, 3] = np.float32(10.0)  # code 5000 at eps 1e-3: beyond int8
    N, D = x.shape
    xt = torch.from_numpy(x).to(dev)
    dig = torch.zeros((N, D // 4), dtype=torch.int64, device=dev)
    codes = torch.zeros(N * D, dtype=torch.int8, device=dev)
    ws = torch.zeros(lam.lam_quantize_workspace_size(), dtype=torch.uint8, device=dev)
    st, *_ = lam.lam_quantize_bands(xt, 1e-3, 1, 4, codes, dig, ws, raise_on_error=False)
    assert st == lam.LAM_ERR_RANGE
    x[5, 5] = np.float32(np.nan)
    xt = torch.from_numpy(x).to(dev)
    st, *_ = lam.lam_quantize_bands(xt, 1e-3, 0, 4, codes, dig, ws, raise_on_error=False)
    assert st == lam.LAM_ERR_NONFINITE
