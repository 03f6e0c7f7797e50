"""Q_eps and dequantisation on the GPU against the CPU oracle: codes and
dequantised values bit-exact (SHA-256 of the code bytes, as the paper checks
determinism by digest), widths, ranges and error statuses."""
import hashlib

import numpy as np
import pytest
import torch

import oracle
import paper_2609_32256_gb300 as lam
from paper_2609_32256_gb300 import inputs
from tests.conftest import golden

pytestmark = pytest.mark.gpu
EPS_SWEEP = (1e-2, 1e-3, 1e-4)
NP_DT = {1: np.int8, 2: np.int16, 4: np.int32}


def digest(a: np.ndarray) -> str:
    return hashlib.sha256(np.ascontiguousarray(a).tobytes()).hexdigest()


def gpu_quantize(x_np, eps, width, dev, offset=0):
    """Quantize through the C ABI; offset > 0 makes both buffers misaligned."""
    n = x_np.size
    xt = torch.zeros(n + offset, dtype=torch.float32, device=dev)
    xt[offset:] = torch.from_numpy(x_np.reshape(-1)).to(dev)
    x = xt[offset:]
    ws = torch.zeros(lam.lam_quantize_workspace_size(), dtype=torch.uint8, device=dev)
    wbytes = 4 if width == 0 else width
    cbuf = torch.zeros(n * wbytes + 4 * offset, dtype=torch.uint8, device=dev)
    codes = cbuf[4 * offset:]  # aligned to any width, not to 16 bytes
    st, w, s, cmin, cmax = lam.lam_quantize(x, eps, width, codes, ws, raise_on_error=False)
    raw = codes.cpu().numpy()[: n * max(w, 1)]
    c = raw.view(NP_DT[w]) if st == 0 else None
    return st, w, s, cmin, cmax, c


@pytest.mark.parametrize("eps", EPS_SWEEP)
@pytest.mark.parametrize("width", [0, 1, 2, 4])
@pytest.mark.parametrize("n", [1, 15, 16, 17, (1 << 16) + 13])
def test_codes_bit_exact(dev, eps, width, n):
    x = inputs.flat_values(n, seed=n)
    oc, rmin, rmax, _ = oracle.quantize(x, eps)
    need = oracle.width(rmin, rmax)
    st, w, s, cmin, cmax, c = gpu_quantize(x, eps, width, dev)
    assert s == oracle.step(eps)
    assert (cmin, cmax) == (int(rmin), int(rmax))
    if width and need > width:
        assert st == lam.LAM_ERR_RANGE
        return
    assert st == 0 and w == (need if width == 0 else width)
    assert digest(c) == digest(oc.astype(NP_DT[w]))


def midpoint_values(eps, kmax=4096, ulps=4, n_random=200000, seed=7):
    """fp32 values within `ulps` ulps of every quotient midpoint (k + 1/2) s,
    |k| < kmax, where the rounded quotient decides the code, plus random bit
    patterns of every magnitude whose quotient stays below 2^30."""
    s = np.float64(oracle.step(eps))
    k = np.arange(-kmax, kmax, dtype=np.float64)
    mid = ((k + 0.5) * s).astype(np.float32)
    xs, up, dn = [mid], mid.copy(), mid.copy()
    for _ in range(ulps):
        up = np.nextafter(up, np.float32(np.inf))
        dn = np.nextafter(dn, np.float32(-np.inf))
        xs += [up, dn]
    bits = np.random.default_rng(seed).integers(0, 2**32, size=n_random, dtype=np.uint64)
    r = bits.astype(np.uint32).view(np.float32)
    r = r[np.isfinite(r)]
    r = r[np.abs(r.astype(np.float64)) < 2.0**30 * s]
    return np.concatenate(xs + [r]).astype(np.float32)


# steps s = 2 eps inside [2^-40, 2^40] take the reciprocal-and-FMA quotient;
# 1e-13 and 1e12 fall outside and take the division for every value
@pytest.mark.parametrize("eps", [1e-2, 1e-3, 1e-4, 0.0123457, 3e-7, 5e-13, 1e11, 1e-13, 1e12])
def test_codes_at_rounding_midpoints(dev, eps):
    """Codes bit-exact with the oracle's IEEE quotient where rounding decides
    them: next to every midpoint between two codes, and at random magnitudes
    down to subnormal values."""
    x = midpoint_values(eps)
    oc, rmin, rmax, _ = oracle.quantize(x, eps)
    st, w, s, cmin, cmax, c = gpu_quantize(x, eps, 4, dev)
    assert st == 0 and w == 4 and s == oracle.step(eps)
    assert (cmin, cmax) == (int(rmin), int(rmax))
    np.testing.assert_array_equal(c, oc.astype(np.int32))


@pytest.mark.parametrize("offset", [1, 2, 3])
@pytest.mark.parametrize("width", [0, 1, 2, 4])
def test_misaligned_buffers(dev, offset, width):
    x = inputs.flat_values(4099, seed=5)
    oc, rmin, rmax, _ = oracle.quantize(x, 1e-4)
    st, w, *_, c = gpu_quantize(x, 1e-4, width, dev, offset=offset)
    if width == 1:
        assert st == lam.LAM_ERR_RANGE
        return
    assert st == 0
    np.testing.assert_array_equal(c.astype(np.int32), oc)


def test_worked_ties(dev):
    rows = golden("q_eps_ties.txt")
    s = np.float32(2.0 ** -9)
    x = np.array([float(r[0]) for r in rows], dtype=np.float32) * s
    want = np.array([int(r[1]) for r in rows])
    st, w, _, cmin, cmax, c = gpu_quantize(x, 2.0 ** -10, 0, dev)
    assert st == 0 and w == 4 and (cmin, cmax) == (want.min(), want.max())
    np.testing.assert_array_equal(c.astype(np.int64), want)


def test_nonfinite_rejected(dev):
    x = inputs.flat_values(1000, seed=1)
    for bad in (np.nan, np.inf, -np.inf):
        y = x.copy()
        y[517] = bad
        for width in (0, 2):
            st, *_ = gpu_quantize(y, 1e-3, width, dev)
            assert st == lam.LAM_ERR_NONFINITE


def test_forced_width_overflow_reports_range(dev):
    s = np.float32(2.0 ** -9)
    x = np.array([0.0, 127.5, -3.0], dtype=np.float32) * s
    st, w, _, cmin, cmax, _ = gpu_quantize(x, 2.0 ** -10, 1, dev)
    assert st == lam.LAM_ERR_RANGE and (cmin, cmax) == (-3, 128)
    # beyond int32 for every width
    y = np.array([1.0, -1.0], dtype=np.float32)
    st, *_ = gpu_quantize(y, 1e-12, 0, dev)
    assert st == lam.LAM_ERR_RANGE


def test_auto_codes_buffer_too_small(dev):
    x = inputs.flat_values(1000, seed=2)
    xt = torch.from_numpy(x).to(dev)
    ws = torch.zeros(lam.lam_quantize_workspace_size(), dtype=torch.uint8, device=dev)
    codes = torch.zeros(1500, dtype=torch.uint8, device=dev)  # int16 needs 2000
    st, w, *_ = lam.lam_quantize(xt, 1e-4, 0, codes, ws, raise_on_error=False)
    assert st == lam.LAM_ERR_WORKSPACE and w == 2


def test_range_only_without_codes(dev):
    x = inputs.flat_values(100000, seed=3)
    _, rmin, rmax, _ = oracle.quantize(x, 1e-4)
    xt = torch.from_numpy(x).to(dev)
    ws = torch.zeros(lam.lam_quantize_workspace_size(), dtype=torch.uint8, device=dev)
    for width in (0, 2, 4):
        st, w, _, cmin, cmax = lam.lam_quantize(xt, 1e-4, width, None, ws)
        assert st == 0 and (cmin, cmax) == (int(rmin), int(rmax))
        assert w == (oracle.width(rmin, rmax) if width == 0 else width)


@pytest.mark.parametrize("width", [1, 2, 4])
@pytest.mark.parametrize("offset", [0, 1])
def test_dequantize_bit_exact(dev, width, offset):
    rng = np.random.default_rng(width)
    lo, hi = {1: (-128, 128), 2: (-32768, 32768), 4: (-(1 << 30), 1 << 30)}[width]
    n = 70001
    c = rng.integers(lo, hi, size=n).astype(NP_DT[width])
    scale = np.float32(2e-3)
    buf = torch.zeros((n + offset) * width, dtype=torch.uint8, device=dev)
    buf[offset * width:] = torch.from_numpy(c.view(np.uint8)).to(dev)
    out = torch.zeros(n + offset, dtype=torch.float32, device=dev)
    lam.lam_dequantize(buf[offset * width:], width, n, float(scale), out[offset:])
    got = out[offset:].cpu().numpy()
    want = oracle.dequantize(c.astype(np.int32), scale)
    assert digest(got) == digest(want)


def test_flat_2p26_sweep_widths_and_round_trip(dev):
    """Flat microbench workload: 2^26 values ~ N(0, 1/768) clipped to [-1, 1]."""
    n = 1 << 26
    x = inputs.flat_values(n, seed=0)
    xt = torch.from_numpy(x).to(dev)
    expect_width = {1e-2: 1, 1e-3: 1, 1e-4: 2}
    for eps in EPS_SWEEP:
        codes, w, scale, cmin, cmax = lam.quantize(xt, eps)
        oc, rmin, rmax, _ = oracle.quantize(x, eps)
        assert w == expect_width[eps] == oracle.width(rmin, rmax)
        assert (cmin, cmax) == (int(rmin), int(rmax))
        got = codes.cpu().numpy()
        assert digest(got) == digest(oc.astype(NP_DT[w]))
        xh = lam.dequantize(codes, scale).cpu().numpy()
        assert digest(xh) == digest(oracle.dequantize(oc, scale))
        err = np.abs(x.astype(np.float64) - xh.astype(np.float64))
        e32 = np.float64(np.float32(eps))
        assert np.all(err <= e32 * (1 + 2.0 ** -23) + np.abs(x) * 2.0 ** -23)
        del codes


def test_planted_chunks_widths(dev):
    """27,986 chunk embeddings with 5% planted near-duplicates, eps sweep."""
    x = inputs.planted_rows(27986, 768, seed=0)
    xt = torch.from_numpy(x).to(dev)
    for eps, want_w in ((1e-2, 1), (1e-3, 1), (1e-4, 2)):
        codes, w, *_ = lam.quantize(xt, eps)
        oc, rmin, rmax, _ = oracle.quantize(x, eps)
        assert w == want_w == oracle.width(rmin, rmax)
        assert digest(codes.cpu().numpy()) == digest(oc.astype(NP_DT[w]))


@pytest.mark.parametrize("outlier,width", [(300.0, 2), (40000.0, 4)])
def test_auto_width_outlier_missed_by_sample(dev, outlier, width):
    # AUTO speculates the width from a fixed sample (four values at each of
    # 64 evenly spaced positions: here x[16384 j .. 16384 j + 3]); one outlier
    # outside the sample forces the exact-width second pass.
    x = inputs.flat_values((1 << 20) + 7, seed=4)
    x[1000 * 256 + 100] = np.float32(outlier * 2 * 1e-2)  # index not sampled
    oc, rmin, rmax, _ = oracle.quantize(x, 1e-2)
    assert oracle.width(rmin, rmax) == width
    st, w, _, cmin, cmax, c = gpu_quantize(x, 1e-2, 0, dev)
    assert st == 0 and w == width and (cmin, cmax) == (int(rmin), int(rmax))
    assert digest(c) == digest(oc.astype(NP_DT[w]))
