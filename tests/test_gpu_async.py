"""The device-resident calls (lam_quantize_async, lam_quantize_result,
lam_dequantize_from, lam_score_topk_from): the same codes, widths, ranges,
values and top-k as the synchronous calls and the oracle, with the width
taken from the quantize status on the device; error statuses carried over."""
import hashlib

import numpy as np
import pytest
import torch

import oracle
import paper_2609_32256_gb300 as lam
from paper_2609_32256_gb300 import inputs
from tests.parity import check_topk, oracle_topk

pytestmark = pytest.mark.gpu
NP_DT = {1: np.int8, 2: np.int16, 4: np.int32}


def digest(a):
    return hashlib.sha256(np.ascontiguousarray(a).tobytes()).hexdigest()


def q_async(dev, x_np, eps, width_req, codes_bytes=None):
    x = torch.from_numpy(np.ascontiguousarray(x_np).reshape(-1)).to(dev)
    n = x.numel()
    codes = torch.full((codes_bytes if codes_bytes is not None else 4 * n,), 0x55,
                       dtype=torch.uint8, device=dev)
    ws = torch.zeros(256, dtype=torch.uint8, device=dev)
    lam.lam_quantize_async(x, eps, width_req, codes, ws)
    res = lam.lam_quantize_result(ws, eps, width_req, raise_on_error=False)
    return res, codes, ws


@pytest.mark.parametrize("eps", [1e-2, 1e-3, 1e-4])
def test_quantize_async_matches_the_oracle(dev, eps):
    x = inputs.flat_values((1 << 20) + 5, seed=7)
    (st, w, s, cmin, cmax), codes, _ = q_async(dev, x, eps, 0)
    oc, rmin, rmax, _ = oracle.quantize(x, eps)
    assert st == 0 and w == oracle.width(rmin, rmax) and (cmin, cmax) == (int(rmin), int(rmax))
    assert s == np.float32(2 * np.float32(eps))
    assert digest(codes.cpu().numpy()[: x.size * w]) == digest(oc.astype(NP_DT[w]))


@pytest.mark.parametrize("outlier,width", [(300.0, 2), (40000.0, 4)])
def test_quantize_async_second_pass_on_the_device(dev, outlier, width):
    # an outlier the AUTO sample misses: the settle step re-quantizes at the
    # exact width without the host
    x = inputs.flat_values((1 << 20) + 7, seed=4)
    x[1000 * 256 + 100] = np.float32(outlier * 2 * 1e-2)
    (st, w, _, cmin, cmax), codes, _ = q_async(dev, x, 1e-2, 0)
    oc, rmin, rmax, _ = oracle.quantize(x, 1e-2)
    assert st == 0 and w == width and (cmin, cmax) == (int(rmin), int(rmax))
    assert digest(codes.cpu().numpy()[: x.size * w]) == digest(oc.astype(NP_DT[w]))


def test_quantize_async_forced_widths_and_errors(dev):
    x = inputs.flat_values(100003, seed=8)
    oc, rmin, rmax, _ = oracle.quantize(x, 1e-3)
    (st, w, *_), codes, _ = q_async(dev, x, 1e-3, 2)
    assert st == 0 and w == 2
    assert digest(codes.cpu().numpy()[: x.size * 2]) == digest(oc.astype(np.int16))
    # a forced width too narrow
    (st, *_), _, _ = q_async(dev, x, 1e-4, 1)
    assert st == lam.LAM_ERR_RANGE
    # non-finite input
    y = x.copy()
    y[77] = np.inf
    (st, *_), _, _ = q_async(dev, y, 1e-2, 0)
    assert st == lam.LAM_ERR_NONFINITE
    # empty input
    (st, w, *_), _, _ = q_async(dev, x[:0], 1e-2, 0)
    assert st == 0 and w == 1


@pytest.mark.parametrize("eps,width", [(1e-2, 0), (1e-4, 0), (1e-4, 4)])
def test_dequantize_from(dev, eps, width):
    x = inputs.flat_values((1 << 18) + 3, seed=9)
    (st, w, s, _, _), codes, ws = q_async(dev, x, eps, width)
    assert st == 0
    out = torch.full((x.size,), 7.0, dtype=torch.float32, device=dev)
    lam.lam_dequantize_from(codes, ws, x.size, eps, out)
    oc = oracle.quantize(x, eps)[0]
    want = oracle.dequantize(oc, s)
    assert np.array_equal(out.cpu().numpy().view(np.uint32), want.view(np.uint32))


def test_dequantize_from_leaves_output_on_error(dev):
    x = inputs.flat_values(4099, seed=10)
    x[5] = np.nan
    (st, *_), codes, ws = q_async(dev, x, 1e-2, 0)
    assert st == lam.LAM_ERR_NONFINITE
    out = torch.full((x.size,), 7.0, dtype=torch.float32, device=dev)
    lam.lam_dequantize_from(codes, ws, x.size, 1e-2, out)
    assert torch.all(out == 7.0).item()


def search_from(dev, q, codes, ws, N, D, eps, k, metric):
    qt = torch.from_numpy(q).to(dev)
    B = q.shape[0]
    nb = lam.lam_score_topk_from_workspace_size(B, N, D, k)
    sws = torch.empty(nb, dtype=torch.uint8, device=dev)
    s = torch.empty((B, k), dtype=torch.float32, device=dev)
    i = torch.empty((B, k), dtype=torch.int64, device=dev)
    lam.lam_score_topk_from(qt, codes, ws, N, D, eps, k, metric, s, i, sws)
    return s, i, lam.lam_score_topk_status(sws)


@pytest.mark.parametrize("path,B", [("bandwidth", 1), ("bandwidth", 2), ("tensor", 20),
                                    ("tensor", 520), ("generic", 5)])
@pytest.mark.parametrize("eps", [1e-2, 1e-4])  # int8 and int16 codes
@pytest.mark.parametrize("metric", [oracle.IP, oracle.COSINE, oracle.L2])
def test_score_topk_from_equals_the_synchronous_search(dev, monkeypatch, score_path, path, B,
                                                       eps, metric):
    """The status-driven search runs the same kernels as the synchronous one
    (bit for bit); the synchronous call's opt-in two-pass tensor search
    rescores its candidates on the CUDA cores instead, so it is compared
    through the oracle."""
    score_path(path)
    N, D, k = 3001, 768, 10
    x = inputs.unit_rows(N, D, seed=B)
    q = inputs.queries(B, D, seed=B + 1)
    (st, w, s, cmin, cmax), codes, ws = q_async(dev, x, eps, 0)
    assert st == 0 and w == (1 if eps == 1e-2 else 2)
    assert lam.lam_score_topk_from_path(B, N, D, k) == {"bandwidth": 0, "tensor": 1,
                                                          "generic": 2}[path]
    gs, gi, gst = search_from(dev, q, codes, ws, N, D, eps, k, metric)
    assert gst == 0
    typed = codes[: N * D * w].view(torch.int8 if w == 1 else torch.int16).view(N, D)
    oc = oracle.quantize(x, eps)[0].reshape(N, D)
    os_, oi = oracle_topk(q, oc, eps, metric, k)
    ss, si = lam.search(torch.from_numpy(q).to(dev), typed, eps, k, metric,
                        code_bound=max(-cmin, cmax))
    assert torch.equal(gs, ss) and torch.equal(gi, si)
    monkeypatch.setenv("LAM_SCORE_HI", "1")
    ss, si = lam.search(torch.from_numpy(q).to(dev), typed, eps, k, metric,
                        code_bound=max(-cmin, cmax))
    check_topk(ss.cpu().numpy(), si.cpu().numpy(), q, oc, eps, metric, os_, oi)
    check_topk(gs.cpu().numpy(), gi.cpu().numpy(), q, oc, eps, metric, os_, oi)


def test_score_topk_from_reports_bad_statuses(dev):
    N, D = 2000, 768
    x = inputs.unit_rows(N, D, seed=3)
    q = inputs.queries(4, D, seed=4)
    # width 4 codes (eps small enough) are not taken
    (st, w, *_), codes, ws = q_async(dev, x, 1e-6, 0)
    assert st == 0 and w == 4
    _, _, gst = search_from(dev, q, codes, ws, N, D, 1e-6, 10, oracle.IP)
    assert gst == lam.LAM_ERR_UNSUPPORTED
    # a failed quantization (non-finite input)
    y = x.copy()
    y[3, 3] = np.nan
    (st, *_), codes, ws = q_async(dev, y, 1e-2, 0)
    assert st == lam.LAM_ERR_NONFINITE
    _, _, gst = search_from(dev, q, codes, ws, N, D, 1e-2, 10, oracle.IP)
    assert gst == lam.LAM_ERR_UNSUPPORTED


def test_score_topk_from_int16_beyond_the_tensor_bound(dev, score_path):
    # int16 codes above 2048 in magnitude cannot take the tensor cores exactly
    score_path("tensor")
    N, D = 1000, 768
    x = inputs.unit_rows(N, D, seed=5)
    (st, w, _, cmin, cmax), codes, ws = q_async(dev, x, 2e-5, 0)
    assert st == 0 and w == 2 and max(-cmin, cmax) > 2048
    _, _, gst = search_from(dev, inputs.queries(20, D, seed=6), codes, ws, N, D, 2e-5, 10,
                            oracle.IP)
    assert gst == lam.LAM_ERR_RANGE
