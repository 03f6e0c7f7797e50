"""Bounded device waits (the failure path of every mbarrier wait).

A test hook of the library (environment: LAM_TEST_WAIT_CYCLES, LAM_TEST_STALL)
gives a search's device waits a budget of a few thousand SM cycles and makes
its copy producers issue nothing, so no copy and no MMA is ever in flight and
every consumer's wait runs out.  The search must then record LAM_ERR_TIMEOUT
in its workspace status (read by lam_score_topk_status), unwind every role,
free its tensor memory, and leave the device usable: the next ordinary
search on the same device matches the oracle."""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_32256_gb300 as lam
from paper_2609_32256_gb300 import inputs
from tests.parity import check_topk, check_topk_fn, oracle_topk

pytestmark = pytest.mark.gpu
NP_DT = {1: np.int8, 2: np.int16}


def stall(monkeypatch, on):
    if on:
        monkeypatch.setenv("LAM_TEST_WAIT_CYCLES", "20000")
        monkeypatch.setenv("LAM_TEST_STALL", "1")
    else:
        monkeypatch.delenv("LAM_TEST_WAIT_CYCLES", raising=False)
        monkeypatch.delenv("LAM_TEST_STALL", raising=False)


@pytest.mark.parametrize("path,B,width,eps,k,metric,bound_known", [
    ("bandwidth", 1, 1, 1e-2, 10, oracle.L2, True),
    ("bandwidth", 2, 2, 1e-3, 100, oracle.IP, True),
    ("tensor", 64, 1, 1e-2, 10, oracle.IP, True),        # stage-loop kernel, one block
    ("tensor", 300, 2, 1e-3, 40, oracle.COSINE, True),   # stage-loop kernel, heaps
    ("tensor", 520, 1, 1e-2, 10, oracle.L2, True),       # conversion pass + scoring kernel
    ("tensor", 520, 2, 1e-3, 10, oracle.IP, False)])     # int16 split (256 h + l)
def test_wait_budget_runs_out_then_device_recovers(dev, monkeypatch, score_path, path, B,
                                                   width, eps, k, metric, bound_known):
    score_path(path)
    n, d = 3000, 768
    x = inputs.unit_rows(n, d, seed=B + k)
    oc, rmin, rmax, _ = oracle.quantize(x, eps)
    oc = oc.reshape(n, d)
    bound = max(-int(rmin), int(rmax)) if bound_known else 0
    codes = torch.from_numpy(oc.astype(NP_DT[width])).to(dev)
    q = inputs.queries(B, d, seed=B)
    qt = torch.from_numpy(q).to(dev)
    assert lam.lam_score_topk_path(B, n, d, k, width, bound) == (
        lam.PATH_BANDWIDTH if path == "bandwidth" else lam.PATH_TENSOR)
    ws = torch.empty(lam.lam_score_topk_workspace_size(B, n, d, k, width, bound),
                     dtype=torch.uint8, device=dev)
    s = torch.empty((B, k), dtype=torch.float32, device=dev)
    i = torch.empty((B, k), dtype=torch.int64, device=dev)
    stall(monkeypatch, True)
    lam.lam_score_topk(qt, codes, width, n, d, eps, bound, k, metric, s, i, ws)
    assert lam.lam_score_topk_status(ws) == lam.LAM_ERR_TIMEOUT
    torch.cuda.synchronize()
    stall(monkeypatch, False)
    # the same workspace, the next ordinary call: status cleared, results right
    lam.lam_score_topk(qt, codes, width, n, d, eps, bound, k, metric, s, i, ws)
    assert lam.lam_score_topk_status(ws) == lam.LAM_OK
    os_, oi = oracle_topk(q, oc, eps, metric, k)
    check_topk(s.cpu().numpy(), i.cpu().numpy(), q, oc, eps, metric, os_, oi)


@pytest.mark.parametrize("B", [1, 200])
def test_wait_budget_runs_out_on_per_vector_rows(dev, monkeypatch, B):
    """The per-vector int8 codec's bandwidth (B = 1) and tensor (B = 200) kernels."""
    n, d, k = 2000, 768, 10
    x = inputs.unit_rows(n, d, seed=B)
    oc, osc, oof = oracle.encode_rows(x, oracle.FMT_INT8_ROWS)
    codes = torch.from_numpy(oc).to(dev)
    scale = torch.from_numpy(osc).to(dev)
    offset = torch.from_numpy(oof).to(dev)
    q = inputs.queries(B, d, seed=B + 1)
    qt = torch.from_numpy(q).to(dev)
    fmt = lam.LAM_ROWS_INT8
    ws = torch.empty(lam.lam_score_topk_rows_workspace_size(B, n, d, k, fmt), dtype=torch.uint8,
                     device=dev)
    s = torch.empty((B, k), dtype=torch.float32, device=dev)
    i = torch.empty((B, k), dtype=torch.int64, device=dev)
    stall(monkeypatch, True)
    lam.lam_score_topk_rows(qt, codes, fmt, scale, offset, n, d, k, oracle.IP, s, i, ws)
    assert lam.lam_score_topk_status(ws) == lam.LAM_ERR_TIMEOUT
    torch.cuda.synchronize()
    stall(monkeypatch, False)
    lam.lam_score_topk_rows(qt, codes, fmt, scale, offset, n, d, k, oracle.IP, s, i, ws)
    assert lam.lam_score_topk_status(ws) == lam.LAM_OK
    rows = oracle.decode_rows(oc, oracle.FMT_INT8_ROWS, d, osc, oof)
    full = oracle.scores_rows(q, rows, oracle.IP)
    os_, oi = oracle.topk(full, k, oracle.IP)
    check_topk_fn(s.cpu().numpy(), i.cpu().numpy(), lambda b, ids: full[b, ids], n, oracle.IP,
                  os_, oi)
