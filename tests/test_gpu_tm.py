"""The opt-in small-batch tensor kernel (LAM_SCORE_TM=1: 3 to 64 queries,
k <= 32, the codes in the MMA M dimension, converted into tensor memory):
parity with the CPU oracle over ragged memories (fewer rows than one 128-row
tile, ragged last tiles, one CTA or many), K extents that end inside a
64-wide slice, both code widths and every metric; the same top-k as the
default stage-loop tensor kernel on the same inputs; and the bounded waits of
its roles."""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_32256_gb300 as lam
from paper_2609_32256_gb300 import inputs
from tests.parity import check_topk, oracle_topk

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def tm_kernel(monkeypatch):
    monkeypatch.setenv("LAM_SCORE_TM", "1")


METRICS = (oracle.IP, oracle.COSINE, oracle.L2)
NP_DT = {1: np.int8, 2: np.int16}


def codes_for(n, d, eps, seed):
    x = inputs.unit_rows(n, d, seed=seed)
    oc, rmin, rmax, _ = oracle.quantize(x, eps)
    return oc.reshape(n, d), max(-int(rmin), int(rmax))


def gpu_search(dev, q, codes, width, eps, k, metric, bound):
    qt = torch.from_numpy(q).to(dev)
    ct = torch.from_numpy(codes.astype(NP_DT[width])).to(dev)
    s, i = lam.search(qt, ct, eps, k, metric, code_bound=bound)
    return s.cpu().numpy(), i.cpu().numpy()


@pytest.mark.parametrize("metric", METRICS)
@pytest.mark.parametrize("width,eps", [(1, 1e-2), (2, 1e-3), (2, 2e-4)])
@pytest.mark.parametrize("B,k", [(3, 1), (16, 10), (33, 32), (64, 10)])
@pytest.mark.parametrize("N", [100, 257, 5000])
def test_parity(dev, score_path, metric, width, eps, B, k, N):
    score_path("tensor")
    codes, bound = codes_for(N, 768, eps, seed=N + B)
    q = inputs.queries(B, 768, seed=B + k)
    assert lam.lam_score_topk_path(B, N, 768, k, width, bound) == lam.PATH_TENSOR
    gs, gi = gpu_search(dev, q, codes, width, eps, min(k, N), metric, bound)
    os_, oi = oracle_topk(q, codes, eps, metric, min(k, N))
    check_topk(gs, gi, q, codes, eps, metric, os_, oi)


@pytest.mark.parametrize("D", [16, 48, 80, 112, 1024])
@pytest.mark.parametrize("width,eps", [(1, 1e-2), (2, 1e-3)])
def test_k_extents(dev, score_path, D, width, eps):
    score_path("tensor")
    codes, bound = codes_for(1500, D, eps, seed=D)
    q = inputs.queries(24, D, seed=D + 1)
    for metric in METRICS:
        gs, gi = gpu_search(dev, q, codes, width, eps, 10, metric, bound)
        os_, oi = oracle_topk(q, codes, eps, metric, 10)
        check_topk(gs, gi, q, codes, eps, metric, os_, oi)


@pytest.mark.parametrize("width,eps", [(1, 1e-2), (2, 1e-3)])
@pytest.mark.parametrize("metric", METRICS)
def test_same_topk_as_stage_loop_kernel(dev, monkeypatch, score_path, width, eps, metric):
    score_path("tensor")
    codes, bound = codes_for(20000, 768, eps, seed=7)
    q = inputs.queries(64, 768, seed=8)
    gs, gi = gpu_search(dev, q, codes, width, eps, 10, metric, bound)
    monkeypatch.setenv("LAM_SCORE_TM", "0")
    hs, hi = gpu_search(dev, q, codes, width, eps, 10, metric, bound)
    monkeypatch.setenv("LAM_SCORE_TM", "1")
    os_, oi = oracle_topk(q, codes, eps, metric, 10)
    check_topk(gs, gi, q, codes, eps, metric, os_, oi)
    check_topk(hs, hi, q, codes, eps, metric, os_, oi)
    # the two kernels differ only in fp32 accumulation order
    tol = 2e-6 + 2e-5 * np.abs(hs)
    assert np.all(np.abs(gs - hs) <= tol)


def test_exact_duplicates_rank_lower_id_first(dev, score_path):
    score_path("tensor")
    codes, bound = codes_for(3000, 768, 1e-2, seed=11)
    codes[1777] = codes[5]
    codes[2900] = codes[5]
    q = inputs.queries(8, 768, seed=12)
    q[3] = codes[5] * 0.02  # query 3 points at the duplicated row
    for metric in METRICS:
        gs, gi = gpu_search(dev, q.astype(np.float32), codes, 1, 1e-2, 5, metric, bound)
        row = list(gi[3])
        assert row.index(5) < row.index(1777) < row.index(2900)
        os_, oi = oracle_topk(q.astype(np.float32), codes, 1e-2, metric, 5)
        check_topk(gs, gi, q.astype(np.float32), codes, 1e-2, metric, os_, oi)


@pytest.mark.parametrize("width,eps,metric", [(1, 1e-2, oracle.L2), (2, 1e-3, oracle.COSINE)])
def test_wait_budget_runs_out_then_device_recovers(dev, monkeypatch, score_path, width, eps,
                                                   metric):
    score_path("tensor")
    n, d, B, k = 3000, 768, 40, 10
    codes, bound = codes_for(n, d, eps, seed=21)
    ct = torch.from_numpy(codes.astype(NP_DT[width])).to(dev)
    q = inputs.queries(B, d, seed=22)
    qt = torch.from_numpy(q).to(dev)
    ws = torch.empty(lam.lam_score_topk_workspace_size(B, n, d, k, width, bound),
                     dtype=torch.uint8, device=dev)
    s = torch.empty((B, k), dtype=torch.float32, device=dev)
    i = torch.empty((B, k), dtype=torch.int64, device=dev)
    monkeypatch.setenv("LAM_TEST_WAIT_CYCLES", "20000")
    monkeypatch.setenv("LAM_TEST_STALL", "1")
    lam.lam_score_topk(qt, ct, width, n, d, eps, bound, k, metric, s, i, ws)
    assert lam.lam_score_topk_status(ws) == lam.LAM_ERR_TIMEOUT
    torch.cuda.synchronize()
    monkeypatch.delenv("LAM_TEST_WAIT_CYCLES")
    monkeypatch.delenv("LAM_TEST_STALL")
    lam.lam_score_topk(qt, ct, width, n, d, eps, bound, k, metric, s, i, ws)
    assert lam.lam_score_topk_status(ws) == lam.LAM_OK
    os_, oi = oracle_topk(q, codes, eps, metric, k)
    check_topk(s.cpu().numpy(), i.cpu().numpy(), q, codes, eps, metric, os_, oi)
