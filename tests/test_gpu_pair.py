"""CTA pairs for the batched tensor kernel (LAM_SCORE_PAIR=1): 2-CTA clusters
over query blocks 2j and 2j + 1, the even CTA issuing M = 256 MMAs for both and
each CTA staging half of every 256-row code block.  Parity with the CPU oracle
over ragged memories, both code widths (int16 beyond +-2048 split as 256 h + l),
every metric and k from 1 to 100, and the per-vector codecs; results
bit-identical to the single-CTA kernel (same operands, same K order); an odd
number of query blocks falling back to single CTAs; and the bounded waits of
the pair's roles."""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_32256_gb300 as lam
from paper_2609_32256_gb300 import inputs
from tests.parity import check_topk, oracle_topk
from tests.test_gpu_rows import FMTS, rows_case

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def pair_kernel(monkeypatch):
    monkeypatch.setenv("LAM_SCORE_PAIR", "1")


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
@pytest.mark.parametrize("width,eps", [(1, 1e-2), (2, 1e-3), (2, 1e-4)])
@pytest.mark.parametrize("B,k", [(512, 1), (512, 10), (768, 32), (512, 100), (600, 10)])
@pytest.mark.parametrize("N", [300, 2100])
def test_parity(dev, score_path, metric, width, eps, B, k, N):
    score_path("tensor")
    codes, bound = codes_for(N, 768, eps, seed=N + B)
    q = inputs.queries(B, 768, seed=B + k)
    gs, gi = gpu_search(dev, q, codes, width, eps, min(k, N), metric, bound)
    os_, oi = oracle_topk(q, codes, eps, metric, min(k, N))
    check_topk(gs, gi, q, codes, eps, metric, os_, oi)


@pytest.mark.parametrize("width,eps", [(1, 1e-2), (2, 1e-3)])
@pytest.mark.parametrize("metric", METRICS)
def test_bit_identical_to_single_cta(dev, monkeypatch, score_path, width, eps, metric):
    score_path("tensor")
    codes, bound = codes_for(20000, 768, eps, seed=3)
    q = inputs.queries(1024, 768, seed=4)
    ps, pi = gpu_search(dev, q, codes, width, eps, 10, metric, bound)
    monkeypatch.setenv("LAM_SCORE_PAIR", "0")
    ss, si = gpu_search(dev, q, codes, width, eps, 10, metric, bound)
    monkeypatch.setenv("LAM_SCORE_PAIR", "1")
    assert np.array_equal(ps.view(np.uint32), ss.view(np.uint32))
    assert np.array_equal(pi, si)
    # and against the oracle on a sample of the queries
    sel = np.arange(0, 1024, 37)
    os_, oi = oracle_topk(q[sel], codes, eps, metric, 10)
    check_topk(ps[sel], pi[sel], q[sel], codes, eps, metric, os_, oi)


@pytest.mark.parametrize("metric", METRICS)
@pytest.mark.parametrize("fmt", FMTS)
@pytest.mark.parametrize("B", [130, 512])
def test_row_codecs(dev, score_path, fmt, metric, B):
    score_path("tensor")
    rows_case(dev, fmt, 3001, 768, B, 10, metric, seed=B + 1)


@pytest.mark.parametrize("D", [16, 80, 1024])
def test_k_extents(dev, score_path, D):
    score_path("tensor")
    codes, bound = codes_for(1500, D, 1e-2, seed=D)
    q = inputs.queries(512, D, seed=D + 1)
    for metric in METRICS:
        gs, gi = gpu_search(dev, q, codes, 1, 1e-2, 10, metric, bound)
        os_, oi = oracle_topk(q, codes, 1e-2, metric, 10)
        check_topk(gs, gi, q, codes, 1e-2, metric, os_, oi)


@pytest.mark.parametrize("width,eps,metric", [(1, 1e-2, oracle.L2), (2, 1e-3, oracle.COSINE)])
def test_wait_budget_runs_out_then_device_recovers(dev, monkeypatch, score_path, width, eps,
                                                   metric):
    score_path("tensor")
    n, d, B, k = 3000, 768, 512, 10
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
