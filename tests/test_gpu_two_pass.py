"""Two-pass tensor-core search (Q_eps codes): a first pass scores with the fp16
hi term of the query alone (half the MMAs), keeps a few more candidates than
k per list, and the merge rescores every candidate exactly on the codes and
certifies the result: a row left out scored no better than the last
candidate by the hi-only score, and the dropped lo term moves a score by at
most 2^-11 ||q|| ||c|| (+ fp32 accumulation).  An uncertified query makes the
full (hi + lo) pass run.  The two-pass search is opt-in (LAM_SCORE_HI=1).
Every outcome must match the oracle: the certified path, the full pass alone
(the default), the full pass forced by a test hook (LAM_TEST_HI_FAIL=1), and
a memory of many exact duplicates, where the certification itself fails."""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_32256_gb300 as lam
from paper_2609_32256_gb300 import inputs
from tests.parity import check_topk, oracle_topk

pytestmark = pytest.mark.gpu
METRICS = (oracle.IP, oracle.COSINE, oracle.L2)
NP_DT = {1: np.int8, 2: np.int16}


def case(dev, n, d, eps, width, seed, B, dup=0):
    x = inputs.unit_rows(n, d, seed=seed)
    q = inputs.queries(B, d, seed=seed + 1)
    if dup:
        x[100:100 + dup] = x[7]  # dup + 1 identical rows
        q[0] = x[7]
    oc, rmin, rmax, _ = oracle.quantize(x, eps)
    assert oracle.width(rmin, rmax) <= width
    oc = oc.reshape(n, d)
    bound = max(-int(rmin), int(rmax))
    codes = torch.from_numpy(oc.astype(NP_DT[width])).to(dev)
    return q, oc, codes, bound


def search_and_check(dev, q, oc, codes, width, eps, k, metric, bound, sel=None):
    s, i = lam.search(torch.from_numpy(q).to(dev), codes, eps, k, metric, bound)
    s, i = s.cpu().numpy(), i.cpu().numpy()
    sel = np.arange(q.shape[0]) if sel is None else sel
    os_, oi = oracle_topk(q[sel], oc, eps, metric, k)
    check_topk(s[sel], i[sel], q[sel], oc, eps, metric, os_, oi)
    return s, i


@pytest.mark.parametrize("mode", ["default", "full_only", "forced_fallback"])
@pytest.mark.parametrize("metric", METRICS)
@pytest.mark.parametrize("B,width,eps,k", [
    (8, 1, 1e-2, 10),      # stage-loop kernel, register lists
    (64, 2, 1e-3, 25),     # stage-loop kernel, int16 codes, heaps
    (300, 1, 1e-2, 100),   # stage-loop kernel, three query blocks, heaps
    (520, 1, 1e-2, 10),    # conversion pass + scoring kernel
    (600, 2, 1e-3, 64)])   # conversion pass, int16, heaps
def test_two_pass_matches_oracle(dev, monkeypatch, mode, metric, B, width, eps, k):
    if mode != "full_only":
        monkeypatch.setenv("LAM_SCORE_HI", "1")
    if mode == "forced_fallback":
        monkeypatch.setenv("LAM_TEST_HI_FAIL", "1")
    q, oc, codes, bound = case(dev, 4000, 768, eps, width, seed=B + k, B=B)
    assert lam.lam_score_topk_path(B, 4000, 768, k, width, bound) == lam.PATH_TENSOR
    sel = np.unique(np.r_[0, 1, B // 2, B - 1])
    search_and_check(dev, q, oc, codes, width, eps, k, metric, bound, sel)


@pytest.mark.parametrize("metric", METRICS)
@pytest.mark.parametrize("B", [4, 520])
@pytest.mark.parametrize("k", [1, 10, 40])
def test_duplicates_beyond_the_candidates_fall_back(dev, monkeypatch, metric, B, k):
    """60 copies of one row (more than any candidate list holds) and a query
    equal to it: the certification cannot separate the copies, the full pass
    runs, and the copies come back in id order."""
    monkeypatch.setenv("LAM_SCORE_HI", "1")
    q, oc, codes, bound = case(dev, 3000, 768, 1e-2, 1, seed=5, B=B, dup=59)
    s, i = search_and_check(dev, q, oc, codes, 1, 1e-2, k, metric, bound, np.array([0, 1]))
    copies = np.r_[7, np.arange(100, 159)]
    np.testing.assert_array_equal(i[0], copies[:k])
