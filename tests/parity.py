"""Element-by-element comparison of the CUDA path with the CPU oracle.

Tolerance for fp32 scores: |gpu - oracle| <= 1e-6 + 1e-5 |oracle|.  Top-k ids
must agree except among scores tied within that tolerance: every GPU score
matches the oracle's score for the same id, the lists are in rank order
(equal scores by lower id), the k-th scores agree, and an id is missing from
either list only if its oracle score is within twice the tolerance of the
oracle's k-th score.
"""
import concurrent.futures as cf
import os

import numpy as np

import oracle

ABS_TOL = 1e-6
REL_TOL = 1e-5
NTHREADS = max(1, os.cpu_count() or 1)

# Largest |gpu - oracle| / tolerance seen by each test (printed in the
# terminal summary), so that the margin left inside the tolerance is visible.
WORST = {}


def _record_margin(ratio):
    name = os.environ.get("PYTEST_CURRENT_TEST", "?").split(" ")[0]
    if ratio > WORST.get(name, -1.0):
        WORST[name] = float(ratio)


def quantize_rows(x, eps, chunk_rows=65536):
    """oracle.quantize over the rows of x [N, D] in chunks on the host cores.

    The oracle call itself is unchanged; the chunks only spread independent
    rows over threads (ctypes releases the GIL).  Returns (codes int32 [N, D],
    rmin, rmax, n_nonfinite) as oracle.quantize does for the whole array."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    N = x.shape[0]
    spans = [(r, min(N, r + chunk_rows)) for r in range(0, N, chunk_rows)]
    with cf.ThreadPoolExecutor(max_workers=NTHREADS) as ex:
        parts = list(ex.map(lambda s: oracle.quantize(x[s[0]:s[1]], eps), spans))
    codes = np.concatenate([p[0] for p in parts]).reshape(x.shape)
    return (codes, min(p[1] for p in parts), max(p[2] for p in parts),
            sum(p[3] for p in parts))


def tol(x):
    return ABS_TOL + REL_TOL * np.abs(np.asarray(x, dtype=np.float64))


def check_topk(g_scores, g_ids, queries, codes_i32, eps, metric, o_scores, o_ids,
               row_offset=0):
    """Compare GPU (scores, ids) [B, k] with the oracle's top-k for the same queries.

    codes_i32: the [N, D] codes (int32) the ids index (ids - row_offset).
    """
    def score_at(b, ids):
        return oracle.scores(queries[b:b + 1], codes_i32[ids - row_offset], eps, metric)[0]
    check_topk_fn(g_scores, g_ids, score_at, codes_i32.shape[0], metric, o_scores, o_ids,
                  row_offset)


def check_topk_fn(g_scores, g_ids, score_at, n_rows, metric, o_scores, o_ids, row_offset=0):
    """check_topk with the oracle's score of (query b, ids) given by score_at."""
    g_scores = np.asarray(g_scores, dtype=np.float32)
    g_ids = np.asarray(g_ids, dtype=np.int64)
    B, k = g_scores.shape
    desc = metric != oracle.L2
    for b in range(B):
        ids = g_ids[b]
        sc = g_scores[b]
        assert len(set(ids.tolist())) == k, "duplicate ids in query %d" % b
        assert ids.min() >= row_offset and ids.max() < row_offset + n_rows
        o_at = score_at(b, ids)
        err = np.abs(sc.astype(np.float64) - o_at.astype(np.float64))
        _record_margin(float(np.max(err / tol(o_at))))
        bad = np.nonzero(err > tol(o_at))[0]
        assert bad.size == 0, "query %d: score of id %d is %r, oracle %r" % (
            b, ids[bad[0]], sc[bad[0]], o_at[bad[0]])
        # rank order on the GPU's own scores, equal scores by lower id
        for j in range(k - 1):
            a, c = sc[j], sc[j + 1]
            better = a > c if desc else a < c
            assert better or (a == c and ids[j] < ids[j + 1]), "query %d not in rank order" % b
        ok = o_scores[b]
        kth = np.float64(ok[k - 1])
        assert abs(np.float64(sc[k - 1]) - kth) <= tol(kth), "query %d: k-th score" % b
        margin = 2 * tol(kth)
        gset, oset = set(ids.tolist()), set(o_ids[b].tolist())
        for i, s in zip(o_ids[b], ok):
            if i not in gset:
                assert abs(np.float64(s) - kth) <= margin, "query %d: oracle id %d missing" % (b, i)
        for i, s in zip(ids, o_at):
            if i not in oset:
                assert abs(np.float64(s) - kth) <= margin, "query %d: extra id %d" % (b, i)


def oracle_topk(queries, codes_i32, eps, metric, k):
    return oracle.search(queries, codes_i32, eps, metric, k, nthreads=NTHREADS)
