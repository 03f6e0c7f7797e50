"""lam_score_topk_noalloc: the search for callers that cannot allocate device
memory (their framework owns all device memory, or cudaMalloc's implicit
synchronisation is not acceptable).  Its scratch is a fixed array inside the
library, so it must give the same results as lam_score_topk with a caller
workspace, call after call, even though every call reuses the same array --
also when consecutive calls lay the array out differently (tensor-core query
images, then bandwidth-kernel partial lists, then tensor-core again).
This file runs last so that a failure here leaves every other test run."""
import ctypes

import numpy as np
import pytest
import torch

import oracle
import paper_2609_32256_gb300 as lam
from paper_2609_32256_gb300 import inputs
from tests.parity import check_topk, oracle_topk, tol

pytestmark = pytest.mark.gpu
NP_DT = {1: np.int8, 2: np.int16}


def noalloc_call(lib, q, codes, width, eps, bound, k, metric):
    B, D = q.shape
    N = codes.shape[0]
    s = torch.full((B, k), float("nan"), dtype=torch.float32, device=q.device)
    i = torch.full((B, k), -1, dtype=torch.int64, device=q.device)
    st = lib.lam_score_topk_noalloc(
        ctypes.c_void_p(q.data_ptr()), B, ctypes.c_void_p(codes.data_ptr()), width, N, D,
        ctypes.c_float(eps), bound, k, metric, ctypes.c_void_p(s.data_ptr()),
        ctypes.c_void_p(i.data_ptr()),
        ctypes.c_void_p(torch.cuda.current_stream(q.device).cuda_stream))
    return st, s.cpu().numpy(), i.cpu().numpy()


def make_case(dev, n, width, eps, seed):
    x = inputs.unit_rows(n, 768, seed=seed)
    oc, rmin, rmax, _ = oracle.quantize(x, eps)
    bound = max(-int(rmin), int(rmax))
    codes = torch.from_numpy(oc.reshape(n, 768).astype(NP_DT[width])).to(dev)
    return codes, bound, oc.reshape(n, 768)


def same_as_workspace_call(lib, q, codes, width, eps, bound, k, metric):
    st, s_na, i_na = noalloc_call(lib, q, codes, width, eps, bound, k, metric)
    assert st == lam.LAM_OK, lam.lam_status_string(st)
    s_ws, i_ws = lam.search(q, codes, eps, k, metric, code_bound=bound)
    s_ws, i_ws = s_ws.cpu().numpy(), i_ws.cpu().numpy()
    assert np.all(np.abs(s_na.astype(np.float64) - s_ws) <= tol(s_ws))
    np.testing.assert_array_equal(i_na, i_ws)
    return s_na, i_na


@pytest.mark.parametrize("B,width,eps,metric,k,path", [
    (64, 1, 1e-2, oracle.IP, 10, lam.PATH_TENSOR),
    (1, 2, 1e-3, oracle.L2, 100, lam.PATH_BANDWIDTH),
    (5, 2, 1e-4, oracle.COSINE, 20, lam.PATH_TENSOR)])
def test_noalloc_matches_workspace_entry_point_twice(dev, B, width, eps, metric, k, path):
    lib = lam.load()
    codes, bound, oc = make_case(dev, 6000, width, eps, seed=B)
    assert lam.lam_score_topk_path(B, 6000, 768, k, width, bound) == path
    for call in range(2):  # two calls in a row reuse the same scratch
        q = torch.from_numpy(inputs.queries(B, 768, seed=100 + call)).to(dev)
        s_na, i_na = same_as_workspace_call(lib, q, codes, width, eps, bound, k, metric)
        if call == 0:  # and once against the oracle directly
            qn = q.cpu().numpy()
            os_, oi = oracle_topk(qn, oc, eps, metric, k)
            check_topk(s_na, i_na, qn, oc, eps, metric, os_, oi)


def test_noalloc_alternating_layouts(dev):
    """Tensor path, bandwidth path, tensor path again through the one array:
    each call must not read what the previous, differently laid out call left."""
    lib = lam.load()
    c8, b8, oc8 = make_case(dev, 5000, 1, 1e-2, seed=41)
    c16, b16, oc16 = make_case(dev, 7000, 2, 1e-3, seed=42)
    plan = [(c8, b8, oc8, 1, 1e-2, 96, oracle.IP, 16, lam.PATH_TENSOR),
            (c16, b16, oc16, 2, 1e-3, 2, oracle.L2, 64, lam.PATH_BANDWIDTH),
            (c8, b8, oc8, 1, 1e-2, 130, oracle.COSINE, 10, lam.PATH_TENSOR),
            (c16, b16, oc16, 2, 1e-3, 1, oracle.IP, 5, lam.PATH_BANDWIDTH)]
    for n, (codes, bound, oc, w, eps, B, metric, k, path) in enumerate(plan):
        assert lam.lam_score_topk_path(B, codes.shape[0], 768, k, w, bound) == path
        q = torch.from_numpy(inputs.queries(B, 768, seed=200 + n)).to(dev)
        s_na, i_na = same_as_workspace_call(lib, q, codes, w, eps, bound, k, metric)
        sel = np.arange(min(B, 8))
        qn = q.cpu().numpy()[sel]
        os_, oi = oracle_topk(qn, oc, eps, metric, k)
        check_topk(s_na[sel], i_na[sel], qn, oc, eps, metric, os_, oi)


def test_noalloc_rejects_shapes_beyond_its_scratch(dev):
    lib = lam.load()
    B, N, D, k = 4096, 361802, 768, 100
    assert lam.lam_score_topk_workspace_size(B, N, D, k, 1, 100) > (16 << 20)
    st = lib.lam_score_topk_noalloc(ctypes.c_void_p(256), B, ctypes.c_void_p(256), 1, N, D,
                                    ctypes.c_float(1e-2), 100, k, 0, ctypes.c_void_p(256),
                                    ctypes.c_void_p(256), None)
    assert st == lam.LAM_ERR_WORKSPACE


def test_noalloc_argument_errors_match_the_workspace_entry_point(dev):
    """Bad arguments get lam_score_topk's own statuses, nothing queued."""
    lib = lam.load()
    fake = ctypes.c_void_p(256)
    # k above N: invalid shape
    st = lib.lam_score_topk_noalloc(fake, 1, fake, 1, 10, 768, ctypes.c_float(1e-2), 0, 11, 0,
                                    fake, fake, None)
    assert st == lam.LAM_ERR_INVALID
    # a metric that does not exist
    st = lib.lam_score_topk_noalloc(fake, 1, fake, 1, 100, 768, ctypes.c_float(1e-2), 0, 10, 7,
                                    fake, fake, None)
    assert st == lam.LAM_ERR_INVALID
