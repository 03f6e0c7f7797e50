"""lam_score_topk_noalloc: the search for callers that cannot allocate device
memory (their framework owns all device memory, or cudaMalloc's implicit
synchronisation is not acceptable).  Its scratch is a fixed array inside the
library, so it must give the same results as lam_score_topk with a caller
workspace, call after call, even though every call reuses the same array.
This file runs last so that a failure here leaves every other test run."""
import ctypes

import numpy as np
import pytest
import torch

import oracle
import paper_2609_32256_gb300 as lam
from paper_2609_32256_gb300 import inputs
from tests.parity import tol

pytestmark = pytest.mark.gpu


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


@pytest.mark.parametrize("B,width,eps,metric,k", [
    (64, 1, 1e-2, oracle.IP, 10),       # tensor-core path
    (1, 2, 1e-3, oracle.L2, 100),       # bandwidth path
    (5, 2, 1e-4, oracle.COSINE, 20)])   # tensor-core path, int16
def test_noalloc_matches_workspace_entry_point_twice(dev, B, width, eps, metric, k):
    lib = lam.load()
    x = inputs.unit_rows(6000, 768, seed=B)
    oc, rmin, rmax, _ = oracle.quantize(x, eps)
    bound = max(-int(rmin), int(rmax))
    dt = {1: np.int8, 2: np.int16}[width]
    codes = torch.from_numpy(oc.reshape(6000, 768).astype(dt)).to(dev)
    for call in range(2):  # two calls in a row reuse the same scratch
        q = torch.from_numpy(inputs.queries(B, 768, seed=100 + call)).to(dev)
        st, s_na, i_na = noalloc_call(lib, q, codes, width, eps, bound, k, metric)
        assert st == lam.LAM_OK, lam.lam_status_string(st)
        s_ws, i_ws = lam.search(q, codes, eps, k, metric, code_bound=bound)
        s_ws, i_ws = s_ws.cpu().numpy(), i_ws.cpu().numpy()
        assert np.all(np.abs(s_na.astype(np.float64) - s_ws) <= tol(s_ws))
        np.testing.assert_array_equal(i_na, i_ws)


def test_noalloc_rejects_shapes_beyond_its_scratch(dev):
    lib = lam.load()
    B, N, D, k = 4096, 361802, 768, 100
    assert lam.lam_score_topk_workspace_size(B, N, D, k, 1, 100) > (16 << 20)
    st = lib.lam_score_topk_noalloc(ctypes.c_void_p(256), B, ctypes.c_void_p(256), 1, N, D,
                                    ctypes.c_float(1e-2), 100, k, 0, ctypes.c_void_p(256),
                                    ctypes.c_void_p(256), None)
    assert st == lam.LAM_ERR_WORKSPACE
