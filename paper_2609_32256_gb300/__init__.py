"""GB300 (sm_103a) library for LAM's quantized agent memory.

The C ABI (include/lam.h, built as liblam.so) computes the error-bounded
quantizer Q_eps(x) = round(x / 2 eps) over fp32 embeddings, its inverse, and
exact top-k retrieval scored directly on the integer codes.  This package is
the Python side: the ctypes binding (`_lib`, same names as the C calls) and a
few conveniences that allocate outputs with PyTorch.  PyTorch only provides
device memory and streams; every step runs in the library's kernels.
"""
from __future__ import annotations

from ._lib import (LAM_ERR_CUDA, LAM_ERR_INVALID, LAM_ERR_NONFINITE, LAM_ERR_RANGE,
                   LAM_ERR_TIMEOUT, LAM_ERR_UNSUPPORTED, LAM_ERR_WORKSPACE, LAM_I8, LAM_I16,
                   LAM_I32, LAM_METRIC_COSINE, LAM_METRIC_IP, LAM_METRIC_L2, LAM_OK,
                   LAM_WIDTH_AUTO, PATH_BANDWIDTH, PATH_GENERIC, PATH_TENSOR, LamError,
                   lam_dequantize, lam_quantize, lam_quantize_workspace_size,
                   lam_score_topk, lam_score_topk_path, lam_score_topk_status,
                   lam_score_topk_workspace_size, lam_status_string, lam_version, load,
                   LAM_TIME_AUX, LAM_TIME_MERGE, LAM_TIME_DEQUANTIZE, LAM_TIME_QUANTIZE, LAM_TIME_SCORE,
                   lam_timing_begin, lam_timing_end, lam_timing_read, lam_code_sqnorms,
                   lam_quantize_bands, lam_admit_batch, lam_admit_batch_workspace_size,
                   lam_lamz_bound, lam_lamz_compress, lam_lamz_decompress,
                   lam_lamz_workspace_size, LAM_ROWS_INT8, LAM_ROWS_FP16, LAM_ROWS_SIGN,
                   lam_encode_rows, lam_decode_rows, lam_score_topk_rows,
                   lam_score_topk_rows_path, lam_score_topk_rows_workspace_size,
                   lam_quantize_async, lam_quantize_result, lam_dequantize_from,
                   lam_score_topk_from, lam_score_topk_from_path,
                   lam_score_topk_from_workspace_size)

CODE_DTYPES = {1: "int8", 2: "int16", 4: "int32"}


def _torch():
    import torch
    return torch


def quantize(x, eps, width=LAM_WIDTH_AUTO, stream=None):
    """Q_eps of a CUDA fp32 tensor.

    Returns (codes, width, scale, code_min, code_max); codes has x's shape and
    the narrowest integer dtype (or the forced one).
    """
    torch = _torch()
    x = x.contiguous()
    n = x.numel()
    ws = torch.empty(max(16, lam_quantize_workspace_size()), dtype=torch.uint8, device=x.device)
    if width == LAM_WIDTH_AUTO:
        _, w, _, _, _ = lam_quantize(x, eps, LAM_WIDTH_AUTO, None, ws, stream)
    else:
        w = width
    codes = torch.empty(x.shape, dtype=getattr(torch, CODE_DTYPES[w]), device=x.device)
    _, w2, scale, cmin, cmax = lam_quantize(x, eps, w, codes if n else None, ws, stream)
    return codes, w2, scale, cmin, cmax


def dequantize(codes, scale, stream=None):
    """scale * codes as a CUDA fp32 tensor of the same shape."""
    torch = _torch()
    w = codes.element_size()
    out = torch.empty(codes.shape, dtype=torch.float32, device=codes.device)
    lam_dequantize(codes.contiguous(), w, codes.numel(), scale, out, stream)
    return out


def search(queries, codes, eps, k, metric=LAM_METRIC_IP, code_bound=None, stream=None):
    """Top-k of every query against every code row: (scores [B,k] f32, ids [B,k] i64).

    code_bound: the largest |code| (max(-code_min, code_max) from quantize),
    or None.  Every int8 code is bounded by 128; for int16 codes, None means
    unknown, and the tensor cores then score the codes split as 256 h + l
    (exact for every int16 code, twice the tensor work of a bound <= 2048)."""
    torch = _torch()
    queries = queries.contiguous()
    codes = codes.contiguous()
    B, D = queries.shape
    N = codes.shape[0]
    w = codes.element_size()
    if code_bound is None:
        code_bound = 128 if w == 1 else 0
    nbytes = lam_score_topk_workspace_size(B, N, D, k, w, code_bound)
    if nbytes == 0:
        raise LamError(LAM_ERR_INVALID, "lam_score_topk_workspace_size")
    ws = torch.empty(nbytes, dtype=torch.uint8, device=queries.device)
    scores = torch.empty((B, k), dtype=torch.float32, device=queries.device)
    ids = torch.empty((B, k), dtype=torch.int64, device=queries.device)
    lam_score_topk(queries, codes, w, N, D, eps, code_bound, k, metric, scores, ids, ws, stream)
    st = lam_score_topk_status(ws, stream)
    if st != LAM_OK:
        raise LamError(st, "lam_score_topk")
    return scores, ids


def encode_rows(x, fmt, stream=None):
    """Per-vector codec of CUDA fp32 rows x [N, D]: (codes, scale, offset),
    scale/offset None where the codec has none."""
    torch = _torch()
    x = x.contiguous()
    N, D = x.shape
    dev = x.device
    if fmt == LAM_ROWS_INT8:
        codes = torch.empty((N, D), dtype=torch.int8, device=dev)
    elif fmt == LAM_ROWS_FP16:
        codes = torch.empty((N, D), dtype=torch.float16, device=dev)
    else:
        codes = torch.empty((N, D // 8), dtype=torch.uint8, device=dev)
    scale = torch.empty(N, dtype=torch.float32, device=dev) if fmt != LAM_ROWS_FP16 else None
    offset = torch.empty(N, dtype=torch.float32, device=dev) if fmt == LAM_ROWS_INT8 else None
    lam_encode_rows(x, fmt, codes, scale, offset, stream)
    return codes, scale, offset


def search_rows(queries, codes, fmt, scale, offset, k, metric=LAM_METRIC_IP, D=None,
                stream=None):
    """Top-k of every query against rows in a per-vector codec."""
    torch = _torch()
    queries = queries.contiguous()
    B, Dq = queries.shape
    D = Dq if D is None else D
    N = codes.shape[0]
    nbytes = lam_score_topk_rows_workspace_size(B, N, D, k, fmt)
    if nbytes == 0:
        raise LamError(LAM_ERR_INVALID, "lam_score_topk_rows_workspace_size")
    ws = torch.empty(nbytes, dtype=torch.uint8, device=queries.device)
    scores = torch.empty((B, k), dtype=torch.float32, device=queries.device)
    ids = torch.empty((B, k), dtype=torch.int64, device=queries.device)
    lam_score_topk_rows(queries, codes, fmt, scale, offset, N, D, k, metric, scores, ids, ws,
                        stream)
    st = lam_score_topk_status(ws, stream)
    if st != LAM_OK:
        raise LamError(st, "lam_score_topk_rows")
    return scores, ids
