"""Thin ctypes binding of the C ABI in include/lam.h (argument marshalling only).

Every function keeps the name of the C entry point it wraps.  Tensors are
passed by device pointer; the CUDA stream defaults to torch's current stream
on the tensor's device.  Every computation runs in liblam.so: if the library
is missing, the first call raises instead of falling back to anything else.
"""
from __future__ import annotations

import ctypes
import os

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "liblam.so")

LAM_OK, LAM_ERR_INVALID, LAM_ERR_RANGE, LAM_ERR_NONFINITE = 0, 1, 2, 3
LAM_ERR_WORKSPACE, LAM_ERR_CUDA, LAM_ERR_TIMEOUT, LAM_ERR_UNSUPPORTED = 4, 5, 6, 7
LAM_WIDTH_AUTO, LAM_I8, LAM_I16, LAM_I32 = 0, 1, 2, 4
LAM_METRIC_IP, LAM_METRIC_COSINE, LAM_METRIC_L2 = 0, 1, 2
PATH_BANDWIDTH, PATH_TENSOR, PATH_GENERIC = 0, 1, 2


class LamError(RuntimeError):
    """A non-OK lam_status."""

    def __init__(self, status: int, where: str):
        self.status = int(status)
        super().__init__("%s: %s (status %d)" % (where, lam_status_string(status), status))


_lib = None


def load():
    """Load liblam.so (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError("liblam.so is not built: call paper_2609_32256_gb300.build.build()")
    lib = ctypes.CDLL(LIB_PATH)
    vp, i32, i64, f32, sz = (ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64,
                             ctypes.c_float, ctypes.c_size_t)
    P = ctypes.POINTER
    sig = {
        "lam_version": (i32, []),
        "lam_status_string": (ctypes.c_char_p, [i32]),
        "lam_quantize_workspace_size": (sz, []),
        "lam_quantize": (i32, [vp, i64, f32, i32, vp, sz, vp, sz, P(i32), P(f32), P(i32),
                               P(i32), vp]),
        "lam_dequantize": (i32, [vp, i32, i64, f32, vp, vp]),
        "lam_score_topk_workspace_size": (sz, [i64, i64, i32, i32, i32, i32]),
        "lam_score_topk": (i32, [vp, i64, vp, i32, i64, i32, f32, i32, i32, i32, vp, vp, vp,
                                 sz, vp]),
        "lam_score_topk_status": (i32, [vp, vp, P(i32)]),
        "lam_score_topk_path": (i32, [i64, i64, i32, i32, i32, i32]),
        "lam_score_topk_noalloc": (i32, [vp, i64, vp, i32, i64, i32, f32, i32, i32, i32, vp,
                                         vp, vp]),
        "lam_code_sqnorms": (i32, [vp, i32, i64, i32, vp, vp]),
        "lam_lamz_bound": (sz, [i64]),
        "lam_lamz_workspace_size": (sz, [i64]),
        "lam_lamz_compress": (i32, [vp, i64, f32, vp, sz, P(sz), vp, sz, vp]),
        "lam_lamz_decompress": (i32, [vp, sz, vp, i64, vp, sz, vp]),
        "lam_admit_batch_workspace_size": (sz, [i64, i32, i64]),
        "lam_admit_batch": (i32, [vp, i64, i32, vp, i32, ctypes.c_double, vp, vp, vp, sz, i64,
                                  P(ctypes.c_double), P(i64), P(i64), vp]),
        "lam_quantize_bands": (i32, [vp, i64, i32, f32, i32, i32, vp, sz, vp, vp, sz, P(i32),
                                     P(f32), P(i32), P(i32), vp]),
        "lam_quantize_async": (i32, [vp, i64, f32, i32, vp, sz, vp, sz, vp]),
        "lam_quantize_result": (i32, [vp, f32, i32, vp, P(i32), P(f32), P(i32), P(i32)]),
        "lam_dequantize_from": (i32, [vp, vp, i64, f32, vp, vp]),
        "lam_score_topk_from_workspace_size": (sz, [i64, i64, i32, i32]),
        "lam_score_topk_from_path": (i32, [i64, i64, i32, i32]),
        "lam_score_topk_from": (i32, [vp, i64, vp, vp, i64, i32, f32, i32, i32, vp, vp, vp, sz,
                                      vp]),
        "lam_encode_rows": (i32, [vp, i64, i32, i32, vp, vp, vp, vp]),
        "lam_decode_rows": (i32, [vp, i32, i64, i32, vp, vp, vp, vp]),
        "lam_score_topk_rows_workspace_size": (sz, [i64, i64, i32, i32, i32]),
        "lam_score_topk_rows_path": (i32, [i64, i64, i32, i32, i32]),
        "lam_score_topk_rows": (i32, [vp, i64, vp, i32, vp, vp, i64, i32, i32, i32, vp, vp, vp,
                                      sz, vp]),
        "lam_timing_begin": (i32, [i32, i64]),
        "lam_timing_read": (i32, [i32, P(ctypes.c_double), P(i64), P(i64)]),
        "lam_timing_end": (i32, []),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _lib = lib
    return lib


def _stream(stream, device=None):
    if stream is not None:
        return ctypes.c_void_p(int(stream))
    import torch
    return ctypes.c_void_p(torch.cuda.current_stream(device).cuda_stream)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _nbytes(t):
    return 0 if t is None else t.numel() * t.element_size()


def _check(status, where):
    if status != LAM_OK:
        raise LamError(status, where)


def lam_version() -> int:
    return int(load().lam_version())


def lam_status_string(status: int) -> str:
    return load().lam_status_string(int(status)).decode()


def lam_quantize_workspace_size() -> int:
    return int(load().lam_quantize_workspace_size())


def lam_quantize(x, eps, width_req=LAM_WIDTH_AUTO, codes=None, workspace=None, stream=None,
                 raise_on_error=True):
    """Q_eps of the fp32 CUDA tensor x into `codes` (a CUDA tensor or None).

    Returns (status, width, scale, code_min, code_max).  `workspace` is a CUDA
    tensor of >= lam_quantize_workspace_size() bytes (16-byte aligned).
    """
    w = ctypes.c_int32(0)
    s = ctypes.c_float(0)
    cmin = ctypes.c_int32(0)
    cmax = ctypes.c_int32(0)
    st = load().lam_quantize(_ptr(x), x.numel(), ctypes.c_float(eps), int(width_req),
                             _ptr(codes), _nbytes(codes), _ptr(workspace), _nbytes(workspace),
                             ctypes.byref(w), ctypes.byref(s), ctypes.byref(cmin),
                             ctypes.byref(cmax), _stream(stream, x.device))
    if raise_on_error and st not in (LAM_OK,):
        raise LamError(st, "lam_quantize")
    return int(st), w.value, s.value, cmin.value, cmax.value


def lam_dequantize(codes, width, n, scale, out, stream=None):
    """out[0:n] = scale * codes[0:n] (fp32), asynchronous on the stream."""
    st = load().lam_dequantize(_ptr(codes), int(width), int(n), ctypes.c_float(scale),
                               _ptr(out), _stream(stream, out.device))
    _check(st, "lam_dequantize")


def lam_score_topk_workspace_size(B, N, D, k, width, code_bound) -> int:
    return int(load().lam_score_topk_workspace_size(int(B), int(N), int(D), int(k), int(width),
                                                    int(code_bound)))


def lam_score_topk_path(B, N, D, k, width, code_bound) -> int:
    return int(load().lam_score_topk_path(int(B), int(N), int(D), int(k), int(width),
                                          int(code_bound)))


def lam_score_topk(queries, codes, width, N, D, eps, code_bound, k, metric, scores, ids,
                   workspace, stream=None):
    """Exact search on the codes; writes scores [B, k] and ids [B, k] (asynchronous)."""
    B = queries.shape[0]
    st = load().lam_score_topk(_ptr(queries), int(B), _ptr(codes), int(width), int(N), int(D),
                               ctypes.c_float(eps), int(code_bound), int(k), int(metric),
                               _ptr(scores), _ptr(ids), _ptr(workspace), _nbytes(workspace),
                               _stream(stream, queries.device))
    _check(st, "lam_score_topk")


def lam_quantize_async(x, eps, width_req, codes, workspace, stream=None):
    """Q_eps of x queued on the stream; the outcome stays in `workspace`."""
    st = load().lam_quantize_async(_ptr(x), x.numel(), ctypes.c_float(eps), int(width_req),
                                   _ptr(codes), _nbytes(codes), _ptr(workspace),
                                   _nbytes(workspace), _stream(stream, x.device))
    _check(st, "lam_quantize_async")


def lam_quantize_result(workspace, eps, width_req=LAM_WIDTH_AUTO, stream=None,
                        raise_on_error=True):
    """(status, width, scale, code_min, code_max) of an asynchronous Q_eps."""
    w = ctypes.c_int32(0)
    s = ctypes.c_float(0)
    cmin = ctypes.c_int32(0)
    cmax = ctypes.c_int32(0)
    st = load().lam_quantize_result(_ptr(workspace), ctypes.c_float(eps), int(width_req),
                                    _stream(stream, workspace.device), ctypes.byref(w),
                                    ctypes.byref(s), ctypes.byref(cmin), ctypes.byref(cmax))
    if raise_on_error and st != LAM_OK:
        raise LamError(st, "lam_quantize_result")
    return int(st), w.value, s.value, cmin.value, cmax.value


def lam_dequantize_from(codes, quant_workspace, n, eps, out, stream=None):
    st = load().lam_dequantize_from(_ptr(codes), _ptr(quant_workspace), int(n),
                                    ctypes.c_float(eps), _ptr(out), _stream(stream, out.device))
    _check(st, "lam_dequantize_from")


def lam_score_topk_from_workspace_size(B, N, D, k) -> int:
    return int(load().lam_score_topk_from_workspace_size(int(B), int(N), int(D), int(k)))


def lam_score_topk_from_path(B, N, D, k) -> int:
    return int(load().lam_score_topk_from_path(int(B), int(N), int(D), int(k)))


def lam_score_topk_from(queries, codes, quant_workspace, N, D, eps, k, metric, scores, ids,
                        workspace, stream=None):
    B = queries.shape[0]
    st = load().lam_score_topk_from(_ptr(queries), int(B), _ptr(codes), _ptr(quant_workspace),
                                    int(N), int(D), ctypes.c_float(eps), int(k), int(metric),
                                    _ptr(scores), _ptr(ids), _ptr(workspace), _nbytes(workspace),
                                    _stream(stream, queries.device))
    _check(st, "lam_score_topk_from")


LAM_ROWS_INT8, LAM_ROWS_FP16, LAM_ROWS_SIGN = 1, 2, 3


def lam_encode_rows(x, fmt, codes, scale=None, offset=None, stream=None):
    """Per-vector codec of the fp32 rows x [N, D] into codes (int8 [N, D],
    fp16 [N, D] or uint8 [N, D/8]) and per-row scale/offset (asynchronous)."""
    N, D = x.shape
    st = load().lam_encode_rows(_ptr(x), int(N), int(D), int(fmt), _ptr(codes), _ptr(scale),
                                _ptr(offset), _stream(stream, x.device))
    _check(st, "lam_encode_rows")


def lam_decode_rows(codes, fmt, N, D, scale, offset, out, stream=None):
    """xhat [N, D] fp32 of per-vector codes (asynchronous)."""
    st = load().lam_decode_rows(_ptr(codes), int(fmt), int(N), int(D), _ptr(scale),
                                _ptr(offset), _ptr(out), _stream(stream, out.device))
    _check(st, "lam_decode_rows")


def lam_score_topk_rows_workspace_size(B, N, D, k, fmt) -> int:
    return int(load().lam_score_topk_rows_workspace_size(int(B), int(N), int(D), int(k),
                                                         int(fmt)))


def lam_score_topk_rows_path(B, N, D, k, fmt) -> int:
    return int(load().lam_score_topk_rows_path(int(B), int(N), int(D), int(k), int(fmt)))


def lam_score_topk_rows(queries, codes, fmt, scale, offset, N, D, k, metric, scores, ids,
                        workspace, stream=None):
    """Exact search over per-vector coded rows; writes scores/ids [B, k]."""
    B = queries.shape[0]
    st = load().lam_score_topk_rows(_ptr(queries), int(B), _ptr(codes), int(fmt), _ptr(scale),
                                    _ptr(offset), int(N), int(D), int(k), int(metric),
                                    _ptr(scores), _ptr(ids), _ptr(workspace), _nbytes(workspace),
                                    _stream(stream, queries.device))
    _check(st, "lam_score_topk_rows")


def lam_score_topk_status(workspace, stream=None) -> int:
    out = ctypes.c_int32(0)
    st = load().lam_score_topk_status(_ptr(workspace), _stream(stream, workspace.device),
                                      ctypes.byref(out))
    _check(st, "lam_score_topk_status")
    return out.value


def lam_score_topk_noalloc(queries, codes, width, N, D, eps, code_bound, k, metric, scores, ids,
                           stream=None):
    """lam_score_topk for callers that cannot allocate: scratch lives in a fixed
    16 MiB device array inside the library (synchronous; see include/lam.h)."""
    import torch
    B = queries.shape[0]
    with torch.cuda.device(queries.device):  # the scratch is the current device's
        st = load().lam_score_topk_noalloc(_ptr(queries), int(B), _ptr(codes), int(width),
                                           int(N), int(D), ctypes.c_float(eps), int(code_bound),
                                           int(k), int(metric), _ptr(scores), _ptr(ids),
                                           _stream(stream, queries.device))
    _check(st, "lam_score_topk_noalloc")


def lam_quantize_bands(x, eps, width_req, r, codes, digests, workspace, stream=None,
                       raise_on_error=True):
    """Q_eps of the fp32 rows x [N, D] fused with the FNV-1a digest of every
    r-coordinate band; digests is a [N, D // r] int64/uint64 CUDA tensor.
    Returns (status, width, scale, code_min, code_max)."""
    N, D = x.shape
    w, sc, cmin, cmax = ctypes.c_int32(0), ctypes.c_float(0), ctypes.c_int32(0), ctypes.c_int32(0)
    st = load().lam_quantize_bands(_ptr(x), int(N), int(D), ctypes.c_float(eps), int(width_req),
                                   int(r), _ptr(codes), _nbytes(codes), _ptr(digests),
                                   _ptr(workspace), _nbytes(workspace), ctypes.byref(w),
                                   ctypes.byref(sc), ctypes.byref(cmin), ctypes.byref(cmax),
                                   _stream(stream, x.device))
    if raise_on_error:
        _check(st, "lam_quantize_bands")
    return st, w.value, sc.value, cmin.value, cmax.value


def lam_admit_batch_workspace_size(N, nb, max_pairs) -> int:
    return int(load().lam_admit_batch_workspace_size(int(N), int(nb), int(max_pairs)))


def lam_admit_batch(e, digests, delta, rep, dist, workspace, max_pairs, stream=None,
                    raise_on_error=True):
    """Batch admission of the fp32 rows e [N, D] over their band digests
    [N, nb]; fills rep (int32 [N]) and dist (float64 [N]).  Returns
    (status, delta_hat, n_retained, n_pairs)."""
    N, D = e.shape
    nb = digests.shape[1]
    dh, kept, np_ = ctypes.c_double(0), ctypes.c_int64(0), ctypes.c_int64(0)
    st = load().lam_admit_batch(_ptr(e), int(N), int(D), _ptr(digests), int(nb),
                                ctypes.c_double(delta), _ptr(rep), _ptr(dist), _ptr(workspace),
                                _nbytes(workspace), int(max_pairs), ctypes.byref(dh),
                                ctypes.byref(kept), ctypes.byref(np_), _stream(stream, e.device))
    if raise_on_error:
        _check(st, "lam_admit_batch")
    return st, dh.value, kept.value, np_.value


def lam_lamz_bound(n) -> int:
    return int(load().lam_lamz_bound(int(n)))


def lam_lamz_workspace_size(n) -> int:
    return int(load().lam_lamz_workspace_size(int(n)))


def lam_lamz_compress(x, rel, out, workspace, stream=None, raise_on_error=True):
    """Error-bounded compression of the fp32 CUDA tensor x into the uint8 CUDA
    tensor out; returns (status, stream bytes)."""
    nb = ctypes.c_size_t(0)
    st = load().lam_lamz_compress(_ptr(x), int(x.numel()), ctypes.c_float(rel), _ptr(out),
                                  _nbytes(out), ctypes.byref(nb), _ptr(workspace),
                                  _nbytes(workspace), _stream(stream, x.device))
    if raise_on_error:
        _check(st, "lam_lamz_compress")
    return st, nb.value


def lam_lamz_decompress(stream_bytes, nbytes, out, workspace, stream=None, raise_on_error=True):
    """Decodes the first nbytes of the uint8 CUDA tensor into out (fp32)."""
    st = load().lam_lamz_decompress(_ptr(stream_bytes), int(nbytes), _ptr(out), int(out.numel()),
                                    _ptr(workspace), _nbytes(workspace),
                                    _stream(stream, out.device))
    if raise_on_error:
        _check(st, "lam_lamz_decompress")
    return st


def lam_code_sqnorms(codes, width, N, D, sqnorm_out, stream=None) -> None:
    """sqnorm_out[i] = fl32(exact sum of squares of code row i)."""
    st = load().lam_code_sqnorms(_ptr(codes), int(width), int(N), int(D), _ptr(sqnorm_out),
                                 _stream(stream, codes.device))
    _check(st, "lam_code_sqnorms")


LAM_TIME_QUANTIZE, LAM_TIME_DEQUANTIZE, LAM_TIME_SCORE, LAM_TIME_AUX, LAM_TIME_MERGE = 1, 2, 4, 8, 16


def lam_timing_begin(mask, capacity) -> None:
    """Bracket launches of the kernel kinds in `mask` with CUDA events (at most
    `capacity` launches) and count all launches by kind."""
    _check(load().lam_timing_begin(int(mask), int(capacity)), "lam_timing_begin")


def lam_timing_read(kind):
    """(summed device ms of the bracketed launches, bracketed count, launch count)."""
    tot, timed, launches = ctypes.c_double(0), ctypes.c_int64(0), ctypes.c_int64(0)
    _check(load().lam_timing_read(int(kind), ctypes.byref(tot), ctypes.byref(timed),
                                  ctypes.byref(launches)), "lam_timing_read")
    return tot.value, timed.value, launches.value


def lam_timing_end() -> None:
    _check(load().lam_timing_end(), "lam_timing_end")
