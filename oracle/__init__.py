"""CPU oracle for LAM's quantized-memory hot path (test infrastructure only).

The oracle is plain C (``lam_oracle.c``), compiled with ``-O2 -ffp-contract=off
-fno-fast-math`` so that no multiply-add is fused on either x86-64 or aarch64.
Only the test suite, the smoke check and the benchmark's CPU-baseline leg may
load it; the product library never does, and the two share no code.

What it follows (paper: "LAM: Lossy Agent Memory"):
  * quantize   -- Sec. 3.2, layer L1: Q_eps(x) = round(x / 2 eps);
  * dequantize -- xhat = 2 eps * Q_eps(x), the reading under which one cell has
                  half-width eps (Sec. 3.1, App. "Rank invariance, in full");
  * scores     -- exact search is a matrix-vector product over the stored
                  vectors (Sec. "Brute-force scan crossover"); metrics inner
                  product, cosine and squared L2 (Eq. 1 ties L2 to cosine);
  * top-k      -- full sort, best first, equal scores by lower id (the
                  lowest-index rule of Algorithm 1).
  * encode_rows / decode_rows / scores_rows -- the per-vector byte codecs
                  of the composite experiment (Sec. "Composite reduction",
                  Table "composite": fp16, per-vector int8 with a scale and an
                  offset per row, sign bits with one scale per row) and the
                  exact scores of their decoded fp32 rows.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "lam_oracle.c")
_LIB = os.path.join(_HERE, "liblam_oracle.so")

IP, COSINE, L2 = 0, 1, 2
CFLAGS = ["-O2", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared",
          "-std=c11", "-pthread"]


def build(force: bool = False) -> str:
    """Compile lam_oracle.c into liblam_oracle.so beside it (gcc)."""
    if (not force and os.path.exists(_LIB)
            and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC)):
        return _LIB
    tmp = _LIB + ".tmp%d" % os.getpid()
    subprocess.run(["gcc", *CFLAGS, "-o", tmp, _SRC, "-lm"], check=True)
    os.replace(tmp, _LIB)
    return _LIB


_lib = None


def _load():
    global _lib
    if _lib is None:
        build()
        lib = ctypes.CDLL(_LIB)
        f32p = ctypes.POINTER(ctypes.c_float)
        i32p = ctypes.POINTER(ctypes.c_int32)
        i64p = ctypes.POINTER(ctypes.c_int64)
        f64p = ctypes.POINTER(ctypes.c_double)
        lib.lam_oracle_step.argtypes = [ctypes.c_float]
        lib.lam_oracle_step.restype = ctypes.c_float
        lib.lam_oracle_quantize.argtypes = [f32p, ctypes.c_int64, ctypes.c_float,
                                            i32p, f64p, f64p, i64p]
        lib.lam_oracle_quantize.restype = None
        lib.lam_oracle_width.argtypes = [ctypes.c_double, ctypes.c_double]
        lib.lam_oracle_width.restype = ctypes.c_int32
        lib.lam_oracle_dequantize.argtypes = [i32p, ctypes.c_int64, ctypes.c_float,
                                              f32p]
        lib.lam_oracle_dequantize.restype = None
        u8p = ctypes.POINTER(ctypes.c_uint8)
        u64p = ctypes.POINTER(ctypes.c_uint64)
        lib.lam_oracle_fnv1a64.argtypes = [u8p, ctypes.c_int64, ctypes.c_uint64]
        lib.lam_oracle_fnv1a64.restype = ctypes.c_uint64
        lib.lam_oracle_band_digests.argtypes = [i32p, ctypes.c_int64, ctypes.c_int32,
                                                ctypes.c_int32, ctypes.c_int32, u64p]
        lib.lam_oracle_band_digests.restype = None
        lib.lam_oracle_admit_batch.argtypes = [f32p, ctypes.c_int64, ctypes.c_int32, u64p,
                                               ctypes.c_int32, ctypes.c_double, i32p,
                                               ctypes.POINTER(ctypes.c_double),
                                               ctypes.POINTER(ctypes.c_double)]
        lib.lam_oracle_admit_batch.restype = ctypes.c_int64
        lib.lam_oracle_lamz_compress.argtypes = [f32p, ctypes.c_int64, ctypes.c_float, u8p,
                                                 ctypes.c_int64]
        lib.lam_oracle_lamz_compress.restype = ctypes.c_int64
        lib.lam_oracle_lamz_decompress.argtypes = [u8p, ctypes.c_int64, f32p, ctypes.c_int64]
        lib.lam_oracle_lamz_decompress.restype = ctypes.c_int32
        i8p = ctypes.POINTER(ctypes.c_int8)
        lib.lam_oracle_encode_int8_rows.argtypes = [f32p, ctypes.c_int64, ctypes.c_int32, i8p,
                                                    f32p, f32p]
        lib.lam_oracle_encode_int8_rows.restype = None
        lib.lam_oracle_encode_sign_rows.argtypes = [f32p, ctypes.c_int64, ctypes.c_int32, u8p,
                                                    f32p]
        lib.lam_oracle_encode_sign_rows.restype = None
        lib.lam_oracle_decode_rows.argtypes = [ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64,
                                               ctypes.c_int32, f32p, f32p, f32p]
        lib.lam_oracle_decode_rows.restype = None
        lib.lam_oracle_scores_rows.argtypes = [f32p, ctypes.c_int64, f32p, ctypes.c_int64,
                                               ctypes.c_int32, ctypes.c_int32, f32p]
        lib.lam_oracle_scores_rows.restype = None
        lib.lam_oracle_code_sqnorms.argtypes = [i32p, ctypes.c_int64, ctypes.c_int32, f32p]
        lib.lam_oracle_code_sqnorms.restype = None
        lib.lam_oracle_scores.argtypes = [f32p, ctypes.c_int64, i32p, ctypes.c_int64,
                                          ctypes.c_int32, ctypes.c_float,
                                          ctypes.c_int32, f32p]
        lib.lam_oracle_scores.restype = None
        lib.lam_oracle_topk.argtypes = [f32p, ctypes.c_int64, ctypes.c_int64,
                                        ctypes.c_int32, ctypes.c_int32, f32p, i64p]
        lib.lam_oracle_topk.restype = ctypes.c_int
        lib.lam_oracle_search.argtypes = [f32p, ctypes.c_int64, i32p,
                                          ctypes.c_int64, ctypes.c_int32,
                                          ctypes.c_float, ctypes.c_int32,
                                          ctypes.c_int32, f32p, i64p,
                                          ctypes.c_int32]
        lib.lam_oracle_search.restype = ctypes.c_int
        _lib = lib
    return _lib


def _ptr(a: np.ndarray, ctype):
    return a.ctypes.data_as(ctypes.POINTER(ctype))


def step(eps: float) -> np.float32:
    """s = fl32(2 eps), the quantizer step."""
    return np.float32(_load().lam_oracle_step(ctypes.c_float(np.float32(eps))))


def quantize(x: np.ndarray, eps: float):
    """Q_eps over a flat fp32 array.

    Returns ``(codes int32, rmin, rmax, n_nonfinite)``; rmin/rmax are the
    smallest/largest rounded quotient over the finite inputs (exact, as float).
    Codes of values outside int32 or non-finite inputs are 0.
    """
    x = np.ascontiguousarray(x, dtype=np.float32).reshape(-1)
    codes = np.empty(x.size, dtype=np.int32)
    rmin = ctypes.c_double()
    rmax = ctypes.c_double()
    nnf = ctypes.c_int64()
    _load().lam_oracle_quantize(_ptr(x, ctypes.c_float), x.size,
                                ctypes.c_float(np.float32(eps)),
                                _ptr(codes, ctypes.c_int32), ctypes.byref(rmin),
                                ctypes.byref(rmax), ctypes.byref(nnf))
    return codes, rmin.value, rmax.value, nnf.value


def width(rmin: float, rmax: float) -> int:
    """Narrowest width in bytes (1, 2, 4) holding [rmin, rmax]; 0 if none."""
    return int(_load().lam_oracle_width(rmin, rmax))


def dequantize(codes: np.ndarray, scale: float) -> np.ndarray:
    """xhat = fl32(scale * code)."""
    c = np.ascontiguousarray(codes, dtype=np.int32).reshape(-1)
    out = np.empty(c.size, dtype=np.float32)
    _load().lam_oracle_dequantize(_ptr(c, ctypes.c_int32), c.size,
                                  ctypes.c_float(np.float32(scale)),
                                  _ptr(out, ctypes.c_float))
    return out.reshape(np.shape(codes))


FNV_OFFSET = 14695981039346656037


def fnv1a64(data: bytes, h: int = FNV_OFFSET) -> int:
    """64-bit FNV-1a of a byte string, continuing from state h."""
    buf = np.frombuffer(bytes(data), dtype=np.uint8).copy()
    return int(_load().lam_oracle_fnv1a64(_ptr(buf, ctypes.c_uint8), buf.size, h))


def band_digests(codes: np.ndarray, r: int, width: int) -> np.ndarray:
    """Digest of every r-coordinate band of every code row [N, D] -> uint64 [N, D // r]."""
    c = np.ascontiguousarray(codes, dtype=np.int32)
    N, D = c.shape
    assert D % r == 0
    out = np.empty((N, D // r), dtype=np.uint64)
    _load().lam_oracle_band_digests(_ptr(c, ctypes.c_int32), N, D, r, width,
                                    _ptr(out, ctypes.c_uint64))
    return out


def admit_batch(e: np.ndarray, digests: np.ndarray, delta: float):
    """Batch admission (Algorithm 2) of the fp32 rows e [N, D] with band
    digests [N, nb]: (rep int32 [N], dist float64 [N], delta_hat, n_retained)."""
    x = np.ascontiguousarray(e, dtype=np.float32)
    dg = np.ascontiguousarray(digests, dtype=np.uint64)
    N, D = x.shape
    nb = dg.shape[1]
    rep = np.empty(N, dtype=np.int32)
    dist = np.empty(N, dtype=np.float64)
    dh = ctypes.c_double(0.0)
    kept = _load().lam_oracle_admit_batch(_ptr(x, ctypes.c_float), N, D,
                                          _ptr(dg, ctypes.c_uint64), nb, float(delta),
                                          _ptr(rep, ctypes.c_int32),
                                          _ptr(dist, ctypes.c_double), ctypes.byref(dh))
    return rep, dist, dh.value, int(kept)


def lamz_compress(x: np.ndarray, rel: float) -> bytes:
    """Error-bounded byte codec (bound rel * max|x|): the compressed bytes."""
    v = np.ascontiguousarray(x, dtype=np.float32).reshape(-1)
    lib = _load()
    size = lib.lam_oracle_lamz_compress(_ptr(v, ctypes.c_float), v.size,
                                        ctypes.c_float(np.float32(rel)), None, 0)
    if size < 0:
        raise ValueError("non-finite input")
    out = np.empty(size, dtype=np.uint8)
    lib.lam_oracle_lamz_compress(_ptr(v, ctypes.c_float), v.size, ctypes.c_float(np.float32(rel)),
                                 _ptr(out, ctypes.c_uint8), size)
    return out.tobytes()


def lamz_decompress(data: bytes, n: int) -> np.ndarray:
    buf = np.frombuffer(data, dtype=np.uint8).copy()
    out = np.empty(n, dtype=np.float32)
    st = _load().lam_oracle_lamz_decompress(_ptr(buf, ctypes.c_uint8), buf.size,
                                            _ptr(out, ctypes.c_float), n)
    if st != 0:
        raise ValueError("malformed stream")
    return out


FMT_INT8_ROWS, FMT_FP16, FMT_SIGN = 1, 2, 3


def encode_rows(x: np.ndarray, fmt: int):
    """Alternative codec of rows [N, D]: (codes, scale, offset) with codes int8
    [N, D] (fmt 1), fp16 [N, D] (fmt 2) or packed sign bits uint8 [N, D/8]
    (fmt 3); scale/offset float32 [N] (offset None unless fmt 1)."""
    v = np.ascontiguousarray(x, dtype=np.float32)
    N, D = v.shape
    if fmt == FMT_FP16:
        return v.astype(np.float16), None, None
    if fmt == FMT_INT8_ROWS:
        c = np.empty((N, D), np.int8)
        sc = np.empty(N, np.float32)
        of = np.empty(N, np.float32)
        _load().lam_oracle_encode_int8_rows(_ptr(v, ctypes.c_float), N, D,
                                            _ptr(c, ctypes.c_int8), _ptr(sc, ctypes.c_float),
                                            _ptr(of, ctypes.c_float))
        return c, sc, of
    assert D % 8 == 0
    bits = np.empty((N, D // 8), np.uint8)
    al = np.empty(N, np.float32)
    _load().lam_oracle_encode_sign_rows(_ptr(v, ctypes.c_float), N, D,
                                        _ptr(bits, ctypes.c_uint8), _ptr(al, ctypes.c_float))
    return bits, al, None


def decode_rows(codes: np.ndarray, fmt: int, D: int, scale=None, offset=None) -> np.ndarray:
    c = np.ascontiguousarray(codes)
    N = c.shape[0]
    out = np.empty((N, D), np.float32)
    sc = np.ascontiguousarray(scale if scale is not None else np.zeros(N), dtype=np.float32)
    of = np.ascontiguousarray(offset if offset is not None else np.zeros(N), dtype=np.float32)
    _load().lam_oracle_decode_rows(c.ctypes.data_as(ctypes.c_void_p), fmt, N, D,
                                   _ptr(sc, ctypes.c_float), _ptr(of, ctypes.c_float),
                                   _ptr(out, ctypes.c_float))
    return out


def scores_rows(queries: np.ndarray, rows: np.ndarray, metric: int) -> np.ndarray:
    """Scores [B, N] of queries [B, D] against decoded fp32 rows [N, D]."""
    q = np.ascontiguousarray(queries, dtype=np.float32)
    r = np.ascontiguousarray(rows, dtype=np.float32)
    B, D = q.shape
    N = r.shape[0]
    out = np.empty((B, N), np.float32)
    _load().lam_oracle_scores_rows(_ptr(q, ctypes.c_float), B, _ptr(r, ctypes.c_float), N, D,
                                   metric, _ptr(out, ctypes.c_float))
    return out


def code_sqnorms(codes: np.ndarray) -> np.ndarray:
    """fl32 of the exact sum of squares of each code row [N, D] -> [N]."""
    c = np.ascontiguousarray(codes, dtype=np.int32)
    N, D = c.shape
    out = np.empty(N, dtype=np.float32)
    _load().lam_oracle_code_sqnorms(_ptr(c, ctypes.c_int32), N, D, _ptr(out, ctypes.c_float))
    return out


def scores(queries: np.ndarray, codes: np.ndarray, eps: float, metric: int):
    """All scores [B, N] of queries [B, D] against code rows [N, D]."""
    q = np.ascontiguousarray(queries, dtype=np.float32)
    c = np.ascontiguousarray(codes, dtype=np.int32)
    B, D = q.shape
    N = c.shape[0]
    assert c.shape[1] == D
    out = np.empty((B, N), dtype=np.float32)
    _load().lam_oracle_scores(_ptr(q, ctypes.c_float), B, _ptr(c, ctypes.c_int32),
                              N, D, ctypes.c_float(np.float32(eps)), metric,
                              _ptr(out, ctypes.c_float))
    return out


def topk(score_matrix: np.ndarray, k: int, metric: int):
    """Top-k per row of a score matrix: (scores [B, k] f32, ids [B, k] i64)."""
    s = np.ascontiguousarray(score_matrix, dtype=np.float32)
    B, N = s.shape
    os_ = np.empty((B, k), dtype=np.float32)
    oi = np.empty((B, k), dtype=np.int64)
    rc = _load().lam_oracle_topk(_ptr(s, ctypes.c_float), B, N, k, metric,
                                 _ptr(os_, ctypes.c_float), _ptr(oi, ctypes.c_int64))
    if rc:
        raise ValueError("oracle topk failed (%d)" % rc)
    return os_, oi


def search(queries: np.ndarray, codes: np.ndarray, eps: float, metric: int,
           k: int, nthreads: int = 1):
    """Exact search: scores of every row, then top-k per query."""
    q = np.ascontiguousarray(queries, dtype=np.float32)
    c = np.ascontiguousarray(codes, dtype=np.int32)
    B, D = q.shape
    N = c.shape[0]
    assert c.shape[1] == D
    os_ = np.empty((B, k), dtype=np.float32)
    oi = np.empty((B, k), dtype=np.int64)
    rc = _load().lam_oracle_search(_ptr(q, ctypes.c_float), B,
                                   _ptr(c, ctypes.c_int32), N, D,
                                   ctypes.c_float(np.float32(eps)), metric, k,
                                   _ptr(os_, ctypes.c_float),
                                   _ptr(oi, ctypes.c_int64), nthreads)
    if rc:
        raise ValueError("oracle search failed (%d)" % rc)
    return os_, oi
