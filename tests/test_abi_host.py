"""The C ABI library builds, loads, exports every declared symbol, and rejects
bad arguments on the host before touching a GPU."""
import ctypes
import os
import re

import pytest

from tests.conftest import ROOT


@pytest.fixture(scope="module")
def lib():
    from paper_2609_32256_gb300 import build as lam_build
    lam_build.build()
    import paper_2609_32256_gb300 as lam
    return lam.load()


def declared_symbols():
    text = open(os.path.join(ROOT, "include", "lam.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(lam_[a-z0-9_]+)\s*\(", text)))


def test_every_declared_symbol_is_exported(lib):
    names = declared_symbols()
    assert len(names) >= 9
    for name in names:
        assert hasattr(lib, name), name


def test_no_extra_exported_entry_points(lib):
    # everything named lam_* in the dynamic symbol table is declared in lam.h
    import subprocess
    out = subprocess.run(["nm", "-D", "--defined-only", lib._name], capture_output=True,
                         text=True).stdout
    exported = {l.split()[-1] for l in out.splitlines() if " T " in l and "lam_" in l}
    assert exported and exported <= set(declared_symbols())


def test_status_strings(lib):
    import paper_2609_32256_gb300 as lam
    assert lam.lam_status_string(0) == "ok"
    assert "invalid" in lam.lam_status_string(1)
    assert lam.lam_version() >= 100
    assert lam.lam_quantize_workspace_size() == 32


@pytest.mark.parametrize("n,eps,width", [
    (-1, 1e-3, 0), (10, 0.0, 0), (10, -1e-3, 0), (10, float("nan"), 0), (10, float("inf"), 0),
    (10, 1e-39, 0), (10, 1e-3, 3), (10, 1e-3, 8)])
def test_quantize_rejects_bad_arguments(lib, n, eps, width):
    c = ctypes
    st = lib.lam_quantize(c.c_void_p(16), n, c.c_float(eps), width, None, 0, c.c_void_p(256), 16,
                          None, None, None, None, None)
    assert st == 1


def test_quantize_null_input_rejected(lib):
    c = ctypes
    assert lib.lam_quantize(None, 5, c.c_float(1e-3), 0, None, 0, c.c_void_p(256), 16, None,
                            None, None, None, None) == 1


def test_quantize_empty_needs_no_device(lib):
    c = ctypes
    w, s, lo, hi = c.c_int32(), c.c_float(), c.c_int32(7), c.c_int32(7)
    st = lib.lam_quantize(None, 0, c.c_float(1e-3), 0, None, 0, None, 0, c.byref(w), c.byref(s),
                          c.byref(lo), c.byref(hi), None)
    assert st == 0 and w.value == 1 and s.value == c.c_float(2e-3).value
    assert (lo.value, hi.value) == (0, 0)


def test_quantize_forced_width_small_buffer(lib):
    c = ctypes
    st = lib.lam_quantize(c.c_void_p(256), 100, c.c_float(1e-3), 2, c.c_void_p(512), 199,
                          c.c_void_p(1024), 16, None, None, None, None, None)
    assert st == 4


@pytest.mark.parametrize("args", [
    dict(B=0), dict(N=0), dict(D=0), dict(k=0), dict(k=1025), dict(k=11, N=10), dict(width=3),
    dict(metric=3), dict(eps=0.0), dict(code_bound=-1)])
def test_score_rejects_bad_arguments(lib, args):
    c = ctypes
    p = dict(B=2, N=10, D=8, k=3, width=1, metric=0, eps=1e-3, code_bound=0)
    p.update(args)
    st = lib.lam_score_topk(c.c_void_p(256), p["B"], c.c_void_p(512), p["width"], p["N"], p["D"],
                            c.c_float(p["eps"]), p["code_bound"], p["k"], p["metric"],
                            c.c_void_p(768), c.c_void_p(1024), c.c_void_p(4096), 1 << 20, None)
    assert st == 1


def test_score_rejects_null_and_misaligned_workspace(lib):
    c = ctypes
    base = (c.c_void_p(256), 2, c.c_void_p(512), 1, 10, 8, c.c_float(1e-3), 0, 3, 0,
            c.c_void_p(768), c.c_void_p(1024))
    assert lib.lam_score_topk(*base, None, 1 << 20, None) == 1
    assert lib.lam_score_topk(*base, c.c_void_p(4096 + 8), 1 << 20, None) == 1


def test_dequantize_rejects_bad_arguments(lib):
    c = ctypes
    assert lib.lam_dequantize(None, 1, 10, c.c_float(1.0), c.c_void_p(256), None) == 1
    assert lib.lam_dequantize(c.c_void_p(256), 3, 10, c.c_float(1.0), c.c_void_p(256), None) == 1
    assert lib.lam_dequantize(c.c_void_p(256), 1, -1, c.c_float(1.0), c.c_void_p(256), None) == 1
    assert lib.lam_dequantize(None, 1, 0, c.c_float(1.0), None, None) == 0


def test_misaligned_buffers_rejected(lib):
    c = ctypes
    ws = c.c_void_p(4096)
    # fp32 input not 4-byte aligned
    assert lib.lam_quantize(c.c_void_p(258), 10, c.c_float(1e-3), 2, c.c_void_p(512), 20, ws, 16,
                            None, None, None, None, None) == 1
    # int16 codes at an odd address; AUTO codes not 4-byte aligned
    assert lib.lam_quantize(c.c_void_p(256), 10, c.c_float(1e-3), 2, c.c_void_p(513), 20, ws, 16,
                            None, None, None, None, None) == 1
    assert lib.lam_quantize(c.c_void_p(256), 10, c.c_float(1e-3), 0, c.c_void_p(514), 40, ws, 16,
                            None, None, None, None, None) == 1
    assert lib.lam_dequantize(c.c_void_p(513), 2, 10, c.c_float(1.0), c.c_void_p(256), None) == 1
    assert lib.lam_dequantize(c.c_void_p(512), 2, 10, c.c_float(1.0), c.c_void_p(258), None) == 1
    base = (c.c_void_p(256), 2, c.c_void_p(513), 2, 10, 8, c.c_float(1e-3), 0, 3, 0,
            c.c_void_p(768), c.c_void_p(1024), c.c_void_p(4096), 1 << 20, None)
    assert lib.lam_score_topk(*base) == 1


@pytest.mark.parametrize("mask,cap", [(0, 10), (32, 10), (-1, 10), (1, -1), (1, (1 << 20) + 1)])
def test_timing_rejects_bad_arguments(lib, mask, cap):
    assert lib.lam_timing_begin(mask, cap) == 1


def test_timing_read_rejects_bad_kind_and_end_is_idempotent(lib):
    import paper_2609_32256_gb300 as lam
    for kind in (0, 3, 32):
        assert lib.lam_timing_read(kind, None, None, None) == 1
    assert lib.lam_timing_begin(lam.LAM_TIME_SCORE, 0) == 0  # no events to create
    tot, timed, launches = lam.lam_timing_read(lam.LAM_TIME_SCORE)
    assert (tot, timed, launches) == (0.0, 0, 0)
    assert lib.lam_timing_end() == 0
    assert lib.lam_timing_end() == 0


@pytest.mark.parametrize("width,N,D,codes,out", [(4, 10, 8, 256, 512), (3, 10, 8, 256, 512),
                                                 (1, -1, 8, 256, 512), (1, 10, 0, 256, 512),
                                                 (2, 10, 8, 257, 512), (1, 10, 8, 256, 514),
                                                 (1, 10, 8, 0, 512)])
def test_code_sqnorms_rejects_bad_arguments(lib, width, N, D, codes, out):
    c = ctypes
    assert lib.lam_code_sqnorms(c.c_void_p(codes), width, N, D, c.c_void_p(out), None) == 1


@pytest.mark.parametrize("N,D,r,width,x,dig", [(4, 8, 3, 0, 256, 512), (4, 8, 0, 0, 256, 512),
                                              (4, 8, 16, 0, 256, 512), (-1, 8, 2, 0, 256, 512),
                                              (4, 8, 2, 3, 256, 512), (4, 8, 2, 0, 258, 512),
                                              (4, 8, 2, 0, 256, 516), (4, 8, 2, 0, 0, 512),
                                              (4, 8, 2, 0, 256, 0)])
def test_quantize_bands_rejects_bad_arguments(lib, N, D, r, width, x, dig):
    c = ctypes
    st = lib.lam_quantize_bands(c.c_void_p(x), N, D, c.c_float(1e-3), width, r, None, 0,
                                c.c_void_p(dig), c.c_void_p(1024), 64, None, None, None, None,
                                None)
    assert st == 1


@pytest.mark.parametrize("n,rel", [(-1, 0.01), (10, 0.0), (10, 1e-7), (10, 2.0),
                                   (10, float("nan"))])
def test_lamz_compress_rejects_bad_arguments(lib, n, rel):
    c = ctypes
    nb = c.c_size_t(0)
    st = lib.lam_lamz_compress(c.c_void_p(256), n, c.c_float(rel), c.c_void_p(512), 1 << 20,
                               c.byref(nb), c.c_void_p(1024), 1 << 20, None)
    assert st == 1


def test_lamz_sizes(lib):
    import paper_2609_32256_gb300 as lam
    assert lam.lam_lamz_bound(0) == 16
    assert lam.lam_lamz_bound(33) == 16 + 4 + 2 * (4 + 4 * 31)
    assert lam.lam_lamz_workspace_size(1 << 20) > 0


# fmt, N, D, codes, scale, offset: each case is invalid before any device work
ROWS_BAD = [(0, 4, 16, 256, 512, 768), (4, 4, 16, 256, 512, 768), (3, 4, 12, 256, 512, 768),
            (1, -1, 16, 256, 512, 768), (1, 4, 0, 256, 512, 768), (1, 4, 16, None, 512, 768),
            (1, 4, 16, 256, None, 768), (1, 4, 16, 256, 512, None), (3, 4, 16, 256, None, None),
            (2, 4, 16, 257, None, None), (1, 4, 16, 256, 514, 768)]


@pytest.mark.parametrize("fmt,N,D,codes,scale,offset", ROWS_BAD)
def test_row_codecs_reject_bad_arguments(lib, fmt, N, D, codes, scale, offset):
    c = ctypes
    p = lambda v: None if v is None else c.c_void_p(v)
    assert lib.lam_encode_rows(c.c_void_p(1024), N, D, fmt, p(codes), p(scale), p(offset),
                               None) == 1
    assert lib.lam_decode_rows(p(codes), fmt, N, D, p(scale), p(offset), c.c_void_p(1024),
                               None) == 1


def test_row_codecs_empty_needs_no_device(lib):
    c = ctypes
    assert lib.lam_encode_rows(None, 0, 16, 1, None, None, None, None) == 0
    assert lib.lam_decode_rows(None, 2, 0, 16, None, None, None, None) == 0


def test_score_rows_rejects_bad_arguments(lib):
    c = ctypes
    v = c.c_void_p
    ok = dict(q=v(1024), B=4, codes=v(4096), fmt=1, scale=v(512), offset=v(768), N=100, D=32,
              k=10, metric=0, scores=v(8192), ids=v(16384), ws=v(1 << 20), wsb=1 << 30)

    def call(**kw):
        a = dict(ok, **kw)
        return lib.lam_score_topk_rows(a["q"], a["B"], a["codes"], a["fmt"], a["scale"],
                                       a["offset"], a["N"], a["D"], a["k"], a["metric"],
                                       a["scores"], a["ids"], a["ws"], a["wsb"], None)
    for bad in (dict(fmt=5), dict(fmt=3, D=20), dict(k=0), dict(k=101), dict(metric=3),
                dict(scale=None), dict(offset=None), dict(q=None), dict(ws=v(1 << 20 | 8)),
                dict(scale=v(514)), dict(B=0), dict(ids=v(16388))):
        assert call(**bad) == 1, bad
    assert lib.lam_score_topk_rows_workspace_size(4, 100, 32, 10, 9) == 0
    assert lib.lam_score_topk_rows_path(4, 100, 20, 10, 3) == -1


def test_async_calls_reject_bad_arguments(lib):
    c = ctypes
    v = c.c_void_p
    # quantize: bad eps, bad width, null workspace, misaligned workspace
    assert lib.lam_quantize_async(v(1024), 16, c.c_float(0.0), 0, v(2048), 64, v(4096), 256,
                                  None) == 1
    assert lib.lam_quantize_async(v(1024), 16, c.c_float(1e-2), 3, v(2048), 64, v(4096), 256,
                                  None) == 1
    assert lib.lam_quantize_async(v(1024), 16, c.c_float(1e-2), 0, v(2048), 64, None, 256,
                                  None) == 1
    assert lib.lam_quantize_async(v(1024), 16, c.c_float(1e-2), 0, v(2048), 64, v(4104), 256,
                                  None) == 1
    # result: null workspace
    w = c.c_int32()
    assert lib.lam_quantize_result(None, c.c_float(1e-2), 0, None, c.byref(w), None, None,
                                   None) == 1
    # dequantize_from: misaligned status, null codes
    assert lib.lam_dequantize_from(v(1024), v(4104), 16, c.c_float(1e-2), v(2048), None) == 1
    assert lib.lam_dequantize_from(None, v(4096), 16, c.c_float(1e-2), v(2048), None) == 1
    # score_from: bad metric, null status, k > N
    assert lib.lam_score_topk_from(v(1024), 2, v(4096), v(8192), 100, 64, c.c_float(1e-2), 10, 5,
                                   v(16384), v(32768), v(1 << 20), 1 << 30, None) == 1
    assert lib.lam_score_topk_from(v(1024), 2, v(4096), None, 100, 64, c.c_float(1e-2), 10, 0,
                                   v(16384), v(32768), v(1 << 20), 1 << 30, None) == 1
    assert lib.lam_score_topk_from(v(1024), 2, v(4096), v(8192), 5, 64, c.c_float(1e-2), 10, 0,
                                   v(16384), v(32768), v(1 << 20), 1 << 30, None) == 1
