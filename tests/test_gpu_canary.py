"""Out-of-bounds writes, checked without a sanitizer: every caller-owned
buffer a call writes (codes, outputs, digests, lists and the workspaces the
library sized itself) is an exact-size view between 4 KB of canary bytes on
each side, the shapes are ragged (n not a multiple of 4, 16 or 32, N not a
multiple of the 256-row tile, k with register lists and with heaps), and
after the call the canaries must be intact and the outputs equal to those of
the plain call."""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_32256_gb300 as lam
from paper_2609_32256_gb300 import _lib, inputs
from tests.parity import check_topk, oracle_topk

pytestmark = pytest.mark.gpu

PAD = 4096
FILL = 0xA5


class Guarded:
    """nbytes of device memory between PAD canary bytes on each side."""

    def __init__(self, dev, nbytes, dtype=torch.uint8):
        esize = torch.empty((), dtype=dtype).element_size()
        assert nbytes % esize == 0
        self.n = nbytes
        self.raw = torch.full((nbytes + 2 * PAD,), FILL, dtype=torch.uint8, device=dev)
        self.view = self.raw[PAD:PAD + nbytes].view(dtype)

    def shaped(self, *shape):
        return self.view.view(*shape)

    def check(self, what):
        torch.cuda.synchronize()
        r = self.raw.cpu().numpy()
        assert (r[:PAD] == FILL).all(), f"{what}: written below the buffer"
        assert (r[PAD + self.n:] == FILL).all(), f"{what}: written past the buffer"


@pytest.mark.parametrize("n", [1, 13, 1000003])
@pytest.mark.parametrize("eps,width", [(1e-2, 0), (1e-2, 1), (1e-4, 2), (1e-4, 4)])
def test_quantize_and_dequantize(dev, n, eps, width):
    x = torch.from_numpy(inputs.flat_values(n, seed=n)).to(dev)
    oc, rmin, rmax, _ = oracle.quantize(x.cpu().numpy(), eps)
    w = width or oracle.width(rmin, rmax)
    codes = Guarded(dev, n * w)
    ws = Guarded(dev, lam.lam_quantize_workspace_size())
    st, gw, scale, _, _ = lam.lam_quantize(x, eps, width, codes.view, ws.view)
    assert st == 0 and gw == w
    codes.check("codes")
    ws.check("quantize workspace")
    dt = {1: np.int8, 2: np.int16, 4: np.int32}[w]
    assert np.array_equal(codes.view.cpu().numpy().view(dt), oc.astype(dt))
    out = Guarded(dev, n * 4, torch.float32)
    lam.lam_dequantize(codes.view, w, n, scale, out.view)
    out.check("dequantize out")
    assert np.array_equal(out.view.cpu().numpy(), oracle.dequantize(oc, scale))


SEARCH_CASES = [  # (B, k, forced path or "")
    (1, 10, "bandwidth"), (2, 100, "bandwidth"), (3, 10, "tensor"), (130, 100, "tensor"),
    (520, 17, "tensor"), (520, 100, "tensor"), (5, 10, "generic"), (1, 1, ""),
]


@pytest.mark.parametrize("B,k,path", SEARCH_CASES)
@pytest.mark.parametrize("width,eps", [(1, 1e-2), (2, 1e-3)])
def test_score_topk(dev, score_path, B, k, path, width, eps):
    if path:
        score_path(path)
    N, D = 3001, 768
    x = inputs.unit_rows(N, D, seed=B + k)
    oc, rmin, rmax, _ = oracle.quantize(x, eps)
    bound = max(-int(rmin), int(rmax))
    codes = torch.from_numpy(oc.reshape(N, D).astype({1: np.int8, 2: np.int16}[width])).to(dev)
    q = torch.from_numpy(inputs.queries(B, D, seed=k)).to(dev)
    for metric in (oracle.IP, oracle.L2):
        s = Guarded(dev, B * k * 4, torch.float32)
        i = Guarded(dev, B * k * 8, torch.int64)
        ws = Guarded(dev, lam.lam_score_topk_workspace_size(B, N, D, k, width, bound))
        lam.lam_score_topk(q, codes, width, N, D, eps, bound, k, metric, s.shaped(B, k),
                           i.shaped(B, k), ws.view)
        assert lam.lam_score_topk_status(ws.view) == lam.LAM_OK
        for g, what in ((s, "scores"), (i, "ids"), (ws, "search workspace")):
            g.check(what)
        ps, pi = lam.search(q, codes, eps, k, metric, code_bound=bound)
        assert np.array_equal(s.shaped(B, k).cpu().numpy(), ps.cpu().numpy())
        assert np.array_equal(i.shaped(B, k).cpu().numpy(), pi.cpu().numpy())
    os_, oi = oracle_topk(q.cpu().numpy(), oc.reshape(N, D), eps, oracle.L2, k)
    check_topk(ps.cpu().numpy(), pi.cpu().numpy(), q.cpu().numpy(), oc.reshape(N, D), eps,
               oracle.L2, os_, oi)


@pytest.mark.parametrize("r", [1, 3, 4, 8])
def test_quantize_bands(dev, r):
    N, D = 1001, 24 * r
    x = torch.from_numpy(inputs.unit_rows(N, D, seed=r)).to(dev)
    codes = Guarded(dev, N * D)  # int8 at this eps
    dig = Guarded(dev, N * (D // r) * 8, torch.int64)
    ws = Guarded(dev, lam.lam_quantize_workspace_size())
    st, w, *_ = lam.lam_quantize_bands(x, 1e-2, 0, r, codes.view, dig.shaped(N, D // r), ws.view)
    assert st == 0 and w == 1
    for g, what in ((codes, "codes"), (dig, "digests"), (ws, "workspace")):
        g.check(what)
    oc, *_ = oracle.quantize(x.cpu().numpy(), 1e-2)
    want = oracle.band_digests(oc.reshape(N, D), r, 1)
    assert np.array_equal(dig.view.cpu().numpy().view(np.uint64), want.reshape(-1))
    assert np.array_equal(codes.view.cpu().numpy().view(np.int8), oc.astype(np.int8))


@pytest.mark.parametrize("fmt", [lam.LAM_ROWS_INT8, lam.LAM_ROWS_FP16, lam.LAM_ROWS_SIGN])
@pytest.mark.parametrize("B", [1, 3, 300])
def test_per_vector_codecs(dev, fmt, B):
    N, D, k = 3001, 768, 10
    x = torch.from_numpy(inputs.unit_rows(N, D, seed=fmt)).to(dev)
    code_bytes = {lam.LAM_ROWS_INT8: N * D, lam.LAM_ROWS_FP16: N * D * 2,
                  lam.LAM_ROWS_SIGN: N * D // 8}[fmt]
    cdt = {lam.LAM_ROWS_INT8: torch.int8, lam.LAM_ROWS_FP16: torch.float16,
           lam.LAM_ROWS_SIGN: torch.uint8}[fmt]
    codes = Guarded(dev, code_bytes, cdt)
    cshape = (N, D // 8) if fmt == lam.LAM_ROWS_SIGN else (N, D)
    scale = Guarded(dev, N * 4, torch.float32) if fmt != lam.LAM_ROWS_FP16 else None
    offset = Guarded(dev, N * 4, torch.float32) if fmt == lam.LAM_ROWS_INT8 else None
    lam.lam_encode_rows(x, fmt, codes.shaped(*cshape), scale and scale.view,
                        offset and offset.view)
    for g, what in ((codes, "codes"), (scale, "scale"), (offset, "offset")):
        if g is not None:
            g.check(what)
    out = Guarded(dev, N * D * 4, torch.float32)
    lam.lam_decode_rows(codes.shaped(*cshape), fmt, N, D, scale and scale.view,
                        offset and offset.view, out.shaped(N, D))
    out.check("decoded rows")
    q = torch.from_numpy(inputs.queries(B, D, seed=B)).to(dev)
    s = Guarded(dev, B * k * 4, torch.float32)
    i = Guarded(dev, B * k * 8, torch.int64)
    ws = Guarded(dev, lam.lam_score_topk_rows_workspace_size(B, N, D, k, fmt))
    lam.lam_score_topk_rows(q, codes.shaped(*cshape), fmt, scale and scale.view,
                            offset and offset.view, N, D, k, oracle.L2, s.shaped(B, k),
                            i.shaped(B, k), ws.view)
    assert lam.lam_score_topk_status(ws.view) == lam.LAM_OK
    for g, what in ((s, "scores"), (i, "ids"), (ws, "rows search workspace")):
        g.check(what)
    ps, pi = lam.search_rows(q, codes.shaped(*cshape), fmt, scale and scale.view,
                             offset and offset.view, k, oracle.L2, D=D)
    assert np.array_equal(i.shaped(B, k).cpu().numpy(), pi.cpu().numpy())


@pytest.mark.parametrize("n", [1, 33, 100003])
def test_byte_codec(dev, n):
    x_np = inputs.flat_values(n, seed=n)
    want = oracle.lamz_compress(x_np, 1e-2)
    x = torch.from_numpy(x_np).to(dev)
    out = Guarded(dev, (len(want) + 3) // 4 * 4)
    ws = Guarded(dev, lam.lam_lamz_workspace_size(n))
    st, nbytes = lam.lam_lamz_compress(x, 1e-2, out.view, ws.view)
    assert st == 0 and nbytes == len(want)
    out.check("stream")
    ws.check("codec workspace")
    assert out.view.cpu().numpy()[:nbytes].tobytes() == want
    if nbytes > lam.lam_lamz_bound(0) + 4:  # a stream one word too long for its buffer
        short = Guarded(dev, nbytes - 4)
        st, need = lam.lam_lamz_compress(x, 1e-2, short.view, ws.view, raise_on_error=False)
        assert st == lam.LAM_ERR_WORKSPACE and need == nbytes
        short.check("short stream buffer")
    y = Guarded(dev, n * 4, torch.float32)
    assert lam.lam_lamz_decompress(out.view, nbytes, y.view, ws.view) == 0
    y.check("decoded values")
    ws.check("codec workspace")
    np.testing.assert_array_equal(y.view.cpu().numpy(), oracle.lamz_decompress(want, n))


def test_admit_batch(dev):
    N, D, r = 2001, 768, 8
    x = torch.from_numpy(inputs.planted_rows(N, D, seed=5)).to(dev)
    nb = D // r
    dig = torch.empty((N, nb), dtype=torch.int64, device=dev)
    lam.lam_quantize_bands(x, 0.3 / D ** 0.5, 0, r, None, dig,
                           torch.empty(lam.lam_quantize_workspace_size(), dtype=torch.uint8,
                                       device=dev))
    delta = (2.0 - 2.0 * 0.95) ** 0.5
    mp = 1 << 16
    rep = Guarded(dev, N * 4, torch.int32)
    dist = Guarded(dev, N * 8, torch.float64)
    ws = Guarded(dev, lam.lam_admit_batch_workspace_size(N, nb, mp))
    st, dh, kept, npairs = lam.lam_admit_batch(x, dig, delta, rep.view, dist.view, ws.view, mp)
    assert st == 0
    for g, what in ((rep, "rep"), (dist, "dist"), (ws, "admission workspace")):
        g.check(what)
    orep, odist, odh, okept = oracle.admit_batch(x.cpu().numpy(), dig.cpu().numpy().view(np.uint64),
                                                 delta)
    assert np.array_equal(rep.view.cpu().numpy(), orep) and kept == okept
    assert np.array_equal(dist.view.cpu().numpy(), odist)


@pytest.mark.parametrize("width", [1, 2])
def test_code_sqnorms(dev, width):
    N, D = 1001, 40
    c = torch.from_numpy(
        np.random.default_rng(width).integers(-100, 100, (N, D)).astype(
            {1: np.int8, 2: np.int16}[width])).to(dev)
    out = Guarded(dev, N * 4, torch.float32)
    lam.lam_code_sqnorms(c, width, N, D, out.view)
    out.check("sqnorms")
    want = (c.cpu().numpy().astype(np.int64) ** 2).sum(axis=1).astype(np.float32)
    assert np.array_equal(out.view.cpu().numpy(), want)


@pytest.mark.parametrize("n", [13, 100003])
def test_device_resident_quantize_and_dequantize(dev, n):
    x_np = inputs.flat_values(n, seed=n + 1)
    x = torch.from_numpy(x_np).to(dev)
    oc, rmin, rmax, _ = oracle.quantize(x_np, 1e-2)
    w = oracle.width(rmin, rmax)
    codes = Guarded(dev, 4 * n)  # room for any width: the width is settled on the device
    qws = Guarded(dev, 256)
    lam.lam_quantize_async(x, 1e-2, 0, codes.view, qws.view)
    st, gw, *_ = lam.lam_quantize_result(qws.view, 1e-2, 0)
    assert st == 0 and gw == w
    codes.check("async codes")
    qws.check("quantize status")
    out = Guarded(dev, 4 * n, torch.float32)
    lam.lam_dequantize_from(codes.view, qws.view, n, 1e-2, out.view)
    out.check("dequantize_from out")
    assert np.array_equal(out.view.cpu().numpy(),
                          oracle.dequantize(oc, np.float32(2 * np.float32(1e-2))))


@pytest.mark.parametrize("B,k", [(1, 10), (3, 100), (520, 10)])
def test_device_resident_search(dev, B, k):
    N, D = 3001, 768
    x_np = inputs.unit_rows(N, D, seed=B)
    x = torch.from_numpy(x_np).to(dev)
    codes = Guarded(dev, 4 * N * D)
    qws = Guarded(dev, 256)
    lam.lam_quantize_async(x.reshape(-1), 1e-2, 0, codes.view, qws.view)
    q = torch.from_numpy(inputs.queries(B, D, seed=k)).to(dev)
    s = Guarded(dev, B * k * 4, torch.float32)
    i = Guarded(dev, B * k * 8, torch.int64)
    ws = Guarded(dev, lam.lam_score_topk_from_workspace_size(B, N, D, k))
    lam.lam_score_topk_from(q, codes.view, qws.view, N, D, 1e-2, k, oracle.L2, s.shaped(B, k),
                            i.shaped(B, k), ws.view)
    assert lam.lam_score_topk_status(ws.view) == lam.LAM_OK
    for g, what in ((codes, "codes"), (qws, "quantize status"), (s, "scores"), (i, "ids"),
                    (ws, "search workspace")):
        g.check(what)
    oc, rmin, rmax, _ = oracle.quantize(x_np, 1e-2)
    ps, pi = lam.search(q, torch.from_numpy(oc.reshape(N, D).astype(np.int8)).to(dev), 1e-2, k,
                        oracle.L2, code_bound=128)
    assert np.array_equal(i.shaped(B, k).cpu().numpy(), pi.cpu().numpy())


def test_noalloc_search(dev):
    B, N, D, k = 64, 6000, 768, 10
    x_np = inputs.unit_rows(N, D, seed=6)
    oc, rmin, rmax, _ = oracle.quantize(x_np, 1e-2)
    codes = torch.from_numpy(oc.reshape(N, D).astype(np.int8)).to(dev)
    q = torch.from_numpy(inputs.queries(B, D, seed=7)).to(dev)
    s = Guarded(dev, B * k * 4, torch.float32)
    i = Guarded(dev, B * k * 8, torch.int64)
    _lib.lam_score_topk_noalloc(q, codes, 1, N, D, 1e-2, 128, k, oracle.IP, s.shaped(B, k),
                                i.shaped(B, k))
    s.check("noalloc scores")
    i.check("noalloc ids")
    ps, pi = lam.search(q, codes, 1e-2, k, oracle.IP, code_bound=128)
    assert np.array_equal(i.shaped(B, k).cpu().numpy(), pi.cpu().numpy())
