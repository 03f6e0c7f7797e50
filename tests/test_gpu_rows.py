"""Per-vector byte codecs of the composite experiment (fp16, per-vector int8,
sign-binary): the CUDA encoders and decoder against the oracle bit for bit
(the sign codec's fp64 scale to one fp32 ulp), and exact search over the
coded rows (lam_score_topk_rows, tensor and generic paths) against the
oracle's scores of the decoded rows."""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_32256_gb300 as lam
from paper_2609_32256_gb300 import inputs
from tests.parity import check_topk_fn

pytestmark = pytest.mark.gpu
METRICS = (oracle.IP, oracle.COSINE, oracle.L2)
FMTS = (lam.LAM_ROWS_INT8, lam.LAM_ROWS_FP16, lam.LAM_ROWS_SIGN)
ORACLE_FMT = {lam.LAM_ROWS_INT8: oracle.FMT_INT8_ROWS, lam.LAM_ROWS_FP16: oracle.FMT_FP16,
              lam.LAM_ROWS_SIGN: oracle.FMT_SIGN}


def special_rows(d):
    """Unit rows plus a constant row, a zero row, a row of -0.0 and a ramp."""
    x = inputs.unit_rows(61, d, seed=d)
    x[3] = 0.25
    x[7] = 0.0
    x[11] = -0.0
    x[13] = np.linspace(-1.0, 1.0, d, dtype=np.float32)
    return x


def encode_both(dev, x, fmt):
    oc, osc, oof = oracle.encode_rows(x, ORACLE_FMT[fmt])
    gc, gsc, gof = lam.encode_rows(torch.from_numpy(x).to(dev), fmt)
    torch.cuda.synchronize()
    return (oc, osc, oof), (gc.cpu().numpy(), None if gsc is None else gsc.cpu().numpy(),
                            None if gof is None else gof.cpu().numpy())


@pytest.mark.parametrize("d", [8, 24, 768, 1000])
def test_encoders_match_the_oracle(dev, d):
    x = special_rows(d)
    for fmt in FMTS:
        if fmt == lam.LAM_ROWS_SIGN and d % 8:
            continue
        (oc, osc, oof), (gc, gsc, gof) = encode_both(dev, x, fmt)
        if fmt == lam.LAM_ROWS_FP16:
            assert np.array_equal(gc.view(np.uint16), oc.view(np.uint16))
        else:
            assert np.array_equal(gc.view(np.uint8), oc.view(np.uint8))
        if fmt == lam.LAM_ROWS_INT8:
            assert np.array_equal(gsc.view(np.uint32), osc.view(np.uint32))
            assert np.array_equal(gof.view(np.uint32), oof.view(np.uint32))
        if fmt == lam.LAM_ROWS_SIGN:
            # fp64 sums in two orders: equal, or one fp32 ulp apart
            ulp = np.abs(gsc.view(np.int32).astype(np.int64) - osc.view(np.int32))
            assert ulp.max() <= 1


def test_encoders_at_the_workload_size(dev):
    x = inputs.unit_rows(27986, 768, seed=3)
    for fmt in FMTS:
        (oc, osc, oof), (gc, gsc, gof) = encode_both(dev, x, fmt)
        assert np.array_equal(gc.view(np.uint8), oc.view(np.uint8))
        if osc is not None:
            ulp = np.abs(gsc.view(np.int32).astype(np.int64) - osc.view(np.int32))
            assert ulp.max() <= (1 if fmt == lam.LAM_ROWS_SIGN else 0)
        if oof is not None:
            assert np.array_equal(gof.view(np.uint32), oof.view(np.uint32))


@pytest.mark.parametrize("fmt", FMTS)
def test_decoder_matches_the_oracle(dev, fmt):
    x = special_rows(64)
    oc, osc, oof = oracle.encode_rows(x, ORACLE_FMT[fmt])
    want = oracle.decode_rows(oc, ORACLE_FMT[fmt], 64, osc, oof)
    t = lambda a: None if a is None else torch.from_numpy(np.ascontiguousarray(a)).to(dev)
    out = torch.empty((61, 64), dtype=torch.float32, device=dev)
    lam.lam_decode_rows(t(oc), fmt, 61, 64, t(osc), t(oof), out)
    assert np.array_equal(out.cpu().numpy().view(np.uint32), want.view(np.uint32))


def rows_case(dev, fmt, n, d, B, k, metric, seed=0, misalign=False):
    """Oracle-encoded rows; GPU top-k against the oracle's decoded-row scores."""
    x = inputs.unit_rows(n, d, seed=seed)
    if n > 40:
        x[17::23] = x[5]  # exact duplicates: equal scores, lower id first
    q = inputs.queries(B, d, seed=seed + 7)
    ofmt = ORACLE_FMT[fmt]
    oc, osc, oof = oracle.encode_rows(x, ofmt)
    rows = oracle.decode_rows(oc, ofmt, d, osc, oof)
    t = lambda a: None if a is None else torch.from_numpy(np.ascontiguousarray(a)).to(dev)
    codes = t(oc)
    if misalign:  # codes one element past a 16-byte boundary
        buf = torch.empty((oc.size + 16,), dtype=codes.dtype, device=dev)
        buf[1:1 + oc.size] = codes.reshape(-1)
        codes = buf[1:1 + oc.size].view(oc.shape)
    gs, gi = lam.search_rows(t(q), codes, fmt, t(osc), t(oof), k, metric, D=d)
    gs, gi = gs.cpu().numpy(), gi.cpu().numpy()
    full = oracle.scores_rows(q, rows, metric)
    os_, oi = oracle.topk(full, k, metric)
    check_topk_fn(gs, gi, lambda b, ids: full[b, ids], n, metric, os_, oi)


@pytest.mark.parametrize("metric", METRICS)
@pytest.mark.parametrize("fmt", FMTS)
@pytest.mark.parametrize("B", [1, 3, 130, 300])
def test_tensor_path(dev, score_path, fmt, metric, B):
    score_path("tensor")
    assert lam.lam_score_topk_rows_path(B, 3001, 768, 10, fmt) == lam.PATH_TENSOR
    rows_case(dev, fmt, 3001, 768, B, 10, metric, seed=B)


@pytest.mark.parametrize("fmt", FMTS)
@pytest.mark.parametrize("k", [1, 16, 17, 32, 100, 128])
def test_tensor_path_k(dev, score_path, fmt, k):
    score_path("tensor")
    for metric in METRICS:
        rows_case(dev, fmt, 700, 256, 140, k, metric, seed=k)


@pytest.mark.parametrize("fmt", FMTS)
@pytest.mark.parametrize("d", [16, 48, 1024])
def test_tensor_path_dims(dev, score_path, fmt, d):
    score_path("tensor")
    for metric in METRICS:
        rows_case(dev, fmt, 513, d, 129, 10, metric, seed=d)


@pytest.mark.parametrize("metric", METRICS)
@pytest.mark.parametrize("fmt", FMTS)
def test_generic_path(dev, score_path, fmt, metric):
    score_path("generic")
    rows_case(dev, fmt, 1201, 768, 5, 10, metric, seed=3)
    rows_case(dev, fmt, 333, 24 if fmt != lam.LAM_ROWS_SIGN else 40, 3, 7, metric, seed=4)


@pytest.mark.parametrize("fmt", FMTS)
def test_auto_paths_large_k_odd_dims_and_misaligned_codes(dev, fmt):
    # k above the tensor path's limit and D not a multiple of 16 go generic
    assert lam.lam_score_topk_rows_path(4, 900, 768, 300, fmt) == lam.PATH_GENERIC
    rows_case(dev, fmt, 900, 768, 4, 300, oracle.IP, seed=5)
    assert lam.lam_score_topk_rows_path(4, 900, 40, 10, fmt) == lam.PATH_GENERIC
    rows_case(dev, fmt, 900, 40, 4, 10, oracle.L2, seed=6)
    # codes one element off a 16-byte boundary
    rows_case(dev, fmt, 900, 768, 200, 10, oracle.COSINE, seed=8, misalign=True)


@pytest.mark.parametrize("fmt", FMTS)
def test_workload_size_sampled(dev, fmt):
    """27,986 rows x 768, 1,024 queries, top-10 inner product (the scoring
    workload), checked on a sample of queries the oracle scores in full."""
    n, d, B, k = 27986, 768, 1024, 10
    x = inputs.unit_rows(n, d, seed=21)
    q = inputs.queries(B, d, seed=22)
    ofmt = ORACLE_FMT[fmt]
    oc, osc, oof = oracle.encode_rows(x, ofmt)
    t = lambda a: None if a is None else torch.from_numpy(np.ascontiguousarray(a)).to(dev)
    gs, gi = lam.search_rows(t(q), t(oc), fmt, t(osc), t(oof), k, oracle.IP)
    gs, gi = gs.cpu().numpy(), gi.cpu().numpy()
    rows = oracle.decode_rows(oc, ofmt, d, osc, oof)
    sample = np.array([0, 1, 127, 128, 511, 700, 1022, 1023])
    full = oracle.scores_rows(q[sample], rows, oracle.IP)
    os_, oi = oracle.topk(full, k, oracle.IP)
    check_topk_fn(gs[sample], gi[sample], lambda b, ids: full[b, ids], n, oracle.IP, os_, oi)


def test_two_slabs_with_first_slab_bound(dev):
    """Per-vector int8 rows over two fp16 slabs (750,000 x 768), L2 top-100:
    the second slab offers only rows at least as good as the first slab's
    k-th best; sampled queries against the oracle."""
    n, d, k = 750000, 768, 100
    x = inputs.unit_rows_device(n, d, seed=78, device=dev)
    x[700100:700140] = x[0:40]
    codes, scale, offset = lam.encode_rows(x, lam.LAM_ROWS_INT8)
    q = inputs.queries(200, d, seed=6)
    x_np = x.cpu().numpy()
    q[7] = x_np[30]
    del x
    # the oracle encodes the same rows: codes and factors bit-exact, and its
    # own rows feed its scores
    oc, osc, oof = oracle.encode_rows(x_np, oracle.FMT_INT8_ROWS)
    del x_np
    assert np.array_equal(codes.cpu().numpy(), oc)
    assert np.array_equal(scale.cpu().numpy().view(np.uint32), osc.view(np.uint32))
    assert np.array_equal(offset.cpu().numpy().view(np.uint32), oof.view(np.uint32))
    gs, gi = lam.search_rows(torch.from_numpy(q).to(dev), codes, lam.LAM_ROWS_INT8, scale,
                             offset, k, oracle.L2)
    gs, gi = gs.cpu().numpy(), gi.cpu().numpy()
    rows = oracle.decode_rows(oc, oracle.FMT_INT8_ROWS, d, osc, oof)
    sel = np.array([0, 7, 128, 199])
    full = oracle.scores_rows(q[sel], rows, oracle.L2)
    os_, oi = oracle.topk(full, k, oracle.L2)
    check_topk_fn(gs[sel], gi[sel], lambda b, ids: full[b, ids], n, oracle.L2, os_, oi)


@pytest.mark.parametrize("metric", METRICS)
@pytest.mark.parametrize("fmt", FMTS)
@pytest.mark.parametrize("B", [1, 2])
@pytest.mark.parametrize("k", [1, 10, 100, 128])
def test_bandwidth_path(dev, score_path, fmt, metric, B, k):
    score_path("bandwidth")
    assert lam.lam_score_topk_rows_path(B, 5003, 768, k, fmt) == lam.PATH_BANDWIDTH
    rows_case(dev, fmt, 5003, 768, B, k, metric, seed=B + k)


@pytest.mark.parametrize("fmt", FMTS)
@pytest.mark.parametrize("d", [128, 256, 1024])
@pytest.mark.parametrize("B", [1, 2])
def test_bandwidth_path_dims(dev, score_path, fmt, d, B):
    score_path("bandwidth")
    for metric in METRICS:
        rows_case(dev, fmt, 777, d, B, 10, metric, seed=d + B)


@pytest.mark.parametrize("fmt", FMTS)
@pytest.mark.parametrize("n", [1, 5, 63, 64, 65, 1029])
def test_bandwidth_path_ragged_rows(dev, score_path, fmt, n):
    # fewer rows than one stage or one warp group, and ragged last stages: the
    # one-query paths prefetch row factors across groups and stages
    score_path("bandwidth")
    for metric in METRICS:
        rows_case(dev, fmt, n, 768, 1, min(10, n), metric, seed=n)


def test_bandwidth_path_routing(dev):
    # small batches go to the bandwidth kernel when a row is a multiple of 16
    # bytes; otherwise to the tensor cores or the generic kernel
    assert lam.lam_score_topk_rows_path(1, 1000, 768, 10, lam.LAM_ROWS_SIGN) == lam.PATH_BANDWIDTH
    assert lam.lam_score_topk_rows_path(1, 1000, 64, 10, lam.LAM_ROWS_SIGN) == lam.PATH_TENSOR
    assert lam.lam_score_topk_rows_path(1, 1000, 24, 10, lam.LAM_ROWS_FP16) == lam.PATH_BANDWIDTH
    assert lam.lam_score_topk_rows_path(1, 1000, 24, 10, lam.LAM_ROWS_INT8) == lam.PATH_GENERIC
    assert lam.lam_score_topk_rows_path(3, 1000, 768, 10, lam.LAM_ROWS_INT8) == lam.PATH_TENSOR
    assert lam.lam_score_topk_rows_path(2, 1000, 768, 200, lam.LAM_ROWS_INT8) == lam.PATH_GENERIC
