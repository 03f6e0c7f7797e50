"""Exact search on the codes (dequantisation fused into the score, then top-k)
against the CPU oracle, per kernel path, metric, width and shape, including
ragged tiles, ragged query blocks, planted exact ties and error statuses."""
import hashlib

import numpy as np
import pytest
import torch

import oracle
import paper_2609_32256_gb300 as lam
from paper_2609_32256_gb300 import inputs
from tests.parity import check_topk, oracle_topk, quantize_rows

pytestmark = pytest.mark.gpu
METRICS = (oracle.IP, oracle.COSINE, oracle.L2)
NP_DT = {1: np.int8, 2: np.int16, 4: np.int32}


def make_codes(n, d, eps, width, seed=0, dup_every=0):
    """Unit rows quantized by the oracle; optionally exact duplicate rows."""
    x = inputs.unit_rows(n, d, seed=seed)
    if dup_every:
        x[dup_every::dup_every] = x[0]
    oc, rmin, rmax, _ = oracle.quantize(x, eps)
    assert oracle.width(rmin, rmax) <= width
    return oc.reshape(n, d), max(-int(rmin), int(rmax))


def run(dev, q, codes_i32, width, eps, k, metric, code_bound):
    qt = torch.from_numpy(q).to(dev)
    ct = torch.from_numpy(codes_i32.astype(NP_DT[width])).to(dev)
    s, i = lam.search(qt, ct, eps, k, metric, code_bound=code_bound)
    return s.cpu().numpy(), i.cpu().numpy()


def check(dev, q, codes, width, eps, k, metric, bound):
    gs, gi = run(dev, q, codes, width, eps, k, metric, bound)
    os_, oi = oracle_topk(q, codes, eps, metric, k)
    check_topk(gs, gi, q, codes, eps, metric, os_, oi)
    return gs, gi, os_, oi


@pytest.mark.parametrize("metric", METRICS)
@pytest.mark.parametrize("width,eps", [(1, 1e-2), (2, 1e-3)])
@pytest.mark.parametrize("B", [1, 2])
@pytest.mark.parametrize("k", [1, 10, 100, 128])
def test_bandwidth_path(dev, score_path, metric, width, eps, B, k):
    score_path("bandwidth")
    codes, bound = make_codes(5003, 768, eps, width)
    q = inputs.queries(B, 768, seed=9)
    assert lam.lam_score_topk_path(B, 5003, 768, k, width, bound) == lam.PATH_BANDWIDTH
    check(dev, q, codes, width, eps, k, metric, bound)


@pytest.mark.parametrize("D", [64, 256, 1024])
def test_bandwidth_path_other_dims(dev, score_path, D):
    score_path("bandwidth")
    codes, bound = make_codes(777, D, 1e-2, 1, seed=D)
    q = inputs.queries(2, D, seed=3)
    for metric in METRICS:
        check(dev, q, codes, 1, 1e-2, 10, metric, bound)


@pytest.mark.parametrize("metric", METRICS)
@pytest.mark.parametrize("width,eps", [(1, 1e-2), (2, 1e-3), (2, 1e-4)])
@pytest.mark.parametrize("B", [3, 16, 64, 65, 130, 500])
def test_tensor_path(dev, score_path, metric, width, eps, B):
    score_path("tensor")
    codes, bound = make_codes(3001, 768, eps, width, seed=B)
    q = inputs.queries(B, 768, seed=B + 100)
    assert lam.lam_score_topk_path(B, 3001, 768, 10, width, bound) == lam.PATH_TENSOR
    check(dev, q, codes, width, eps, 10, metric, bound)


@pytest.mark.parametrize("D", [16, 48, 80, 1024])
@pytest.mark.parametrize("k", [1, 16, 17, 32, 64, 112])
@pytest.mark.parametrize("B", [20, 300, 520])  # 1 and 3 query blocks (stage-loop conversion); 5 (conversion pass)
def test_tensor_path_dims_and_k(dev, score_path, D, k, B):
    score_path("tensor")
    codes, bound = make_codes(700, D, 1e-2, 1, seed=D + k)
    q = inputs.queries(B, D, seed=k)
    for metric in METRICS:
        check(dev, q, codes, 1, 1e-2, k, metric, bound)


@pytest.mark.parametrize("width,eps", [(1, 1e-2), (2, 1e-4), (4, 1e-6)])
@pytest.mark.parametrize("D", [33, 768])
def test_generic_path(dev, score_path, width, eps, D):
    score_path("generic")
    codes, bound = make_codes(1500, D, eps, width, seed=D)
    q = inputs.queries(5, D, seed=D)
    for metric in METRICS:
        for k in (1, 10, 1024):
            check(dev, q, codes, width, eps, k, metric, bound)


@pytest.mark.parametrize("path,B", [("bandwidth", 2), ("tensor", 8), ("tensor", 136),
                                    ("generic", 8)])
def test_exact_ties_rank_lower_id_first(dev, score_path, path, B):
    score_path(path)
    codes, bound = make_codes(2000, 768, 1e-2, 1, dup_every=97)  # rows 0,97,194,... identical
    q = inputs.unit_rows(2000, 768, seed=0)[:B]
    for metric in METRICS:
        gs, gi, os_, oi = check(dev, q, codes, 1, 1e-2, 25, metric, bound)
        # query 0 equals row 0, so the 21 copies of it lead, in id order
        dup = np.arange(0, 2000, 97)
        np.testing.assert_array_equal(gi[0][: dup.size], dup)
        np.testing.assert_array_equal(oi[0][: dup.size], dup)


def test_auto_selects_paths(dev):
    assert lam.lam_score_topk_path(1, 361802, 768, 10, 2, 120) == lam.PATH_BANDWIDTH
    assert lam.lam_score_topk_path(64, 361802, 768, 10, 2, 120) == lam.PATH_TENSOR
    # int16 codes with no bound, or beyond 2048, take the split (256 h + l) tensor path
    assert lam.lam_score_topk_path(64, 361802, 768, 10, 2, 0) == lam.PATH_TENSOR
    assert lam.lam_score_topk_path(64, 361802, 768, 10, 2, 4000) == lam.PATH_TENSOR
    assert lam.lam_score_topk_path(64, 361802, 768, 10, 4, 0) == lam.PATH_GENERIC
    assert (lam.lam_score_topk_workspace_size(64, 361802, 768, 10, 2, 4000) >
            lam.lam_score_topk_workspace_size(64, 361802, 768, 10, 2, 120))
    assert lam.lam_score_topk_path(256, 8388608, 768, 100, 1, 0) == lam.PATH_TENSOR
    assert lam.lam_score_topk_path(4, 1000, 768, 500, 1, 0) == lam.PATH_GENERIC


@pytest.mark.parametrize("metric", METRICS)
@pytest.mark.parametrize("B", [3, 64, 130, 520])
@pytest.mark.parametrize("eps,known", [(2e-5, True), (2e-5, False), (1e-3, False)])
def test_tensor_path_int16_split(dev, score_path, metric, B, eps, known):
    """int16 codes the fp16 operands cannot hold (|c| up to ~8,000 at eps=2e-5),
    or with no bound given: the tensor path splits each code as 256 h + l."""
    score_path("tensor")
    codes, bound = make_codes(2500, 768, eps, 2, seed=B + 7)
    assert (bound > 2048) == (eps == 2e-5)
    cb = bound if known else 0
    assert lam.lam_score_topk_path(B, 2500, 768, 10, 2, cb) == lam.PATH_TENSOR
    q = inputs.queries(B, 768, seed=B + 8)
    check(dev, q, codes, 2, eps, 10, metric, cb)


@pytest.mark.parametrize("k", [1, 32, 100])
def test_tensor_path_int16_full_range(dev, score_path, k):
    """Codes spanning the whole int16 range (the largest |c| = 32767 and
    -32768), ragged tile and query block, D not a multiple of 32."""
    score_path("tensor")
    n, d = 1300, 272
    x = inputs.unit_rows(n, d, seed=k)
    x[5, 7] = 0.999
    x[9, 3] = -0.999
    eps = float(np.float32(0.999 / 2 / 32767.4))
    oc, rmin, rmax, _ = oracle.quantize(x, eps)
    assert oracle.width(rmin, rmax) == 2 and max(-rmin, rmax) >= 32767
    codes = oc.reshape(n, d)
    codes[11, :] = -32768
    q = inputs.queries(140, d, seed=k + 1)
    for metric in METRICS:
        check(dev, q, codes, 2, eps, k, metric, 0)


def test_forced_path_unsupported(dev, score_path):
    score_path("bandwidth")
    codes, bound = make_codes(100, 768, 1e-2, 1)
    q = torch.from_numpy(inputs.queries(5, 768, seed=1)).to(dev)
    ct = torch.from_numpy(codes.astype(np.int8)).to(dev)
    assert lam.lam_score_topk_workspace_size(5, 100, 768, 10, 1, bound) == 0
    ws = torch.empty(1 << 20, dtype=torch.uint8, device=dev)
    s = torch.empty((5, 10), dtype=torch.float32, device=dev)
    i = torch.empty((5, 10), dtype=torch.int64, device=dev)
    with pytest.raises(lam.LamError) as e:
        lam.lam_score_topk(q, ct, 1, 100, 768, 1e-2, bound, 10, oracle.IP, s, i, ws)
    assert e.value.status == lam.LAM_ERR_UNSUPPORTED


@pytest.mark.parametrize("B", [4, 200])
def test_code_bound_violation_reported(dev, score_path, B):
    score_path("tensor")
    codes, _ = make_codes(600, 64, 1e-4, 2)
    codes[5, 3] = 3000  # beyond what the tensor path can hold exactly
    q = inputs.queries(B, 64, seed=2)
    with pytest.raises(lam.LamError) as e:
        run(dev, q, codes, 2, 1e-4, 10, oracle.IP, 2048)
    assert e.value.status == lam.LAM_ERR_RANGE


def test_k_equals_n_and_single_row(dev):
    for path_n in (1, 7, 300):
        codes, bound = make_codes(path_n, 768, 1e-2, 1, seed=path_n)
        q = inputs.queries(3, 768, seed=4)
        for metric in METRICS:
            check(dev, q, codes, 1, 1e-2, path_n, metric, bound) if path_n <= 128 else \
                check(dev, q, codes, 1, 1e-2, 128, metric, bound)


@pytest.mark.parametrize("B", [4, 140])
def test_zero_rows_and_zero_query_cosine(dev, B):
    codes, bound = make_codes(500, 768, 1e-2, 1)
    codes[10:20] = 0
    q = inputs.queries(B, 768, seed=5)
    q[1] = 0.0
    for metric in METRICS:
        check(dev, q, codes, 1, 1e-2, 30, metric, bound)


@pytest.mark.parametrize("width", [1, 2])
@pytest.mark.parametrize("N,D", [(1, 1), (1000, 33), (777, 768)])
def test_code_sqnorms_bit_exact(dev, width, N, D):
    rng = np.random.default_rng(N + D + width)
    lo, hi = (-128, 128) if width == 1 else (-32768, 32768)
    c = rng.integers(lo, hi, size=(N, D)).astype(NP_DT[width])
    c[0, :] = lo  # the extreme code everywhere in one row
    want = oracle.code_sqnorms(c.astype(np.int32))
    ct = torch.from_numpy(c).to(dev)
    out = torch.empty(N, dtype=torch.float32, device=dev)
    lam.lam_code_sqnorms(ct, width, N, D, out)
    np.testing.assert_array_equal(out.cpu().numpy().view(np.uint32), want.view(np.uint32))


@pytest.mark.parametrize("metric,k", [(oracle.IP, 10), (oracle.L2, 100), (oracle.COSINE, 128)])
def test_tensor_two_slabs_with_first_slab_bound(dev, score_path, metric, k):
    """750,000 rows take two fp16 slabs: the second slab only offers rows at
    least as good as the first slab's k-th best.  Duplicated rows across the
    slab boundary tie exactly; sampled queries against the oracle."""
    score_path("tensor")
    n, d, eps = 750000, 768, 1e-2
    x = inputs.unit_rows_device(n, d, seed=77, device=dev)
    x[720000:720050] = x[10:60]  # second-slab copies of first-slab rows
    codes = torch.empty((n, d), dtype=torch.int8, device=dev)
    ws = torch.zeros(64, dtype=torch.uint8, device=dev)
    st, w, scale, cmin, cmax = lam.lam_quantize(x, eps, 1, codes, ws)
    assert st == 0 and w == 1
    # the oracle quantizes the same rows: every code bit-exact, and its own
    # codes feed its search
    oc, rmin, rmax, nnf = quantize_rows(x.cpu().numpy(), eps)
    del x
    assert nnf == 0 and (cmin, cmax) == (int(rmin), int(rmax))
    assert hashlib.sha256(codes.cpu().numpy().tobytes()).hexdigest() == \
        hashlib.sha256(oc.astype(np.int8).tobytes()).hexdigest()
    q = inputs.queries(520, d, seed=5)  # five query blocks: the conversion pass, in slabs
    # plant queries equal to duplicated rows so that the ties reach the top-k
    q[3] = oracle.dequantize(oc[20], scale)
    q[129] = oracle.dequantize(oc[45], scale)
    gs, gi = lam.search(torch.from_numpy(q).to(dev), codes, eps, k, metric,
                        code_bound=max(-cmin, cmax))
    gs, gi = gs.cpu().numpy(), gi.cpu().numpy()
    sel = np.array([0, 3, 129, 257, 519])
    os_, oi = oracle_topk(q[sel], oc, eps, metric, k)
    check_topk(gs[sel], gi[sel], q[sel], oc, eps, metric, os_, oi)


def test_tensor_k128_needs_the_conversion_pass(dev, score_path):
    """k = 128 fits the conversion-pass kernel only: five query blocks take the
    tensor path, one block the generic path."""
    codes, bound = make_codes(2000, 768, 1e-2, 1, seed=128)
    assert lam.lam_score_topk_path(520, 2000, 768, 128, 1, bound) == lam.PATH_TENSOR
    assert lam.lam_score_topk_path(100, 2000, 768, 128, 1, bound) == lam.PATH_GENERIC
    score_path("tensor")
    q = inputs.queries(520, 768, seed=128)
    for metric in METRICS:
        check(dev, q, codes, 1, 1e-2, 128, metric, bound)


@pytest.mark.parametrize("path", ["bandwidth", "tensor", "generic"])
@pytest.mark.parametrize("qscale", [1e-30, 1e-3, 1e20])
def test_query_scale_extremes(dev, score_path, path, qscale):
    """Queries far from unit norm: the integer-digit (int8, bandwidth) and
    split-fp16 (tensor) encodings of the query rescale by a power of two, so
    inner-product and cosine scores keep their relative accuracy."""
    score_path(path)
    codes, bound = make_codes(1500, 768, 1e-2, 1, seed=31)
    B = 2 if path == "bandwidth" else 130
    q = (inputs.queries(B, 768, seed=32).astype(np.float64) * qscale).astype(np.float32)
    q[1, 5:] = 0.0  # one query with a few coordinates only
    for metric in (oracle.IP, oracle.COSINE):
        check(dev, q, codes, 1, 1e-2, 10, metric, bound)
