"""Pins of the CPU oracle to what the paper and the mathematics fix.

None of these compares the oracle with itself: each checks a value the paper
prints, a hand computation, a closed form, an invariant of Q_eps, or a brute
force over tiny inputs.  A dropped factor of 2 in the step, a different tie
rule, a transposed code index, a wrong norm in the cosine, a sign slip in the
L2 cross term or a reversed ranking direction each fails at least one test.
"""
import math

import numpy as np
import pytest

import oracle
from tests.conftest import golden
from paper_2609_32256_gb300 import inputs

EPS_SWEEP = (1e-2, 1e-3, 1e-4)


# --- Q_eps (Sec. 3.2, layer L1) -------------------------------------------------

def test_worked_ties_half_to_even():
    eps = np.float32(2.0 ** -10)
    s = np.float32(2.0 ** -9)
    rows = golden("q_eps_ties.txt")
    v = np.array([float(r[0]) for r in rows], dtype=np.float32)
    want = np.array([int(r[1]) for r in rows], dtype=np.int64)
    x = v * s  # power-of-two scaling: exact
    codes, rmin, rmax, nnf = oracle.quantize(x, eps)
    assert nnf == 0
    np.testing.assert_array_equal(codes.astype(np.int64), want)
    assert rmin == want.min() and rmax == want.max()


def test_step_is_two_eps():
    # x = 0.9 * 2eps must land in cell 1 (a step of eps would give 2).
    for eps in EPS_SWEEP:
        s = np.float32(2.0) * np.float32(eps)
        x = np.array([0.9, -0.9, 1.9, 0.45], dtype=np.float32) * s
        codes, *_ = oracle.quantize(x, eps)
        assert list(codes) == [1, -1, 2, 0]
    assert oracle.step(np.float32(1e-3)) == np.float32(2.0) * np.float32(1e-3)


def _bound_slack(x, eps):
    # |x - s*c| <= eps + one rounding of the quotient and one of the product.
    return eps * (1 + 2.0 ** -23) + np.abs(x.astype(np.float64)) * 2.0 ** -23


@pytest.mark.parametrize("eps", EPS_SWEEP)
def test_dequant_error_bound_and_tight(eps):
    x = inputs.flat_values(1 << 20, seed=7)
    codes, *_ = oracle.quantize(x, eps)
    xh = oracle.dequantize(codes, oracle.step(eps))
    err = np.abs(x.astype(np.float64) - xh.astype(np.float64))
    assert np.all(err <= _bound_slack(x, np.float64(np.float32(eps))))
    # Tightness: the cell half-width is eps, so dense inputs reach it.
    dense = np.linspace(-50 * eps, 50 * eps, 200001, dtype=np.float32)
    c2, *_ = oracle.quantize(dense, eps)
    e2 = np.abs(dense.astype(np.float64) - oracle.dequantize(c2, oracle.step(eps)))
    assert e2.max() > 0.99 * eps


@pytest.mark.parametrize("eps", EPS_SWEEP)
def test_idempotent_on_every_int16_code(eps):
    c = np.arange(-32768, 32768, dtype=np.int32)
    xh = oracle.dequantize(c, oracle.step(eps))
    c2, rmin, rmax, nnf = oracle.quantize(xh, eps)
    np.testing.assert_array_equal(c2, c)
    assert (rmin, rmax, nnf) == (-32768, 32767, 0)


def test_monotone_and_odd():
    x = np.sort(inputs.flat_values(200000, seed=3))
    for eps in EPS_SWEEP:
        c, *_ = oracle.quantize(x, eps)
        assert np.all(np.diff(c) >= 0)
        cn, *_ = oracle.quantize(-x, eps)
        np.testing.assert_array_equal(cn, -c)


@pytest.mark.parametrize("lo,hi,w", [
    (0, 0, 1), (-128, 127, 1), (-129, 0, 2), (0, 128, 2), (-32768, 32767, 2),
    (-32769, 0, 4), (0, 32768, 4), (-2147483648, 2147483647, 4),
    (-2147483649, 0, 0), (0, 2147483648, 0)])
def test_width_boundaries(lo, hi, w):
    assert oracle.width(float(lo), float(hi)) == w


def test_width_from_quantized_range():
    eps = np.float32(2.0 ** -10)
    s = np.float32(2.0 ** -9)
    for vals, w in [([127.4, -128.4], 1), ([127.5], 2), ([-128.6], 2),
                    ([32767.4], 2), ([32767.5], 4)]:
        x = np.array(vals, dtype=np.float32) * s
        _, rmin, rmax, _ = oracle.quantize(x, eps)
        assert oracle.width(rmin, rmax) == w


def test_nonfinite_counted():
    x = np.array([0.1, np.nan, np.inf, -np.inf, 0.2], dtype=np.float32)
    codes, rmin, rmax, nnf = oracle.quantize(x, 1e-2)
    assert nnf == 3
    assert list(codes) == [5, 0, 0, 0, 10]
    assert (rmin, rmax) == (5, 10)


def test_empty_input():
    codes, rmin, rmax, nnf = oracle.quantize(np.zeros(0, np.float32), 1e-3)
    assert codes.size == 0 and (rmin, rmax, nnf) == (0, 0, 0)


# --- scores (exact search, Sec. "Brute-force scan crossover"; Eq. 1) -----------

def test_scores_d2_hand_computed():
    q = np.array([[0.6, 0.8]], dtype=np.float32)
    c = np.array([[3, -1]], dtype=np.int32)
    for metric, want in golden("scores_d2_hand.txt"):
        got = oracle.scores(q, c, 0.25, int(metric))[0, 0]
        assert got == np.float32(float(want))


def test_scores_d1_closed_form():
    eps = 0.125  # s = 0.25
    q = np.array([[-2.0], [0.0], [3.0]], dtype=np.float32)
    c = np.array([[4], [-3], [0]], dtype=np.int32)
    ip = oracle.scores(q, c, eps, oracle.IP)
    np.testing.assert_array_equal(ip, np.outer(q[:, 0], 0.25 * c[:, 0]).astype(np.float32))
    cos = oracle.scores(q, c, eps, oracle.COSINE)
    np.testing.assert_array_equal(
        cos, np.array([[-1, 1, 0], [0, 0, 0], [1, -1, 0]], dtype=np.float32))
    l2 = oracle.scores(q, c, eps, oracle.L2)
    want = (q[:, 0][:, None] - 0.25 * c[:, 0][None, :]) ** 2
    np.testing.assert_array_equal(l2, want.astype(np.float32))


def test_basis_queries_read_codes():
    # IP with the unit vector e_d equals s * c[i, d]: pins the code indexing.
    rng = np.random.default_rng(5)
    N, D, eps = 7, 5, 1e-2
    c = rng.integers(-100, 100, size=(N, D), dtype=np.int32)
    q = np.eye(D, dtype=np.float32)
    ip = oracle.scores(q, c, eps, oracle.IP)
    s = oracle.step(eps)
    np.testing.assert_array_equal(ip, (s * c.T.astype(np.float32)).astype(np.float32))


def test_self_query_cosine_one_l2_zero():
    x = inputs.unit_rows(64, 768, seed=11)
    eps = 1e-3
    codes, *_ = oracle.quantize(x, eps)
    codes = codes.reshape(x.shape)
    xh = oracle.dequantize(codes, oracle.step(eps))
    cos = oracle.scores(xh, codes, eps, oracle.COSINE)
    assert np.all(np.abs(np.diag(cos) - 1.0) <= 2 ** -23)
    l2 = oracle.scores(xh, codes, eps, oracle.L2)
    assert np.all(np.diag(l2) == 0.0)
    assert np.all(l2[~np.eye(64, dtype=bool)] > 0.5)


def test_margin_constants_match_paper():
    for eps, printed in golden("margin_bound_constants.txt"):
        assert round(2 * float(eps) * math.sqrt(768), 4) == float(printed)


@pytest.mark.parametrize("eps", (1e-3, 1e-2))
def test_score_deviation_within_paper_bound(eps):
    # One vector quantized to within eps per coordinate moves an inner product
    # by at most ||q||_1 eps (Hoelder) <= sqrt(D) eps ||q||_2, i.e. half the
    # pairwise 2 eps sqrt(D) constant the paper prints.
    x = inputs.unit_rows(300, 768, seed=21)
    q = inputs.queries(40, 768, seed=22)
    codes, *_ = oracle.quantize(x, eps)
    codes = codes.reshape(x.shape)
    ip_q = oracle.scores(q, codes, eps, oracle.IP).astype(np.float64)
    ip_x = q.astype(np.float64) @ x.astype(np.float64).T
    l1 = np.abs(q.astype(np.float64)).sum(1)[:, None]
    slack = 1e-6
    assert np.all(np.abs(ip_q - ip_x) <= l1 * eps * (1 + 1e-6) + slack)
    printed = {1e-3: 0.0554, 1e-2: 0.5543}[eps]
    assert np.abs(ip_q - ip_x).max() <= printed / 2 + 1e-4
    # cosine: |cos(q,x) - cos(q,xh)| <= 2 ||x - xh|| / ||x|| <= 2 eps sqrt(D)
    cos_q = oracle.scores(q, codes, eps, oracle.COSINE).astype(np.float64)
    cos_x = ip_x  # unit rows, unit queries
    assert np.abs(cos_q - cos_x).max() <= printed + 1e-4
    # L2: | ||q-x|| - ||q-xh|| | <= ||x - xh|| <= eps sqrt(D)
    l2_q = oracle.scores(q, codes, eps, oracle.L2).astype(np.float64)
    l2_x = ((q.astype(np.float64)[:, None, :] - x.astype(np.float64)[None]) ** 2).sum(-1)
    assert np.abs(np.sqrt(l2_q) - np.sqrt(l2_x)).max() <= printed / 2 + 1e-4


# --- top-k ---------------------------------------------------------------------

def _brute_rank(scores_row, k, ascending):
    n = scores_row.size
    better = np.zeros(n, dtype=np.int64)
    for i in range(n):
        for j in range(n):
            if ascending:
                b = scores_row[j] < scores_row[i] or (scores_row[j] == scores_row[i] and j < i)
            else:
                b = scores_row[j] > scores_row[i] or (scores_row[j] == scores_row[i] and j < i)
            better[i] += b
    order = np.argsort(better)
    return order[:k]


@pytest.mark.parametrize("metric", [oracle.IP, oracle.COSINE, oracle.L2])
def test_topk_brute_force_with_ties(metric):
    rng = np.random.default_rng(metric + 1)
    for n in (1, 2, 7, 33, 64):
        s = rng.integers(-4, 5, size=(3, n)).astype(np.float32) / 4  # many exact ties
        for k in sorted({1, min(3, n), n}):
            got_s, got_i = oracle.topk(s, k, metric)
            for b in range(3):
                want = _brute_rank(s[b], k, ascending=(metric == oracle.L2))
                np.testing.assert_array_equal(got_i[b], want)
                np.testing.assert_array_equal(got_s[b], s[b][want])


def test_topk_direction_and_lowest_index():
    s = np.array([[0.5, 0.9, 0.9, -0.1]], dtype=np.float32)
    _, ids = oracle.topk(s, 3, oracle.IP)
    assert list(ids[0]) == [1, 2, 0]
    _, ids = oracle.topk(s, 3, oracle.L2)
    assert list(ids[0]) == [3, 0, 1]


def test_search_driver_threads_agree():
    x = inputs.unit_rows(500, 64, seed=2)
    q = inputs.queries(5, 64, seed=3)
    codes, *_ = oracle.quantize(x, 1e-2)
    codes = codes.reshape(x.shape)
    for metric in (oracle.IP, oracle.COSINE, oracle.L2):
        full = oracle.scores(q, codes, 1e-2, metric)
        ws, wi = oracle.topk(full, 17, metric)
        for nt in (1, 3, 8):
            gs, gi = oracle.search(q, codes, 1e-2, metric, 17, nthreads=nt)
            np.testing.assert_array_equal(gi, wi)
            np.testing.assert_array_equal(gs, ws)


def test_numpy_rint_cross_check():
    # Not a pin (it restates the formula), but a guard on the C build flags.
    x = inputs.flat_values(1 << 21, seed=9)
    for eps in EPS_SWEEP:
        codes, *_ = oracle.quantize(x, eps)
        s = np.float32(2.0) * np.float32(eps)
        np.testing.assert_array_equal(codes, np.rint(x / s).astype(np.int32))


def test_code_sqnorms_closed_forms_and_invariants():
    # constant rows: D v^2 (the exact integer, rounded once to fp32)
    for D in (1, 7, 768):
        for v in (0, 1, -3, 127, -128, 2048, 32767, -32768):
            got = oracle.code_sqnorms(np.full((1, D), v, dtype=np.int32))[0]
            assert got == np.float32(float(D * v * v))
    # one non-zero coordinate reads back its square wherever it sits
    D = 33
    basis = np.zeros((D, D), dtype=np.int32)
    basis[np.arange(D), np.arange(D)] = np.arange(1, D + 1) * 7
    np.testing.assert_array_equal(oracle.code_sqnorms(basis),
                                  (np.arange(1, D + 1, dtype=np.float32) * 7) ** 2)
    rng = np.random.default_rng(5)
    c = rng.integers(-300, 300, size=(50, 96)).astype(np.int32)
    base = oracle.code_sqnorms(c)
    # sign and coordinate-order invariance
    np.testing.assert_array_equal(oracle.code_sqnorms(-c), base)
    np.testing.assert_array_equal(oracle.code_sqnorms(c[:, rng.permutation(96)]), base)
    # additivity over a split of the coordinates (sums here stay exact in fp32)
    np.testing.assert_array_equal(oracle.code_sqnorms(c[:, :40]) + oracle.code_sqnorms(c[:, 40:]),
                                  base)


def test_code_sqnorms_agree_with_the_l2_score_of_a_zero_query():
    # ||0 - s c||^2 = s^2 sum c^2: the two oracle functions must agree to fp32 rounding
    x = inputs.unit_rows(40, 64, seed=6)
    codes, *_ = oracle.quantize(x, 1e-3)
    codes = codes.reshape(x.shape)
    s = float(oracle.step(1e-3))
    l2 = oracle.scores(np.zeros((1, 64), np.float32), codes, 1e-3, oracle.L2)[0]
    np.testing.assert_allclose(l2, s * s * oracle.code_sqnorms(codes).astype(np.float64),
                               rtol=3e-7)


def test_fnv1a64_published_vectors():
    for text, want in golden("fnv1a64_vectors.txt"):
        data = b"" if text == "-" else text.encode("ascii")
        assert oracle.fnv1a64(data) == int(want, 16), text


def test_band_digests_depend_on_every_code_and_the_band_position():
    rng = np.random.default_rng(12)
    for r, width, (lo, hi) in ((2, 1, (-128, 128)), (4, 2, (-32768, 32768)), (32, 1, (-5, 6)),
                               (8, 4, (-2**31, 2**31))):
        D = 4 * r
        row = rng.integers(lo, hi, size=(1, D)).astype(np.int64).astype(np.int32)
        base = oracle.band_digests(row, r, width)
        assert base.shape == (1, D // r)
        # the same codes in every band still give a different digest per band
        same = np.tile(row[:, :r], (1, D // r))
        dig = oracle.band_digests(same, r, width)[0]
        assert len(set(dig.tolist())) == D // r
        # changing any one coordinate changes only its own band's digest
        for d in range(D):
            mod = row.copy()
            mod[0, d] = mod[0, d] + 1 if mod[0, d] < hi - 1 else mod[0, d] - 1
            got = oracle.band_digests(mod, r, width)[0]
            changed = np.nonzero(got != base[0])[0].tolist()
            assert changed == [d // r], (r, width, d)
        # identical rows share every digest; rows are independent of each other
        two = np.vstack([row, row[:, ::-1]])
        dd = oracle.band_digests(two, r, width)
        np.testing.assert_array_equal(dd[0], base[0])
        np.testing.assert_array_equal(oracle.band_digests(two[1:], r, width)[0], dd[1])


def test_band_digest_of_a_single_band_is_the_fnv_of_its_bytes():
    # one band, one code: the digest is FNV-1a of the two index bytes then the
    # code's little-endian bytes, checked through the published FNV function
    for width, code in ((1, -3), (2, 1234), (4, -70000)):
        got = oracle.band_digests(np.array([[code]], dtype=np.int32), 1, width)[0, 0]
        want = oracle.fnv1a64(int(code).to_bytes(4, "little", signed=True)[:width],
                              oracle.fnv1a64(b"\x00\x00"))
        assert int(got) == want


def test_admit_batch_worked_line_cases():
    for case, delta, pos, reps, dh in golden("admit_line.txt"):
        x = np.array([[float(p), 0.0] for p in pos.split(",")], dtype=np.float32)
        rep, dist, delta_hat, kept = oracle.admit_batch(x, np.zeros((len(x), 1), np.uint64),
                                                        float(delta))
        assert rep.tolist() == [int(v) for v in reps.split(",")], case
        assert abs(delta_hat - float(dh)) < 1e-6, case
        assert kept == len(set(rep.tolist()))


def _lsh_rows(n, seed, dup_every=7):
    x = inputs.unit_rows(n, 64, seed=seed)
    rng = np.random.default_rng(seed)
    for i in range(dup_every, n, dup_every):  # near-duplicates of earlier rows
        j = int(rng.integers(0, i))
        v = x[j] + rng.normal(0, 0.03, size=64).astype(np.float32)
        x[i] = v / np.linalg.norm(v)
    return x


def test_admit_batch_cover_packing_and_lowest_index_with_all_pairs_candidates():
    x = _lsh_rows(300, 21)
    delta = float(np.sqrt(2 - 2 * 0.95))
    rep, dist, dh, kept = oracle.admit_batch(x, np.zeros((300, 1), np.uint64), delta)
    R = np.nonzero(rep == np.arange(300))[0]
    d = np.linalg.norm(x[:, None, :].astype(np.float64) - x[None, :, :], axis=2)
    # cover: every merged row lies within delta of an earlier retained row
    for i in np.nonzero(rep != np.arange(300))[0]:
        assert rep[i] < i and rep[rep[i]] == rep[i] and d[i, rep[i]] <= delta
        # lowest index: no retained row below the representative is within delta
        assert not np.any(d[i, R[R < rep[i]]] <= delta)
    # packing: retained rows are pairwise farther apart than delta (Prop. 2)
    dr = d[np.ix_(R, R)] + np.eye(len(R)) * 10
    assert dr.min() > delta
    assert kept == len(R) and dh == pytest.approx(max(dist.max(), 0.0))


def test_admit_batch_score_deficit_bound_and_prefix_stability():
    x = _lsh_rows(400, 22)
    delta = float(np.sqrt(2 - 2 * 0.9))
    oc, *_ = oracle.quantize(x, 0.05)
    dig = oracle.band_digests(oc.reshape(x.shape), 4, oracle.width(*oracle.quantize(x, 0.05)[1:3]))
    rep, dist, dh, kept = oracle.admit_batch(x, dig, delta)
    R = np.nonzero(rep == np.arange(400))[0]
    # Theorem 1: for unit queries 0 <= max_S q.x - max_R q.z <= delta_hat <= delta
    q = inputs.queries(200, 64, seed=5).astype(np.float64)
    gap = (q @ x.T.astype(np.float64)).max(1) - (q @ x[R].T.astype(np.float64)).max(1)
    assert gap.min() >= 0 and gap.max() <= dh + 1e-12 and dh <= delta
    # decisions are never revised: a prefix decides exactly as in the whole run
    rep_p, *_ = oracle.admit_batch(x[:250], dig[:250], delta)
    np.testing.assert_array_equal(rep_p, rep[:250])


def test_admit_batch_only_band_candidates_merge():
    # two identical rows with no digest in common are not candidates
    x = np.array([[1.0, 0.0], [1.0, 0.0], [1.0, 0.0]], dtype=np.float32)
    dig = np.array([[5], [6], [5]], dtype=np.uint64)
    rep, dist, dh, kept = oracle.admit_batch(x, dig, 0.1)
    assert rep.tolist() == [0, 1, 0] and kept == 2
    # digests match only within the same band position
    dig2 = np.array([[5, 9], [9, 5]], dtype=np.uint64)
    rep, *_ = oracle.admit_batch(x[:2], dig2, 0.1)
    assert rep.tolist() == [0, 1]


def test_lamz_worked_stream():
    for vals, rel, hexs in golden("lamz_small.txt"):
        x = np.array([float(v) for v in vals.split(",")], dtype=np.float32)
        b = oracle.lamz_compress(x, float(rel))
        assert b.hex() == hexs
        np.testing.assert_array_equal(oracle.lamz_decompress(b, x.size), x)


@pytest.mark.parametrize("rel", [1e-3, 1e-2, 3e-2])
def test_lamz_round_trip_is_q_eps_at_the_codec_bound(rel):
    x = inputs.flat_values((1 << 16) + 13, seed=8)  # ragged tail block
    b = oracle.lamz_compress(x, rel)
    y = oracle.lamz_decompress(b, x.size)
    eb = np.float32(rel) * np.abs(x).max()
    # the decoded values are exactly the quantizer's at eps = eb (an
    # independent function: its own division, rounding and dequantisation)
    codes, *_ = oracle.quantize(x, float(eb))
    np.testing.assert_array_equal(y, oracle.dequantize(codes, oracle.step(float(eb))))
    err = np.abs(x.astype(np.float64) - y)
    assert np.all(err <= eb * (1 + 2.0 ** -23) + np.abs(x) * 2.0 ** -23)


def test_lamz_sizes_of_zero_and_constant_inputs():
    n = 1000
    nb = (n + 31) // 32
    head = 16 + (nb + 3) // 4 * 4
    assert len(oracle.lamz_compress(np.zeros(n, np.float32), 0.01)) == head
    # a constant c: one non-zero delta per block, c / s = 1 / (2 rel) = 50
    b = oracle.lamz_compress(np.full(n, 0.37, np.float32), 0.01)
    assert len(b) == head + nb * (4 + 4 * 6)  # |50| needs 6 bits
    y = oracle.lamz_decompress(b, n)
    assert np.all(y == y[0]) and abs(float(y[0]) - 0.37) <= 0.0037
    with pytest.raises(ValueError):
        oracle.lamz_compress(np.array([1.0, np.inf], np.float32), 0.01)
    with pytest.raises(ValueError):
        oracle.lamz_decompress(b[:-4], n)  # truncated


# --- per-vector byte codecs (Sec. "Composite reduction", Table "composite") --

def _row_cases():
    for line in golden("row_codecs_hand.txt"):
        yield line


def test_row_codecs_hand_worked_rows():
    for codec, vals, codes, scale, offset, xhat in _row_cases():
        x = np.array([float(v) for v in vals.split(",")], np.float32)[None, :]
        want = np.array([float(v) for v in xhat.split(",")], np.float32)
        if codec == "int8":
            c, sc, of = oracle.encode_rows(x, oracle.FMT_INT8_ROWS)
            assert c[0].tolist() == [int(v) for v in codes.split(",")]
            assert sc[0] == np.float32(scale) and of[0] == np.float32(offset)
            got = oracle.decode_rows(c, oracle.FMT_INT8_ROWS, x.shape[1], sc, of)
        else:
            c, al, _ = oracle.encode_rows(x, oracle.FMT_SIGN)
            assert c[0].tolist() == [int(codes, 16)]
            assert al[0] == np.float32(scale)
            got = oracle.decode_rows(c, oracle.FMT_SIGN, x.shape[1], al)
        assert np.array_equal(got[0], want)


def test_row_codec_sizes_give_the_papers_ratios():
    # bytes per row: int8 D + two fp32 factors, sign D/8 + one fp32
    D = 768
    x = inputs.unit_rows(3, D, seed=5)
    c, sc, of = oracle.encode_rows(x, oracle.FMT_INT8_ROWS)
    int8_bytes = c[0].nbytes + sc[:1].nbytes + of[:1].nbytes
    b, al, _ = oracle.encode_rows(x, oracle.FMT_SIGN)
    sign_bytes = b[0].nbytes + al[:1].nbytes
    h, _, _ = oracle.encode_rows(x, oracle.FMT_FP16)
    assert round(4 * D / int8_bytes, 2) == 3.96
    assert round(4 * D / sign_bytes, 2) == 30.72
    assert 4 * D / h[0].nbytes == 2.0


def test_fp16_decode_is_exact_for_every_bit_pattern():
    # the C decoder against the IEEE binary16 definition as numpy implements it
    pats = np.arange(1 << 16, dtype=np.uint32).astype(np.uint16)[None, :]
    got = oracle.decode_rows(pats, oracle.FMT_FP16, pats.shape[1])[0]
    want = pats.view(np.float16).astype(np.float32)[0]
    fin = np.isfinite(want)
    assert np.array_equal(got[fin].view(np.uint32), want[fin].view(np.uint32))
    assert np.array_equal(np.isnan(got), np.isnan(want))
    assert np.array_equal(got[np.isinf(want)], want[np.isinf(want)])


def test_int8_rows_error_bound_extremes_and_order():
    x = inputs.unit_rows(64, 96, seed=11)
    c, sc, of = oracle.encode_rows(x, oracle.FMT_INT8_ROWS)
    xh = oracle.decode_rows(c, oracle.FMT_INT8_ROWS, 96, sc, of)
    for i in range(64):
        lo, hi = x[i].min(), x[i].max()
        assert sc[i] == np.float32((hi - lo) / np.float32(255))
        # the row minimum takes code -128 and the maximum 127
        assert c[i][x[i].argmin()] == -128 and c[i][x[i].argmax()] == 127
        # half a step, plus the fp32 roundings of the encode and the decode
        assert np.abs(xh[i] - x[i]).max() <= 0.5 * sc[i] * (1 + 1e-4) + 4e-7
        # codes are monotone in x
        o = np.argsort(x[i], kind="stable")
        assert np.all(np.diff(c[i][o].astype(int)) >= 0)


def test_sign_rows_alpha_is_the_least_squares_scale():
    # for fixed signs b, ||x - a (2b - 1)||^2 is smallest at a = mean |x|
    x = inputs.unit_rows(16, 64, seed=12)
    b, al, _ = oracle.encode_rows(x, oracle.FMT_SIGN)
    xh = oracle.decode_rows(b, oracle.FMT_SIGN, 64, al)
    for i in range(16):
        assert np.array_equal(np.sign(xh[i]), np.where(x[i] >= 0, 1.0, -1.0))
        assert abs(al[i] - np.abs(x[i].astype(np.float64)).mean()) <= 1e-7 * al[i]
        sg = np.sign(xh[i]).astype(np.float64)
        err = lambda a: ((x[i] - a * sg) ** 2).sum()
        assert err(al[i]) <= min(err(al[i] * 1.01), err(al[i] * 0.99))


def test_fp16_rows_are_round_to_nearest():
    x = inputs.unit_rows(8, 64, seed=13)
    h, _, _ = oracle.encode_rows(x, oracle.FMT_FP16)
    xh = oracle.decode_rows(h, oracle.FMT_FP16, 64)
    # no fp16 value lies strictly closer to x than the chosen one
    up = np.nextafter(h, np.float16(np.inf)).astype(np.float32)
    dn = np.nextafter(h, np.float16(-np.inf)).astype(np.float32)
    d = np.abs(xh - x)
    assert np.all(d <= np.abs(up - x)) and np.all(d <= np.abs(dn - x))


def test_row_scores_agree_with_the_code_scores_on_dequantised_rows():
    # Q_eps rows s c are a per-row affine code with offset 0; the fp32-row
    # scorer must reproduce the code scorer (pinned above) on them
    eps = 1e-2
    x = inputs.unit_rows(40, 64, seed=14)
    q = inputs.unit_rows(5, 64, seed=15)
    codes = oracle.quantize(x, eps)[0].reshape(x.shape)
    rows = oracle.dequantize(codes, oracle.step(eps))
    for metric in (oracle.IP, oracle.COSINE, oracle.L2):
        a = oracle.scores_rows(q, rows, metric)
        b = oracle.scores(q, codes, eps, metric)
        np.testing.assert_allclose(a, b, rtol=2e-7, atol=1e-7)


def test_row_scores_closed_forms():
    rows = np.array([[3.0, 4.0], [0.0, 0.0], [-1.0, 0.5]], np.float32)
    q = np.array([[1.0, 2.0]], np.float32)
    ip = oracle.scores_rows(q, rows, oracle.IP)[0]
    cs = oracle.scores_rows(q, rows, oracle.COSINE)[0]
    l2 = oracle.scores_rows(q, rows, oracle.L2)[0]
    assert ip.tolist() == [11.0, 0.0, 0.0]
    assert cs[1] == 0.0 and cs[2] == 0.0
    assert cs[0] == np.float32(11.0 / (5.0 * math.sqrt(5.0)))
    assert l2.tolist() == [8.0, 5.0, 6.25]
