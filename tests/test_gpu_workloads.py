"""The five synthetic workloads at full size, in the launch configuration the
benchmark times: codes bit-exact, and top-k within tolerance of the oracle
(all queries where the oracle finishes in seconds, a seeded sample otherwise)."""
import hashlib

import numpy as np
import pytest
import torch

import oracle
import paper_2609_32256_gb300 as lam
from paper_2609_32256_gb300 import inputs
from tests.parity import NTHREADS, check_topk, oracle_topk, quantize_rows

pytestmark = pytest.mark.gpu
NP_DT = {1: np.int8, 2: np.int16, 4: np.int32}


def digest(a):
    return hashlib.sha256(np.ascontiguousarray(a).tobytes()).hexdigest()


def quantize_checked(x_np, eps, width, dev):
    xt = torch.from_numpy(x_np).to(dev)
    codes, w, scale, cmin, cmax = lam.quantize(xt, eps, width)
    oc, rmin, rmax, _ = oracle.quantize(x_np, eps)
    assert (cmin, cmax) == (int(rmin), int(rmax))
    assert w == (oracle.width(rmin, rmax) if width == 0 else width)
    assert digest(codes.cpu().numpy()) == digest(oc.astype(NP_DT[w]))
    return codes, w, max(-cmin, cmax), oc.reshape(x_np.shape)


def test_pr1_n4096_cosine_int16(dev):
    x = inputs.unit_rows(4096, 768, seed=0)
    q = inputs.queries(16, 768, seed=1)
    codes, w, bound, oc = quantize_checked(x, 1e-3, 2, dev)
    s, i = lam.search(torch.from_numpy(q).to(dev), codes, 1e-3, 10, lam.LAM_METRIC_COSINE, bound)
    os_, oi = oracle_topk(q, oc, 1e-3, oracle.COSINE, 10)
    check_topk(s.cpu().numpy(), i.cpu().numpy(), q, oc, 1e-3, oracle.COSINE, os_, oi)


@pytest.mark.parametrize("eps", [1e-2, 1e-3, 1e-4])
def test_chunks_n27986_planted_ip(dev, eps):
    x = inputs.planted_rows(27986, 768, seed=0)
    q = inputs.queries(1024, 768, seed=1)
    codes, w, bound, oc = quantize_checked(x, eps, 0, dev)
    assert lam.lam_score_topk_path(1024, 27986, 768, 10, w, bound) == lam.PATH_TENSOR
    s, i = lam.search(torch.from_numpy(q).to(dev), codes, eps, 10, lam.LAM_METRIC_IP, bound)
    s, i = s.cpu().numpy(), i.cpu().numpy()
    sel = np.arange(1024) if eps == 1e-3 else np.random.default_rng(7).choice(1024, 128, False)
    os_, oi = oracle_topk(q[sel], oc, eps, oracle.IP, 10)
    check_topk(s[sel], i[sel], q[sel], oc, eps, oracle.IP, os_, oi)


@pytest.mark.parametrize("eps,bound_known", [(1e-4, False), (2e-5, True)])
def test_flat_2p26_rows_int16_tensor(dev, score_path, eps, bound_known):
    """The flat 2^26 values read as 87,381 rows of 768, int16 codes searched on
    the tensor cores: at eps = 2e-5 the codes exceed 2048 (the split 256 h + l
    path), at eps = 1e-4 with no bound given the same split path on small codes."""
    score_path("tensor")
    n = (1 << 26) // 768
    x = inputs.flat_values(1 << 26, seed=0)[: n * 768].reshape(n, 768)
    codes, w, bound, oc = quantize_checked(x, eps, 0, dev)
    assert w == 2 and (bound > 2048) == (eps == 2e-5)
    cb = bound if bound_known else 0
    assert lam.lam_score_topk_path(130, n, 768, 10, 2, cb) == lam.PATH_TENSOR
    q = inputs.queries(130, 768, seed=1)
    sel = np.array([0, 1, 63, 64, 127, 128, 129])
    for metric in (oracle.IP, oracle.L2):
        s, i = lam.search(torch.from_numpy(q).to(dev), codes, eps, 10, metric, cb)
        s, i = s.cpu().numpy(), i.cpu().numpy()
        os_, oi = oracle_topk(q[sel], oc, eps, metric, 10)
        check_topk(s[sel], i[sel], q[sel], oc, eps, metric, os_, oi)


def test_records_n361802_ip_int16(dev):
    x = inputs.unit_rows(361802, 768, seed=0)
    codes, w, bound, oc = quantize_checked(x, 1e-3, 2, dev)
    del x
    for B, sample in ((1, None), (64, None), (4096, 64)):
        q = inputs.queries(B, 768, seed=1)
        s, i = lam.search(torch.from_numpy(q).to(dev), codes, 1e-3, 10, lam.LAM_METRIC_IP, bound)
        s, i = s.cpu().numpy(), i.cpu().numpy()
        sel = np.arange(B) if sample is None else np.random.default_rng(B).choice(B, sample, False)
        os_, oi = oracle_topk(q[sel], oc, 1e-3, oracle.IP, 10)
        check_topk(s[sel], i[sel], q[sel], oc, 1e-3, oracle.IP, os_, oi)


def test_mem_n8388608_l2_int8_slabs(dev):
    """8,388,608 rows drawn and quantized in 1M-row slabs to int8 at eps=1e-2;
    L2 top-100 over the whole resident code matrix.  Every code of every slab
    is compared with the oracle's (SHA-256 of the bytes), and the oracle's own
    codes feed its search: B = 1 and a seeded 32 of the 256 queries."""
    N, D, slab, eps, k = 8388608, 768, 1 << 20, 1e-2, 100
    codes = torch.empty((N, D), dtype=torch.int8, device=dev)
    ws = torch.zeros(lam.lam_quantize_workspace_size(), dtype=torch.uint8, device=dev)
    bound = 0
    ranges = []
    for j in range(N // slab):
        x = inputs.unit_rows_device(slab, D, seed=1000 + j, device=dev)
        st, w, scale, cmin, cmax = lam.lam_quantize(x, eps, 1, codes[j * slab:(j + 1) * slab], ws)
        assert st == 0 and w == 1
        ranges.append((cmin, cmax))
        bound = max(bound, -cmin, cmax)
        del x
    torch.cuda.synchronize()
    q = inputs.queries(256, D, seed=1)
    qt = torch.from_numpy(q).to(dev)
    s1, i1 = lam.search(qt[:1], codes, eps, k, lam.LAM_METRIC_L2, bound)
    s256, i256 = lam.search(qt, codes, eps, k, lam.LAM_METRIC_L2, bound)
    sel = np.sort(np.random.default_rng(3).choice(256, 32, False))
    g_s = np.concatenate([s1.cpu().numpy(), s256.cpu().numpy()[sel]])
    g_i = np.concatenate([i1.cpu().numpy(), i256.cpu().numpy()[sel]])
    qs = np.concatenate([q[:1], q[sel]])
    nq = qs.shape[0]
    # per slab: the oracle quantizes the same fp32 rows (all of them, bit-exact
    # against the GPU codes), searches them with its own codes, and keeps its
    # codes of the rows either side's lists name
    cand_s, cand_i = [], []
    kept = {}
    for j in range(N // slab):
        x = inputs.unit_rows_device(slab, D, seed=1000 + j, device=dev).cpu().numpy()
        oc, rmin, rmax, nnf = quantize_rows(x, eps)
        del x
        assert nnf == 0 and oracle.width(rmin, rmax) == 1
        assert ranges[j] == (int(rmin), int(rmax))
        got = codes[j * slab:(j + 1) * slab].cpu().numpy()
        assert digest(got) == digest(oc.astype(np.int8)), "slab %d codes differ" % j
        del got
        os_, oi = oracle.search(qs, oc, eps, oracle.L2, k, nthreads=NTHREADS)
        cand_s.append(os_)
        cand_i.append(oi + j * slab)
        want = np.union1d(g_i.reshape(-1), (oi + j * slab).reshape(-1))
        want = want[(want >= j * slab) & (want < (j + 1) * slab)]
        for r in want:
            kept[int(r)] = oc[int(r) - j * slab].copy()
        del oc
    cs, ci = np.concatenate(cand_s, 1), np.concatenate(cand_i, 1)
    o_s = np.empty((nq, k), np.float32)
    o_i = np.empty((nq, k), np.int64)
    for b in range(nq):
        order = np.lexsort((ci[b], cs[b]))[:k]
        o_s[b], o_i[b] = cs[b][order], ci[b][order]
    for b in range(nq):
        ids = np.union1d(g_i[b], o_i[b])
        sub = np.stack([kept[int(r)] for r in ids])
        remap = {int(r): n for n, r in enumerate(ids)}
        gi_local = np.array([remap[int(r)] for r in g_i[b]])
        oi_local = np.array([remap[int(r)] for r in o_i[b]])
        # ids are remapped monotonically, so the lower-id tie rule is preserved
        check_topk(g_s[b:b + 1], gi_local[None], qs[b:b + 1], sub, eps, oracle.L2,
                   o_s[b:b + 1], oi_local[None])
