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
from tests.parity import NTHREADS, check_topk, oracle_topk

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
    L2 top-100 over the whole resident code matrix."""
    N, D, slab, eps, k = 8388608, 768, 1 << 20, 1e-2, 100
    codes = torch.empty((N, D), dtype=torch.int8, device=dev)
    ws = torch.zeros(lam.lam_quantize_workspace_size(), dtype=torch.uint8, device=dev)
    rng = np.random.default_rng(11)
    bound = 0
    for j in range(N // slab):
        x = inputs.unit_rows_device(slab, D, seed=1000 + j, device=dev)
        st, w, scale, cmin, cmax = lam.lam_quantize(x, eps, 1, codes[j * slab:(j + 1) * slab], ws)
        bound = max(bound, -cmin, cmax)
        rows = rng.choice(slab, 256, replace=False)
        xs = x[torch.from_numpy(rows).to(dev)].cpu().numpy()
        oc, *_ = oracle.quantize(xs, eps)
        got = codes[j * slab + torch.from_numpy(rows).to(dev)].cpu().numpy().reshape(-1)
        assert digest(got) == digest(oc.astype(np.int8))
        del x
    torch.cuda.synchronize()
    q = inputs.queries(256, D, seed=1)
    qt = torch.from_numpy(q).to(dev)
    s1, i1 = lam.search(qt[:1], codes, eps, k, lam.LAM_METRIC_L2, bound)
    s256, i256 = lam.search(qt, codes, eps, k, lam.LAM_METRIC_L2, bound)
    sel = np.concatenate([[0], np.random.default_rng(3).choice(np.arange(1, 256), 7, False)])
    g_s = np.concatenate([s1.cpu().numpy(), s256.cpu().numpy()[sel]])
    g_i = np.concatenate([i1.cpu().numpy(), i256.cpu().numpy()[sel]])
    qs = np.concatenate([q[:1], q[sel]])
    # oracle: top-k of every slab, then the k best of their union (same rule)
    cand_s, cand_i = [], []
    for j in range(N // slab):
        oc = codes[j * slab:(j + 1) * slab].cpu().numpy().astype(np.int32)
        os_, oi = oracle.search(qs, oc, eps, oracle.L2, k, nthreads=NTHREADS)
        cand_s.append(os_)
        cand_i.append(oi + j * slab)
    cs, ci = np.concatenate(cand_s, 1), np.concatenate(cand_i, 1)
    o_s = np.empty((qs.shape[0], k), np.float32)
    o_i = np.empty((qs.shape[0], k), np.int64)
    for b in range(qs.shape[0]):
        order = np.lexsort((ci[b], cs[b]))[:k]
        o_s[b], o_i[b] = cs[b][order], ci[b][order]
    # the checker needs the codes of the GPU ids: gather them per query
    for b in range(qs.shape[0]):
        ids = np.union1d(g_i[b], o_i[b])
        sub = codes[torch.from_numpy(ids).to(dev)].cpu().numpy().astype(np.int32)
        remap = {int(r): n for n, r in enumerate(ids)}
        gi_local = np.array([remap[int(r)] for r in g_i[b]])
        oi_local = np.array([remap[int(r)] for r in o_i[b]])
        # ids are remapped monotonically, so the lower-id tie rule is preserved
        check_topk(g_s[b:b + 1], gi_local[None], qs[b:b + 1], sub, eps, oracle.L2,
                   o_s[b:b + 1], oi_local[None])
