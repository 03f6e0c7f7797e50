"""Batch admission (Algorithm 2) on the GPU against the oracle: band
candidates from the fused Q_eps + digest pass, full-precision l2
verification, greedy first-occurrence representatives, delta_hat and |R|,
all bit-exact; hand-worked line cases; the candidate-pair overflow status."""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_32256_gb300 as lam
from paper_2609_32256_gb300 import inputs
from tests.conftest import golden

pytestmark = pytest.mark.gpu
SIGMA = 1.0 / np.sqrt(768.0)


def near_dup_rows(n, d, seed, every=5, noise=0.005):
    x = inputs.unit_rows(n, d, seed=seed)
    rng = np.random.default_rng(seed + 1)
    for i in range(every, n, every):
        j = int(rng.integers(0, i))
        v = x[j] + rng.normal(0, noise, size=d).astype(np.float32)
        x[i] = v / np.linalg.norm(v)
    return x


def gpu_admit(dev, x, dig, delta, max_pairs=1 << 22):
    N = x.shape[0]
    xt = torch.from_numpy(np.ascontiguousarray(x)).to(dev)
    dt = torch.from_numpy(np.ascontiguousarray(dig).view(np.int64)).to(dev)
    rep = torch.empty(N, dtype=torch.int32, device=dev)
    dist = torch.empty(N, dtype=torch.float64, device=dev)
    ws = torch.empty(lam.lam_admit_batch_workspace_size(N, dig.shape[1], max_pairs),
                     dtype=torch.uint8, device=dev)
    st, dh, kept, npairs = lam.lam_admit_batch(xt, dt, delta, rep, dist, ws, max_pairs,
                                               raise_on_error=False)
    return st, rep.cpu().numpy(), dist.cpu().numpy(), dh, kept, npairs


def gpu_digests(dev, x, eps, r):
    N, D = x.shape
    dig = torch.empty((N, D // r), dtype=torch.int64, device=dev)
    ws = torch.zeros(lam.lam_quantize_workspace_size(), dtype=torch.uint8, device=dev)
    lam.lam_quantize_bands(torch.from_numpy(x).to(dev), eps, 0, r, None, dig, ws)
    return dig.cpu().numpy().view(np.uint64)


@pytest.mark.parametrize("t", [0.95, 0.99])
@pytest.mark.parametrize("n,r,rel", [(2000, 4, 0.2), (2000, 8, 0.3), (27986, 8, 0.3),
                                     (27986, 16, 0.2)])
def test_admission_matches_the_oracle(dev, t, n, r, rel):
    # (at r = 4 unrelated unit rows already share a band with probability
    # ~3%, so 27,986 rows give ~10^7 candidate pairs: kept to the small case)
    x = near_dup_rows(n, 768, seed=n + r)
    eps = rel * SIGMA
    dig = gpu_digests(dev, x, eps, r)
    oc, rmin, rmax, _ = oracle.quantize(x, eps)
    np.testing.assert_array_equal(dig, oracle.band_digests(oc.reshape(x.shape), r,
                                                           oracle.width(rmin, rmax)))
    delta = float(np.sqrt(2.0 - 2.0 * t))
    o_rep, o_dist, o_dh, o_kept = oracle.admit_batch(x, dig, delta)
    st, rep, dist, dh, kept, npairs = gpu_admit(dev, x, dig, delta)
    assert st == 0
    np.testing.assert_array_equal(rep, o_rep)
    np.testing.assert_array_equal(dist.view(np.uint64), o_dist.view(np.uint64))
    assert dh == o_dh and kept == o_kept
    assert kept < n  # the planted near-duplicates merge


def test_worked_line_cases(dev):
    for case, delta, pos, reps, dh in golden("admit_line.txt"):
        x = np.array([[float(p), 0.0] for p in pos.split(",")], dtype=np.float32)
        st, rep, dist, got_dh, kept, _ = gpu_admit(dev, x, np.zeros((len(x), 1), np.uint64),
                                                   float(delta))
        assert st == 0 and rep.tolist() == [int(v) for v in reps.split(",")], case
        assert abs(got_dh - float(dh)) < 1e-6, case


def test_candidate_pair_overflow_is_reported(dev):
    x = near_dup_rows(300, 64, seed=3)
    dig = np.zeros((300, 2), np.uint64)  # every pair shares both bands: 2 * 300 * 299 / 2
    st, *_, npairs = gpu_admit(dev, x, dig, 0.3, max_pairs=1000)
    assert st == lam.LAM_ERR_WORKSPACE and npairs == 300 * 299
    st, rep, *_ = gpu_admit(dev, x, dig, 0.3, max_pairs=300 * 299)
    assert st == 0
    o_rep, *_ = oracle.admit_batch(x, dig, 0.3)
    np.testing.assert_array_equal(rep, o_rep)
