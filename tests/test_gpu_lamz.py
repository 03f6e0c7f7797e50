"""The error-bounded byte codec on the GPU against the oracle: streams
byte-identical (SHA-256), decoded values bit-exact, ragged tails, the
paper's relative bounds, zero/constant inputs, and the error statuses."""
import hashlib

import numpy as np
import pytest
import torch

import oracle
import paper_2609_32256_gb300 as lam
from paper_2609_32256_gb300 import inputs

pytestmark = pytest.mark.gpu


def compress(dev, x_np, rel, cap=None):
    n = x_np.size
    x = torch.from_numpy(np.ascontiguousarray(x_np.reshape(-1))).to(dev)
    out = torch.zeros(cap if cap is not None else lam.lam_lamz_bound(n), dtype=torch.uint8,
                      device=dev)
    ws = torch.zeros(lam.lam_lamz_workspace_size(n), dtype=torch.uint8, device=dev)
    st, nbytes = lam.lam_lamz_compress(x, rel, out, ws, raise_on_error=False)
    return st, nbytes, out, ws


def decompress(dev, stream_t, nbytes, n, ws):
    out = torch.empty(n, dtype=torch.float32, device=dev)
    st = lam.lam_lamz_decompress(stream_t, nbytes, out, ws, raise_on_error=False)
    return st, out.cpu().numpy()


@pytest.mark.parametrize("rel", [1e-3, 1e-2, 3e-2])
@pytest.mark.parametrize("n", [1, 31, 32, 33, 100003, 1 << 22])
def test_stream_and_decode_bit_exact(dev, rel, n):
    x = inputs.flat_values(n, seed=n % 97)
    want = oracle.lamz_compress(x, rel)
    st, nbytes, out, ws = compress(dev, x, rel)
    assert st == 0 and nbytes == len(want)
    got = out[:nbytes].cpu().numpy().tobytes()
    assert hashlib.sha256(got).hexdigest() == hashlib.sha256(want).hexdigest()
    st, y = decompress(dev, out, nbytes, n, ws)
    assert st == 0
    np.testing.assert_array_equal(y.view(np.uint32), oracle.lamz_decompress(want, n).view(np.uint32))


def test_embedding_rows_and_special_inputs(dev):
    x = inputs.unit_rows(2000, 768, seed=4)
    want = oracle.lamz_compress(x, 1e-2)
    st, nbytes, out, ws = compress(dev, x, 1e-2)
    assert st == 0 and out[:nbytes].cpu().numpy().tobytes() == want
    for x in (np.zeros(1000, np.float32), np.full(1000, -0.25, np.float32)):
        want = oracle.lamz_compress(x, 1e-2)
        st, nbytes, out, ws = compress(dev, x, 1e-2)
        assert st == 0 and out[:nbytes].cpu().numpy().tobytes() == want
        st, y = decompress(dev, out, nbytes, x.size, ws)
        np.testing.assert_array_equal(y, oracle.lamz_decompress(want, x.size))


def test_statuses(dev):
    x = inputs.flat_values(4096, seed=2)
    need = len(oracle.lamz_compress(x, 1e-2))
    st, nbytes, out, ws = compress(dev, x, 1e-2, cap=need - 4)
    assert st == lam.LAM_ERR_WORKSPACE and nbytes == need
    st, nbytes, out, ws = compress(dev, x, 1e-2)
    assert st == 0
    st, _ = decompress(dev, out, nbytes - 4, x.size, ws)  # truncated
    assert st == lam.LAM_ERR_INVALID
    bad = x.copy()
    bad[17] = np.inf
    st, *_ = compress(dev, bad, 1e-2)
    assert st == lam.LAM_ERR_NONFINITE


def test_malformed_streams_write_nothing(dev):
    """The stream is checked on the device before any payload word is read:
    a bad magic, a different n, a bit length above 31 or a payload past the
    end each give LAM_ERR_INVALID and leave the output untouched."""
    x = inputs.flat_values(10000, seed=3)
    st, nbytes, out, ws = compress(dev, x, 1e-2)
    assert st == 0
    good = out[:nbytes].clone()

    def run(stream_t, size, n):
        y = torch.full((n,), 7.0, dtype=torch.float32, device=dev)
        s = lam.lam_lamz_decompress(stream_t, size, y, ws, raise_on_error=False)
        return s, y.cpu().numpy()

    bad = good.clone()
    bad[1] = ord("X")  # magic
    st, y = run(bad, nbytes, x.size)
    assert st == lam.LAM_ERR_INVALID and np.all(y == 7.0)
    ws_big = torch.zeros(lam.lam_lamz_workspace_size(x.size - 5), dtype=torch.uint8, device=dev)
    y = torch.full((x.size - 5,), 7.0, dtype=torch.float32, device=dev)
    st = lam.lam_lamz_decompress(good, nbytes, y, ws_big, raise_on_error=False)  # n differs
    assert st == lam.LAM_ERR_INVALID and np.all(y.cpu().numpy() == 7.0)
    bad = good.clone()
    bad[16 + 5] = 40  # block 5's bit length
    st, y = run(bad, nbytes, x.size)
    assert st == lam.LAM_ERR_INVALID and np.all(y == 7.0)
    st, y = run(good, nbytes - 1, x.size)  # last payload word cut
    assert st == lam.LAM_ERR_INVALID and np.all(y == 7.0)
    st, y = run(good, nbytes, x.size)  # and the intact stream still decodes
    assert st == 0
    np.testing.assert_array_equal(y, oracle.lamz_decompress(good.cpu().numpy().tobytes(),
                                                            x.size))


def test_lookback_budget_runs_out_then_device_recovers(dev, monkeypatch):
    """The compressor's look-back is a bounded wait: with tile 0 publishing
    nothing (a test hook) every later tile's look-back runs out, the call
    returns LAM_ERR_TIMEOUT, and the next ordinary call on the same workspace
    writes the oracle's stream."""
    x_np = inputs.flat_values(100003, seed=9)  # 13 tiles of 256 blocks
    want = oracle.lamz_compress(x_np, 1e-2)
    x = torch.from_numpy(x_np).to(dev)
    out = torch.zeros(lam.lam_lamz_bound(x_np.size), dtype=torch.uint8, device=dev)
    ws = torch.zeros(lam.lam_lamz_workspace_size(x_np.size), dtype=torch.uint8, device=dev)
    monkeypatch.setenv("LAM_TEST_WAIT_CYCLES", "20000")
    monkeypatch.setenv("LAM_TEST_STALL", "1")
    st, _ = lam.lam_lamz_compress(x, 1e-2, out, ws, raise_on_error=False)
    assert st == lam.LAM_ERR_TIMEOUT
    monkeypatch.delenv("LAM_TEST_WAIT_CYCLES")
    monkeypatch.delenv("LAM_TEST_STALL")
    st, nbytes = lam.lam_lamz_compress(x, 1e-2, out, ws, raise_on_error=False)
    assert st == 0 and out[:nbytes].cpu().numpy().tobytes() == want
