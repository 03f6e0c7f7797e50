import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")


def golden(name):
    """Rows of a whitespace-separated fixture under tests/golden (comments skipped)."""
    rows = []
    with open(os.path.join(ROOT, "tests", "golden", name)) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            rows.append(line.split())
    return rows


@pytest.fixture(scope="session")
def dev():
    """cuda:0 with the library built and loaded (GPU tests only)."""
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_32256_gb300 import build as lam_build
    lam_build.build()
    import paper_2609_32256_gb300 as lam
    lam.load()
    return torch.device("cuda:0")


@pytest.fixture
def score_path(monkeypatch):
    """Force one kernel path of lam_score_topk for the duration of a test."""
    def force(name):
        monkeypatch.setenv("LAM_SCORE_PATH", name)
    return force


def pytest_terminal_summary(terminalreporter):
    """Prints, per parity test, the largest |gpu - oracle| / tolerance of its
    scores (1.0 would be at the tolerance)."""
    try:
        from tests.parity import WORST
    except Exception:
        return
    if not WORST:
        return
    tr = terminalreporter
    tr.section("score margin: max |gpu - oracle| / (1e-6 + 1e-5 |oracle|) per test")
    for name, r in sorted(WORST.items(), key=lambda kv: -kv[1]):
        tr.write_line("%8.4f  %s" % (r, name))
