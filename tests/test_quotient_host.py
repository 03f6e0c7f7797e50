"""Host check of the quotient scheme of the quantize kernels: the reciprocal
RN(1/s) and two fused multiply-add refinements give the IEEE-rounded single
quotient x / s (Markstein's theorem), on random fp32 values of every magnitude
and values next to the quotient midpoints (k + 1/2) s where the code is
decided; the plain reciprocal product fails the same check.  (The kernels
themselves are compared with the oracle on the GPU.)"""
import os
import shutil
import subprocess

import pytest

HERE = os.path.dirname(os.path.abspath(__file__))


def run_check(tmp_path, *defines, samples=1 << 20):
    if shutil.which("gcc") is None:
        pytest.skip("gcc not found")
    exe = str(tmp_path / "fqc")
    subprocess.run(["gcc", "-std=c99", "-O2", "-ffp-contract=off", *defines, "-o", exe,
                    os.path.join(HERE, "fma_quotient_check.c"), "-lm"], check=True)
    out = subprocess.run([exe, str(samples)], capture_output=True, text=True, check=True)
    checked, bad_q, bad_c = (int(v) for v in out.stdout.split())
    return checked, bad_q, bad_c


def test_fma_quotient_equals_ieee_division(tmp_path):
    checked, bad_q, bad_c = run_check(tmp_path)
    assert checked > 8_000_000
    assert bad_q == 0 and bad_c == 0


def test_plain_reciprocal_product_is_caught(tmp_path):
    _, bad_q, bad_c = run_check(tmp_path, "-DNO_REFINE", samples=1 << 16)
    assert bad_q > 0 and bad_c > 0
