"""include/copes.h from plain C: a C99 program compiles against the header alone (no CUDA
or C++ headers), links libcopes.so, and its host helpers agree with the Python binding's
results.  No GPU is needed."""
import os
import shutil
import subprocess

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PKG = os.path.join(ROOT, "paper_2608_02391_gb300")


@pytest.fixture(scope="module")
def program(tmp_path_factory):
    from paper_2608_02391_gb300 import copes
    copes.load()  # builds libcopes.so if it is missing
    if not shutil.which("gcc"):
        pytest.skip("gcc is not available")
    exe = str(tmp_path_factory.mktemp("cabi") / "c_abi_main")
    subprocess.run(["gcc", "-std=c99", "-Wall", "-Werror", "-I", os.path.join(ROOT, "include"),
                    os.path.join(ROOT, "tests", "c_abi_main.c"), "-L", PKG, "-lcopes",
                    "-Wl,-rpath," + PKG, "-o", exe], check=True, capture_output=True, text=True)
    out = subprocess.run([exe], check=True, capture_output=True, text=True).stdout
    return dict(line.split(" ", 1) for line in out.strip().splitlines())


def test_c_program_agrees_with_the_binding(program):
    from paper_2608_02391_gb300 import copes
    assert program["version"] == copes.version()
    layout = copes.Layout([1000, 7, 130])
    assert [int(v) for v in program["offsets"].split()] == [int(v) for v in layout.offsets]
    nid, sign, P = copes.member_table(6, copes.ANTITHETIC)
    got = program["members"].split()
    assert int(got[0]) == P == 3
    assert got[1:] == [f"{int(n)}:{int(s)}" for n, s in zip(nid, sign)]
    assert int(program["seed"]) == int(copes.member_seeds(33, 2, 1, 6)[5])
    assert float(program["sigma"]) == copes.sigma_eff(1e-3, 4000, 1000, True) == 2e-3
    assert np.isclose(float(program["coef"]), 5e-4 / (32 * 1e-3), rtol=0, atol=1e-18)
    code, msg = program["error"].split(" ", 1)
    assert int(code) == copes.ERR_INVALID_ARG and "antithetic" in msg
