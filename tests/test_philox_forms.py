"""The CUDA path's three Philox4x32-10 forms, built for the host: the plain rounds, the
precomputed round keys, and the folded form of the update (round 0's product given, the
key-only terms of rounds 0..2 precomputed), checked word for word against the oracle's
independent Philox4x32-10 (itself pinned by the published known-answer vectors) on the
counter layout (lo32(q), hi32(q), 0, tag), for every tag, edge counters and keys, and
random ones.  A slip in the folding algebra (a dropped key term, a swapped word) fails
here without a GPU."""
import os
import shutil
import subprocess

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _cuda_include():
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    inc = os.path.join(os.path.dirname(os.path.dirname(os.path.realpath(nvcc))), "include")
    return inc if os.path.exists(os.path.join(inc, "cuda_runtime.h")) else None


@pytest.fixture(scope="module")
def program(tmp_path_factory):
    cxx = shutil.which("g++")
    inc = _cuda_include()
    if not cxx or not inc:
        pytest.skip("g++ or the CUDA headers are not available")
    exe = str(tmp_path_factory.mktemp("philox") / "philox_forms")
    subprocess.run([cxx, "-std=c++17", "-O1", "-Wall", "-I", inc, os.path.join(ROOT, "tests", "philox_forms_main.cpp"),
                    "-o", exe], check=True, capture_output=True, text=True)
    return exe


def test_philox_forms_match_the_oracle(program):
    import oracle
    rng = np.random.default_rng(20)
    keys = [0, 1, 33, 0xFFFFFFFF, 0xFFFFFFFF00000000, 0xFFFFFFFFFFFFFFFF] + \
        [int(v) for v in rng.integers(0, 2**63, 6, dtype=np.uint64)]
    ctrs = [0, 1, 2**31, 2**32 - 1, 2**32, 2**40 + 3, 2**62] + \
        [int(v) for v in rng.integers(0, 2**32, 6, dtype=np.uint64)]
    cases = [(k, c, t) for k in keys for c in ctrs for t in range(5)]
    inp = "".join(f"{k} {c} {t}\n" for k, c, t in cases)
    out = subprocess.run([program], input=inp, capture_output=True, text=True, check=True).stdout.splitlines()
    assert len(out) == len(cases)
    folded_seen = 0
    for (k, c, t), line in zip(cases, out):
        plain, viark, rest = line.split("|")
        ref = oracle.philox4x32_10([c & 0xFFFFFFFF, c >> 32, 0, t], [k & 0xFFFFFFFF, k >> 32])
        assert [int(v) for v in plain.split()] == [int(v) for v in ref], (k, c, t)
        assert [int(v) for v in viark.split()] == [int(v) for v in ref], (k, c, t)
        has, *words = rest.split()
        if c >> 32 == 0:
            assert has == "1" and [int(v) for v in words] == [int(v) for v in ref], (k, c, t)
            folded_seen += 1
    assert folded_seen == len(keys) * 10 * 5
