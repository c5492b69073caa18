"""One ES visit driven from plain C: tests/c_abi_visit.c allocates with cudaMalloc and
calls only include/copes.h -- copes_subspace_build, N x copes_perturb,
copes_perturb_two_pairs on four working copies, copes_restore, copes_shape_fitness,
copes_update (fuse_commit = 0) and copes_context_commit -- on a 3-tensor layout; its
dumps are checked here against the oracle (Sec. 3.2, Eq. 8, Eq. 5, Eq. 13) at the
tolerances of tests/tolerances.py."""
import os
import shutil
import subprocess

import numpy as np
import pytest

from tolerances import assert_bf16_close, assert_fitness_close, assert_update_close

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PKG = os.path.join(ROOT, "paper_2608_02391_gb300")
NUMEL = [300001, 4099, 150000]
K, k, N, SIGMA = 3, 1, 8, 1e-3


def _cuda_home():
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    return os.path.dirname(os.path.dirname(os.path.realpath(nvcc)))


@pytest.fixture(scope="module")
def visit(tmp_path_factory):
    from paper_2608_02391_gb300 import copes
    copes.load()
    if not shutil.which("gcc"):
        pytest.skip("gcc is not available")
    cuda = _cuda_home()
    lib64 = os.path.join(cuda, "lib64")
    out = tmp_path_factory.mktemp("cvisit")
    exe = str(out / "c_abi_visit")
    subprocess.run(["gcc", "-std=c99", "-Wall", "-Werror", "-I", os.path.join(ROOT, "include"),
                    "-I", os.path.join(cuda, "include"), os.path.join(ROOT, "tests", "c_abi_visit.c"),
                    "-L", PKG, "-lcopes", "-L", lib64, "-lcudart", "-lm",
                    "-Wl,-rpath," + PKG, "-Wl,-rpath," + lib64, "-o", exe],
                   check=True, capture_output=True, text=True)
    res = subprocess.run([exe, str(out)], capture_output=True, text=True, timeout=600)
    assert res.returncode == 0, res.stderr
    lines = dict(line.split(" ", 1) for line in res.stdout.strip().splitlines())
    n = int(lines["n_alloc"])
    load = lambda name, dt: np.fromfile(out / name, dtype=dt)
    d = {name: load(name + ".bin", dt) for name, dt in [
        ("theta", np.float32), ("rewards", np.float32), ("fitness", np.float32), ("master_after", np.float32),
        ("w_member0", np.uint16), ("w_member1", np.uint16), ("w_restored", np.uint16),
        ("w_before_commit", np.uint16), ("w_after", np.uint16), ("tiles", np.uint64),
        *[(f"w_two_pairs{c}", np.uint16) for c in range(4)]]}
    d.update(n=n, P=int(lines["P"]), seeds=np.array(lines["seeds"].split(), dtype=np.uint64),
             coef=np.float32(float(lines["coef"])))
    assert all(d[x].size == n for x in ("theta", "master_after", "w_after"))
    return d


def _subspace(oracle):
    """S's global-index ranges (the contiguous cut crosses from tensor 0 into tensor 1),
    its indices g and a membership mask over the arena."""
    ranges = oracle.contiguous_ranges(NUMEL, K, k)
    g = np.concatenate([np.arange(b, e, dtype=np.uint64) for b, e in ranges])
    n = int(oracle.layout(NUMEL)[-1])
    inside = np.zeros(n, dtype=bool)
    inside[g.astype(np.int64)] = True
    return ranges, g, inside


def test_subspace_and_members_from_c(visit):
    import oracle
    from paper_2608_02391_gb300 import copes
    ranges, _, _ = _subspace(oracle)
    assert len(ranges) == 2  # the cut crosses a tensor boundary and its padding
    expected = [(s, min(s + 4096, e)) for b, e in ranges for s in range(b, e, 4096)]
    assert [tuple(int(v) for v in t) for t in visit["tiles"].reshape(-1, 2)] == expected
    assert visit["n"] == int(oracle.layout(NUMEL)[-1])
    assert visit["P"] == N // 2
    assert [int(s) for s in visit["seeds"]] == [oracle.member_seed(33, 0, k, j) for j in range(N // 2)]
    # the C program passes sigma as the fp32 value 1e-3f
    assert np.float32(copes.step_coef(5e-4, N, float(np.float32(SIGMA)), copes.COEF_OPENAI)) == visit["coef"]


def test_perturb_and_restore_from_c(visit):
    import oracle
    _, g, inside = _subspace(oracle)
    gi = g.astype(np.int64)
    theta = visit["theta"]
    context = oracle.bf16_bits_array(theta)
    nid, sign = oracle.member_table(N, 1)[:2]
    for i in (0, 1):
        seed, s = int(visit["seeds"][nid[i]]), float(sign[i]) * SIGMA
        ref, _ = oracle.perturb_at(g, theta[gi], seed, s, oracle.BF16)
        scale = np.maximum(np.abs(theta[gi]), np.abs(np.float32(SIGMA) * oracle.noise(seed, g)))
        got = visit[f"w_member{i}"]
        assert_bf16_close(got[gi], ref.astype(np.uint16), scale)
        # outside S (other subspaces and the layout's padding) the context is untouched
        assert np.array_equal(got[~inside], context[~inside])
    assert np.array_equal(visit["w_restored"], context)


def test_shaping_update_and_commit_from_c(visit):
    import oracle
    _, g, inside = _subspace(oracle)
    gi = g.astype(np.int64)
    theta, after = visit["theta"], visit["master_after"]
    f_ref = oracle.shape_fitness(visit["rewards"], oracle.SHAPE_ZSCORE)
    assert_fitness_close(visit["fitness"], f_ref)
    nid, sign, P = oracle.member_table(N, 1)
    wj = oracle.noise_weights(nid, sign, f_ref, P)
    _, exact, scale = oracle.update_at(g, theta[gi], visit["seeds"], wj, visit["coef"])
    assert_update_close(after[gi], exact, scale)
    # outside S the master keeps its bits; without the fused commit the update left w alone
    assert np.array_equal(after[~inside].view(np.uint32), theta[~inside].view(np.uint32))
    assert np.array_equal(visit["w_before_commit"], visit["w_restored"])
    # the commit published round(theta) of the new master
    assert np.array_equal(visit["w_after"], oracle.bf16_bits_array(after))


def test_two_pairs_from_c(visit):
    """copes_perturb_two_pairs from C: copies 0 and 1 equal the plain perturbs of members 0
    and 1 bit for bit, copies 2 and 3 (members 2 and 3) agree with the oracle on S, and
    outside S every copy holds the committed context."""
    import oracle
    _, g, inside = _subspace(oracle)
    gi = g.astype(np.int64)
    theta = visit["theta"]
    context = oracle.bf16_bits_array(theta)
    assert np.array_equal(visit["w_two_pairs0"], visit["w_member0"])
    assert np.array_equal(visit["w_two_pairs1"], visit["w_member1"])
    nid, sign = oracle.member_table(N, 1)[:2]
    for i in (2, 3):
        seed, s = int(visit["seeds"][nid[i]]), float(sign[i]) * SIGMA
        ref, _ = oracle.perturb_at(g, theta[gi], seed, s, oracle.BF16)
        scale = np.maximum(np.abs(theta[gi]), np.abs(np.float32(SIGMA) * oracle.noise(seed, g)))
        got = visit[f"w_two_pairs{i}"]
        assert_bf16_close(got[gi], ref.astype(np.uint16), scale)
        assert np.array_equal(got[~inside], context[~inside])
