"""The hash partition that allocates nothing (copes_hash_partition_static).

Callers that cannot allocate device scratch use this entry point, for example a trainer
sharing the GPU with a rollout engine that reserved nearly all free HBM for its KV
cache. It builds the same sorted index lists as copes_hash_count + copes_hash_fill on a
fixed scratch array inside the library. Index lists are integers, so its output must
equal the workspace version's bit for bit, call after call: the scratch is reused and
keeps the previous call's contents.
"""
import ctypes

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu

NUMEL = [50_000, 333, 16_384, 16_385, 64, 40_000, 7]
TENSOR_IDS = [10, 11, 12, 13, 14, 15, 16]


@pytest.fixture(scope="module")
def copes():
    from paper_2608_02391_gb300 import copes as c
    c.load()
    return c


def _static_call(copes, layout, K, seed, lists=None, capacity=None):
    lib = copes.load()
    counts = np.zeros(K, np.uint64)
    ptrs = None if lists is None else (ctypes.c_void_p * K)(*[t.data_ptr() for t in lists])
    caps = None if capacity is None else np.ascontiguousarray(capacity, np.uint64)
    rc = lib.copes_hash_partition_static(ctypes.byref(layout.desc), K, seed, ptrs,
                                         None if caps is None else caps.ctypes.data_as(ctypes.c_void_p),
                                         counts.ctypes.data_as(ctypes.c_void_p),
                                         ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    return rc, counts


@pytest.mark.parametrize("K,seed", [(16, 1088), (5, 7)])
def test_static_scratch_matches_workspace_version_twice(copes, K, seed):
    layout = copes.Layout(NUMEL, TENSOR_IDS)
    ref = copes.hash_partition(layout, K, seed)  # workspace version
    ref_counts = np.array([s.numel for s in ref], np.uint64)
    rc, counts = _static_call(copes, layout, K, seed)  # count only
    assert rc == copes.OK, copes.last_error()
    assert np.array_equal(counts, ref_counts)
    for _ in range(2):  # the second call starts from the first call's scratch contents
        lists = [torch.full((max(int(c), 1),), -1, dtype=torch.int64, device="cuda") for c in ref_counts]
        rc, counts = _static_call(copes, layout, K, seed, lists, ref_counts)
        assert rc == copes.OK, copes.last_error()
        torch.cuda.synchronize()
        assert np.array_equal(counts, ref_counts)
        for k in range(K):
            assert torch.equal(lists[k][:int(ref_counts[k])], ref[k].tensor), k
    copes.check()


def test_static_scratch_lists_match_the_oracle(copes):
    """The static entry point's lists against the oracle's hash partition (Eq. 7: element
    e of tensor tid goes to subspace floor(x K / 2^32), x its partition Philox word),
    on a fresh scratch state and after another partition reused it."""
    import oracle
    layout = copes.Layout(NUMEL, TENSOR_IDS)
    for K, seed in ((3, 21), (8, 1088)):
        subs = copes.hash_partition_static(layout, K, seed)
        torch.cuda.synchronize()
        for k in range(K):
            ref = oracle.hash_list(NUMEL, TENSOR_IDS, K, seed, k)
            assert np.array_equal(subs[k].tensor.cpu().numpy(), ref), (K, k)
    copes.check()


def test_static_scratch_rejects_oversize_and_short_lists(copes):
    big = copes.Layout([1 << 31, 1 << 31])  # needs far more than the fixed scratch
    rc, _ = _static_call(copes, big, 16, 1)
    assert rc == copes.ERR_SIZE and "static" in copes.last_error()
    layout = copes.Layout(NUMEL, TENSOR_IDS)
    rc, counts = _static_call(copes, layout, 4, 3)
    assert rc == copes.OK
    short = [torch.empty(max(int(c) - 1, 1), dtype=torch.int64, device="cuda") for c in counts]
    rc, _ = _static_call(copes, layout, 4, 3, short, [t.numel() for t in short])
    assert rc == copes.ERR_WORKSPACE
