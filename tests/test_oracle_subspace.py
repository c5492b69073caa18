"""Pins for the oracle's parameter layout and subspace builds (CPU only).

Eq. 7 asks for disjoint, covering subspaces of equal size; the builds are checked for
exactly that, for sizes given by closed forms, and (hash / random chunks) against the
independent big-int Philox and numpy's sort.
"""
import numpy as np
import pytest

import oracle
import philox_bigint
from paper_2608_02391_gb300 import workloads as wl


def _members(ranges):
    out = []
    for b, e in ranges:
        out.extend(range(b, e))
    return out


def _real_indices(numel):
    off = oracle.layout(numel)
    s = set()
    for t, n in enumerate(numel):
        s.update(range(int(off[t]), int(off[t]) + int(n)))
    return s


ODD_LAYOUT = [1000, 64, 7, 4096, 130, 1, 2500]  # numels that force padding


def test_layout_offsets_are_64_aligned_and_padded():
    off = oracle.layout(ODD_LAYOUT)
    assert off[0] == 0
    for t, n in enumerate(ODD_LAYOUT):
        assert off[t] % 64 == 0
        assert off[t + 1] - off[t] == (n + 63) // 64 * 64
    assert list(off) == wl.layout_offsets([wl.Tensor(str(i), n, "x") for i, n in enumerate(ODD_LAYOUT)])


@pytest.mark.parametrize("K", [1, 3, 4, 7])
def test_contiguous_partition(K):
    real = _real_indices(ODD_LAYOUT)
    n = len(real)
    seen = set()
    order = sorted(real)
    for k in range(K):
        rs = oracle.contiguous_ranges(ODD_LAYOUT, K, k)
        m = _members(rs)
        assert m == sorted(m)
        assert len(m) == (n * (k + 1)) // K - (n * k) // K
        assert m == order[(n * k) // K:(n * (k + 1)) // K]
        assert not (seen & set(m))
        seen |= set(m)
        for a, b in zip(rs, rs[1:]):
            assert a[1] < b[0]  # merged: no two ranges touch
    assert seen == real


def test_group_ranges_union_of_tensors():
    off = oracle.layout(ODD_LAYOUT)
    groups = [0, 1, 1, 0, 2, 2, 1]
    seen = set()
    for k in range(3):
        m = set(_members(oracle.group_ranges(ODD_LAYOUT, groups, k)))
        expect = set()
        for t, g in enumerate(groups):
            if g == k:
                expect |= set(range(int(off[t]), int(off[t]) + ODD_LAYOUT[t]))
        assert m == expect
        assert not (seen & m)
        seen |= m
    assert seen == _real_indices(ODD_LAYOUT)


def test_hash_partition_properties():
    numel = [5000, 333, 12000, 64, 4099]
    tids = [0, 1, 2, 3, 4]
    K, seed = 16, 1088
    off = oracle.layout(numel)
    lists = [oracle.hash_list(numel, tids, K, seed, k) for k in range(K)]
    allidx = np.concatenate(lists)
    assert allidx.size == sum(numel)
    assert len(set(allidx.tolist())) == allidx.size
    assert set(allidx.tolist()) == _real_indices(numel)
    n = sum(numel)
    for lst in lists:
        assert np.all(np.diff(lst) > 0)
        sd = np.sqrt(n * (1 / K) * (1 - 1 / K))
        assert abs(lst.size - n / K) < 5 * sd
    # membership from the independent big-int Philox for sampled elements
    rng = np.random.default_rng(0)
    for _ in range(200):
        t = int(rng.integers(0, len(numel)))
        e = int(rng.integers(0, numel[t]))
        x = philox_bigint.words(seed, e >> 2, aux=tids[t], tag=oracle.TAG_PARTITION)[e & 3]
        k = (x * K) >> 32
        assert oracle.hash_subspace(seed, tids[t], e, K) == k
        assert int(off[t]) + e in set(lists[k].tolist())


def test_random_chunks_equal_sizes_and_replay():
    for n_chunks, K in [(1, 1), (10, 4), (61, 8), (1000, 16)]:
        seed = 1088 + n_chunks
        cs = oracle.random_chunks(n_chunks, K, seed)
        counts = np.bincount(cs, minlength=K)
        assert counts.sum() == n_chunks
        assert counts.max() - counts.min() <= 1
        # the same map from numpy's lexsort of keys drawn with the big-int Philox
        keys = np.array([philox_bigint.words(seed, c, tag=oracle.TAG_CHUNK)[0] for c in range(n_chunks)],
                        dtype=np.uint64)
        order = np.lexsort((np.arange(n_chunks), keys))
        ref = np.zeros(n_chunks, np.uint32)
        ref[order] = (np.arange(n_chunks) * K) // n_chunks
        assert np.array_equal(cs, ref)
        assert np.array_equal(cs, oracle.random_chunks(n_chunks, K, seed))  # replay


def test_chunk_ranges_cover_real_elements_once():
    numel = ODD_LAYOUT
    chunk = 256
    d_pad = int(oracle.layout(numel)[-1])
    n_chunks = (d_pad + chunk - 1) // chunk
    K = 3
    cs = oracle.random_chunks(n_chunks, K, 5)
    seen = set()
    for k in range(K):
        m = set(_members(oracle.chunk_ranges(numel, chunk, cs, k)))
        for g in m:
            assert cs[g // chunk] == k
        assert not (seen & m)
        seen |= m
    assert seen == _real_indices(numel)


def test_workload_parameter_counts():
    assert wl.workload("tiny").d == 1_048_576
    assert wl.workload("0.5b").d == 494_032_768
    assert wl.workload("4b").d == 4_022_468_096
    assert wl.workload("8b").d == 8_190_735_360
    for name in ("0.5b", "4b", "8b"):
        w = wl.workload(name)
        assert w.d_pad == w.d  # every tensor size is a multiple of 64: no padding


def test_workload_groupings():
    w8 = wl.workload("8b")
    sizes = np.bincount(w8.group_of, weights=w8.numel).astype(np.int64)
    assert list(sizes) == [1_509_949_440, 5_435_817_984, 622_638_080, 622_329_856]
    w4 = wl.workload("4b")
    layers = [t.layer for t in w4.tensors]
    blocks = {}
    for g, l in zip(w4.group_of, layers):
        if l >= 0:
            blocks.setdefault(g, set()).add(l)
    assert [len(blocks[k]) for k in range(8)] == [4, 5, 4, 5, 4, 5, 4, 5]
    for k in range(8):  # layer blocks are contiguous in the layout: one range each
        assert len(oracle.group_ranges(w4.numel, w4.group_of, k)) == 1
    w05 = wl.workload("0.5b")
    blocks = {}
    for g, l in zip(w05.group_of, [t.layer for t in w05.tensors]):
        if l >= 0:
            blocks.setdefault(g, set()).add(l)
    assert [len(blocks[k]) for k in range(1, 8)] == [3, 3, 4, 3, 4, 3, 4]
    assert len(oracle.group_ranges(w05.numel, w05.group_of, 0)) == 2  # embedding + final norm
