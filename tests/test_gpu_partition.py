"""GPU-vs-oracle parity of the subspace builds: tile tables of the range modes, the
random-chunk map and the hash partition's sorted index lists, all bit-exact."""
import numpy as np
import pytest
import torch

import oracle

pytestmark = pytest.mark.gpu

ODD_LAYOUT = [1000, 64, 7, 4096, 130, 1, 2500, 70_000, 33]


@pytest.fixture(scope="module")
def copes():
    from paper_2608_02391_gb300 import copes as c
    c.load()
    return c


def tiles_to_ranges(sub):
    t = sub.tensor.cpu().numpy().astype(np.uint64)
    out = []
    for b, e in t:
        if out and out[-1][1] == int(b):
            out[-1] = (out[-1][0], int(e))
        else:
            out.append((int(b), int(e)))
    return out


def check_tiles(sub, ranges, tile):
    t = sub.tensor.cpu().numpy()
    assert np.all(t[:, 1] - t[:, 0] <= tile) and np.all(t[:, 1] > t[:, 0])
    assert tiles_to_ranges(sub) == ranges


@pytest.mark.parametrize("K", [1, 3, 4, 8])
@pytest.mark.parametrize("tile", [64, 1000, 1 << 14])
def test_contiguous_tiles(copes, K, tile):
    L = copes.Layout(ODD_LAYOUT)
    for k in range(K):
        sub = copes.subspace_build(L, copes.PART_CONTIGUOUS, K, k, tile_size=tile)
        check_tiles(sub, oracle.contiguous_ranges(ODD_LAYOUT, K, k), tile)


def test_group_tiles(copes):
    L = copes.Layout(ODD_LAYOUT)
    groups = [0, 1, 1, 0, 2, 2, 1, 2, 0]
    for k in range(3):
        sub = copes.subspace_build(L, copes.PART_TENSOR_GROUPS, 3, k, group_of=groups, tile_size=512)
        check_tiles(sub, oracle.group_ranges(ODD_LAYOUT, groups, k), 512)


@pytest.mark.parametrize("n_chunks,K", [(1, 1), (10, 4), (61, 8), (3000, 16), (4096, 3), (4097, 5),
                                         (8192, 64), (70_000, 7), (1 << 20, 13)])
def test_random_chunk_map(copes, n_chunks, K):
    seed = 1088 + n_chunks
    got = copes.random_chunk_map(n_chunks, K, seed).cpu().numpy().view(np.uint32)
    assert np.array_equal(got, oracle.random_chunks(n_chunks, K, seed))


def test_random_chunk_tiles(copes):
    L = copes.Layout(ODD_LAYOUT)
    chunk, K = 256, 5
    n_chunks = (L.d_pad + chunk - 1) // chunk
    cmap = copes.random_chunk_map(n_chunks, K, 77)
    ref_map = oracle.random_chunks(n_chunks, K, 77)
    for k in range(K):
        sub = copes.subspace_build(L, copes.PART_RANDOM_CHUNKS, K, k, seed=77, chunk=chunk,
                                   chunk_map=cmap, tile_size=300)
        check_tiles(sub, oracle.chunk_ranges(ODD_LAYOUT, chunk, ref_map, k), 300)


@pytest.mark.parametrize("K", [1, 5, 16, 64])
def test_hash_lists_bit_exact(copes, K):
    numel = [50_000, 333, 16_384, 16_385, 64, 40_000]
    tids = [10, 11, 12, 13, 14, 15]
    L = copes.Layout(numel, tids)
    lists = copes.hash_partition(L, K, 1088)
    total = 0
    for k, sub in enumerate(lists):
        got = sub.tensor.cpu().numpy()
        ref = oracle.hash_list(numel, tids, K, 1088, k)
        assert np.array_equal(got, ref), k
        total += got.size
    assert total == sum(numel)


@pytest.mark.parametrize("n_ranges", [1, 999, 1000, 1001, 3000])
@pytest.mark.parametrize("tile", [1, 777, 4096])
def test_tile_tables_either_side_of_the_device_expansion_limit(copes, n_ranges, tile):
    """Up to 1,000 ranges the table is written by a device kernel, beyond that it is split
    on the host and copied: both give every range cut into [b + i tile, min(b + (i+1)
    tile, e)) pieces, in range order, bit for bit."""
    rng = np.random.default_rng(n_ranges * 7 + tile)
    lens = rng.integers(1, 3 * tile + 5, n_ranges) if tile > 1 else rng.integers(1, 6, n_ranges)
    gaps = rng.integers(1, 50, n_ranges)  # ranges apart, so none merge
    b = np.cumsum(gaps + np.concatenate([[0], lens[:-1]])).astype(np.int64) + (1 << 33)
    ranges = [(int(x), int(x + l)) for x, l in zip(b, lens)]
    expected = np.array([(s, min(s + tile, e)) for s0, e in ranges for s in range(s0, e, tile)], dtype=np.int64)
    sub = copes.tiles_from_ranges(ranges, tile_size=tile)
    torch.cuda.synchronize()
    got = sub.tensor.cpu().numpy().astype(np.int64).reshape(-1, 2)
    assert np.array_equal(got, expected)
