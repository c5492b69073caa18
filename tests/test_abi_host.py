"""The C ABI library without a GPU: it loads, exports every function include/copes.h
declares, its host-side logic matches the oracle, and invalid arguments come back as
error codes before any CUDA call."""
import ctypes
import os
import re

import numpy as np
import pytest

import oracle

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2608_02391_gb300 import build, copes
    if not os.path.exists(copes.LIB_PATH):
        try:
            build.build()
        except RuntimeError as e:
            pytest.skip(f"cannot build libcopes.so here: {e}")
    return copes.load()


def declared_functions():
    text = open(os.path.join(ROOT, "include", "copes.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(copes_[a-z0-9_]+)\s*\(", text)))


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert len(names) >= 20
    for name in names:
        assert hasattr(lib, name), name
    from paper_2608_02391_gb300 import copes
    assert set(names) == set(copes.SIGNATURES)


def test_version_and_error_strings(lib):
    assert b"sm_103a" in lib.copes_version()
    assert lib.copes_perturb(None, None, 0, 1.0, None) == -1
    buf = ctypes.create_string_buffer(256)
    n = lib.copes_last_error(buf, 256)
    assert n > 0 and b"copes_perturb" in buf.value


def test_host_helpers_match_oracle(lib):
    from paper_2608_02391_gb300 import copes
    for args in [(33, 0, 0, 0), (33, 5, 7, 63), (2**63 + 11, 2**31, 3, 1)]:
        assert copes.member_seed(*args) == oracle.member_seed(*args)
    for n, pairing in [(8, copes.ANTITHETIC), (128, copes.ANTITHETIC), (5, copes.ONE_SIDED)]:
        a = copes.member_table(n, pairing)
        b = oracle.member_table(n, pairing)
        assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1]) and a[2] == b[2]
    assert copes.sigma_eff(1e-3, 4e9, 1e9) == oracle.sigma_eff(1e-3, 4e9, 1e9)
    for conv in (copes.COEF_PAPER, copes.COEF_OPENAI):
        assert copes.step_coef(5e-4, 32, 1e-3, conv) == oracle.step_coef(5e-4, 32, 1e-3, conv)
    numel = [1000, 64, 7, 4096, 130, 1, 2500]
    assert np.array_equal(copes.Layout(numel).offsets, oracle.layout(numel))


def _expected_tiles(ranges, tile):
    out = []
    for b, e in ranges:
        for s in range(b, e, tile):
            out.append((s, min(s + tile, e)))
    return out


def test_subspace_build_tile_counts_match_oracle_ranges(lib):
    from paper_2608_02391_gb300 import copes
    numel = [1000, 64, 7, 4096, 130, 1, 2500]
    L = copes.Layout(numel)
    count = ctypes.c_uint64()
    for K in (1, 3, 4):
        for k in range(K):
            spec = copes.PartitionSpec(copes.PART_CONTIGUOUS, K, 0, 0, None)
            rc = lib.copes_subspace_build(ctypes.byref(L.desc), ctypes.byref(spec), k, 100, None, None, 0,
                                          ctypes.byref(count), None)
            assert rc == 0
            assert count.value == len(_expected_tiles(oracle.contiguous_ranges(numel, K, k), 100))
    groups = np.array([0, 1, 1, 0, 2, 2, 1], np.int32)
    for k in range(3):
        spec = copes.PartitionSpec(copes.PART_TENSOR_GROUPS, 3, 0, 0, groups.ctypes.data_as(ctypes.c_void_p))
        assert lib.copes_subspace_build(ctypes.byref(L.desc), ctypes.byref(spec), k, 512, None, None, 0,
                                        ctypes.byref(count), None) == 0
        assert count.value == len(_expected_tiles(oracle.group_ranges(numel, groups, k), 512))


def test_invalid_arguments_are_rejected_before_any_launch(lib):
    from paper_2608_02391_gb300 import copes
    fake = 0x10000  # never dereferenced: every case below fails validation first
    p = copes.Params(fake, fake + 3, 100, copes.BF16)  # misaligned master
    s = copes.Subspace(copes.SUBSPACE_TILES, fake, 1, None, 0)
    assert lib.copes_perturb(ctypes.byref(p), ctypes.byref(s), 1, 1e-3, None) == copes.ERR_ALIGNMENT
    p = copes.Params(fake, fake + (1 << 24), 100, 7)
    assert lib.copes_restore(ctypes.byref(p), ctypes.byref(s), None) == copes.ERR_INVALID_ARG
    p = copes.Params(fake, fake + (1 << 24), 100, copes.BF16)
    bad = copes.Subspace(9, None, 0, None, 0)
    assert lib.copes_context_commit(ctypes.byref(p), ctypes.byref(bad), None) == copes.ERR_INVALID_ARG
    idx = copes.Subspace(copes.SUBSPACE_INDICES, None, 0, fake + 8, 10)
    assert lib.copes_restore(ctypes.byref(p), ctypes.byref(idx), None) == copes.ERR_ALIGNMENT
    assert lib.copes_perturb(ctypes.byref(p), ctypes.byref(s), 1, float("nan"), None) == copes.ERR_INVALID_ARG
    assert lib.copes_shape_fitness(fake, 0, None, copes.SHAPE_ZSCORE, fake, None) == copes.ERR_SIZE
    assert lib.copes_shape_fitness(fake, 300, None, copes.SHAPE_ZSCORE, fake, None) == copes.ERR_SIZE
    assert lib.copes_shape_fitness(fake, 8, None, copes.SHAPE_ZSCORE_GROUPED, fake, None) == copes.ERR_INVALID_ARG
    nid = np.array([0, 0, 1, 5], np.int32)
    sg = np.array([1, -1, 1, -1], np.int8)
    seeds = np.zeros(2, np.uint64)
    P = ctypes.c_void_p
    assert lib.copes_update(ctypes.byref(p), ctypes.byref(s), 4, nid.ctypes.data_as(P), sg.ctypes.data_as(P),
                            fake, 2, seeds.ctypes.data_as(P), 0.1, 1, None) == copes.ERR_INVALID_ARG
    nid[3] = 1
    sg[3] = 0
    assert lib.copes_update(ctypes.byref(p), ctypes.byref(s), 4, nid.ctypes.data_as(P), sg.ctypes.data_as(P),
                            fake, 2, seeds.ctypes.data_as(P), 0.1, 1, None) == copes.ERR_INVALID_ARG
    assert lib.copes_update(ctypes.byref(p), ctypes.byref(s), 300, nid.ctypes.data_as(P), sg.ctypes.data_as(P),
                            fake, 2, seeds.ctypes.data_as(P), 0.1, 1, None) == copes.ERR_SIZE
    L = copes.Layout([1000, 2000])
    need = lib.copes_hash_workspace_bytes(ctypes.byref(L.desc), 16)
    assert need > 0
    counts = np.zeros(16, np.uint64)
    assert lib.copes_hash_count(ctypes.byref(L.desc), 16, 1, fake, need - 16, counts.ctypes.data_as(P),
                                None) == copes.ERR_WORKSPACE
    assert lib.copes_hash_count(ctypes.byref(L.desc), 65, 1, fake, need, counts.ctypes.data_as(P),
                                None) == copes.ERR_INVALID_ARG
    assert lib.copes_random_chunk_map(0, 4, 1, fake, fake, 1 << 20, None) == copes.ERR_SIZE
    assert lib.copes_random_chunk_map((1 << 20) + 1, 4, 1, fake, fake, 1 << 24, None) == copes.ERR_SIZE
    # the sort workspace: 8 bytes per chunk, the count rounded up to a power of two >= 4096
    assert lib.copes_random_chunk_map_workspace_bytes(1) == 8 * 4096
    assert lib.copes_random_chunk_map_workspace_bytes(4097) == 8 * 8192
    assert lib.copes_random_chunk_map_workspace_bytes(1 << 20) == 8 << 20
    assert lib.copes_random_chunk_map_workspace_bytes((1 << 20) + 1) == 0
    assert lib.copes_random_chunk_map(5000, 4, 1, fake, fake, 8 * 4096, None) == copes.ERR_WORKSPACE
    assert lib.copes_random_chunk_map(5000, 4, 1, fake, None, 8 * 8192, None) == copes.ERR_WORKSPACE
    assert lib.copes_random_chunk_map(5000, 4, 1, fake, fake + 8, 8 * 8192, None) == copes.ERR_ALIGNMENT
    spec = copes.PartitionSpec(copes.PART_HASH, 4, 0, 0, None)
    cnt = ctypes.c_uint64()
    assert lib.copes_subspace_build(ctypes.byref(L.desc), ctypes.byref(spec), 0, 100, None, None, 0,
                                    ctypes.byref(cnt), None) == copes.ERR_INVALID_ARG
    spec = copes.PartitionSpec(copes.PART_CONTIGUOUS, 4, 0, 0, None)
    assert lib.copes_subspace_build(ctypes.byref(L.desc), ctypes.byref(spec), 4, 100, None, None, 0,
                                    ctypes.byref(cnt), None) == copes.ERR_INVALID_ARG
    assert lib.copes_subspace_build(ctypes.byref(L.desc), ctypes.byref(spec), 0, 0, None, None, 0,
                                    ctypes.byref(cnt), None) == copes.ERR_SIZE
    assert lib.copes_member_table(7, copes.ANTITHETIC, fake, fake) == copes.ERR_INVALID_ARG


def test_hash_replay_arguments_are_rejected_before_any_copy(lib):
    from paper_2608_02391_gb300 import copes
    fake = 0x10000  # never dereferenced: every case below fails validation first
    P = ctypes.c_void_p
    L = copes.Layout([1000, 0, 2000])
    # 32 bytes per non-empty tensor, then 4 per 16,384-element tile (2 tiles), each rounded to 16
    assert lib.copes_hash_replay_bytes(ctypes.byref(L.desc)) == 80
    assert lib.copes_hash_replay_bytes(None) == 0
    out = copes.Subspace()
    for K, k, table, nbytes, code in [(0, 0, fake, 80, copes.ERR_INVALID_ARG),
                                      (65, 0, fake, 80, copes.ERR_INVALID_ARG),
                                      (4, 4, fake, 80, copes.ERR_INVALID_ARG),
                                      (4, -1, fake, 80, copes.ERR_INVALID_ARG),
                                      (4, 1, None, 80, copes.ERR_WORKSPACE),
                                      (4, 1, fake, 64, copes.ERR_WORKSPACE),
                                      (4, 1, fake + 8, 80, copes.ERR_ALIGNMENT)]:
        assert lib.copes_hash_replay_subspace(ctypes.byref(L.desc), K, 7, k, table, nbytes, None,
                                              ctypes.byref(out)) == code, (K, k, table, nbytes)
    assert lib.copes_hash_replay_subspace(ctypes.byref(L.desc), 4, 7, 1, fake, 80, None, None) == \
        copes.ERR_INVALID_ARG
    p = copes.Params(fake, fake + (1 << 24), 3072, copes.BF16)
    def replay(**kw):
        f = dict(kind=copes.SUBSPACE_HASH_REPLAY, replay=fake, n_replay_tiles=2, n_replay_tensors=2, K=4,
                 k=1, seed=7)
        f.update(kw)
        return copes.Subspace(**f)
    for S, code in [(replay(K=0), copes.ERR_INVALID_ARG), (replay(k=4), copes.ERR_INVALID_ARG),
                    (replay(replay=None), copes.ERR_INVALID_ARG), (replay(replay=fake + 4), copes.ERR_ALIGNMENT),
                    (replay(n_replay_tiles=0), copes.ERR_INVALID_ARG),
                    (replay(n_replay_tiles=1 << 31), copes.ERR_SIZE)]:
        assert lib.copes_perturb(ctypes.byref(p), ctypes.byref(S), 1, 1e-3, None) == code
        assert lib.copes_restore(ctypes.byref(p), ctypes.byref(S), None) == code
    nid = np.array([0, 0], np.int32)
    sg = np.array([1, -1], np.int8)
    seeds = np.zeros(1, np.uint64)
    S = replay(K=65)
    assert lib.copes_update(ctypes.byref(p), ctypes.byref(S), 2, nid.ctypes.data_as(P), sg.ctypes.data_as(P),
                            fake, 1, seeds.ctypes.data_as(P), 0.1, 1, None) == copes.ERR_INVALID_ARG


def test_backup_mode_arguments_are_rejected_before_any_launch(lib):
    from paper_2608_02391_gb300 import copes
    fake = 0x10000  # never dereferenced: every case below fails validation first
    P = ctypes.c_void_p
    tiles = copes.Subspace(copes.SUBSPACE_TILES, fake, 1, None, 0)
    idx = copes.Subspace(copes.SUBSPACE_INDICES, None, 0, fake, 4)
    cases = [(None, tiles, copes.ERR_INVALID_ARG),
             (copes.BackupParams(fake, None, 100), tiles, copes.ERR_INVALID_ARG),
             (copes.BackupParams(fake + 2, fake, 100), tiles, copes.ERR_ALIGNMENT),
             (copes.BackupParams(fake, fake + 8, 100), tiles, copes.ERR_ALIGNMENT),
             (copes.BackupParams(fake, fake, 0), tiles, copes.ERR_SIZE),
             (copes.BackupParams(fake, fake, 100), idx, copes.ERR_UNSUPPORTED)]
    for prm, S, code in cases:
        pp = None if prm is None else ctypes.byref(prm)
        assert lib.copes_backup_save(pp, ctypes.byref(S), None) == code
        assert lib.copes_backup_restore(pp, ctypes.byref(S), None) == code
        assert lib.copes_backup_perturb(pp, ctypes.byref(S), 1, 1e-3, None) == code
    prm = copes.BackupParams(fake, fake, 100)
    assert lib.copes_backup_perturb(ctypes.byref(prm), ctypes.byref(tiles), 1, float("inf"), None) == \
        copes.ERR_INVALID_ARG
    nid = np.array([0, 0], np.int32)
    sg = np.array([1, -1], np.int8)
    seeds = np.zeros(1, np.uint64)
    assert lib.copes_backup_update(ctypes.byref(prm), ctypes.byref(tiles), 300, nid.ctypes.data_as(P),
                                   sg.ctypes.data_as(P), fake, 1, seeds.ctypes.data_as(P), 0.1, None) == \
        copes.ERR_SIZE
    assert lib.copes_backup_update(ctypes.byref(prm), ctypes.byref(idx), 2, nid.ctypes.data_as(P),
                                   sg.ctypes.data_as(P), fake, 1, seeds.ctypes.data_as(P), 0.1, None) == \
        copes.ERR_UNSUPPORTED


def test_gathered_master_arguments_are_rejected_before_any_launch(lib):
    from paper_2608_02391_gb300 import copes
    fake = 0x10000  # never dereferenced: every case below fails validation first
    p = copes.Params(fake, fake + (1 << 24), 100, copes.BF16)
    tiles = copes.Subspace(copes.SUBSPACE_TILES, fake, 1, None, 0)
    tiles.gathered = fake
    assert lib.copes_perturb(ctypes.byref(p), ctypes.byref(tiles), 1, 1e-3, None) == copes.ERR_INVALID_ARG
    idx = copes.Subspace(copes.SUBSPACE_INDICES, None, 0, fake, 4)
    assert lib.copes_gather_master(ctypes.byref(p), ctypes.byref(idx), None) == copes.ERR_INVALID_ARG
    assert lib.copes_scatter_master(ctypes.byref(p), ctypes.byref(idx), None) == copes.ERR_INVALID_ARG
    idx.gathered = fake + 4
    assert lib.copes_gather_master(ctypes.byref(p), ctypes.byref(idx), None) == copes.ERR_ALIGNMENT
    assert lib.copes_restore(ctypes.byref(p), ctypes.byref(idx), None) == copes.ERR_ALIGNMENT


def test_replay_mask_arguments_are_rejected_before_any_launch(lib):
    from paper_2608_02391_gb300 import copes
    fake = 0x10000  # never dereferenced: every case below fails validation first
    p = copes.Params(fake, fake + (1 << 24), 100, copes.BF16)
    tiles = copes.Subspace(copes.SUBSPACE_TILES, fake, 1, None, 0)
    tiles.replay_mask = fake
    assert lib.copes_perturb(ctypes.byref(p), ctypes.byref(tiles), 1, 1e-3, None) == copes.ERR_INVALID_ARG
    S = copes.Subspace(kind=copes.SUBSPACE_HASH_REPLAY, replay=fake, n_replay_tiles=2, n_replay_tensors=1,
                       K=4, k=1, seed=7)
    assert lib.copes_hash_replay_mask(ctypes.byref(p), ctypes.byref(S), None) == copes.ERR_INVALID_ARG
    S.replay_mask = fake + 4
    assert lib.copes_hash_replay_mask(ctypes.byref(p), ctypes.byref(S), None) == copes.ERR_ALIGNMENT


def test_partner_buffer_arguments_are_rejected_before_any_launch(lib):
    """copes_perturb_pair / copes_perturb_partner: the partner buffer must be non-NULL,
    16-byte aligned, start at a multiple of 4, lie inside the arena and overlap neither the
    working weights nor the master."""
    from paper_2608_02391_gb300 import copes
    fake = 0x10000  # never dereferenced: every case below fails validation first
    mst, buf = fake + (1 << 24), fake + (1 << 26)  # the master and a partner buffer, apart from w
    p = copes.Params(fake, mst, 1000, copes.BF16)
    s = copes.Subspace(copes.SUBSPACE_TILES, fake, 1, None, 0)
    pair, partner = lib.copes_perturb_pair, lib.copes_perturb_partner
    assert pair(ctypes.byref(p), ctypes.byref(s), 1, 1e-3, None, 0, 1000, None) == copes.ERR_INVALID_ARG
    assert pair(ctypes.byref(p), ctypes.byref(s), 1, 1e-3, buf + 2, 0, 1000, None) == copes.ERR_ALIGNMENT
    assert pair(ctypes.byref(p), ctypes.byref(s), 1, 1e-3, buf, 6, 900, None) == copes.ERR_ALIGNMENT
    assert pair(ctypes.byref(p), ctypes.byref(s), 1, 1e-3, buf, 8, 993, None) == copes.ERR_SIZE
    assert pair(ctypes.byref(p), ctypes.byref(s), 1, 1e-3, buf, 1004, 0, None) == copes.ERR_SIZE
    assert pair(ctypes.byref(p), ctypes.byref(s), 1, float("inf"), buf, 0, 1000, None) == copes.ERR_INVALID_ARG
    assert partner(ctypes.byref(p), ctypes.byref(s), None, 0, 1000, None) == copes.ERR_INVALID_ARG
    assert partner(ctypes.byref(p), ctypes.byref(s), buf + 8, 0, 1000, None) == copes.ERR_ALIGNMENT
    assert partner(ctypes.byref(p), ctypes.byref(s), buf, 2, 10, None) == copes.ERR_ALIGNMENT
    assert partner(ctypes.byref(p), ctypes.byref(s), buf, 0, 1001, None) == copes.ERR_SIZE
    bad = copes.Subspace(9, None, 0, None, 0)
    assert partner(ctypes.byref(p), ctypes.byref(bad), buf, 0, 1000, None) == copes.ERR_INVALID_ARG
    q = copes.Params(fake, fake + 4, 1000, copes.BF16)  # misaligned master
    assert partner(ctypes.byref(q), ctypes.byref(s), buf, 0, 1000, None) == copes.ERR_ALIGNMENT
    # a partner buffer inside the working weights is rejected
    assert pair(ctypes.byref(p), ctypes.byref(s), 1, 1e-3, fake + 1024, 0, 100, None) == copes.ERR_INVALID_ARG
    assert partner(ctypes.byref(p), ctypes.byref(s), fake + 1984, 0, 8, None) == copes.ERR_INVALID_ARG
    # ... and so is one that overlaps the fp32 master, whose values the pair perturb reads
    assert pair(ctypes.byref(p), ctypes.byref(s), 1, 1e-3, mst + 64, 0, 100, None) == copes.ERR_INVALID_ARG
    assert pair(ctypes.byref(p), ctypes.byref(s), 1, 1e-3, mst - 192, 0, 100, None) == copes.ERR_INVALID_ARG
    assert partner(ctypes.byref(p), ctypes.byref(s), mst + 3984, 0, 8, None) == copes.ERR_INVALID_ARG


def test_second_working_buffer_is_validated(lib):
    from paper_2608_02391_gb300 import copes
    fake = 0x10000  # never dereferenced: every case below fails validation first
    s = copes.Subspace(copes.SUBSPACE_TILES, fake, 1, None, 0)
    p = copes.Params(fake, fake + 64, 100, copes.BF16, fake + 8)  # misaligned w2
    assert lib.copes_restore(ctypes.byref(p), ctypes.byref(s), None) == copes.ERR_ALIGNMENT
    p = copes.Params(fake, fake + 64, 100, copes.BF16, fake)  # w2 aliases w
    assert lib.copes_restore(ctypes.byref(p), ctypes.byref(s), None) == copes.ERR_INVALID_ARG
    p = copes.Params(fake, fake + 64, 100, copes.BF16, fake + 64)  # w2 aliases master
    assert lib.copes_context_commit(ctypes.byref(p), ctypes.byref(s), None) == copes.ERR_INVALID_ARG
    mst = fake + (1 << 24)
    p = copes.Params(fake, fake + 64, 100, copes.BF16)  # w (200 B) runs into master
    assert lib.copes_restore(ctypes.byref(p), ctypes.byref(s), None) == copes.ERR_INVALID_ARG
    p = copes.Params(fake, mst, 100, copes.BF16, fake + 176)  # w2 starts inside w
    assert lib.copes_restore(ctypes.byref(p), ctypes.byref(s), None) == copes.ERR_INVALID_ARG
    p = copes.Params(fake, mst, 100, copes.BF16, mst - 192)  # w2 runs into master
    assert lib.copes_restore(ctypes.byref(p), ctypes.byref(s), None) == copes.ERR_INVALID_ARG
    p = copes.Params(fake, mst, 100, copes.BF16, mst + 384)  # w2 starts inside master (400 B)
    assert lib.copes_context_commit(ctypes.byref(p), ctypes.byref(s), None) == copes.ERR_INVALID_ARG
    p = copes.Params(fake, mst, 100, copes.FP32, fake + 384)  # fp32 w is 400 B: w2 inside it
    assert lib.copes_restore(ctypes.byref(p), ctypes.byref(s), None) == copes.ERR_INVALID_ARG


def test_four_working_copies_are_validated(lib):
    """w3 and w4 come together and only with w2, 16-byte aligned, each disjoint from w, the
    master and the other copies; copes_perturb_two_pairs needs all four copies and a TILES
    subspace.  Every case fails before any CUDA call."""
    from paper_2608_02391_gb300 import copes
    fake = 0x10000  # never dereferenced: every case below fails validation first
    mst = fake + (1 << 24)
    w2, w3, w4 = fake + 1024, fake + 2048, fake + 3072  # 200 B each (100 bf16)
    s = copes.Subspace(copes.SUBSPACE_TILES, fake, 1, None, 0)
    R = lambda p: lib.copes_restore(ctypes.byref(p), ctypes.byref(s), None)
    assert R(copes.Params(fake, mst, 100, copes.BF16, w2, w3, None)) == copes.ERR_INVALID_ARG  # w3 alone
    assert R(copes.Params(fake, mst, 100, copes.BF16, w2, None, w4)) == copes.ERR_INVALID_ARG  # w4 alone
    assert R(copes.Params(fake, mst, 100, copes.BF16, None, w3, w4)) == copes.ERR_INVALID_ARG  # without w2
    assert R(copes.Params(fake, mst, 100, copes.BF16, w2, w3 + 8, w4)) == copes.ERR_ALIGNMENT
    assert R(copes.Params(fake, mst, 100, copes.BF16, w2, w3, w4 + 4)) == copes.ERR_ALIGNMENT
    assert R(copes.Params(fake, mst, 100, copes.BF16, w2, w3, fake)) == copes.ERR_INVALID_ARG  # w4 aliases w
    assert R(copes.Params(fake, mst, 100, copes.BF16, w2, mst, w4)) == copes.ERR_INVALID_ARG  # w3 aliases master
    assert R(copes.Params(fake, mst, 100, copes.BF16, w2, w2, w4)) == copes.ERR_INVALID_ARG  # w3 aliases w2
    assert R(copes.Params(fake, mst, 100, copes.BF16, w2, w3, w2 + 176)) == copes.ERR_INVALID_ARG  # w4 in w2
    assert R(copes.Params(fake, mst, 100, copes.BF16, w2, w3, w3 + 160)) == copes.ERR_INVALID_ARG  # w4 in w3
    assert R(copes.Params(fake, mst, 100, copes.BF16, w2, mst - 192, w4)) == copes.ERR_INVALID_ARG  # into master
    assert R(copes.Params(fake, mst, 100, copes.FP32, w2, w2 + 256, w4)) == copes.ERR_INVALID_ARG  # fp32 w2: 400 B
    T = lambda p, sub, sigma=1e-3: lib.copes_perturb_two_pairs(ctypes.byref(p), ctypes.byref(sub), 1, 2, sigma, None)
    dual = copes.Params(fake, mst, 100, copes.BF16, w2)
    assert T(dual, s) == copes.ERR_INVALID_ARG  # two copies only
    quad = copes.Params(fake, mst, 100, copes.BF16, w2, w3, w4)
    assert T(quad, s, float("inf")) == copes.ERR_INVALID_ARG
    idx = copes.Subspace(copes.SUBSPACE_INDICES, None, 0, fake, 10)
    assert T(quad, idx) == copes.ERR_UNSUPPORTED
    assert lib.copes_perturb_two_pairs(None, ctypes.byref(s), 1, 2, 1e-3, None) == copes.ERR_INVALID_ARG


def test_backup_partner_arguments_are_rejected_before_any_launch(lib):
    from paper_2608_02391_gb300 import copes
    fake = 0x10000  # never dereferenced: every case below fails validation first
    s = copes.Subspace(copes.SUBSPACE_TILES, fake, 1, None, 0)
    p = copes.BackupParams(fake + 8, fake, 1000)  # misaligned w
    assert lib.copes_backup_perturb_pair(ctypes.byref(p), ctypes.byref(s), 1, 1e-3, fake, 0, 1000,
                                         None) == copes.ERR_ALIGNMENT
    assert lib.copes_backup_perturb_pair(ctypes.byref(p), ctypes.byref(s), 1, float("nan"), fake, 0, 1000,
                                         None) == copes.ERR_INVALID_ARG
    assert lib.copes_backup_perturb_partner(None, ctypes.byref(s), fake, 0, 1000, None) == copes.ERR_INVALID_ARG
