"""Host logic of es.perturb_members: which members are perturbed by copes_perturb_two_pairs
or copes_perturb_pair, which are copied in from the partner buffer, and which take a plain
copes_perturb (no GPU: the calls are recorded, not run)."""
import numpy as np
import pytest

from paper_2608_02391_gb300 import copes, es


@pytest.fixture
def calls(monkeypatch):
    log = []
    monkeypatch.setattr(copes, "perturb", lambda a, s, seed, ss: log.append(("perturb", seed, ss)))
    monkeypatch.setattr(copes, "perturb_pair",
                        lambda a, s, seed, ss, buf, base: log.append(("pair", seed, ss, base)))
    monkeypatch.setattr(copes, "perturb_partner", lambda a, s, buf, base: log.append(("partner", base)))
    monkeypatch.setattr(copes, "perturb_two_pairs",
                        lambda a, s, sa, sb, ss: log.append(("two_pairs", sa, sb, ss)))
    return log


def run(calls, members, nid, sign, partner):
    seeds = np.arange(100, 100 + max(nid) + 1, dtype=np.uint64)
    live = []
    es.perturb_members(None, None, members, nid, sign, seeds, 0.5, live.append, partner)
    return live


def test_antithetic_pairs_use_one_generation_each(calls):
    nid, sign, P = copes.member_table(8, copes.ANTITHETIC)
    live = run(calls, range(8), nid, sign, es.Partner(None, 12))
    assert live == list(range(8))
    expect = []
    for j in range(4):
        expect += [("pair", 100 + j, 0.5, 12), ("partner", 12)]
    assert calls == expect


def test_without_a_partner_buffer_every_member_is_perturbed(calls):
    nid, sign, P = copes.member_table(4, copes.ANTITHETIC)
    run(calls, range(4), nid, sign, None)
    assert calls == [("perturb", 100, 0.5), ("perturb", 100, -0.5), ("perturb", 101, 0.5),
                     ("perturb", 101, -0.5)]


def test_one_sided_members_have_no_partner(calls):
    nid, sign, P = copes.member_table(3, copes.ONE_SIDED)
    run(calls, range(3), nid, sign, es.Partner(None, 0))
    assert calls == [("perturb", 100, 0.5), ("perturb", 101, 0.5), ("perturb", 102, 0.5)]


def test_a_slice_that_splits_a_pair(calls):
    """Members 3 .. 5 of an antithetic population (a population-parallel slice): member 3's
    partner (2) is not in the slice, so 3 is perturbed alone; 4 and 5 form a pair."""
    nid, sign, P = copes.member_table(8, copes.ANTITHETIC)
    live = run(calls, es.member_slice(1, 3, 8), nid, sign, es.Partner(None, 0))
    assert live == [3, 4, 5]
    assert calls == [("perturb", 101, -0.5), ("pair", 102, 0.5, 0), ("partner", 0)]


def test_in_place_partner_evaluates_the_second_member_on_w2(calls):
    """With the arena's second working buffer as the partner, member 2j + 1 is evaluated on
    w2: no copy, and arena.live points at the buffer that holds the live member."""
    from types import SimpleNamespace
    arena = SimpleNamespace(w="w", w2="w2", live="w")
    nid, sign, P = copes.member_table(6, copes.ANTITHETIC)
    seeds = np.arange(100, 103, dtype=np.uint64)
    seen = []
    es.perturb_members(arena, None, range(6), nid, sign, seeds, 0.5, lambda i: seen.append((i, arena.live)),
                       es.Partner("w2", 0, True))
    assert seen == [(0, "w"), (1, "w2"), (2, "w"), (3, "w2"), (4, "w"), (5, "w2")]
    assert calls == [("pair", 100, 0.5, 0), ("pair", 101, 0.5, 0), ("pair", 102, 0.5, 0)]
    assert arena.live == "w"


def four_copy_run(members, n_members, kind=copes.SUBSPACE_TILES):
    from types import SimpleNamespace
    arena = SimpleNamespace(w="w", w2="w2", w3="w3", w4="w4", live="w")
    sub = SimpleNamespace(kind=kind)
    nid, sign, P = copes.member_table(n_members, copes.ANTITHETIC)
    seeds = np.arange(100, 100 + P, dtype=np.uint64)
    seen = []
    es.perturb_members(arena, sub, members, nid, sign, seeds, 0.5, lambda i: seen.append((i, arena.live)),
                       es.Partner(arena.w2, 0, True, True))
    assert arena.live == "w"
    return seen


def test_four_copies_take_two_pairs_per_pass(calls):
    """Members 4m .. 4m+3 are written by one two-pairs pass and evaluated on w, w2, w3, w4;
    a pair left over at the end goes to w and w2."""
    seen = four_copy_run(range(10), 10)
    assert seen == [(0, "w"), (1, "w2"), (2, "w3"), (3, "w4"), (4, "w"), (5, "w2"), (6, "w3"), (7, "w4"),
                    (8, "w"), (9, "w2")]
    assert calls == [("two_pairs", 100, 101, 0.5), ("two_pairs", 102, 103, 0.5), ("pair", 104, 0.5, 0)]


def test_four_copies_on_other_subspace_kinds_take_pairs(calls):
    """The two-pairs kernel takes tile subspaces only: index-list and replay subspaces run
    their pairs one at a time on w and w2."""
    seen = four_copy_run(range(4), 4, kind=copes.SUBSPACE_INDICES)
    assert seen == [(0, "w"), (1, "w2"), (2, "w"), (3, "w2")]
    assert calls == [("pair", 100, 0.5, 0), ("pair", 101, 0.5, 0)]


def test_four_copies_on_a_slice_that_splits_the_groups(calls):
    """Members 3 .. 9 of 12: member 3 alone, then 4 .. 7 in one pass, then the pair 8, 9."""
    seen = four_copy_run(range(3, 10), 12)
    assert [i for i, _ in seen] == list(range(3, 10))
    assert calls == [("perturb", 101, -0.5), ("two_pairs", 102, 103, 0.5), ("pair", 104, 0.5, 0)]
