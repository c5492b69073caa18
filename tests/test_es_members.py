"""Host logic of es.perturb_members: which members are perturbed by copes_perturb_pair,
which are copied in from the partner buffer, and which take a plain copes_perturb (no GPU:
the three calls are recorded, not run)."""
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
