"""Pins for the planner oracle: Eq. 1 / Eq. 2 closed forms, brute force, hand cases."""
import itertools

import pytest

from oracle import planner as P


def test_memory_first_fill_hand_cases():
    GB = 10 ** 9
    # 80 layers of 1.7113 GB, 60 GB budget, 4.2 GB fixed, 0.36 GB KV, 2 slots:
    # (60 - 4.2 - 0.36 - 2*1.7113) / 1.7113 = 30.4 -> 30 resident
    R, ok = P.memory_first_fill(80, 1_711_308_800, 60 * GB, 4_200_000_000, 360_000_000, 2)
    assert ok and R == 30
    R3, _ = P.memory_first_fill(80, 1_711_308_800, 60 * GB, 4_200_000_000, 360_000_000, 3)
    assert R3 == 29
    # everything fits: no slot reserved
    assert P.memory_first_fill(4, 100, 1000, 100, 50, 2) == (4, True)
    # exactly one layer short of fitting -> slots are needed
    assert P.memory_first_fill(4, 100, 549, 100, 50, 2) == (1, True)
    # cannot hold the slots
    assert P.memory_first_fill(4, 100, 349, 100, 50, 2) == (0, False)


def test_evenly_spaced_counts_and_gaps():
    for L in (8, 10, 32, 80):
        for m in range(L + 1):
            mask = P.evenly_spaced(L, m)
            assert sum(mask) == m
            if 0 < m < L:
                idx = [i for i, o in enumerate(mask) if o]
                gaps = [(idx[(j + 1) % m] - idx[j]) % L or L for j in range(m)]
                assert max(gaps) - min(gaps) <= 1


def test_single_slot_simulation_equals_eq1_when_gaps_uniform():
    # K = 1: each load overlaps only the resident layers before its layer (Eq. 2 window).
    L, m = 12, 4                       # gaps of 3 layers (2 resident + 1 offloaded)
    mask = P.evenly_spaced(L, m)
    for t, c in ((1.0, 0.5), (1.0, 2.0), (1.0, 5.0), (0.3, 0.31)):
        comp, load = [t] * L, [c] * L
        assert P.simulate(comp, load, mask, 1) == pytest.approx(P.eq1_single_device(comp, load, mask), rel=1e-12)


def test_double_slot_closed_forms():
    L, m = 10, 5
    mask = P.evenly_spaced(L, m)
    # link bound: the copy stream never idles -> T = m * c
    assert P.simulate([1.0] * L, [7.0] * L, mask, 2) == pytest.approx(m * 7.0)
    # compute bound: T = sum of compute
    assert P.simulate([1.0] * L, [0.5] * L, mask, 2) == pytest.approx(L * 1.0)
    # nothing offloaded
    assert P.simulate([1.0] * L, [9.0] * L, [False] * L, 2) == pytest.approx(L)
    # never below max(compute, copy)
    for K in (1, 2, 3):
        for c in (0.2, 1.0, 1.7, 4.0):
            assert P.simulate([1.0] * L, [c] * L, mask, K) >= P.step_lower_bound([1.0] * L, [c] * L, mask) - 1e-12


def test_evenly_spaced_is_optimal_single_slot_brute_force():
    L = 10
    for m in (2, 3, 4, 6):
        for c in (1.5, 2.5, 4.0):
            comp, load = [1.0] * L, [c] * L
            best = min(P.simulate(comp, load, [i in s for i in range(L)], 1)
                       for s in itertools.combinations(range(L), m))
            assert P.simulate(comp, load, P.evenly_spaced(L, m), 1) == pytest.approx(best)


def test_plan_and_threshold():
    plan = P.plan(80, 1_711_308_800, 60 * 10 ** 9, 4_200_000_000, 360_000_000, 2, 6.7e12, 2.1e11)
    assert plan["R"] == 30 and sum(plan["offloaded"]) == 50
    assert plan["pred_step_s"] == pytest.approx(50 * 1_711_308_800 / 2.1e11, rel=1e-9)
    assert P.plan(4, 100, 349, 100, 50, 2, 1.0, 1.0) is None
    # Eq. 6 reading: tokens until the KV cache exhausts what is left
    assert P.kv_threshold_tokens(1000, 100, 100, 6, 2, 10) == 10
    assert P.kv_threshold_tokens(1000, 100, 100, 8, 2, 10) == 0


def _max_resident_run(mask):
    """Longest cyclic run of resident layers (brute force over start points)."""
    L = len(mask)
    if not any(mask):
        return L
    best = 0
    for s in range(L):
        run = 0
        while run < L and not mask[(s + run) % L]:
            run += 1
        best = max(best, run)
    return best


def test_demote_one_hand_cases():
    # nothing offloaded: the last layer goes first (where m = 1 even spacing puts it)
    assert P.demote_one([False] * 8) == ([False] * 7 + [True], 7)
    # L = 8: 7 -> 3 (middle of 0..6) -> 5 (first of two runs of 3, 4..6) -> 1
    mask, order = [False] * 8, []
    for _ in range(4):
        mask, v = P.demote_one(mask)
        order.append(v)
    assert order == [7, 3, 5, 1]
    assert mask == [False, True] * 4
    # even-length run: the lower middle (L = 5: after 4, run 0..3 -> layer 1)
    assert P.demote_one(P.demote_one([False] * 5)[0])[1] == 1
    # the run may wrap around the end of the layer order: offloaded {2}, run 3,4,0,1 -> layer 4
    assert P.demote_one([False, False, True, False, False]) == ([False, False, True, False, True], 4)
    # everything offloaded: no victim
    assert P.demote_one([True] * 3) == ([True] * 3, None)


def test_demote_one_minimises_longest_resident_run_brute_force():
    import random
    rng = random.Random(5)
    for _ in range(300):
        L = rng.randint(2, 24)
        mask = [rng.random() < 0.3 for _ in range(L)]
        if all(mask):
            continue
        new, v = P.demote_one(mask)
        assert not mask[v] and new[v] and sum(new) == sum(mask) + 1
        assert all(new[i] == mask[i] for i in range(L) if i != v)
        best = min(_max_resident_run(mask[:i] + [True] + mask[i + 1:]) for i in range(L) if not mask[i])
        assert _max_resident_run(new) == best


def test_refine_blocks_hand_cases():
    A, M = 30, 140  # MHA and MLP block bytes of a 170-byte layer (p_A ~ 0.18)
    off = [False, True, False, True, True]
    # 150 left: layer 1 keeps its MLP block (140), 10 left -> nothing more
    assert P.refine_blocks(150, off, A, M) == ([3, 2, 3, 0, 0], 10)
    # 100 left: no MLP block fits; MHA blocks of layers 1, 3, 4 (90), 10 left
    assert P.refine_blocks(100, off, A, M) == ([3, 1, 3, 1, 1], 10)
    # 200 left: MLP of layer 1, then MHA of layers 3 and 4 (140 + 30 + 30 = 200)
    assert P.refine_blocks(200, off, A, M) == ([3, 2, 3, 1, 1], 0)
    # nothing offloaded or nothing left: unchanged
    assert P.refine_blocks(500, [False] * 3, A, M) == ([3, 3, 3], 500)
    assert P.refine_blocks(29, off, A, M) == ([3, 0, 3, 0, 0], 29)


def test_refine_blocks_never_exceeds_memory_and_streams_less():
    import random
    rng = random.Random(3)
    for _ in range(200):
        L = rng.randint(1, 12)
        off = [rng.random() < 0.5 for _ in range(L)]
        A, M = rng.randint(1, 50), rng.randint(1, 200)
        left0 = rng.randint(0, 600)
        masks, left = P.refine_blocks(left0, off, A, M)
        kept = sum((A if m & 1 else 0) + (M if m & 2 else 0) for m, o in zip(masks, off) if o)
        assert left == left0 - kept >= 0
        assert all(m == 3 for m, o in zip(masks, off) if not o)
        # a layer left fully offloaded means no block fits any more
        if any(m == 0 and o for m, o in zip(masks, off)):
            assert left < min(A, M)


def test_eq7_choice_brute_force():
    import random
    rng = random.Random(4)
    assert P.eq7_choice(10, 3, 2, 30, 140) == (1, 0)   # one MHA block covers it
    assert P.eq7_choice(100, 3, 2, 30, 140) == (0, 1)  # 140 beats 4 x 30 (not available) and 3 x 30 + 1 x 140
    assert P.eq7_choice(80, 3, 2, 30, 140) == (3, 0)   # 90 < 140
    assert P.eq7_choice(0, 3, 2, 30, 140) == (0, 0)
    assert P.eq7_choice(10 ** 6, 3, 2, 30, 140) is None
    for _ in range(300):
        A, M = rng.randint(1, 60), rng.randint(1, 300)
        na, nm = rng.randint(0, 6), rng.randint(0, 4)
        need = rng.randint(0, na * A + nm * M + 50)
        got = P.eq7_choice(need, na, nm, A, M)
        cands = [(a * A + b * M, a + b, (a, b)) for a in range(na + 1) for b in range(nm + 1) if a * A + b * M >= need]
        if not cands:
            assert got is None
        else:
            best = min(cands)
            assert got is not None and (got[0] * A + got[1] * M, sum(got)) == best[:2]
