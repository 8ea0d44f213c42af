"""The schedule of the one-launch decode step, checked on the host (no GPU):
af1_step_plan_dry returns the tiles af1_step_create deals to the CTAs.

Every sign tile of every phase of every linear must be covered exactly once,
within its matrix; each CTA's tiles must run in stage order (level, phase 1,
phase 2), which with every CTA resident is what makes the step free of
deadlock; and each row block must be split into exactly the K slices the
consumers of its partial sums expect."""
import ctypes

import numpy as np
import pytest

import synth
from oracle import af1_oracle as O


@pytest.fixture(scope="module")
def P():
    import paper_2609_06161_gb300 as P
    return P


def dry_plan(P, shapes, levels, tokens, ctas, producer=None, producer2=None):
    lib = P._lib
    f = lib.af1_step_plan_dry
    i64p, i32p = ctypes.POINTER(ctypes.c_int64), ctypes.POINTER(ctypes.c_int32)
    f.argtypes = [i64p, i64p, i64p, i32p, i32p, i32p, ctypes.c_int, ctypes.c_int64, ctypes.c_int32, i32p, i32p,
                  ctypes.c_int64, i32p, i32p, i64p, ctypes.POINTER(ctypes.c_double)]
    f.restype = ctypes.c_int
    k = len(shapes)
    m = (ctypes.c_int64 * k)(*[s[0] for s in shapes])
    n = (ctypes.c_int64 * k)(*[s[1] for s in shapes])
    r = (ctypes.c_int64 * k)(*[s[2] for s in shapes])
    lv = (ctypes.c_int32 * k)(*levels)
    pr = None if producer is None else (ctypes.c_int32 * k)(*producer)
    pr2 = None if producer2 is None else (ctypes.c_int32 * k)(*producer2)
    nt = ctypes.c_int64()
    us = ctypes.c_double()
    assert f(m, n, r, lv, pr, pr2, k, tokens, ctas, None, None, 0, None, None, ctypes.byref(nt), ctypes.byref(us)) == 0
    order = (ctypes.c_int32 * k)()
    tasks = (ctypes.c_int32 * (7 * nt.value))()
    first = (ctypes.c_int32 * (ctas + 1))()
    ks = (ctypes.c_int32 * (2 * k))()
    assert f(m, n, r, lv, pr, pr2, k, tokens, ctas, order, tasks, nt.value, first, ks, ctypes.byref(nt),
             ctypes.byref(us)) == 0, P.last_error()
    return (list(order), np.array(tasks, dtype=np.int64).reshape(-1, 7), list(first), list(ks), us.value)


def check_plan(P, shapes, levels, tokens=1, ctas=304, producer=None, producer2=None):
    """Stage of a tile: 3 level + 0 (phase 1), 1 (phase 2) or 2 (storing y);
    the y tiles of level L come after level L + 1's phase 1 (3 L + 3.5) when
    every linear of level L + 1 is chained."""
    order, tasks, first, ks, model_us = dry_plan(P, shapes, levels, tokens, ctas, producer, producer2)
    chained = None if producer is None else [p >= 0 for p in producer]
    assert sorted(order) == list(range(len(shapes)))
    lv_sorted = [levels[i] for i in order]
    assert lv_sorted == sorted(lv_sorted)
    dense = {v: i for i, v in enumerate(sorted(set(levels)))}
    nlev = len(dense)
    ext = [False] * nlev
    for i, lvv in enumerate(levels):
        if dense[lvv] > 0 and (chained is None or not chained[i]):
            ext[dense[lvv]] = True
    probs = []  # (R, C, RB, NCH, level, phase)
    for i in order:
        m, n, r = shapes[i]
        for (R, C, ph) in ((r, n, 1), (m, r, 2)):
            probs.append((R, C, -(-R // 128), -(-C // 128), dense[levels[i]], ph))
    cover = [np.zeros((p[2], p[3]), dtype=np.int64) for p in probs]
    outs = [np.zeros(p[2], dtype=np.int64) for p in probs]
    slices = [dict() for _ in probs]
    assert first[0] == 0 and first[-1] == len(tasks)
    assert all(first[c] <= first[c + 1] for c in range(ctas))
    for c in range(ctas):
        stages = []
        for (q, rb0, G, c0, nch, kslice, kind) in tasks[first[c]:first[c + 1]]:
            R, C, RB, NCH, lev, ph = probs[q]
            assert 1 <= G <= 4 and 0 <= rb0 and rb0 + G <= RB
            if kind == 1:
                assert ph == 2 and nch == 0
                outs[q][rb0:rb0 + G] += 1
                deferred = lev + 1 < nlev and not ext[lev + 1]
                stages.append(3 * lev + 3.5 if deferred else 3 * lev + 2)
                continue
            assert kind == 0
            assert 1 <= nch and 0 <= c0 and c0 + nch <= NCH
            assert 0 <= kslice < ks[q]
            cover[q][rb0:rb0 + G, c0:c0 + nch] += 1
            for rb in range(rb0, rb0 + G):
                slices[q].setdefault(rb, []).append((kslice, c0, nch))
            stages.append(3 * lev + ph - 1)
        assert stages == sorted(stages), f"CTA {c} runs its tiles out of stage order"
    for q, cv in enumerate(cover):
        assert (cv == 1).all(), f"problem {q}: tiles do not cover its matrix exactly once"
        for rb, sl in slices[q].items():
            assert sorted(s[0] for s in sl) == list(range(ks[q])), f"problem {q} row block {rb}: K slices"
        if probs[q][5] == 2:
            assert (outs[q] == 1).all(), f"problem {q}: every row block of y is stored exactly once"
        else:
            assert (outs[q] == 0).all()
    # Phase 2's K slices are ranks: its chunks are the row blocks of phase 1.
    for j in range(len(order)):
        assert probs[2 * j][2] == probs[2 * j + 1][3]
    assert model_us > 0
    return tasks, first, model_us


def test_plan_one_decoder_layer(P):
    shapes = [(m, n, O.rank_for_budget(m, n, 1)) for (_nm, m, n) in synth.LLAMA3_8B_LINEARS]
    check_plan(P, shapes, [0, 0, 0, 1, 2, 2, 3])


@pytest.mark.parametrize("tokens", [1, 2, 4])
def test_plan_32_layer_stack(P, tokens):
    base = [(m, n, O.rank_for_budget(m, n, 1)) for (_nm, m, n) in synth.LLAMA3_8B_LINEARS]
    shapes = base * 32
    levels = [4 * (i // 7) + [0, 0, 0, 1, 2, 2, 3][i % 7] for i in range(len(shapes))]
    tasks, first, model_us = check_plan(P, shapes, levels, tokens)
    # every CTA works in most stages: the tiles are spread
    per_cta = np.diff(first)
    assert per_cta.min() >= 64


def test_plan_32_layer_chained_stack(P):
    """The decoder data flow: every linear above level 0 reads earlier
    outputs, so each level's y tiles follow the next level's phase 1."""
    base = [(m, n, O.rank_for_budget(m, n, 1)) for (_nm, m, n) in synth.LLAMA3_8B_LINEARS]
    shapes = base * 32
    levels = [4 * (i // 7) + [0, 0, 0, 1, 2, 2, 3][i % 7] for i in range(len(shapes))]
    producer, producer2 = [], []
    for li in range(32):
        b = 7 * li
        prev_down = b - 1 if li > 0 else -1
        producer += [prev_down, prev_down, prev_down, b + 0, b + 3, b + 3, b + 4]
        producer2 += [-1, -1, -1, -1, -1, -1, b + 5]
    check_plan(P, shapes, levels, 1, producer=producer, producer2=producer2)


def test_plan_ragged_shapes_unsorted_levels(P):
    shapes = [(100, 130, 77), (1000, 700, 321), (33, 70, 31), (520, 2000, 600), (257, 129, 200), (16, 16, 8)]
    levels = [5, 0, 5, 2, 9, 0]
    check_plan(P, shapes, levels, tokens=3, ctas=37)


def test_plan_more_ctas_than_tiles(P):
    check_plan(P, [(16, 16, 8), (64, 64, 32)], [0, 1], tokens=1, ctas=304)


def test_plan_rejects_bad_arguments(P):
    lib = P._lib
    f = lib.af1_step_plan_dry
    one = (ctypes.c_int64 * 1)(64)
    lv = (ctypes.c_int32 * 1)(0)
    nt = ctypes.c_int64()
    assert f(one, one, one, lv, None, None, 1, 5, 304, None, None, 0, None, None, ctypes.byref(nt), None) == -1
    assert f(one, one, one, lv, None, None, 1, 1, 0, None, None, 0, None, None, ctypes.byref(nt), None) == -1
    neg = (ctypes.c_int32 * 1)(-1)
    assert f(one, one, one, neg, None, None, 1, 1, 304, None, None, 0, None, None, ctypes.byref(nt), None) == -1
