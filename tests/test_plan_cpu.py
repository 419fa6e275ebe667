"""The fused kernel's launcher plan on the host (no GPU): CTAs per
(product, 1024-row segment) run, and when a multi-product launch is issued
as two.  Through the library's internal entry point duo_test_plan_runs.

The plan gives each run whole CTAs, greedily, in proportion to its cost
w = 4 (128 + 2 d 1024) + (128 + 2 d rows): mostly its record count (one
warp's walk over 1024 rows per record whatever the segment holds), a little
its bytes.  The greedy (next CTA to the largest w / n) is the min-max
allocation; the launch splits when that max is above 1.25 x the mean.
"""
import ctypes
import random

import pytest

MASK_BYTES = 128


@pytest.fixture(scope="module")
def lib():
    from paper_2506_20194_gb300.build import build_library
    build_library()
    from paper_2506_20194_gb300 import duo
    return duo.load_library()


def plan(lib, Os, dens, grid=152):
    np_ = len(Os)
    O = (ctypes.c_int * np_)(*Os)
    d = (ctypes.c_float * np_)(*dens)
    n = (ctypes.c_int * 128)()
    split = ctypes.c_int(-7)
    nr = lib.duo_test_plan_runs(np_, O, d, grid, n, ctypes.byref(split))
    return nr, list(n[:max(nr, 0)]), split.value


def weights(Os, dens):
    w = []
    for O, d in zip(Os, dens):
        d = float(ctypes.c_float(d).value)
        full = MASK_BYTES + 2.0 * d * 1024
        for s in range((O + 1023) // 1024):
            rows = min(1024, O - 1024 * s)
            w.append(4.0 * full + MASK_BYTES + 2.0 * d * rows)
    return w


def test_llama2_7b_launches(lib):
    nr, n, split = plan(lib, [4096] * 3, [0.5] * 3)      # q/k/v
    assert (nr, split, sum(n)) == (12, 0, 152) and set(n) == {12, 13}
    nr, n, split = plan(lib, [11008] * 2, [0.5] * 2)     # gate/up: 10 full segments + 768 rows each
    assert (nr, split, sum(n)) == (22, 0, 152)
    assert n[10] == n[21] == 6 and all(c == 7 for i, c in enumerate(n) if i not in (10, 21))
    nr, n, split = plan(lib, [4096], [0.5])              # o, down
    assert (nr, split, n) == (4, 0, [38] * 4)


def test_short_last_segment_counts_as_records(lib):
    # LLaMA-2-13B gate/up: 13 full segments + 512 rows each; by bytes alone the
    # 512-row runs got 3 CTAs (854 of k = 2560 records per CTA)
    nr, n, split = plan(lib, [13824] * 2, [0.5] * 2)
    assert (nr, split, sum(n)) == (28, 0, 152)
    assert n[13] >= 5 and n[27] >= 5
    assert max(-(-2560 // c) for c in n) <= 512


def test_unbalanced_multi_launch_splits(lib):
    # LLaMA-2-70B gate/up: 56 runs on 152 CTAs (2 or 3 each, 1.36x the mean)
    nr, n, split = plan(lib, [28672] * 2, [0.5] * 2)
    assert (nr, split, sum(n)) == (56, 1, 152) and set(n) == {2, 3}
    nr, n, split = plan(lib, [28672], [0.5])            # each half: 28 runs, 5 or 6 CTAs
    assert (nr, split, sum(n)) == (28, 0, 152) and set(n) == {5, 6}
    # one product never splits, however unbalanced
    nr, n, split = plan(lib, [57 * 1024], [0.5])
    assert (nr, split, sum(n)) == (57, 0, 152)


def test_bad_arguments(lib):
    n = (ctypes.c_int * 128)()
    sp = ctypes.c_int()
    O = (ctypes.c_int * 1)(4096)
    d = (ctypes.c_float * 1)(0.5)
    assert lib.duo_test_plan_runs(0, O, d, 152, n, ctypes.byref(sp)) == -1
    assert lib.duo_test_plan_runs(5, O, d, 152, n, ctypes.byref(sp)) == -1       # more than 4 products
    assert lib.duo_test_plan_runs(1, O, d, 3, n, ctypes.byref(sp)) == -1         # 4 runs on 3 CTAs
    O0 = (ctypes.c_int * 1)(0)
    assert lib.duo_test_plan_runs(1, O0, d, 152, n, ctypes.byref(sp)) == -1      # no rows


def test_min_max_allocation_on_random_shapes(lib):
    rng = random.Random(5)
    for _ in range(300):
        np_ = rng.randint(1, 4)
        Os = [rng.randint(1, 40 * 1024) for _ in range(np_)]
        dens = [rng.choice([0.1, 0.3, 0.5, 0.8]) for _ in range(np_)]
        runs = sum((O + 1023) // 1024 for O in Os)
        grid = rng.randint(1, 152)
        nr, n, split = plan(lib, Os, dens, grid)
        if runs > 128 or runs > grid:
            assert nr == -1
            continue
        assert nr == runs and sum(n) == grid and min(n) >= 1
        w = weights(Os, dens)
        top = max(wq / nq for wq, nq in zip(w, n))
        # no CTA can move without some run's cost per CTA reaching the max
        for wq, nq in zip(w, n):
            if nq > 1:
                assert wq / (nq - 1) >= top * (1 - 1e-12)
        assert split == (1 if (np_ >= 2 and top > 1.25 * sum(w) / grid) else 0)
