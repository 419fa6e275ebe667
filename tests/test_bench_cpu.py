"""Host-side arithmetic of bench.py that needs no GPU: the byte companions
of the required bytes (kept values, densest-channel worst case, loaded
fractions), checked on small layers against sums written out here from the
definitions, with kept sets from the CPU oracle's sparsifier."""
import os
import sys

import numpy as np
import pytest
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
import oracle  # noqa: E402
from paper_2506_20194_gb300 import synth  # noqa: E402

SHAPE = synth.llama_shapes(96, 32, 160, "tiny")


def _layer(seed, density=0.5):
    rng = np.random.default_rng(seed)
    W = {}
    for p in synth.PROJS:
        O, I = SHAPE.O(p), SHAPE.I(p)
        w = (rng.standard_normal((O, I)) * 0.02).astype(np.float16)
        w[rng.random((O, I)) >= density] = 0
        W[p] = w
    x = {s: rng.laplace(0, 1, size=SHAPE.I(s)).astype(np.float16) for s in bench.STAGE_SRC}
    nnz = {p: torch.from_numpy((W[p] != 0).sum(axis=0).astype(np.int64)) for p in synth.PROJS}
    return W, x, nnz


def _kept(x, px):
    out = []
    for st, src in zip(bench.STAGES, bench.STAGE_SRC):
        k = bench.k_of(SHAPE.I(st[0]), px)
        if k == 0:
            out.append(None)
            continue
        K, _ = oracle.oracle_sparsify(x[src], k)
        out.append(torch.from_numpy(K.astype(np.int64)))
    return out


def _required(W, kept, px):
    """Σ over stages of Σ_p [2 Σ_{j∈K} nnz_j + k O/8 + 4 O] + 2 I + 4 k."""
    total = 0.0
    for si, st in enumerate(bench.STAGES):
        I = SHAPE.I(st[0])
        k = bench.k_of(I, px)
        for p in st:
            O = SHAPE.O(p)
            nz = 0 if k == 0 else int((W[p][:, kept[si].numpy()] != 0).sum())
            total += 2.0 * nz + k * O / 8.0 + 4.0 * O
        total += 2.0 * I + 4.0 * k
    return total


@pytest.mark.parametrize("px", [25, 50, 70])
def test_side_bytes_against_the_definitions(px):
    W, x, nnz = _layer(px)
    kept = _kept(x, px)
    vals, worst, frac, wfrac = bench.side_bytes_from_sets(SHAPE, nnz, kept, px)
    want_vals = sum(2.0 * int((W[p][:, kept[si].numpy()] != 0).sum())
                    for si, st in enumerate(bench.STAGES) for p in st)
    dense = sum(2.0 * SHAPE.O(p) * SHAPE.I(p) for p in synth.PROJS)
    assert vals == want_vals
    assert frac == pytest.approx(vals / dense, rel=1e-12)
    # the densest channels bound any selection of the same size from above
    assert worst >= _required(W, kept, px)
    assert wfrac >= frac
    # roughly (1 - p^w)(1 - p^x) for i.i.d. masks
    assert frac == pytest.approx(0.5 * (100 - px) / 100, abs=0.06)


def test_side_bytes_edge_sparsities():
    W, x, nnz = _layer(7)
    dense = sum(2.0 * SHAPE.O(p) * SHAPE.I(p) for p in synth.PROJS)
    # px = 0: every channel is kept, so the worst case is the actual selection
    kept = _kept(x, 0)
    vals, worst, frac, wfrac = bench.side_bytes_from_sets(SHAPE, nnz, kept, 0)
    assert vals == sum(2.0 * int((W[p] != 0).sum()) for p in synth.PROJS)
    assert worst == _required(W, kept, 0) and wfrac == frac == vals / dense
    # px = 100: nothing kept; only x is read
    vals, worst, frac, wfrac = bench.side_bytes_from_sets(SHAPE, nnz, _kept(x, 100), 100)
    assert vals == 0.0 and frac == 0.0 and wfrac == 0.0
    assert worst == sum(2.0 * SHAPE.I(st[0]) for st in bench.STAGES)


BRUTE_SHAPE = synth.llama_shapes(8, 4, 10, "brute")


def _brute_layer(seed):
    """A tiny layer whose products have different per-channel densities, so
    a shared-input stage's densest set differs from any one product's."""
    rng = np.random.default_rng(seed)
    nnz = {}
    for p in synth.PROJS:
        O, I = BRUTE_SHAPE.O(p), BRUTE_SHAPE.I(p)
        keep = rng.random((O, I)) < rng.uniform(0.1, 0.9, size=I)
        nnz[p] = torch.from_numpy(keep.sum(0).astype(np.int64))
    return nnz


def _check_worst_case_bruteforce(side_bytes, seed, px):
    """The worst case of the required bytes (App. B.3: the densest channels
    kept) is the largest required-bytes total over every k-subset of each
    stage's channels; its value bytes over the dense weights are the
    worst-case loaded fraction.  Stages are independent, so the per-stage
    maxima add up."""
    import itertools
    nnz = _brute_layer(seed)
    worst = wvals = dense = 0.0
    kept = []
    for st in bench.STAGES:
        I = BRUTE_SHAPE.I(st[0])
        k = bench.k_of(I, px)
        kept.append(torch.arange(k, dtype=torch.int64) if k > 0 else None)
        best_req = best_vals = None
        for K in itertools.combinations(range(I), k):
            v = sum(2.0 * int(nnz[p][j]) for p in st for j in K)
            req = v + sum(k * BRUTE_SHAPE.O(p) / 8.0 + 4.0 * BRUTE_SHAPE.O(p) for p in st)
            req += 2.0 * I + 4.0 * k
            best_req = req if best_req is None else max(best_req, req)
            best_vals = v if best_vals is None else max(best_vals, v)
        worst += best_req
        wvals += best_vals
        dense += sum(2.0 * BRUTE_SHAPE.O(p) * BRUTE_SHAPE.I(p) for p in st)
    _, got_worst, _, got_wfrac = side_bytes(BRUTE_SHAPE, nnz, kept, px)
    assert got_worst == worst, (seed, px)
    assert got_wfrac == pytest.approx(wvals / dense, rel=1e-12, abs=0.0), (seed, px)


@pytest.mark.parametrize("seed", range(4))
@pytest.mark.parametrize("px", [0, 25, 50, 70])
def test_worst_case_bytes_bruteforce(seed, px):
    _check_worst_case_bruteforce(bench.side_bytes_from_sets, seed, px)


def test_worst_case_of_one_product_is_caught():
    """Planted mistake: a shared-input stage takes the densest channels of
    its first product instead of those of the stage's summed non-zeros."""
    def mutant(shape, nnz, kept, px):
        orig_topk = torch.topk

        def topk_first(t, k):   # the stage total swapped for its first product's counts
            for st in bench.STAGES:
                if torch.equal(t, sum(nnz[p] for p in st)):
                    return orig_topk(nnz[st[0]], k)
            return orig_topk(t, k)

        torch.topk = topk_first
        try:
            return bench.side_bytes_from_sets(shape, nnz, kept, px)
        finally:
            torch.topk = orig_topk

    with pytest.raises(AssertionError):
        for seed in range(4):
            _check_worst_case_bruteforce(mutant, seed, 50)


def test_worst_case_without_the_k_cut_is_caught():
    """Planted mistake: every channel's values counted in the worst case."""
    def mutant(shape, nnz, kept, px):
        orig_topk = torch.topk
        torch.topk = lambda t, k: orig_topk(t, t.numel())
        try:
            return bench.side_bytes_from_sets(shape, nnz, kept, px)
        finally:
            torch.topk = orig_topk

    with pytest.raises(AssertionError):
        _check_worst_case_bruteforce(mutant, 0, 50)
