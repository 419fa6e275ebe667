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
