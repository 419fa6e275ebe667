"""A decode token over a small stack, replayed as one CUDA graph.

Two LLaMA-3-8B-shaped layers (q/o 4096 x 4096, k/v 1024 x 4096, gate/up
14336 x 4096, down 4096 x 14336; 60% weight, 50% activation sparsity), each
layer's four launches (q/k/v and gate/up as shared-input launches, o, down)
captured once, the way bench.py times the per-token stack, and replayed
twice.  Every projection's output is then checked against the CPU oracle on
sampled rows (first and last, both sides of every 1024-row segment border,
and a seeded sample), within 2e-3 * sum_{j in K} |W_ij| |x_j|.
"""
import os
import sys

import numpy as np
import pytest
import torch

import oracle as orc

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def duo():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    from paper_2506_20194_gb300 import duo as d
    d.load_library()
    return d


def _rows(O, seed):
    rng = np.random.default_rng(seed)
    borders = [r for s in range(1, (O + 1023) // 1024) for r in (1024 * s - 1, 1024 * s)]
    return np.unique(np.concatenate([[0, O - 1], borders, rng.integers(0, O, 48)]).astype(np.int64))


def test_two_layer_token_graph_matches_oracle(duo):
    import bench
    from paper_2506_20194_gb300 import synth
    dev = torch.device("cuda", 0)
    wl = synth.WORKLOADS["llama3-8b-stack"]
    shape = wl["shape"]
    px = 50
    layers, dense = [], []
    for l in range(2):
        Ws = {p: synth.layer_weight(wl, p, layer=l, device=dev) for p in synth.PROJS}
        hs = {p: duo.duo_pack(Ws[p], "bitmask") for p in synth.PROJS}
        xs = {s: synth.layer_input(wl, s, layer=l, device=dev) for s in bench.STAGE_SRC}
        ys = {p: torch.full((shape.O(p),), float("nan"), dtype=torch.float32, device=dev)
              for p in synth.PROJS}
        layers.append(dict(h=hs, x=xs, y=ys))
        dense.append(Ws)

    def token():
        for lay in layers:
            for si in range(len(bench.STAGES)):
                bench.stage_call(duo, shape, lay, px, si)

    g = bench.capture(token)
    for _ in range(2):
        g.replay()
    torch.cuda.synchronize()
    assert duo.duo_device_status() == duo.DUO_OK
    for l, (lay, Ws) in enumerate(zip(layers, dense)):
        for si, st in enumerate(bench.STAGES):
            x16 = lay["x"][bench.STAGE_SRC[si]].cpu().numpy()
            k = bench.k_of(shape.I(st[0]), px)
            K, _ = orc.oracle_sparsify(x16, k)
            for p in st:
                rows = _rows(shape.O(p), 100 * l + si)
                W16 = Ws[p][torch.from_numpy(rows).to(dev)].cpu().numpy()
                y_ref = orc.oracle_spmspv(W16, x16, k)
                tol = orc.tolerance_rows(W16, x16, K, 2e-3)
                y = lay["y"][p].cpu().numpy()[rows].astype(np.float64)
                err = np.abs(y - y_ref)
                assert np.all(err <= tol), (l, p, int(rows[np.argmax(err - tol)]), float(err.max()))
    for lay in layers:
        for h in lay["h"].values():
            h.free()
