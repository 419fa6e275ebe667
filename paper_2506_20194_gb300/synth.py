"""Seeded synthetic inputs shaped like the paper's LLaMA workloads.

This module holds none of the method's arithmetic: it only draws weights,
pruning masks and activation vectors.  Both the CUDA path (tests, bench) and
the CPU oracle consume its outputs, so they see identical inputs.

The paper evaluates LLaMA-2 7B/13B/70B and LLaMA-3 8B (§5, Table 1) with all
seeds fixed to 0.  Trained weights and calibration data are not available
here, so every tensor is synthetic:
  * W ~ N(0, sigma) in fp32, cast to fp16;
  * pruning: either an i.i.d. Bernoulli keep mask, or magnitude pruning with
    an exact pruned count per block of 128 input channels (the block size of
    Algorithm 1); ties prune the lower flat index (row-major inside the
    block) first; a surviving weight that rounds to 0 in fp16 becomes
    +-2**-24 so that "stored non-zero" and "not pruned" coincide;
  * x ~ Laplace(0, 1) for attention / gate / up inputs, optionally with a
    seeded 1% of channels scaled by 20 (outliers); x = SiLU(g) * u with
    g, u ~ N(0, 1) for the down-projection input.
Seeds: seed = base * 1_000_003 + layer * 64 + proj * 4 + kind, with
proj in (q, k, v, o, gate, up, down) = 0..6 and kind in (W, mask, x, aux).
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import torch

PROJS = ("q", "k", "v", "o", "gate", "up", "down")
KIND_W, KIND_MASK, KIND_X, KIND_AUX = 0, 1, 2, 3
PRUNE_BLOCK = 128


def seed_of(base: int, layer: int, proj: int, kind: int) -> int:
    return base * 1_000_003 + layer * 64 + proj * 4 + kind


def _gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return g


def gen_weight(O: int, I: int, sigma: float, pw: float, prune: str, seed_w: int,
               seed_mask: int, device="cpu") -> torch.Tensor:
    """O x I fp16 weight with pruned entries set to zero."""
    g = _gen(seed_w, device)
    w32 = torch.randn((O, I), generator=g, device=device, dtype=torch.float32) * sigma
    w = w32.to(torch.float16)
    if pw <= 0.0:
        keep = torch.ones((O, I), dtype=torch.bool, device=device)
    elif prune == "bernoulli":
        gm = _gen(seed_mask, device)
        keep = torch.rand((O, I), generator=gm, device=device) >= pw
    elif prune == "magnitude":
        keep = torch.ones((O, I), dtype=torch.bool, device=device)
        a = w.abs().to(torch.float32)
        nfull = I // PRUNE_BLOCK
        if nfull:
            # all full blocks at once: [nb, O*128], flat index r*128 + c
            blk = a[:, : nfull * PRUNE_BLOCK].reshape(O, nfull, PRUNE_BLOCK).permute(1, 0, 2)
            blk = blk.reshape(nfull, O * PRUNE_BLOCK)
            n_prune = int(round(pw * O * PRUNE_BLOCK))
            if n_prune:
                order = torch.sort(blk, dim=1, stable=True).indices[:, :n_prune]
                kb = torch.ones_like(blk, dtype=torch.bool)
                kb.scatter_(1, order, False)
                keep[:, : nfull * PRUNE_BLOCK] = kb.view(nfull, O, PRUNE_BLOCK).permute(1, 0, 2) \
                    .reshape(O, nfull * PRUNE_BLOCK)
        for b0 in range(nfull * PRUNE_BLOCK, I, PRUNE_BLOCK):
            b1 = min(I, b0 + PRUNE_BLOCK)
            blk = a[:, b0:b1].reshape(-1)
            n_prune = int(round(pw * blk.numel()))
            if n_prune == 0:
                continue
            order = torch.sort(blk, stable=True).indices[:n_prune]
            kb = torch.ones(blk.numel(), dtype=torch.bool, device=device)
            kb[order] = False
            keep[:, b0:b1] = kb.view(O, b1 - b0)
    else:
        raise ValueError(f"unknown pruning mode {prune!r}")
    tiny = torch.where(w32 < 0, -2.0**-24, 2.0**-24).to(torch.float16)
    w = torch.where(keep & (w == 0), tiny, w)
    w = torch.where(keep, w, torch.zeros_like(w))
    return w


def gen_x_laplace(I: int, seed: int, device="cpu", outlier_frac: float = 0.0,
                  outlier_scale: float = 20.0, seed_aux: int | None = None) -> torch.Tensor:
    g = _gen(seed, device)
    u = torch.rand(I, generator=g, device=device, dtype=torch.float64) - 0.5
    x = -torch.sign(u) * torch.log1p(-2.0 * u.abs())
    x = x.to(torch.float32)
    if outlier_frac > 0:
        n_out = int(math.floor(outlier_frac * I))
        ga = _gen(seed_aux if seed_aux is not None else seed + 1, device)
        idx = torch.randperm(I, generator=ga, device=device)[:n_out]
        x[idx] = x[idx] * outlier_scale
    return x.to(torch.float16)


def gen_x_swiglu(I: int, seed: int, device="cpu") -> torch.Tensor:
    g = _gen(seed, device)
    gg = torch.randn(I, generator=g, device=device, dtype=torch.float32)
    uu = torch.randn(I, generator=g, device=device, dtype=torch.float32)
    return (torch.nn.functional.silu(gg) * uu).to(torch.float16)


@dataclass
class LayerShape:
    """One decoder layer: per projection (O, I)."""
    name: str
    shapes: dict = field(default_factory=dict)

    def O(self, p):
        return self.shapes[p][0]

    def I(self, p):
        return self.shapes[p][1]


def llama_shapes(hidden: int, kv: int, ffn: int, name: str) -> LayerShape:
    return LayerShape(name, {
        "q": (hidden, hidden), "k": (kv, hidden), "v": (kv, hidden),
        "o": (hidden, hidden), "gate": (ffn, hidden), "up": (ffn, hidden),
        "down": (hidden, ffn)})


LLAMA2_7B = llama_shapes(4096, 4096, 11008, "llama2-7b")
LLAMA3_8B = llama_shapes(4096, 1024, 14336, "llama3-8b")
LLAMA2_13B = llama_shapes(5120, 5120, 13824, "llama2-13b")
LLAMA2_70B = llama_shapes(8192, 1024, 28672, "llama2-70b")

# The five workloads (single layer / decoder layer / stacks).
WORKLOADS = {
    "single-4096": dict(shape=None, O=4096, I=4096, sigma=0.02, pw=0.5,
                        prune="bernoulli", px=50, x="laplace", layers=1),
    "llama2-7b-layer": dict(shape=LLAMA2_7B, sigma=0.02, pw=0.5, prune="magnitude",
                            px=50, px_sweep=(0, 25, 50, 70), layers=1),
    "llama3-8b-stack": dict(shape=LLAMA3_8B, sigma=0.02, pw=0.6, prune="magnitude",
                            px=50, layers=32),
    "llama2-13b-stack": dict(shape=LLAMA2_13B, sigma=0.02, pw=0.5, prune="magnitude",
                             px=50, pw_sweep=(0.4, 0.5, 0.6), px_sweep=(30, 50, 70),
                             outliers=0.01, layers=40),
    "llama2-70b-stack": dict(shape=LLAMA2_70B, sigma=0.01, pw=0.5, prune="magnitude",
                             px=50, layers=80),
}


def layer_weight(wl: dict, proj: str, layer: int = 0, base: int = 0, device="cpu",
                 pw: float | None = None) -> torch.Tensor:
    p = PROJS.index(proj)
    shape = wl["shape"]
    O, I = shape.shapes[proj]
    return gen_weight(O, I, wl["sigma"], wl["pw"] if pw is None else pw, wl["prune"],
                      seed_of(base, layer, p, KIND_W), seed_of(base, layer, p, KIND_MASK),
                      device)


def layer_input(wl: dict, proj: str, layer: int = 0, base: int = 0, device="cpu") -> torch.Tensor:
    """Input vector of a projection.  q/k/v share the q seed and gate/up share
    the gate seed (one sparsified input each, as in a real decoder layer)."""
    shape = wl["shape"]
    I = shape.shapes[proj][1]
    src = {"k": "q", "v": "q", "up": "gate"}.get(proj, proj)
    p = PROJS.index(src)
    if proj == "down":
        return gen_x_swiglu(I, seed_of(base, layer, p, KIND_X), device)
    return gen_x_laplace(I, seed_of(base, layer, p, KIND_X), device,
                         outlier_frac=wl.get("outliers", 0.0),
                         seed_aux=seed_of(base, layer, p, KIND_AUX))


def single_layer(O=4096, I=4096, sigma=0.02, pw=0.5, prune="bernoulli", base=0, device="cpu"):
    """The single out=in=4096 layer: fp16 W ~ N(0, 0.02) with a Bernoulli
    mask and x ~ Laplace(0, 1)."""
    W = gen_weight(O, I, sigma, pw, prune, seed_of(base, 0, 0, KIND_W),
                   seed_of(base, 0, 0, KIND_MASK), device)
    x = gen_x_laplace(I, seed_of(base, 0, 0, KIND_X), device)
    return W, x
