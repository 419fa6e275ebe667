"""Plain CPU oracle (numpy, fp64) for DuoGPT's calibration precompute.

TEST INFRASTRUCTURE ONLY (see the package docstring): only tests/, smoke()
and bench.py's baseline legs may import it; it shares no code with the CUDA
library.

What it computes follows §4.3 ("Efficient DuoGPT Algorithm") and the
precompute lines of Algorithm 1, in the paper's notation: W (n x k) is the
layer weight, the calibration input X (k x m) has one column per token; the
sparse input X_hat keeps, in every column, the channels of largest
magnitude (§3, "Activation Sparsity"); X_tilde is the dense input.

    H = X_hat X_hat^T,   L = Inverse_Cholesky(H)  (H^-1 = L L^T, L lower)
    dX = X_tilde - X_hat
    Q = dX X_hat^T L,    U = Q (.) M_u   (M_u: ones strictly above the diagonal)
    a = diag(dX dX^T),   b = diag(U U^T),   c = diag(Q) / diag(L),   D = U L^T
    S[:, p] = W[:, p]^2 (1 / L_pp^2 + a_p - b_p + 2 c_p)      (the efficient score)

Readings (the paper's calibration settings, App. B.1, plus points it leaves
open; each is listed in the design doc):
  * X_hat keeps, per token column, the keep = floor(k (100 - pct) / 100)
    channels of largest |x| (ties to the lower channel index), as the decode
    sparsifier does;
  * a channel whose Hessian diagonal is 0 (never kept) gets H_ii = 1;
  * act_order: channels are reordered by the Hessian diagonal, largest first
    (ties keep the lower index first), and every quantity is in that order;
    perm[i] is the original channel at position i.  The order is decided on
    the exact diagonal (a sum of squared fp16 values, compared as integers
    in units of 2^-48), so no rounding can reorder near-equal channels;
  * dampening: H += 0.1 * mean(diag(H)) * I, after the reordering;
  * X_tilde here is the dense input itself (one layer, no earlier pruned
    layer), so dX holds exactly the dropped activations.
"""
from __future__ import annotations

import numpy as np

from .duo_oracle import _as_f16, oracle_sparsify

DAMP = 0.1


def sparsify_columns(X16, keep: int):
    """X_hat: in every column (token) of the k x m input, the `keep`
    channels of largest |x| survive (ties to the lower index), the rest are
    zero (§3).  Returns fp16."""
    X = _as_f16(X16)
    k, m = X.shape
    Xh = np.zeros_like(X)
    for t in range(m):
        K, V = oracle_sparsify(X[:, t].copy(), keep)
        Xh[K.astype(np.int64), t] = V
    return Xh


def exact_diag_keys(Xh16) -> list[int]:
    """diag(X_hat X_hat^T) * 2^48 as exact Python integers (every fp16 value
    is an integer multiple of 2^-24)."""
    Xh = _as_f16(Xh16)
    v = np.abs((Xh.astype(np.float64) * 2.0**24).astype(np.int64))   # < 2^40
    hi, lo = v >> 20, v & ((1 << 20) - 1)                            # v = hi 2^20 + lo
    # v^2 = hi^2 2^40 + 2 hi lo 2^20 + lo^2; each column sum stays below 2^63
    shh = (hi * hi).sum(axis=1)
    shl = (hi * lo).sum(axis=1)
    sll = (lo * lo).sum(axis=1)
    return [(int(a) << 40) + (int(b) << 21) + int(c) for a, b, c in zip(shh, shl, sll)]


def oracle_calib_precompute(X16, keep: int, damp: float = DAMP, act_order: bool = True):
    """The precompute of Algorithm 1 (readings in the module docstring).

    Returns a dict of fp64 arrays in the act_order channel order: perm,
    H (dampened), L, dX, Xh (rows reordered), Q, U, a, b, c, D."""
    X = _as_f16(X16)
    k, m = X.shape
    Xh16 = sparsify_columns(X, keep)
    Xh = Xh16.astype(np.float64)
    Xt = X.astype(np.float64)
    H = Xh @ Xh.T
    key = exact_diag_keys(Xh16)
    dead = np.array([kk == 0 for kk in key])
    H[dead, dead] = 1.0
    key = [kk if kk != 0 else 1 << 48 for kk in key]   # H_ii = 1 for a dead channel
    if act_order:
        perm = np.array(sorted(range(k), key=lambda i: (-key[i], i)), dtype=np.int64)
    else:
        perm = np.arange(k)
    H = H[np.ix_(perm, perm)]
    Xh = Xh[perm]
    Xt = Xt[perm]
    H[np.diag_indices(k)] += damp * np.mean(np.diag(H))
    Hinv = np.linalg.inv(H)
    Hinv = (Hinv + Hinv.T) / 2
    L = np.linalg.cholesky(Hinv)
    dX = Xt - Xh
    Q = dX @ Xh.T @ L
    U = np.triu(Q, 1)
    a = np.sum(dX * dX, axis=1)
    b = np.sum(U * U, axis=1)
    c = np.diag(Q) / np.diag(L)
    D = U @ L.T
    return dict(perm=perm, H=H, L=L, dX=dX, Xh=Xh, Q=Q, U=U, a=a, b=b, c=c, D=D)


def oracle_calib_score(W16, pre) -> np.ndarray:
    """S = W^2 (1 / L_pp^2 + a - b + 2 c) per column p (the efficient score
    of §4.3), with W's columns in the act_order order of `pre`."""
    W = _as_f16(W16).astype(np.float64)[:, pre["perm"]]
    L = pre["L"]
    col = 1.0 / np.diag(L) ** 2 + pre["a"] - pre["b"] + 2.0 * pre["c"]
    return W * W * col[None, :]
