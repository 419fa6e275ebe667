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
open):
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


def oracle_calib_prune(W16, pre, pw_pct: int, block: int = 128):
    """Algorithm 1's column sweep (§4.3) after the precompute `pre`, written
    unblocked: columns in the processing order; at the first column of every
    block of `block` columns, the scores of the block's current weights
    S = W^2 (1 / L_pp^2 + a - b + 2 c) decide its mask: the
    floor(n * B_j * pw_pct / 100) weights of the block with the lowest scores
    are pruned (equal scores: the lower flat index r * B_j + c first); then
    for each column j, P_j = W_j (.) M_j, E_j = (W_j - P_j) / L_jj, and every
    later column q gets W_q -= E_j L_qj - W_j D_jq (W_j as it is at step j),
    after which W_j = P_j.  This equals the blocked form with lazy batch
    updates when the trailing columns see the same W_j (the reading taken).

    Returns (W_pruned fp64 n x k in the ORIGINAL channel order, keep mask
    bool n x k in the original order)."""
    W = _as_f16(W16).astype(np.float64)
    n, k = W.shape
    perm = pre["perm"]
    L, D = pre["L"], pre["D"]
    col = 1.0 / np.diag(L) ** 2 + pre["a"] - pre["b"] + 2.0 * pre["c"]
    Wp = W[:, perm].copy()
    keep = np.ones((n, k), dtype=bool)
    for i in range(0, k, block):
        bj = min(block, k - i)
        S = Wp[:, i:i + bj] ** 2 * col[None, i:i + bj]
        cnt = (n * bj * pw_pct) // 100
        flat = S.reshape(-1)
        order = np.lexsort((np.arange(flat.size), flat))     # score, then flat index
        m = np.ones(flat.size, dtype=bool)
        m[order[:cnt]] = False
        keep[:, i:i + bj] = m.reshape(n, bj)
        for j in range(i, i + bj):
            wj = Wp[:, j].copy()
            pj = np.where(keep[:, j], wj, 0.0)
            E = (wj - pj) / L[j, j]
            if j + 1 < k:
                Wp[:, j + 1:] -= np.outer(E, L[j + 1:, j]) - np.outer(wj, D[j, j + 1:])
            Wp[:, j] = pj
    out = np.zeros_like(Wp)
    out[:, perm] = Wp
    mask = np.zeros_like(keep)
    mask[:, perm] = keep
    return out, mask


def oracle_calib_prune_blocked(W16, pre, pw_pct: int, block: int = 128):
    """The same sweep in Algorithm 1's blocked form: within a block the
    updates reach only the block's columns; at the block's end the trailing
    columns get W_T -= E L_T,blk^T - W_pre D_blk,T in one product (lazy
    batch), W_pre holding each block column as it was at its step."""
    W = _as_f16(W16).astype(np.float64)
    n, k = W.shape
    perm = pre["perm"]
    L, D = pre["L"], pre["D"]
    col = 1.0 / np.diag(L) ** 2 + pre["a"] - pre["b"] + 2.0 * pre["c"]
    Wp = W[:, perm].copy()
    keep = np.ones((n, k), dtype=bool)
    for i in range(0, k, block):
        bj = min(block, k - i)
        S = Wp[:, i:i + bj] ** 2 * col[None, i:i + bj]
        cnt = (n * bj * pw_pct) // 100
        flat = S.reshape(-1)
        order = np.lexsort((np.arange(flat.size), flat))
        m = np.ones(flat.size, dtype=bool)
        m[order[:cnt]] = False
        keep[:, i:i + bj] = m.reshape(n, bj)
        E = np.zeros((n, bj))
        Wpre = np.zeros((n, bj))
        for jj in range(bj):
            j = i + jj
            Wpre[:, jj] = Wp[:, j]
            pj = np.where(keep[:, j], Wp[:, j], 0.0)
            E[:, jj] = (Wp[:, j] - pj) / L[j, j]
            if jj + 1 < bj:
                Wp[:, j + 1:i + bj] -= np.outer(E[:, jj], L[j + 1:i + bj, j]) - np.outer(Wpre[:, jj], D[j, j + 1:i + bj])
            Wp[:, j] = pj
        if i + bj < k:
            T = slice(i + bj, k)
            Wp[:, T] -= E @ L[T, i:i + bj].T - Wpre @ D[i:i + bj, T]
    out = np.zeros_like(Wp)
    out[:, perm] = Wp
    mask = np.zeros_like(keep)
    mask[:, perm] = keep
    return out, mask
