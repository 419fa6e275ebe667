"""Pins of the calibration-precompute oracle (§4.3, Algorithm 1) against
things other than itself (CPU only):
  * a hand-worked fixture (tests/golden/calib_worked_example.txt);
  * the unvectorised definitions: b_p, c_p and the compensation row D_p from
    the inverse Hessian after sequential Gaussian elimination (§3's update
    rule), and 1 / [H^-1]_pp, against the Cholesky forms the efficient
    algorithm uses (App. A.2-A.4 state these are equal);
  * the R-decomposed score (Eq. 5 of §4.3, before a, b, c are named) against
    the efficient score;
  * closed forms: no activation sparsity (X_hat = X) gives dX = 0, so
    a = b = c = D = 0 and S is SparseGPT's W^2 / [H^-1]_pp;
  * invariants of L, of the act_order permutation and of X_hat.
"""
import math
import os

import numpy as np
import pytest

import oracle as orc

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "calib_worked_example.txt")


def _parse_golden():
    env = {"sqrt": math.sqrt, "__builtins__": {}}
    out = {}
    with open(GOLDEN) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            name, val = [p.strip() for p in line.split("=", 1)]
            rows = [[eval(tok, env) for tok in r.split()] for r in val.split(";")]
            out[name] = np.array(rows if len(rows) > 1 else rows[0], dtype=np.float64)
    return out


def test_golden_worked_example():
    g = _parse_golden()
    X = g["X"].astype(np.float16)
    pre = orc.oracle_calib_precompute(X, int(g["keep"].reshape(-1)[0]))
    assert pre["perm"].tolist() == g["perm"].astype(int).tolist()
    for name in ("H", "L", "Q", "U", "a", "b", "c", "D"):
        np.testing.assert_allclose(pre[name], g[name], rtol=1e-12, atol=1e-15, err_msg=name)
    S = orc.oracle_calib_score(g["W"].astype(np.float16)[None, :], pre)
    np.testing.assert_allclose(S[0], g["S"], rtol=1e-12)


def _inputs(rng, k, m, dead=False, ties=False):
    X = rng.laplace(0, 1, size=(k, m)).astype(np.float16)
    if dead:
        X[3] = np.float16(1e-3)      # never among the largest: a channel with H_ii = 0
    if ties:
        X[5] = X[6]                  # two channels with equal Hessian diagonals
    return X


def _naive(pre):
    """b, c, D and [H^-1]_pp by sequential Gaussian elimination of H^-1 in
    the processing order (§3's update rule applied column after column)."""
    H, dX, Xh = pre["H"], pre["dX"], pre["Xh"]
    k = H.shape[0]
    cur = np.linalg.inv(H)
    b = np.zeros(k)
    c = np.zeros(k)
    hpp = np.zeros(k)
    D = np.zeros((k, k))
    for p in range(k):
        z = dX[p] @ Xh.T                 # dX_p X_hat^T
        hpp[p] = cur[p, p]
        c[p] = z @ cur[:, p] / cur[p, p]
        cur = cur - np.outer(cur[:, p], cur[p, :]) / cur[p, p]   # H^-1_{-p}
        b[p] = z @ cur @ z
        D[p] = z @ cur
    return b, c, D, hpp


@pytest.mark.parametrize("act_order", [True, False])
@pytest.mark.parametrize("k,m,keep,dead,ties", [(6, 9, 3, False, False), (12, 20, 6, True, True),
                                                 (16, 40, 4, False, True)])
def test_efficient_terms_equal_sequential_elimination(act_order, k, m, keep, dead, ties):
    rng = np.random.default_rng(k * 100 + m)
    X = _inputs(rng, k, m, dead, ties)
    pre = orc.oracle_calib_precompute(X, keep, act_order=act_order)
    b, c, D, hpp = _naive(pre)
    L = pre["L"]
    scale = np.abs(D).max() + 1e-300
    np.testing.assert_allclose(pre["b"], b, rtol=1e-9, atol=1e-12 * np.abs(b).max())
    np.testing.assert_allclose(pre["c"], c, rtol=1e-9, atol=1e-12 * (np.abs(c).max() + 1))
    np.testing.assert_allclose(pre["D"], D, rtol=1e-8, atol=1e-11 * scale)
    np.testing.assert_allclose(np.diag(L) ** 2, hpp, rtol=1e-10)


def test_score_equals_r_decomposed_form():
    """S from the named terms against S written out from the residual
    decomposition R_p = W_:,p dX_p (before a, b and c are named)."""
    rng = np.random.default_rng(7)
    k, m, n = 10, 24, 5
    X = _inputs(rng, k, m)
    W = (rng.standard_normal((n, k)) * 0.02).astype(np.float16)
    pre = orc.oracle_calib_precompute(X, 5)
    S = orc.oracle_calib_score(W, pre)
    Wp = W.astype(np.float64)[:, pre["perm"]]
    H, dX, Xh = pre["H"], pre["dX"], pre["Xh"]
    cur = np.linalg.inv(H)
    for p in range(k):
        hpp = cur[p, p]
        colp = cur[:, p].copy()
        nxt = cur - np.outer(cur[:, p], cur[p, :]) / hpp
        for i in range(n):
            w = Wp[i, p]
            Rp = w * dX[p]                               # row i of R_p
            term2 = Rp @ Rp
            term3 = (w * dX[p] @ Xh.T) @ nxt @ (Xh @ dX[p] * w)
            term4 = 2 * w / hpp * (w * dX[p] @ Xh.T @ colp)
            want = w * w / hpp + term2 - term3 + term4
            assert abs(S[i, p] - want) <= 1e-9 * (abs(want) + w * w / hpp)
        cur = nxt


def test_no_activation_sparsity_reduces_to_sparsegpt():
    rng = np.random.default_rng(3)
    k, m = 12, 30
    X = _inputs(rng, k, m)
    W = (rng.standard_normal((4, k)) * 0.02).astype(np.float16)
    pre = orc.oracle_calib_precompute(X, k)
    for name in ("dX", "a", "b", "c", "D", "Q", "U"):
        assert np.all(pre[name] == 0), name
    S = orc.oracle_calib_score(W, pre)
    Hinv = np.linalg.inv(pre["H"])
    hpp = np.zeros(k)
    cur = Hinv.copy()
    for p in range(k):
        hpp[p] = cur[p, p]
        cur = cur - np.outer(cur[:, p], cur[p, :]) / cur[p, p]
    Wp = W.astype(np.float64)[:, pre["perm"]]
    np.testing.assert_allclose(S, Wp * Wp / hpp[None, :], rtol=1e-10)


def test_invariants_of_L_perm_and_sparse_input():
    rng = np.random.default_rng(11)
    k, m, keep = 16, 33, 7
    X = _inputs(rng, k, m, dead=True, ties=True)
    pre = orc.oracle_calib_precompute(X, keep)
    L, H = pre["L"], pre["H"]
    assert np.all(np.triu(L, 1) == 0) and np.all(np.diag(L) > 0)
    np.testing.assert_allclose(L @ L.T @ H, np.eye(k), atol=1e-9)
    # act_order: largest undampened diagonal first, ties by channel index
    Xh = orc.sparsify_columns(X, keep).astype(np.float64)
    d = np.diag(Xh @ Xh.T).copy()
    d[d == 0] = 1.0
    order = sorted(range(k), key=lambda i: (-d[i], i))
    assert pre["perm"].tolist() == order
    # dampening: H = P (X_hat X_hat^T, dead fixed) P^T + 0.1 mean(diag) I
    Hd = (Xh @ Xh.T)
    Hd[np.diag_indices(k)] = d
    Hd = Hd[np.ix_(order, order)]
    np.testing.assert_allclose(H, Hd + 0.1 * np.mean(d) * np.eye(k), rtol=1e-12)
    # X_hat: exactly `keep` survivors per token, none smaller than a dropped one
    Xs = orc.sparsify_columns(X, keep).astype(np.float64)
    for t in range(m):
        kept = Xs[:, t] != 0
        assert (np.abs(X[:, t].astype(np.float64)) > 0).sum() < keep or kept.sum() == keep
        if kept.any() and (~kept).any():
            assert np.abs(X[kept, t].astype(np.float64)).min() >= np.abs(X[~kept, t].astype(np.float64)).max()
    # a = per-channel energy of the dropped activations
    np.testing.assert_allclose(pre["a"], np.sum(pre["dX"] ** 2, axis=1))
    assert np.all(pre["dX"] * pre["Xh"] == 0)   # each entry is kept or dropped, not both


# ------------------------------------------------------------ column sweep ----

def test_sweep_golden_cases():
    g = _parse_golden()
    pre = orc.oracle_calib_precompute(g["X"].astype(np.float16), 1)
    for wn, rn in (("Wsweep1", "result1"), ("Wsweep2", "result2")):
        W = g[wn].astype(np.float16)[None, :]
        Wf, keep = orc.oracle_calib_prune(W, pre, 50, block=2)
        np.testing.assert_allclose(Wf[0], g[rn], rtol=1e-12, atol=1e-15)
        assert keep[0].tolist() == [bool(v != 0) for v in g[rn]]


def _sweep_inputs(seed, n, k, m, keep):
    rng = np.random.default_rng(seed)
    X = rng.laplace(0, 1, size=(k, m)).astype(np.float16)
    W = (rng.standard_normal((n, k)) * 0.05).astype(np.float16)
    return X, W, orc.oracle_calib_precompute(X, keep)


@pytest.mark.parametrize("n,k,m,keep,block,pw", [(8, 24, 40, 12, 8, 50), (5, 30, 50, 10, 7, 60),
                                                 (6, 16, 30, 16, 16, 25)])
def test_sweep_blocked_equals_unblocked(n, k, m, keep, block, pw):
    """Algorithm 1's blocked form (lazy batch updates) against the column by
    column form: the same masks and, up to rounding, the same weights."""
    X, W, pre = _sweep_inputs(n * k + m, n, k, m, keep)
    Wu, mu = orc.oracle_calib_prune(W, pre, pw, block)
    Wb, mb = orc.oracle_calib_prune_blocked(W, pre, pw, block)
    assert np.array_equal(mu, mb)
    np.testing.assert_allclose(Wb, Wu, rtol=1e-10, atol=1e-12 * np.abs(Wu).max())


def test_sweep_masks_and_pruned_zeros():
    n, k, m, block, pw = 10, 40, 60, 16, 50
    X, W, pre = _sweep_inputs(9, n, k, m, 20)
    Wf, keep = orc.oracle_calib_prune(W, pre, pw, block)
    assert np.all(Wf[~keep] == 0)
    kp = keep[:, pre["perm"]]                       # processing order
    for i in range(0, k, block):
        bj = min(block, k - i)
        assert (~kp[:, i:i + bj]).sum() == (n * bj * pw) // 100
    # the first block's decision is on the original weights: its pruned
    # scores are all at or below its kept ones
    col = 1.0 / np.diag(pre["L"]) ** 2 + pre["a"] - pre["b"] + 2 * pre["c"]
    S0 = W.astype(np.float64)[:, pre["perm"][:block]] ** 2 * col[:block]
    assert S0[~kp[:, :block]].max() <= S0[kp[:, :block]].min()


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_sweep_compensation_lowers_the_calibration_loss(seed):
    """The point of the sweep (§4.2): with the same mask, the compensated
    weights reproduce the dense output W X_tilde from the sparse input better
    than the masked weights alone."""
    n, k, m = 12, 48, 200
    X, W, pre = _sweep_inputs(100 + seed, n, k, m, 24)
    Wf, keep = orc.oracle_calib_prune(W, pre, 50, 16)
    Xh = orc.sparsify_columns(X, 24).astype(np.float64)
    target = W.astype(np.float64) @ X.astype(np.float64)
    loss_comp = np.linalg.norm(Wf @ Xh - target)
    loss_mask = np.linalg.norm(np.where(keep, W.astype(np.float64), 0.0) @ Xh - target)
    assert loss_comp < loss_mask
