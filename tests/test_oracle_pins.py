"""Pins of the CPU oracle against things other than itself (CPU only).

Each test fixes a property that a plausible mistake in the oracle (a dropped
term, a wrong sign or index, a transposed operand, a wrong tie rule, an
off-by-one in the packer) would break:
  * exact integer arithmetic on fp16 (every fp16 is an integer * 2**-24);
  * the exactly-rounded sum math.fsum;
  * pure-Python brute force on tiny inputs (all k-subsets for the kept set);
  * closed forms: dense special case, k = 0, all-equal magnitudes, linearity;
  * a hand-worked fixture (tests/golden/tiny_worked_example.txt);
  * packer round trips and hand-derived record bytes.
"""
import itertools
import math
import os

import numpy as np
import pytest

import oracle as orc

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "tiny_worked_example.txt")
U = 2.0 ** -53   # fp64 unit roundoff


def _rand_w(rng, O, I, pw=0.5, scale=0.05):
    W = (rng.standard_normal((O, I)) * scale).astype(np.float16)
    W[rng.random((O, I)) < pw] = 0
    return W


def _rand_x(rng, I, ties=True):
    if ties:   # few distinct magnitudes -> many ties
        x = rng.integers(-4, 5, size=I).astype(np.float16) * np.float16(0.5)
    else:
        x = rng.laplace(0, 1, size=I).astype(np.float16)
    return x


# ---------------------------------------------------------------- golden ----

def _parse_golden():
    W, x, cases, recs = [], None, [], []
    with open(GOLDEN) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            tok = line.split()
            if tok[0] == "W":
                W.append([float(t) for t in tok[1:]])
            elif tok[0] == "x":
                x = [float(t) for t in tok[1:]]
            elif tok[0] == "case":
                k = int(tok[1].split("=")[1])
                yi = tok.index("y")
                K = [int(t) for t in tok[3:yi]]
                y = [float(t) for t in tok[yi + 1:]]
                cases.append((k, K, y))
            elif tok[0] == "thresh":
                tau = float(tok[1].split("=")[1])
                yi = tok.index("y")
                K = [int(t) for t in tok[3:yi]]
                y = [float(t) for t in tok[yi + 1:]]
                cases.append(("tau", tau, K, y))
            elif tok[0] == "cmb_record":
                j = int(tok[1].split("=")[1])
                word0 = int(tok[3])
                vi, ui = tok.index("vals"), tok.index("units")
                vals = [int(t, 16) for t in tok[vi + 1:ui]]
                recs.append((j, word0, vals, int(tok[ui + 1])))
    return np.array(W, dtype=np.float16), np.array(x, dtype=np.float16), cases, recs


def test_golden_hand_worked_example():
    W, x, cases, _ = _parse_golden()
    for case in cases:
        if case[0] == "tau":
            continue
        k, K, y = case
        Kc, vals = orc.oracle_sparsify(x, k)
        assert list(Kc) == K
        assert np.array_equal(vals.view(np.uint16), x[K].view(np.uint16))
        assert np.array_equal(orc.oracle_spmspv(W, x, k), np.array(y))


def test_golden_threshold_cases():
    W, x, cases, _ = _parse_golden()
    tcases = [c for c in cases if c[0] == "tau"]
    assert len(tcases) == 5
    for _, tau, K, y in tcases:
        Kc, vals = orc.oracle_sparsify_threshold(x, tau)
        assert list(Kc) == K
        assert np.array_equal(vals.view(np.uint16), x[K].view(np.uint16))
        assert np.array_equal(orc.oracle_spmspv_threshold(W, x, tau), np.array(y))
        assert np.array_equal(orc.oracle_spmspv_threshold(W, x, -tau), np.array(y))   # sign ignored


def test_threshold_equals_topk_between_magnitudes():
    """Two independent definitions agree: with no tie at the boundary, the
    channels above the (k+1)-th largest magnitude are the top-k set."""
    rng = np.random.default_rng(11)
    for trial in range(200):
        I = int(rng.integers(2, 300))
        x = rng.laplace(size=I).astype(np.float16)
        a = np.sort(np.abs(x.astype(np.float64)))[::-1]
        k = int(rng.integers(0, I))
        if k > 0 and a[k - 1] == a[k]:
            continue   # tie at the boundary: top-k breaks it by index, a threshold cannot
        Kt, _ = orc.oracle_sparsify_threshold(x, a[k])
        Kk, _ = orc.oracle_sparsify(x, k)
        assert np.array_equal(Kt, Kk)


def test_threshold_special_cases():
    x = np.array([0.0, -0.0, 1.5, -3.0, 0.0, 2.0, -1.5, 65504.0], dtype=np.float16)
    assert list(orc.oracle_sparsify_threshold(x, 0.0)[0]) == [2, 3, 5, 6, 7]   # the non-zeros
    assert list(orc.oracle_sparsify_threshold(x, 1.5)[0]) == [3, 5, 7]          # strict
    assert len(orc.oracle_sparsify_threshold(x, 65504.0)[0]) == 0
    assert len(orc.oracle_sparsify_threshold(x, np.inf)[0]) == 0
    inf_x = np.array([np.inf, -np.inf, 1.0], dtype=np.float16)
    assert list(orc.oracle_sparsify_threshold(inf_x, 65504.0)[0]) == [0, 1]
    with pytest.raises(ValueError):
        orc.oracle_sparsify_threshold(np.array([np.nan, 1.0], dtype=np.float16), 0.5)
    # nested: a larger threshold keeps a subset
    rng = np.random.default_rng(5)
    xr = rng.laplace(size=500).astype(np.float16)
    prev = set(range(500))
    for tau in (0.0, 0.1, 0.5, 1.0, 2.0, 4.0):
        cur = set(int(j) for j in orc.oracle_sparsify_threshold(xr, tau)[0])
        assert cur <= prev
        prev = cur


def test_golden_cmb_records():
    W, _, _, recs = _parse_golden()
    hdr, off, data = orc.ref_pack_cmb(W)
    assert hdr["nseg"] == 1 and hdr["nnz"] == int((W != 0).sum())
    for j, word0, vals, units in recs:
        b0 = int(off[j]) * 16
        assert int(off[j + 1] - off[j]) == units
        words = np.frombuffer(data[b0:b0 + 128].tobytes(), dtype="<u4")
        assert int(words[0]) == word0 and not words[1:].any()
        got = np.frombuffer(data[b0 + 128:b0 + 128 + 2 * len(vals)].tobytes(), dtype="<u2")
        assert [int(v) for v in got] == vals
        assert not data[b0 + 128 + 2 * len(vals): b0 + 16 * units].any()


# -------------------------------------------------------------- sparsify ----

def _brute_kept_set(x, k):
    """All k-subsets; the valid one has every kept j beating every dropped j'
    (|x_j| > |x_j'|, or equal and j < j')."""
    I = len(x)
    a = [abs(float(v)) for v in x]
    found = []
    for S in itertools.combinations(range(I), k):
        Sset = set(S)
        ok = all((a[j] > a[d]) or (a[j] == a[d] and j < d)
                 for j in S for d in range(I) if d not in Sset)
        if ok:
            found.append(list(S))
    assert len(found) == 1, "the kept set is unique"
    return found[0]


@pytest.mark.parametrize("I", [1, 2, 5, 8, 11])
def test_sparsify_matches_bruteforce(I):
    rng = np.random.default_rng(100 + I)
    for trial in range(6):
        x = _rand_x(rng, I, ties=(trial % 2 == 0))
        if trial == 5:
            x[:] = np.float16(0.0)
            x[::2] = np.float16(-0.0)
        for k in range(I + 1):
            K, vals = orc.oracle_sparsify(x, k)
            assert list(K) == _brute_kept_set(x, k)
            assert len(K) == k


def test_sparsify_all_equal_keeps_lowest_indices():
    for v in (1.5, -1.5, 0.0):
        x = np.full(37, v, dtype=np.float16)
        x[::3] = -x[::3]
        for k in (0, 1, 17, 37):
            K, _ = orc.oracle_sparsify(x, k)
            assert list(K) == list(range(k))


def test_sparsify_rejects_bad_k_and_nan():
    x = np.ones(4, dtype=np.float16)
    with pytest.raises(ValueError):
        orc.oracle_sparsify(x, 5)
    with pytest.raises(ValueError):
        orc.oracle_sparsify(x, -1)
    x[1] = np.float16(np.nan)
    with pytest.raises(ValueError):
        orc.oracle_sparsify(x, 2)


def test_fp16_magnitude_order_equals_integer_key_order():
    """For every finite or infinite fp16, ordering by |x| (fp64) equals
    ordering by the 15 low bits of the pattern; the CUDA selector relies on
    this IEEE property and the oracle on the magnitude definition."""
    keys = np.arange(0, 0x7C01, dtype=np.uint16)          # +0 .. +inf
    mags = np.abs(keys.view(np.float16).astype(np.float64))
    assert np.all(np.diff(mags) > 0)
    neg = (keys | 0x8000).view(np.float16)
    assert np.array_equal(np.abs(neg.astype(np.float64)), mags)


def test_k_from_pct():
    assert orc.k_from_pct(4096, 50) == 2048
    assert orc.k_from_pct(11008, 70) == 3302
    assert orc.k_from_pct(11008, 25) == 8256
    assert orc.k_from_pct(7, 0) == 7 and orc.k_from_pct(7, 100) == 0


# ---------------------------------------------------------------- spmspv ----

def _bound(W, x, K):
    Kl = np.asarray(K, dtype=np.int64)
    s = np.abs(W[:, Kl].astype(np.float64)) @ np.abs(x[Kl].astype(np.float64))
    return (len(K) + 2) * U * s


@pytest.mark.parametrize("O,I,pw,k", [(7, 9, 0.5, 4), (33, 65, 0.3, 40), (130, 257, 0.6, 100),
                                      (64, 300, 0.0, 300), (5, 40, 0.9, 1)])
def test_spmspv_exact_integer(O, I, pw, k):
    rng = np.random.default_rng(O * 1000 + I)
    W = _rand_w(rng, O, I, pw)
    x = _rand_x(rng, I, ties=False)
    y = orc.oracle_spmspv(W, x, k)
    K, _ = orc.oracle_sparsify(x, k)
    ex = orc.exact_spmspv_rows_scaled(W, x, K)
    for i in range(O):
        exact = ex[i] / 2.0 ** 48       # one rounding of the exact value
        assert abs(y[i] - exact) <= _bound(W, x, K)[i] + abs(exact) * U
    assert np.all(np.abs(y - orc.fsum_spmspv_rows(W, x, K)) <= _bound(W, x, K))


def test_spmspv_pure_python_bruteforce():
    rng = np.random.default_rng(7)
    for O, I in ((1, 1), (3, 4), (6, 5), (2, 12)):
        W = _rand_w(rng, O, I, 0.4)
        x = _rand_x(rng, I)
        for k in range(I + 1):
            K = _brute_kept_set(x, k)
            want = [0.0] * O
            for i in range(O):
                terms = [float(W[i, j]) * float(x[j]) for j in K if float(W[i, j]) != 0.0]
                want[i] = math.fsum(terms)
            got = orc.oracle_spmspv(W, x, k)
            assert np.allclose(got, want, rtol=0, atol=1e-12)


def test_dense_special_case_is_plain_gemv():
    """p^w = p^x = 0: y is the dense GEMV, checked with exact integers."""
    rng = np.random.default_rng(3)
    O, I = 40, 96
    W = (rng.standard_normal((O, I)) * 0.1).astype(np.float16)
    x = rng.standard_normal(I).astype(np.float16)
    y = orc.oracle_spmspv(W, x, I)
    ex = orc.exact_spmspv_rows_scaled(W, x, np.arange(I))
    b = _bound(W, x, np.arange(I))
    for i in range(O):
        assert abs(y[i] - ex[i] / 2.0 ** 48) <= b[i] + abs(ex[i]) / 2.0 ** 48 * U


def test_k_zero_gives_zero_and_row_bound_zero():
    rng = np.random.default_rng(4)
    W = _rand_w(rng, 9, 13)
    x = _rand_x(rng, 13)
    assert not orc.oracle_spmspv(W, x, 0).any()
    assert not orc.tolerance_rows(W, x, []).any()


def test_linearity_scaling_and_additivity():
    rng = np.random.default_rng(5)
    O, I, k = 50, 80, 30
    W = _rand_w(rng, O, I)
    x = _rand_x(rng, I, ties=False)
    y1 = orc.oracle_spmspv(W, x, k)
    y2 = orc.oracle_spmspv(W, (x.astype(np.float32) * 2).astype(np.float16), k)
    assert np.array_equal(y2, 2 * y1)            # power-of-two scaling is exact
    # additivity for a fixed kept set: W[:,K](x1+x2) = W[:,K]x1 + W[:,K]x2
    K, _ = orc.oracle_sparsify(x, k)
    x1 = np.zeros(I, np.float16)
    x2 = np.zeros(I, np.float16)
    Kl = K.astype(np.int64)
    x1[Kl[::2]] = x[Kl[::2]]
    x2[Kl[1::2]] = x[Kl[1::2]]
    ya = orc.oracle_spmspv(W, x1, k) + orc.oracle_spmspv(W, x2, k)
    assert np.all(np.abs(ya - y1) <= 2 * _bound(W, x, K))


def test_transposed_operand_is_caught():
    """W x differs from W^T x on a non-symmetric square case: the oracle uses
    columns of W for channels (§3: W[:, i] multiplies x_i)."""
    W = np.zeros((3, 3), np.float16)
    W[0, 2] = 1
    x = np.array([0, 0, 1], np.float16)
    assert list(orc.oracle_spmspv(W, x, 3)) == [1.0, 0.0, 0.0]


# ---------------------------------------------------------------- packers ----

@pytest.mark.parametrize("O,I", [(1, 1), (31, 3), (32, 2), (1023, 2), (1024, 3), (1025, 2),
                                 (2100, 3), (5, 17)])
def test_cmb_round_trip_and_structure(O, I):
    rng = np.random.default_rng(O + 7 * I)
    W = _rand_w(rng, O, I, pw=0.5)
    if I >= 2:
        W[:, 0] = 0                             # an empty channel
        W[:, 1] = np.float16(0.5)               # a full channel
    W[0, -1] = np.float16(-0.0)                 # -0 counts as pruned
    hdr, off, data = orc.ref_pack_cmb(W)
    S = (O + 1023) // 1024
    assert hdr["nseg"] == S and hdr["out"] == O and hdr["inp"] == I
    assert hdr["nnz"] == int((W != 0).sum())
    assert off.dtype == np.uint32 and off.size == I * S + 1 and off[0] == 0
    assert len(data) == 16 * int(off[-1])
    canon = np.where(W == 0, np.float16(0), W)
    assert np.array_equal(orc.ref_unpack_cmb(hdr, off, data).view(np.uint16), canon.view(np.uint16))
    for j in range(I):
        for s in range(S):
            b0 = int(off[j * S + s]) * 16
            words = np.frombuffer(data[b0:b0 + 128].tobytes(), dtype="<u4")
            n = sum(bin(int(w)).count("1") for w in words)
            assert int(off[j * S + s + 1] - off[j * S + s]) * 16 == (128 + 2 * n + 15) // 16 * 16
            nrows = min(O, (s + 1) * 1024) - s * 1024
            bits = np.unpackbits(words.view(np.uint8), bitorder="little")
            assert not bits[nrows:].any()        # tail rows carry no bits


def test_cmb_single_nonzero_position():
    """Closed form of the bit convention: a lone non-zero at (r, j) sets bit
    r % 32 of word (r % 1024) // 32 in record (j, r // 1024)."""
    O, I = 2500, 3
    for r in (0, 31, 32, 1023, 1024, 2047, 2499):
        W = np.zeros((O, I), np.float16)
        W[r, 1] = np.float16(-3.0)
        hdr, off, data = orc.ref_pack_cmb(W)
        S = hdr["nseg"]
        s = r // 1024
        b0 = int(off[1 * S + s]) * 16
        words = np.frombuffer(data[b0:b0 + 128].tobytes(), dtype="<u4")
        want = np.zeros(32, np.uint32)
        want[(r % 1024) // 32] = 1 << (r % 32)
        assert np.array_equal(words, want)
        assert data[b0 + 128] == 0x00 and data[b0 + 129] == 0xC2    # -3.0 = 0xC200
        assert hdr["nnz"] == 1


@pytest.mark.parametrize("O,I", [(1, 1), (17, 9), (300, 4)])
def test_idx16_round_trip_and_structure(O, I):
    rng = np.random.default_rng(O * 3 + I)
    W = _rand_w(rng, O, I, pw=0.6)
    hdr, colptr, cnt, data = orc.ref_pack_idx16(W)
    canon = np.where(W == 0, np.float16(0), W)
    assert np.array_equal(orc.ref_unpack_idx16(hdr, colptr, cnt, data).view(np.uint16),
                          canon.view(np.uint16))
    for j in range(I):
        n = int(cnt[j])
        assert n == int((W[:, j] != 0).sum())
        assert int(colptr[j + 1] - colptr[j]) == 2 * ((2 * n + 15) // 16 * 16)
        r0 = int(colptr[j]) + (2 * n + 15) // 16 * 16
        rows = np.frombuffer(data[r0:r0 + 2 * n].tobytes(), dtype="<u2")
        assert np.all(np.diff(rows.astype(np.int64)) > 0)


# ------------------------------------------------------ bytes and loads ----

def test_required_bytes_closed_form():
    nnz = np.array([3, 0, 5, 8])
    # K = {0, 2}: 2*(3+5) value bytes + 2 * 16/8 mask bytes + 2*4 (x) + 4*2 + 4*16
    assert orc.required_bytes(nnz, [0, 2], O=16, I=4) == 16 + 4 + 8 + 8 + 64


def test_loaded_fraction_matches_dual_sparsity_product():
    """§5: about (1 - p^w)(1 - p^x) of the weights are loaded when the kept
    channels are independent of the weight mask; the App. B.3 worst case
    (densest channels) bounds it from above."""
    rng = np.random.default_rng(11)
    O, I, pw = 512, 1024, 0.5
    keep = rng.random((O, I)) >= pw
    nnz = keep.sum(0)
    for px in (0, 30, 50, 70):
        k = orc.k_from_pct(I, px)
        K = np.sort(rng.permutation(I)[:k])
        f = orc.loaded_fraction(nnz, K, O, I)
        expect = (1 - pw) * (1 - px / 100)
        assert abs(f - expect) < 0.01
        assert orc.worst_case_loaded_fraction(nnz, k, O, I) >= f - 1e-12
    assert orc.loaded_fraction(nnz, np.arange(I), O, I) == nnz.sum() / (O * I)


def _worst_case_cases():
    """Tiny layers with channel non-zero counts spread out (distinct enough
    that the densest, sparsest and first-k sets all differ)."""
    out = []
    for seed in range(6):
        rng = np.random.default_rng(100 + seed)
        O, I = 7, int(rng.integers(5, 11))
        keep = rng.random((O, I)) < rng.uniform(0.2, 0.8, size=I)
        out.append((O, I, keep.sum(0)))
    return out


def test_worst_case_loaded_fraction_is_the_max_over_kept_sets():
    """App. B.3 bounds the loaded fraction by the case where the k densest
    channels are the kept ones: over every k-subset K of a tiny layer, the
    largest Σ_{j∈K} nnz_j / (O I) must equal the function, exactly (integer
    sums over the same denominator)."""
    for O, I, nnz in _worst_case_cases():
        for k in range(I + 1):
            best = max(sum(int(nnz[j]) for j in K) for K in itertools.combinations(range(I), k))
            assert orc.worst_case_loaded_fraction(nnz, k, O, I) == best / (O * I), (O, I, k)
