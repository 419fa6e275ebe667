"""Pins of the quantised-value oracle (§5, weight-only quantisation with
channel-wise RTN and group size 128, Table 4) against things other than
itself (CPU only):
  * a hand-worked fixture (tests/golden/quant_worked_example.txt);
  * brute force in exact rational arithmetic: the nearest fp16 scale, the
    nearest zero point and, per weight, the nearest grid point in range
    (ties to an even offset from z), searched over every code;
  * closed forms: weights placed on a grid come back exactly; the error
    bound of round-to-nearest;
  * exact integer arithmetic for y from the codes themselves;
  * packer round trips and hand-derived record and table bytes.
"""
import math
import os
from fractions import Fraction

import numpy as np
import pytest

import oracle as orc

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "quant_worked_example.txt")


def _expand(tokens):
    out = []
    for t in tokens:
        if "*" in t:
            v, n = t.split("*")
            out += [v] * int(n)
        else:
            out.append(t)
    return out


def _parse_golden():
    rows = []
    with open(GOLDEN) as f:
        for line in f:
            line = line.strip()
            if not line.startswith("qrow"):
                continue
            parts = [p.split() for p in line.split("|")]
            bits = int(parts[0][1])
            fields = {p[0]: _expand(p[1:]) for p in parts[1:]}
            rows.append(dict(
                bits=bits,
                w=[float(v) for v in fields["w"]],
                s=[int(v, 16) for v in fields["s"]],
                z=[int(v) for v in fields["z"]],
                q=[None if v == "-" else int(v) for v in fields["q"]],
                what=[float(v) for v in fields["what"]]))
    return rows


def test_golden_rows():
    rows = _parse_golden()
    assert len(rows) == 9
    for r in rows:
        W = np.array([r["w"]], dtype=np.float16)
        q, s16, z = orc.oracle_quantize_rtn(W, r["bits"])
        assert s16[0].view(np.uint16).tolist() == r["s"], r
        assert z[0].tolist() == r["z"], r
        got_q = [None if r["w"][j] == 0 else int(q[0, j]) for j in range(W.shape[1])]
        assert got_q == r["q"], r
        deq = orc.oracle_dequantize(W, r["bits"])[0]
        assert deq.tolist() == r["what"], r


# ------------------------------------------------------------ brute force ----

def _fp16_value(bits):
    return Fraction(float(np.uint16(bits).view(np.float16)))


def _fp16_nearest(r: Fraction) -> int:
    """Bits of the fp16 nearest to r >= 0 (ties to an even significand),
    found by exact comparison, not by a float conversion."""
    assert r >= 0
    if r == 0:
        return 0
    if r < Fraction(1, 2**14):           # subnormal: multiples of 2**-24
        m = round(r * 2**24)             # Fraction rounds half to even
        return int(m)                    # m == 1024 is the smallest normal's bits
    e = 0
    while r >= Fraction(2) ** (e + 1):
        e += 1
    while r < Fraction(2) ** e:
        e -= 1
    m = round((r / Fraction(2) ** e - 1) * 1024)   # half to even
    if m == 1024:
        e, m = e + 1, 0
    assert -14 <= e <= 15
    return ((e + 15) << 10) | int(m)


def _brute_group(w_vals, bits):
    """(s bits, z, codes) of one group by exact search."""
    maxq = (1 << bits) - 1
    ws = [Fraction(float(v)) for v in w_vals]
    nzv = [v for v in ws if v != 0]
    lo = min([Fraction(0)] + nzv)
    hi = max([Fraction(0)] + nzv)
    if hi == lo:
        sb = 0x3C00
    else:
        sb = _fp16_nearest((hi - lo) / maxq)
        if sb == 0:
            sb = 1
    s = _fp16_value(sb)
    z = min(max(round(-lo / s), 0), maxq)
    codes = []
    for v in ws:
        if v == 0:
            codes.append(None)
            continue
        best = None
        for c in range(maxq + 1):
            d = abs(v - s * (c - z))
            key = (d, (c - z) % 2)        # nearest, then an even offset from z
            if best is None or key < best[0]:
                best = (key, c)
        codes.append(best[1])
    return sb, z, codes


@pytest.mark.parametrize("bits", [8, 4])
def test_brute_force_groups(bits):
    rng = np.random.default_rng(10 + bits)
    for trial in range(60 if bits == 4 else 16):   # every one of 2**b codes is tried
        O, I = 3, int(rng.integers(1, 300 if bits == 4 else 160))
        kind = trial % 4
        if kind == 0:     # Gaussian weights, half pruned
            W = (rng.standard_normal((O, I)) * 0.02).astype(np.float16)
            W[rng.random((O, I)) < 0.5] = 0
        elif kind == 1:   # one-signed groups
            W = (np.abs(rng.standard_normal((O, I))) * (1 if (trial // 4) % 2 else -1)).astype(np.float16)
        elif kind == 2:   # few distinct values: half-way cases on power-of-two grids
            W = (rng.integers(-8, 9, size=(O, I)) * 0.125).astype(np.float16)
        else:             # wide dynamic range, tiny values included
            W = (rng.standard_normal((O, I)) * 2.0 ** rng.integers(-20, 4, size=(O, I))).astype(np.float16)
        q, s16, z = orc.oracle_quantize_rtn(W, bits)
        for i in range(O):
            for g in range((I + 127) // 128):
                c0, c1 = 128 * g, min(I, 128 * g + 128)
                sb, zz, codes = _brute_group(W[i, c0:c1], bits)
                assert int(s16[i, g].view(np.uint16)) == sb, (trial, i, g)
                assert int(z[i, g]) == zz, (trial, i, g)
                for c, want in zip(range(c0, c1), codes):
                    if want is not None:
                        assert int(q[i, c]) == want, (trial, i, c)


@pytest.mark.parametrize("bits", [8, 4])
def test_weights_on_a_grid_come_back_exactly(bits):
    """W = s (q - z) with s a power of two and both ends of the code range
    present reproduces q, z and W exactly."""
    maxq = (1 << bits) - 1
    rng = np.random.default_rng(bits)
    O, I = 5, 256 + 37
    G = (I + 127) // 128
    W = np.zeros((O, I), dtype=np.float16)
    want_q = np.zeros((O, I), dtype=np.int64)
    for i in range(O):
        for g in range(G):
            c0, c1 = 128 * g, min(I, 128 * g + 128)
            s = 2.0 ** int(rng.integers(-12, -4))
            zz = int(rng.integers(1, maxq))
            codes = rng.integers(0, maxq + 1, size=c1 - c0)
            codes[0], codes[-1] = 0, maxq
            codes[codes == zz] = 0            # keep every stored weight non-zero
            W[i, c0:c1] = (s * (codes - zz)).astype(np.float16)
            want_q[i, c0:c1] = codes
    q, s16, z = orc.oracle_quantize_rtn(W, bits)
    assert np.array_equal(q, want_q)
    assert np.array_equal(orc.oracle_dequantize(W, bits), W.astype(np.float64))


@pytest.mark.parametrize("bits", [8, 4])
def test_rtn_error_bound(bits):
    """|w_hat - w| <= s/2 up to the fp16 rounding of s (at most maxq * 2**-11
    grid steps at the ends of the range)."""
    maxq = (1 << bits) - 1
    rng = np.random.default_rng(20 + bits)
    W = (rng.standard_normal((64, 500)) * 0.02).astype(np.float16)
    W[rng.random(W.shape) < 0.5] = 0
    q, s16, z = orc.oracle_quantize_rtn(W, bits)
    deq = orc.oracle_dequantize(W, bits)
    s = s16.astype(np.float64)[:, np.arange(500) // 128]
    err = np.abs(deq - W.astype(np.float64))
    assert np.all(err <= s * (0.5 + maxq * 2.0**-11))
    assert np.all(deq[W == 0] == 0)
    inner = (q > 0) & (q < maxq)
    assert np.all(err[inner] <= s[inner] * 0.5)


def test_pruned_stay_pruned_and_sign_of_zero():
    W = np.array([[0.0, -0.0, 0.5, -0.25]], dtype=np.float16)
    for bits in (8, 4):
        deq = orc.oracle_dequantize(W, bits)
        assert deq[0, 0] == 0 and deq[0, 1] == 0
        hdr, off, data, table = orc.ref_pack_cmb_q(W, bits)
        nz, q, s16, z = orc.ref_unpack_cmb_q(hdr, off, data, table)
        assert nz[0].tolist() == [False, False, True, True]


# ------------------------------------------------------------------ exact y ----

@pytest.mark.parametrize("bits", [8, 4])
def test_spmspv_q_matches_exact_integer_arithmetic(bits):
    rng = np.random.default_rng(30 + bits)
    O, I, k = 40, 300, 170
    W = (rng.standard_normal((O, I)) * 0.02).astype(np.float16)
    W[rng.random((O, I)) < 0.5] = 0
    x = rng.laplace(0, 1, size=I).astype(np.float16)
    y = orc.oracle_spmspv_q(W, x, k, bits)
    K, _ = orc.oracle_sparsify(x, k)
    q, s16, z = orc.oracle_quantize_rtn(W, bits)
    nz = W != 0
    ex = orc.exact_spmspv_q_rows_scaled(q, s16, z, nz, x, K)
    Wd = orc.oracle_dequantize(W, bits)
    mag = np.abs(Wd[:, K.astype(np.int64)]) @ np.abs(x[K.astype(np.int64)].astype(np.float64))
    for i in range(O):
        exact = Fraction(ex[i], 2**48)
        assert abs(Fraction(float(y[i])) - exact) <= Fraction(k * 2.0**-52) * Fraction(float(mag[i])) + Fraction(1, 2**1074)


def test_spmspv_q_reduces_to_fp16_path_on_grid_weights():
    """A weight already on its grid dequantises to itself, so the quantised
    product equals the fp16 product (§3's sum) exactly."""
    rng = np.random.default_rng(5)
    O, I = 16, 256
    codes = rng.integers(0, 16, size=(O, I))
    codes[:, 0], codes[:, 128] = 0, 0
    codes[:, 1], codes[:, 129] = 15, 15
    codes[codes == 7] = 8
    W = (0.0625 * (codes - 7)).astype(np.float16)
    x = rng.laplace(0, 1, size=I).astype(np.float16)
    for k in (0, 1, 100, I):
        assert np.array_equal(orc.oracle_spmspv_q(W, x, k, 4), orc.oracle_spmspv(W, x, k))
    tau = 0.7
    assert np.array_equal(orc.oracle_spmspv_q_threshold(W, x, tau, 4),
                          orc.oracle_spmspv_threshold(W, x, tau))


# ------------------------------------------------------------------ packer ----

@pytest.mark.parametrize("bits", [8, 4])
@pytest.mark.parametrize("O,I", [(1, 1), (5, 130), (1024, 3), (1025, 129), (2100, 40)])
def test_pack_q_round_trip(bits, O, I):
    rng = np.random.default_rng(O * 7 + I + bits)
    W = (rng.standard_normal((O, I)) * 0.02).astype(np.float16)
    W[rng.random((O, I)) < 0.6] = 0
    hdr, off, data, table = orc.ref_pack_cmb_q(W, bits)
    nz, q, s16, z = orc.ref_unpack_cmb_q(hdr, off, data, table)
    q0, s0, z0 = orc.oracle_quantize_rtn(W, bits)
    assert np.array_equal(nz, W != 0)
    assert np.array_equal(q, q0)
    assert np.array_equal(s16.view(np.uint16), s0.view(np.uint16))
    assert np.array_equal(z, z0)
    S = hdr["nseg"]
    assert hdr["nnz"] == int((W != 0).sum())
    for j in range(I):
        for s in range(S):
            b0, b1 = int(off[j * S + s]) * 16, int(off[j * S + s + 1]) * 16
            n = int(np.unpackbits(data[b0:b0 + 128]).sum())
            code_bytes = n if bits == 8 else (n + 1) // 2
            assert b1 - b0 == (128 + code_bytes + 15) // 16 * 16
            assert np.all(data[b0 + 128 + code_bytes:b1] == 0)


def test_pack_q_hand_bytes():
    """One column, rows 0, 1, 2 and 33 stored, 4-bit codes: the mask words,
    the nibble order of the record, and where each row's grid sits.  Each row
    has its own grid (one weight per group here):
      row 0,  0.25: s = fp16(0.25/15) = 1.0667 * 2^-6 -> 0x2400 + 68 = 0x2444,
                    z = 0, code rint(15.004) = 15;
      row 1, -0.5 : s = fp16(0.5/15) -> 0x2844, z = rint(15.004) = 15, code 0;
      row 2,  1.0 : s = 0x2C44, z = 0, code 15;
      row 33, 0.125: s = fp16(0.125/15) -> 0x2044, z = 0, code 15."""
    W = np.zeros((40, 1), dtype=np.float16)
    W[[0, 1, 2, 33], 0] = [0.25, -0.5, 1.0, 0.125]
    hdr, off, data, table = orc.ref_pack_cmb_q(W, 4)
    rec = data[:int(off[1]) * 16]
    assert len(rec) == 144
    assert rec[:4].tolist() == [0b111, 0, 0, 0]      # word 0: rows 0, 1, 2
    assert rec[4:8].tolist() == [0b10, 0, 0, 0]      # word 1: row 33
    assert rec[128:130].tolist() == [0x0F, 0xFF]     # codes 15, 0 | 15, 15, low nibble first
    # row 32 l + t sits at index 32 t + l
    assert table[0 * 32 + 0] == 0x2444
    assert table[1 * 32 + 0] == 0x2844 | (15 << 16)
    assert table[2 * 32 + 0] == 0x2C44
    assert table[1 * 32 + 1] == 0x2044
    assert table[3 * 32 + 0] == 0x3C00               # row 3: no weight, s = 1
    assert table[0 * 32 + 2] == 0                    # row 64 >= O


def test_required_bytes_q_closed_form():
    nnz = np.array([3, 0, 5, 2, 7] + [1] * 200)
    K = np.array([0, 2, 130])
    O, I = 10, 205
    for bits in (8, 4):
        got = orc.required_bytes_q(nnz, K, O, I, bits)
        want = bits / 8 * (3 + 5 + 1) + 3 * 10 / 8 + (2 + bits / 8) * 10 * 2 + 2 * I + 12 + 40
        assert math.isclose(got, want, rel_tol=0, abs_tol=1e-9)
