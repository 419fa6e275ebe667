"""Plain, slow, obviously-correct CPU oracle (numpy, fp64).

TEST INFRASTRUCTURE ONLY -- see the package docstring.  Nothing here is tuned.

Notation follows the paper (DuoGPT, arXiv 2506.20194, §3 "Preliminaries"):
the layer weight is W in R^{n x k} with n output rows and k input channels
(here O = n rows, I = k channels, to keep the letter k for the number of kept
channels), the input is a column vector x, and activation sparsity multiplies
x by a binary mask m^x chosen by magnitude at decode time (§3, "Activation
Sparsity").  The decode-time product is

    y = W (x ⊙ m^x) = sum_{i : m^x_i = 1} W[:, i] * x_i          (§3)

and only the weight columns of the surviving channels are fetched (§4.1).
Weight sparsity is unstructured: a pruned weight is stored as zero (§3, mask
m^w), and each kept column is stored compressed (§4.1).

Readings taken where the paper is silent:
  * the number of kept channels is k = floor(I * (100 - pct) / 100) for an
    integer activation-sparsity percentage pct;
  * the kept set is the k channels of largest |x_j|; ties between equal
    magnitudes go to the LOWER channel index; -0 and +0 have magnitude 0;
    when fewer than k entries are non-zero, zero channels fill the set in
    index order (they contribute nothing);
  * the oracle requires x to be NaN-free (the CUDA path orders NaN above Inf
    by bit pattern; the paper does not define either);
  * a weight entry is pruned iff it compares equal to zero (+0 or -0);
  * the threshold mask (§5's threshold-based activation sparsity) keeps
    |x_j| > |tau| strictly, as the thresholding function it cites zeroes
    entries at or below the threshold;
  * y is accumulated and returned in fp64 here (fp32 on the GPU).
"""
from __future__ import annotations

import math

import numpy as np

# Rows per segment of the channel-major bitmask ("CMB") format.  The paper
# does not fix a storage format (§4.1 only says each column is stored
# compressed); this layout is the one defined for this library and the
# reference packer below is normative for it.
SEG_ROWS = 1024
CMB_MAGIC = 0x31424D43      # b"CMB1" little-endian
IDX16_MAGIC = 0x30584449    # b"IDX0" little-endian
CMB_VERSION = 1
IDX16_VERSION = 0


def _as_f16(a) -> np.ndarray:
    a = np.asarray(a)
    if a.dtype == np.uint16:
        return a.view(np.float16)
    if a.dtype != np.float16:
        raise TypeError(f"expected float16 (or uint16 bit patterns), got {a.dtype}")
    return a


def k_from_pct(I: int, pct: int) -> int:
    """Number of kept channels for an activation sparsity of ``pct`` percent.

    §3 defines p^x as the proportion of zeros in m^x; with an integer
    percentage the kept count is floor(I * (100 - pct) / 100).
    """
    if not (0 <= pct <= 100):
        raise ValueError("pct must be in [0, 100]")
    return (I * (100 - pct)) // 100


def oracle_sparsify(x16, k: int):
    """Magnitude top-k activation mask (§3, "Activation Sparsity").

    Returns ``(kept_idx, kept_val)``: the k channel ids with the largest
    |x_j| (ties to the lower index), in ASCENDING id order as uint16, and the
    unchanged fp16 values x[kept_idx].
    """
    x = _as_f16(x16).reshape(-1)
    I = x.shape[0]
    if not (0 <= k <= I):
        raise ValueError(f"k={k} outside [0, {I}]")
    if I > 65535:
        raise ValueError("channel ids are uint16: I must be <= 65535")
    a = np.abs(x.astype(np.float64))
    if np.isnan(a).any():
        raise ValueError("the oracle defines the kept set for NaN-free x only")
    j = np.arange(I)
    order = np.lexsort((j, -a))          # by |x| descending, then j ascending
    K = np.sort(order[:k])
    return K.astype(np.uint16), x[K].copy()


def oracle_sparsify_threshold(x16, tau):
    """Threshold activation mask (§5, compatibility with threshold-based
    activation sparsity, Table 3(b)): instead of the k largest magnitudes,
    the mask keeps every channel whose magnitude exceeds a threshold fixed
    beforehand for the layer.  Entries with |x_j| <= |tau| are dropped, so the
    comparison is strict; the sign of ``tau`` is ignored.

    Returns ``(kept_idx, kept_val)``: the kept channel ids in ASCENDING order
    as uint16 and the unchanged fp16 values x[kept_idx].  The number kept
    depends on x.
    """
    x = _as_f16(x16).reshape(-1)
    I = x.shape[0]
    if I > 65535:
        raise ValueError("channel ids are uint16: I must be <= 65535")
    a = np.abs(x.astype(np.float64))
    t = abs(float(np.float16(tau)))
    if np.isnan(a).any() or math.isnan(t):
        raise ValueError("the oracle defines the kept set for NaN-free x and tau only")
    K = np.nonzero(a > t)[0]
    return K.astype(np.uint16), x[K].copy()


def oracle_spmspv_threshold(W16, x16, tau) -> np.ndarray:
    """y = W (x ⊙ m^x) in fp64 (§3) with the threshold mask of
    :func:`oracle_sparsify_threshold`."""
    W = _as_f16(W16)
    if W.ndim != 2 or W.shape[1] != _as_f16(x16).size:
        raise ValueError("W must be O x I with I = len(x)")
    K, xv = oracle_sparsify_threshold(x16, tau)
    return W[:, K.astype(np.int64)].astype(np.float64) @ xv.astype(np.float64)


def oracle_spmspv(W16, x16, k: int) -> np.ndarray:
    """y = W (x ⊙ m^x) in fp64 over the dense masked weight (§3).

    ``W16`` is the O x I fp16 weight with pruned entries stored as zero.
    The product over kept columns is a plain matrix-vector product in fp64;
    pruned (zero) entries contribute exactly zero, so this equals the sum
    over stored non-zeros of kept columns.
    """
    W = _as_f16(W16)
    if W.ndim != 2:
        raise ValueError("W must be 2-D (O x I)")
    K, xv = oracle_sparsify(x16, k)
    if W.shape[1] != _as_f16(x16).size:
        raise ValueError("W and x disagree on I")
    Kl = K.astype(np.int64)
    return W[:, Kl].astype(np.float64) @ xv.astype(np.float64)


def oracle_spmspv_rows(W_rows16, x16, k: int) -> np.ndarray:
    """Same as :func:`oracle_spmspv` for a subset of rows of W (sampled
    parity at full size): ``W_rows16`` holds those rows (r x I)."""
    return oracle_spmspv(W_rows16, x16, k)


def exact_spmspv_rows_scaled(W_rows16, x16, K) -> list[int]:
    """Exact y_i * 2**48 as Python integers for the given kept set K.

    Every finite fp16 value is an integer multiple of 2**-24, so
    y_i * 2**48 = sum_j (W_ij * 2**24) * (x_j * 2**24) holds exactly in
    integer arithmetic (§3's sum, no rounding anywhere).
    """
    W = _as_f16(W_rows16)
    x = _as_f16(x16).reshape(-1)
    Kl = np.asarray(K, dtype=np.int64)
    Wi = (W[:, Kl].astype(np.float64) * 2.0**24).astype(np.int64)
    xi = (x[Kl].astype(np.float64) * 2.0**24).astype(np.int64)
    xs = [int(v) for v in xi]
    out = []
    for r in range(Wi.shape[0]):
        row = Wi[r]
        nz = np.nonzero(row)[0]
        out.append(sum(int(row[c]) * xs[c] for c in nz))
    return out


def fsum_spmspv_rows(W_rows16, x16, K) -> np.ndarray:
    """Correctly rounded fp64 y_i via math.fsum of the (exact) fp64
    products W_ij * x_j over the kept set K (fp16 x fp16 fits fp64 exactly)."""
    W = _as_f16(W_rows16)
    x = _as_f16(x16).reshape(-1)
    Kl = np.asarray(K, dtype=np.int64)
    P = W[:, Kl].astype(np.float64) * x[Kl].astype(np.float64)[None, :]
    return np.array([math.fsum(P[r]) for r in range(P.shape[0])], dtype=np.float64)


def tolerance_rows(W_rows16, x16, K, rel: float = 2e-3) -> np.ndarray:
    """Per-row acceptance bound rel * sum_{j in K} |W_ij| |x_j| for an fp16-in,
    fp32-accumulate result (a row whose bound is 0 must come out exactly 0)."""
    W = _as_f16(W_rows16)
    x = _as_f16(x16).reshape(-1)
    Kl = np.asarray(K, dtype=np.int64)
    return rel * (np.abs(W[:, Kl].astype(np.float64)) @ np.abs(x[Kl].astype(np.float64)))


# --------------------------------------------------------------------------
# Reference packers (the storage step of §4.1: "each weight row is stored in
# compressed format", with the paper's column-major convention of §3's
# footnote, i.e. one compressed run per input channel).
# --------------------------------------------------------------------------

def _pad16(n: int) -> int:
    return (n + 15) // 16 * 16


def ref_pack_cmb(W16):
    """Channel-major bitmask ("CMB") packing, normative reference.

    Layout: rows are cut into S = ceil(O / 1024) segments.  For each input
    channel j (outer) and segment s (inner) there is one record at byte
    offset 16 * off[j*S + s]:
        32 little-endian uint32 mask words; bit b of word w is set iff
        W[s*1024 + 32*w + b, j] != 0 (rows >= O give 0 bits);
        the fp16 bit patterns of those non-zero entries in increasing row
        order;
        zero bytes up to the next multiple of 16.
    off[I*S] is the total size in 16-byte units.

    Returns ``(header, off, data)`` with off uint32[I*S+1] and data uint8.
    """
    W = _as_f16(W16)
    O, I = W.shape
    S = (O + SEG_ROWS - 1) // SEG_ROWS
    bits = W.view(np.uint16)
    nzmask = (bits & 0x7FFF) != 0
    off = np.zeros(I * S + 1, dtype=np.uint32)
    pieces = []
    pos = 0
    nnz = 0
    for j in range(I):
        col_nz = nzmask[:, j]
        col_bits = bits[:, j]
        for s in range(S):
            r0, r1 = s * SEG_ROWS, min(O, (s + 1) * SEG_ROWS)
            m = np.zeros(SEG_ROWS, dtype=bool)
            m[: r1 - r0] = col_nz[r0:r1]
            mask_bytes = np.packbits(m, bitorder="little").tobytes()   # 128 bytes
            vals = col_bits[r0:r1][col_nz[r0:r1]].astype("<u2").tobytes()
            nnz += len(vals) // 2
            rec = mask_bytes + vals
            rec = rec + b"\x00" * (_pad16(len(rec)) - len(rec))
            off[j * S + s] = pos // 16
            pos += len(rec)
            pieces.append(rec)
    off[I * S] = pos // 16
    if pos // 16 >= 2**32:
        raise ValueError("packed size exceeds the uint32 offset range")
    data = np.frombuffer(b"".join(pieces), dtype=np.uint8).copy()
    header = dict(magic=CMB_MAGIC, version=CMB_VERSION, out=O, inp=I,
                  seg_rows=SEG_ROWS, nseg=S, nnz=nnz)
    return header, off, data


def ref_unpack_cmb(header, off, data) -> np.ndarray:
    """Inverse of :func:`ref_pack_cmb` (returns the O x I fp16 weight)."""
    O, I, S = header["out"], header["inp"], header["nseg"]
    out = np.zeros((O, I), dtype=np.uint16)
    data = np.asarray(data, dtype=np.uint8)
    for j in range(I):
        for s in range(S):
            b0 = int(off[j * S + s]) * 16
            words = np.frombuffer(data[b0:b0 + 128].tobytes(), dtype="<u4")
            m = np.unpackbits(words.view(np.uint8), bitorder="little").astype(bool)
            n = int(m.sum())
            vals = np.frombuffer(data[b0 + 128:b0 + 128 + 2 * n].tobytes(), dtype="<u2")
            rows = np.nonzero(m)[0] + s * SEG_ROWS
            if rows.size and rows[-1] >= O:
                raise ValueError("mask bit set beyond the last row")
            out[rows, j] = vals
    return out.view(np.float16)


def ref_pack_idx16(W16):
    """Index format ("IDX16", parity format): per input channel j a block at
    byte offset colptr[j]: the fp16 non-zeros in increasing row order, zero
    padded to 16 bytes, then their uint16 row ids, zero padded to 16 bytes.
    cnt[j] is the number of non-zeros; colptr[I] is the total size.
    Requires O <= 65536 (row ids fit uint16)."""
    W = _as_f16(W16)
    O, I = W.shape
    if O > 65536:
        raise ValueError("IDX16 needs O <= 65536")
    bits = W.view(np.uint16)
    nzmask = (bits & 0x7FFF) != 0
    colptr = np.zeros(I + 1, dtype=np.uint64)
    cnt = np.zeros(I, dtype=np.uint32)
    pieces = []
    pos = 0
    for j in range(I):
        rows = np.nonzero(nzmask[:, j])[0]
        v = bits[rows, j].astype("<u2").tobytes()
        r = rows.astype("<u2").tobytes()
        blk = v + b"\x00" * (_pad16(len(v)) - len(v)) + r + b"\x00" * (_pad16(len(r)) - len(r))
        colptr[j] = pos
        cnt[j] = rows.size
        pos += len(blk)
        pieces.append(blk)
    colptr[I] = pos
    data = np.frombuffer(b"".join(pieces), dtype=np.uint8).copy()
    header = dict(magic=IDX16_MAGIC, version=IDX16_VERSION, out=O, inp=I,
                  seg_rows=0, nseg=0, nnz=int(cnt.sum()))
    return header, colptr, cnt, data


def ref_unpack_idx16(header, colptr, cnt, data) -> np.ndarray:
    O, I = header["out"], header["inp"]
    out = np.zeros((O, I), dtype=np.uint16)
    data = np.asarray(data, dtype=np.uint8)
    for j in range(I):
        b0, n = int(colptr[j]), int(cnt[j])
        vals = np.frombuffer(data[b0:b0 + 2 * n].tobytes(), dtype="<u2")
        r0 = b0 + _pad16(2 * n)
        rows = np.frombuffer(data[r0:r0 + 2 * n].tobytes(), dtype="<u2").astype(np.int64)
        out[rows, j] = vals
    return out.view(np.float16)


# --------------------------------------------------------------------------
# Byte and load accounting (§4.1, §5 "weights loaded to SRAM", App. B.3).
# --------------------------------------------------------------------------

def required_bytes(nnz_per_channel, K, O: int, I: int) -> float:
    """Format-neutral bytes one call must move: for every kept channel its
    fp16 non-zeros plus one mask bit per (kept channel, row) position, plus
    x (2I), the kept ids and values (4k) and the fp32 output (4O)."""
    n = np.asarray(nnz_per_channel, dtype=np.float64)
    Kl = np.asarray(K, dtype=np.int64)
    k = Kl.size
    return float(2.0 * n[Kl].sum() + k * O / 8.0 + 2.0 * I + 4.0 * k + 4.0 * O)


def loaded_fraction(nnz_per_channel, K, O: int, I: int) -> float:
    """Fraction of the dense weight count fetched for kept set K (§5: about
    (1 - p^w)(1 - p^x) for a dual-sparse layer)."""
    n = np.asarray(nnz_per_channel, dtype=np.float64)
    return float(n[np.asarray(K, dtype=np.int64)].sum() / (O * I))


def worst_case_loaded_fraction(nnz_per_channel, k: int, O: int, I: int) -> float:
    """Upper bound of App. B.3: the k densest channels are the ones kept."""
    n = np.sort(np.asarray(nnz_per_channel, dtype=np.float64))[::-1]
    return float(n[:k].sum() / (O * I))


# --------------------------------------------------------------------------
# Weight-only quantisation of the stored values (§5, compatibility with
# weight-only quantisation, Table 4): b-bit uniform integers (b = 8 or 4),
# round-to-nearest ("RTN", no error feedback), one grid per output row and
# group of 128 consecutive input channels.
#
# Readings (the paper names only "uniform integer", "channel-wise RTN" and the
# group size; it follows the GPTQ / OBC line of work, whose quantiser is the
# asymmetric min-max grid):
#   * per (row i, group g): lo = min(0, min W), hi = max(0, max W) over the
#     group's entries; scale s = (hi - lo) / (2**b - 1), computed in fp64 and
#     rounded to the nearest fp16 (ties to even); s = 1 for a group with no
#     non-zero entry, s = 2**-24 if a non-zero quotient rounds to 0;
#   * zero point z = rint(-lo / s) (ties to even), clamped to [0, 2**b - 1];
#   * code q = clamp(rint(w / s) + z, 0, 2**b - 1) for every stored (non-zero)
#     entry, the quotients in fp64; pruned entries stay pruned (no code, mask
#     bit 0), and a code equal to z keeps its mask bit although it stands for 0;
#   * the dequantised weight is s * (q - z) (exact in fp64); y sums it against
#     x over the kept channels in fp64.
# --------------------------------------------------------------------------

QUANT_GROUP = 128
QUANT_BITS = (8, 4)


def _check_bits(bits):
    if bits not in QUANT_BITS:
        raise ValueError(f"bits must be one of {QUANT_BITS}")
    return (1 << bits) - 1


def oracle_quantize_rtn(W16, bits: int):
    """RTN quantisation of the non-zero entries of W (readings above).

    Returns ``(q, s16, z)``: q int64 O x I (the code of every non-zero entry,
    0 where pruned), s16 float16 O x G and z int64 O x G with
    G = ceil(I / 128); group g holds channels 128 g .. 128 g + 127.
    """
    W = _as_f16(W16)
    if W.ndim != 2:
        raise ValueError("W must be O x I")
    maxq = _check_bits(bits)
    O, I = W.shape
    G = (I + QUANT_GROUP - 1) // QUANT_GROUP
    nz = (W.view(np.uint16) & 0x7FFF) != 0
    Wd = np.where(nz, W.astype(np.float64), 0.0)
    q = np.zeros((O, I), dtype=np.int64)
    s16 = np.zeros((O, G), dtype=np.float16)
    z = np.zeros((O, G), dtype=np.int64)
    for g in range(G):
        c0, c1 = g * QUANT_GROUP, min(I, (g + 1) * QUANT_GROUP)
        blk = Wd[:, c0:c1]
        lo = np.minimum(blk.min(axis=1), 0.0)
        hi = np.maximum(blk.max(axis=1), 0.0)
        sg = ((hi - lo) / maxq).astype(np.float16)
        empty = hi == lo
        sg[empty] = np.float16(1.0)
        sg[(sg == 0) & ~empty] = np.uint16(1).view(np.float16)   # 2**-24
        sd = sg.astype(np.float64)
        zg = np.clip(np.rint(-lo / sd), 0, maxq).astype(np.int64)
        qg = np.clip(np.rint(blk / sd[:, None]) + zg[:, None], 0, maxq).astype(np.int64)
        q[:, c0:c1] = np.where(nz[:, c0:c1], qg, 0)
        s16[:, g] = sg
        z[:, g] = zg
    return q, s16, z


def oracle_dequantize(W16, bits: int) -> np.ndarray:
    """The weight the quantised store stands for: s * (q - z) at every
    non-zero entry of W, 0 at pruned ones (fp64, exact)."""
    W = _as_f16(W16)
    q, s16, z = oracle_quantize_rtn(W, bits)
    g = np.arange(W.shape[1]) // QUANT_GROUP
    nz = (W.view(np.uint16) & 0x7FFF) != 0
    deq = s16.astype(np.float64)[:, g] * (q - z[:, g]).astype(np.float64)
    return np.where(nz, deq, 0.0)


def oracle_spmspv_q(W16, x16, k: int, bits: int) -> np.ndarray:
    """y = W_q (x ⊙ m^x) in fp64 with the top-k mask (§3) and the RTN-quantised
    weight of :func:`oracle_dequantize` (§5, Table 4)."""
    Wq = oracle_dequantize(W16, bits)
    K, xv = oracle_sparsify(x16, k)
    if Wq.shape[1] != _as_f16(x16).size:
        raise ValueError("W and x disagree on I")
    return Wq[:, K.astype(np.int64)] @ xv.astype(np.float64)


def oracle_spmspv_q_threshold(W16, x16, tau, bits: int) -> np.ndarray:
    """As :func:`oracle_spmspv_q` with the threshold mask of
    :func:`oracle_sparsify_threshold`."""
    Wq = oracle_dequantize(W16, bits)
    K, xv = oracle_sparsify_threshold(x16, tau)
    if Wq.shape[1] != _as_f16(x16).size:
        raise ValueError("W and x disagree on I")
    return Wq[:, K.astype(np.int64)] @ xv.astype(np.float64)


def exact_spmspv_q_rows_scaled(q_rows, s16_rows, z_rows, nz_rows, x16, K) -> list[int]:
    """Exact y_i * 2**48 as Python integers from the codes themselves: every
    fp16 scale is an integer multiple of 2**-24, so
    y_i * 2**48 = sum_j (s_ig * 2**24) * (q_ij - z_ig) * (x_j * 2**24)."""
    x = _as_f16(x16).reshape(-1)
    s_int = (np.asarray(s16_rows, dtype=np.float16).astype(np.float64) * 2.0**24).astype(np.int64)
    out = []
    for r in range(len(q_rows)):
        acc = 0
        for j in (int(c) for c in K):
            if not nz_rows[r][j]:
                continue
            g = j // QUANT_GROUP
            xi = int(float(x[j]) * 2.0**24)
            acc += int(s_int[r][g]) * (int(q_rows[r][j]) - int(z_rows[r][g])) * xi
        out.append(acc)
    return out


def tolerance_rows_f64(Wd_rows, x16, K, rel: float = 2e-3) -> np.ndarray:
    """rel * sum_{j in K} |W_ij| |x_j| for an fp64 weight (the dequantised one)."""
    x = _as_f16(x16).reshape(-1)
    Kl = np.asarray(K, dtype=np.int64)
    return rel * (np.abs(np.asarray(Wd_rows, dtype=np.float64)[:, Kl]) @ np.abs(x[Kl].astype(np.float64)))


def ref_pack_cmb_q(W16, bits: int):
    """Bitmask packing with b-bit codes in place of the fp16 values.

    Records are laid out as in :func:`ref_pack_cmb` (32 mask words, then the
    stored entries in increasing row order, zero padding to 16 bytes), but an
    entry is its code: one byte each for b = 8; for b = 4 two per byte, the
    n-th entry of the record in byte n // 2, low nibble first when n is even.

    The grids sit in a separate table of uint32 entries, s's fp16 bits in the
    low half and z in the high half.  The entry of row i = 1024 s + 32 l + t
    (segment s, lane l, bit t) and group g is at index
    ((s * G + g) * 32 + t) * 32 + l; rows >= O hold 0.

    Returns ``(header, off, data, table)``.
    """
    W = _as_f16(W16)
    maxq = _check_bits(bits)
    O, I = W.shape
    S = (O + SEG_ROWS - 1) // SEG_ROWS
    G = (I + QUANT_GROUP - 1) // QUANT_GROUP
    q, s16, z = oracle_quantize_rtn(W, bits)
    nzmask = (W.view(np.uint16) & 0x7FFF) != 0
    off = np.zeros(I * S + 1, dtype=np.uint32)
    pieces = []
    pos = 0
    nnz = 0
    for j in range(I):
        for s in range(S):
            r0, r1 = s * SEG_ROWS, min(O, (s + 1) * SEG_ROWS)
            m = np.zeros(SEG_ROWS, dtype=bool)
            m[: r1 - r0] = nzmask[r0:r1, j]
            codes = q[r0:r1, j][nzmask[r0:r1, j]]
            assert codes.size == 0 or (codes.min() >= 0 and codes.max() <= maxq)
            nnz += codes.size
            if bits == 8:
                cb = codes.astype(np.uint8).tobytes()
            else:
                nb = bytearray((codes.size + 1) // 2)
                for n, c in enumerate(codes):
                    nb[n // 2] |= int(c) << (4 * (n % 2))
                cb = bytes(nb)
            rec = np.packbits(m, bitorder="little").tobytes() + cb
            rec = rec + b"\x00" * (_pad16(len(rec)) - len(rec))
            off[j * S + s] = pos // 16
            pos += len(rec)
            pieces.append(rec)
    off[I * S] = pos // 16
    if pos // 16 >= 2**32:
        raise ValueError("packed size exceeds the uint32 offset range")
    data = np.frombuffer(b"".join(pieces), dtype=np.uint8).copy()
    table = np.zeros(S * G * SEG_ROWS, dtype=np.uint32)
    for s in range(S):
        for g in range(G):
            for t in range(32):
                for l in range(32):
                    i = s * SEG_ROWS + 32 * l + t
                    if i < O:
                        table[((s * G + g) * 32 + t) * 32 + l] = (
                            int(s16[i, g].view(np.uint16)) | (int(z[i, g]) << 16))
    header = dict(magic=CMB_MAGIC, version=CMB_VERSION, out=O, inp=I,
                  seg_rows=SEG_ROWS, nseg=S, nnz=nnz, bits=bits, group=QUANT_GROUP)
    return header, off, data, table


def ref_unpack_cmb_q(header, off, data, table):
    """Inverse of :func:`ref_pack_cmb_q`: returns ``(nz, q, s16, z)`` (the
    non-zero mask O x I, the codes O x I with 0 where pruned, the grids)."""
    O, I, S, bits = header["out"], header["inp"], header["nseg"], header["bits"]
    G = (I + QUANT_GROUP - 1) // QUANT_GROUP
    data = np.asarray(data, dtype=np.uint8)
    nz = np.zeros((O, I), dtype=bool)
    q = np.zeros((O, I), dtype=np.int64)
    for j in range(I):
        for s in range(S):
            b0 = int(off[j * S + s]) * 16
            words = np.frombuffer(data[b0:b0 + 128].tobytes(), dtype="<u4")
            m = np.unpackbits(words.view(np.uint8), bitorder="little").astype(bool)
            rows = np.nonzero(m)[0] + s * SEG_ROWS
            if rows.size and rows[-1] >= O:
                raise ValueError("mask bit set beyond the last row")
            n = rows.size
            cb = data[b0 + 128:b0 + 128 + (n if bits == 8 else (n + 1) // 2)]
            if bits == 8:
                codes = cb.astype(np.int64)
            else:
                codes = np.array([(int(cb[e // 2]) >> (4 * (e % 2))) & 15 for e in range(n)],
                                 dtype=np.int64)
            nz[rows, j] = True
            q[rows, j] = codes
    tab = np.asarray(table, dtype=np.uint32).reshape(S, G, 32, 32)   # [s][g][t][l]
    rows_tab = tab.transpose(0, 3, 2, 1).reshape(S * SEG_ROWS, G)[:O]   # row 1024 s + 32 l + t
    s16 = (rows_tab & 0xFFFF).astype(np.uint16).view(np.float16)
    z = (rows_tab >> 16).astype(np.int64)
    return nz, q, s16, z


def required_bytes_q(nnz_per_channel, K, O: int, I: int, bits: int) -> float:
    """Format-neutral bytes of a quantised call: b/8 bytes per stored entry of
    the kept channels, one mask bit per (kept channel, row) position, an fp16
    scale and a b-bit zero point per (row, group holding a kept channel), plus
    x (2I), the kept ids and values (4k) and the fp32 output (4O)."""
    _check_bits(bits)
    n = np.asarray(nnz_per_channel, dtype=np.float64)
    Kl = np.asarray(K, dtype=np.int64)
    k = Kl.size
    groups = np.unique(Kl // QUANT_GROUP).size
    return float(bits / 8.0 * n[Kl].sum() + k * O / 8.0 + (2.0 + bits / 8.0) * O * groups
                 + 2.0 * I + 4.0 * k + 4.0 * O)
