"""Planted mistakes in the oracle, on the CPU: each test patches one
plausible error into the oracle for its own duration and checks that the
pins guarding that part fail. The errors covered: a reversed tie rule,
ranking by signed value instead of magnitude, a dropped term, a wrong sign,
a transposed operand, an ignored kept set, a non-strict threshold, mask
bits in the wrong order, a zero point off by one, a scale rounded through
fp32, codes rounded half up, a sign flip or a dropped term in the efficient
score, a transposed factor, no dampening, act_order ignored, and the sweep
without its activation-sparsity term. Nothing here touches a GPU."""
import numpy as np
import pytest

import oracle as orc
from oracle import calib_oracle as cal_o
from oracle import duo_oracle as duo_o

import test_oracle_calib as calib_pins
import test_oracle_pins as pins
import test_oracle_quant as quant_pins


def _fails(pin, *args):
    with pytest.raises((AssertionError, ValueError, IndexError)):
        pin(*args)


# ------------------------------------------------------------ sparsifier ----

def test_reversed_tie_rule_is_caught(monkeypatch):
    orig = duo_o.oracle_sparsify

    def mutant(x16, k):   # ties go to the HIGHER index
        x = np.asarray(x16, dtype=np.float16).reshape(-1)
        K, _ = orig(x[::-1].copy(), k)
        K = np.sort(x.size - 1 - K.astype(np.int64))
        return K.astype(np.uint16), x[K].copy()

    monkeypatch.setattr(orc, "oracle_sparsify", mutant)
    _fails(pins.test_sparsify_matches_bruteforce, 8)
    _fails(pins.test_sparsify_all_equal_keeps_lowest_indices)


def test_signed_order_is_caught(monkeypatch):
    def mutant(x16, k):   # largest x_j instead of largest |x_j|
        x = np.asarray(x16, dtype=np.float16).reshape(-1)
        order = np.lexsort((np.arange(x.size), -x.astype(np.float64)))
        K = np.sort(order[:k])
        return K.astype(np.uint16), x[K].copy()

    monkeypatch.setattr(orc, "oracle_sparsify", mutant)
    _fails(pins.test_sparsify_matches_bruteforce, 8)


def test_non_strict_threshold_is_caught(monkeypatch):
    def mutant(x16, tau):   # keeps |x_j| >= |tau| instead of > |tau|
        x = np.asarray(x16, dtype=np.float16).reshape(-1)
        K = np.nonzero(np.abs(x.astype(np.float64)) >= abs(float(np.float16(tau))))[0]
        return K.astype(np.uint16), x[K].copy()

    monkeypatch.setattr(orc, "oracle_sparsify_threshold", mutant)
    _fails(pins.test_golden_threshold_cases)


# ---------------------------------------------------------------- spMspV ----

def test_dropped_term_is_caught(monkeypatch):
    orig = duo_o.oracle_spmspv

    def mutant(W16, x16, k):   # forgets the last kept channel
        y = orig(W16, x16, k)
        if k == 0:
            return y
        K, xv = duo_o.oracle_sparsify(x16, k)
        j = int(K[-1])
        return y - np.asarray(W16, np.float16)[:, j].astype(np.float64) * float(xv[-1])

    monkeypatch.setattr(orc, "oracle_spmspv", mutant)
    _fails(pins.test_spmspv_exact_integer, 7, 9, 0.5, 4)
    _fails(pins.test_spmspv_pure_python_bruteforce)


def test_wrong_sign_is_caught(monkeypatch):
    orig = duo_o.oracle_spmspv
    monkeypatch.setattr(orc, "oracle_spmspv", lambda W, x, k: -orig(W, x, k))
    _fails(pins.test_spmspv_pure_python_bruteforce)
    _fails(pins.test_spmspv_exact_integer, 33, 65, 0.3, 40)


def test_transposed_operand_is_caught(monkeypatch):
    orig = duo_o.oracle_spmspv

    def mutant(W16, x16, k):   # rows of W for channels (square shapes only)
        W = np.asarray(W16, np.float16)
        return orig(np.ascontiguousarray(W.T), x16, k) if W.shape[0] == W.shape[1] else orig(W, x16, k)

    monkeypatch.setattr(orc, "oracle_spmspv", mutant)
    _fails(pins.test_transposed_operand_is_caught)


def test_ignored_kept_set_is_caught(monkeypatch):
    orig = duo_o.oracle_spmspv
    monkeypatch.setattr(orc, "oracle_spmspv", lambda W, x, k: orig(W, x, np.asarray(x).size))
    _fails(pins.test_spmspv_exact_integer, 7, 9, 0.5, 4)
    _fails(pins.test_k_zero_gives_zero_and_row_bound_zero)


# ---------------------------------------------------------------- packer ----

def test_reversed_mask_bit_order_is_caught(monkeypatch):
    orig = duo_o.ref_pack_cmb

    def mutant(W16):   # bit b of a mask word for row 32 w + 31 - b
        header, off, data = orig(W16)
        data = data.copy()
        for u in np.asarray(off[:-1], dtype=np.int64):
            b0 = int(u) * 16
            words = data[b0:b0 + 128].view("<u4")
            rev = np.array([int(f"{int(v):032b}"[::-1], 2) for v in words], dtype="<u4")
            data[b0:b0 + 128] = rev.view(np.uint8)
        return header, off, data

    monkeypatch.setattr(orc, "ref_pack_cmb", mutant)
    _fails(pins.test_golden_cmb_records)


# ---------------------------------------------------------- quantisation ----

def test_zero_point_off_by_one_is_caught(monkeypatch):
    orig = duo_o.oracle_quantize_rtn

    def mutant(W16, bits):
        q, s16, z = orig(W16, bits)
        return q, s16, z + 1

    monkeypatch.setattr(orc, "oracle_quantize_rtn", mutant)
    _fails(quant_pins.test_golden_rows)


def _rtn_mutant(scale_fp32=False, half_up=False):
    """The RTN grid with one planted change: the scale's quotient rounded to
    fp32 before fp16, or codes rounded half up instead of half to even."""
    rnd = (lambda v: np.floor(v + 0.5)) if half_up else np.rint

    def mutant(W16, bits):
        W = np.asarray(W16, np.float16)
        maxq = (1 << bits) - 1
        O, I = W.shape
        G = (I + orc.QUANT_GROUP - 1) // orc.QUANT_GROUP
        nz = (W.view(np.uint16) & 0x7FFF) != 0
        Wd = np.where(nz, W.astype(np.float64), 0.0)
        q = np.zeros((O, I), np.int64)
        s16 = np.zeros((O, G), np.float16)
        z = np.zeros((O, G), np.int64)
        for g in range(G):
            c0, c1 = g * orc.QUANT_GROUP, min(I, (g + 1) * orc.QUANT_GROUP)
            blk = Wd[:, c0:c1]
            lo = np.minimum(blk.min(axis=1), 0.0)
            hi = np.maximum(blk.max(axis=1), 0.0)
            quot = (hi - lo) / maxq
            sg = (quot.astype(np.float32) if scale_fp32 else quot).astype(np.float16)
            empty = hi == lo
            sg[empty] = np.float16(1.0)
            sg[(sg == 0) & ~empty] = np.uint16(1).view(np.float16)
            sd = sg.astype(np.float64)
            zg = np.clip(rnd(-lo / sd), 0, maxq).astype(np.int64)
            qg = np.clip(rnd(blk / sd[:, None]) + zg[:, None], 0, maxq).astype(np.int64)
            q[:, c0:c1] = np.where(nz[:, c0:c1], qg, 0)
            s16[:, g] = sg
            z[:, g] = zg
        return q, s16, z

    return mutant


def test_scale_rounded_through_fp32_is_caught(monkeypatch):
    monkeypatch.setattr(orc, "oracle_quantize_rtn", _rtn_mutant(scale_fp32=True))
    _fails(quant_pins.test_golden_rows)


def test_codes_rounded_half_up_are_caught(monkeypatch):
    monkeypatch.setattr(orc, "oracle_quantize_rtn", _rtn_mutant(half_up=True))
    _fails(quant_pins.test_golden_rows)
    _fails(quant_pins.test_brute_force_groups, 4)


# ----------------------------------------------------------- calibration ----

def _patch_precompute(monkeypatch, edit):
    orig = cal_o.oracle_calib_precompute

    def mutant(*args, **kwargs):
        pre = orig(*args, **kwargs)
        edit(pre)
        return pre

    monkeypatch.setattr(orc, "oracle_calib_precompute", mutant)


def test_sign_of_c_is_caught(monkeypatch):
    _patch_precompute(monkeypatch, lambda pre: pre.__setitem__("c", -pre["c"]))
    _fails(calib_pins.test_efficient_terms_equal_sequential_elimination, True, 6, 9, 3, False, False)


def test_dropped_b_is_caught(monkeypatch):
    _patch_precompute(monkeypatch, lambda pre: pre.__setitem__("b", 0.0 * pre["b"]))
    _fails(calib_pins.test_efficient_terms_equal_sequential_elimination, True, 6, 9, 3, False, False)


def test_transposed_factor_is_caught(monkeypatch):
    _patch_precompute(monkeypatch, lambda pre: pre.__setitem__("L", pre["L"].T.copy()))
    _fails(calib_pins.test_invariants_of_L_perm_and_sparse_input)


def test_missing_dampening_is_caught(monkeypatch):
    orig = cal_o.oracle_calib_precompute
    monkeypatch.setattr(orc, "oracle_calib_precompute",
                        lambda X, keep, damp=0.1, act_order=True: orig(X, keep, 0.0, act_order))
    _fails(calib_pins.test_invariants_of_L_perm_and_sparse_input)


def test_ignored_act_order_is_caught(monkeypatch):
    orig = cal_o.oracle_calib_precompute
    monkeypatch.setattr(orc, "oracle_calib_precompute",
                        lambda X, keep, damp=0.1, act_order=True: orig(X, keep, damp, False))
    _fails(calib_pins.test_invariants_of_L_perm_and_sparse_input)


def test_sweep_without_the_activation_term_is_caught(monkeypatch):
    orig = cal_o.oracle_calib_prune_blocked

    def mutant(W16, pre, pw_pct, block=128):   # W_j D_jq dropped from every update
        pre2 = dict(pre)
        pre2["D"] = 0.0 * pre["D"]
        return orig(W16, pre2, pw_pct, block)

    monkeypatch.setattr(orc, "oracle_calib_prune_blocked", mutant)
    _fails(calib_pins.test_sweep_blocked_equals_unblocked, 8, 24, 40, 12, 8, 50)


# ------------------------------------------------------- byte accounting ----

def test_worst_case_without_the_k_cut_is_caught(monkeypatch):
    def mutant(nnz_per_channel, k, O, I):   # forgets to keep only k channels
        n = np.sort(np.asarray(nnz_per_channel, dtype=np.float64))[::-1]
        return float(n.sum() / (O * I))

    monkeypatch.setattr(orc, "worst_case_loaded_fraction", mutant)
    _fails(pins.test_worst_case_loaded_fraction_is_the_max_over_kept_sets)


def test_worst_case_sparsest_channels_is_caught(monkeypatch):
    def mutant(nnz_per_channel, k, O, I):   # ascending sort: the k sparsest
        n = np.sort(np.asarray(nnz_per_channel, dtype=np.float64))
        return float(n[:k].sum() / (O * I))

    monkeypatch.setattr(orc, "worst_case_loaded_fraction", mutant)
    _fails(pins.test_worst_case_loaded_fraction_is_the_max_over_kept_sets)
