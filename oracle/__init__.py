"""CPU oracle for the dual-sparse batch-1 spMspV of DuoGPT (arXiv 2506.20194).

TEST INFRASTRUCTURE ONLY.  Nothing in the product path imports this package:
only ``tests/``, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` /
``--impl reference`` legs of ``bench.py`` may import or call it.  It shares no
code with the CUDA library (no kernels, headers, tables or helpers) and does
not import ``paper_2506_20194_gb300``.

Every function is pinned by ``tests/test_oracle_*.py`` against something other
than itself (exact integer arithmetic, exactly-rounded summation, brute force
on tiny inputs, closed forms and invariants).  No function here is "parity
unpinned".
"""
from .duo_oracle import (  # noqa: F401
    SEG_ROWS,
    CMB_MAGIC,
    IDX16_MAGIC,
    k_from_pct,
    oracle_sparsify,
    oracle_sparsify_threshold,
    oracle_spmspv_threshold,
    oracle_spmspv,
    oracle_spmspv_rows,
    exact_spmspv_rows_scaled,
    fsum_spmspv_rows,
    tolerance_rows,
    ref_pack_cmb,
    ref_unpack_cmb,
    ref_pack_idx16,
    ref_unpack_idx16,
    required_bytes,
    loaded_fraction,
    worst_case_loaded_fraction,
    QUANT_GROUP,
    QUANT_BITS,
    oracle_quantize_rtn,
    oracle_dequantize,
    oracle_spmspv_q,
    oracle_spmspv_q_threshold,
    exact_spmspv_q_rows_scaled,
    tolerance_rows_f64,
    ref_pack_cmb_q,
    ref_unpack_cmb_q,
    required_bytes_q,
)
from .calib_oracle import (  # noqa: F401
    DAMP,
    sparsify_columns,
    exact_diag_keys,
    oracle_calib_precompute,
    oracle_calib_score,
    oracle_calib_prune,
    oracle_calib_prune_blocked,
)
