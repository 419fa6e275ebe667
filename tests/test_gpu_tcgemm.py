"""GPU parity of the tcgen05 GEMM behind the calibration's contractions
(Algorithm 1, §4.3), through the library's internal test entry
duo_test_tc_gemm: C = alpha A B^T + beta C with strided operands.

Reference: the same product in fp64 on the CPU from the same inputs.  Bar
per element: |C - C_ref| <= 4e-6 (1 + K / 256) sum_l |alpha A_il B_jl| +
|beta C0_ij| 2^-23: fp16 operands multiply exactly and accumulate in fp32;
fp32 operands are split into three bf16 pieces (24 bits), of whose nine
piece products the six largest are summed, the dropped ones below 2^-24 of
|A_il B_jl|.  Tiles skipped by `lower` must keep C's old values exactly.
Shapes cover ragged edges in M, N and K, both layouts of each operand,
batches, more tiles than SMs, and persistent CTAs capped at a few.
"""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    from paper_2506_20194_gb300 import duo as d
    return d.load_library()


CASES = [
    # dtype, M, N, K, batch, A col-major, B col-major, C col-major, alpha, beta, lower, max_ctas
    ("f16", 128, 128, 64, 1, 0, 0, 0, 1.0, 0.0, 0, 0),
    ("f16", 200, 130, 100, 1, 0, 0, 0, 1.0, 0.0, 0, 0),
    ("f16", 129, 257, 77, 2, 1, 0, 1, 0.5, 1.0, 0, 0),
    ("f16", 1664, 1664, 64, 1, 0, 1, 1, 1.0, 0.0, 0, 0),
    ("f32", 33, 17, 5, 2, 0, 1, 0, 2.0, 0.5, 0, 0),
    ("f32", 256, 256, 640, 1, 1, 0, 1, -1.0, 1.0, 0, 0),
    ("f32", 300, 300, 200, 1, 1, 1, 1, -1.0, 1.0, 1, 0),
    ("f32", 1280, 2176, 96, 1, 1, 0, 1, -1.0, 1.0, 0, 0),
    ("f32", 640, 640, 200, 1, 1, 1, 1, 1.0, 0.5, 0, 3),
    ("f32", 1152, 1152, 128, 1, 1, 1, 1, -1.0, 1.0, 1, 5),
    ("f32", 256, 256, 64, 7, 1, 0, 1, -1.0, 0.0, 0, -2),
]


def _layout(rows, cols, batch, colmajor):
    """Strides (row, col, batch) of a rows x cols matrix stored row- or
    column-major, batch entries back to back."""
    return (1, rows, rows * cols) if colmajor else (cols, 1, rows * cols)


@pytest.mark.parametrize("case", CASES, ids=[f"{c[0]}-{c[1]}x{c[2]}x{c[3]}-b{c[4]}-l{c[10]}-c{c[11]}" for c in CASES])
def test_tc_gemm_matches_fp64(lib, case):
    dt, M, N, K, Bt, acm, bcm, ccm, alpha, beta, lower, ctas = case
    rng = np.random.default_rng(M * 7 + N + K)
    npdt = np.float16 if dt == "f16" else np.float32
    A = rng.standard_normal((Bt, M, K)).astype(npdt)
    B = rng.standard_normal((Bt, N, K)).astype(npdt)
    C0 = rng.standard_normal((Bt, M, N)).astype(np.float32)
    sa, sb, sc = _layout(M, K, Bt, acm), _layout(N, K, Bt, bcm), _layout(M, N, Bt, ccm)

    def store(X, colmajor):
        return np.ascontiguousarray(X.transpose(0, 2, 1) if colmajor else X).ravel()

    dA = torch.from_numpy(store(A, acm)).cuda()
    dB = torch.from_numpy(store(B, bcm)).cuda()
    dC = torch.from_numpy(store(C0, ccm)).cuda()
    stream = torch.cuda.current_stream().cuda_stream
    rc = lib.duo_test_tc_gemm(0 if dt == "f16" else 1, M, N, K, Bt, dA.data_ptr(), *sa, dB.data_ptr(), *sb,
                              dC.data_ptr(), *sc, alpha, beta, lower, ctas, stream)
    assert rc == 0
    got = dC.cpu().numpy().reshape((Bt, N, M) if ccm else (Bt, M, N))
    if ccm:
        got = got.transpose(0, 2, 1)
    A64, B64 = A.astype(np.float64), B.astype(np.float64)
    ref = alpha * np.einsum("zik,zjk->zij", A64, B64) + beta * C0.astype(np.float64)
    mag = np.abs(alpha) * np.einsum("zik,zjk->zij", np.abs(A64), np.abs(B64))
    tol = 4e-6 * (1 + K / 256) * mag + np.abs(beta * C0.astype(np.float64)) * 2.0 ** -23 + 1e-30
    if lower:
        ti = np.arange(M)[:, None] // 128
        tj = np.arange(N)[None, :] // 128
        skip = np.broadcast_to(tj > ti, (Bt, M, N))
        assert np.array_equal(got[skip], C0[skip])
        keep = ~skip
        assert np.all(np.abs(got[keep] - ref[keep]) <= tol[keep])
    else:
        assert np.all(np.abs(got - ref) <= tol), float((np.abs(got - ref) / tol).max())


def test_tc_gemm_rejects_bad_shapes(lib):
    x = torch.zeros(16, device="cuda")
    stream = torch.cuda.current_stream().cuda_stream
    args = (x.data_ptr(), 1, 4, 16, x.data_ptr(), 1, 4, 16, x.data_ptr(), 1, 4, 16, 1.0, 0.0)
    assert lib.duo_test_tc_gemm(1, 4, 4, 0, 1, *args, 0, 0, stream) == -1       # K < 1
    assert lib.duo_test_tc_gemm(1, 4, 3, 4, 1, *args, 1, 0, stream) == -1       # lower with M != N
    assert lib.duo_test_tc_gemm(2, 4, 4, 4, 1, *args, 0, 0, stream) == -1       # no such type
