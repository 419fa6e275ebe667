// Dense GEMM on the tcgen05 tensor cores (kernels: tcgemm.cu).
//
//     C(i, j) = alpha * sum_l A(i, l) B(j, l) + beta * C(i, j)
//
// for i < M, j < N, l < K and each batch index z < batch.  C is fp32,
// addressed through element strides: C(i, j) = C[z c_bs + i c_m + j c_n].
// A and B are first brought into the tensor-core operand layout by tc_prep,
// which reads any strided matrix X(r, l) = X[z s_b + r s_r + l s_k] of rows
// x K (fp16 or fp32) into a buffer of tc_operand_bytes: 128-row x 64-column
// tiles, each stored as the shared-memory image the MMAs read (K-major
// no-swizzle core matrices), zero beyond rows and K.  A prepared operand is
// reused by every product that reads it.
//
// Arithmetic: fp16 operands multiply exactly and accumulate in fp32.  fp32
// operands are split by tc_prep into three bf16 pieces each (x = x0 + x1 +
// x2 to 24 significant bits; each residual is exact), and the product is the
// sum of the six piece products whose indices add to at most 2.  The dropped
// terms are below 2^-24 of |A| |B|, so the result is within a few fp32
// roundings of the fp32 product.
//
// With `lower` set only the 128 x 128 output tiles whose first column is not
// right of their first row are written (the lower triangle of a square C, in
// whole tiles).  beta == 0 never reads C.
#pragma once
#include <cstddef>
#include <cstdint>
#include <cuda_runtime.h>

namespace duo {

enum TcType : int { TC_F16 = 0, TC_F32 = 1 };

// Bytes of a prepared operand of rows x K (per batch entry, times batch).
size_t tc_operand_bytes(int dtype, int64_t rows, int64_t K, int64_t batch);

// Writes the prepared image of X (rows x K, strides s_r, s_k, batch stride
// s_b) to dst (device, 16-byte aligned, tc_operand_bytes long).
cudaError_t tc_prep(int dtype, const void* X, int64_t rows, int64_t K, int64_t batch, int64_t s_r, int64_t s_k,
                    int64_t s_b, void* dst, cudaStream_t st);

struct TcGemm {
  int dtype = TC_F32;
  int M = 0, N = 0, K = 0, batch = 1;
  const void* A = nullptr;   // prepared: M rows x K
  const void* B = nullptr;   // prepared: N rows x K
  float* C = nullptr;
  int64_t c_m = 0, c_n = 0, c_bs = 0;
  float alpha = 1.f, beta = 0.f;
  int lower = 0;      // lower tiles only (M == N)
  int max_ctas = 0;   // persistent CTAs at most: 0 one per SM, n > 0 at most n, n < 0 all SMs but |n|
                      // (SMs left free for kernels on other streams)
};

// Enqueues the product on `st`.  M, N or batch of 0 is a no-op; K < 1, a
// batch above 65535 or `lower` with M != N is cudaErrorInvalidValue.
cudaError_t launch_tc_gemm(const TcGemm& g, cudaStream_t st);

// Reads and clears the tensor-core GEMM status word: bit 0 is set when a
// bounded wait ran out (that tile is then not written).
cudaError_t tc_gemm_take_status(unsigned int* out);

}  // namespace duo
