// Calibration precompute of DuoGPT (§4.3, Algorithm 1) on one GPU: the
// per-token sparse input, the Hessian and its inverse-Cholesky factor, Q, U,
// a, b, c, D and the efficient pruning score (C ABI: include/duo_calib.h).
//
// Every dense contraction runs on the tcgen05 GEMM of tcgemm.cu: H = X_hat
// X_hat^T and dX X_hat^T with fp16 operands (exact products, fp32 sums), the
// products with L, the factorisation's panels and updates, the triangular
// inverse and the sweep's lazy batch update with fp32 operands (three bf16
// pieces each, six piece products: fp32-level results).  Everything else is
// a kernel here.
//
// L (lower, H^-1 = L L^T) comes from one Cholesky factorisation and one
// triangular inverse: with J the index reversal, factor J H J = C C^T; then
// H^-1 = J C^-T C^-1 J = (J C^-T J)(J C^-T J)^T and J C^-T J is lower with a
// positive diagonal, so it is L.  (Forming H^-1 and factoring it again would
// take twice the flops.)  The factorisation is blocked and right-looking
// with 128-column blocks: one CTA factors a diagonal block C11 and inverts
// it in the same elimination (the row operations that reduce the block to
// C11^T turn the identity into C11^-1), the panel below is A21 C11^-T on the
// tensor cores, and the trailing matrix takes the rank-128 update
// -L21 L21^T (lower tiles only).  The triangular inverse is computed by
// recursive doubling: 64 x 64 diagonal blocks are inverted in shared memory,
// then for s = 64, 128, ... each pair [A 0; B D] of s x s diagonal blocks
// gets its off-diagonal block -D^-1 B A^-1 from two batched GEMMs.  C is kept
// in a kp x kp buffer, kp = 64 * 2^j >= k, whose trailing diagonal block is
// the identity.
#include <cstdint>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <new>
#include <unordered_set>

#include <cuda_runtime.h>

#include "duo_calib.h"
#include "duo_device.cuh"
#include "tcgemm.h"

namespace duo {
namespace calib {

constexpr int TOK_THREADS = 1024;   // the selection wants 512..1024 threads
constexpr int STAT_STRIDES = 16;    // channel statistics: 32 channels x 16 token strides
constexpr int RANK_THREADS = 256;
constexpr int EPI_THREADS = 256;
constexpr int TRI_BASE = 64;        // diagonal blocks inverted directly

// Padded order of the triangular factor: TRI_BASE * 2^j >= k.
inline int64_t tri_pad(int64_t k) {
  int64_t kp = TRI_BASE;
  while (kp < k) kp *= 2;
  return kp;
}
__host__ __device__ inline size_t tok_xs_bytes(int k) { return (2 * (size_t)k + 63) / 64 * 64; }

// X_hat and dX rows of one token (§3: keep the `keep` largest |x|, ties to
// the lower channel; the same selection as the decode sparsifier).
__global__ void __launch_bounds__(TOK_THREADS) token_sparsify_kernel(const uint16_t* __restrict__ X,
                                                                     int k, int keep,
                                                                     uint16_t* __restrict__ Xh,
                                                                     uint16_t* __restrict__ dX) {
  extern __shared__ __align__(128) uint8_t sm[];
  uint16_t* xs = reinterpret_cast<uint16_t*>(sm);
  SelShared* sel = reinterpret_cast<SelShared*>(sm + tok_xs_bytes(k));
  const size_t row = (size_t)blockIdx.x * k;
  load_x_to_smem(xs, X + row, k);
  select_clear(sel);
  __syncthreads();
  int T, cut;
  select_threshold(xs, k, keep, sel, &T, &cut);
  for (int i = threadIdx.x; i < k; i += TOK_THREADS) {
    const uint16_t v = xs[i];
    const int key = v & 0x7FFF;
    const bool kept = key > T || (key == T && i <= cut);
    Xh[row + i] = kept ? v : (uint16_t)0;
    dX[row + i] = kept ? (uint16_t)0 : v;
  }
}

// |x| * 2^24 of a finite fp16 value, an integer below 2^40.
__device__ __forceinline__ uint64_t fp16_scaled_int(uint16_t b) {
  const uint32_t e = (b >> 10) & 31u, mnt = b & 1023u;
  return e == 0 ? (uint64_t)mnt : (uint64_t)(mnt | 1024u) << (e - 1);
}

struct U128 {
  uint64_t hi, lo;
};

__device__ __forceinline__ void add128(U128& s, uint64_t hi, uint64_t lo) {
  s.lo += lo;
  s.hi += hi + (s.lo < lo ? 1u : 0u);
}

// Per channel i: key_i = diag(X_hat X_hat^T)_i * 2^48 exactly (128-bit), and
// a_i = sum_t dX[t][i]^2 (fp32).  Block: 32 channels x 16 token strides.
__global__ void __launch_bounds__(32 * STAT_STRIDES) channel_stats_kernel(
    const uint16_t* __restrict__ Xh, const uint16_t* __restrict__ dX, int k, int m,
    uint64_t* __restrict__ key_hi, uint64_t* __restrict__ key_lo, float* __restrict__ a) {
  __shared__ uint64_t shi[STAT_STRIDES][32], slo[STAT_STRIDES][32];
  __shared__ float sa[STAT_STRIDES][32];
  const int c = threadIdx.x & 31, r = threadIdx.x >> 5;
  const int i = blockIdx.x * 32 + c;
  U128 s{0, 0};
  float acc = 0.f;
  if (i < k) {
    for (int t = r; t < m; t += STAT_STRIDES) {
      const uint64_t v = fp16_scaled_int(Xh[(size_t)t * k + i] & 0x7FFFu);
      add128(s, __umul64hi(v, v), v * v);
      const float d = __half2float(__ushort_as_half(dX[(size_t)t * k + i]));
      acc = fmaf(d, d, acc);
    }
  }
  shi[r][c] = s.hi;
  slo[r][c] = s.lo;
  sa[r][c] = acc;
  __syncthreads();
  if (r == 0 && i < k) {
    for (int q = 1; q < STAT_STRIDES; ++q) {
      add128(s, shi[q][c], slo[q][c]);
      acc += sa[q][c];
    }
    key_hi[i] = s.hi;
    key_lo[i] = s.lo;
    a[i] = acc;
  }
}

// A channel never kept has H_ii = 0; it gets H_ii = 1 (key 2^48).
__device__ __forceinline__ U128 eff_key(const uint64_t* hi, const uint64_t* lo, int i) {
  U128 v{hi[i], lo[i]};
  if (v.hi == 0 && v.lo == 0) v.lo = 1ull << 48;
  return v;
}

__device__ __forceinline__ bool key_before(U128 a, int ia, U128 b, int ib) {   // a sorts before b
  if (a.hi != b.hi) return a.hi > b.hi;
  if (a.lo != b.lo) return a.lo > b.lo;
  return ia < ib;
}

// act_order: perm[rank(i)] = i, rank = channels sorting before i (largest
// diagonal first, ties to the lower index).  rank_count_kernel: one thread
// per channel i, CTA y of RANK_SPLIT compares i with the channels of its
// slice of j (keys streamed through shared memory) and adds its count to
// rank[i] (zeroed beforehand); rank_place_kernel scatters.
constexpr int RANK_SPLIT = 16;

__global__ void __launch_bounds__(RANK_THREADS) rank_count_kernel(const uint64_t* __restrict__ key_hi,
                                                                  const uint64_t* __restrict__ key_lo, int k,
                                                                  int* __restrict__ rank) {
  __shared__ uint64_t th[RANK_THREADS], tl[RANK_THREADS];
  const int i = blockIdx.x * RANK_THREADS + threadIdx.x;
  const U128 ki = i < k ? eff_key(key_hi, key_lo, i) : U128{0, 0};
  const int per = (k + RANK_SPLIT - 1) / RANK_SPLIT;
  const int jb = blockIdx.y * per, je = min(k, jb + per);
  int cnt = 0;
  for (int j0 = jb; j0 < je; j0 += RANK_THREADS) {
    __syncthreads();
    const int j = j0 + threadIdx.x;
    if (j < je) {
      const U128 kj = eff_key(key_hi, key_lo, j);
      th[threadIdx.x] = kj.hi;
      tl[threadIdx.x] = kj.lo;
    }
    __syncthreads();
    const int n = min(RANK_THREADS, je - j0);
    if (i < k)
      for (int q = 0; q < n; ++q) cnt += key_before(U128{th[q], tl[q]}, j0 + q, ki, i) ? 1 : 0;
  }
  if (i < k && cnt > 0) atomicAdd(rank + i, cnt);
}

__global__ void rank_place_kernel(const int* __restrict__ rank, int k, int act_order, int* __restrict__ perm) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < k) perm[act_order ? rank[i] : i] = i;
}

// damp * mean(diag(H)) from the exact keys (one block).
__global__ void damp_kernel(const uint64_t* __restrict__ key_hi, const uint64_t* __restrict__ key_lo,
                            int k, float damp, float* __restrict__ out) {
  __shared__ double part[256];
  double s = 0.0;
  for (int i = threadIdx.x; i < k; i += 256) {
    const U128 v = eff_key(key_hi, key_lo, i);
    s += ((double)v.hi * 18446744073709551616.0 + (double)v.lo) * 3.552713678800501e-15;   // 2^-48
  }
  part[threadIdx.x] = s;
  __syncthreads();
  for (int o = 128; o > 0; o >>= 1) {
    if (threadIdx.x < o) part[threadIdx.x] += part[threadIdx.x + o];
    __syncthreads();
  }
  if (threadIdx.x == 0) *out = (float)((double)damp * part[0] / (double)k);
}

// Reordered, dampened H (row-major Hp, and its index reversal Hr for the
// factorisation) and reordered G = dX X_hat^T (row-major Gp).  H (symmetric)
// and GT hold H_ij and G_ij at [j + i k], so output row p reads the one
// contiguous column perm[p] of each (16 KB at k = 4096) in permuted order.
__global__ void gather_kernel(const float* __restrict__ H, const float* __restrict__ GT,
                              const int* __restrict__ perm, const uint64_t* __restrict__ key_hi,
                              const uint64_t* __restrict__ key_lo, int k, int kp,
                              const float* __restrict__ dampadd, float* __restrict__ Hp,
                              float* __restrict__ Hr, float* __restrict__ Gp) {
  const int q = blockIdx.x * blockDim.x + threadIdx.x;
  const int p = blockIdx.y;
  if (q >= k) return;
  const int op = perm[p], oq = perm[q];
  float h = H[(size_t)oq + (size_t)op * k];
  if (p == q) {
    if (key_hi[op] == 0 && key_lo[op] == 0) h = 1.f;
    h += *dampadd;
  }
  Hp[(size_t)p * k + q] = h;
  Hr[(size_t)(k - 1 - p) * kp + (k - 1 - q)] = h;
  Gp[(size_t)p * k + q] = GT[(size_t)oq + (size_t)op * k];
}

// L (row-major) from C^-1 (column-major, lower, leading dimension kp):
// L[p][q] = C^-1[k-1-q][k-1-p] for p >= q, 0 above the diagonal.
__global__ void l_from_cinv_kernel(const float* __restrict__ Cinv, int k, int kp, float* __restrict__ L) {
  const int q = blockIdx.x * blockDim.x + threadIdx.x;
  const int p = blockIdx.y;
  if (q >= k) return;
  L[(size_t)p * k + q] = p >= q ? Cinv[(size_t)(k - 1 - q) + (size_t)(k - 1 - p) * kp] : 0.f;
}

// Identity on the padded trailing block of the factor buffer (rows and
// columns >= k), zeros elsewhere outside the leading k x k block.
__global__ void pad_identity_kernel(float* __restrict__ C, int k, int kp) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  const int j = blockIdx.y;
  if (i >= kp || (i < k && j < k)) return;
  C[(size_t)i + (size_t)j * kp] = i == j ? 1.f : 0.f;
}

// Zeros above the diagonal of the column-major kp x kp factor (the
// factorisation leaves the input's upper triangle there).
__global__ void zero_upper_kernel(float* __restrict__ C, int kp) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  const int j = blockIdx.y;
  if (i < j) C[(size_t)i + (size_t)j * kp] = 0.f;
}

// In-place inverse of each TRI_BASE x TRI_BASE diagonal block of the lower
// triangular C (column-major, leading dimension ld): thread j computes
// column j of the inverse by forward substitution.
__global__ void __launch_bounds__(TRI_BASE) tri_base_inverse_kernel(float* __restrict__ C, int ld) {
  __shared__ float a[TRI_BASE][TRI_BASE + 1];
  __shared__ float x[TRI_BASE][TRI_BASE + 1];
  float* blk = C + (size_t)blockIdx.x * TRI_BASE * ((size_t)ld + 1);
  const int t = threadIdx.x;
  for (int c = 0; c < TRI_BASE; ++c) a[t][c] = blk[t + (size_t)c * ld];
  __syncthreads();
  const int j = t;
  for (int i = 0; i < TRI_BASE; ++i) {
    float v = 0.f;
    if (i >= j) {
      float s = i == j ? 1.f : 0.f;
      for (int l = j; l < i; ++l) s = fmaf(-a[i][l], x[l][j], s);
      v = s / a[i][i];
    }
    x[i][j] = v;
  }
  __syncthreads();
  for (int c = 0; c < TRI_BASE; ++c) blk[t + (size_t)c * ld] = x[t][c];
}

// ---- blocked Cholesky factorisation ----

constexpr int CHOL_NB = 128;                 // columns per block
constexpr int CHOL_SUB = 32;                 // columns per sub-block (one warp)
constexpr int CHOL_THREADS = 256;
constexpr int CHOL_P = CHOL_NB + 1;          // pitch of the shared 128 x 128 arrays
constexpr int CHOL_SMEM = (2 * CHOL_NB * CHOL_P + 3 * CHOL_SUB) * (int)sizeof(float);

// The warp's factorisation of the 32 x 32 block F (pitch fp, lower
// triangle read, factor written in place).  Lane j holds column j of the
// Schur complement in a.  Step c: lane c publishes its column in shared
// memory (cbuf, two buffers), every lane reads it back with eight 16-byte
// broadcast loads, l_ic = a_ic / sqrt(a_cc), lane j >= c writes l_jc to
// F[j][c], and lanes j > c take a_ij -= l_ic l_jc over all 32 rows (rows
// above j are not used).  1 / l_cc goes to rdiag[c].  Returns the first
// pivot (1-based) that was not positive and finite, 0 if none; such a pivot
// is taken as 1.
__device__ __forceinline__ int chol_warp_factor(float* F, int fp, float* rdiag, float* cbuf, int lane) {
  float a[32];
#pragma unroll
  for (int i = 0; i < 32; ++i) a[i] = i >= lane ? F[i * fp + lane] : 0.f;
  int bad = 0;
#pragma unroll 1
  for (int c = 0; c < 32; ++c) {
    float4* cb = reinterpret_cast<float4*>(cbuf + 32 * (c & 1));
    if (lane == c) {
#pragma unroll
      for (int q = 0; q < 8; ++q) cb[q] = make_float4(a[4 * q], a[4 * q + 1], a[4 * q + 2], a[4 * q + 3]);
    }
    __syncwarp();
    float v[32];
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      const float4 t = cb[q];
      v[4 * q] = t.x;
      v[4 * q + 1] = t.y;
      v[4 * q + 2] = t.z;
      v[4 * q + 3] = t.w;
    }
    const float* cs = cbuf + 32 * (c & 1);
    float p = cs[c];
    if (!(p > 0.f) || !(p < INFINITY)) {   // warp-uniform
      if (bad == 0) bad = c + 1;
      p = 1.f;
    }
    const float inv = rsqrtf(p);
    const float lj = lane == c ? p * inv : cs[lane] * inv;   // l_(lane)c
    if (lane >= c) F[lane * fp + c] = lj;
    if (lane == c) rdiag[c] = inv;   // 1 / l_cc
    if (lane > c) {
      const float w = lj * inv;
#pragma unroll
      for (int i = 0; i < 32; ++i) a[i] = fmaf(-v[i], w, a[i]);
    }
  }
  return bad;
}

// Forward substitution with the 32 x 32 lower factor F (pitch fp, reciprocal
// diagonal rd): v <- F^-1 v, in registers (every index a constant).
__device__ __forceinline__ void chol_forward(float (&v)[32], const float* F, int fp, const float* rd) {
#pragma unroll
  for (int j = 0; j < 32; ++j) {
    float s0 = v[j], s1 = 0.f, s2 = 0.f, s3 = 0.f;   // four chains against the FMA latency
#pragma unroll
    for (int t = 0; t < j; t += 4) {
      s0 = fmaf(-F[j * fp + t], v[t], s0);
      if (t + 1 < j) s1 = fmaf(-F[j * fp + t + 1], v[t + 1], s1);
      if (t + 2 < j) s2 = fmaf(-F[j * fp + t + 2], v[t + 2], s2);
      if (t + 3 < j) s3 = fmaf(-F[j * fp + t + 3], v[t + 3], s3);
    }
    v[j] = ((s0 + s1) + (s2 + s3)) * rd[j];
  }
}

// Factor of one diagonal block and its inverse.  The block is E(j0 + i,
// j0 + j), i, j < b <= 128, of the column-major buffer E (leading dimension
// kp), lower triangle read; it holds the Schur complement left by the
// earlier blocks (the identity stands in beyond b).  Writes C11 (lower,
// zeros above the diagonal) back in place and X = C11^-1 to Linv (row-major
// 128 x 128, the identity beyond b).
//
// Four sub-blocks of 32 columns, o = 0, 32, 64, 96, each in three phases
// separated by barriers:
//  1. warp 0 factors the 32 x 32 diagonal sub-block, D = C_ss C_ss^T
//     (chol_warp_factor).
//  2. one forward substitution with C_ss per thread (128 threads): each
//     panel row below, L_is^T = C_ss^-1 A_is^T; each of the o columns of X
//     already started on rows o .. o+31, X_s = C_ss^-1 X_s (the row
//     operations of this sub-block applied to what the earlier ones left);
//     and the 32 columns of C_ss^-1 itself (X's diagonal sub-block).
//  3. the rank-32 updates of everything below, in 4 x 4 register tiles: the
//     trailing block A_ij -= L_is L_js^T (lower tiles), and X_i -= L_is X_s
//     on rows i >= o + 32 (columns < o + 32; right of those X is still 0).
// Rows of X above the current sub-block are final once their sub-block is
// done: X = C11^-1 is the elimination's row operations applied to I.  A
// pivot that is not positive and finite marks info (first column, 1-based,
// as a Cholesky routine reports it) and is replaced by 1.
__global__ void __launch_bounds__(CHOL_THREADS, 1) chol_diag_kernel(float* __restrict__ E, int kp, int j0, int b,
                                                                 float* __restrict__ Linv,
                                                                 int* __restrict__ info) {
  extern __shared__ float csm[];
  float* A = csm;                               // [128][CHOL_P]: the block, then C11 (lower)
  float* X = csm + CHOL_NB * CHOL_P;            // [128][CHOL_P]: C11^-1 (lower)
  float* rd = X + CHOL_NB * CHOL_P;             // [32]: 1 / diagonal of the current C_ss
  float* cbuf = rd + CHOL_SUB;                  // [2][32]: the warp factor's broadcast column
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  float* blk = E + (size_t)j0 * ((size_t)kp + 1);
  // the block in batches of 32 independent loads per thread (a loop that
  // stored each load before issuing the next would pay the memory latency
  // on every element)
  constexpr int LOAD_BATCH = 32;
#pragma unroll 1
  for (int base = 0; base < CHOL_NB * CHOL_NB; base += LOAD_BATCH * CHOL_THREADS) {
    float v[LOAD_BATCH];
#pragma unroll
    for (int u = 0; u < LOAD_BATCH; ++u) {
      const int idx = base + u * CHOL_THREADS + tid;
      const int i = idx & (CHOL_NB - 1), j = idx >> 7;   // i fastest: E is column-major
      v[u] = (i < b && j < b) ? (i >= j ? __ldg(blk + i + (size_t)j * kp) : 0.f) : (i == j ? 1.f : 0.f);
    }
#pragma unroll
    for (int u = 0; u < LOAD_BATCH; ++u) {
      const int idx = base + u * CHOL_THREADS + tid;
      const int i = idx & (CHOL_NB - 1), j = idx >> 7;
      A[i * CHOL_P + j] = v[u];
      X[i * CHOL_P + j] = 0.f;
    }
  }
  __syncthreads();
  for (int o = 0; o < CHOL_NB; o += CHOL_SUB) {
    float* F = A + o * CHOL_P + o;              // the sub-block's factor, pitch CHOL_P
    // ---- 1. factor the diagonal sub-block (warp 0) ----
    if (warp == 0) {
      const int bad = chol_warp_factor(F, CHOL_P, rd, cbuf, lane);
      if (lane == 0 && bad > 0 && o + bad - 1 < b) atomicCAS(info, 0, j0 + o + bad);
    }
    __syncthreads();
    // ---- 2. forward substitutions: panel rows, columns of X ----
    const int below = CHOL_NB - o - CHOL_SUB;   // rows under the sub-block
    if (tid < CHOL_NB) {                         // below + o + 32 == 128 solves
      float v[CHOL_SUB];
      if (tid < below) {                         // panel row o + 32 + tid
        const float* ar = A + (o + CHOL_SUB + tid) * CHOL_P + o;
#pragma unroll
        for (int t = 0; t < CHOL_SUB; ++t) v[t] = ar[t];
      } else if (tid < below + o) {              // column c < o of X's rows o .. o+31
        const int c = tid - below;
#pragma unroll
        for (int t = 0; t < CHOL_SUB; ++t) v[t] = X[(o + t) * CHOL_P + c];
      } else {                                   // column q of the identity
        const int q = tid - below - o;
#pragma unroll
        for (int t = 0; t < CHOL_SUB; ++t) v[t] = t == q ? 1.f : 0.f;
      }
      chol_forward(v, F, CHOL_P, rd);
      if (tid < below) {
        float* ar = A + (o + CHOL_SUB + tid) * CHOL_P + o;
#pragma unroll
        for (int t = 0; t < CHOL_SUB; ++t) ar[t] = v[t];
      } else {
        const int c = tid - below;               // o + q for the identity columns
#pragma unroll
        for (int t = 0; t < CHOL_SUB; ++t) X[(o + t) * CHOL_P + c] = v[t];
      }
    }
    __syncthreads();
    if (below == 0) break;
    // ---- 3. rank-32 updates below, in 4 x 4 tiles ----
    const int nrt = below / 4;                        // row tiles
    const int xct = (o + CHOL_SUB) / 4;               // X column tiles
    const int nx = nrt * xct, ntask = nx + nrt * (nrt + 1) / 2;
    for (int task = tid; task < ntask; task += CHOL_THREADS) {
      int i0, c0;
      const float* Y;                                 // Y(t, c): X[o + t][c] or A[c][o + t]
      int ys_t, ys_c;
      float* out;
      if (task < nx) {
        i0 = o + CHOL_SUB + 4 * (task / xct);
        c0 = 4 * (task % xct);
        Y = X + o * CHOL_P;
        ys_t = CHOL_P;
        ys_c = 1;
        out = X;
      } else {
        int tt = task - nx, ti = 0;                   // lower tile (ti, tj), tj <= ti
        while (tt > ti) {
          tt -= ti + 1;
          ++ti;
        }
        i0 = o + CHOL_SUB + 4 * ti;
        c0 = o + CHOL_SUB + 4 * tt;
        Y = A + o;
        ys_t = 1;
        ys_c = CHOL_P;
        out = A;
      }
      float acc[4][4] = {};
      const float* Lr = A + i0 * CHOL_P + o;
#pragma unroll 4
      for (int t = 0; t < CHOL_SUB; ++t) {
        float lv[4], yv[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          lv[e] = Lr[e * CHOL_P + t];
          yv[e] = Y[t * ys_t + (c0 + e) * ys_c];
        }
#pragma unroll
        for (int e = 0; e < 4; ++e)
#pragma unroll
          for (int f = 0; f < 4; ++f) acc[e][f] = fmaf(lv[e], yv[f], acc[e][f]);
      }
#pragma unroll
      for (int e = 0; e < 4; ++e)
#pragma unroll
        for (int f = 0; f < 4; ++f) out[(i0 + e) * CHOL_P + c0 + f] -= acc[e][f];
    }
    __syncthreads();
  }
  // C11 back into E (column-major, zeros above the diagonal), X to Linv
  for (int idx = tid; idx < CHOL_NB * CHOL_NB; idx += CHOL_THREADS) {
    const int i = idx & (CHOL_NB - 1), j = idx >> 7;
    if (i < b && j < b) blk[i + (size_t)j * kp] = i >= j ? A[i * CHOL_P + j] : 0.f;
  }
  for (int idx = tid; idx < CHOL_NB * CHOL_NB; idx += CHOL_THREADS) {
    const int i = idx >> 7, j = idx & (CHOL_NB - 1);   // j fastest: Linv is row-major
    Linv[idx] = j <= i ? X[i * CHOL_P + j] : 0.f;
  }
}

// Row p of Q (row-major): U = its part right of the diagonal, b_p = |U_p|^2,
// c_p = Q_pp / L_pp, col_p = 1 / L_pp^2 + a_p - b_p + 2 c_p (a in the
// original channel order, gathered through perm).
__global__ void __launch_bounds__(EPI_THREADS) q_epilogue_kernel(
    const float* __restrict__ Q, const float* __restrict__ L, const float* __restrict__ a_orig,
    const int* __restrict__ perm, int k, float* __restrict__ U, float* __restrict__ a,
    float* __restrict__ b, float* __restrict__ c, float* __restrict__ col) {
  __shared__ float part[EPI_THREADS / 32];
  const int p = blockIdx.x;
  const float* q = Q + (size_t)p * k;
  float* u = U + (size_t)p * k;
  float s = 0.f;
  for (int i = threadIdx.x; i < k; i += EPI_THREADS) {
    const float v = q[i];
    const bool up = i > p;
    u[i] = up ? v : 0.f;
    if (up) s = fmaf(v, v, s);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(FULL_MASK, s, o);
  if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = s;
  __syncthreads();
  if (threadIdx.x == 0) {
    float bp = 0.f;
    for (int w = 0; w < EPI_THREADS / 32; ++w) bp += part[w];
    const float lpp = L[(size_t)p * k + p];
    const float cp = q[p] / lpp;
    const float ap = a_orig[perm[p]];
    a[p] = ap;
    b[p] = bp;
    c[p] = cp;
    col[p] = 1.f / (lpp * lpp) + ap - bp + 2.f * cp;
  }
}

// S[r][p] = W[r][perm[p]]^2 col[p].
__global__ void score_kernel(const uint16_t* __restrict__ W, int64_t ldw, int k,
                             const int* __restrict__ perm, const float* __restrict__ col,
                             float* __restrict__ S) {
  const int p = blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t r = blockIdx.y;
  if (p >= k) return;
  const float w = __half2float(__ushort_as_half(W[r * ldw + perm[p]]));
  S[r * k + p] = w * w * col[p];
}

// ---- Algorithm 1's column sweep ----

constexpr int SWEEP_ROWS = 32;     // rows (one warp each) per CTA of the in-block sweep

// W32[r][p] = W[r][perm[p]] (fp16 -> fp32, processing order).
__global__ void load_permuted_kernel(const uint16_t* __restrict__ W, int64_t ldw, int k,
                                     const int* __restrict__ perm, float* __restrict__ W32) {
  const int p = blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t r = blockIdx.y;
  if (p >= k) return;
  W32[r * k + p] = __half2float(__ushort_as_half(W[r * ldw + perm[p]]));
}

// Monotone uint32 key of a float score (+0 and -0 map to the same key).
__device__ __forceinline__ uint32_t score_key(float s) {
  const uint32_t b = __float_as_uint(s + 0.f);
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

// Mask of one block (columns i .. i+bj-1, n rows): prune the `cnt` weights
// with the lowest S = W^2 col (equal scores: lower flat index f = r*bj + c
// first).  Multi-CTA radix select on the monotone keys: three passes of 11,
// 11 and 10 bits, each a histogram (per-CTA in shared memory, merged into a
// global one over the non-empty bins) followed by a one-CTA pick of the
// digit, give the cnt-th smallest key T and `want`, the number of elements
// equal to T to prune; per-CTA tie counts and their scan then give every tie
// its rank in flat order.  The histogram kernels are grid-strided; the tie
// and mask kernels split the elements into contiguous flat ranges of
// SELM_PER_CTA per CTA, SELM_PER_THREAD consecutive ones per thread.
constexpr int SELM_THREADS = 256;
constexpr int SELM_PER_THREAD = 8;
constexpr int SELM_PER_CTA = SELM_THREADS * SELM_PER_THREAD;
constexpr int SEL_DIGIT_BINS = 2048;   // the largest digit (11 bits)

struct SelState {
  uint32_t prefix;   // T once all passes have run
  uint32_t want;     // rank of T among the keys matching the prefix (1-based)
};

__device__ __forceinline__ int sel_shift(int pass) { return pass == 0 ? 21 : (pass == 1 ? 10 : 0); }
__device__ __forceinline__ uint32_t sel_bins(int pass) { return pass == 2 ? 1024u : 2048u; }

// Keys of the block in flat order (f = r*bj + c), and the histogram of their
// top 11 bits.  Grid-strided; (r, c) advance by the stride without a division.
__global__ void __launch_bounds__(SELM_THREADS) sel_keys_kernel(const float* __restrict__ W32, int n, int k,
                                                                int i, int bj,
                                                                const float* __restrict__ col,
                                                                uint32_t* __restrict__ keys,
                                                                uint32_t* __restrict__ hist) {
  __shared__ uint32_t h[SEL_DIGIT_BINS];
  for (int b = threadIdx.x; b < SEL_DIGIT_BINS; b += SELM_THREADS) h[b] = 0u;
  __syncthreads();
  const int64_t N = (int64_t)n * bj;
  const int stride = (int)gridDim.x * SELM_THREADS;
  const int dr = stride / bj, dc = stride - dr * bj;
  const int f0 = (int)blockIdx.x * SELM_THREADS + (int)threadIdx.x;
  int64_t r = f0 / bj;
  int c = f0 - (int)r * bj;
  for (int64_t f = f0; f < N; f += stride) {
    const float w = W32[r * k + i + c];
    const uint32_t key = score_key(w * w * col[i + c]);
    keys[f] = key;
    atomicAdd(&h[key >> 21], 1u);
    r += dr;
    c += dc;
    if (c >= bj) {
      c -= bj;
      ++r;
    }
  }
  __syncthreads();
  for (int b = threadIdx.x; b < SEL_DIGIT_BINS; b += SELM_THREADS)
    if (h[b]) atomicAdd(&hist[b], h[b]);
}

// Histogram of pass 1 or 2's digit among the keys matching the prefix.
__global__ void __launch_bounds__(SELM_THREADS) sel_hist_kernel(const uint32_t* __restrict__ keys, int64_t N,
                                                                const SelState* __restrict__ st, int pass,
                                                                uint32_t* __restrict__ hist) {
  __shared__ uint32_t h[SEL_DIGIT_BINS];
  for (int b = threadIdx.x; b < SEL_DIGIT_BINS; b += SELM_THREADS) h[b] = 0u;
  __syncthreads();
  const int sh = sel_shift(pass);
  const uint32_t hi = st->prefix >> (sh + (pass == 1 ? 11 : 10));
  const uint32_t dmask = sel_bins(pass) - 1u;
  for (int64_t f = (int64_t)blockIdx.x * SELM_THREADS + threadIdx.x; f < N; f += (int64_t)gridDim.x * SELM_THREADS) {
    const uint32_t key = keys[f];
    if ((key >> (sh + (pass == 1 ? 11 : 10))) == hi) atomicAdd(&h[(key >> sh) & dmask], 1u);
  }
  __syncthreads();
  for (int b = threadIdx.x; b < SEL_DIGIT_BINS; b += SELM_THREADS)
    if (h[b]) atomicAdd(&hist[b], h[b]);
}

// One CTA: the digit where the cumulative count reaches `want` (pass 0:
// want = cnt), the prefix extended by it; clears the histogram.
__global__ void __launch_bounds__(1024) sel_pick_kernel(uint32_t* __restrict__ hist, SelState* __restrict__ st,
                                                        int pass, uint32_t cnt) {
  __shared__ uint32_t wsum[32];
  __shared__ uint32_t s_digit, s_before;
  const int t = threadIdx.x, lane = t & 31, wid = t >> 5;
  const uint32_t want = pass == 0 ? cnt : st->want;
  if (t == 0) {   // stays so only when want == 0 (nothing to prune)
    s_digit = 0;
    s_before = 0;
  }
  // thread t: bins 2t, 2t+1 (2048 bins; pass 2 uses the first 1024)
  const uint2 hv = reinterpret_cast<const uint2*>(hist)[t];
  const uint32_t sum = hv.x + hv.y;
  uint32_t inc = sum;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t v = __shfl_up_sync(FULL_MASK, inc, o);
    if (lane >= o) inc += v;
  }
  if (lane == 31) wsum[wid] = inc;
  __syncthreads();
  if (wid == 0) {
    uint32_t v = wsum[lane];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t u = __shfl_up_sync(FULL_MASK, v, o);
      if (lane >= o) v += u;
    }
    wsum[lane] = v;
  }
  __syncthreads();
  const uint32_t excl = (wid > 0 ? wsum[wid - 1] : 0u) + inc - sum;
  if (excl < want && want <= excl + sum) {   // this thread's two bins hold the rank
    const bool first = excl + hv.x >= want;
    s_digit = 2u * (uint32_t)t + (first ? 0u : 1u);
    s_before = first ? excl : excl + hv.x;
  }
  __syncthreads();
  reinterpret_cast<uint2*>(hist)[t] = make_uint2(0u, 0u);
  if (t == 0) {
    const uint32_t d = s_digit << sel_shift(pass);
    st->prefix = pass == 0 ? d : (st->prefix | d);
    st->want = want - s_before;
  }
}

// Per CTA: how many keys equal T.
__global__ void __launch_bounds__(SELM_THREADS) sel_tie_count_kernel(const uint32_t* __restrict__ keys, int64_t N,
                                                                     const SelState* __restrict__ st,
                                                                     uint32_t* __restrict__ ctacnt) {
  __shared__ uint32_t part[SELM_THREADS / 32];
  const uint32_t T = st->prefix;
  const int64_t f0 = (int64_t)blockIdx.x * SELM_PER_CTA + (int64_t)threadIdx.x * SELM_PER_THREAD;
  uint32_t c = 0;
#pragma unroll
  for (int e = 0; e < SELM_PER_THREAD; ++e) c += (f0 + e < N && keys[f0 + e] == T) ? 1u : 0u;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) c += __shfl_xor_sync(FULL_MASK, c, o);
  if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = c;
  __syncthreads();
  if (threadIdx.x == 0) {
    uint32_t s2 = 0;
    for (int w = 0; w < SELM_THREADS / 32; ++w) s2 += part[w];
    ctacnt[blockIdx.x] = s2;
  }
}

// One CTA: exclusive scan of the per-CTA tie counts (nb <= 65536).
__global__ void __launch_bounds__(1024) sel_tie_scan_kernel(uint32_t* __restrict__ ctacnt, int nb) {
  __shared__ uint32_t part[1024];
  const int t = threadIdx.x;
  const int per = (nb + 1023) / 1024;
  uint32_t sum = 0;
  for (int b = t * per; b < min(nb, t * per + per); ++b) sum += ctacnt[b];
  part[t] = sum;
  __syncthreads();
  for (int o = 1; o < 1024; o <<= 1) {
    const uint32_t v = t >= o ? part[t - o] : 0u;
    __syncthreads();
    part[t] += v;
    __syncthreads();
  }
  uint32_t run = part[t] - sum;
  for (int b = t * per; b < min(nb, t * per + per); ++b) {
    const uint32_t c = ctacnt[b];
    ctacnt[b] = run;
    run += c;
  }
}

// Keep flags: pruned iff key < T, or key == T with flat tie rank < want.
__global__ void __launch_bounds__(SELM_THREADS) sel_mask_kernel(const uint32_t* __restrict__ keys, int64_t N,
                                                                int k, int i, int bj,
                                                                const SelState* __restrict__ st,
                                                                const uint32_t* __restrict__ ctaoff,
                                                                int none, uint8_t* __restrict__ keep) {
  __shared__ uint32_t part[SELM_THREADS / 32];
  const uint32_t T = st->prefix, want = st->want;
  const int64_t f0 = (int64_t)blockIdx.x * SELM_PER_CTA + (int64_t)threadIdx.x * SELM_PER_THREAD;
  uint32_t kv[SELM_PER_THREAD];
  uint32_t c = 0;
#pragma unroll
  for (int e = 0; e < SELM_PER_THREAD; ++e) {
    kv[e] = f0 + e < N ? keys[f0 + e] : 0xFFFFFFFFu;
    c += (f0 + e < N && kv[e] == T) ? 1u : 0u;
  }
  // rank of this thread's first tie within the CTA
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  uint32_t inc = c;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t v = __shfl_up_sync(FULL_MASK, inc, o);
    if (lane >= o) inc += v;
  }
  if (lane == 31) part[wid] = inc;
  __syncthreads();
  uint32_t wbefore = 0;
  for (int w = 0; w < wid; ++w) wbefore += part[w];
  uint32_t rank = ctaoff[blockIdx.x] + wbefore + inc - c;
#pragma unroll
  for (int e = 0; e < SELM_PER_THREAD; ++e) {
    const int64_t f = f0 + e;
    if (f < N) {
      bool pruned = false;
      if (!none) {
        if (kv[e] < T) {
          pruned = true;
        } else if (kv[e] == T) {
          pruned = rank < want;
          ++rank;
        }
      }
      const int64_t r = f / bj;
      const int cc = (int)(f - r * bj);
      keep[r * k + i + cc] = pruned ? 0 : 1;
    }
  }
}

// The block's sequential steps, one warp per row (lane l holds block
// columns l, l+32, l+64, l+96): for column j, the owner lane broadcasts W_j;
// P = W_j M_j, E_j = (W_j - P) / L_jj; later block columns q get
// W_q -= E_j L_qj - W_j D_jq; W_j = P.  The pairs {E_j, W_j as it was at its
// step} are kept for the lazy update of the trailing columns.  The block's
// coefficients come from Z (Z[q][j] = {-L_qj, D_jq}) into shared memory as
// T[j][q] (pitch SWEEP_TP), zero for q <= j, so that every lane applies
// every step to its columns without a predicate; L_jj separately.  The keep
// bits of a row are four warp-uniform ballots.  Rows per CTA: launch-time
// (warps of the block), one CTA per SM.
constexpr int SWEEP_TP = 129;   // float2 pitch of T's rows (q), padded against bank conflicts
constexpr size_t SWEEP_SMEM = (size_t)128 * SWEEP_TP * sizeof(float2) + 128 * sizeof(float);

__global__ void __launch_bounds__(1024, 1) block_sweep_kernel(float* __restrict__ W32, int n, int k, int i,
                                                              int bj, const float2* __restrict__ Z,
                                                              const float* __restrict__ L,
                                                              const uint8_t* __restrict__ keep,
                                                              float2* __restrict__ EW) {
  extern __shared__ __align__(128) uint8_t sm[];
  float2* T = reinterpret_cast<float2*>(sm);
  float* Ld = reinterpret_cast<float*>(sm + (size_t)128 * SWEEP_TP * sizeof(float2));
  for (int e = threadIdx.x; e < 128 * 128; e += blockDim.x) {   // j fastest: Z's rows are read in order
    const int q = e >> 7, j = e & 127;
    T[j * SWEEP_TP + q] = (q > j && q < bj) ? Z[(size_t)(i + q) * k + i + j] : make_float2(0.f, 0.f);
  }
  for (int t = threadIdx.x; t < 128; t += blockDim.x) Ld[t] = t < bj ? L[(size_t)(i + t) * (k + 1)] : 1.f;
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r = blockIdx.x * (blockDim.x >> 5) + warp;
  if (r >= n) return;
  float w[4];
  uint32_t km[4];
  float2 ew[4];
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    const int q = lane + 32 * u;
    w[u] = q < bj ? W32[(size_t)r * k + i + q] : 0.f;
    km[u] = __ballot_sync(FULL_MASK, q < bj && keep[(size_t)r * k + i + q] != 0);
    ew[u] = make_float2(0.f, 0.f);
  }
#pragma unroll
  for (int uj = 0; uj < 4; ++uj) {
#pragma unroll
    for (int jj = 0; jj < 32; ++jj) {
      const int j = uj * 32 + jj;
      if (j < bj) {
        const float wj = __shfl_sync(FULL_MASK, w[uj], jj);
        const bool kj = ((km[uj] >> jj) & 1u) != 0u;
        const float ej = kj ? 0.f : wj / Ld[j];
        const float2* Tj = T + j * SWEEP_TP + lane;
#pragma unroll
        for (int u = uj; u < 4; ++u) {
          const float2 z = Tj[32 * u];
          w[u] = fmaf(ej, z.x, fmaf(wj, z.y, w[u]));
        }
        if (lane == jj) {
          w[uj] = kj ? wj : 0.f;
          ew[uj] = make_float2(ej, wj);
        }
      }
    }
  }
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    const int q = lane + 32 * u;
    if (q < bj) {
      W32[(size_t)r * k + i + q] = w[u];
      EW[(size_t)r * bj + q] = ew[u];
    }
  }
}

// Z (k x 2k row-major, as float2 pairs): Z[r][c] = {-L[r][c], D[c][r]}, so that
// the lazy batch of a block is one product of K = 2 B_j: for row q after the
// block, sum over the block's columns c of -L[q][c] E[.][c] + D[c][q] W_pre[.][c].
// 32 x 32 tiles; D's tile goes through shared memory to be read transposed.
__global__ void __launch_bounds__(256) build_z_kernel(const float* __restrict__ L, const float* __restrict__ D,
                                                      int k, float2* __restrict__ Z) {
  __shared__ float t[32][33];
  const int c0 = blockIdx.x * 32, r0 = blockIdx.y * 32;
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;   // 32 x 8
  for (int y = ty; y < 32; y += 8) {   // t[c - c0][r - r0] = D[c][r]
    const int c = c0 + y, r = r0 + tx;
    t[y][tx] = (c < k && r < k) ? D[(size_t)c * k + r] : 0.f;
  }
  __syncthreads();
  for (int y = ty; y < 32; y += 8) {
    const int r = r0 + y, c = c0 + tx;
    if (r < k && c < k) Z[(size_t)r * k + c] = make_float2(-L[(size_t)r * k + c], t[tx][y]);
  }
}

// Back to the original channel order: Wout[r][perm[p]] = W32[r][p] and the
// keep mask likewise.
__global__ void store_unpermuted_kernel(const float* __restrict__ W32, const uint8_t* __restrict__ keepP,
                                        int k, const int* __restrict__ perm, float* __restrict__ Wout,
                                        uint8_t* __restrict__ keep_out) {
  const int p = blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t r = blockIdx.y;
  if (p >= k) return;
  const int o = perm[p];
  Wout[r * k + o] = W32[r * k + p];
  if (keep_out != nullptr) keep_out[r * k + o] = keepP[r * k + p];
}

}  // namespace calib
}  // namespace duo

// ---------------------------------------------------------------------------
// C ABI
// ---------------------------------------------------------------------------
namespace {

constexpr uint32_t kCalibMagic = 0x434C4243u;   // "CBLC"

}  // namespace

struct duo_calib {
  uint32_t magic;
  int device;
  int64_t k, m, kp;   // kp: padded order of the triangular factor
  uint16_t *Xh, *dX;
  float *H, *G, *Hp, *Hr, *L, *Gp, *Q, *U, *D;
  float *a_orig, *a, *b, *c, *col, *dampadd;
  uint64_t *key_hi, *key_lo;
  int* perm;
  int* rank;   // act_order ranks (scratch)
  int* info;   // factorisation status
  float* linv;                    // inverse of the current diagonal block (128 x 128)
  cudaStream_t side;              // the factorisation's diagonal blocks (high priority)
  cudaEvent_t ev_fork, ev_join;
  uint8_t *tcA, *tcB;             // prepared GEMM operands (tc_bytes each)
  size_t tc_bytes;
  void* allocs[32];
  int nalloc;
  // column sweep scratch, grown on demand: W32 (n x k fp32), keep (n x k),
  // {E, W_pre} pairs (n x 128 float2); Z (k x k float2) is rebuilt after
  // every precompute (z_ok = 0)
  float* sw_W32;
  float2* sw_EW;
  float2* sw_Z;
  int z_ok;
  uint8_t* sw_keep;
  uint32_t *sw_keys, *sw_ctacnt;
  uint8_t *sw_tcZ, *sw_tcEW;      // prepared operands of the lazy update
  int64_t sw_rows;
  uint32_t* sel_hist;             // SEL_DIGIT_BINS counters, zero between passes
  duo::calib::SelState* sel_state;
};

namespace {

std::mutex g_calib_mu;
std::unordered_set<const duo_calib*>& live_calibs() {
  static std::unordered_set<const duo_calib*> s;
  return s;
}

bool calib_live(const duo_calib* h) {
  std::lock_guard<std::mutex> lk(g_calib_mu);
  return live_calibs().count(h) != 0 && h->magic == kCalibMagic;
}

int map_cuda(cudaError_t e) {
  if (e == cudaSuccess) return DUO_OK;
  if (e == cudaErrorMemoryAllocation) return DUO_ENOMEM;
  return DUO_ECUDA;
}

void release(duo_calib* h) {
  if (h->ev_fork) cudaEventDestroy(h->ev_fork);
  if (h->ev_join) cudaEventDestroy(h->ev_join);
  if (h->side) cudaStreamDestroy(h->side);
  for (int i = 0; i < h->nalloc; ++i) cudaFree(h->allocs[i]);
  cudaFree(h->sw_W32);
  cudaFree(h->sw_EW);
  cudaFree(h->sw_Z);
  cudaFree(h->sw_keep);
  cudaFree(h->sw_keys);
  cudaFree(h->sw_ctacnt);
  cudaFree(h->sw_tcZ);
  cudaFree(h->sw_tcEW);
  delete h;
}

template <typename T>
cudaError_t alloc(duo_calib* h, T** p, size_t count) {
  void* q = nullptr;
  cudaError_t e = cudaMalloc(&q, count * sizeof(T) == 0 ? 16 : count * sizeof(T));
  if (e != cudaSuccess) return e;
  h->allocs[h->nalloc++] = q;
  *p = static_cast<T*>(q);
  return cudaSuccess;
}

bool aligned2(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 1u) == 0; }

// Bytes of one prepared-operand buffer: H and G read k x m fp16 operands,
// Q, D and the factorisation k x k (or k x 128, 128 x 128) fp32 ones, the
// triangular inverse's doubling step s a batch of kp / (2 s) s x s blocks.
size_t tc_scratch_bytes(int64_t k, int64_t m, int64_t kp) {
  using duo::TC_F16;
  using duo::TC_F32;
  using duo::tc_operand_bytes;
  size_t b = tc_operand_bytes(TC_F16, k, m, 1);
  const size_t sizes[] = {tc_operand_bytes(TC_F32, k, k, 1), tc_operand_bytes(TC_F32, k, duo::calib::CHOL_NB, 1),
                          tc_operand_bytes(TC_F32, duo::calib::CHOL_NB, duo::calib::CHOL_NB, 1)};
  for (size_t v : sizes) b = v > b ? v : b;
  for (int64_t sz = duo::calib::TRI_BASE; sz < kp; sz *= 2) {
    const size_t v = tc_operand_bytes(TC_F32, sz, sz, kp / (2 * sz));
    b = v > b ? v : b;
  }
  return b;
}

int map_tc(cudaError_t e) { return e == cudaSuccess ? DUO_OK : DUO_ECUDA; }

// Blocked right-looking Cholesky factorisation of the leading k x k block of
// the column-major factor buffer Hr (leading dimension kp), lower triangle,
// in place; a failed pivot sets info[0].  Per 128-column block at j0, with
// C11 and C11^-1 from chol_diag_kernel: the panel L21 = A21 C11^-T, then
// the trailing update A22 -= L21 L21^T in two parts: first the next block
// column, then (lower tiles) the rest.  The next block's diagonal kernel
// only needs the first part, so it runs on the context's side stream (high
// priority) while the rest of the update runs on `st`; `st` waits for it
// before the next panel.  The GEMMs read prepared copies of their operands,
// so the panel product may overwrite its own input.
int factor_blocked(duo_calib* h, cudaStream_t st) {
  using namespace duo::calib;
  using duo::TC_F32;
  const int k = (int)h->k, kp = (int)h->kp;
  float* E = h->Hr;
  cudaError_t e = cudaFuncSetAttribute(chol_diag_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, CHOL_SMEM);
  if (e != cudaSuccess) return map_cuda(e);
  chol_diag_kernel<<<1, CHOL_THREADS, CHOL_SMEM, st>>>(E, kp, 0, k < CHOL_NB ? k : CHOL_NB, h->linv, h->info);
  e = cudaGetLastError();
  // one prepared row tile of the 128-column panel: 2 chunks of 3 pieces
  const size_t tile_bytes = duo::tc_operand_bytes(TC_F32, CHOL_NB, CHOL_NB, 1);
  for (int j0 = 0; j0 + CHOL_NB < k && e == cudaSuccess; j0 += CHOL_NB) {
    const int rest = k - j0 - CHOL_NB;                     // rows below the block
    const int nb = rest < CHOL_NB ? rest : CHOL_NB;        // the next block's width
    float* P = E + (j0 + CHOL_NB) + (size_t)j0 * kp;       // E(j0 + 128 + i, j0 + l)
    duo::TcGemm g;
    g.dtype = TC_F32;
    g.M = rest;
    g.N = g.K = CHOL_NB;
    g.A = h->tcA;
    g.B = h->tcB;
    g.C = P;
    g.c_m = 1;
    g.c_n = kp;
    e = duo::tc_prep(TC_F32, P, rest, CHOL_NB, 1, 1, kp, 0, h->tcA, st);
    if (e == cudaSuccess) e = duo::tc_prep(TC_F32, h->linv, CHOL_NB, CHOL_NB, 1, CHOL_NB, 1, 0, h->tcB, st);
    if (e == cudaSuccess) e = duo::launch_tc_gemm(g, st);   // L21(i, j) = sum_l A21(i, l) C11^-1(j, l)
    if (e == cudaSuccess) e = duo::tc_prep(TC_F32, P, rest, CHOL_NB, 1, 1, kp, 0, h->tcA, st);
    // the next block column: E(j0 + 128 + i, j0 + 128 + j) -= L21_i . L21_j, j < nb
    duo::TcGemm t;
    t.dtype = TC_F32;
    t.M = rest;
    t.N = nb;
    t.K = CHOL_NB;
    t.A = t.B = h->tcA;
    t.C = E + (size_t)(j0 + CHOL_NB) * ((size_t)kp + 1);
    t.c_m = 1;
    t.c_n = kp;
    t.alpha = -1.f;
    t.beta = 1.f;
    if (e == cudaSuccess) e = duo::launch_tc_gemm(t, st);
    // the next diagonal block on the side stream
    if (e == cudaSuccess) e = cudaEventRecord(h->ev_fork, st);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(h->side, h->ev_fork, 0);
    if (e == cudaSuccess) {
      chol_diag_kernel<<<1, CHOL_THREADS, CHOL_SMEM, h->side>>>(E, kp, j0 + CHOL_NB, nb, h->linv, h->info);
      e = cudaGetLastError();
    }
    if (e == cudaSuccess) e = cudaEventRecord(h->ev_join, h->side);
    // the rest of the trailing matrix (rows and columns from j0 + 256)
    if (e == cudaSuccess && rest > CHOL_NB) {
      t.M = t.N = rest - CHOL_NB;
      t.A = t.B = h->tcA + tile_bytes;
      t.C = E + (size_t)(j0 + 2 * CHOL_NB) * ((size_t)kp + 1);
      t.lower = 1;
      t.max_ctas = -2;   // SMs left for the side stream's diagonal block
      e = duo::launch_tc_gemm(t, st);
    }
    if (e == cudaSuccess) e = cudaStreamWaitEvent(st, h->ev_join, 0);
  }
  return map_cuda(e);
}

}  // namespace

extern "C" {

int duo_calib_create(int64_t k, int64_t m, void* stream, duo_calib** out) {
  if (out == nullptr || k < 1 || k > 32768 || m < 1 || m > (1 << 20)) return DUO_EINVAL;
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    return DUO_ECUDA;
  }
  duo_calib* h = new (std::nothrow) duo_calib();
  if (h == nullptr) return DUO_ENOMEM;
  h->device = dev;
  h->k = k;
  h->m = m;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  auto fail = [&](int code) {
    release(h);
    return code;
  };
  const size_t kk = (size_t)k * k, km = (size_t)k * m;
  h->kp = duo::calib::tri_pad(k);
  cudaError_t e = cudaSuccess;
  float** mats[] = {&h->H, &h->G, &h->Hp, &h->L, &h->Gp, &h->Q, &h->U, &h->D};
  for (float** q : mats)
    if (e == cudaSuccess) e = alloc(h, q, kk);
  if (e == cudaSuccess) e = alloc(h, &h->Hr, (size_t)h->kp * h->kp);
  float** vecs[] = {&h->a_orig, &h->a, &h->b, &h->c, &h->col};
  for (float** q : vecs)
    if (e == cudaSuccess) e = alloc(h, q, (size_t)k);
  if (e == cudaSuccess) e = alloc(h, &h->dampadd, 1);
  if (e == cudaSuccess) e = alloc(h, &h->Xh, km);
  if (e == cudaSuccess) e = alloc(h, &h->dX, km);
  if (e == cudaSuccess) e = alloc(h, &h->key_hi, (size_t)k);
  if (e == cudaSuccess) e = alloc(h, &h->key_lo, (size_t)k);
  if (e == cudaSuccess) e = alloc(h, &h->perm, (size_t)k);
  if (e == cudaSuccess) e = alloc(h, &h->rank, (size_t)k);
  if (e == cudaSuccess) e = alloc(h, &h->info, 2);
  if (e == cudaSuccess) e = alloc(h, &h->sel_hist, (size_t)duo::calib::SEL_DIGIT_BINS);
  if (e == cudaSuccess) e = alloc(h, &h->sel_state, 1);
  if (e == cudaSuccess) e = cudaMemsetAsync(h->sel_hist, 0, sizeof(uint32_t) * duo::calib::SEL_DIGIT_BINS, st);
  if (e != cudaSuccess) return fail(map_cuda(e));
  // the factorisation's side stream and its fork / join events
  int prio_lo = 0, prio_hi = 0;
  if (e == cudaSuccess) e = cudaDeviceGetStreamPriorityRange(&prio_lo, &prio_hi);
  if (e == cudaSuccess) e = cudaStreamCreateWithPriority(&h->side, cudaStreamNonBlocking, prio_hi);
  if (e == cudaSuccess) e = cudaEventCreateWithFlags(&h->ev_fork, cudaEventDisableTiming);
  if (e == cudaSuccess) e = cudaEventCreateWithFlags(&h->ev_join, cudaEventDisableTiming);
  // prepared GEMM operands: the largest of the precompute's products
  h->tc_bytes = tc_scratch_bytes(k, m, h->kp);
  if (e == cudaSuccess) e = alloc(h, &h->tcA, h->tc_bytes);
  if (e == cudaSuccess) e = alloc(h, &h->tcB, h->tc_bytes);
  if (e == cudaSuccess) e = alloc(h, &h->linv, (size_t)duo::calib::CHOL_NB * duo::calib::CHOL_NB);
  if (e != cudaSuccess) return fail(map_cuda(e));
  e = cudaMemsetAsync(h->info, 0, 2 * sizeof(int), st);
  if (e == cudaSuccess) {
    const dim3 gp((unsigned)((h->kp + 255) / 256), (unsigned)h->kp);
    duo::calib::pad_identity_kernel<<<gp, 256, 0, st>>>(h->Hr, (int)k, (int)h->kp);
    e = cudaGetLastError();
  }
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) return fail(map_cuda(e));
  h->magic = kCalibMagic;
  {
    std::lock_guard<std::mutex> lk(g_calib_mu);
    live_calibs().insert(h);
  }
  *out = h;
  return DUO_OK;
}

int duo_calib_precompute(duo_calib* h, const void* X_fp16_dev, int64_t keep, float damp,
                         int act_order, void* stream) {
  if (h == nullptr || X_fp16_dev == nullptr || !calib_live(h)) return DUO_EINVAL;
  if (keep < 0 || keep > h->k || !(damp >= 0.f) || !aligned2(X_fp16_dev)) return DUO_EINVAL;
  using namespace duo::calib;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const int k = (int)h->k, m = (int)h->m;
  const uint16_t* X = static_cast<const uint16_t*>(X_fp16_dev);
  h->z_ok = 0;   // the sweep's Z follows this precompute's L and D
  // 1. X_hat and dX, one token per CTA
  const size_t tsm = tok_xs_bytes(k) + sizeof(duo::SelShared);
  cudaError_t e = cudaFuncSetAttribute(token_sparsify_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)tsm);
  if (e != cudaSuccess) return map_cuda(e);
  token_sparsify_kernel<<<m, TOK_THREADS, tsm, st>>>(X, k, (int)keep, h->Xh, h->dX);
  // 2. exact Hessian diagonal, a, act_order, dampening
  channel_stats_kernel<<<(k + 31) / 32, 32 * STAT_STRIDES, 0, st>>>(h->Xh, h->dX, k, m, h->key_hi,
                                                                    h->key_lo, h->a_orig);
  e = cudaMemsetAsync(h->rank, 0, sizeof(int) * (size_t)k, st);
  if (e != cudaSuccess) return map_cuda(e);
  if (act_order)
    rank_count_kernel<<<dim3((k + RANK_THREADS - 1) / RANK_THREADS, RANK_SPLIT), RANK_THREADS, 0, st>>>(
        h->key_hi, h->key_lo, k, h->rank);
  rank_place_kernel<<<(k + 255) / 256, 256, 0, st>>>(h->rank, k, act_order ? 1 : 0, h->perm);
  damp_kernel<<<1, 256, 0, st>>>(h->key_hi, h->key_lo, k, damp, h->dampadd);
  e = cudaGetLastError();
  if (e != cudaSuccess) return map_cuda(e);
  // 3. H = X_hat X_hat^T and G = dX X_hat^T, fp16 operands: the
  //    token-major buffers are column-major k x m matrices, so row i of an
  //    operand is channel i (stride 1) over tokens (stride k).  Outputs
  //    column-major: H[i + j k] = H_ij, and G transposed, G[i + j k] = G_ji
  //    (the product X_hat dX^T).
  using duo::TcGemm;
  using duo::TC_F16;
  using duo::TC_F32;
  int rc = map_tc(duo::tc_prep(TC_F16, h->Xh, k, m, 1, 1, k, 0, h->tcA, st));
  if (rc == DUO_OK) rc = map_tc(duo::tc_prep(TC_F16, h->dX, k, m, 1, 1, k, 0, h->tcB, st));
  if (rc != DUO_OK) return rc;
  {
    TcGemm g;
    g.dtype = TC_F16;
    g.M = g.N = k;
    g.K = m;
    g.A = g.B = h->tcA;
    g.C = h->H;
    g.c_m = 1;
    g.c_n = k;
    rc = map_tc(duo::launch_tc_gemm(g, st));
    if (rc != DUO_OK) return rc;
    g.B = h->tcB;
    g.C = h->G;
    rc = map_tc(duo::launch_tc_gemm(g, st));
    if (rc != DUO_OK) return rc;
  }
  // 4. reorder and dampen, then L
  const dim3 g2((k + 255) / 256, k);
  const int kp = (int)h->kp;
  gather_kernel<<<g2, 256, 0, st>>>(h->H, h->G, h->perm, h->key_hi, h->key_lo, k, kp, h->dampadd, h->Hp,
                                    h->Hr, h->Gp);
  e = cudaMemsetAsync(h->info, 0, 2 * sizeof(int), st);
  if (e == cudaSuccess) e = cudaGetLastError();
  if (e != cudaSuccess) return map_cuda(e);
  rc = factor_blocked(h, st);
  if (rc != DUO_OK) return rc;
  // C^-1 in place: base blocks, then one doubling step per level.  The
  // step's product B A^-1 goes to the H buffer (no longer needed; it holds
  // kp s / 2 <= k^2 floats).
  {
    const dim3 gz((unsigned)((kp + 255) / 256), (unsigned)kp);
    zero_upper_kernel<<<gz, 256, 0, st>>>(h->Hr, kp);
    tri_base_inverse_kernel<<<kp / TRI_BASE, TRI_BASE, 0, st>>>(h->Hr, kp);
    e = cudaGetLastError();
    if (e != cudaSuccess) return map_cuda(e);
    for (int sz = TRI_BASE; sz < kp; sz *= 2) {
      const int batch = kp / (2 * sz);
      const int64_t stride = 2LL * sz * ((int64_t)kp + 1);   // between diagonal block pairs
      float* A = h->Hr;                                      // upper-left s x s block of a pair
      float* B = h->Hr + sz;                                 // lower-left
      float* Dg = h->Hr + sz + (size_t)sz * kp;              // lower-right
      // T = B A^-1: T(i, j) = sum_l B(i, l) A^-1(l, j)
      rc = map_tc(duo::tc_prep(TC_F32, B, sz, sz, batch, 1, kp, stride, h->tcA, st));
      if (rc == DUO_OK) rc = map_tc(duo::tc_prep(TC_F32, A, sz, sz, batch, kp, 1, stride, h->tcB, st));
      TcGemm g;
      g.dtype = TC_F32;
      g.M = g.N = g.K = sz;
      g.batch = batch;
      g.A = h->tcA;
      g.B = h->tcB;
      g.C = h->H;
      g.c_m = 1;
      g.c_n = sz;
      g.c_bs = (int64_t)sz * sz;
      if (rc == DUO_OK) rc = map_tc(duo::launch_tc_gemm(g, st));
      // B <- -D^-1 T
      if (rc == DUO_OK) rc = map_tc(duo::tc_prep(TC_F32, Dg, sz, sz, batch, 1, kp, stride, h->tcA, st));
      if (rc == DUO_OK)
        rc = map_tc(duo::tc_prep(TC_F32, h->H, sz, sz, batch, sz, 1, (int64_t)sz * sz, h->tcB, st));
      g.C = B;
      g.c_n = kp;
      g.c_bs = stride;
      g.alpha = -1.f;
      if (rc == DUO_OK) rc = map_tc(duo::launch_tc_gemm(g, st));
      if (rc != DUO_OK) return rc;
    }
  }
  l_from_cinv_kernel<<<g2, 256, 0, st>>>(h->Hr, k, kp, h->L);
  e = cudaGetLastError();
  if (e != cudaSuccess) return map_cuda(e);
  // 5. Q = Gp L (row-major buffers): Q^T(i, j) = sum_l L(l, i) Gp(j, l), so
  //    with column-major output A(i, l) = L[l k + i] and B(j, l) = Gp[j k + l].
  TcGemm g;
  g.dtype = TC_F32;
  g.M = g.N = g.K = k;
  g.c_m = 1;
  g.c_n = k;
  g.A = h->tcA;
  g.B = h->tcB;
  rc = map_tc(duo::tc_prep(TC_F32, h->L, k, k, 1, 1, k, 0, h->tcA, st));
  if (rc == DUO_OK) rc = map_tc(duo::tc_prep(TC_F32, h->Gp, k, k, 1, k, 1, 0, h->tcB, st));
  g.C = h->Q;
  if (rc == DUO_OK) rc = map_tc(duo::launch_tc_gemm(g, st));
  if (rc != DUO_OK) return rc;
  // 6. U, a (reordered), b, c and the score's column factor
  q_epilogue_kernel<<<k, EPI_THREADS, 0, st>>>(h->Q, h->L, h->a_orig, h->perm, k, h->U, h->a, h->b, h->c,
                                               h->col);
  e = cudaGetLastError();
  if (e != cudaSuccess) return map_cuda(e);
  // 7. D = U L^T (row-major): D^T(i, j) = sum_l L(i, l) U(j, l), A(i, l) =
  //    L[i k + l], B(j, l) = U[j k + l].
  rc = map_tc(duo::tc_prep(TC_F32, h->L, k, k, 1, k, 1, 0, h->tcA, st));
  if (rc == DUO_OK) rc = map_tc(duo::tc_prep(TC_F32, h->U, k, k, 1, k, 1, 0, h->tcB, st));
  g.C = h->D;
  if (rc == DUO_OK) rc = map_tc(duo::launch_tc_gemm(g, st));
  return rc;
}

int duo_calib_status(const duo_calib* h, void* stream) {
  if (h == nullptr || !calib_live(h)) return DUO_EINVAL;
  cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return DUO_ECUDA;
  int info[2] = {0, 0};
  e = cudaMemcpy(info, h->info, sizeof(info), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return DUO_ECUDA;
  unsigned int tc = 0;
  if (duo::tc_gemm_take_status(&tc) != cudaSuccess) return DUO_ECUDA;
  if (tc != 0) return DUO_ETIMEOUT;
  return info[0] != 0 ? DUO_ERANGE : DUO_OK;
}

int duo_calib_query(const duo_calib* h, duo_calib_info* info) {
  if (h == nullptr || info == nullptr || !calib_live(h)) return DUO_EINVAL;
  std::memset(info, 0, sizeof(*info));
  info->k = h->k;
  info->m = h->m;
  info->perm_dev = h->perm;
  info->H_dev = h->Hp;
  info->L_dev = h->L;
  info->Q_dev = h->Q;
  info->U_dev = h->U;
  info->D_dev = h->D;
  info->a_dev = h->a;
  info->b_dev = h->b;
  info->c_dev = h->c;
  info->col_dev = h->col;
  return DUO_OK;
}

int duo_calib_export(const duo_calib* h, int which, void* dst_dev, int64_t bytes, void* stream) {
  if (h == nullptr || dst_dev == nullptr || !calib_live(h)) return DUO_EINVAL;
  const int64_t kk = h->k * h->k * 4, kv = h->k * 4;
  const void* src = nullptr;
  int64_t n = 0;
  switch (which) {
    case 0: src = h->perm; n = kv; break;
    case 1: src = h->Hp; n = kk; break;
    case 2: src = h->L; n = kk; break;
    case 3: src = h->Q; n = kk; break;
    case 4: src = h->U; n = kk; break;
    case 5: src = h->D; n = kk; break;
    case 6: src = h->a; n = kv; break;
    case 7: src = h->b; n = kv; break;
    case 8: src = h->c; n = kv; break;
    case 9: src = h->col; n = kv; break;
    default: return DUO_EINVAL;
  }
  if (bytes != n) return DUO_EINVAL;
  return map_cuda(cudaMemcpyAsync(dst_dev, src, (size_t)n, cudaMemcpyDeviceToDevice,
                                  static_cast<cudaStream_t>(stream)));
}

int duo_calib_score(const duo_calib* h, const void* W_fp16_dev, int64_t n, int64_t ldw, float* S_dev,
                    void* stream) {
  if (h == nullptr || W_fp16_dev == nullptr || S_dev == nullptr || !calib_live(h)) return DUO_EINVAL;
  if (n < 1 || n > 65535 || ldw < h->k || !aligned2(W_fp16_dev) ||
      (reinterpret_cast<uintptr_t>(S_dev) & 3u) != 0)
    return DUO_EINVAL;
  const int k = (int)h->k;
  const dim3 grid((k + 255) / 256, (unsigned)n);
  duo::calib::score_kernel<<<grid, 256, 0, static_cast<cudaStream_t>(stream)>>>(
      static_cast<const uint16_t*>(W_fp16_dev), ldw, k, h->perm, h->col, S_dev);
  return map_cuda(cudaGetLastError());
}

int duo_calib_prune(duo_calib* h, const void* W_fp16_dev, int64_t n, int64_t ldw, int pw_pct, int block,
                    float* Wout_dev, uint8_t* keep_dev, void* stream) {
  if (h == nullptr || W_fp16_dev == nullptr || Wout_dev == nullptr || !calib_live(h)) return DUO_EINVAL;
  if (n < 1 || n > 65535 || ldw < h->k || pw_pct < 0 || pw_pct > 100 || block < 1 || block > 128 ||
      !aligned2(W_fp16_dev) || (reinterpret_cast<uintptr_t>(Wout_dev) & 3u) != 0)
    return DUO_EINVAL;
  using namespace duo::calib;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const int k = (int)h->k;
  cudaError_t e = cudaSuccess;
  if (h->sw_rows < n) {   // grow the scratch (the stream's earlier work may still use it)
    e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return map_cuda(e);
    cudaFree(h->sw_W32);
    cudaFree(h->sw_EW);
    cudaFree(h->sw_keep);
    cudaFree(h->sw_keys);
    cudaFree(h->sw_ctacnt);
    cudaFree(h->sw_tcEW);
    h->sw_tcEW = nullptr;
    h->sw_W32 = nullptr;
    h->sw_EW = nullptr;
    h->sw_keep = nullptr;
    h->sw_keys = h->sw_ctacnt = nullptr;
    h->sw_rows = 0;
    const size_t nk = (size_t)n * k;
    e = cudaMalloc(&h->sw_W32, nk * sizeof(float));
    if (e == cudaSuccess) e = cudaMalloc(&h->sw_EW, (size_t)n * 128 * sizeof(float2));
    if (e == cudaSuccess) e = cudaMalloc(&h->sw_keep, nk);
    if (e == cudaSuccess) e = cudaMalloc(&h->sw_keys, (size_t)n * 128 * sizeof(uint32_t));
    if (e == cudaSuccess)
      e = cudaMalloc(&h->sw_ctacnt, ((size_t)n * 128 / SELM_PER_CTA + 1) * sizeof(uint32_t));
    if (e == cudaSuccess) e = cudaMalloc(&h->sw_tcEW, duo::tc_operand_bytes(duo::TC_F32, n, 2 * 128, 1));
    if (e != cudaSuccess) return map_cuda(e);
    h->sw_rows = n;
  }
  float* W32 = h->sw_W32;
  float2* EW = h->sw_EW;
  if (h->sw_Z == nullptr) {
    e = cudaMalloc(&h->sw_Z, (size_t)k * k * sizeof(float2));
    if (e == cudaSuccess && h->sw_tcZ == nullptr)
      e = cudaMalloc(&h->sw_tcZ, duo::tc_operand_bytes(duo::TC_F32, k, 2 * 128, 1));
    if (e != cudaSuccess) return map_cuda(e);
    h->z_ok = 0;
  }
  if (!h->z_ok) {
    const dim3 gz((k + 31) / 32, (k + 31) / 32);
    build_z_kernel<<<gz, 256, 0, st>>>(h->L, h->D, k, h->sw_Z);
    h->z_ok = 1;
  }
  uint8_t* keepP = h->sw_keep;
  const dim3 gk((k + 255) / 256, (unsigned)n);
  load_permuted_kernel<<<gk, 256, 0, st>>>(static_cast<const uint16_t*>(W_fp16_dev), ldw, k, h->perm, W32);
  e = cudaFuncSetAttribute(block_sweep_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)SWEEP_SMEM);
  if (e != cudaSuccess) return map_cuda(e);
  // rows (warps) per CTA of the in-block sweep: one CTA per SM, waves of 152
  const int64_t waves = (n + (int64_t)152 * SWEEP_ROWS - 1) / ((int64_t)152 * SWEEP_ROWS);
  const int rpc = (int)((n + 152 * waves - 1) / (152 * waves));
  for (int i = 0; i < k; i += block) {
    const int bj = k - i < block ? k - i : block;
    const int64_t cnt = (int64_t)n * bj * pw_pct / 100;
    const int64_t N = (int64_t)n * bj;
    const unsigned nb = (unsigned)((N + SELM_PER_CTA - 1) / SELM_PER_CTA);
    const unsigned nh = nb < 2u * 152u ? nb : 2u * 152u;   // histogram CTAs, grid-strided
    sel_keys_kernel<<<nh, SELM_THREADS, 0, st>>>(W32, (int)n, k, i, bj, h->col, h->sw_keys, h->sel_hist);
    sel_pick_kernel<<<1, 1024, 0, st>>>(h->sel_hist, h->sel_state, 0, (uint32_t)cnt);
    sel_hist_kernel<<<nh, SELM_THREADS, 0, st>>>(h->sw_keys, N, h->sel_state, 1, h->sel_hist);
    sel_pick_kernel<<<1, 1024, 0, st>>>(h->sel_hist, h->sel_state, 1, (uint32_t)cnt);
    sel_hist_kernel<<<nh, SELM_THREADS, 0, st>>>(h->sw_keys, N, h->sel_state, 2, h->sel_hist);
    sel_pick_kernel<<<1, 1024, 0, st>>>(h->sel_hist, h->sel_state, 2, (uint32_t)cnt);
    sel_tie_count_kernel<<<nb, SELM_THREADS, 0, st>>>(h->sw_keys, N, h->sel_state, h->sw_ctacnt);
    sel_tie_scan_kernel<<<1, 1024, 0, st>>>(h->sw_ctacnt, (int)nb);
    sel_mask_kernel<<<nb, SELM_THREADS, 0, st>>>(h->sw_keys, N, k, i, bj, h->sel_state, h->sw_ctacnt,
                                                 cnt == 0 ? 1 : 0, keepP);
    block_sweep_kernel<<<(unsigned)((n + rpc - 1) / rpc), (unsigned)rpc * 32, SWEEP_SMEM, st>>>(
        W32, (int)n, k, i, bj, h->sw_Z, h->L, keepP, EW);
    e = cudaGetLastError();
    if (e != cudaSuccess) return map_cuda(e);
    const int nt = k - i - bj;   // trailing columns
    if (nt > 0) {
      // Lazy batch: W_T -= E L_T,blk^T - W_pre D_blk,T as one product of
      // K = 2 B_j over the pairs.  With column-major output over W32's rows
      // (C(t, r) = W32[r k + i + bj + t]): A(t, l) = Z[i + bj + t] as floats
      // (Z[q][j] = {-L_qj, D_jq}, pairs of block columns j), B(r, l) =
      // {E, W_pre} of row r.
      const float* Zb = reinterpret_cast<const float*>(h->sw_Z) + (size_t)(i + bj) * 2 * k + 2 * (size_t)i;
      duo::TcGemm g;
      g.dtype = duo::TC_F32;
      g.M = nt;
      g.N = (int)n;
      g.K = 2 * bj;
      g.A = h->sw_tcZ;
      g.B = h->sw_tcEW;
      g.C = W32 + i + bj;
      g.c_m = 1;
      g.c_n = k;
      g.beta = 1.f;
      e = duo::tc_prep(duo::TC_F32, Zb, nt, 2 * bj, 1, 2 * (int64_t)k, 1, 0, h->sw_tcZ, st);
      if (e == cudaSuccess)
        e = duo::tc_prep(duo::TC_F32, EW, n, 2 * bj, 1, 2 * (int64_t)bj, 1, 0, h->sw_tcEW, st);
      if (e == cudaSuccess) e = duo::launch_tc_gemm(g, st);
      if (e != cudaSuccess) return map_cuda(e);
    }
  }
  store_unpermuted_kernel<<<gk, 256, 0, st>>>(W32, keepP, k, h->perm, Wout_dev, keep_dev);
  return map_cuda(cudaGetLastError());
}

int duo_calib_free(duo_calib* h) {
  if (h == nullptr) return DUO_OK;
  {
    std::lock_guard<std::mutex> lk(g_calib_mu);
    auto& s = live_calibs();
    auto it = s.find(h);
    if (it == s.end()) return DUO_EINVAL;
    s.erase(it);
  }
  h->magic = 0;
  release(h);
  return DUO_OK;
}

}  // extern "C"
