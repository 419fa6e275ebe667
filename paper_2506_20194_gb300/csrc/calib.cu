// Calibration precompute of DuoGPT (§4.3, Algorithm 1) on one GPU: the
// per-token sparse input, the Hessian and its inverse-Cholesky factor, Q, U,
// a, b, c, D and the efficient pruning score (C ABI: include/duo_calib.h).
//
// Plain GEMMs go to cuBLAS: H = X_hat X_hat^T and dX X_hat^T with fp16
// inputs and fp32 accumulation on the tensor cores, the products with L in
// fp32 (emulated with bf16 tensor-core products, see kL_COMPUTE).  The
// factorisation goes to cuSOLVER.  Everything else is a kernel here.
//
// L (lower, H^-1 = L L^T) comes from one Cholesky factorisation and one
// triangular inverse: with J the index reversal, factor J H J = C C^T; then
// H^-1 = J C^-T C^-1 J = (J C^-T J)(J C^-T J)^T and J C^-T J is lower with a
// positive diagonal, so it is L.  (Forming H^-1 and factoring it again would
// take twice the flops.)  The triangular inverse is computed here by
// recursive doubling: 64 x 64 diagonal blocks are inverted in shared memory,
// then for s = 64, 128, ... each pair [A 0; B D] of s x s diagonal blocks
// gets its off-diagonal block -D^-1 B A^-1 from two batched tensor-core
// GEMMs.  (cuSOLVER's trtri took 8.3 ms at k = 4096 on GB300, its
// factorisation 2.1 ms.)  C is kept in a kp x kp buffer, kp = 64 * 2^j >= k,
// whose trailing diagonal block is the identity.
#include <cstdint>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <new>
#include <unordered_set>

#include <cublas_v2.h>
#include <cuda_runtime.h>
#include <cusolverDn.h>

#include "duo_calib.h"
#include "duo_device.cuh"

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
// Products with L in fp32 through cuBLAS's BF16x9 emulation on the tensor
// cores: measured on GB300 at k = 4096, 215 TFLOP/s with a max error of
// 7e-7 relative, against 67 TFLOP/s and 2.5e-6 for the plain fp32 path.
constexpr cublasComputeType_t kL_COMPUTE = CUBLAS_COMPUTE_32F_EMULATED_16BFX9;

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
// diagonal first, ties to the lower index).  One thread per channel, keys
// streamed through shared memory.
__global__ void __launch_bounds__(RANK_THREADS) rank_kernel(const uint64_t* __restrict__ key_hi,
                                                            const uint64_t* __restrict__ key_lo, int k,
                                                            int act_order, int* __restrict__ perm) {
  __shared__ uint64_t th[RANK_THREADS], tl[RANK_THREADS];
  const int i = blockIdx.x * RANK_THREADS + threadIdx.x;
  const U128 ki = i < k ? eff_key(key_hi, key_lo, i) : U128{0, 0};
  int rank = 0;
  for (int j0 = 0; j0 < k; j0 += RANK_THREADS) {
    __syncthreads();
    const int j = j0 + threadIdx.x;
    if (j < k) {
      const U128 kj = eff_key(key_hi, key_lo, j);
      th[threadIdx.x] = kj.hi;
      tl[threadIdx.x] = kj.lo;
    }
    __syncthreads();
    const int n = min(RANK_THREADS, k - j0);
    if (i < k && act_order)
      for (int q = 0; q < n; ++q) rank += key_before(U128{th[q], tl[q]}, j0 + q, ki, i) ? 1 : 0;
  }
  if (i < k) perm[act_order ? rank : i] = i;
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
// factorisation) and reordered G = dX X_hat^T (row-major Gp).  H and G are
// cuBLAS column-major: G[i + j k] = (dX X_hat^T)_ij.
__global__ void gather_kernel(const float* __restrict__ H, const float* __restrict__ G,
                              const int* __restrict__ perm, const uint64_t* __restrict__ key_hi,
                              const uint64_t* __restrict__ key_lo, int k, int kp,
                              const float* __restrict__ dampadd, float* __restrict__ Hp,
                              float* __restrict__ Hr, float* __restrict__ Gp) {
  const int q = blockIdx.x * blockDim.x + threadIdx.x;
  const int p = blockIdx.y;
  if (q >= k) return;
  const int op = perm[p], oq = perm[q];
  float h = H[(size_t)op + (size_t)oq * k];
  if (p == q) {
    if (key_hi[op] == 0 && key_lo[op] == 0) h = 1.f;
    h += *dampadd;
  }
  Hp[(size_t)p * k + q] = h;
  Hr[(size_t)(k - 1 - p) * kp + (k - 1 - q)] = h;
  Gp[(size_t)p * k + q] = G[(size_t)op + (size_t)oq * k];
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
  cublasHandle_t blas;
  cusolverDnHandle_t solver;
  cusolverDnParams_t params;
  uint16_t *Xh, *dX;
  float *H, *G, *Hp, *Hr, *L, *Gp, *Q, *U, *D;
  float *a_orig, *a, *b, *c, *col, *dampadd;
  uint64_t *key_hi, *key_lo;
  int* perm;
  int* info;   // factorisation status
  void* dwork;
  size_t dwork_bytes;
  void* hwork;
  size_t hwork_bytes;
  void* allocs[32];
  int nalloc;
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

int map_blas(cublasStatus_t s) { return s == CUBLAS_STATUS_SUCCESS ? DUO_OK : DUO_ECUDA; }
int map_solver(cusolverStatus_t s) { return s == CUSOLVER_STATUS_SUCCESS ? DUO_OK : DUO_ECUDA; }

void release(duo_calib* h) {
  if (h->blas) cublasDestroy(h->blas);
  if (h->params) cusolverDnDestroyParams(h->params);
  if (h->solver) cusolverDnDestroy(h->solver);
  for (int i = 0; i < h->nalloc; ++i) cudaFree(h->allocs[i]);
  if (h->hwork) std::free(h->hwork);
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
  if (cublasCreate(&h->blas) != CUBLAS_STATUS_SUCCESS) return fail(DUO_ECUDA);
  if (cusolverDnCreate(&h->solver) != CUSOLVER_STATUS_SUCCESS) return fail(DUO_ECUDA);
  if (cusolverDnCreateParams(&h->params) != CUSOLVER_STATUS_SUCCESS) return fail(DUO_ECUDA);
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
  if (e == cudaSuccess) e = alloc(h, &h->info, 2);
  if (e != cudaSuccess) return fail(map_cuda(e));
  // cuSOLVER workspace of the factorisation.
  size_t d1 = 0, h1 = 0;
  cusolverDnSetStream(h->solver, st);
  if (cusolverDnXpotrf_bufferSize(h->solver, h->params, CUBLAS_FILL_MODE_LOWER, k, CUDA_R_32F, h->Hr,
                                  h->kp, CUDA_R_32F, &d1, &h1) != CUSOLVER_STATUS_SUCCESS)
    return fail(DUO_ECUDA);
  h->dwork_bytes = d1;
  h->hwork_bytes = h1;
  uint8_t* dw = nullptr;
  e = alloc(h, &dw, h->dwork_bytes);
  if (e != cudaSuccess) return fail(map_cuda(e));
  h->dwork = dw;
  if (h->hwork_bytes > 0) {
    h->hwork = std::malloc(h->hwork_bytes);
    if (h->hwork == nullptr) return fail(DUO_ENOMEM);
  }
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
  // 1. X_hat and dX, one token per CTA
  const size_t tsm = tok_xs_bytes(k) + sizeof(duo::SelShared);
  cudaError_t e = cudaFuncSetAttribute(token_sparsify_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)tsm);
  if (e != cudaSuccess) return map_cuda(e);
  token_sparsify_kernel<<<m, TOK_THREADS, tsm, st>>>(X, k, (int)keep, h->Xh, h->dX);
  // 2. exact Hessian diagonal, a, act_order, dampening
  channel_stats_kernel<<<(k + 31) / 32, 32 * STAT_STRIDES, 0, st>>>(h->Xh, h->dX, k, m, h->key_hi,
                                                                    h->key_lo, h->a_orig);
  rank_kernel<<<(k + RANK_THREADS - 1) / RANK_THREADS, RANK_THREADS, 0, st>>>(h->key_hi, h->key_lo, k,
                                                                              act_order ? 1 : 0, h->perm);
  damp_kernel<<<1, 256, 0, st>>>(h->key_hi, h->key_lo, k, damp, h->dampadd);
  e = cudaGetLastError();
  if (e != cudaSuccess) return map_cuda(e);
  // 3. H = X_hat X_hat^T and G = dX X_hat^T (fp16 in, fp32 accumulate):
  //    the token-major buffers are column-major k x m matrices.
  if (cublasSetStream(h->blas, st) != CUBLAS_STATUS_SUCCESS) return DUO_ECUDA;
  const float one = 1.f, zero = 0.f;
  int rc = map_blas(cublasGemmEx(h->blas, CUBLAS_OP_N, CUBLAS_OP_T, k, k, m, &one, h->Xh, CUDA_R_16F, k,
                                 h->Xh, CUDA_R_16F, k, &zero, h->H, CUDA_R_32F, k, CUBLAS_COMPUTE_32F,
                                 CUBLAS_GEMM_DEFAULT));
  if (rc != DUO_OK) return rc;
  rc = map_blas(cublasGemmEx(h->blas, CUBLAS_OP_N, CUBLAS_OP_T, k, k, m, &one, h->dX, CUDA_R_16F, k, h->Xh,
                             CUDA_R_16F, k, &zero, h->G, CUDA_R_32F, k, CUBLAS_COMPUTE_32F,
                             CUBLAS_GEMM_DEFAULT));
  if (rc != DUO_OK) return rc;
  // 4. reorder and dampen, then L
  const dim3 g2((k + 255) / 256, k);
  const int kp = (int)h->kp;
  gather_kernel<<<g2, 256, 0, st>>>(h->H, h->G, h->perm, h->key_hi, h->key_lo, k, kp, h->dampadd, h->Hp,
                                    h->Hr, h->Gp);
  e = cudaGetLastError();
  if (e != cudaSuccess) return map_cuda(e);
  if (cusolverDnSetStream(h->solver, st) != CUSOLVER_STATUS_SUCCESS) return DUO_ECUDA;
  rc = map_solver(cusolverDnXpotrf(h->solver, h->params, CUBLAS_FILL_MODE_LOWER, k, CUDA_R_32F, h->Hr, kp,
                                   CUDA_R_32F, h->dwork, h->dwork_bytes, h->hwork, h->hwork_bytes, h->info));
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
    const float minus_one = -1.f;
    for (int sz = TRI_BASE; sz < kp; sz *= 2) {
      const int batch = kp / (2 * sz);
      const long long stride = 2LL * sz * ((long long)kp + 1);
      float* A = h->Hr;
      float* B = h->Hr + sz;
      float* Dg = h->Hr + sz + (size_t)sz * kp;
      rc = map_blas(cublasGemmStridedBatchedEx(h->blas, CUBLAS_OP_N, CUBLAS_OP_N, sz, sz, sz, &one, B,
                                               CUDA_R_32F, kp, stride, A, CUDA_R_32F, kp, stride, &zero,
                                               h->H, CUDA_R_32F, sz, (long long)sz * sz, batch, kL_COMPUTE,
                                               CUBLAS_GEMM_DEFAULT));
      if (rc != DUO_OK) return rc;
      rc = map_blas(cublasGemmStridedBatchedEx(h->blas, CUBLAS_OP_N, CUBLAS_OP_N, sz, sz, sz, &minus_one,
                                               Dg, CUDA_R_32F, kp, stride, h->H, CUDA_R_32F, sz,
                                               (long long)sz * sz, &zero, B, CUDA_R_32F, kp, stride, batch,
                                               kL_COMPUTE, CUBLAS_GEMM_DEFAULT));
      if (rc != DUO_OK) return rc;
    }
  }
  l_from_cinv_kernel<<<g2, 256, 0, st>>>(h->Hr, k, kp, h->L);
  e = cudaGetLastError();
  if (e != cudaSuccess) return map_cuda(e);
  // 5. Q = Gp L.  Row-major buffers are the column-major transposes, so
  //    Q^T = L^T Gp^T is a plain product of the two buffers.
  rc = map_blas(cublasGemmEx(h->blas, CUBLAS_OP_N, CUBLAS_OP_N, k, k, k, &one, h->L, CUDA_R_32F, k, h->Gp,
                             CUDA_R_32F, k, &zero, h->Q, CUDA_R_32F, k, kL_COMPUTE,
                             CUBLAS_GEMM_DEFAULT));
  if (rc != DUO_OK) return rc;
  // 6. U, a (reordered), b, c and the score's column factor
  q_epilogue_kernel<<<k, EPI_THREADS, 0, st>>>(h->Q, h->L, h->a_orig, h->perm, k, h->U, h->a, h->b, h->c,
                                               h->col);
  e = cudaGetLastError();
  if (e != cudaSuccess) return map_cuda(e);
  // 7. D = U L^T: D^T = L U^T, i.e. op(L buffer) = L and the U buffer as is.
  rc = map_blas(cublasGemmEx(h->blas, CUBLAS_OP_T, CUBLAS_OP_N, k, k, k, &one, h->L, CUDA_R_32F, k, h->U,
                             CUDA_R_32F, k, &zero, h->D, CUDA_R_32F, k, kL_COMPUTE,
                             CUBLAS_GEMM_DEFAULT));
  return rc;
}

int duo_calib_status(const duo_calib* h, void* stream) {
  if (h == nullptr || !calib_live(h)) return DUO_EINVAL;
  cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return DUO_ECUDA;
  int info[2] = {0, 0};
  e = cudaMemcpy(info, h->info, sizeof(info), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return DUO_ECUDA;
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
