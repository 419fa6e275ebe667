// Dense GEMM on the 5th-generation tensor cores (tcgen05); interface and
// arithmetic in tcgemm.h.  It carries the calibration's contractions
// (Algorithm 1, §4.3): the Hessian products, the blocked Cholesky
// factorisation, the triangular inverse, Q = G L, D = U L^T and the column
// sweep's lazy batch update.
//
// tc_prep writes an operand as the image the MMAs read: for every 128-row
// tile and 64-column chunk, its P pieces (fp16: the values; fp32: three bf16
// pieces) one after the other, each 16 KB in the canonical K-major
// no-swizzle layout (core matrices of 8 rows x 16 bytes; neighbours along K
// 128 bytes apart, along rows 8 x 128 bytes apart).  One chunk of one
// operand is then a single contiguous block of P x 16 KB that a bulk copy
// (cp.async.bulk) moves into shared memory unchanged.
//
// tc_gemm_kernel: persistent, one CTA per SM (or fewer), 128 x 128 output
// tiles handed out round-robin.  Lane 0 of warp 0 streams the chunks of A
// and B through an S-stage ring of shared-memory buffers (full / empty
// mbarriers, the copies completing transaction bytes on `full`); lane 0 of
// warp 1 issues each chunk's MMAs (K = 16 each, 6 products per step for
// fp32) into one of two TMEM accumulators and commits the stage to `empty`
// and the finished tile to `acc_full`; warps 2..5 read the accumulator with
// tcgen05.ld, write C and release it on `acc_empty`, so a tile's epilogue
// runs under the next tile's MMAs.  Every wait is bounded by a wall-clock
// limit; a CTA that gives up still waits (bounded) for its copies in flight
// and frees its TMEM.
#include <cstdint>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include "tcgemm.h"

namespace duo {
namespace {

constexpr int TG_M = 128, TG_N = 128, TG_K = 64;
constexpr int TG_CTA_THREADS = 192;                // producer, MMA and four epilogue warps
constexpr int TG_TILE = TG_M * TG_K * 2;            // bytes of one 128 x 64 16-bit tile
constexpr int PREP_THREADS = 256;
constexpr uint64_t TG_WAIT_NS = 1000000000ull;      // 1 s per bounded wait

__device__ unsigned int g_tg_status = 0u;           // bit 0: a wait ran out

__device__ __forceinline__ uint32_t su32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ uint64_t now_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ uint64_t smem_desc(uint32_t saddr) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);           // start address >> 4
  d |= (uint64_t)(128u >> 4) << 16;                    // leading byte offset: next core matrix along K
  d |= (uint64_t)((8u * 128u) >> 4) << 32;             // stride byte offset: next 8 rows
  d |= (uint64_t)1 << 46;                              // fixed 0b001; no swizzle
  return d;
}

// kind::f16 instruction descriptor: fp32 D, A and B of type t (0 fp16,
// 1 bf16), both K-major, N = 128, M = 128.
__host__ __device__ constexpr uint32_t idesc_f16(uint32_t t) {
  return (1u << 4) | (t << 7) | (t << 10) | ((uint32_t)(TG_N >> 3) << 17) | ((uint32_t)(TG_M >> 4) << 24);
}

__device__ __forceinline__ void mma(uint32_t d, uint64_t a, uint64_t b, uint32_t idesc, uint32_t acc) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d),
      "l"(a), "l"(b), "r"(idesc), "r"(acc)
      : "memory");
}

__device__ __forceinline__ void commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(su32(bar))
               : "memory");
}

__device__ __forceinline__ void bar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(su32(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(su32(bar)), "r"(bytes) : "memory");
}

// bytes (a multiple of 16) from global src to shared dst, both 16-byte
// aligned, completing on bar
__device__ __forceinline__ void bulk_copy(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(su32(dst)),
      "l"(src), "r"(bytes), "r"(su32(bar))
      : "memory");
}

__device__ __forceinline__ bool try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(su32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

__device__ __forceinline__ bool bar_wait(uint64_t* bar, uint32_t parity) {
  if (try_wait(bar, parity)) return true;
  const uint64_t t0 = now_ns();
  while (!try_wait(bar, parity)) {
    if (now_ns() - t0 > TG_WAIT_NS) {
      atomicOr(&g_tg_status, 1u);
      return false;
    }
  }
  return true;
}

// bf16 pieces of two fp32 values, x = x0 + x1 + x2 to 24 bits: each residual
// x - x0 (and x - x0 - x1) is exact in fp32, a multiple of the value's last
// place below 2^16 of them.  Piece p of (a, b) packed in one 32-bit word.
template <int P>
__device__ __forceinline__ void split2(float a, float b, uint32_t (&w)[P]) {
#pragma unroll
  for (int p = 0; p < P; ++p) {
    const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
    w[p] = *reinterpret_cast<const uint32_t*>(&h);
    if (p + 1 < P) {
      a -= __low2float(h);
      b -= __high2float(h);
    }
  }
}

// One 16-byte unit per thread: row r, columns k .. k + 7 of batch entry z.
// A warp covers 8 rows x 4 column groups, so its loads read 8 row segments
// of 4 groups and its stores fill 4 whole core matrices.
template <typename T, int P>
__global__ void __launch_bounds__(PREP_THREADS) tc_prep_kernel(const T* __restrict__ X, int64_t rows, int64_t K,
                                                               int64_t s_r, int64_t s_k, int64_t s_b, int64_t nrt,
                                                               int64_t nkc, int vec, uint8_t* __restrict__ dst) {
  const int64_t u = (int64_t)blockIdx.x * PREP_THREADS + threadIdx.x;
  const int lane = threadIdx.x & 31;
  const int64_t w = u >> 5;
  const int64_t nq = 2 * nkc;                     // quads of column groups per 8 rows
  const int64_t quad = w % nq, w2 = w / nq;
  const int64_t ro = w2 % (nrt * 16), z = w2 / (nrt * 16);
  const int64_t r = ro * 8 + (lane & 7);
  const int64_t k = (quad * 4 + (lane >> 3)) * 8;
  const int64_t blk = ((z * nrt + (r >> 7)) * nkc + (k >> 6)) * P;
  uint8_t* out = dst + blk * TG_TILE + ((((r & 127) >> 3) * 8 + ((k & 63) >> 3)) << 7) + ((r & 7) << 4);
  const T* row = X + z * s_b + (r < rows ? r : 0) * s_r;
  if constexpr (sizeof(T) == 4) {
    float v[8];
    if (vec && r < rows && k + 8 <= K) {
      const float4 a = __ldg(reinterpret_cast<const float4*>(row + k));
      const float4 b = __ldg(reinterpret_cast<const float4*>(row + k) + 1);
      v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
      v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
    } else {
#pragma unroll
      for (int j = 0; j < 8; ++j) v[j] = (r < rows && k + j < K) ? __ldg(row + (k + j) * s_k) : 0.f;
    }
    uint32_t wd[4][P];
#pragma unroll
    for (int q = 0; q < 4; ++q) split2<P>(v[2 * q], v[2 * q + 1], wd[q]);
#pragma unroll
    for (int p = 0; p < P; ++p)
      *reinterpret_cast<uint4*>(out + p * TG_TILE) = make_uint4(wd[0][p], wd[1][p], wd[2][p], wd[3][p]);
  } else {
    uint4 q;
    if (vec && r < rows && k + 8 <= K) {
      q = __ldg(reinterpret_cast<const uint4*>(row + k));
    } else {
      const uint16_t* rb = reinterpret_cast<const uint16_t*>(row);
      uint32_t h[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) h[j] = (r < rows && k + j < K) ? __ldg(rb + (k + j) * s_k) : 0u;
      q = make_uint4(h[0] | (h[1] << 16), h[2] | (h[3] << 16), h[4] | (h[5] << 16), h[6] | (h[7] << 16));
    }
    *reinterpret_cast<uint4*>(out) = q;
  }
}

// Output tile t of the product (nt fastest, so that consecutive tiles share
// their A rows): batch entry z, row tile mt, column tile nt; with `lower`
// only tiles nt <= mt are enumerated.
__device__ __forceinline__ void tile_of(int64_t t, int MT, int NT, int lower, int& z, int& mt, int& nt) {
  if (!lower) {
    const int64_t per = (int64_t)MT * NT, r = t % per;
    z = (int)(t / per);
    mt = (int)(r / NT);
    nt = (int)(r % NT);
  } else {
    const int64_t per = (int64_t)MT * (MT + 1) / 2, r = t % per;
    z = (int)(t / per);
    int m = (int)((sqrtf(8.f * (float)r + 1.f) - 1.f) * 0.5f);
    while ((int64_t)m * (m + 1) / 2 > r) --m;
    while ((int64_t)(m + 1) * (m + 2) / 2 <= r) ++m;
    mt = m;
    nt = (int)(r - (int64_t)m * (m + 1) / 2);
  }
}

// Persistent, warp-specialised: each CTA walks the tiles t = blockIdx.x,
// blockIdx.x + gridDim.x, ...  Warp 0 (lane 0) streams every tile's chunks
// through the S-stage ring; warp 1 (lane 0) issues the MMAs into one of two
// TMEM accumulators (128 columns each) and commits the accumulator to
// acc_full; warps 2..5 drain an accumulator (warp w reads TMEM lanes
// 32 (w % 4) ..) into C and release it on acc_empty, so a tile's epilogue
// overlaps the next tile's MMAs.
template <int P>
__global__ void __launch_bounds__(TG_CTA_THREADS, 1) tc_gemm_kernel(const TcGemm g) {
  constexpr int NPROD = P == 1 ? 1 : 6;
  constexpr int S = P == 1 ? 4 : 2;                    // ring stages
  constexpr uint32_t OPB = P * TG_TILE;                // one operand's chunk
  constexpr uint32_t STB = 2 * OPB;                    // one stage: A chunk, then B chunk
  extern __shared__ __align__(1024) uint8_t sm[];
  __shared__ __align__(8) uint64_t full[S], empty[S], acc_full[2], acc_empty[2], mma_done;
  __shared__ uint32_t tmem_base;
  __shared__ int fail_flag;
  volatile int& fail = fail_flag;                      // set by any role that gives up
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int nkc = (g.K + TG_K - 1) / TG_K;
  const int MT = (g.M + TG_M - 1) / TG_M, NT = (g.N + TG_N - 1) / TG_N;
  const int64_t ntiles = (int64_t)g.batch * (g.lower ? (int64_t)MT * (MT + 1) / 2 : (int64_t)MT * NT);

  if (tid == 0) {
    for (int s = 0; s < S; ++s) {
      bar_init(&full[s], 1);
      bar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      bar_init(&acc_full[a], 1);
      bar_init(&acc_empty[a], 4);                      // one arrival per epilogue warp
    }
    bar_init(&mma_done, 1);
    fail = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], 256;" ::"r"(su32(&tmem_base))
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = tmem_base;

  if (warp == 0) {
    if (lane == 0) {   // producer
      int64_t q = 0, issued = 0;                       // chunks over all of this CTA's tiles
      for (int64_t t = blockIdx.x; t < ntiles && !fail; t += gridDim.x) {
        int z, mt, nt;
        tile_of(t, MT, NT, g.lower, z, mt, nt);
        const uint8_t* Ach = static_cast<const uint8_t*>(g.A) + ((int64_t)z * MT + mt) * nkc * (int64_t)OPB;
        const uint8_t* Bch = static_cast<const uint8_t*>(g.B) + ((int64_t)z * NT + nt) * nkc * (int64_t)OPB;
        for (int c = 0; c < nkc; ++c, ++q) {
          const int s = (int)(q % S);
          const int64_t round = q / S;
          if (round > 0 && !bar_wait(&empty[s], (uint32_t)((round - 1) & 1))) {
            fail = 1;
            break;
          }
          expect_tx(&full[s], STB);
          bulk_copy(sm + s * STB, Ach + (int64_t)c * OPB, OPB, &full[s]);
          bulk_copy(sm + s * STB + OPB, Bch + (int64_t)c * OPB, OPB, &full[s]);
          issued = q + 1;
        }
      }
      // every issued copy has landed before the CTA may exit
      for (int64_t c = issued > S ? issued - S : 0; c < issued; ++c)
        if (!bar_wait(&full[c % S], (uint32_t)((c / S) & 1))) fail = 1;
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {   // MMA issuer
      constexpr int PA[6] = {0, 0, 1, 0, 1, 2};         // (A piece, B piece) of each product
      constexpr int PB[6] = {0, 1, 0, 2, 1, 0};
      constexpr uint32_t ID = idesc_f16(P == 1 ? 0u : 1u);
      int64_t q = 0, u = 0;
      for (int64_t t = blockIdx.x; t < ntiles && !fail; t += gridDim.x, ++u) {
        const int ab = (int)(u & 1);
        const int64_t use = u >> 1;
        if (use > 0 && !bar_wait(&acc_empty[ab], (uint32_t)((use - 1) & 1))) {
          fail = 1;
          break;
        }
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        const uint32_t d = tmem + (uint32_t)(ab * TG_N);
        bool ok = true;
        for (int c = 0; c < nkc; ++c, ++q) {
          const int s = (int)(q % S);
          if (!bar_wait(&full[s], (uint32_t)((q / S) & 1))) {
            ok = false;
            break;
          }
          asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
          const uint32_t a0 = su32(sm + s * STB), b0 = a0 + OPB;
#pragma unroll
          for (int ks = 0; ks < TG_K / 16; ++ks) {
#pragma unroll
            for (int pr = 0; pr < NPROD; ++pr) {
              const uint32_t off = (uint32_t)ks * 256u;   // 16 columns = two core matrices along K
              const uint32_t acc = (c > 0 || ks > 0 || pr > 0) ? 1u : 0u;
              mma(d, smem_desc(a0 + PA[pr] * TG_TILE + off), smem_desc(b0 + PB[pr] * TG_TILE + off), ID, acc);
            }
          }
          commit(&empty[s]);
        }
        if (!ok) {
          fail = 1;
          break;
        }
        commit(&acc_full[ab]);   // arrives once this tile's MMAs have completed
      }
      // no MMA may still be writing TMEM when it is freed
      commit(&mma_done);
      if (!bar_wait(&mma_done, 0u)) fail = 1;
    }
    __syncwarp();
  } else {   // epilogue: warps 2..5
    const int quarter = warp & 3;                      // TMEM lanes 32 quarter .. 32 quarter + 31
    int64_t u = 0;
    for (int64_t t = blockIdx.x; t < ntiles; t += gridDim.x, ++u) {
      const int ab = (int)(u & 1);
      const bool got = bar_wait(&acc_full[ab], (uint32_t)((u >> 1) & 1));
      if (!__all_sync(0xffffffffu, got) || fail) {
        fail = 1;
        break;
      }
      asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      int z, mt, nt;
      tile_of(t, MT, NT, g.lower, z, mt, nt);
      const int r = mt * TG_M + 32 * quarter + lane;
      const int n0 = nt * TG_N;
      float* C = g.C + (int64_t)z * g.c_bs;
#pragma unroll 1
      for (int c16 = 0; c16 < TG_N; c16 += 16) {
        uint32_t v[16];
        const uint32_t addr = tmem + (uint32_t)(ab * TG_N) + ((uint32_t)(32 * quarter) << 16) + (uint32_t)c16;
        asm volatile(
            "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, "
            "[%16];"
            : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]),
              "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]),
              "=r"(v[15])
            : "r"(addr));
        asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
        if (r < g.M) {
          float* cr = C + (int64_t)r * g.c_m + (int64_t)(n0 + c16) * g.c_n;
          float old[16];
          // all 16 reads of C before any write: the stores may alias as far
          // as the compiler knows, which would serialise each read behind
          // the previous write
#pragma unroll
          for (int j = 0; j < 16; ++j)
            old[j] = (g.beta != 0.f && n0 + c16 + j < g.N) ? cr[(int64_t)j * g.c_n] : 0.f;
#pragma unroll
          for (int j = 0; j < 16; ++j)
            if (n0 + c16 + j < g.N) cr[(int64_t)j * g.c_n] = fmaf(g.beta, old[j], g.alpha * __uint_as_float(v[j]));
        }
      }
      // this warp's reads of the accumulator are done: release it
      asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
      __syncwarp();
      if (lane == 0) asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(su32(&acc_empty[ab])) : "memory");
    }
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  if (warp == 0)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, 256;" ::"r"(tmem) : "memory");
}

int pieces(int dtype) { return dtype == TC_F16 ? 1 : 3; }

}  // namespace

size_t tc_operand_bytes(int dtype, int64_t rows, int64_t K, int64_t batch) {
  const int64_t nrt = (rows + TG_M - 1) / TG_M, nkc = (K + TG_K - 1) / TG_K;
  return (size_t)(batch * nrt * nkc * pieces(dtype)) * TG_TILE;
}

cudaError_t tc_prep(int dtype, const void* X, int64_t rows, int64_t K, int64_t batch, int64_t s_r, int64_t s_k,
                    int64_t s_b, void* dst, cudaStream_t st) {
  if (rows <= 0 || K <= 0 || batch <= 0) return cudaSuccess;
  if (X == nullptr || dst == nullptr || (reinterpret_cast<uintptr_t>(dst) & 15u) != 0 ||
      (dtype != TC_F16 && dtype != TC_F32))
    return cudaErrorInvalidValue;
  const int64_t nrt = (rows + TG_M - 1) / TG_M, nkc = (K + TG_K - 1) / TG_K;
  const int64_t blocks = batch * nrt * nkc * (TG_M * TG_K / 8) / PREP_THREADS;
  if (blocks > 0x7FFFFFFF) return cudaErrorInvalidValue;
  const int esz = dtype == TC_F16 ? 2 : 4, per16 = 16 / esz;
  const int vec = s_k == 1 && (reinterpret_cast<uintptr_t>(X) & 15u) == 0 && s_r % per16 == 0 &&
                  s_b % per16 == 0;
  uint8_t* d = static_cast<uint8_t*>(dst);
  if (dtype == TC_F16)
    tc_prep_kernel<__half, 1><<<(unsigned)blocks, PREP_THREADS, 0, st>>>(static_cast<const __half*>(X), rows, K,
                                                                        s_r, s_k, s_b, nrt, nkc, vec, d);
  else
    tc_prep_kernel<float, 3><<<(unsigned)blocks, PREP_THREADS, 0, st>>>(static_cast<const float*>(X), rows, K,
                                                                       s_r, s_k, s_b, nrt, nkc, vec, d);
  return cudaGetLastError();
}

cudaError_t launch_tc_gemm(const TcGemm& g, cudaStream_t st) {
  if (g.M <= 0 || g.N <= 0 || g.batch <= 0) return cudaSuccess;
  if (g.K <= 0 || g.batch > 65535 || (g.lower && g.M != g.N)) return cudaErrorInvalidValue;
  if (g.A == nullptr || g.B == nullptr || g.C == nullptr || (reinterpret_cast<uintptr_t>(g.A) & 15u) != 0 ||
      (reinterpret_cast<uintptr_t>(g.B) & 15u) != 0)
    return cudaErrorInvalidValue;
  const int64_t MT = (g.M + TG_M - 1) / TG_M, NT = (g.N + TG_N - 1) / TG_N;
  const int64_t ntiles = (int64_t)g.batch * (g.lower ? MT * (MT + 1) / 2 : MT * NT);
  int dev = 0, sms = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return e;
  int64_t ctas = sms;
  if (g.max_ctas > 0 && g.max_ctas < sms) ctas = g.max_ctas;
  if (g.max_ctas < 0 && sms + g.max_ctas >= 1) ctas = sms + g.max_ctas;
  if (ctas > ntiles) ctas = ntiles;
  if (g.dtype == TC_F16) {
    constexpr int smem = 4 * 2 * TG_TILE;
    e = cudaFuncSetAttribute(tc_gemm_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    tc_gemm_kernel<1><<<(unsigned)ctas, TG_CTA_THREADS, smem, st>>>(g);
  } else if (g.dtype == TC_F32) {
    constexpr int smem = 2 * 2 * 3 * TG_TILE;
    e = cudaFuncSetAttribute(tc_gemm_kernel<3>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    tc_gemm_kernel<3><<<(unsigned)ctas, TG_CTA_THREADS, smem, st>>>(g);
  } else {
    return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

cudaError_t tc_gemm_take_status(unsigned int* out) {
  unsigned int v = 0, zero = 0;
  cudaError_t e = cudaMemcpyFromSymbol(&v, g_tg_status, sizeof(v));
  if (e == cudaSuccess) e = cudaMemcpyToSymbol(g_tg_status, &zero, sizeof(zero));
  *out = v;
  return e;
}

}  // namespace duo

// ---------------------------------------------------------------------------
// Internal, for the GEMM's own parity tests (not declared in the public
// headers): prepares A and B (strided, fp16 when dtype == 0, fp32 when 1)
// into temporary buffers, runs the product into C and synchronises.
// Returns 0, -1 (invalid arguments), -4 (CUDA error) or -6 (a bounded wait
// ran out), the codes of include/duo.h.
// ---------------------------------------------------------------------------
extern "C" int duo_test_tc_gemm(int dtype, int M, int N, int K, int batch, const void* A, int64_t a_m, int64_t a_k,
                                int64_t a_bs, const void* B, int64_t b_n, int64_t b_k, int64_t b_bs, float* C,
                                int64_t c_m, int64_t c_n, int64_t c_bs, float alpha, float beta, int lower,
                                int max_ctas, void* stream) {
  using namespace duo;
  if ((dtype != TC_F16 && dtype != TC_F32) || M < 1 || N < 1 || K < 1 || batch < 1 || A == nullptr ||
      B == nullptr || C == nullptr || (lower && M != N))
    return -1;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  void *pa = nullptr, *pb = nullptr;
  cudaError_t e = cudaMalloc(&pa, tc_operand_bytes(dtype, M, K, batch));
  if (e == cudaSuccess) e = cudaMalloc(&pb, tc_operand_bytes(dtype, N, K, batch));
  if (e == cudaSuccess) e = tc_prep(dtype, A, M, K, batch, a_m, a_k, a_bs, pa, st);
  if (e == cudaSuccess) e = tc_prep(dtype, B, N, K, batch, b_n, b_k, b_bs, pb, st);
  TcGemm g;
  g.dtype = dtype;
  g.M = M;
  g.N = N;
  g.K = K;
  g.batch = batch;
  g.A = pa;
  g.B = pb;
  g.C = C;
  g.c_m = c_m;
  g.c_n = c_n;
  g.c_bs = c_bs;
  g.alpha = alpha;
  g.beta = beta;
  g.lower = lower;
  g.max_ctas = max_ctas;
  if (e == cudaSuccess) e = launch_tc_gemm(g, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  cudaFree(pa);
  cudaFree(pb);
  if (e != cudaSuccess) return -4;
  unsigned int v = 0;
  if (tc_gemm_take_status(&v) != cudaSuccess) return -4;
  return v != 0 ? -6 : 0;
}
