// Device helpers shared by the kernels of libduo: mbarrier / bulk-copy
// wrappers (inline PTX for sm_103a), bounded waits, block scans and the
// exact top-k magnitude selection of §3 ("Activation Sparsity").
#pragma once

#include <cstdint>
#include <cuda_fp16.h>

namespace duo {

constexpr uint32_t FULL_MASK = 0xFFFFFFFFu;
constexpr int SEG_ROWS = 1024;           // rows per CMB segment
constexpr int SEG_WORDS = SEG_ROWS / 32; // mask words per record
constexpr int MASK_BYTES = SEG_ROWS / 8; // 128
constexpr int MAX_RECORD_BYTES = MASK_BYTES + 2 * SEG_ROWS;  // 2176
constexpr int MAXP = 4;                  // products per multi launch
constexpr uint64_t WAIT_LIMIT_NS = 1000000000ull;  // 1 s per bounded wait

// Device status word (bit 0: a bounded wait ran out; bit 1: a record size or
// channel id outside the format's bounds).  Defined here because this header
// is included by exactly one translation unit (kernels.cu).
__device__ unsigned int g_status = 0u;
constexpr unsigned int STATUS_TIMEOUT = 1u;
constexpr unsigned int STATUS_FORMAT = 2u;

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.release.cta.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.release.cta.shared::cta.b64 _, [%0], %1;"
               ::"r"(smem_u32(bar)), "r"(bytes) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cta.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Waits for the phase of `parity` with a wall-clock limit.  On timeout the
// device status word and the CTA's abort flag are set and false returned;
// a wait also gives up (false) once another warp has raised the abort flag.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t* bar, uint32_t parity,
                                                  volatile int* abort_flag) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  while (true) {
    if (mbar_try_wait(bar, parity)) return true;
    if (*abort_flag) return false;
    if (globaltimer_ns() - t0 > WAIT_LIMIT_NS) {
      atomicOr(&g_status, STATUS_TIMEOUT);
      *abort_flag = 1;
      return false;
    }
  }
}

// Same, without an abort flag (used while draining after an abort).
__device__ __forceinline__ bool mbar_wait_limited(uint64_t* bar, uint32_t parity) {
  const uint64_t t0 = globaltimer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (globaltimer_ns() - t0 > WAIT_LIMIT_NS) {
      atomicOr(&g_status, STATUS_TIMEOUT);
      return false;
    }
  }
  return true;
}

// 1-D bulk copy global -> shared (the CTA is its own cluster), completing
// `bytes` transaction bytes on `bar`.  dst, src 16-byte aligned, bytes % 16 == 0.
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar,
                                         uint64_t policy) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint "
      "[%0], [%1], %2, [%3], %4;" ::"r"(smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar)), "l"(policy)
      : "memory");
}

__device__ __forceinline__ uint64_t policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}

__device__ __forceinline__ unsigned int ld_acquire_gpu(const unsigned int* p) {
  unsigned int v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void named_bar_sync(int id, int nthreads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}

// acc + w * x with w, x fp16 (exact product) and one fp32 rounding.
__device__ __forceinline__ float fma_f16_f32(uint16_t w, uint16_t x, float acc) {
  asm("{\n\t.reg .f16 a, b;\n\tmov.b16 a, %1;\n\tmov.b16 b, %2;\n\t"
      "fma.rn.f32.f16 %0, a, b, %0;\n\t}"
      : "+f"(acc)
      : "h"(w), "h"(x));
  return acc;
}

__device__ __forceinline__ void red_add_v4(float* p, float a, float b, float c, float d) {
  asm volatile("red.global.add.v4.f32 [%0], {%1, %2, %3, %4};" ::"l"(p), "f"(a), "f"(b), "f"(c),
               "f"(d)
               : "memory");
}

__device__ __forceinline__ uint32_t warp_inclusive_scan(uint32_t v, int lane) {
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t t = __shfl_up_sync(FULL_MASK, v, o);
    if (lane >= o) v += t;
  }
  return v;
}

// In-place exclusive scan of a[0..n) in shared memory by the whole block;
// returns the total.  wsum needs 32 entries.  Contains __syncthreads.
__device__ inline uint32_t block_exclusive_scan(uint32_t* a, int n, uint32_t* wsum) {
  const int tid = threadIdx.x, nt = blockDim.x, lane = tid & 31, wid = tid >> 5;
  const int nwarps = nt >> 5;
  const int per = (n + nt - 1) / nt;
  const int beg = min(n, tid * per), end = min(n, beg + per);
  uint32_t s = 0;
  for (int i = beg; i < end; ++i) s += a[i];
  const uint32_t inc = warp_inclusive_scan(s, lane);
  if (lane == 31) wsum[wid] = inc;
  __syncthreads();
  if (wid == 0) {
    uint32_t w = lane < nwarps ? wsum[lane] : 0u;
    w = warp_inclusive_scan(w, lane);
    wsum[lane] = w;
  }
  __syncthreads();
  uint32_t base = (wid > 0 ? wsum[wid - 1] : 0u) + inc - s;
  for (int i = beg; i < end; ++i) {
    const uint32_t v = a[i];
    a[i] = base;
    base += v;
  }
  const uint32_t total = wsum[nwarps - 1];
  __syncthreads();
  return total;
}

// Position of the r-th (0-based) set bit of m; requires r < popc(m).
__device__ __forceinline__ int select_bit(uint32_t m, int r) {
  int pos = 0, c;
  c = __popc(m & 0xFFFFu); if (r >= c) { r -= c; m >>= 16; pos += 16; }
  c = __popc(m & 0xFFu);   if (r >= c) { r -= c; m >>= 8;  pos += 8; }
  c = __popc(m & 0xFu);    if (r >= c) { r -= c; m >>= 4;  pos += 4; }
  c = __popc(m & 0x3u);    if (r >= c) { r -= c; m >>= 2;  pos += 2; }
  c = m & 1u;              if (r >= c) { pos += 1; }
  return pos;
}

// Block-cooperative copy of x (fp16 bits) into shared memory.
__device__ inline void load_x_to_smem(uint16_t* xs, const uint16_t* x, int I) {
  const int tid = threadIdx.x, nt = blockDim.x;
  if ((reinterpret_cast<uintptr_t>(x) & 15u) == 0) {
    const int nvec = I >> 3;
    const uint4* xv = reinterpret_cast<const uint4*>(x);
    uint4* sv = reinterpret_cast<uint4*>(xs);
    for (int i = tid; i < nvec; i += nt) sv[i] = __ldg(xv + i);
    for (int i = (nvec << 3) + tid; i < I; i += nt) xs[i] = x[i];
  } else {
    for (int i = tid; i < I; i += nt) xs[i] = x[i];
  }
}

struct SelShared {
  uint32_t hist[256];
  uint32_t wsum[32];
  int b1;
  uint32_t above1;
  uint32_t T;
  int q;
};

// Exact top-k by magnitude (§3): keeps the k channels with the largest
// |x_j|, ties to the lower index.  The key of x_j is its fp16 bit pattern
// with the sign cleared; for IEEE fp16 this integer order equals the order of
// |x_j| (NaN patterns sort above Inf).  Two radix passes (8 high key bits,
// then 7 low bits) find the threshold key T and the number q of channels
// with key == T to keep (the q lowest-indexed ones).
//
// Output, in shared memory, for nw = ceil(I/32) words:
//   kb[w]  kept-channel bitmap (bit b <-> channel 32w+b),
//   kp[w]  number of kept channels before word w, kp[nw] = k.
// eqw is nw words of scratch.  All threads of the block must call it.
__device__ inline void select_topk(const uint16_t* xs, int I, int k, uint32_t* kb, uint32_t* kp,
                                   uint32_t* eqw, SelShared* sh) {
  const int tid = threadIdx.x, nt = blockDim.x, lane = tid & 31, wid = tid >> 5;
  const int nwarps = nt >> 5;
  const int nw = (I + 31) >> 5;
  if (k <= 0 || k >= I) {
    for (int w = tid; w < nw; w += nt) {
      const int rem = I - 32 * w;
      const uint32_t full = rem >= 32 ? FULL_MASK : ((1u << rem) - 1u);
      kb[w] = k > 0 ? full : 0u;
    }
    __syncthreads();
  } else {
    for (int i = tid; i < 256; i += nt) sh->hist[i] = 0u;
    __syncthreads();
    for (int j = tid; j < I; j += nt) atomicAdd(&sh->hist[(xs[j] & 0x7FFFu) >> 7], 1u);
    __syncthreads();
    if (wid == 0) {
      uint32_t c[8], s = 0;
#pragma unroll
      for (int q = 0; q < 8; ++q) { c[q] = sh->hist[8 * lane + q]; s += c[q]; }
      uint32_t sfx = s;   // inclusive suffix sum over lanes >= lane
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t t = __shfl_down_sync(FULL_MASK, sfx, o);
        if (lane + o < 32) sfx += t;
      }
      const uint32_t above = sfx - s;
      if (above < (uint32_t)k && (uint32_t)k <= sfx) {
        uint32_t acc = above;
        int b = 8 * lane;
        for (int q = 7; q >= 0; --q) {
          if (acc + c[q] >= (uint32_t)k) { b = 8 * lane + q; break; }
          acc += c[q];
        }
        sh->b1 = b;
        sh->above1 = acc;
      }
    }
    __syncthreads();
    const uint32_t b1 = (uint32_t)sh->b1;
    const uint32_t above1 = sh->above1;
    for (int i = tid; i < 128; i += nt) sh->hist[i] = 0u;
    __syncthreads();
    for (int j = tid; j < I; j += nt) {
      const uint32_t key = xs[j] & 0x7FFFu;
      if ((key >> 7) == b1) atomicAdd(&sh->hist[key & 127u], 1u);
    }
    __syncthreads();
    if (wid == 0) {
      const uint32_t need = (uint32_t)k - above1;
      uint32_t c[4], s = 0;
#pragma unroll
      for (int q = 0; q < 4; ++q) { c[q] = sh->hist[4 * lane + q]; s += c[q]; }
      uint32_t sfx = s;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t t = __shfl_down_sync(FULL_MASK, sfx, o);
        if (lane + o < 32) sfx += t;
      }
      const uint32_t above = sfx - s;
      if (above < need && need <= sfx) {
        uint32_t acc = above;
        int b2 = 4 * lane;
        for (int q = 3; q >= 0; --q) {
          if (acc + c[q] >= need) { b2 = 4 * lane + q; break; }
          acc += c[q];
        }
        sh->T = b1 * 128u + (uint32_t)b2;
        sh->q = (int)(need - acc);
      }
    }
    __syncthreads();
    const uint32_t T = sh->T;
    const int q = sh->q;
    for (int w = wid; w < nw; w += nwarps) {
      const int j = 32 * w + lane;
      const bool valid = j < I;
      const uint32_t key = valid ? (xs[j] & 0x7FFFu) : 0u;
      const uint32_t gt = __ballot_sync(FULL_MASK, valid && key > T);
      const uint32_t eq = __ballot_sync(FULL_MASK, valid && key == T);
      if (lane == 0) { kb[w] = gt; eqw[w] = eq; kp[w] = __popc(eq); }
    }
    __syncthreads();
    block_exclusive_scan(kp, nw, sh->wsum);   // kp[w] = ties before word w
    for (int w = tid; w < nw; w += nt) {
      const int allowed = q - (int)kp[w];
      const uint32_t eq = eqw[w];
      if (allowed > 0 && eq != 0u) {
        uint32_t take = eq;
        if (allowed < __popc(eq)) {
          uint32_t r = eq;
          for (int t = 0; t < allowed; ++t) r &= r - 1u;
          take = eq & ~r;
        }
        kb[w] |= take;
      }
    }
    __syncthreads();
  }
  for (int w = tid; w < nw; w += nt) kp[w] = __popc(kb[w]);
  __syncthreads();
  const uint32_t tot = block_exclusive_scan(kp, nw, sh->wsum);
  if (tid == 0) kp[nw] = tot;
  __syncthreads();
}

// Channel id of kept index i (0 <= i < kp[nw]) from the bitmap + prefix.
__device__ __forceinline__ int kept_channel(const uint32_t* kb, const uint32_t* kp, int nw, uint32_t i) {
  int lo = 0, hi = nw - 1;   // find the last w with kp[w] <= i
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (kp[mid] <= i) lo = mid; else hi = mid - 1;
  }
  return 32 * lo + select_bit(kb[lo], (int)(i - kp[lo]));
}

}  // namespace duo
