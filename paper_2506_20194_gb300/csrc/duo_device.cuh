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

// L2 prefetch of [src, src + bytes) (16-byte aligned, bytes % 16 == 0).
__device__ __forceinline__ void prefetch_l2(const void* src, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(src), "r"(bytes) : "memory");
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

__device__ __forceinline__ unsigned int ld_relaxed_gpu(const unsigned int* p) {
  unsigned int v;
  asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ unsigned int atom_add_acq_rel_gpu(unsigned int* p, unsigned int v) {
  unsigned int old;
  asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
  return old;
}

__device__ __forceinline__ void red_add_release_gpu(unsigned int* p, unsigned int v) {
  asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
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

constexpr int SEL_BINS = 2048;   // histogram of key >> 4

// Shared state of the selection.
struct SelShared {
  uint32_t hist[SEL_BINS];
  uint32_t sub[16];      // key & 15 inside the threshold bin
  uint32_t wtot[32];     // per-warp partial sums
  uint32_t C;            // threshold bin
  uint32_t aboveC;       // channels in bins above it
};

// Clears the histograms (before the __syncthreads that precedes select_topk).
__device__ __forceinline__ void select_clear(SelShared* sh) {
  uint4* h = reinterpret_cast<uint4*>(sh->hist);
  for (int i = threadIdx.x; i < SEL_BINS / 4; i += blockDim.x) h[i] = make_uint4(0u, 0u, 0u, 0u);
  if (threadIdx.x < 16) sh->sub[threadIdx.x] = 0u;
}

// Exact top-k by magnitude (§3): keeps the k channels with the largest
// |x_j|, ties to the lower index.  The key of x_j is its fp16 bit pattern
// with the sign cleared; for IEEE fp16 this integer order equals the order of
// |x_j| (NaN patterns sort above Inf).  xs holds the fp16 bits of x in
// shared memory (room for a whole number of 32-channel words).
//
//  1. histogram of key >> 4 (2048 bins, shared-memory atomics);
//  2. suffix scan of the histogram (512 threads x 4 bins) to find the bin C
//     where the count from the top reaches k;
//  3. histogram of key & 15 over the few channels in bin C, giving the
//     threshold key T and the count above it; the q = k - count(key > T)
//     lowest-indexed channels with key == T are kept;
//  4. every thread builds the "above T" / "equal to T" masks of its own
//     32-channel words from 16-byte loads of x, a block exclusive scan of the
//     packed counts orders the words, and the thread writes kb[w] (kept
//     bitmap, bit b <-> channel 32w+b) and kp[w] (kept channels before word
//     w; kp[nw] = k);
//  5. if klist / kvals are given, warps emit klist[r] (channel of kept rank
//     r, ascending) and kvals[r] (its fp16 bits), lane = bit.
// Shared-memory accesses are arranged to be bank-conflict free.
//
// select_clear() and the loading of xs come first, then a __syncthreads.
// All threads of the block take part (blockDim.x >= 512, a multiple of 32);
// it ends with a __syncthreads.
__device__ __forceinline__ uint32_t key_of(const uint16_t* xs, int j) { return xs[j] & 0x7FFFu; }

// Masks of the channels of word w (32 channels) above T and equal to T.  The
// four 16-byte chunks are read in an order rotated by (w >> 1) so that the
// eight threads of a quarter warp (consecutive words) hit distinct banks.
__device__ __forceinline__ void word_masks(const uint16_t* xs, int I, int w, bool all, bool none,
                                           uint32_t T, uint32_t& gt, uint32_t& eq) {
  const uint4* p = reinterpret_cast<const uint4*>(xs + 32 * w);
  const int rot = (w >> 1) & 3;
  gt = 0u;
  eq = 0u;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int ci = (i + rot) & 3;
    const uint4 c = p[ci];
    const uint32_t v[4] = {c.x, c.y, c.z, c.w};
#pragma unroll
    for (int h = 0; h < 8; ++h) {
      const uint32_t key = (v[h >> 1] >> (16 * (h & 1))) & 0x7FFFu;
      const int b = 8 * ci + h;
      gt |= (uint32_t)(key > T) << b;
      eq |= (uint32_t)(key == T) << b;
    }
  }
  const int valid = min(32, I - 32 * w);
  const uint32_t vmask = valid >= 32 ? FULL_MASK : ((1u << valid) - 1u);
  if (all) { gt = FULL_MASK; eq = 0u; }
  if (none) { gt = 0u; eq = 0u; }
  gt &= vmask;
  eq &= vmask;
}

__device__ inline void select_topk(const uint16_t* xs, int I, int k, uint32_t* kb, uint32_t* kp,
                                   uint16_t* klist, uint16_t* kvals, SelShared* sh) {
  const int tid = threadIdx.x, nt = blockDim.x, lane = tid & 31, wid = tid >> 5;
  const int nwarps = nt >> 5;
  const int nw = (I + 31) >> 5;
  const bool all = k >= I, none = k <= 0;
  uint32_t T = 0u;
  int q = 0;
  if (!all && !none) {
    // 1. histogram of the high 11 key bits
    {
      int j = tid;
      for (; j + 3 * nt < I; j += 4 * nt) {
        const uint32_t k0 = key_of(xs, j), k1 = key_of(xs, j + nt);
        const uint32_t k2 = key_of(xs, j + 2 * nt), k3 = key_of(xs, j + 3 * nt);
        atomicAdd(&sh->hist[k0 >> 4], 1u);
        atomicAdd(&sh->hist[k1 >> 4], 1u);
        atomicAdd(&sh->hist[k2 >> 4], 1u);
        atomicAdd(&sh->hist[k3 >> 4], 1u);
      }
      for (; j < I; j += nt) atomicAdd(&sh->hist[key_of(xs, j) >> 4], 1u);
    }
    __syncthreads();
    // 2. suffix scan: thread t < 512 owns bins [4t, 4t + 4)
    uint32_t c[4] = {0u, 0u, 0u, 0u}, s = 0, incl = 0;
    if (tid < 512) {
      const uint4 h = reinterpret_cast<const uint4*>(sh->hist)[tid];
      c[0] = h.x; c[1] = h.y; c[2] = h.z; c[3] = h.w;
      s = c[0] + c[1] + c[2] + c[3];
      incl = s;   // suffix over lanes >= lane inside the warp
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t t = __shfl_down_sync(FULL_MASK, incl, o);
        if (lane + o < 32) incl += t;
      }
      if (lane == 0) sh->wtot[wid] = incl;
    }
    __syncthreads();
    if (tid < 512) {
      uint32_t above_w = (lane > wid && lane < 16) ? sh->wtot[lane] : 0u;
      above_w = __reduce_add_sync(FULL_MASK, above_w);
      const uint32_t hi = above_w + incl;   // channels in bins >= 4*tid
      const uint32_t lo = hi - s;           // channels in bins >= 4*tid + 4
      if (lo < (uint32_t)k && (uint32_t)k <= hi) {
        uint32_t acc = lo;
        int b = 0;
#pragma unroll
        for (int i = 3; i >= 0; --i) {
          if (acc + c[i] >= (uint32_t)k) { b = i; break; }
          acc += c[i];
        }
        sh->C = 4u * tid + (uint32_t)b;
        sh->aboveC = acc;
      }
    }
    __syncthreads();
    // 3. the 16 keys of bin C (few channels: contention-free atomics)
    const uint32_t C = sh->C;
    for (int j = tid; j < I; j += nt) {
      const uint32_t key = key_of(xs, j);
      if ((key >> 4) == C) atomicAdd(&sh->sub[key & 15u], 1u);
    }
    __syncthreads();
    uint32_t sub[16];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const uint4 v = reinterpret_cast<const uint4*>(sh->sub)[i];
      sub[4 * i] = v.x; sub[4 * i + 1] = v.y; sub[4 * i + 2] = v.z; sub[4 * i + 3] = v.w;
    }
    uint32_t above = sh->aboveC;
    int b = -1;
#pragma unroll
    for (int v = 15; v >= 0; --v) {
      if (b < 0) {
        if (above + sub[v] >= (uint32_t)k) b = v;
        else above += sub[v];
      }
    }
    if (b < 0) b = 0;
    T = 16u * C + (uint32_t)b;
    q = k - (int)above;
  }
  // 4. thread tid owns words [w0, w1)
  const int per = (nw + nt - 1) / nt;
  const int w0 = min(nw, tid * per), w1 = min(nw, w0 + per);
  uint32_t packed = 0;   // greater-count | tie-count << 16 (each <= 65535)
  for (int w = w0; w < w1; ++w) {
    uint32_t gt, eq;
    word_masks(xs, I, w, all, none, T, gt, eq);
    kb[w] = gt;   // provisional: the masks are kept in kb / kp until ranked
    kp[w] = eq;
    packed += (uint32_t)__popc(gt) | ((uint32_t)__popc(eq) << 16);
  }
  const uint32_t inc = warp_inclusive_scan(packed, lane);
  if (lane == 31) sh->wtot[wid] = inc;   // step 2's wtot reads ended two barriers ago
  __syncthreads();
  if (wid == 0) {
    uint32_t t = lane < nwarps ? sh->wtot[lane] : 0u;
    t = warp_inclusive_scan(t, lane);
    sh->wtot[lane] = t;
  }
  __syncthreads();
  const uint32_t base = (wid > 0 ? sh->wtot[wid - 1] : 0u) + inc - packed;
  uint32_t gpre = base & 0xFFFFu, epre = base >> 16;
  for (int w = w0; w < w1; ++w) {
    const uint32_t gt = kb[w], eq = kp[w];
    const int allowed = q - (int)epre;
    uint32_t take = 0u;
    if (allowed > 0 && eq != 0u)
      take = allowed >= __popc(eq) ? eq : (eq & ((1u << select_bit(eq, allowed)) - 1u));
    kb[w] = gt | take;
    kp[w] = gpre + min(epre, (uint32_t)q);
    gpre += __popc(gt);
    epre += __popc(eq);
  }
  if (tid == 0) kp[nw] = all ? (uint32_t)I : (none ? 0u : (uint32_t)k);
  __syncthreads();
  // 5. warp-parallel emission of the kept list
  if (klist != nullptr || kvals != nullptr) {
    const uint32_t lt = (1u << lane) - 1u;
    for (int w = wid; w < nw; w += nwarps) {
      const uint32_t kbw = kb[w];
      if ((kbw >> lane) & 1u) {
        const uint32_t rank = kp[w] + __popc(kbw & lt);
        const int j = 32 * w + lane;
        if (klist != nullptr) klist[rank] = (uint16_t)j;
        if (kvals != nullptr) kvals[rank] = xs[j];
      }
    }
    __syncthreads();
  }
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
