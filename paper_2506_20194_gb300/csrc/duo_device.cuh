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

// Same, but the thread may be suspended for up to hint_ns until the phase
// completes, so a waiting warp takes no issue slots from the others.
__device__ __forceinline__ bool mbar_try_wait_suspend(uint64_t* bar, uint32_t parity,
                                                      uint32_t hint_ns) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cta.shared::cta.b64 p, [%1], %2, %3;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity), "r"(hint_ns)
      : "memory");
  return ok != 0;
}

constexpr uint32_t SUSPEND_HINT_NS = 2000;

// Waits for the phase of `parity` with a wall-clock limit.  On timeout the
// device status word and the CTA's abort flag are set and false returned;
// a wait also gives up (false) once another warp has raised the abort flag.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t* bar, uint32_t parity,
                                                  volatile int* abort_flag) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  while (true) {
    if (mbar_try_wait_suspend(bar, parity, SUSPEND_HINT_NS)) return true;
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

__device__ __forceinline__ int ld_acquire_cta_shared(const int* p) {
  int v;
  asm volatile("ld.acquire.cta.shared::cta.b32 %0, [%1];" : "=r"(v) : "r"(smem_u32(p)) : "memory");
  return v;
}

__device__ __forceinline__ void st_release_cta_shared(int* p, int v) {
  asm volatile("st.release.cta.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(p)), "r"(v) : "memory");
}

// Spins (bounded, like mbar_wait_bounded) until the shared word at p equals
// want.  Used to check the exact identity of a ring slot's fill, which an
// mbarrier parity alone cannot tell apart from a fill two phases earlier.
__device__ __forceinline__ bool wait_shared_eq(const int* p, int want, volatile int* abort_flag) {
  if (ld_acquire_cta_shared(p) == want) return true;
  const uint64_t t0 = globaltimer_ns();
  while (true) {
    if (ld_acquire_cta_shared(p) == want) return true;
    if (*abort_flag) return false;
    if (globaltimer_ns() - t0 > WAIT_LIMIT_NS) {
      atomicOr(&g_status, STATUS_TIMEOUT);
      *abort_flag = 1;
      return false;
    }
  }
}

// Programmatic dependent launch: wait until the previous kernel of the
// stream has completed and its memory is visible (returns at once when the
// launch has no programmatic dependency), and let the next kernel of the
// stream be scheduled as soon as this grid's CTAs leave their SMs.
__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void griddep_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
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
constexpr int SEL_MAX_WARPS = 32;

// Shared state of the selection.
struct SelShared {
  uint32_t hist[SEL_BINS];
  uint32_t subw[SEL_MAX_WARPS][16];   // per warp: its keys of bin C by key & 15
  uint32_t wgt[SEL_MAX_WARPS];        // per warp: its keys in bins above C
  uint32_t wpre[SEL_MAX_WARPS];       // per warp: keys above T | ties << 16 in lower warps
  uint32_t wown[SEL_MAX_WARPS];       // per warp: its own keys above T | ties << 16
  uint32_t C, aboveC, T, q;
};

// Clears the histograms (before the __syncthreads that precedes select_topk).
__device__ __forceinline__ void select_clear(SelShared* sh) {
  uint4* h = reinterpret_cast<uint4*>(sh->hist);
  for (int i = threadIdx.x; i < (SEL_BINS + 16 * SEL_MAX_WARPS) / 4; i += blockDim.x)
    h[i] = make_uint4(0u, 0u, 0u, 0u);   // hist and subw are contiguous
}

// Exact top-k by magnitude (§3): keeps the k channels with the largest
// |x_j|, ties to the lower index.  The key of x_j is its fp16 bit pattern
// with the sign cleared; for IEEE fp16 this integer order equals the order of
// |x_j| (NaN patterns sort above Inf).  xs holds the fp16 bits of x in
// shared memory (room for a whole number of 32-channel words).
//
//  1. histogram of key >> 4 (2048 bins, shared-memory atomics);
//  2. one warp finds, by suffix scans over 32 blocks of 64 bins and then
//     over the bins of the block that holds the crossing, the bin C where the
//     count from the top reaches k;
//  3. warp w walks its contiguous run of 32-channel words (lane = channel)
//     and counts its keys in bins above C (ballots) and, by key & 15, its
//     keys in bin C (its own 16 counters);
//  4. one warp sums the per-warp counters of bin C to find the threshold
//     key T = 16 C + b and q = k - count(key > T), the number of channels
//     with key == T that are kept (the lowest-indexed ones), and scans the
//     per-warp counts to give every warp the "above T" and "tie" counts
//     before its own run;
//  5. warps whose kept ranks meet the requested window walk their words
//     again: kept channel j has rank r = (channels above T before j) +
//     min(q, ties before j); if d = (r - r0) mod k is below rn it writes
//     klist[d] = j and kvals[d] = its fp16 bits.
//
// The window is the cyclic rank range r0, r0 + 1, ... (mod k) of length
// min(rn, k); with r0 = 0 and rn = k the lists are indexed by rank.
//
// select_clear() and the loading of xs come first, then a __syncthreads.
// All threads of the block take part (512 <= blockDim.x <= 1024, a multiple
// of 32); it ends with a __syncthreads.
constexpr uint32_t KEY_NONE = 0xFFFFu;
__device__ __forceinline__ uint32_t key_of(const uint16_t* xs, int j) { return xs[j] & 0x7FFFu; }

__device__ __forceinline__ bool ranges_meet(uint32_t a0, uint32_t a1, uint32_t b0, uint32_t b1) {
  return a0 < b1 && b0 < a1;
}

__device__ inline void select_topk(const uint16_t* xs, int I, int k, uint32_t r0, uint32_t rn,
                                   uint16_t* klist, uint16_t* kvals, SelShared* sh) {
  const int tid = threadIdx.x, nt = blockDim.x, lane = tid & 31, wid = tid >> 5;
  const int nwarps = nt >> 5;
  const int nw = (I + 31) >> 5;
  const uint32_t kk = (uint32_t)k;
  const bool whole = rn >= kk;
  // list position of rank r, or -1 outside the window
  auto slot_of = [&](uint32_t r) -> int {
    const uint32_t d = r >= r0 ? r - r0 : r + kk - r0;
    return (whole || d < rn) ? (int)d : -1;
  };
  if (k <= 0) {   // nothing kept
    __syncthreads();
    return;
  }
  if (k >= I) {   // everything kept: rank = channel
    for (int j = tid; j < I; j += nt) {
      const int d = slot_of((uint32_t)j);
      if (d >= 0) {
        if (klist != nullptr) klist[d] = (uint16_t)j;
        if (kvals != nullptr) kvals[d] = xs[j];
      }
    }
    __syncthreads();
    return;
  }
  // 1. histogram of the high 11 key bits (4 independent loads in flight)
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
  // 2. threshold bin C, by warp 0 alone: lane l totals bins [64 l, 64 l + 64),
  //    a suffix scan over lanes finds the lane whose bins hold the crossing,
  //    and a second scan over that lane's 64 bins (2 per lane) finds C.
  if (wid == 0) {
    const uint4* h4 = reinterpret_cast<const uint4*>(sh->hist) + 16 * lane;
    uint32_t s64 = 0;
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const uint4 h = h4[(i + lane) & 15];   // rotated: a quarter warp hits 8 bank groups
      s64 += (h.x + h.y) + (h.z + h.w);
    }
    uint32_t sl = s64;   // keys in bins >= 64 * lane
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t t = __shfl_down_sync(FULL_MASK, sl, o);
      if (lane + o < 32) sl += t;
    }
    const int L = 31 - __clz(__ballot_sync(FULL_MASK, sl >= kk));
    const uint32_t above_l = __shfl_sync(FULL_MASK, sl - s64, L);   // keys in bins >= 64 (L + 1)
    const uint2 h2 = reinterpret_cast<const uint2*>(sh->hist)[32 * L + lane];   // bins 64 L + 2 lane, +1
    const uint32_t s2 = h2.x + h2.y;
    uint32_t sp = s2;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t t = __shfl_down_sync(FULL_MASK, sp, o);
      if (lane + o < 32) sp += t;
    }
    const int M = 31 - __clz(__ballot_sync(FULL_MASK, above_l + sp >= kk));
    if (lane == M) {
      const uint32_t above = above_l + sp - s2;   // keys above bin 64 L + 2 M + 1
      const bool hi = above + h2.y >= kk;
      sh->C = 64u * (uint32_t)L + 2u * (uint32_t)M + (hi ? 1u : 0u);
      sh->aboveC = hi ? above : above + h2.y;
    }
  }
  __syncthreads();
  // 3. per-warp counts over the warp's words [w0, w1)
  const int per = (nw + nwarps - 1) / nwarps;
  const int w0 = min(nw, wid * per), w1 = min(nw, w0 + per);
  {
    const uint32_t C = sh->C;
    uint32_t ngt = 0;
    for (int w = w0; w < w1; w += 4) {
      uint32_t key[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int j = 32 * (w + u) + lane;
        key[u] = (w + u < w1 && j < I) ? key_of(xs, j) : KEY_NONE;
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const bool valid = key[u] != KEY_NONE;
        ngt += (uint32_t)__popc(__ballot_sync(FULL_MASK, valid && (key[u] >> 4) > C));
        if (valid && (key[u] >> 4) == C) atomicAdd(&sh->subw[wid][key[u] & 15u], 1u);
      }
    }
    if (lane == 0) sh->wgt[wid] = ngt;
  }
  __syncthreads();
  // 4. by warp 0 alone: the threshold key T = 16 C + b (lane v < 16 = key & 15
  //    inside bin C), q, and for every warp w (lane w) its own and its lower
  //    warps' counts above T and equal to T.
  if (wid == 0) {
    uint32_t part[4] = {0u, 0u, 0u, 0u};
    if (lane < 16) {
#pragma unroll
      for (int w = 0; w < SEL_MAX_WARPS; ++w)
        if (w < nwarps) part[w & 3] += sh->subw[w][lane];
    }
    const uint32_t sv = (part[0] + part[1]) + (part[2] + part[3]);
    uint32_t suf = sv;   // keys of bin C with key & 15 >= lane
#pragma unroll
    for (int o = 1; o < 16; o <<= 1) {
      const uint32_t t = __shfl_down_sync(FULL_MASK, suf, o);
      if (lane + o < 16) suf += t;
    }
    const uint32_t need = kk - sh->aboveC;   // >= 1, <= hist[C]
    const int b = 31 - __clz(__ballot_sync(FULL_MASK, lane < 16 && suf >= need));
    const uint32_t above_in_c = __shfl_sync(FULL_MASK, suf - sv, b);
    uint32_t al = 0, tl = 0;
    if (lane < nwarps) {
      const uint4* row = reinterpret_cast<const uint4*>(sh->subw[lane]);
      al = sh->wgt[lane];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int c = (i + (lane >> 1)) & 3;   // rotated: conflict-free quarter warps
        const uint4 r4 = row[c];
        const uint32_t v4[4] = {r4.x, r4.y, r4.z, r4.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int v = 4 * c + e;
          al += v > b ? v4[e] : 0u;
          tl += v == b ? v4[e] : 0u;
        }
      }
    }
    const uint32_t own = al | (tl << 16);   // each <= 65535
    const uint32_t pre = warp_inclusive_scan(own, lane) - own;
    if (lane < nwarps) {
      sh->wpre[lane] = pre;
      sh->wown[lane] = own;
    }
    if (lane == 0) {
      sh->T = 16u * sh->C + (uint32_t)b;
      sh->q = need - above_in_c;   // >= 1
    }
  }
  __syncthreads();
  const uint32_t T = sh->T, q = sh->q;
  uint32_t gpre, epre, a_own, t_own;
  {
    const uint32_t pre = sh->wpre[wid], own = sh->wown[wid];
    gpre = pre & 0xFFFFu;
    epre = pre >> 16;
    a_own = own & 0xFFFFu;
    t_own = own >> 16;
  }
  // 5. emission by the warps whose kept ranks meet the window
  if (klist != nullptr || kvals != nullptr) {
    const uint32_t R = gpre + min(epre, q);
    const uint32_t Kw = a_own + min(epre + t_own, q) - min(epre, q);
    bool meet = whole;
    if (!meet && Kw > 0) {
      const uint32_t e0 = r0 + rn;   // window [r0, e0), wrapping past kk
      meet = ranges_meet(R, R + Kw, r0, min(e0, kk)) || (e0 > kk && ranges_meet(R, R + Kw, 0u, e0 - kk));
    }
    if (meet) {
      const uint32_t lt = (1u << lane) - 1u;
      for (int w = w0; w < w1; w += 4) {
        uint32_t key[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int j = 32 * (w + u) + lane;
          key[u] = (w + u < w1 && j < I) ? key_of(xs, j) : KEY_NONE;
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const bool valid = key[u] != KEY_NONE;
          const bool isg = valid && key[u] > T;
          const bool ise = valid && key[u] == T;
          const uint32_t g = __ballot_sync(FULL_MASK, isg);
          const uint32_t e = __ballot_sync(FULL_MASK, ise);
          const uint32_t tr = epre + (uint32_t)__popc(e & lt);   // ties before this channel
          if (isg || (ise && tr < q)) {
            const int d = slot_of(gpre + (uint32_t)__popc(g & lt) + min(tr, q));
            if (d >= 0) {
              const int j = 32 * (w + u) + lane;
              if (klist != nullptr) klist[d] = (uint16_t)j;
              if (kvals != nullptr) kvals[d] = xs[j];
            }
          }
          gpre += (uint32_t)__popc(g);
          epre += (uint32_t)__popc(e);
        }
      }
    }
  }
  __syncthreads();
}

// Threshold mask (§5, threshold-based activation sparsity): writes the
// channels j in [c0, c1) with key_j > T in ascending order to klist[0..n) (and
// their fp16 bits to kvals if given) and returns n to every thread.  Warps
// take contiguous runs of the range's 32-channel words (lane = channel): one
// ballot pass counts, a block barrier and a sum over lower warps place each
// warp's run, a second pass writes.  wcnt needs one entry per warp.  All
// threads take part; it ends with a __syncthreads.
__device__ inline int thresh_compact(const uint16_t* xs, int c0, int c1, uint32_t T, uint16_t* klist,
                                     uint16_t* kvals, uint32_t* wcnt) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
  const int wb = c0 >> 5, nwd = c1 > c0 ? ((c1 + 31) >> 5) - wb : 0;
  const int per = (nwd + nwarps - 1) / nwarps;
  const int w0 = wb + min(nwd, wid * per), w1 = wb + min(nwd, wid * per + per);
  auto kept = [&](int j) { return j >= c0 && j < c1 && key_of(xs, j) > T; };
  uint32_t cnt = 0;
  for (int w = w0; w < w1; ++w) cnt += (uint32_t)__popc(__ballot_sync(FULL_MASK, kept(32 * w + lane)));
  if (lane == 0) wcnt[wid] = cnt;
  __syncthreads();
  const uint32_t c = lane < nwarps ? wcnt[lane] : 0u;
  uint32_t base = __reduce_add_sync(FULL_MASK, lane < wid ? c : 0u);
  const uint32_t total = __reduce_add_sync(FULL_MASK, c);
  const uint32_t lt = (1u << lane) - 1u;
  for (int w = w0; w < w1; ++w) {
    const int j = 32 * w + lane;
    const bool keep = kept(j);
    const uint32_t m = __ballot_sync(FULL_MASK, keep);
    if (keep) {
      const uint32_t pos = base + (uint32_t)__popc(m & lt);
      klist[pos] = (uint16_t)j;
      if (kvals != nullptr) kvals[pos] = xs[j];
    }
    base += (uint32_t)__popc(m);
  }
  __syncthreads();
  return (int)total;
}

}  // namespace duo
