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
// channel id outside the format's bounds), read by duo_device_status.  The
// translation unit that owns it (kernels.cu) defines DUO_STATUS_OWNER; any
// other unit including this header gets a private copy nobody reads.
#ifdef DUO_STATUS_OWNER
__device__ unsigned int g_status = 0u;
#else
static __device__ unsigned int g_status = 0u;
#endif
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

// ---- Quantised values (§5, weight-only quantisation, Table 4) ----
// A b-bit code q of row i in input-channel group g (128 channels) stands for
// s (q - z), with {fp16 s, z} the grid of (i, g).  Grid tables hold one
// (segment, group) each: entry 32 t + l is row 32 l + t of the segment.
constexpr int QGROUP = 128;                    // input channels per grid
constexpr int QTAB_BYTES = SEG_ROWS * 4;       // one table: 1024 uint32 entries
constexpr int QNTB = 4;                        // tables a CTA holds at once

// Walk over one lane's codes in a record, from its first code on.  at()
// reads the code at the current position whether or not the row has one
// (the byte after a lane's last code is still inside the record's slot or
// the 16 bytes of slack after the ring), and step(bit) moves on by one code
// when bit is 1: no branch per row.
template <int VB>
struct CodeWalk;

template <>
struct CodeWalk<8> {   // one byte per code
  const uint8_t* p;
  __device__ __forceinline__ void init(const uint8_t* codes, uint32_t first) { p = codes + first; }
  __device__ __forceinline__ uint32_t at() const { return *p; }
  __device__ __forceinline__ void step(uint32_t bit) { p += bit; }
};

template <>
struct CodeWalk<4> {   // two codes per byte, the even one in the low nibble
  const uint8_t* p;
  uint32_t sh;
  __device__ __forceinline__ void init(const uint8_t* codes, uint32_t first) {
    p = codes + (first >> 1);
    sh = (first & 1u) << 2;
  }
  __device__ __forceinline__ uint32_t at() const { return ((uint32_t)*p >> sh) & 15u; }
  __device__ __forceinline__ void step(uint32_t bit) {
    p += (sh >> 2) & bit;
    sh ^= bit << 2;
  }
};

// acc + bit * s (q - z) x (bit 0 or 1, no branch), with e = s's fp16 bits |
// z << 16 (z <= 255): q - z is the exact difference of 2^23 + q and
// 2^23 + z, s x is exact in fp32 (fp16 x fp16), and the fma rounds once.
__device__ __forceinline__ float q_fma_sel(uint32_t bit, uint32_t q, uint32_t e, uint16_t x, float acc) {
  const float d = __uint_as_float(0x4B000000u | q) -
                  __uint_as_float(__byte_perm(e, 0x4B000000u, 0x7542));
  const float sx = fma_f16_f32((uint16_t)(e & 0xFFFFu), x, 0.f);
  return fmaf(bit ? d : 0.f, sx, acc);
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

// Block-cooperative copy of x (fp16 bits) into shared memory.  Up to four
// 16-byte loads per thread are issued before the first store, so a thread
// waits for one memory round trip per 4 blocks of the input, not per block.
__device__ inline void load_x_to_smem(uint16_t* xs, const uint16_t* x, int I) {
  const int tid = threadIdx.x, nt = blockDim.x;
  if ((reinterpret_cast<uintptr_t>(x) & 15u) == 0) {
    const int nvec = I >> 3;
    const uint4* xv = reinterpret_cast<const uint4*>(x);
    uint4* sv = reinterpret_cast<uint4*>(xs);
    for (int i0 = tid; i0 < nvec; i0 += 4 * nt) {
      uint4 v[4];
#pragma unroll
      for (int u = 0; u < 4; ++u)
        if (i0 + u * nt < nvec) v[u] = __ldg(xv + i0 + u * nt);
#pragma unroll
      for (int u = 0; u < 4; ++u)
        if (i0 + u * nt < nvec) sv[i0 + u * nt] = v[u];
    }
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
  uint32_t sub[16];               // keys of bin C by key & 15
  uint32_t wcnt[SEL_MAX_WARPS];   // per-warp counts
  uint32_t C, aboveC;
  int T, cut;                     // the selection's result (see select_threshold)
};

// Clears the histograms (before the __syncthreads that precedes the selection).
__device__ __forceinline__ void select_clear(SelShared* sh) {
  uint4* h = reinterpret_cast<uint4*>(sh->hist);
  for (int i = threadIdx.x; i < (SEL_BINS + 16) / 4; i += blockDim.x)
    h[i] = make_uint4(0u, 0u, 0u, 0u);   // hist and sub are contiguous
}

// The key of x_j is its fp16 bit pattern with the sign cleared; for IEEE
// fp16 this integer order equals the order of |x_j| (NaN patterns sort above
// Inf).
__device__ __forceinline__ int key_of(const uint16_t* xs, int j) { return xs[j] & 0x7FFF; }

// Exact top-k by magnitude (§3) as a threshold: keeps the k channels with
// the largest |x_j|, ties to the lower index.  On return (to every thread)
// channel j is kept iff key_j > T, or key_j == T and j <= cut.
//
//  1. histogram of key >> 4 (2048 bins, shared-memory atomics);
//  2. one warp finds the bin C where the count from the top reaches k: a
//     suffix scan over 32 lanes x 64 bins, then over the 64 bins of the
//     crossing lane (2 per lane);
//  3. histogram of key & 15 over the keys of bin C (few: contention-free
//     atomics);
//  4. one warp gets T = 16 C + b and q = k - count(key > T), the number of
//     channels with key == T to keep (the lowest-indexed ones);
//  5. only if fewer than all of them are kept: each warp counts the ties in
//     its contiguous run of 32-channel words, and the warp holding the q-th
//     tie finds its channel, cut; otherwise cut = I.
// k <= 0 keeps nothing (T = 0x7FFF, cut = -1), k >= I everything (T = -1).
// xs holds the fp16 bits of x (room for a whole number of 32-channel words);
// select_clear() and the loading of xs come first, then a __syncthreads.  All
// threads of the block take part (512 <= blockDim.x <= 1024, a multiple of
// 32); it ends with a __syncthreads.
__device__ inline void select_threshold(const uint16_t* xs, int I, int k, SelShared* sh, int* T_out,
                                        int* cut_out) {
  const int tid = threadIdx.x, nt = blockDim.x, lane = tid & 31, wid = tid >> 5;
  const int nwarps = nt >> 5;
  const uint32_t kk = (uint32_t)k;
  if (k <= 0 || k >= I) {
    *T_out = k <= 0 ? 0x7FFF : -1;   // no key exceeds 0x7FFF; every key exceeds -1
    *cut_out = -1;
    __syncthreads();
    return;
  }
  // 1. histogram of the high 11 key bits (4 independent loads in flight)
  {
    int j = tid;
    for (; j + 3 * nt < I; j += 4 * nt) {
      const int k0 = key_of(xs, j), k1 = key_of(xs, j + nt);
      const int k2 = key_of(xs, j + 2 * nt), k3 = key_of(xs, j + 3 * nt);
      atomicAdd(&sh->hist[k0 >> 4], 1u);
      atomicAdd(&sh->hist[k1 >> 4], 1u);
      atomicAdd(&sh->hist[k2 >> 4], 1u);
      atomicAdd(&sh->hist[k3 >> 4], 1u);
    }
    for (; j < I; j += nt) atomicAdd(&sh->hist[key_of(xs, j) >> 4], 1u);
  }
  __syncthreads();
  // 2. threshold bin C, by warp 0
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
  // 3. the 16 keys of bin C
  {
    const int C = (int)sh->C;
    int j = tid;
    for (; j + 3 * nt < I; j += 4 * nt) {
      const int k0 = key_of(xs, j), k1 = key_of(xs, j + nt);
      const int k2 = key_of(xs, j + 2 * nt), k3 = key_of(xs, j + 3 * nt);
      if ((k0 >> 4) == C) atomicAdd(&sh->sub[k0 & 15], 1u);
      if ((k1 >> 4) == C) atomicAdd(&sh->sub[k1 & 15], 1u);
      if ((k2 >> 4) == C) atomicAdd(&sh->sub[k2 & 15], 1u);
      if ((k3 >> 4) == C) atomicAdd(&sh->sub[k3 & 15], 1u);
    }
    for (; j < I; j += nt) {
      const int key = key_of(xs, j);
      if ((key >> 4) == C) atomicAdd(&sh->sub[key & 15], 1u);
    }
  }
  __syncthreads();
  // 4. T and q (lane v < 16 = key & 15 inside bin C), by every warp: the
  //    result is read by all, with no further barrier.
  int T, q, ties;
  {
    const uint32_t sv = lane < 16 ? sh->sub[lane] : 0u;
    uint32_t suf = sv;   // keys of bin C with key & 15 >= lane
#pragma unroll
    for (int o = 1; o < 16; o <<= 1) {
      const uint32_t t = __shfl_down_sync(FULL_MASK, suf, o);
      if (lane + o < 16) suf += t;
    }
    const uint32_t need = kk - sh->aboveC;   // >= 1, <= hist[C]
    const int b = 31 - __clz(__ballot_sync(FULL_MASK, lane < 16 && suf >= need));
    T = 16 * (int)sh->C + b;
    q = (int)(need - __shfl_sync(FULL_MASK, suf - sv, b));   // >= 1
    ties = (int)__shfl_sync(FULL_MASK, sv, b);
  }
  int cut = I;
  if (q < ties) {
    // 5. the q-th channel with key == T in index order
    const int nw = (I + 31) >> 5;
    const int per = (nw + nwarps - 1) / nwarps;
    const int w0 = min(nw, wid * per), w1 = min(nw, w0 + per);
    uint32_t cnt = 0;
    for (int w = w0; w < w1; ++w) {
      const int j = 32 * w + lane;
      cnt += (uint32_t)__popc(__ballot_sync(FULL_MASK, j < I && key_of(xs, j) == T));
    }
    if (lane == 0) sh->wcnt[wid] = cnt;
    __syncthreads();
    const uint32_t c = lane < nwarps ? sh->wcnt[lane] : 0u;   // lane l: warp l's count
    uint32_t before = __reduce_add_sync(FULL_MASK, lane < wid ? c : 0u);
    const uint32_t own = __shfl_sync(FULL_MASK, c, wid);   // this warp's count, in every lane
    if (before < (uint32_t)q && (uint32_t)q <= before + own) {   // this warp holds the q-th tie
      for (int w = w0; w < w1; ++w) {
        const int j = 32 * w + lane;
        const uint32_t m = __ballot_sync(FULL_MASK, j < I && key_of(xs, j) == T);
        const uint32_t n = (uint32_t)__popc(m);
        if (before + n >= (uint32_t)q) {
          if (lane == 0) sh->cut = 32 * w + select_bit(m, q - 1 - (int)before);
          break;
        }
        before += n;
      }
    }
    __syncthreads();
    cut = sh->cut;
  }
  *T_out = T;
  *cut_out = cut;
  __syncthreads();
}

// Writes the channels j in [c0, c1) that a threshold keeps (key_j > T, or
// key_j == T and j <= cut) in ascending order to klist[0..n) (and their fp16
// bits to kvals if given) and returns n to every thread.  Warps take
// contiguous runs of the range's 32-channel words (lane = channel): one
// ballot pass counts, a block barrier and a sum over lower warps place each
// warp's run, a second pass writes.  wcnt needs one entry per warp.  All
// threads take part; it ends with a __syncthreads.  Used for the threshold
// mask of §5 (T = tau, cut = -1) and for the top-k set as a threshold.
__device__ inline int thresh_compact(const uint16_t* xs, int c0, int c1, int T, int cut,
                                     uint16_t* klist, uint16_t* kvals, uint32_t* wcnt) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
  const int wb = c0 >> 5, nwd = c1 > c0 ? ((c1 + 31) >> 5) - wb : 0;
  const int per = (nwd + nwarps - 1) / nwarps;
  const int w0 = wb + min(nwd, wid * per), w1 = wb + min(nwd, wid * per + per);
  auto kept = [&](int j) {
    if (j < c0 || j >= c1) return false;
    const int key = key_of(xs, j);
    return key > T || (key == T && j <= cut);
  };
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
