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

// Device status words (bit 0: a bounded wait ran out; bit 1: a record size
// or channel id outside the format's bounds).  A launch with a packed handle
// writes that handle's word (kept next to its grid-barrier words); the
// process-wide word below is for kernels without a handle.  The translation
// unit that owns it (kernels.cu) defines DUO_STATUS_OWNER; any other unit
// including this header gets a private copy nobody reads.
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
// status word (bit STATUS_TIMEOUT) and the CTA's abort flag are set and
// false returned; a wait also gives up (false) once another warp has raised
// the abort flag.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t* bar, uint32_t parity,
                                                  volatile int* abort_flag, unsigned int* status,
                                                  uint64_t limit_ns = WAIT_LIMIT_NS) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  while (true) {
    if (mbar_try_wait_suspend(bar, parity, SUSPEND_HINT_NS)) return true;
    if (*abort_flag) return false;
    if (globaltimer_ns() - t0 > limit_ns) {
      atomicOr(status, STATUS_TIMEOUT);
      *abort_flag = 1;
      return false;
    }
  }
}

// Same, without an abort flag (used while draining after an abort).
__device__ __forceinline__ bool mbar_wait_limited(uint64_t* bar, uint32_t parity, unsigned int* status,
                                                   uint64_t limit_ns = WAIT_LIMIT_NS) {
  const uint64_t t0 = globaltimer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (globaltimer_ns() - t0 > limit_ns) {
      atomicOr(status, STATUS_TIMEOUT);
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

// L2 prefetch of the 128-byte line holding p (any alignment).
__device__ __forceinline__ void prefetch_line_l2(const void* p) {
  asm volatile("prefetch.global.L2 [%0];" ::"l"(p));
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
// How a consumer lane walks its b-bit codes along its 32 positions (the
// lane's codes are consecutive in the record, from the code index its mask
// prefix gives).  8-bit codes: one byte load per position and a pointer
// that advances on set bits (the cheapest in instructions: measured faster
// than windows for this width).  4-bit codes: a window of 8 codes from two
// aligned 32-bit loads and a funnel shift, reloaded every 8 positions, with
// a shift per consumed code (a nibble walk costs a shift, a mask and a
// parity update per position).  A window reads up to 7 bytes past the
// lane's last code: the ring keeps 16 bytes of slack after its last slot.
template <int VB>
struct CodeWalk;

template <>
struct CodeWalk<8> {   // one byte per code
  static constexpr int G = 32;   // positions per (re)load: the whole record
  const uint8_t* p;
  __device__ __forceinline__ void load(const uint8_t* codes, uint32_t first) { p = codes + first; }
  __device__ __forceinline__ uint32_t at() const { return *p; }
  __device__ __forceinline__ void step(uint32_t bit) { p += bit; }
};

template <>
struct CodeWalk<4> {   // two codes per byte, the even one in the low nibble
  static constexpr int G = 8;
  uint32_t w;
  __device__ __forceinline__ void load(const uint8_t* codes, uint32_t first) {
    const uint32_t* wd = reinterpret_cast<const uint32_t*>(codes);
    const uint32_t i = first >> 3;
    w = __funnelshift_r(wd[i], wd[i + 1], (first & 7u) << 2);
  }
  __device__ __forceinline__ uint32_t at() const { return w & 15u; }
  __device__ __forceinline__ void step(uint32_t bit) { w >>= bit << 2; }
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
  uint32_t tmp[6 * SEL_MAX_WARPS];   // select_window's scratch
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

// Step 2 of select_threshold, by warp 0 only (after the histogram of key >> 4
// is complete): the bin C where the count of keys from the top reaches k,
// and the number of keys above it, into sh->C and sh->aboveC.  1 <= k < I.
__device__ __forceinline__ void select_find_bin(SelShared* sh, uint32_t kk, int lane) {
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

// Steps 4 and 5 of select_threshold (after the histogram of key & 15 over
// the keys of bin C is complete): T, and the tie cut when fewer than all
// keys equal to T are kept.  Every thread of the block calls it; it ends
// with a __syncthreads.
__device__ inline void select_finish(const uint16_t* xs, int I, int k, SelShared* sh, int* T_out,
                                     int* cut_out) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
  const uint32_t kk = (uint32_t)k;
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
  if (wid == 0) select_find_bin(sh, kk, lane);
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
  select_finish(xs, I, k, sh, T_out, cut_out);
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

// Whether select_window<..., NT>() can hold this x in registers: 16-byte
// aligned, at most four 16-byte chunks per thread.
template <int NT>
__device__ __forceinline__ bool select_window_ok(const uint16_t* x, int I) {
  return (reinterpret_cast<uintptr_t>(x) & 15u) == 0 && (I >> 3) <= 4 * NT;
}

// x into shared memory (fp16 bits), the kept set, and this CTA's share of
// the kept list, all from registers: each thread holds NCH 16-byte chunks
// of x (chunk c of thread t: channels 8 (t + c NT) .. + 7; the last
// I % 8 channels, one per thread, after them).
//  * top-k: a histogram of key >> 4 (2048 bins) counted straight from the
//    registers; every warp finds the bin C where the count from the top
//    reaches k (each warp sums 128 bins; then each warp reads the crossing
//    warp's bins again); the keys of bin C give T = 16 C + b, and q, the
//    number of channels with key == T to keep (the lowest-indexed ones).
//    The threshold mask keeps key > tau (T = tau, q = 0).
//  * one block scan of per-chunk counts of key > T and key == T (in channel
//    order) ranks every channel: a kept channel (key > T, or key == T with
//    fewer than q equal keys before it) has rank #(key > T before it) +
//    min(q, #(key == T before it)); each thread writes its kept channels
//    whose rank lies in this CTA's window [K m / nr, K (m + 1) / nr), K the
//    number kept (m = bits 32..47 of `run`, this CTA's index in its run,
//    nr = bits 48..63, the run's CTAs), to klist (ascending).  Every CTA of
//    a run thus gets the same number of channels (+-1) however x is spread.
// Returns the window size; ends with a barrier.  NCH = ceil((I / 8) /
// NT), 1..4 (select_window_ok() tells whether it fits).  All NT threads of the
// block take part; tmp needs 6 NT / 32 words.
template <bool TOPK, int NCH, int NT>
__device__ __noinline__ int select_window(const uint16_t* x, int I, int k, int tau_key,
                                             uint16_t* xs, SelShared* sh, uint64_t run,
                                             uint16_t* klist, uint32_t* tmp) {
  constexpr int ST_THREADS = NT, ST_WARPS = NT / 32;
  static_assert(ST_WARPS * 128 == SEL_BINS, "each warp sums 128 histogram bins");
  static_assert(NCH * 8 <= 32 && NCH >= 1, "at most four chunks (32 channels) a thread");
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  const int nvec = I >> 3;
  const uint4* x4 = reinterpret_cast<const uint4*>(x);
  uint32_t w[4 * NCH];   // the chunks, 2 channels per word
  bool have[NCH];
#pragma unroll
  for (int c = 0; c < NCH; ++c) {
    const int i = tid + c * ST_THREADS;
    have[c] = i < nvec;
    const uint4 v = have[c] ? __ldg(x4 + i) : make_uint4(0u, 0u, 0u, 0u);
    w[4 * c] = v.x;
    w[4 * c + 1] = v.y;
    w[4 * c + 2] = v.z;
    w[4 * c + 3] = v.w;
    if (have[c]) reinterpret_cast<uint4*>(xs)[i] = v;
  }
  const int jt = (nvec << 3) + tid;   // the tail channel of this thread, if < I
  const bool tail = jt < I;
  const uint16_t xt = tail ? x[jt] : (uint16_t)0;
  if (tail) xs[jt] = xt;
  auto key_at = [&](int c, int h) { return (int)((w[4 * c + (h >> 1)] >> (16 * (h & 1))) & 0x7FFFu); };
  int T, q = 0;
  if (!TOPK) {
    T = tau_key;
  } else if (k <= 0 || k >= I) {
    T = k <= 0 ? 0x7FFF : -1;
  } else {
    const uint32_t kk = (uint32_t)k;
#pragma unroll
    for (int c = 0; c < NCH; ++c)
      if (have[c])
#pragma unroll
        for (int h = 0; h < 8; ++h) atomicAdd(&sh->hist[key_at(c, h) >> 4], 1u);
    if (tail) atomicAdd(&sh->hist[(xt & 0x7FFFu) >> 4], 1u);
    __syncthreads();
    // bin C: warp v sums bins 128 v .. 128 v + 127; every warp then scans the
    // 16 sums and the crossing warp's bins (lane l: bins 4 l .. 4 l + 3)
    {
      const uint4 h4 = reinterpret_cast<const uint4*>(sh->hist)[32 * wid + lane];
      const uint32_t wsum = __reduce_add_sync(FULL_MASK, (h4.x + h4.y) + (h4.z + h4.w));
      if (lane == 0) tmp[wid] = wsum;
    }
    __syncthreads();
    {
      const uint32_t wv = lane < ST_WARPS ? tmp[lane] : 0u;
      uint32_t suf = wv;   // keys in bins >= 128 lane
#pragma unroll
      for (int o = 1; o < ST_WARPS; o <<= 1) {
        const uint32_t t = __shfl_down_sync(FULL_MASK, suf, o);
        if (lane + o < ST_WARPS) suf += t;
      }
      const int W = 31 - __clz(__ballot_sync(FULL_MASK, lane < ST_WARPS && suf >= kk));
      const uint32_t above_w = __shfl_sync(FULL_MASK, suf - wv, W);   // keys above warp W's bins
      const uint4 h4 = reinterpret_cast<const uint4*>(sh->hist)[32 * W + lane];
      const uint32_t s4 = (h4.x + h4.y) + (h4.z + h4.w);
      uint32_t ls = s4;   // keys in warp W's bins >= 4 lane
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t t = __shfl_down_sync(FULL_MASK, ls, o);
        if (lane + o < 32) ls += t;
      }
      const int L = 31 - __clz(__ballot_sync(FULL_MASK, above_w + ls >= kk));
      uint32_t above = above_w + ls - s4;   // keys above bin 4 L + 3 of warp W
      int b = 3;
      if (above + h4.w < kk) {
        above += h4.w;
        b = 2;
        if (above + h4.z < kk) {
          above += h4.z;
          b = 1;
          if (above + h4.y < kk) {
            above += h4.y;
            b = 0;
          }
        }
      }
      const int C = 128 * W + 4 * L + __shfl_sync(FULL_MASK, b, L);
      const uint32_t aboveC = __shfl_sync(FULL_MASK, above, L);
      // the keys of bin C, by their low 4 bits.  A chunk is tested two keys
      // a word first: a 16-bit half of (key >> 4) ^ C is 0 exactly for a key
      // of bin C, and subtracting 1 then sets the half's top bit (the halves
      // hold 11 bits; a borrow from the low half can also set the high
      // half's: a false alarm, which the exact loop rules out)
      const uint32_t CC = (uint32_t)C * 0x10001u;
#pragma unroll
      for (int c = 0; c < NCH; ++c)
        if (have[c]) {
          uint32_t z = 0;
#pragma unroll
          for (int u = 0; u < 4; ++u) z |= (((w[4 * c + u] >> 4) & 0x07FF07FFu) ^ CC) - 0x00010001u;
          if (z & 0x80008000u)
#pragma unroll
            for (int h = 0; h < 8; ++h) {
              const int key = key_at(c, h);
              if ((key >> 4) == C) atomicAdd(&sh->sub[key & 15], 1u);
            }
        }
      if (tail && (int)((xt & 0x7FFFu) >> 4) == C) atomicAdd(&sh->sub[xt & 15u], 1u);
      __syncthreads();
      // T and q, in every warp: the 16 keys of bin C from the top
      const uint32_t sv = lane < 16 ? sh->sub[lane] : 0u;
      uint32_t sfx = sv;   // keys of bin C with key & 15 >= lane
#pragma unroll
      for (int o = 1; o < 16; o <<= 1) {
        const uint32_t t = __shfl_down_sync(FULL_MASK, sfx, o);
        if (lane + o < 16) sfx += t;
      }
      const uint32_t need = kk - aboveC;   // >= 1
      const int bb = 31 - __clz(__ballot_sync(FULL_MASK, lane < 16 && sfx >= need));
      T = 16 * C + bb;
      q = (int)(need - __shfl_sync(FULL_MASK, sfx - sv, bb));   // >= 1
    }
  }
  // per chunk: bits and counts of key > T and key == T, two keys a word:
  // with the sign bit set, (key | 0x8000) - t has bit 15 set exactly when
  // key >= t (0 <= t <= 0x8000: no borrow leaves the half), so t = T + 1
  // gives key > T and t = max(T, 0) key >= T; the words' bits 15 and 31 are
  // then gathered into the chunk's 8-bit masks (bit h: channel h)
  uint32_t gb[NCH], eb[NCH];
  uint32_t p[5] = {0u, 0u, 0u, 0u, 0u};   // gt of chunks 0|1, 2|3, eq 0|1, 2|3, {gt, eq} of the tail
  const uint32_t T1 = (uint32_t)(T + 1) * 0x10001u, T0 = (uint32_t)(T < 0 ? 0 : T) * 0x10001u;
#pragma unroll
  for (int c = 0; c < NCH; ++c) {
    uint32_t g = 0, e = 0;
    if (have[c]) {
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const uint32_t o = w[4 * c + u] | 0x80008000u;
        const uint32_t gw = (o - T1) & 0x80008000u, ew = (o - T0) & ~gw & 0x80008000u;
        g |= gw >> (15 - 2 * u);
        e |= ew >> (15 - 2 * u);
      }
      g = (g | (g >> 15)) & 0xFFu;
      e = (e | (e >> 15)) & 0xFFu;
    }
    gb[c] = g;
    eb[c] = e;
    p[c >> 1] |= (uint32_t)__popc(g) << (16 * (c & 1));
    p[2 + (c >> 1)] |= (uint32_t)__popc(e) << (16 * (c & 1));
  }
  const int tkey = (int)(xt & 0x7FFFu);
  const uint32_t tg = (tail && tkey > T) ? 1u : 0u, te = (tail && tkey == T) ? 1u : 0u;
  p[4] = tg | (te << 16);
  // block exclusive scan of the packed counters (16-bit fields: at most
  // 8 ST_THREADS per field).  Words 1 and 3 (chunks 2 and 3) exist only for
  // NCH > 2 and word 4 only when I % 8 != 0 (block-uniform); the others are
  // zero and not scanned.  Across warps: the exclusive prefix and the total
  // of the warp totals, each one warp reduction.
  const bool ftail = (I & 7) != 0;
  auto live = [&](int f) { return (f & 1) == 0 ? (f < 4 || ftail) : NCH > 2; };
  uint32_t incl[5];
#pragma unroll
  for (int f = 0; f < 5; ++f) incl[f] = live(f) ? warp_inclusive_scan(p[f], lane) : 0u;
  if (lane == 31)
#pragma unroll
    for (int f = 0; f < 5; ++f)
      if (live(f)) tmp[ST_WARPS + 5 * wid + f] = incl[f];
  __syncthreads();
  uint32_t ex[5], tot[5];
#pragma unroll
  for (int f = 0; f < 5; ++f) {
    ex[f] = tot[f] = 0u;
    if (live(f)) {
      const uint32_t v = lane < ST_WARPS ? tmp[ST_WARPS + 5 * lane + f] : 0u;
      ex[f] = __reduce_add_sync(FULL_MASK, lane < wid ? v : 0u) + incl[f] - p[f];
      tot[f] = __reduce_add_sync(FULL_MASK, v);
    }
  }
  auto field = [](uint32_t v, int c) { return (v >> (16 * (c & 1))) & 0xFFFFu; };
  uint32_t GT = (tot[4] & 0xFFFFu), EQ = (tot[4] >> 16);
#pragma unroll
  for (int c = 0; c < 4; ++c) {
    GT += field(tot[c >> 1], c);
    EQ += field(tot[2 + (c >> 1)], c);
  }
  const uint32_t qq = (uint32_t)q;
  const uint32_t K = GT + (EQ < qq ? EQ : qq);
  const uint32_t m = (uint32_t)(run >> 32) & 0xFFFFu, nr = (uint32_t)(run >> 48);
  const uint32_t R0 = K * m / nr, R1 = K * (m + 1) / nr;
  uint32_t gbase = 0, ebase = 0;
#pragma unroll
  for (int c = 0; c < 4; ++c) {
    if (c < NCH) {
      // the chunk's 8 channels, each ranked on its own (no loop-carried
      // find-first-set): kept when key > T, or key == T within the first q
      const uint32_t g0 = gbase + field(ex[c >> 1], c), e0 = ebase + field(ex[2 + (c >> 1)], c);
      const uint32_t gbc = gb[c], ebc = eb[c];
      // the chunk's kept channels take ranks from r0c on, at most 8 of them:
      // only chunks that can reach this CTA's window [R0, R1) are ranked
      // (a few threads of the CTA; the others skip it)
      const uint32_t r0c = g0 + (e0 < qq ? e0 : qq);
      if (r0c < R1 && r0c + 8u > R0) {
#pragma unroll
        for (int h = 0; h < 8; ++h) {
          const uint32_t below = (1u << h) - 1u;
          const uint32_t g = g0 + (uint32_t)__popc(gbc & below), e = e0 + (uint32_t)__popc(ebc & below);
          const bool kept = ((gbc >> h) & 1u) || (((ebc >> h) & 1u) && e < qq);
          const uint32_t r = g + (e < qq ? e : qq);
          if (kept && r >= R0 && r < R1) klist[r - R0] = (uint16_t)(8 * (tid + c * ST_THREADS) + h);
        }
      }
    }
    gbase += field(tot[c >> 1], c);
    ebase += field(tot[2 + (c >> 1)], c);
  }
  if (tg | te) {
    const uint32_t g = gbase + (ex[4] & 0xFFFFu), e = ebase + (ex[4] >> 16);
    if (tg || e < qq) {
      const uint32_t r = g + (e < qq ? e : qq);
      if (r >= R0 && r < R1) klist[r - R0] = (uint16_t)jt;
    }
  }
  __syncthreads();
  return (int)(R1 - R0);
}

}  // namespace duo
