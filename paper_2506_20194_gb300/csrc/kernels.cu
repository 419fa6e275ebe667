// Kernels of libduo (sm_103a): the channel-major packer (§4.1 storage), the
// exact magnitude top-k sparsifier (§3), and the dual-sparse spMspV
// y = W (x ⊙ m^x) (§3) over the bitmask ("CMB") and index ("IDX16")
// formats.  All device code lives in this one translation unit so the
// device status word needs no relocatable device code.
#include <algorithm>
#include <cstdio>
#include <mutex>

#define DUO_STATUS_OWNER
#include "duo_device.cuh"
#include "duo_launch.h"

namespace duo {

// ------------------------------------------------------------------------
// Device properties (cached per device).
// ------------------------------------------------------------------------
cudaError_t dev_props(DevProps* out) {
  static std::mutex mu;
  static DevProps cache[64];
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lk(mu);
  if (cache[dev].nsm == 0) {
    DevProps p;
    e = cudaDeviceGetAttribute(&p.nsm, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    e = cudaDeviceGetAttribute(&p.smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    if (e != cudaSuccess) return e;
    cache[dev] = p;
  }
  *out = cache[dev];
  return cudaSuccess;
}

__host__ __device__ inline size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

// ------------------------------------------------------------------------
// Packing (§4.1: each kept column is stored compressed; column-major
// storage per the footnote of §3).  A CTA loads a 1024-row x 32-channel tile
// of the row-major weight with coalesced loads into shared memory (row pitch
// 34 halves so that the column walk below is bank-conflict free); warp w
// then walks channels w, w+8, ...: for mask word t, lane b tests row 32t+b,
// a ballot gives the word, and popcounts give each value's slot.
// ------------------------------------------------------------------------
constexpr int PACK_THREADS = 256;
constexpr int PACK_PITCH = 34;  // halves per tile row
constexpr size_t PACK_SMEM = (size_t)SEG_ROWS * PACK_PITCH * 2;
constexpr int QT_PITCH = 33;    // uint32 per row of a grid table staged for the scatter
constexpr size_t PACK_QSMEM = PACK_SMEM + (size_t)32 * QT_PITCH * 4;

enum PackMode { PACK_COUNT = 0, PACK_CMB = 1, PACK_IDX16 = 2 };

struct PackArgs {
  const uint16_t* W;
  int64_t O, I, ldw;
  int S;
  uint32_t* cnt_js;          // COUNT: output
  const uint32_t* cnt_js_in; // IDX16: per-segment counts
  const uint32_t* off;       // CMB
  const uint32_t* cnt;       // IDX16
  const uint64_t* colptr;    // IDX16
  const uint32_t* qtab;      // CMB, VB < 16: grid tables
  int G;                     // CMB, VB < 16: input-channel groups
  uint8_t* data;
};

// RTN code of a stored weight w (fp16 bits) on the grid e = {fp16 s, z}
// (§5, weight-only quantisation): clamp(rint(w / s) + z, 0, maxq), the
// quotient in fp64.
__device__ __forceinline__ uint32_t rtn_code(uint16_t w, uint32_t e, int maxq) {
  const double s = (double)__half2float(__ushort_as_half((unsigned short)(e & 0xFFFFu)));
  const double q = rint((double)__half2float(__ushort_as_half(w)) / s) + (double)(e >> 16);
  return (uint32_t)fmin(fmax(q, 0.0), (double)maxq);
}

template <int MODE, int VB>
__global__ void __launch_bounds__(PACK_THREADS) pack_tile_kernel(const PackArgs a) {
  extern __shared__ __align__(16) uint16_t tile[];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t j0 = (int64_t)blockIdx.x * 32;
  const int s = blockIdx.y;
  const int64_t r0 = (int64_t)s * SEG_ROWS;
  const int64_t rows64 = a.O - r0;
  const int rows = rows64 < SEG_ROWS ? (int)rows64 : SEG_ROWS;
  const int64_t ncol64 = a.I - j0;
  const int ncol = ncol64 < 32 ? (int)ncol64 : 32;
  constexpr bool QUANT = MODE == PACK_CMB && VB < 16;
  uint32_t* qs = reinterpret_cast<uint32_t*>(tile + (size_t)SEG_ROWS * PACK_PITCH);
  for (int e = tid; e < SEG_ROWS * 32; e += PACK_THREADS) {
    const int r = e >> 5, c = e & 31;
    uint16_t v = 0;
    if (r < rows && c < ncol) v = a.W[(r0 + r) * a.ldw + j0 + c];
    tile[r * PACK_PITCH + c] = v;
  }
  if (QUANT) {
    // The grid table of (segment s, group j0 / 128): the 32 channels of the
    // tile share it.  Entry 32 b + t (row 32 t + b) goes to qs[b * 33 + t],
    // so the walk below (lane b, word t) reads distinct banks.
    const uint32_t* src = a.qtab + ((size_t)s * a.G + (size_t)(j0 / QGROUP)) * SEG_ROWS;
    for (int e = tid; e < SEG_ROWS; e += PACK_THREADS) qs[(e >> 5) * QT_PITCH + (e & 31)] = src[e];
  }
  __syncthreads();
  const uint32_t lt = (1u << lane) - 1u;
  for (int c = warp; c < ncol; c += PACK_THREADS / 32) {
    const int64_t j = j0 + c;
    uint32_t total = 0, myword = 0;
    uint16_t* vals = nullptr;
    uint8_t* codes = nullptr;
    uint16_t* rowids = nullptr;
    uint32_t pend = 0;   // VB == 4: the code waiting for its byte's high nibble
    if (MODE == PACK_CMB) {
      const uint32_t o = a.off[j * a.S + s];
      vals = reinterpret_cast<uint16_t*>(a.data + (size_t)o * 16 + MASK_BYTES);
      codes = a.data + (size_t)o * 16 + MASK_BYTES;
    } else if (MODE == PACK_IDX16) {
      uint32_t pre = 0;
      for (int s2 = 0; s2 < s; ++s2) pre += a.cnt_js_in[j * a.S + s2];
      const uint32_t n = a.cnt[j];
      uint8_t* blk = a.data + a.colptr[j];
      vals = reinterpret_cast<uint16_t*>(blk) + pre;
      rowids = reinterpret_cast<uint16_t*>(blk + align_up((size_t)2 * n, 16)) + pre;
    }
#pragma unroll 4
    for (int t = 0; t < SEG_WORDS; ++t) {
      const uint16_t v = tile[(32 * t + lane) * PACK_PITCH + c];
      const bool nz = (v & 0x7FFFu) != 0u;
      const uint32_t word = __ballot_sync(FULL_MASK, nz);
      if (MODE == PACK_CMB) {
        if (lane == t) myword = word;
        const uint32_t pos = total + __popc(word & lt);
        if (VB == 16) {
          if (nz) vals[pos] = v;
        } else {
          const uint32_t q = nz ? rtn_code(v, qs[lane * QT_PITCH + t], (1 << VB) - 1) : 0u;
          if (VB == 8) {
            if (nz) codes[pos] = (uint8_t)q;
          } else {
            // Code n goes to byte n / 2, low nibble when n is even.  A lane
            // at an odd position writes its byte with the code before it:
            // the previous set lane's, or the word's carried-over last code.
            const uint32_t below = word & lt;
            const int prev = below ? 31 - __clz(below) : lane;
            const uint32_t qprev = __shfl_sync(FULL_MASK, q, prev);
            if (nz && (pos & 1u)) codes[pos >> 1] = (uint8_t)((below ? qprev : pend) | (q << 4));
            if (word != 0u) pend = __shfl_sync(FULL_MASK, q, 31 - __clz(word));
          }
        }
      } else if (MODE == PACK_IDX16) {
        if (nz) {
          const uint32_t pos = total + __popc(word & lt);
          vals[pos] = v;
          rowids[pos] = (uint16_t)(r0 + 32 * t + lane);
        }
      }
      total += __popc(word);
    }
    if (MODE == PACK_COUNT) {
      if (lane == 0) a.cnt_js[j * a.S + s] = total;
    } else if (MODE == PACK_CMB) {
      const uint32_t o = a.off[j * a.S + s];
      reinterpret_cast<uint32_t*>(a.data + (size_t)o * 16)[lane] = myword;
      if (VB == 4 && (total & 1u) && lane == 0) codes[total >> 1] = (uint8_t)pend;
    }
  }
}

template <int MODE, int VB>
static cudaError_t launch_pack_tiles_t(const PackArgs& a, cudaStream_t st) {
  const dim3 grid((unsigned)((a.I + 31) / 32), (unsigned)a.S);
  const size_t smem = (MODE == PACK_CMB && VB < 16) ? PACK_QSMEM : PACK_SMEM;
  cudaError_t e = cudaFuncSetAttribute(pack_tile_kernel<MODE, VB>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  pack_tile_kernel<MODE, VB><<<grid, PACK_THREADS, smem, st>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_pack_count(const uint16_t* W, int64_t O, int64_t I, int64_t ldw, int S,
                              uint32_t* cnt_js, cudaStream_t st) {
  PackArgs a{};
  a.W = W; a.O = O; a.I = I; a.ldw = ldw; a.S = S; a.cnt_js = cnt_js;
  return launch_pack_tiles_t<PACK_COUNT, 16>(a, st);
}

cudaError_t launch_cmb_scatter(const uint16_t* W, int64_t O, int64_t I, int64_t ldw, int S,
                               int vbits, const uint32_t* table, const uint32_t* off,
                               uint8_t* data, cudaStream_t st) {
  PackArgs a{};
  a.W = W; a.O = O; a.I = I; a.ldw = ldw; a.S = S; a.off = off; a.data = data;
  a.qtab = table;
  a.G = (int)((I + QGROUP - 1) / QGROUP);
  switch (vbits) {
    case 16: return launch_pack_tiles_t<PACK_CMB, 16>(a, st);
    case 8: return launch_pack_tiles_t<PACK_CMB, 8>(a, st);
    case 4: return launch_pack_tiles_t<PACK_CMB, 4>(a, st);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_idx16_scatter(const uint16_t* W, int64_t O, int64_t I, int64_t ldw, int S,
                                 const uint32_t* cnt_js, const uint32_t* cnt,
                                 const uint64_t* colptr, uint8_t* data, cudaStream_t st) {
  PackArgs a{};
  a.W = W; a.O = O; a.I = I; a.ldw = ldw; a.S = S; a.cnt_js_in = cnt_js; a.cnt = cnt;
  a.colptr = colptr; a.data = data;
  return launch_pack_tiles_t<PACK_IDX16, 16>(a, st);
}

// RTN grids (§5, weight-only quantisation with channel-wise RTN, group size
// 128): one warp per (row i, group g), lanes covering four channels each.
// lo = min(0, min w), hi = max(0, max w) over the group's stored weights;
// s = fp16((hi - lo) / maxq) from an fp64 quotient (1 for an empty group,
// 2^-24 if it rounds to 0); z = rint(-lo / s) clamped to [0, maxq].
constexpr int QGRID_THREADS = 256;

__global__ void __launch_bounds__(QGRID_THREADS) quant_grid_kernel(const uint16_t* __restrict__ W,
                                                                    int64_t O, int64_t I, int64_t ldw,
                                                                    int G, int maxq,
                                                                    uint32_t* __restrict__ table) {
  const int lane = threadIdx.x & 31;
  const int64_t wg = (int64_t)blockIdx.x * (QGRID_THREADS / 32) + (threadIdx.x >> 5);
  if (wg >= O * G) return;   // whole warps
  const int64_t i = wg / G;
  const int g = (int)(wg - i * G);
  float lo = 0.f, hi = 0.f;   // fp16 values are exact in fp32
  for (int e = lane; e < QGROUP; e += 32) {
    const int64_t j = (int64_t)g * QGROUP + e;
    if (j < I) {
      const uint16_t b = W[i * ldw + j];
      if (b & 0x7FFFu) {
        const float v = __half2float(__ushort_as_half(b));
        lo = fminf(lo, v);
        hi = fmaxf(hi, v);
      }
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    lo = fminf(lo, __shfl_xor_sync(FULL_MASK, lo, o));
    hi = fmaxf(hi, __shfl_xor_sync(FULL_MASK, hi, o));
  }
  if (lane == 0) {
    uint32_t sb = 0x3C00u;
    if (hi != lo) {
      sb = __half_as_ushort(__double2half(((double)hi - (double)lo) / (double)maxq));
      if (sb == 0u) sb = 1u;
    }
    const double sd = (double)__half2float(__ushort_as_half((unsigned short)sb));
    const double zd = fmin(fmax(rint(-(double)lo / sd), 0.0), (double)maxq);
    const int64_t seg = i / SEG_ROWS, r = i - seg * SEG_ROWS;
    table[((seg * G + g) * 32 + (r & 31)) * 32 + (r >> 5)] = sb | ((uint32_t)zd << 16);
  }
}

cudaError_t launch_quant_grid(const uint16_t* W, int64_t O, int64_t I, int64_t ldw, int S, int bits,
                              uint32_t* table, cudaStream_t st) {
  (void)S;
  if (bits != 8 && bits != 4) return cudaErrorInvalidValue;
  const int64_t G = (I + QGROUP - 1) / QGROUP;
  const int64_t warps = O * G;
  const int64_t blocks = (warps + QGRID_THREADS / 32 - 1) / (QGRID_THREADS / 32);
  if (blocks > 0x7FFFFFFF) return cudaErrorInvalidValue;
  quant_grid_kernel<<<(unsigned)blocks, QGRID_THREADS, 0, st>>>(W, O, I, ldw, (int)G, (1 << bits) - 1,
                                                               table);
  return cudaGetLastError();
}

// Single-CTA chunked exclusive scan (packing is an offline step; one CTA
// walking a few million entries takes well under a millisecond).
constexpr int SCAN_THREADS = 1024;
constexpr int SCAN_PER = 8;

template <typename F, typename G>
__device__ void chunked_scan(int64_t n, F value, G emit, unsigned long long* total_out) {
  __shared__ unsigned long long wsum[32];
  __shared__ unsigned long long carry;
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  if (tid == 0) carry = 0ull;
  __syncthreads();
  for (int64_t base = 0; base < n; base += (int64_t)SCAN_THREADS * SCAN_PER) {
    unsigned long long v[SCAN_PER], s = 0;
#pragma unroll
    for (int q = 0; q < SCAN_PER; ++q) {
      const int64_t i = base + (int64_t)tid * SCAN_PER + q;
      v[q] = i < n ? value(i) : 0ull;
      s += v[q];
    }
    unsigned long long inc = s;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const unsigned long long t = __shfl_up_sync(FULL_MASK, inc, o);
      if (lane >= o) inc += t;
    }
    if (lane == 31) wsum[wid] = inc;
    __syncthreads();
    if (wid == 0) {
      unsigned long long w = wsum[lane];
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const unsigned long long t = __shfl_up_sync(FULL_MASK, w, o);
        if (lane >= o) w += t;
      }
      wsum[lane] = w;
    }
    __syncthreads();
    unsigned long long run = carry + (wid > 0 ? wsum[wid - 1] : 0ull) + inc - s;
#pragma unroll
    for (int q = 0; q < SCAN_PER; ++q) {
      const int64_t i = base + (int64_t)tid * SCAN_PER + q;
      if (i < n) emit(i, run);
      run += v[q];
    }
    __syncthreads();
    if (tid == 0) carry += wsum[31];
    __syncthreads();
  }
  if (tid == 0) *total_out = carry;
}

__global__ void __launch_bounds__(SCAN_THREADS) cmb_offsets_kernel(const uint32_t* cnt_js, int64_t n,
                                                                   int vbits, uint32_t* off,
                                                                   unsigned long long* totals) {
  // record units = (128 + pad16(ceil(cnt * vbits / 8))) / 16 = 8 + ceil(cnt * vbits / 128)
  chunked_scan(
      n, [&](int64_t i) { return 8ull + ((unsigned long long)cnt_js[i] * vbits + 127ull) / 128ull; },
      [&](int64_t i, unsigned long long pre) { off[i] = (uint32_t)pre; }, &totals[0]);
  __syncthreads();
  chunked_scan(
      n, [&](int64_t i) { return (unsigned long long)cnt_js[i]; },
      [&](int64_t, unsigned long long) {}, &totals[1]);
  // largest record non-zero count
  __shared__ uint32_t wmax[SCAN_THREADS / 32];
  uint32_t m = 0;
  for (int64_t i = threadIdx.x; i < n; i += SCAN_THREADS) m = max(m, cnt_js[i]);
  m = __reduce_max_sync(FULL_MASK, m);
  if ((threadIdx.x & 31) == 0) wmax[threadIdx.x >> 5] = m;
  __syncthreads();
  if (threadIdx.x == 0) {
    uint32_t mm = 0;
    for (int w = 0; w < SCAN_THREADS / 32; ++w) mm = max(mm, wmax[w]);
    totals[2] = mm;
    off[n] = (uint32_t)totals[0];
  }
}

cudaError_t launch_cmb_offsets(const uint32_t* cnt_js, int64_t n, int vbits, uint32_t* off,
                               unsigned long long* totals, cudaStream_t st) {
  if (vbits != 16 && vbits != 8 && vbits != 4) return cudaErrorInvalidValue;
  cmb_offsets_kernel<<<1, SCAN_THREADS, 0, st>>>(cnt_js, n, vbits, off, totals);
  return cudaGetLastError();
}

__global__ void __launch_bounds__(SCAN_THREADS) idx16_offsets_kernel(const uint32_t* cnt_js,
                                                                     int64_t I, int S,
                                                                     uint32_t* cnt,
                                                                     uint64_t* colptr,
                                                                     unsigned long long* totals) {
  for (int64_t j = threadIdx.x; j < I; j += SCAN_THREADS) {
    uint32_t c = 0;
    for (int s = 0; s < S; ++s) c += cnt_js[j * S + s];
    cnt[j] = c;
  }
  __syncthreads();
  chunked_scan(
      I, [&](int64_t j) { return 2ull * align_up(2ull * cnt[j], 16ull); },
      [&](int64_t j, unsigned long long pre) { colptr[j] = pre; }, &totals[0]);
  __syncthreads();
  chunked_scan(
      I, [&](int64_t j) { return (unsigned long long)cnt[j]; },
      [&](int64_t, unsigned long long) {}, &totals[1]);
  __syncthreads();
  if (threadIdx.x == 0) colptr[I] = totals[0];
}

cudaError_t launch_idx16_offsets(const uint32_t* cnt_js, int64_t I, int S, uint32_t* cnt,
                                 uint64_t* colptr, unsigned long long* totals, cudaStream_t st) {
  idx16_offsets_kernel<<<1, SCAN_THREADS, 0, st>>>(cnt_js, I, S, cnt, colptr, totals);
  return cudaGetLastError();
}

// ------------------------------------------------------------------------
// Sparsifier (§3): one CTA selects and writes the kept ids and values.
// ------------------------------------------------------------------------
constexpr int SPARSIFY_THREADS = 1024;

struct SelLayout {
  size_t xs, klist, sel, end;
};

// list_entries: room for that many kept-list entries in shared memory (0: none).
__host__ __device__ inline SelLayout sel_layout(int I, size_t base, int list_entries) {
  SelLayout L;
  size_t o = base;
  L.xs = o;    o += align_up(2 * (size_t)I, 64);   // whole 32-channel words
  L.klist = o; o += align_up(2 * (size_t)list_entries, 16);
  L.sel = o;   o += align_up(sizeof(SelShared), 16);
  L.end = o;
  return L;
}

__global__ void __launch_bounds__(SPARSIFY_THREADS) sparsify_kernel(const uint16_t* __restrict__ x,
                                                                    int I, int k,
                                                                    uint16_t* __restrict__ kidx,
                                                                    uint16_t* __restrict__ kval) {
  extern __shared__ __align__(128) uint8_t sm[];
  const SelLayout L = sel_layout(I, 0, 0);
  uint16_t* xs = reinterpret_cast<uint16_t*>(sm + L.xs);
  SelShared* sel = reinterpret_cast<SelShared*>(sm + L.sel);
  load_x_to_smem(xs, x, I);
  select_clear(sel);
  __syncthreads();
  int T, cut;
  select_threshold(xs, I, k, sel, &T, &cut);
  thresh_compact(xs, 0, I, T, cut, kidx, kval, sel->wcnt);
}

cudaError_t launch_sparsify(const uint16_t* x, int I, int k, uint16_t* kidx, uint16_t* kval,
                            cudaStream_t st) {
  const size_t smem = sel_layout(I, 0, 0).end;
  cudaError_t e = cudaFuncSetAttribute(sparsify_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  sparsify_kernel<<<1, SPARSIFY_THREADS, smem, st>>>(x, I, k, kidx, kval);
  return cudaGetLastError();
}

// Threshold mask alone (parity and standalone use): one CTA.
__global__ void __launch_bounds__(SPARSIFY_THREADS) sparsify_threshold_kernel(
    const uint16_t* __restrict__ x, int I, uint32_t T, uint16_t* __restrict__ kidx,
    uint16_t* __restrict__ kval, int* __restrict__ count) {
  extern __shared__ __align__(128) uint8_t sm[];
  const SelLayout L = sel_layout(I, 0, 0);
  uint16_t* xs = reinterpret_cast<uint16_t*>(sm + L.xs);
  SelShared* sel = reinterpret_cast<SelShared*>(sm + L.sel);
  load_x_to_smem(xs, x, I);
  __syncthreads();
  const int n = thresh_compact(xs, 0, I, (int)T, -1, kidx, kval, sel->wcnt);
  if (threadIdx.x == 0) *count = n;
}

cudaError_t launch_sparsify_threshold(const uint16_t* x, int I, uint32_t tau_key, uint16_t* kidx,
                                      uint16_t* kval, int* count, cudaStream_t st) {
  const size_t smem = sel_layout(I, 0, 0).end;
  cudaError_t e = cudaFuncSetAttribute(sparsify_threshold_kernel,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  sparsify_threshold_kernel<<<1, SPARSIFY_THREADS, smem, st>>>(x, I, tau_key & 0x7FFFu, kidx, kval, count);
  return cudaGetLastError();
}

// ------------------------------------------------------------------------
// spMspV over the bitmask format (§3 product; §4.1: only the columns of
// surviving channels are fetched).
//
// Persistent cooperative CTAs, one per SM.  Work items are (product p, row
// segment s, kept rank i), ordered p, s, i; CTA b takes the contiguous item
// range [total*b/G, total*(b+1)/G).
//
// Warp 0 produces: lane l resolves items l, l+32, ... (kept channel id,
// record offset and size; the next PQ-1 items of the lane are resolved ahead
// so their offset loads are in flight) and issues a 1-D bulk copy of each
// record into ring slot v % nslot, signalled on the slot's "full" mbarrier
// with the byte count.  Every slot carries the index of the item it holds
// (tag, written by the producer) and of the item last consumed from it (rel,
// written by the consumer); each side checks the exact index before relying
// on the mbarrier, whose parity cannot tell a fill from one two phases
// earlier.  Slots are as large as the largest record of the
// launch's weights (about 1.3 KB at 50% weight density), so the ring holds
// as many records as the shared memory allows.
//
// Warps 1..NC consume: item v goes to consumer v % NC.  A consumer lane owns
// rows 32*lane .. 32*lane+31 of the current segment in fp32 registers: it
// reads its mask word, finds where its values start with a warp prefix sum
// of popcounts, and walks its bits, multiplying each stored fp16 weight by
// the channel's fp16 activation (exact product, fp32 accumulation).  When a
// segment ends the consumers add their registers into a shared-memory row
// tile (rotated so lanes hit distinct banks) and add the tile to y with
// vector reductions.
//
// y is zeroed by the kernel itself: each CTA clears a slice of the outputs,
// then arrives on a split-phase grid barrier whose completion it checks only
// before its first reduction into y.  The launch is cooperative, so all CTAs
// are co-resident and the barrier cannot deadlock.
// ------------------------------------------------------------------------
constexpr int CMB_NC = 15;   // 16 warps in all: 4 per scheduler, up to 128 registers
constexpr int CMB_THREADS = 32 * (1 + CMB_NC);
constexpr int CMB_MAX_SLOTS = 256;

struct CmbLayout {
  SelLayout sel;
  size_t tile, full, empty, xval, tfull, qtab, ring, total;
};

// quant: room for QNTB grid tables and their mbarriers.
__host__ __device__ inline CmbLayout cmb_layout(int I, bool fused, int list_cap, int nslot,
                                                int slot_bytes, bool quant) {
  CmbLayout L;
  size_t o = 0;
  if (fused) {
    L.sel = sel_layout(I, 0, list_cap);
    o = L.sel.end;
  }
  L.tile = o;  o += 2 * SEG_ROWS * sizeof(float);
  L.full = o;  o += 8 * (size_t)nslot;
  L.empty = o; o += 8 * (size_t)nslot;
  L.xval = o;  o += align_up(4 * (size_t)nslot, 16);
  L.tfull = o; o += quant ? 8 * (size_t)QNTB : 0;
  o = align_up(o, 128);
  L.qtab = o;  o += quant ? (size_t)QNTB * QTAB_BYTES : 0;
  L.ring = o;  o += (size_t)nslot * slot_bytes;
  o += quant ? 16 : 0;   // coded walks read one byte past a lane's codes
  L.total = o;
  return L;
}

__device__ __forceinline__ int tile_index(int r) { return (r & ~31) | ((r + (r >> 5)) & 31); }

// One consumer warp decodes two records of the same segment at once: one
// warp prefix sum serves both masks (16-bit halves) and the two records'
// loads interleave.  Lane owns rows 32*lane + t.
__device__ __forceinline__ void decode_two(const uint8_t* ra, uint16_t xa, const uint8_t* rb,
                                           uint16_t xb, float (&acc)[32], int lane) {
  const uint32_t ma = reinterpret_cast<const uint32_t*>(ra)[lane];
  const uint32_t mb = reinterpret_cast<const uint32_t*>(rb)[lane];
  const uint32_t c = (uint32_t)__popc(ma) | ((uint32_t)__popc(mb) << 16);
  const uint32_t ex = warp_inclusive_scan(c, lane) - c;
  const uint16_t* pa = reinterpret_cast<const uint16_t*>(ra + MASK_BYTES) + (ex & 0xFFFFu);
  const uint16_t* pb = reinterpret_cast<const uint16_t*>(rb + MASK_BYTES) + (ex >> 16);
#pragma unroll
  for (int t = 0; t < 32; ++t) {
    if (ma & (1u << t)) {
      acc[t] = fma_f16_f32(*pa, xa, acc[t]);
      ++pa;
    }
    if (mb & (1u << t)) {
      acc[t] = fma_f16_f32(*pb, xb, acc[t]);
      ++pb;
    }
  }
}

// One consumer warp decodes one record: lane owns rows 32*lane + t.
__device__ __forceinline__ void decode_record(const uint8_t* rec, uint16_t xb, float (&acc)[32],
                                              int lane) {
  const uint32_t m = reinterpret_cast<const uint32_t*>(rec)[lane];
  const uint32_t c = __popc(m);
  const uint32_t incl = warp_inclusive_scan(c, lane);
  const uint16_t* vp = reinterpret_cast<const uint16_t*>(rec + MASK_BYTES) + (incl - c);
#pragma unroll
  for (int t = 0; t < 32; ++t) {
    if (m & (1u << t)) {
      acc[t] = fma_f16_f32(*vp, xb, acc[t]);
      ++vp;
    }
  }
}

// Coded records (§5, weight-only quantisation): as decode_record / decode_two
// with b-bit codes in place of the fp16 values; tab is the record's grid
// table plus lane, so row 32 lane + t's grid is tab[32 t] (conflict-free).
// The lane's codes come through a CodeWalk, (re)loaded every G positions
// at the code index the mask prefix gives (independent loads).
template <int VB>
__device__ __forceinline__ void decode_record_q(const uint8_t* rec, uint16_t xb, const uint32_t* tab,
                                                float (&acc)[32], int lane) {
  constexpr int G = CodeWalk<VB>::G, NG = 32 / G;
  const uint32_t m = reinterpret_cast<const uint32_t*>(rec)[lane];
  const uint32_t c = __popc(m);
  const uint32_t c0 = warp_inclusive_scan(c, lane) - c;
  CodeWalk<VB> w[NG];
#pragma unroll
  for (int g = 0; g < NG; ++g) w[g].load(rec + MASK_BYTES, c0 + (uint32_t)__popc(m & ((1ull << (G * g)) - 1u)));
#pragma unroll
  for (int g = 0; g < NG; ++g)
#pragma unroll
    for (int j = 0; j < G; ++j) {
      const int t = G * g + j;
      const uint32_t bit = (m >> t) & 1u;
      acc[t] = q_fma_sel(bit, w[g].at(), tab[32 * t], xb, acc[t]);
      w[g].step(bit);
    }
}

// Two records of one group (one table) at once: one warp prefix sum serves
// both masks (16-bit halves) and the two records' loads interleave.
template <int VB>
__device__ __forceinline__ void decode_two_q(const uint8_t* ra, uint16_t xa, const uint8_t* rb, uint16_t xb,
                                             const uint32_t* tab, float (&acc)[32], int lane) {
  constexpr int G = CodeWalk<VB>::G, NG = 32 / G;
  const uint32_t ma = reinterpret_cast<const uint32_t*>(ra)[lane];
  const uint32_t mb = reinterpret_cast<const uint32_t*>(rb)[lane];
  const uint32_t c = (uint32_t)__popc(ma) | ((uint32_t)__popc(mb) << 16);
  const uint32_t ex = warp_inclusive_scan(c, lane) - c;
  const uint32_t ca = ex & 0xFFFFu, cb = ex >> 16;
  CodeWalk<VB> wa[NG], wb[NG];
#pragma unroll
  for (int g = 0; g < NG; ++g) {
    const uint32_t below = (uint32_t)((1ull << (G * g)) - 1u);
    wa[g].load(ra + MASK_BYTES, ca + (uint32_t)__popc(ma & below));
    wb[g].load(rb + MASK_BYTES, cb + (uint32_t)__popc(mb & below));
  }
#pragma unroll
  for (int g = 0; g < NG; ++g)
#pragma unroll
    for (int j = 0; j < G; ++j) {
      const int t = G * g + j;
      const uint32_t ba = (ma >> t) & 1u, bb = (mb >> t) & 1u;
      const uint32_t e = tab[32 * t];
      acc[t] = q_fma_sel(ba, wa[g].at(), e, xa, acc[t]);
      acc[t] = q_fma_sel(bb, wb[g].at(), e, xb, acc[t]);
      wa[g].step(ba);
      wb[g].step(bb);
    }
}

// Item cursor: (product p, segment s, kept rank i) of a linear item index.
struct ItemCursor {
  int p, s, i;
  __device__ __forceinline__ void set(const CmbArgs& a, uint32_t u) {   // item counts < 2^31
    const uint32_t k = (uint32_t)a.k;
    uint32_t base = 0;
    p = 0;
    while (p < a.np - 1 && u >= base + (uint32_t)a.p[p].S * k) {
      base += (uint32_t)a.p[p].S * k;
      ++p;
    }
    const uint32_t rem = u - base;
    s = (int)(rem / k);
    i = (int)(rem - (uint32_t)s * k);
  }
  __device__ __forceinline__ void advance(const CmbArgs& a, int n) {
    i += n;
    while (i >= a.k) {
      i -= a.k;
      if (++s == a.p[p].S) {
        s = 0;
        if (p < a.np - 1) ++p;
      }
    }
  }
};

// Ring position of an item: slot = v % nslot, fill number n = v / nslot.
struct SlotCursor {
  int slot, n;
  __device__ __forceinline__ void set(int v, int nslot) { n = v / nslot; slot = v - n * nslot; }
  __device__ __forceinline__ void advance(int by, int nslot) {   // by <= nslot
    slot += by;
    if (slot >= nslot) { slot -= nslot; ++n; }
  }
};

// Where an item's record lives.  The two offset loads stay in flight until
// the item is issued, PQ rounds later: nothing here reads their results, so
// the producer never waits a memory latency per round.
struct Resolved {
  const uint8_t* data;   // the product's packed data
  uint32_t o0, o1;       // off[j * S + s], off[j * S + s + 1] (16-byte units)
  uint16_t xb;
  int g;                 // input-channel group j / 128 (quantised formats)
  bool bad_j;            // channel id out of range
  __device__ __forceinline__ uint32_t bytes() const { return (o1 - o0) * 16u; }
  __device__ __forceinline__ bool bad(int slot_bytes) const {
    const uint32_t b = bytes();
    return bad_j || o1 < o0 || b < (uint32_t)MASK_BYTES || b > (uint32_t)slot_bytes;
  }
};

template <bool FUSED>
__device__ __forceinline__ Resolved resolve_item(const CmbArgs& a, const ItemCursor& c,
                                                 const uint16_t* klist, const uint16_t* xs, int r0) {
  Resolved r;
  int j;
  if (FUSED) {
    const int d = c.i >= r0 ? c.i - r0 : c.i + a.k - r0;   // position in this CTA's list window
    j = klist[d];
    r.xb = xs[j];
  } else {
    j = __ldg(a.kidx + c.i);
    r.xb = __ldg(a.kval + c.i);
  }
  r.bad_j = j >= a.I;
  if (r.bad_j) j = 0;   // keep the loads below in bounds; the item is rejected
  r.g = j / QGROUP;
  const CmbProb& P = a.p[c.p];
  const int64_t ri = (int64_t)j * P.S + c.s;
  r.o0 = __ldg(P.off + ri);
  r.o1 = __ldg(P.off + ri + 1);
  r.data = P.data;
  return r;
}

// Whether consumers may decode two records at once (one scan for both
// masks, interleaved loads) when the ring allows it.  Measured on the 7B
// layer (us per layer, with / without): fp16 64.5 / 66.4, 8-bit codes
// 85.4 / 86.7, 4-bit codes 103.3 / 101.4 -- so 4-bit launches decode one
// record at a time (and their kernels carry no pair code).
#ifndef CMB_PAIRS
#define CMB_PAIRS 1
#endif

// The run of this CTA: the r with run_cta[r] <= blockIdx.x < run_cta[r + 1]
// (run_cta ascending from 0), by binary search over the kernel parameters.
__device__ __forceinline__ int run_of_cta(const CmbArgs& a) {
  int lo = 0, hi = a.nruns - 1;   // the answer lies in [lo, hi]
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if ((unsigned)a.run_cta[mid] <= blockIdx.x) lo = mid;
    else hi = mid - 1;
  }
  return lo;
}

template <int MODE, int VB>
__global__ void __launch_bounds__(CMB_THREADS, 1) cmb_spmspv_kernel(const CmbArgs a) {
  constexpr bool FUSED = MODE != CMB_LISTED;   // the kernel builds its own kept list
  constexpr bool QUANT = VB < 16;              // b-bit codes + grid tables (§5)
  extern __shared__ __align__(128) uint8_t sm[];
  __shared__ volatile int abort_flag;
  __shared__ int grid_open;   // 1 once every CTA has zeroed its slice of y
  __shared__ int cons[CMB_NC];    // QUANT: items each consumer has released
  __shared__ int tfirst[QNTB];    // QUANT: first item of each table in flight
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int nslot = a.nslot, slot_bytes = a.slot_bytes;
  const CmbLayout L = cmb_layout(a.I, FUSED, a.list_cap, nslot, slot_bytes, QUANT);
  float* tile = reinterpret_cast<float*>(sm + L.tile);
  uint64_t* full = reinterpret_cast<uint64_t*>(sm + L.full);
  uint64_t* empty = reinterpret_cast<uint64_t*>(sm + L.empty);
  uint32_t* xval = reinterpret_cast<uint32_t*>(sm + L.xval);
  uint8_t* ring = sm + L.ring;
  uint64_t* tfull = reinterpret_cast<uint64_t*>(sm + L.tfull);
  uint32_t* qt = reinterpret_cast<uint32_t*>(sm + L.qtab);
  uint16_t* xs = FUSED ? reinterpret_cast<uint16_t*>(sm + L.sel.xs) : nullptr;
  uint16_t* klist = FUSED ? reinterpret_cast<uint16_t*>(sm + L.sel.klist) : nullptr;
  SelShared* sel = FUSED ? reinterpret_cast<SelShared*>(sm + L.sel.sel) : nullptr;

  // ---- prologue ----
  // Work that touches nothing the previous kernel of the stream may write
  // runs before griddep_wait(), overlapping that kernel's last CTAs: ring
  // mbarriers, shared-memory state, and an L2 warm-up of this CTA's share of
  // every offset table (a hint only).
  griddep_launch_dependents();
  for (int i = tid; i < nslot; i += CMB_THREADS) {
    mbar_init(&full[i], 1);
    mbar_init(&empty[i], 1);
  }
  if (QUANT && tid < QNTB) mbar_init(&tfull[tid], 1);
  if (QUANT && tid < CMB_NC) cons[tid] = 0;
  fence_mbar_init();
  if (tid == 0) {
    abort_flag = 0;
    grid_open = 0;
  }
  if (warp < a.np && lane == 0) {   // one warp per product (its parameters: one
                                    // uniform load each), slices from the launcher
    const CmbProb& P = a.p[warp];
    const uint32_t lo = P.pf_chunk * blockIdx.x;
    const uint32_t hi = lo + P.pf_chunk < P.pf_bytes ? lo + P.pf_chunk : P.pf_bytes;
    if (hi > lo) prefetch_l2(reinterpret_cast<const uint8_t*>(P.off) + lo, hi - lo);
  }
  for (int i = tid; i < SEG_ROWS / 2; i += CMB_THREADS)   // 2 SEG_ROWS floats, 16 B a store
    reinterpret_cast<float4*>(tile)[i] = make_float4(0.f, 0.f, 0.f, 0.f);
  if (MODE == CMB_TOPK) select_clear(sel);
  // x into L2 while the previous kernel finishes: a prefetch reads nothing
  // into this CTA, and L2 is coherent, so a later write to x by that kernel
  // is what the loads after the wait see.
  if (FUSED && tid < (2 * a.I + 127) / 128)
    prefetch_line_l2(reinterpret_cast<const uint8_t*>(a.x) + 128 * tid);
  // This CTA's run identity (a kernel parameter, not the previous kernel's
  // output): read before the wait so that its cold parameter-cache miss
  // overlaps the wait.
  const uint64_t cinfo = (FUSED && a.cta_info_ok) ? a.cta_info[blockIdx.x] : 0ull;
  // Inputs, y and the grid barrier words may be the previous kernel's.
  griddep_wait();
  // Fused modes: x and the selection straight from registers when x fits
  // (select_window), else through shared memory.
  const bool regs = FUSED && select_window_ok<CMB_THREADS>(a.x, a.I);
  if (FUSED && !regs) load_x_to_smem(xs, a.x, a.I);
  uint32_t u0, u1;   // this CTA's items (32-bit: the launcher keeps counts < 2^31)
  int r0 = 0;        // kept rank of its first item
  int pr = 0, sr = 0;   // fused modes: run (product, segment)
  // Fused modes: the run identity p << 8 | s << 10 | m << 32 | n << 48 (this
  // CTA is the m-th of the n CTAs of product p's segment s).  Every CTA of a
  // run takes an equal share of the run's kept channels in index order
  // (select_window), or, on the shared-memory path, the kept channels of its
  // own channel range.  The launcher's word is decoded only where it is
  // used, so that its parameter load overlaps the loads of x.
  uint64_t ci = cinfo;
  if (FUSED) {
    if (!a.cta_info_ok) {
      const int r = run_of_cta(a);
      int p = 0, sg = r;
      while (p < a.np - 1 && sg >= a.p[p].S) sg -= a.p[p++].S;
      ci = (uint64_t)p << 8 | (uint64_t)sg << 10 | (uint64_t)(blockIdx.x - a.run_cta[r]) << 32 |
           (uint64_t)(a.run_cta[r + 1] - a.run_cta[r]) << 48;
    }
    u0 = u1 = 0;
  } else if (a.nruns > 0) {
    const int r = run_of_cta(a);
    const uint32_t n = a.run_cta[r + 1] - a.run_cta[r], m = blockIdx.x - a.run_cta[r];
    const uint32_t k = (uint32_t)a.k;   // k * m < 2^32: k <= 65535, m < 1024
    u0 = (uint32_t)r * k + k * m / n;
    u1 = (uint32_t)r * k + k * (m + 1) / n;
    r0 = (int)(k * m / n);
  } else {
    uint32_t total = 0;
    for (int p = 0; p < a.np; ++p) total += (uint32_t)a.p[p].S * (uint32_t)a.k;
    u0 = (uint32_t)((uint64_t)total * blockIdx.x / gridDim.x);
    u1 = (uint32_t)((uint64_t)total * (blockIdx.x + 1) / gridDim.x);
  }
  __syncthreads();
  if (FUSED && regs) {
    constexpr bool TK = MODE == CMB_TOPK;
    const int nch = ((a.I >> 3) + CMB_THREADS - 1) / CMB_THREADS;
    const int tk = (int)a.tau_key;
    int nw;
    if (nch <= 1) nw = select_window<TK, 1, CMB_THREADS>(a.x, a.I, a.k, tk, xs, sel, ci, klist, sel->tmp);
    else if (nch == 2) nw = select_window<TK, 2, CMB_THREADS>(a.x, a.I, a.k, tk, xs, sel, ci, klist, sel->tmp);
    else if (nch == 3) nw = select_window<TK, 3, CMB_THREADS>(a.x, a.I, a.k, tk, xs, sel, ci, klist, sel->tmp);
    else nw = select_window<TK, 4, CMB_THREADS>(a.x, a.I, a.k, tk, xs, sel, ci, klist, sel->tmp);
    u1 = (uint32_t)nw;
  } else if (FUSED) {
    // The kept set as a threshold (top-k: computed here; threshold mask:
    // given), then this CTA's kept channels of its range, numbered from 0.
    const uint32_t rm = (uint32_t)(ci >> 32) & 0xFFFFu, rn = (uint32_t)(ci >> 48);
    const int c0 = (int)((uint32_t)a.I * rm / rn), c1 = (int)((uint32_t)a.I * (rm + 1) / rn);
    int T = (int)a.tau_key, cut = -1;
    if (MODE == CMB_TOPK) select_threshold(xs, a.I, a.k, sel, &T, &cut);
    u1 = (uint32_t)thresh_compact(xs, c0, c1, T, cut, klist, nullptr, sel->wcnt);
  }
  if (FUSED) {
    pr = (int)((ci >> 8) & 3u);
    sr = (int)((ci >> 10) & 0x3FFFFFu);
  }
  const int nv = (int)(u1 - u0);
  // Generation of the grid barrier before this CTA arrives on it: read after
  // the selection (no warp has arrived yet: consumers arrive after the role
  // split) and used only once every copy is issued, so its round trip is
  // off the path.
  unsigned int gen0 = 0;
  if (tid == 0) gen0 = ld_relaxed_gpu(a.bar + 1);
  // An item cursor at item u of this CTA.
  auto cursor_at = [&](uint32_t u) {
    ItemCursor c;
    if (FUSED) {
      c.p = pr;
      c.s = sr;
      c.i = (int)u;   // u < nv <= k (top-k) or a.k above any count: advance() never wraps
    } else {
      c.set(a, u);
    }
    return c;
  };

  if (warp == 0) {
    // ---------------- producer ----------------
    constexpr int PQ = 2;   // rounds queued ahead: deeper queues only add code and start-up work
    const uint64_t pol = policy_evict_first();
    int last_v = -1;
    bool stop = false;
    ItemCursor cur = cursor_at(u0 + lane);
    SlotCursor sc;
    sc.set(lane, nslot);
    Resolved q[PQ] = {};
#pragma unroll
    for (int d = 0; d < PQ; ++d) {
      if (lane + 32 * d < nv) {
        if (d > 0) cur.advance(a, 32);
        q[d] = resolve_item<FUSED>(a, cur, klist, xs, r0);
      }
    }
    // Coded formats: the grid tables of the CTA's run, group gA on, go
    // through QNTB buffers in order.  Table n (group gA + n) is armed once
    // every item of a group <= gA + n - QNTB has been released, and an item
    // is issued only after its table is armed, so a consumer that waits for
    // table n finds phase n - QNTB of its buffer complete (exact parity).
    int tarm = 0, last_seq = 0, gA = 0;
    const uint32_t* qsrc = nullptr;
    if (QUANT) {
      const ItemCursor ci = cursor_at(u0);   // a CTA of a coded launch serves one run
      gA = FUSED ? (nv > 0 ? klist[0] / QGROUP : 0) : __shfl_sync(FULL_MASK, q[0].g, 0);
      const CmbProb& P = a.p[ci.p];
      qsrc = P.qtab + ((size_t)ci.s * P.G + gA) * SEG_ROWS;
    }
    // Rounds of 32 items: round R issues items 32 R .. 32 R + 31, lane l the
    // item 32 R + l.  A __syncwarp opens every round, so the rounds run in
    // lockstep and items are issued in increasing round order.
    for (int R0 = 0; R0 < nv; R0 += 32 * PQ) {
#pragma unroll
      for (int d = 0; d < PQ; ++d) {
        __syncwarp();
        stop = __any_sync(FULL_MASK, stop || abort_flag != 0);
        if (stop) break;
        const int v = R0 + 32 * d + lane;
        if (!QUANT) {
          if (v >= nv) continue;
          const Resolved r = q[d];
          if (r.bad(slot_bytes)) {
            atomicOr(a.status, STATUS_FORMAT);
            abort_flag = 1;
            stop = true;
            continue;
          }
          if (v + 32 * PQ < nv) {                 // refill: this lane's item v + 32*PQ
            cur.advance(a, 32);
            q[d] = resolve_item<FUSED>(a, cur, klist, xs, r0);
          }
          // Fill n of a slot waits until fill n - 1 has been consumed.  Fill
          // n - 1 was issued in an earlier round (nslot >= 32), after fill
          // n - 2 had been released, so the "empty" phase parity is exact.
          if (sc.n > 0 && !mbar_wait_bounded(&empty[sc.slot], (uint32_t)((sc.n - 1) & 1), &abort_flag, a.status, a.wait_ns)) {
            stop = true;
            continue;
          }
          xval[sc.slot] = r.xb;
          mbar_arrive_expect_tx(&full[sc.slot], r.bytes());
          bulk_g2s(ring + (size_t)sc.slot * slot_bytes, r.data + (size_t)r.o0 * 16, r.bytes(),
                   &full[sc.slot], pol);
          last_v = v;
          sc.advance(32, nslot);
        } else {
          bool pend = v < nv;
          const Resolved r = q[d];
          int seq = 0;
          if (pend) {
            if (r.bad(slot_bytes)) {
              atomicOr(a.status, STATUS_FORMAT);
              abort_flag = 1;
              stop = true;
              pend = false;
            }
            if (v + 32 * PQ < nv) {
              cur.advance(a, 32);
              q[d] = resolve_item<FUSED>(a, cur, klist, xs, r0);
            }
            seq = r.g - gA;
          }
          // Groups must not decrease along the items (pending lanes are a
          // prefix of the warp); a kept list out of group order is rejected.
          const int prev = __shfl_up_sync(FULL_MASK, seq, 1);
          if (pend && (seq < 0 || seq < (lane == 0 ? last_seq : prev))) {
            atomicOr(a.status, STATUS_FORMAT);
            abort_flag = 1;
            stop = true;
            pend = false;
          }
          last_seq = max(last_seq, __reduce_max_sync(FULL_MASK, pend ? seq : 0));
          while (true) {
            if (pend && seq < tarm) {   // table armed: issue
              if (sc.n > 0 &&
                  !mbar_wait_bounded(&empty[sc.slot], (uint32_t)((sc.n - 1) & 1), &abort_flag, a.status, a.wait_ns)) {
                stop = true;
              } else {
                xval[sc.slot] = (uint32_t)r.xb | ((uint32_t)seq << 16);
                mbar_arrive_expect_tx(&full[sc.slot], r.bytes());
                bulk_g2s(ring + (size_t)sc.slot * slot_bytes, r.data + (size_t)r.o0 * 16, r.bytes(),
                         &full[sc.slot], pol);
                last_v = v;
              }
              pend = false;
            }
            const uint32_t pm = __ballot_sync(FULL_MASK, pend);
            stop = __any_sync(FULL_MASK, stop);
            if (pm == 0u || stop) break;
            // Arm table tarm.  Every item of a lower table is issued; the
            // first item of table >= tarm is the lowest pending lane's.
            const int b = tarm % QNTB;
            bool ok = true;
            if (tarm >= QNTB) {
              // Its buffer's previous load (table tarm - QNTB) has landed ...
              if (lane == 0) ok = mbar_wait_bounded(&tfull[b], (uint32_t)((tarm / QNTB - 1) & 1), &abort_flag, a.status, a.wait_ns);
              ok = __shfl_sync(FULL_MASK, ok, 0);
              // ... and every item before the first of table tarm - QNTB + 1
              // is released: lane c checks consumer c's count.
              const int E = tfirst[(tarm + 1) % QNTB] - 1;
              const int need = (lane < CMB_NC && E >= lane) ? (E - lane) / CMB_NC + 1 : 0;
              const int* cw = &cons[lane < CMB_NC ? lane : 0];
              const uint64_t t0 = globaltimer_ns();
              while (ok && !__all_sync(FULL_MASK, ld_acquire_cta_shared(cw) >= need)) {
                const bool late = globaltimer_ns() - t0 > a.wait_ns;
                if (__any_sync(FULL_MASK, late || abort_flag != 0)) {
                  if (lane == 0 && late) {
                    atomicOr(a.status, STATUS_TIMEOUT);
                    abort_flag = 1;
                  }
                  ok = false;
                }
                __nanosleep(32);
              }
            }
            if (!ok) {
              stop = true;
              break;
            }
            if (lane == 0) {
              tfirst[b] = R0 + 32 * d + __ffs(pm) - 1;
              mbar_arrive_expect_tx(&tfull[b], QTAB_BYTES);
              bulk_g2s(qt + (size_t)b * SEG_ROWS, qsrc + (size_t)tarm * SEG_ROWS, QTAB_BYTES, &tfull[b],
                       pol);
            }
            __syncwarp();
            ++tarm;
          }
          sc.advance(32, nslot);
        }
      }
      if (stop) break;
    }
    // Every copy is issued: wait here, off the consumers' path, for the grid
    // barrier, and tell the consumers through shared memory.
    if (lane == 0) {
      const uint64_t t0 = globaltimer_ns();
      while (ld_acquire_gpu(a.bar + 1) == gen0) {
        __nanosleep(64);
        if (globaltimer_ns() - t0 > a.wait_ns) {
          atomicOr(a.status, STATUS_TIMEOUT);
          abort_flag = 1;
          break;
        }
      }
      st_release_cta_shared(&grid_open, 1);
    }
    if (abort_flag) {
      // Let this lane's copies still in flight land before the CTA exits.
      for (int v = last_v; v >= 0 && v > last_v - nslot; v -= 32) {
        SlotCursor w;
        w.set(v, nslot);
        mbar_wait_limited(&full[w.slot], (uint32_t)(w.n & 1), a.status, a.wait_ns);
      }
    }
    if (QUANT && lane == 0) {
      // A table no consumer waited on (a group without kept channels) may
      // still be landing: wait for the last QNTB before the CTA exits.
      for (int t = tarm > QNTB ? tarm - QNTB : 0; t < tarm; ++t)
        mbar_wait_limited(&tfull[t % QNTB], (uint32_t)((t / QNTB) & 1), a.status, a.wait_ns);
    }
  } else {
    // ---------------- consumers ----------------
    const int c = warp - 1;
    const int ctid = tid - 32;
    // Zero this CTA's slice of the outputs and arrive on the grid barrier:
    // done here, off the selection's path, while the first records are in
    // flight.  The named barrier orders every consumer's stores before
    // consumer 0's release.
    {
      int64_t ytot = 0;
      for (int p = 0; p < a.np; ++p) ytot += a.p[p].O;
      const int64_t z0 = ytot * blockIdx.x / gridDim.x, z1 = ytot * (blockIdx.x + 1) / gridDim.x;
      int64_t base = 0;
      for (int p = 0; p < a.np; ++p) {
        const int64_t lo = z0 > base ? z0 : base;
        const int64_t hi = z1 < base + a.p[p].O ? z1 : base + a.p[p].O;
        for (int64_t r = lo + ctid; r < hi; r += CMB_NC * 32) a.p[p].y[r - base] = 0.f;
        base += a.p[p].O;
      }
    }
    named_bar_sync(1, CMB_NC * 32);
    unsigned int gen0c = 0;
    if (ctid == 0) {
      gen0c = ld_relaxed_gpu(a.bar + 1);
      if (atom_add_acq_rel_gpu(a.bar, 1u) == gridDim.x - 1) {   // last arriver opens it
        a.bar[0] = 0u;
        red_add_release_gpu(a.bar + 1, 1u);
      }
    }
    float acc[32];
    // Item v sits in slot v % nslot.  nslot is a multiple of CMB_NC, so a
    // slot only ever holds items of this consumer, which it takes in
    // increasing order and releases before waiting on any item nslot later
    // (group * CMB_NC <= nslot): when it waits for fill n, fill n - 1 is
    // consumed and fill n + 1 not yet issued, so the "full" parity is exact.
    auto wait_item = [&](const SlotCursor& q) -> bool {
      return mbar_wait_bounded(&full[q.slot], (uint32_t)(q.n & 1), &abort_flag, a.status, a.wait_ns);
    };
    auto release = [&](const SlotCursor& q) { mbar_arrive(&empty[q.slot]); };
    // Coded formats: the grid table of an item's group (its table number is
    // in the slot's xval word), waited for once per table; and the count of
    // released items, which tells the producer when a table buffer is free.
    // (Copying the group's grid into 32 registers per lane measured no faster
    // than reading it from shared memory per row.)
    int ncons = 0, cur_seq = -1;
    const uint32_t* tcur = nullptr;
    auto table_for = [&](uint32_t seq) -> const uint32_t* {
      if ((int)seq != cur_seq) {
        if (!mbar_wait_bounded(&tfull[seq % QNTB], (seq / QNTB) & 1u, &abort_flag, a.status, a.wait_ns)) return nullptr;
        cur_seq = (int)seq;
        tcur = qt + (size_t)(seq % QNTB) * SEG_ROWS + lane;
      }
      return tcur;
    };
    auto released = [&](int n) {   // lane 0, after release()
      ncons += n;
      st_release_cta_shared(&cons[c], ncons);
    };
    // One coded item, decoded and released before anything else is waited for.
    auto single_q = [&](const SlotCursor& q, bool& any) {
      if constexpr (QUANT) {
        if (!abort_flag && wait_item(q)) {
          const uint32_t xv = xval[q.slot];
          const uint32_t* tb = table_for(xv >> 16);
          if (tb != nullptr) {
            decode_record_q<VB>(ring + (size_t)q.slot * slot_bytes, (uint16_t)xv, tb, acc, lane);
            any = true;
          }
        }
      }
      __syncwarp();
      if (lane == 0) {
        release(q);
        released(1);
      }
    };
    // The ring can hold every consumer's partial rows for the final flush.
    const bool scratch_ok = (size_t)nslot * slot_bytes >= (size_t)CMB_NC * SEG_ROWS * sizeof(float);
    uint32_t u = u0;
    int piece = 0;
    while (u < u1) {
      const ItemCursor pc = cursor_at(u);
      const uint32_t seg_end = u + (uint32_t)(a.k - pc.i);   // end of this (p, s) run
      const uint32_t pend = seg_end < u1 ? seg_end : u1;
      const int va = (int)(u - u0), vb = (int)(pend - u0);
#pragma unroll
      for (int t = 0; t < 32; ++t) acc[t] = 0.f;
      bool any = false;
      int v = va + ((c - va % CMB_NC) % CMB_NC + CMB_NC) % CMB_NC;
      // this consumer's items in pairs, then alone
      SlotCursor sc, sc2;
      sc.set(v, nslot);
      if (CMB_PAIRS && VB != 4 && a.group >= 2) {
        sc2.set(v + CMB_NC, nslot);
        for (; v + CMB_NC < vb; v += 2 * CMB_NC) {   // pairs
          if constexpr (!QUANT) {
            if (!abort_flag && wait_item(sc) && wait_item(sc2)) {
              decode_two(ring + (size_t)sc.slot * slot_bytes, (uint16_t)xval[sc.slot],
                         ring + (size_t)sc2.slot * slot_bytes, (uint16_t)xval[sc2.slot], acc, lane);
              any = true;
            }
            __syncwarp();
            if (lane == 0) {
              release(sc);
              release(sc2);
            }
          } else if (FUSED && klist[v] / QGROUP == klist[v + CMB_NC] / QGROUP) {
            // Same group, same table: holding the first item while waiting
            // for the second never holds up the arming of a table.
            if (!abort_flag && wait_item(sc) && wait_item(sc2)) {
              const uint32_t xa = xval[sc.slot], xb2 = xval[sc2.slot];
              const uint32_t* tb = table_for(xa >> 16);
              if (tb != nullptr) {
                decode_two_q<VB>(ring + (size_t)sc.slot * slot_bytes, (uint16_t)xa,
                                 ring + (size_t)sc2.slot * slot_bytes, (uint16_t)xb2, tb, acc, lane);
                any = true;
              }
            }
            __syncwarp();
            if (lane == 0) {
              release(sc);
              release(sc2);
              released(2);
            }
          } else {
            single_q(sc, any);
            single_q(sc2, any);
          }
          sc.advance(2 * CMB_NC, nslot);
          sc2.advance(2 * CMB_NC, nslot);
        }
      }
      for (; v < vb; v += CMB_NC) {   // singles
        if constexpr (!QUANT) {
          if (!abort_flag && wait_item(sc)) {
            decode_record(ring + (size_t)sc.slot * slot_bytes, (uint16_t)xval[sc.slot], acc, lane);
            any = true;
          }
          __syncwarp();
          if (lane == 0) release(sc);
        } else {
          single_q(sc, any);
        }
        sc.advance(CMB_NC, nslot);
      }
      const CmbProb& P = a.p[pc.p];
      const int rows = min(SEG_ROWS, P.O - pc.s * SEG_ROWS);
      float* yb = P.y + (size_t)pc.s * SEG_ROWS;
      // First reduction into y: every CTA must have zeroed its slice.  The
      // producer, once it has issued every copy, waits for the grid barrier
      // and sets grid_open; a flush that comes earlier polls the barrier
      // itself (it must not wait for the producer, which may be waiting for
      // this flush's consumers to free slots).
      auto wait_grid = [&]() {
        if (ld_acquire_cta_shared(&grid_open) == 1) return;
        const uint64_t t0 = globaltimer_ns();
        while (ld_acquire_gpu(a.bar + 1) == gen0c) {
          if (ld_acquire_cta_shared(&grid_open) == 1) return;
          __nanosleep(64);
          if (globaltimer_ns() - t0 > a.wait_ns) {
            atomicOr(a.status, STATUS_TIMEOUT);
            abort_flag = 1;
            return;
          }
        }
      };
      auto add_rows = [&](int g, const float (&vv)[4]) {
        if (4 * g + 3 < rows) {
          red_add_v4(yb + 4 * g, vv[0], vv[1], vv[2], vv[3]);
        } else {
          for (int e = 0; e < 4 && 4 * g + e < rows; ++e) atomicAdd(yb + 4 * g + e, vv[e]);
        }
      };
      if (pend == u1 && scratch_ok) {
        // This CTA's last piece: once every consumer passes the barrier all
        // items are consumed and no copy is in flight, so the ring is free.
        // Each consumer stores its partial rows to its own SEG_ROWS floats
        // of it, then the partials are summed four rows at a time, with no
        // shared-memory atomics.  Rows 32 L + 4 i .. + 3 sit in 16-byte chunk
        // (i + L) % 8 of block L, so both the stores and the loads of eight
        // consecutive lanes hit eight different bank groups.
        named_bar_sync(1, CMB_NC * 32);
        float4* mine = reinterpret_cast<float4*>(ring) + (size_t)c * (SEG_ROWS / 4);
#pragma unroll
        for (int i = 0; i < 8; ++i)
          mine[8 * lane + ((i + lane) & 7)] =
              make_float4(acc[4 * i], acc[4 * i + 1], acc[4 * i + 2], acc[4 * i + 3]);
        if (piece == 0 && ctid == 0) wait_grid();
        named_bar_sync(1, CMB_NC * 32);
        const float4* part = reinterpret_cast<const float4*>(ring);
        for (int g = ctid; 4 * g < rows; g += CMB_NC * 32) {
          const int at = 8 * (g >> 3) + (((g & 7) + (g >> 3)) & 7);
          float vv[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
          for (int w = 0; w < CMB_NC; ++w) {
            const float4 q4 = part[(size_t)w * (SEG_ROWS / 4) + at];
            vv[0] += q4.x; vv[1] += q4.y; vv[2] += q4.z; vv[3] += q4.w;
          }
          add_rows(g, vv);
        }
      } else {
        float* tb = tile + (piece & 1) * SEG_ROWS;
        if (any) {
#pragma unroll
          for (int t = 0; t < 32; ++t) atomicAdd(&tb[32 * lane + ((t + lane) & 31)], acc[t]);
        }
        if (piece == 0 && ctid == 0) wait_grid();
        named_bar_sync(1, CMB_NC * 32);
        for (int g = ctid; 4 * g < rows; g += CMB_NC * 32) {
          float vv[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const int r = 4 * g + e;
            if (r < rows) {
              const int ix = tile_index(r);
              vv[e] = tb[ix];
              tb[ix] = 0.f;
            } else {
              vv[e] = 0.f;
            }
          }
          add_rows(g, vv);
        }
      }
      ++piece;
      u = pend;
    }
  }
}

// Host: whole CTAs for each (product, segment) run of a launch (runs in
// product order, at most kMaxRuns, at most grid of them) into n, greedily in
// proportion to each run's estimated cost.  A run's cost is its k records,
// each one warp's walk over 1024 rows whatever the segment holds (a 768-row
// record measured 0.99 of a full one in the stream), plus its bytes: a short
// last segment (13824 rows: 512) weighed by bytes alone got 3 CTAs of 854
// records where the others had 5 or 6 of 427-512.  Returns true when the
// launch should rather be two launches of half the products each: a launch
// ends with its busiest CTA, and when whole CTAs per run leave that CTA far
// above the mean (56 gate/up runs of a 70B layer on 152 CTAs: runs of 2 and
// 3 CTAs, 1.36x the mean), half the products per launch do better (28 runs:
// 5 or 6 CTAs, 1.09x) than one launch saves in selection and prologue.
bool plan_runs(const CmbArgs& a, int grid, int* n) {
  double w[kMaxRuns];
  int nruns = 0;
  for (int p = 0; p < a.np; ++p)
    for (int s = 0; s < a.p[p].S; ++s, ++nruns) {
      const int rows = std::min(SEG_ROWS, a.p[p].O - s * SEG_ROWS);
      const double full = (double)MASK_BYTES + 2.0 * (double)a.p[p].dens * SEG_ROWS;
      w[nruns] = 4.0 * full + (double)MASK_BYTES + 2.0 * (double)a.p[p].dens * rows;
      n[nruns] = 1;
    }
  for (int extra = grid - nruns; extra > 0; --extra) {
    int best = 0;
    for (int q = 1; q < nruns; ++q)
      if (w[q] * n[best] > w[best] * n[q]) best = q;
    ++n[best];
  }
  if (a.np < 2) return false;
  double wsum = 0.0, wmax = 0.0;
  for (int q = 0; q < nruns; ++q) {
    wsum += w[q];
    wmax = std::max(wmax, w[q] / n[q]);
  }
  return wmax > 1.25 * wsum / grid;
}

cudaError_t launch_cmb_spmspv(const CmbArgs& a0, cudaStream_t st) {
  CmbArgs a = a0;
  if (a.wait_ns == 0) a.wait_ns = WAIT_LIMIT_NS;
  DevProps dp;
  cudaError_t e = dev_props(&dp);
  if (e != cudaSuccess) return e;
  const bool thresh = a.thresh != 0;
  const bool fused = thresh || a.kidx == nullptr;
  const bool quant = a.vbits != 16;
  if (a.vbits != 16 && a.vbits != 8 && a.vbits != 4) return cudaErrorInvalidValue;
  int64_t total = 0;
  for (int p = 0; p < a.np; ++p) total += (int64_t)a.p[p].S * (thresh ? a.I : a.k);
  if (total <= 0) return cudaSuccess;
  if (total >= ((int64_t)1 << 31)) return cudaErrorInvalidValue;   // item indices are 32-bit
  const int grid = (int)std::min<int64_t>(dp.nsm, total);
  if ((total + grid - 1) / grid >= (int64_t)1 << 30) return cudaErrorInvalidValue;
  if (thresh) a.k = 1 << 16;   // no rank space: cursors never wrap
  // Item split.  Items are the (problem, segment) runs of kept channels, in
  // order.  When every run can have CTAs of its own, runs get CTAs in
  // proportion to their estimated cost (plan_runs: mostly the number of
  // records) and no CTA spans two runs: a run boundary inside a CTA would
  // cost a mid-stream flush of all its consumers' rows.  A CTA of a fused mode
  // takes a channel range of its run (the kept set is a threshold, so it can
  // find its own kept channels); with a kept list it takes a rank range.
  // Otherwise (more runs than CTAs) a kept list is split evenly, and the
  // fused modes are not launched.
  int nruns = 0;
  for (int p = 0; p < a.np; ++p) nruns += a.p[p].S;
  int64_t per_cta = (total + grid - 1) / grid;
  a.nruns = 0;
  if (nruns <= kMaxRuns && nruns <= grid) {
    int n[kMaxRuns];
    if (plan_runs(a, grid, n)) {   // two launches of half the products each
      CmbArgs b0 = a0, b1 = a0;
      const int h = a0.np / 2;
      b0.np = h;
      b1.np = a0.np - h;
      for (int p = 0; p < b1.np; ++p) b1.p[p] = a0.p[h + p];
      e = launch_cmb_spmspv(b0, st);
      return e != cudaSuccess ? e : launch_cmb_spmspv(b1, st);
    }
    a.run_cta[0] = 0;
    per_cta = 0;
    for (int q = 0; q < nruns; ++q) {
      a.run_cta[q + 1] = (uint16_t)(a.run_cta[q] + n[q]);
      per_cta = std::max<int64_t>(per_cta, (a.k + n[q] - 1) / n[q]);
    }
    a.nruns = nruns;
    a.cta_info_ok = grid <= kMaxCtaInfo ? 1 : 0;
    if (a.cta_info_ok) {
      int q = 0;
      for (int p = 0; p < a.np; ++p)
        for (int s = 0; s < a.p[p].S; ++s, ++q)
          for (int m = 0; m < n[q]; ++m)
            a.cta_info[a.run_cta[q] + m] = (uint64_t)q | (uint64_t)p << 8 | (uint64_t)s << 10 |
                                           (uint64_t)m << 32 | (uint64_t)n[q] << 48;
    }
    if (fused) {   // channel ranges: at most ceil(I / n) kept per CTA
      per_cta = 0;
      for (int q = 0; q < nruns; ++q) per_cta = std::max<int64_t>(per_cta, (a.I + n[q] - 1) / n[q]);
    }
  } else if (thresh || quant) {
    return cudaErrorInvalidValue;   // these launches need CTAs of their own per run
  } else if (fused) {
    return cudaErrorNotSupported;   // the caller selects first and launches with a kept list
  }
  // Kept-list window of a CTA: at most its item count, at most k.
  a.list_cap = fused ? (int)std::min<int64_t>(per_cta, a.k) : 0;
  // Slot size: the largest record among the launch's weights (given by the
  // caller in a.slot_bytes); slot count: as many as the shared memory holds,
  // a multiple of the consumer count.
  const int slot_bytes = (int)align_up((size_t)std::max(a.slot_bytes, MASK_BYTES + 16), 16);
  if (slot_bytes > MAX_RECORD_BYTES) return cudaErrorInvalidValue;
  const size_t avail = (size_t)dp.smem_optin - 256;   // static shared memory headroom
  const size_t fixed = cmb_layout(a.I, fused, a.list_cap, 0, slot_bytes, quant).total + 128;
  if (fixed >= avail) return cudaErrorInvalidValue;
  int nslot = (int)((avail - fixed) / (slot_bytes + 20));
  nslot = std::min(nslot, CMB_MAX_SLOTS);
  nslot -= nslot % CMB_NC;
  if (nslot < std::max(32, CMB_NC)) return cudaErrorInvalidValue;
  // Pairs (waiting for more records costs more than it gains); coded
  // formats pair only items of one group, which a consumer can tell ahead
  // only from the kept list in shared memory (fused modes).
  a.group = (CMB_PAIRS && a.vbits != 4 && nslot >= 2 * CMB_NC && (fused || !quant)) ? 2 : 1;
  a.nslot = nslot;
  a.slot_bytes = slot_bytes;
  const size_t smem = cmb_layout(a.I, fused, a.list_cap, nslot, slot_bytes, quant).total;
  void (*kern)(const CmbArgs) = nullptr;
  const int mode = thresh ? CMB_THRESH : (fused ? CMB_TOPK : CMB_LISTED);
#define DUO_CMB_PICK(M, B) \
  if (mode == M && a.vbits == B) kern = cmb_spmspv_kernel<M, B>;
  DUO_CMB_PICK(CMB_LISTED, 16) DUO_CMB_PICK(CMB_TOPK, 16) DUO_CMB_PICK(CMB_THRESH, 16)
  DUO_CMB_PICK(CMB_LISTED, 8) DUO_CMB_PICK(CMB_TOPK, 8) DUO_CMB_PICK(CMB_THRESH, 8)
  DUO_CMB_PICK(CMB_LISTED, 4) DUO_CMB_PICK(CMB_TOPK, 4) DUO_CMB_PICK(CMB_THRESH, 4)
#undef DUO_CMB_PICK
  if (kern == nullptr) return cudaErrorInvalidValue;
  // L2 warm-up of the offset tables: each CTA one slice of every product's
  for (int p = 0; p < a.np; ++p) {
    const uint64_t bytes = align_up(((uint64_t)a.I * a.p[p].S + 1) * 4, 16);
    const bool fits = bytes < (1ull << 31);
    a.p[p].pf_bytes = fits ? (uint32_t)bytes : 0u;
    a.p[p].pf_chunk = fits ? (uint32_t)align_up((bytes + grid - 1) / grid, 16) : 0u;
  }
  e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(CMB_THREADS);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  // Cooperative: all CTAs are co-resident (the in-kernel grid barrier).
  // Programmatic stream serialization: this launch may start while the
  // previous kernel of the stream finishes; the kernel waits for it
  // (griddepcontrol.wait) before it reads its inputs or writes y.
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  e = cudaLaunchKernelEx(&cfg, kern, a);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

// ------------------------------------------------------------------------
// spMspV over the index format (parity format): one warp per kept channel,
// lanes stride its non-zeros and add w * x into y[row] atomically.
// ------------------------------------------------------------------------
constexpr int IDX16_THREADS = 512;   // the selection needs >= 512 threads

template <bool FUSED>
__global__ void __launch_bounds__(IDX16_THREADS, 1) idx16_spmspv_kernel(const Idx16Args a) {
  extern __shared__ __align__(128) uint8_t sm[];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const SelLayout L = sel_layout(a.I, 0, a.I);
  uint16_t* xs = reinterpret_cast<uint16_t*>(sm + L.xs);
  uint16_t* klist = reinterpret_cast<uint16_t*>(sm + L.klist);
  if (FUSED) {
    SelShared* sel = reinterpret_cast<SelShared*>(sm + L.sel);
    load_x_to_smem(xs, a.x, a.I);
    select_clear(sel);
    __syncthreads();
    int T, cut;
    select_threshold(xs, a.I, a.k, sel, &T, &cut);
    thresh_compact(xs, 0, a.I, T, cut, klist, nullptr, sel->wcnt);
  }
  const int nwt = gridDim.x * (IDX16_THREADS / 32);
  for (int i = blockIdx.x * (IDX16_THREADS / 32) + warp; i < a.k; i += nwt) {
    int j;
    uint16_t xb;
    if (FUSED) {
      j = klist[i];
      xb = xs[j];
    } else {
      j = __ldg(a.kidx + i);
      xb = __ldg(a.kval + i);
    }
    if (j >= a.I) {
      if (lane == 0) atomicOr(a.status, STATUS_FORMAT);
      continue;
    }
    const uint32_t n = __ldg(a.cnt + j);
    const uint8_t* blk = a.data + __ldg(a.colptr + j);
    const uint16_t* vals = reinterpret_cast<const uint16_t*>(blk);
    const uint16_t* rows = reinterpret_cast<const uint16_t*>(blk + align_up((size_t)2 * n, 16));
    for (uint32_t e = lane; e < n; e += 32) {
      const uint32_t r = __ldg(rows + e);
      if (r < (uint32_t)a.O) atomicAdd(a.y + r, fma_f16_f32(__ldg(vals + e), xb, 0.f));
    }
  }
}

}  // namespace duo

// Internal test entry point (not part of include/duo.h): the launcher's run
// plan for np products of O[p] rows and density dens[p] on grid CTAs.  Host
// only (no device call).  Writes each run's CTA count to n_out (runs in
// product order; room for 128) and returns their number, with *split = 1
// when the launch would be issued as two; -1 on bad arguments.
extern "C" int duo_test_plan_runs(int np, const int* O, const float* dens, int grid, int* n_out,
                                  int* split) {
  if (np < 1 || np > duo::kMaxProblems || O == nullptr || dens == nullptr || n_out == nullptr ||
      split == nullptr || grid < 1)
    return -1;
  duo::CmbArgs a{};
  a.np = np;
  int nruns = 0;
  for (int p = 0; p < np; ++p) {
    if (O[p] < 1) return -1;
    a.p[p].O = O[p];
    a.p[p].S = (O[p] + duo::SEG_ROWS - 1) / duo::SEG_ROWS;
    a.p[p].dens = dens[p];
    nruns += a.p[p].S;
  }
  if (nruns > duo::kMaxRuns || nruns > grid) return -1;
  *split = duo::plan_runs(a, grid, n_out) ? 1 : 0;
  return nruns;
}

namespace duo {

cudaError_t launch_idx16_spmspv(const Idx16Args& a, cudaStream_t st) {
  DevProps dp;
  cudaError_t e = dev_props(&dp);
  if (e != cudaSuccess) return e;
  if (a.k <= 0) return cudaSuccess;
  const bool fused = a.kidx == nullptr;
  const size_t smem = fused ? sel_layout(a.I, 0, a.I).end : 0;
  const int warps = IDX16_THREADS / 32;
  const int grid = (int)std::min<int64_t>((int64_t)dp.nsm * 2, ((int64_t)a.k + warps - 1) / warps);
  if (fused) {
    e = cudaFuncSetAttribute(idx16_spmspv_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem);
    if (e != cudaSuccess) return e;
    idx16_spmspv_kernel<true><<<grid, IDX16_THREADS, smem, st>>>(a);
  } else {
    idx16_spmspv_kernel<false><<<grid, IDX16_THREADS, 0, st>>>(a);
  }
  return cudaGetLastError();
}

cudaError_t read_and_clear_status(unsigned int* out) {
  unsigned int v = 0, zero = 0;
  cudaError_t e = cudaMemcpyFromSymbol(&v, g_status, sizeof(v));
  if (e != cudaSuccess) return e;
  e = cudaMemcpyToSymbol(g_status, &zero, sizeof(zero));
  *out = v;
  return e;
}

}  // namespace duo
