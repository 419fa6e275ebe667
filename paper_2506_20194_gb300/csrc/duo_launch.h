// Host-side interface between the C ABI (api.cu) and the kernels
// (kernels.cu).  Plain structs of device pointers and sizes.
#pragma once

#include <cstddef>
#include <cstdint>

#include <cuda_runtime.h>

namespace duo {

constexpr int kMaxProblems = 4;
constexpr int kMaxRuns = 128;   // (problem, segment) runs a launch may split by
constexpr int kMaxCtaInfo = 256;   // CTAs whose run identity the launcher precomputes
// Modes of the fused bitmask kernel.
constexpr int CMB_LISTED = 0;   // kept list given by the caller
constexpr int CMB_TOPK = 1;     // exact top-k selection in the kernel
constexpr int CMB_THRESH = 2;   // threshold mask in the kernel
constexpr int kSegRows = 1024;

struct CmbProb {
  const uint8_t* data;   // records
  const uint32_t* off;   // off[I*S + 1], 16-byte units
  float* y;              // fp32[O], zeroed before the launch
  const uint32_t* qtab;  // quantised formats: grid tables [S][G][1024] ({fp16 s, z})
  int O;
  int S;
  int G;                 // quantised formats: input-channel groups ceil(I / 128)
  float dens;            // non-zeros / (O * I): to estimate record sizes
  uint32_t pf_bytes;     // set by the launcher: bytes of off[], 16-byte aligned (0: no warm-up)
  uint32_t pf_chunk;     // set by the launcher: bytes of off[] each CTA warms in L2
};

struct CmbArgs {
  CmbProb p[kMaxProblems];
  int np;
  int I;
  int k;
  int cta_info_ok;       // set by the launcher: cta_info holds every CTA's run (see below);
                         // next to I and x, whose parameter line the kernel reads first
  const uint16_t* x;     // fused mode: fp16 bits [I]
  const uint16_t* kidx;  // listed mode: uint16 [k]
  const uint16_t* kval;  // listed mode: fp16 bits [k]
  unsigned int* bar;     // 2 words {count, generation} of a grid barrier, zero
                         // between launches; owned by the first handle
  int slot_bytes;        // in: largest record of the launch's weights (bytes);
                         // the launcher rounds it and picks the slot count
  int nslot;             // set by the launcher (a multiple of the consumer count)
  int group;             // set by the launcher: records a consumer waits for at once (1 or 2)
  int list_cap;          // set by the launcher: kept-list entries a CTA emits
  int thresh;            // in: 1 = threshold mask (keep key > tau_key), 0 = top-k / listed
  uint32_t tau_key;      // in: threshold as an fp16 magnitude bit pattern (bits & 0x7FFF)
  int vbits;             // in: bits of a stored value: 16 (fp16), 8 or 4 (RTN codes)
  unsigned int* status;  // device status word of the launch (the first handle's):
                         // bit 0 a bounded wait ran out, bit 1 a bad record or id
  unsigned long long wait_ns;   // limit of every bounded wait (0: the 1 s default)
  int nruns;             // set by the launcher: > 0 when each (problem, segment)
                         // run has CTAs of its own: run r (items r*k .. r*k+k-1)
                         // goes to CTAs run_cta[r] .. run_cta[r+1]-1
  uint16_t run_cta[kMaxRuns + 1];
  // set by the launcher when nruns > 0 and the grid has at most kMaxCtaInfo
  // CTAs (cta_info_ok = 1; else 0 and the kernel searches run_cta): per CTA
  // its run r, the run's product p and segment s, the CTA's index m in the
  // run and the run's CTA count n, packed as r | p << 8 | s << 10 | m << 32 |
  // n << 48 (one parameter load instead of a search)
  uint64_t cta_info[kMaxCtaInfo];
};

struct Idx16Args {
  unsigned int* status;  // device status word of the launch (the handle's)
  const uint8_t* data;
  const uint64_t* colptr;
  const uint32_t* cnt;
  float* y;
  int O;
  int I;
  int k;
  const uint16_t* x;
  const uint16_t* kidx;
  const uint16_t* kval;
};

// SM count and opt-in shared memory per block of the current device
// (cached per device).
struct DevProps {
  int nsm = 0;
  int smem_optin = 0;
};
cudaError_t dev_props(DevProps* out);

// spMspV over the bitmask format (fused when a.kidx == nullptr).  Zeroes
// every y itself (no memset needed before it).
cudaError_t launch_cmb_spmspv(const CmbArgs& a, cudaStream_t st);
// spMspV over the index format (fused when a.kidx == nullptr).
cudaError_t launch_idx16_spmspv(const Idx16Args& a, cudaStream_t st);
// Exact top-k sparsifier: kept ids ascending + their values.
cudaError_t launch_sparsify_threshold(const uint16_t* x, int I, uint32_t tau_key, uint16_t* kidx,
                                      uint16_t* kval, int* count, cudaStream_t st);
cudaError_t launch_sparsify(const uint16_t* x, int I, int k, uint16_t* kidx, uint16_t* kval,
                            cudaStream_t st);

// Packing.  cnt_js[j*S + s] = non-zeros of channel j in row segment s.
cudaError_t launch_pack_count(const uint16_t* W, int64_t O, int64_t I, int64_t ldw, int S,
                              uint32_t* cnt_js, cudaStream_t st);
// off[n] exclusive prefix (16-byte units) of the CMB record sizes for
// vbits-bit values (16, 8 or 4); totals[0] = total units (64-bit),
// totals[1] = total non-zeros, totals[2] = largest per-record non-zero count.
cudaError_t launch_cmb_offsets(const uint32_t* cnt_js, int64_t n, int vbits, uint32_t* off,
                               unsigned long long* totals, cudaStream_t st);
// RTN grids of every (row, 128-channel group) into table[S][G][1024]
// (zeroed by the caller; rows >= O stay 0).
cudaError_t launch_quant_grid(const uint16_t* W, int64_t O, int64_t I, int64_t ldw, int S, int bits,
                              uint32_t* table, cudaStream_t st);
// Records: fp16 values (vbits 16) or the codes of the grids in table.
cudaError_t launch_cmb_scatter(const uint16_t* W, int64_t O, int64_t I, int64_t ldw, int S,
                               int vbits, const uint32_t* table, const uint32_t* off,
                               uint8_t* data, cudaStream_t st);
// cnt[j] = sum_s cnt_js, colptr[j] byte offsets of the IDX16 blocks;
// totals[0] = total bytes, totals[1] = total non-zeros.
cudaError_t launch_idx16_offsets(const uint32_t* cnt_js, int64_t I, int S, uint32_t* cnt,
                                 uint64_t* colptr, unsigned long long* totals, cudaStream_t st);
cudaError_t launch_idx16_scatter(const uint16_t* W, int64_t O, int64_t I, int64_t ldw, int S,
                                 const uint32_t* cnt_js, const uint32_t* cnt,
                                 const uint64_t* colptr, uint8_t* data, cudaStream_t st);

// Reads and clears the process-wide device status word of the kernels that
// run without a handle (the sparsifiers): bit 0 a bounded wait ran out,
// bit 1 a record size or id outside the format's bounds.
cudaError_t read_and_clear_status(unsigned int* out);

}  // namespace duo
