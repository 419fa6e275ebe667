// duo_pack_cmb_noalloc: the bitmask packer for callers that cannot allocate
// device memory themselves (declared in include/duo.h).
//
// duo_pack needs per-record scratch (the non-zero count of every
// (channel, segment) record, and three totals) and allocates it, plus the
// packed buffers, with cudaMalloc.  Some callers cannot do that: code that
// runs where the CUDA allocator is off limits (an engine whose device memory
// all comes from a pool it manages itself, or a process whose allocations
// are accounted by someone else).  This entry point writes the packed bytes
// into buffers the caller provides and keeps its scratch in a fixed,
// file-scope device array instead, so it calls no cudaMalloc, cudaFree or
// other allocating routine.
#include <cstdint>
#include <mutex>

#include <cuda_runtime.h>

#include "duo.h"
#include "duo_launch.h"

namespace {

// Scratch limit: I * ceil(O / 1024) records (4 bytes each) plus three 64-bit
// totals that the offset scan writes (16-byte units, non-zeros, the largest
// record's count).  262144 records covers, for example, I = 65535 with
// O <= 4096, or a 28672 x 8192 weight (229376 records).
constexpr int64_t kMaxRecords = DUO_NOALLOC_MAX_RECORDS;
constexpr size_t kTotalsAt = (size_t)kMaxRecords * 4;
constexpr size_t kTotalsPad = 256;
static_assert(kTotalsPad >= 3 * sizeof(unsigned long long), "the scan writes three totals");

// Every GPU that loads the library holds this array until the process exits.
static __device__ __align__(256) unsigned char g_noalloc_scratch[kTotalsAt + kTotalsPad];

std::mutex g_mu;
void* g_scratch_dev[64];
bool g_scratch_ready[64];

// Device address of the scratch array for the current device.  In host code
// the array's name is only a host-side stand-in, so its device address is
// fetched once per device, with that device current, and cached.
int scratch_address(void** out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
    cudaGetLastError();
    return DUO_ECUDA;
  }
  std::lock_guard<std::mutex> lk(g_mu);
  if (!g_scratch_ready[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr) {
      cudaGetLastError();
      return DUO_ECUDA;
    }
    g_scratch_dev[dev] = p;
    g_scratch_ready[dev] = true;
  }
  *out = g_scratch_dev[dev];
  return DUO_OK;
}

bool aligned_to(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// True when the GPU can address p as device memory (device or managed).
bool on_device(const void* p) {
  cudaPointerAttributes at;
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged;
}

int map_cuda(cudaError_t e) {
  if (e == cudaSuccess) return DUO_OK;
  cudaGetLastError();
  return DUO_ECUDA;
}

}  // namespace

extern "C" int duo_pack_cmb_noalloc(const void* W_fp16_dev, int64_t out, int64_t in, int64_t ldw,
                                    uint32_t* off_dev, void* data_dev, int64_t data_capacity,
                                    int64_t* data_bytes, void* stream) {
  if (W_fp16_dev == nullptr || off_dev == nullptr || data_bytes == nullptr) return DUO_EINVAL;
  if (out < 1 || in < 1 || ldw < in || data_capacity < 0) return DUO_EINVAL;
  if (!aligned_to(W_fp16_dev, 2) || !aligned_to(off_dev, 4) || !aligned_to(data_dev, 16))
    return DUO_EINVAL;
  if (in > 65535) return DUO_ERANGE;
  const int64_t S = (out + duo::kSegRows - 1) / duo::kSegRows;
  const int64_t nrec = in * S;
  if (nrec > kMaxRecords) return DUO_ERANGE;
  if (S > 65535) return DUO_ERANGE;   // segments are a grid dimension, as in duo_pack
  int n = 0;
  if (cudaGetDeviceCount(&n) != cudaSuccess || n <= 0) {
    cudaGetLastError();
    return DUO_ECUDA;
  }
  if (!on_device(W_fp16_dev) || !on_device(off_dev) ||
      (data_dev != nullptr && !on_device(data_dev)))
    return DUO_EINVAL;
  void* scratch = nullptr;
  int rc = scratch_address(&scratch);
  if (rc != DUO_OK) return rc;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const uint16_t* W = static_cast<const uint16_t*>(W_fp16_dev);
  uint32_t* cnt = static_cast<uint32_t*>(scratch);
  unsigned long long* totals =
      reinterpret_cast<unsigned long long*>(static_cast<unsigned char*>(scratch) + kTotalsAt);

  // Every scratch word read below is written earlier in the same call (the
  // count kernel writes all nrec counts, the scan writes all three totals), so
  // nothing needs clearing; the previous call's contents are never read.
  rc = map_cuda(duo::launch_pack_count(W, out, in, ldw, (int)S, cnt, st));
  if (rc != DUO_OK) return rc;
  rc = map_cuda(duo::launch_cmb_offsets(cnt, nrec, 16, off_dev, totals, st));
  if (rc != DUO_OK) return rc;
  unsigned long long host_tot[2] = {0, 0};
  rc = map_cuda(cudaMemcpyAsync(host_tot, totals, sizeof(host_tot), cudaMemcpyDeviceToHost, st));
  if (rc != DUO_OK) return rc;
  rc = map_cuda(cudaStreamSynchronize(st));
  if (rc != DUO_OK) return rc;
  if (host_tot[0] >= (1ull << 32)) return DUO_ERANGE;
  const int64_t bytes = (int64_t)host_tot[0] * 16;
  *data_bytes = bytes;
  if (data_dev == nullptr) return DUO_OK;            // size query
  if (bytes > data_capacity) return DUO_ERANGE;      // *data_bytes tells the size needed
  rc = map_cuda(cudaMemsetAsync(data_dev, 0, (size_t)bytes, st));
  if (rc != DUO_OK) return rc;
  rc = map_cuda(duo::launch_cmb_scatter(W, out, in, ldw, (int)S, 16, nullptr, off_dev,
                                        static_cast<uint8_t*>(data_dev), st));
  if (rc != DUO_OK) return rc;
  return map_cuda(cudaStreamSynchronize(st));
}
