// duo_copy (include/duo.h): a copy between two addresses the GPU can reach
// (device memory, or page-locked host memory mapped into the device's address
// space), done by a kernel on the SMs instead of the copy engine.  In a
// captured decode step the step's inputs come in and its outputs go out this
// way: a copy-engine node costs a few microseconds of scheduling on each side
// of the kernels, a small kernel about half of that.
#include <cstdint>

#include <cuda_runtime.h>

#include "duo.h"
#include "duo_device.cuh"

namespace duo {

// 16-byte words when both ends are 16-byte aligned, else bytes.  Waits for the
// previous kernel of the stream first (programmatic dependent launch: the
// copy may start while that kernel drains, never before its data is final).
__global__ void __launch_bounds__(256) copy_kernel(uint8_t* __restrict__ d, const uint8_t* __restrict__ s,
                                                   int64_t bytes) {
  griddep_wait();
  const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t nt = (int64_t)gridDim.x * blockDim.x;
  if (((reinterpret_cast<uintptr_t>(d) | reinterpret_cast<uintptr_t>(s)) & 15u) == 0) {
    const int64_t n16 = bytes >> 4;
    uint4* d16 = reinterpret_cast<uint4*>(d);
    const uint4* s16 = reinterpret_cast<const uint4*>(s);
    for (int64_t i = t; i < n16; i += nt) d16[i] = s16[i];
    for (int64_t i = (n16 << 4) + t; i < bytes; i += nt) d[i] = s[i];
  } else {
    for (int64_t i = t; i < bytes; i += nt) d[i] = s[i];
  }
  griddep_launch_dependents();
}

}  // namespace duo

namespace {

// The address the current device dereferences for p, or nullptr when p is
// not memory that device can reach (unregistered host memory, another
// device's memory, an unknown address).
void* device_view(const void* p, int dev) {
  cudaPointerAttributes at;
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  if (at.type == cudaMemoryTypeDevice) return at.device == dev ? at.devicePointer : nullptr;
  if (at.type == cudaMemoryTypeManaged || at.type == cudaMemoryTypeHost) return at.devicePointer;
  return nullptr;
}

}  // namespace

extern "C" int duo_copy(void* dst, const void* src, int64_t bytes, void* stream) {
  if (bytes < 0) return DUO_EINVAL;
  if (bytes == 0) return DUO_OK;   // nothing to copy: no pointer is looked at
  if (dst == nullptr || src == nullptr) return DUO_EINVAL;
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    return DUO_ECUDA;
  }
  void* d = device_view(dst, dev);
  const void* s = device_view(src, dev);
  if (d == nullptr || s == nullptr) return DUO_EINVAL;
  const int64_t words = (bytes + 15) / 16;
  const int64_t want = (words + 255) / 256;
  const unsigned grid = (unsigned)(want < 4 * 152 ? want : 4 * 152);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(256);
  cfg.stream = static_cast<cudaStream_t>(stream);
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, duo::copy_kernel, static_cast<uint8_t*>(d),
                                           static_cast<const uint8_t*>(s), bytes);
  if (e == cudaSuccess) return DUO_OK;
  cudaGetLastError();
  return DUO_ECUDA;
}
