// Zero-copy swap-in kernel (the GPU-side counterpart of the paper's
// copy-free dispatch, Sec. 4.2.2): SM threads read the block's parameters
// straight from page-locked, mapped host memory and write them into the
// arena slot, 16 bytes per access, with several independent loads in flight
// per thread to cover the host-link latency.
#include <algorithm>
#include <cstring>

#include "device.cuh"
#include "internal.h"
#include "kernels.h"

namespace swapnet {

namespace {

constexpr int kZcMaxSeg = 48;
constexpr int kZcThreads = 512;
constexpr int kZcUnroll = 8;

struct ZcArgs {
  int nseg;
  ZcSeg seg[kZcMaxSeg];
};

__device__ __forceinline__ uint4 ld_host16(const uint4* p) {
  uint4 r;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p));
  return r;
}

__global__ void __launch_bounds__(kZcThreads) zerocopy_kernel(const __grid_constant__ ZcArgs a) {
  const uint64_t tid = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const uint64_t nthr = (uint64_t)gridDim.x * blockDim.x;
  for (int s = 0; s < a.nseg; ++s) {
    const uint4* __restrict__ src = static_cast<const uint4*>(a.seg[s].src);
    uint4* __restrict__ dst = static_cast<uint4*>(a.seg[s].dst);
    const uint64_t n16 = a.seg[s].bytes >> 4;
    uint64_t i = tid;
    // main body: kZcUnroll independent 16-byte loads in flight per thread
    for (; i + (kZcUnroll - 1) * nthr < n16; i += kZcUnroll * nthr) {
      uint4 v[kZcUnroll];
#pragma unroll
      for (int u = 0; u < kZcUnroll; ++u) v[u] = ld_host16(src + i + u * nthr);
#pragma unroll
      for (int u = 0; u < kZcUnroll; ++u) dst[i + u * nthr] = v[u];
    }
    for (; i < n16; i += nthr) dst[i] = ld_host16(src + i);
    // tail bytes (segment sizes need not be multiples of 16)
    const uint64_t tail = a.seg[s].bytes & 15;
    if (tail && tid < tail) {
      const uint8_t* s8 = static_cast<const uint8_t*>(a.seg[s].src) + (n16 << 4);
      uint8_t* d8 = static_cast<uint8_t*>(a.seg[s].dst) + (n16 << 4);
      d8[tid] = s8[tid];
    }
  }
}

}  // namespace

int launch_zerocopy(const ZcSeg* segs, int nseg, int ctas, cudaStream_t s) {
  if (nseg <= 0) return SWAPNET_OK;
  if (ctas <= 0) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "zero-copy: ctas must be positive");
  for (int i = 0; i < nseg; ++i)
    if (((uintptr_t)segs[i].src | (uintptr_t)segs[i].dst) & 15)
      SN_FAIL(SWAPNET_ERR_MISALIGNED, "zero-copy: segment not 16-byte aligned");
  for (int base = 0; base < nseg; base += kZcMaxSeg) {
    ZcArgs a;
    std::memset(&a, 0, sizeof(a));
    a.nseg = std::min(kZcMaxSeg, nseg - base);
    for (int i = 0; i < a.nseg; ++i) a.seg[i] = segs[base + i];
    zerocopy_kernel<<<ctas, kZcThreads, 0, s>>>(a);
    const cudaError_t err = cudaGetLastError();
    if (err != cudaSuccess) SN_FAIL(SWAPNET_ERR_CUDA, std::string("zero-copy launch: ") + cudaGetErrorString(err));
  }
  return SWAPNET_OK;
}

}  // namespace swapnet
