// Unpacking swap-in kernel of the packed swap variant (layout in pack.h):
// one warp per chunk, its header and body read straight from page-locked,
// mapped host memory (every load issued before any is used, so one link
// round trip per chunk; the body in whole 128-byte lines), decoded in
// registers and written to the arena with 16-byte stores.  Lane l takes elements 512 g + 16 l .. + 16 of its
// chunk for g = 0..7, so each warp-wide load reads one contiguous range:
// 8 bytes of codes (256 bytes a warp) and 16 sign-mantissa bytes (512).
// Four elements are decoded at once as byte lanes of 32-bit words: the
// exponents are x0 + code (no carry between bytes, since x0 + 15 <= 255),
// then the high and low bytes of the four bf16 values are assembled with
// masks and interleaved with byte permutes.  An escaped element (code 15)
// gets the exponent its record header lists, patched before the store.
#include <cstring>

#include "internal.h"
#include "kernels.h"
#include "pack.h"

namespace swapnet {

namespace {

constexpr int kUpMaxJobs = 1024;

__device__ __forceinline__ uint4 ld_host16(const void* p) {
  uint4 r;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p));
  return r;
}

__device__ __forceinline__ uint2 ld_host8(const void* p) {
  uint2 r;
  asm volatile("ld.global.nc.L1::no_allocate.v2.u32 {%0,%1}, [%2];" : "=r"(r.x), "=r"(r.y) : "l"(p));
  return r;
}

// four 4-bit codes (16 bits, element i in bits 4i..4i+3) -> one per byte
__device__ __forceinline__ uint32_t spread4(uint32_t sel) {
  uint32_t t = (sel | (sel << 8)) & 0x00ff00ffu;
  return (t | (t << 4)) & 0x0f0f0f0fu;
}

// four elements: codes (16 bits) and sign-mantissa bytes -> two words of
// two bf16 values each
__device__ __forceinline__ void decode4(uint32_t sel, uint32_t sm, uint32_t x0x4, uint32_t& w0, uint32_t& w1) {
  const uint32_t x = spread4(sel) + x0x4;  // exponents, one per byte
  const uint32_t hi = (sm & 0x80808080u) | ((x >> 1) & 0x7f7f7f7fu);
  const uint32_t lo = ((x << 7) & 0x80808080u) | (sm & 0x7f7f7f7fu);
  w0 = __byte_perm(lo, hi, 0x5140);
  w1 = __byte_perm(lo, hi, 0x7362);
}

__global__ void __launch_bounds__(kUnpackThreads, 1) unpack_kernel(const PkJob* __restrict__ jobs, int njobs,
                                                                uint32_t total) {
  __shared__ uint32_t s_first[kUpMaxJobs];
  for (int j = threadIdx.x; j < njobs; j += blockDim.x) s_first[j] = jobs[j].first;
  __syncthreads();
  const int lane = threadIdx.x & 31;
  const uint32_t nwarps = (gridDim.x * blockDim.x) >> 5;
  for (uint32_t g = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; g < total; g += nwarps) {
    int lo = 0, hi = njobs - 1;  // the last job starting at or before chunk g
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (s_first[mid] <= g) lo = mid;
      else hi = mid - 1;
    }
    const PkJob* J = jobs + lo;
    const uint32_t rel = g - J->first;
    const uint8_t* base = J->base;
    const uint64_t c = J->c0 + rel;
    const uint8_t* body = base + J->body_off + c * kPkBody;
    uint4* out = reinterpret_cast<uint4*>(J->dst + (uint64_t)rel * kPkChunk);
    const uint32_t x0x4 = J->x0 * 0x01010101u;
    const uint4 hdr = ld_host16(base + 16 + kPkHeader * c);
    uint2 cd[8];
    uint4 sm[8];
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      cd[q] = ld_host8(body + q * 256 + lane * 8);
      sm[q] = ld_host16(body + kPkChunk / 2 + q * 512 + lane * 16);
    }
    const uint32_t k = hdr.x & 0xffu;
    if (k == (uint32_t)kPkRaw) {  // stored unpacked in the overflow area
      const uint8_t* src = base + J->overflow_off + (uint64_t)hdr.y * kPkChunkBytes;
      uint4 v[16];
#pragma unroll
      for (int i = 0; i < 16; ++i) v[i] = ld_host16(src + (uint64_t)(i * 32 + lane) * 16);
#pragma unroll
      for (int i = 0; i < 16; ++i) out[i * 32 + lane] = v[i];
      continue;
    }
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      uint32_t w[8];  // elements 2i, 2i + 1 of this lane's 16
      decode4(cd[q].x & 0xffffu, sm[q].x, x0x4, w[0], w[1]);
      decode4(cd[q].x >> 16, sm[q].y, x0x4, w[2], w[3]);
      decode4(cd[q].y & 0xffffu, sm[q].z, x0x4, w[4], w[5]);
      decode4(cd[q].y >> 16, sm[q].w, x0x4, w[6], w[7]);
      const uint32_t e0 = q * 512 + lane * 16;  // this lane's first element
#pragma unroll
      for (uint32_t i = 0; i < (uint32_t)kPkMaxEsc; ++i) {  // k is the same for the whole warp
        const uint32_t pos = ((i < 2 ? hdr.y : hdr.z) >> ((i & 1) * 16)) & 0xffffu;
        if (i < k && pos - e0 < 16u) {
          const uint32_t j = pos - e0, sh = (j & 1) * 16;
          const uint32_t m = 0x7f80u << sh, v = ((hdr.w >> (i * 8)) & 0xffu) << (7 + sh);
#pragma unroll
          for (int t = 0; t < 8; ++t) {  // masks, not an indexed store: w stays in registers
            const uint32_t mt = (j >> 1) == (uint32_t)t ? m : 0u;
            w[t] = (w[t] & ~mt) | (v & mt);
          }
        }
      }
      out[e0 / 8] = make_uint4(w[0], w[1], w[2], w[3]);
      out[e0 / 8 + 1] = make_uint4(w[4], w[5], w[6], w[7]);
    }
  }
}

}  // namespace

int launch_unpack(const PkJob* jobs, int njobs, uint32_t total, int ctas, cudaStream_t s) {
  if (njobs <= 0 || total == 0) return SWAPNET_OK;
  if (njobs > kUpMaxJobs) SN_FAIL(SWAPNET_ERR_UNSUPPORTED, "unpack: too many jobs in one launch");
  if (ctas <= 0) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "unpack: ctas must be positive");
  unpack_kernel<<<ctas, kUnpackThreads, 0, s>>>(jobs, njobs, total);
  const cudaError_t err = cudaGetLastError();
  if (err != cudaSuccess) SN_FAIL(SWAPNET_ERR_CUDA, std::string("unpack launch: ") + cudaGetErrorString(err));
  return SWAPNET_OK;
}

}  // namespace swapnet
