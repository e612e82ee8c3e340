// Unpacking swap-in kernel of the packed swap variant (layout in pack.h):
// one warp per chunk record, read straight from page-locked, mapped host
// memory with 16-byte loads (all of a record's loads issued before any is
// used, so one link round trip per record), decoded in registers and
// written to the arena with 16-byte stores.  Lane l of a warp decodes
// elements d * 1024 + 32 l .. + 32 of its chunk for d = 0..3: 16 bytes of
// codes and 32 bytes of sign-mantissa bytes each, 64 bytes of output.
#include <cstring>

#include "internal.h"
#include "kernels.h"
#include "pack.h"

namespace swapnet {

namespace {

constexpr int kUpThreads = 512;
constexpr int kUpMaxJobs = 1024;

__device__ __forceinline__ uint4 ld_host16(const void* p) {
  uint4 r;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p));
  return r;
}

__device__ __forceinline__ uint32_t word_of(const uint4& v, int i) {
  return i == 0 ? v.x : i == 1 ? v.y : i == 2 ? v.z : v.w;
}

// exponent of code c (< 15) from the 16 table bytes in t
__device__ __forceinline__ uint32_t table_exp(uint32_t c, const uint4& t) {
  const uint32_t lo = __byte_perm(t.x, t.y, c & 7u);
  const uint32_t hi = __byte_perm(t.z, t.w, c & 7u);
  return (c < 8u ? lo : hi) & 0xffu;
}

// exponent of the escaped element at position pos of the chunk (the header
// lists k <= 4 positions in hdr.y, hdr.z and their exponents in hdr.w)
__device__ __forceinline__ uint32_t escape_exp(uint32_t pos, uint32_t k, const uint4& hdr) {
  uint32_t x = 0;
#pragma unroll
  for (uint32_t i = 0; i < (uint32_t)kPkMaxEsc; ++i) {
    const uint32_t p = ((i < 2 ? hdr.y : hdr.z) >> ((i & 1) * 16)) & 0xffffu;
    if (i < k && p == pos) x = (hdr.w >> (i * 8)) & 0xffu;
  }
  return x;
}

__global__ void __launch_bounds__(kUpThreads) unpack_kernel(const PkJob* __restrict__ jobs, int njobs,
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
    const uint8_t* rec = base + kPkHeader + (uint64_t)(J->c0 + rel) * kPkRecord;
    uint4* out = reinterpret_cast<uint4*>(J->dst + (uint64_t)rel * kPkChunk);
    const uint4 t = make_uint4(J->table[0], J->table[1], J->table[2], J->table[3]);
    const uint4 hdr = ld_host16(rec);
    uint4 cd[4], s0[4], s1[4];
#pragma unroll
    for (int d = 0; d < 4; ++d) {
      cd[d] = ld_host16(rec + 16 + d * 512 + lane * 16);
      s0[d] = ld_host16(rec + 16 + kPkChunk / 2 + d * 1024 + lane * 32);
      s1[d] = ld_host16(rec + 16 + kPkChunk / 2 + d * 1024 + lane * 32 + 16);
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
    for (int d = 0; d < 4; ++d) {
      const uint32_t e0 = d * 1024 + lane * 32;  // first element of this group
      uint32_t w[16];
#pragma unroll
      for (int j = 0; j < 32; ++j) {
        const uint32_t c = (word_of(cd[d], j >> 3) >> ((j & 7) * 4)) & 0xfu;
        const uint32_t s = (word_of(j < 16 ? s0[d] : s1[d], (j & 15) >> 2) >> ((j & 3) * 8)) & 0xffu;
        const uint32_t x = c < 15u ? table_exp(c, t) : escape_exp(e0 + j, k, hdr);
        const uint32_t v = ((s & 0x80u) << 8) | (x << 7) | (s & 0x7fu);
        if (j & 1) w[j >> 1] |= v << 16;
        else w[j >> 1] = v;
      }
#pragma unroll
      for (int q = 0; q < 4; ++q) out[e0 / 8 + q] = make_uint4(w[4 * q], w[4 * q + 1], w[4 * q + 2], w[4 * q + 3]);
    }
  }
}

}  // namespace

int launch_unpack(const PkJob* jobs, int njobs, uint32_t total, int ctas, cudaStream_t s) {
  if (njobs <= 0 || total == 0) return SWAPNET_OK;
  if (njobs > kUpMaxJobs) SN_FAIL(SWAPNET_ERR_UNSUPPORTED, "unpack: too many jobs in one launch");
  if (ctas <= 0) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "unpack: ctas must be positive");
  unpack_kernel<<<ctas, kUpThreads, 0, s>>>(jobs, njobs, total);
  const cudaError_t err = cudaGetLastError();
  if (err != cudaSuccess) SN_FAIL(SWAPNET_ERR_CUDA, std::string("unpack launch: ") + cudaGetErrorString(err));
  return SWAPNET_OK;
}

}  // namespace swapnet
