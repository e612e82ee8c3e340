// Shared pieces of the tcgen05 GEMM kernels: launch arguments and the
// register-only fused epilogue (bias, residual, activation, conversion).
#pragma once
#include "device.cuh"
#include "kernels.h"

namespace swapnet {
namespace {

struct TcArgs {
  int M, N, K;
  const void* x;  // conv input (gather)
  int H, Wd, C, Ho, Wo, kh, kw, stride, pad;
  Epi e;
  void* y;
  int64_t ldy;
  int* err;
  int kb_per_split;  // k-blocks per split; gridDim.z splits
  float* partial;    // [splits][M][N] fp32 partial sums (global split-K only)
  int* counters;     // per output tile, zero between launches (global split-K only)
  int cluster;       // 1: the splits of a tile form a cluster and reduce through DSMEM
  // TMA im2col (persistent kernel): output tiles are wt x ht pixel patches of
  // one image, tiles_w x tiles_h of them per image; rows >= wt * ht are unused
  int wt, ht, tiles_w, tiles_h;
};

// ---- register-only epilogue helpers
template <typename T> __device__ __forceinline__ uint32_t pack2(float lo, float hi);
template <> __device__ __forceinline__ uint32_t pack2<__half>(float lo, float hi) {
  uint32_t r;
  asm("cvt.rn.f16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
  return r;
}
template <> __device__ __forceinline__ uint32_t pack2<__nv_bfloat16>(float lo, float hi) {
  uint32_t r;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
  return r;
}
template <typename T> __device__ __forceinline__ float lo_f(uint32_t u);
template <typename T> __device__ __forceinline__ float hi_f(uint32_t u);
template <> __device__ __forceinline__ float lo_f<__half>(uint32_t u) {
  return __half2float(__ushort_as_half((unsigned short)(u & 0xffffu)));
}
template <> __device__ __forceinline__ float hi_f<__half>(uint32_t u) {
  return __half2float(__ushort_as_half((unsigned short)(u >> 16)));
}
template <> __device__ __forceinline__ float lo_f<__nv_bfloat16>(uint32_t u) { return __uint_as_float(u << 16); }
template <> __device__ __forceinline__ float hi_f<__nv_bfloat16>(uint32_t u) { return __uint_as_float(u & 0xffff0000u); }

// 8 consecutive outputs (16 bytes): acc -> bias, residual (the 8 stored
// values r, when has_res), activation -> T.
template <typename T>
__device__ __forceinline__ void epi8r(const float (&a)[8], const float* sb, uint4 r, bool has_res, T* out, int act,
                                      int res_post) {
  const float4 b0 = *reinterpret_cast<const float4*>(sb);
  const float4 b1 = *reinterpret_cast<const float4*>(sb + 4);
  const float bf[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
  const uint32_t rw[4] = {r.x, r.y, r.z, r.w};
  uint32_t o[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float v0 = epilogue(a[2 * i], bf[2 * i], lo_f<T>(rw[i]), has_res, act, res_post);
    const float v1 = epilogue(a[2 * i + 1], bf[2 * i + 1], hi_f<T>(rw[i]), has_res, act, res_post);
    o[i] = pack2<T>(v0, v1);
  }
  *reinterpret_cast<uint4*>(out) = make_uint4(o[0], o[1], o[2], o[3]);
}

// The residual of 32 columns [n, n+32) of row m as four 16-byte loads, for
// the vector path of finish32 (zeros when there is no residual or the
// vector path does not apply).  Issued a chunk ahead, so that the loads'
// latency overlaps the accumulator reads and the arithmetic of the chunk
// before.
template <typename T>
__device__ __forceinline__ void res_prefetch32(uint4 (&r)[4], const TcArgs& p, int m, int n, bool vec_ok) {
  const T* res = static_cast<const T*>(p.e.res);
  const bool ok = res && m >= 0 && vec_ok && n + 32 <= p.N;
#pragma unroll
  for (int q = 0; q < 4; ++q)
    r[q] = ok ? *reinterpret_cast<const uint4*>(res + (int64_t)m * p.e.ldr + n + 8 * q) : make_uint4(0, 0, 0, 0);
}

// 8 consecutive outputs (16 bytes): acc -> bias, residual, activation -> T.
template <typename T>
__device__ __forceinline__ void epi8(const float (&a)[8], const float* sb, const T* res, T* out, int act,
                                     int res_post) {
  const float4 b0 = *reinterpret_cast<const float4*>(sb);
  const float4 b1 = *reinterpret_cast<const float4*>(sb + 4);
  const float bf[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
  uint4 r = make_uint4(0, 0, 0, 0);
  if (res) r = *reinterpret_cast<const uint4*>(res);
  const uint32_t rw[4] = {r.x, r.y, r.z, r.w};
  uint32_t o[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float v0 = epilogue(a[2 * i], bf[2 * i], lo_f<T>(rw[i]), res != nullptr, act, res_post);
    const float v1 = epilogue(a[2 * i + 1], bf[2 * i + 1], hi_f<T>(rw[i]), res != nullptr, act, res_post);
    o[i] = pack2<T>(v0, v1);
  }
  *reinterpret_cast<uint4*>(out) = make_uint4(o[0], o[1], o[2], o[3]);
}

// Final epilogue of 32 columns [n, n+32) of row m from fp32 values v.
template <typename T>
__device__ __forceinline__ void finish32(const float (&v)[32], const float* sb, const TcArgs& p, int m, int n,
                                         bool vec_ok) {
  const T* res = static_cast<const T*>(p.e.res);
  T* y = static_cast<T*>(p.y) + (int64_t)m * p.ldy;
  const T* rrow = res ? res + (int64_t)m * p.e.ldr : nullptr;
  if (vec_ok && n + 32 <= p.N) {
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      float a[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) a[j] = v[8 * q + j];
      epi8<T>(a, sb + 8 * q, rrow ? rrow + n + 8 * q : nullptr, y + n + 8 * q, p.e.act, p.e.res_post);
    }
  } else {
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      if (n + j < p.N) {
        const float rv = rrow ? to_f<T>(rrow[n + j]) : 0.f;
        y[n + j] = from_f<T>(epilogue(v[j], sb[j], rv, rrow != nullptr, p.e.act, p.e.res_post));
      }
    }
  }
}

// finish32 with the residual already loaded by res_prefetch32 (same
// arithmetic; the scalar path, for ragged or unaligned columns, loads it
// itself).
template <typename T>
__device__ __forceinline__ void finish32r(const float (&v)[32], const float* sb, const TcArgs& p, int m, int n,
                                          bool vec_ok, const uint4 (&r)[4]) {
  if (vec_ok && n + 32 <= p.N) {
    T* y = static_cast<T*>(p.y) + (int64_t)m * p.ldy;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      float a[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) a[j] = v[8 * q + j];
      epi8r<T>(a, sb + 8 * q, r[q], p.e.res != nullptr, y + n + 8 * q, p.e.act, p.e.res_post);
    }
  } else {
    finish32<T>(v, sb, p, m, n, vec_ok);
  }
}

__device__ __forceinline__ void epi_bar() { asm volatile("bar.sync 1, 128;" ::: "memory"); }

// Final epilogue of 4 columns [n, n+4) of row m.
template <typename T>
__device__ __forceinline__ void finish4(const float4& v, const float* sb, const TcArgs& p, int m, int n) {
  const T* res = static_cast<const T*>(p.e.res);
  T* y = static_cast<T*>(p.y) + (int64_t)m * p.ldy;
  const T* rrow = res ? res + (int64_t)m * p.e.ldr : nullptr;
  const float a[4] = {v.x, v.y, v.z, v.w};
  const bool vec = n + 4 <= p.N && ((p.ldy | n) % 4 == 0) && (!rrow || (p.e.ldr % 4 == 0));
  if (vec) {
    uint2 rr = make_uint2(0, 0);
    if (rrow) rr = *reinterpret_cast<const uint2*>(rrow + n);
    const float b0 = sb[0], b1 = sb[1], b2 = sb[2], b3 = sb[3];
    const float r0 = lo_f<T>(rr.x), r1 = hi_f<T>(rr.x), r2 = lo_f<T>(rr.y), r3 = hi_f<T>(rr.y);
    const int hr = rrow != nullptr;
    const uint32_t w0 = pack2<T>(epilogue(a[0], b0, r0, hr, p.e.act, p.e.res_post),
                                 epilogue(a[1], b1, r1, hr, p.e.act, p.e.res_post));
    const uint32_t w1 = pack2<T>(epilogue(a[2], b2, r2, hr, p.e.act, p.e.res_post),
                                 epilogue(a[3], b3, r3, hr, p.e.act, p.e.res_post));
    *reinterpret_cast<uint2*>(y + n) = make_uint2(w0, w1);
  } else {
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      if (n + j < p.N) {
        const float rv = rrow ? to_f<T>(rrow[n + j]) : 0.f;
        y[n + j] = from_f<T>(epilogue(a[j], sb[j], rv, rrow != nullptr, p.e.act, p.e.res_post));
      }
    }
  }
}

}  // namespace
}  // namespace swapnet
