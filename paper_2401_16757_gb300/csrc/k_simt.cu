// SIMT layer kernels: skinny linear (M <= 16, HBM-bound GEMV family),
// direct convolution for channel counts the tensor-core path cannot tile,
// pooling, upsampling and channel concatenation.  NHWC everywhere.
#include <cstdio>
#include <cstring>

#include "device.cuh"
#include "internal.h"
#include "kernels.h"

namespace swapnet {

namespace {

template <typename T> struct Vec16 { static constexpr int N = 16 / sizeof(T); };

// Launch with programmatic stream serialization: the kernel may start while
// the previous kernel on the stream drains; it waits (pdl_wait) before
// reading that kernel's output.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s, Args... args) {
  cudaLaunchConfig_t cfg;
  std::memset(&cfg, 0, sizeof(cfg));
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, static_cast<KArgs>(args)...);
}

__device__ __forceinline__ uint4 ld_stream16(const void* p) {
  uint4 r;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p));
  return r;
}

template <typename T> __device__ __forceinline__ void unpack16(const uint4& v, float* f) {
  const T* e = reinterpret_cast<const T*>(&v);
#pragma unroll
  for (int i = 0; i < Vec16<T>::N; ++i) f[i] = to_f<T>(e[i]);
}

template <typename T> __device__ __forceinline__ uint4 pack16(const float* f) {
  uint4 v;
  T* e = reinterpret_cast<T*>(&v);
#pragma unroll
  for (int i = 0; i < Vec16<T>::N; ++i) e[i] = from_f<T>(f[i]);
  return v;
}

// ------------------------------------------------------------ skinny linear
// One warp per output feature, for all M rows: lane l reads the 16-byte
// chunks l, l+32, ... of the feature's weight row, kSkBatch loads in flight
// per lane, and keeps one fp32 partial sum per row in chunk order; a
// butterfly combines the lanes, so the result does not depend on
// scheduling.  The weights do not depend on the kernel before (they are in
// place before this kernel is launched), so the first batch is requested
// before the programmatic wait and overlaps that kernel's drain.
constexpr int kSkWarps = 8;
constexpr int kSkBatch = 8;

template <typename T, int MT>
__global__ void __launch_bounds__(kSkWarps * 32) linear_skinny_kernel(const T* __restrict__ x, int M, int K,
                                                                      const T* __restrict__ W, int N, Epi e,
                                                                      T* __restrict__ y, int64_t ldy) {
  constexpr int V = Vec16<T>::N;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int o = blockIdx.x * kSkWarps + warp;
  const int kchunks = K / V;  // K % V == 0 (checked on the host)
  const T* wrow = W + (int64_t)min(o, N - 1) * K;
  uint4 wv[kSkBatch];
  auto load_batch = [&](int c0) {
#pragma unroll
    for (int u = 0; u < kSkBatch; ++u) {
      const int ch = c0 + u * 32;
      wv[u] = ch < kchunks ? ld_stream16(wrow + (int64_t)ch * V) : make_uint4(0u, 0u, 0u, 0u);
    }
  };
  if (o < N) load_batch(lane);
  pdl_wait();
  pdl_launch_dependents();
  if (o >= N) return;
  float acc[MT];
#pragma unroll
  for (int m = 0; m < MT; ++m) acc[m] = 0.f;
  for (int c0 = lane; c0 < kchunks; c0 += 32 * kSkBatch) {
    if (c0 != lane) load_batch(c0);
#pragma unroll
    for (int u = 0; u < kSkBatch; ++u) {
      const int ch = c0 + u * 32;
      if (ch < kchunks) {
        float wf[V];
        unpack16<T>(wv[u], wf);
#pragma unroll
        for (int m = 0; m < MT; ++m) {
          if (m < M) {
            float xv[V];
            unpack16<T>(__ldg(reinterpret_cast<const uint4*>(x + (int64_t)m * K + (int64_t)ch * V)), xv);
#pragma unroll
            for (int i = 0; i < V; ++i) acc[m] = fmaf(wf[i], xv[i], acc[m]);
          }
        }
      }
    }
  }
  const float b = e.bias ? to_f<T>(reinterpret_cast<const T*>(e.bias)[o]) : 0.f;
#pragma unroll
  for (int m = 0; m < MT; ++m) {
    float v = acc[m];
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
    if (lane == m && m < M) {
      float r = 0.f;
      if (e.res) r = to_f<T>(reinterpret_cast<const T*>(e.res)[(int64_t)m * e.ldr + o]);
      y[(int64_t)m * ldy + o] = from_f<T>(epilogue(v, b, r, e.res != nullptr, e.act, e.res_post));
    }
  }
}

template <typename T>
int skinny_dispatch(const void* x, int M, int K, const void* W, int N, const Epi& e, void* y, int64_t ldy,
                    cudaStream_t s) {
  const dim3 grid((N + kSkWarps - 1) / kSkWarps), block(kSkWarps * 32);
  const T* xp = static_cast<const T*>(x);
  const T* wp = static_cast<const T*>(W);
  T* yp = static_cast<T*>(y);
  if (M <= 1) launch_pdl(linear_skinny_kernel<T, 1>, grid, block, 0, s, xp, M, K, wp, N, e, yp, ldy);
  else if (M <= 2) launch_pdl(linear_skinny_kernel<T, 2>, grid, block, 0, s, xp, M, K, wp, N, e, yp, ldy);
  else if (M <= 4) launch_pdl(linear_skinny_kernel<T, 4>, grid, block, 0, s, xp, M, K, wp, N, e, yp, ldy);
  else if (M <= 8) launch_pdl(linear_skinny_kernel<T, 8>, grid, block, 0, s, xp, M, K, wp, N, e, yp, ldy);
  else launch_pdl(linear_skinny_kernel<T, 16>, grid, block, 0, s, xp, M, K, wp, N, e, yp, ldy);
  return cudaGetLastError() == cudaSuccess ? SWAPNET_OK : SWAPNET_ERR_CUDA;
}

// ------------------------------------------------------------ tiled linear
// General fallback for any M, K, N and dtype: 64 x 64 output tile per CTA,
// 16 x 16 threads with 4 x 4 outputs each, K staged through shared memory
// in steps of 16, fp32 accumulation in a fixed order.
template <typename T>
__global__ void __launch_bounds__(256) linear_tiled_kernel(const T* __restrict__ x, int M, int K,
                                                           const T* __restrict__ W, int N, Epi e,
                                                           T* __restrict__ y, int64_t ldy) {
  __shared__ float xs[16][64 + 1];
  __shared__ float ws[16][64 + 1];
  pdl_wait();
  pdl_launch_dependents();
  const int tx = threadIdx.x % 16, ty = threadIdx.x / 16;
  const int m0 = blockIdx.y * 64, n0 = blockIdx.x * 64;
  float acc[4][4] = {};
  for (int k0 = 0; k0 < K; k0 += 16) {
    for (int i = threadIdx.x; i < 16 * 64; i += 256) {
      const int kk = i % 16, r = i / 16;
      const int m = m0 + r, n = n0 + r, k = k0 + kk;
      xs[kk][r] = (m < M && k < K) ? to_f<T>(x[(int64_t)m * K + k]) : 0.f;
      ws[kk][r] = (n < N && k < K) ? to_f<T>(W[(int64_t)n * K + k]) : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < 16; ++kk) {
      float a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) { a[i] = xs[kk][ty + 16 * i]; b[i] = ws[kk][tx + 16 * i]; }
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
  const T* bias = reinterpret_cast<const T*>(e.bias);
  const T* res = reinterpret_cast<const T*>(e.res);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int m = m0 + ty + 16 * i;
    if (m >= M) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int n = n0 + tx + 16 * j;
      if (n >= N) continue;
      const float rv = res ? to_f<T>(res[(int64_t)m * e.ldr + n]) : 0.f;
      y[(int64_t)m * ldy + n] =
          from_f<T>(epilogue(acc[i][j], bias ? to_f<T>(bias[n]) : 0.f, rv, res != nullptr, e.act, e.res_post));
    }
  }
}

// ------------------------------------------------------------ direct conv
// Thread = one output pixel x 16 output channels.  The CTA's 16 filters are
// staged in shared memory as fp32, laid out [tap][cin][16] so each input
// value meets 16 weights read as four broadcast float4 loads.  Used for
// channel counts the tensor-core path cannot tile (e.g. a 3-channel image).
constexpr int kDcCo = 16;

template <typename T>
__global__ void __launch_bounds__(128) conv_direct_kernel(const T* __restrict__ x, int n, int h, int w, int cin,
                                                          const T* __restrict__ W, int cout, int kh, int kw,
                                                          int stride, int pad, int oh, int ow, Epi e,
                                                          T* __restrict__ y) {
  extern __shared__ float ws[];  // [kh*kw*cin][kDcCo]
  const int co0 = blockIdx.y * kDcCo;
  const int taps = kh * kw * cin;
  for (int i = threadIdx.x; i < taps * kDcCo; i += blockDim.x) {
    const int j = i % kDcCo, tc = i / kDcCo;  // tc = (r*kw + s)*cin + c
    const int co = co0 + j;
    ws[i] = co < cout ? to_f<T>(W[(int64_t)co * taps + tc]) : 0.f;
  }
  pdl_wait();  // the filters come from the arena; the input from the previous kernel
  pdl_launch_dependents();
  __syncthreads();
  const int64_t pix = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t npix = (int64_t)n * oh * ow;
  if (pix >= npix) return;
  const int img = (int)(pix / ((int64_t)oh * ow));
  const int rem = (int)(pix % ((int64_t)oh * ow));
  const int oy = rem / ow, ox = rem % ow;
  float acc[kDcCo];
#pragma unroll
  for (int j = 0; j < kDcCo; ++j) acc[j] = 0.f;
  for (int r = 0; r < kh; ++r) {
    const int iy = oy * stride + r - pad;
    if (iy < 0 || iy >= h) continue;
    for (int s = 0; s < kw; ++s) {
      const int ix = ox * stride + s - pad;
      if (ix < 0 || ix >= w) continue;
      const T* xp = x + (((int64_t)img * h + iy) * w + ix) * cin;
      const float4* wp = reinterpret_cast<const float4*>(ws + (int64_t)((r * kw + s) * cin) * kDcCo);
      for (int c = 0; c < cin; ++c) {
        const float xv = to_f<T>(xp[c]);
#pragma unroll
        for (int q = 0; q < kDcCo / 4; ++q) {
          const float4 wv = wp[c * (kDcCo / 4) + q];
          acc[4 * q + 0] = fmaf(xv, wv.x, acc[4 * q + 0]);
          acc[4 * q + 1] = fmaf(xv, wv.y, acc[4 * q + 1]);
          acc[4 * q + 2] = fmaf(xv, wv.z, acc[4 * q + 2]);
          acc[4 * q + 3] = fmaf(xv, wv.w, acc[4 * q + 3]);
        }
      }
    }
  }
  const T* bias = reinterpret_cast<const T*>(e.bias);
  const T* res = reinterpret_cast<const T*>(e.res);
#pragma unroll
  for (int j = 0; j < kDcCo; ++j) {
    const int co = co0 + j;
    if (co < cout) {
      const float rv = res ? to_f<T>(res[pix * e.ldr + co]) : 0.f;
      y[pix * cout + co] =
        from_f<T>(epilogue(acc[j], bias ? to_f<T>(bias[co]) : 0.f, rv, res != nullptr, e.act, e.res_post));
    }
  }
}

// ------------------------------------------------------------ pooling etc.
template <typename T>
__global__ void maxpool_kernel(const T* __restrict__ x, int n, int h, int w, int c, int kh, int kw, int stride,
                               int pad, int oh, int ow, T* __restrict__ y) {
  pdl_wait();
  pdl_launch_dependents();
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t total = (int64_t)n * oh * ow * c;
  if (idx >= total) return;
  const int ch = (int)(idx % c);
  const int64_t p = idx / c;
  const int ox = (int)(p % ow);
  const int oy = (int)((p / ow) % oh);
  const int img = (int)(p / ((int64_t)ow * oh));
  float m = -INFINITY;
  for (int r = 0; r < kh; ++r) {
    const int iy = oy * stride + r - pad;
    if (iy < 0 || iy >= h) continue;
    for (int s = 0; s < kw; ++s) {
      const int ix = ox * stride + s - pad;
      if (ix < 0 || ix >= w) continue;
      m = fmaxf(m, to_f<T>(x[(((int64_t)img * h + iy) * w + ix) * c + ch]));
    }
  }
  y[idx] = from_f<T>(m);
}

template <typename T>
__global__ void gap_kernel(const T* __restrict__ x, int n, int hw, int c, T* __restrict__ y) {
  pdl_wait();
  pdl_launch_dependents();
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= (int64_t)n * c) return;
  const int img = (int)(idx / c), ch = (int)(idx % c);
  const T* p = x + (int64_t)img * hw * c + ch;
  float s = 0.f;
  for (int i = 0; i < hw; ++i) s += to_f<T>(p[(int64_t)i * c]);
  y[idx] = from_f<T>(s / (float)hw);
}

template <typename T>
__global__ void upsample2x_kernel(const T* __restrict__ x, int n, int h, int w, int c, T* __restrict__ y) {
  pdl_wait();
  pdl_launch_dependents();
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t total = (int64_t)n * 2 * h * 2 * w * c;
  if (idx >= total) return;
  const int ch = (int)(idx % c);
  const int64_t p = idx / c;
  const int ox = (int)(p % (2 * w));
  const int oy = (int)((p / (2 * w)) % (2 * h));
  const int img = (int)(p / ((int64_t)4 * w * h));
  y[idx] = x[(((int64_t)img * h + oy / 2) * w + ox / 2) * c + ch];
}

template <typename T>
__global__ void concat_kernel(const T* __restrict__ a, int ca, const T* __restrict__ b, int cb, int64_t pixels,
                              T* __restrict__ y) {
  pdl_wait();
  pdl_launch_dependents();
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int c = ca + cb;
  if (idx >= pixels * c) return;
  const int64_t p = idx / c;
  const int ch = (int)(idx % c);
  y[idx] = ch < ca ? a[p * ca + ch] : b[p * cb + (ch - ca)];
}

// Vectorised variants: a thread handles 16 bytes of channels (channels a
// multiple of the vector width, rows 16-byte aligned).  Max is exact, so
// the result equals the scalar kernels'.
template <typename T>
__global__ void maxpool_vec_kernel(const uint4* __restrict__ x, int n, int h, int w, int cv, int kh, int kw,
                                   int stride, int pad, int oh, int ow, uint4* __restrict__ y) {
  constexpr int V = Vec16<T>::N;
  pdl_wait();
  pdl_launch_dependents();
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t total = (int64_t)n * oh * ow * cv;
  if (idx >= total) return;
  const int ch = (int)(idx % cv);
  const int64_t p = idx / cv;
  const int ox = (int)(p % ow);
  const int64_t q = p / ow;
  const int oy = (int)(q % oh);
  const int img = (int)(q / oh);
  float m[V];
#pragma unroll
  for (int i = 0; i < V; ++i) m[i] = -INFINITY;
  for (int r = 0; r < kh; ++r) {
    const int iy = oy * stride + r - pad;
    if (iy < 0 || iy >= h) continue;
    for (int s = 0; s < kw; ++s) {
      const int ix = ox * stride + s - pad;
      if (ix < 0 || ix >= w) continue;
      float f[V];
      unpack16<T>(__ldg(x + (((int64_t)img * h + iy) * w + ix) * cv + ch), f);
#pragma unroll
      for (int i = 0; i < V; ++i) m[i] = fmaxf(m[i], f[i]);
    }
  }
  y[idx] = pack16<T>(m);
}

__global__ void upsample2x_vec_kernel(const uint4* __restrict__ x, int n, int h, int w, int cv,
                                      uint4* __restrict__ y) {
  pdl_wait();
  pdl_launch_dependents();
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t total = (int64_t)n * 2 * h * 2 * w * cv;
  if (idx >= total) return;
  const int ch = (int)(idx % cv);
  const int64_t p = idx / cv;
  const int ox = (int)(p % (2 * w));
  const int64_t q = p / (2 * w);
  const int oy = (int)(q % (2 * h));
  const int img = (int)(q / (2 * h));
  y[idx] = x[(((int64_t)img * h + oy / 2) * w + ox / 2) * cv + ch];
}

__global__ void concat_vec_kernel(const uint4* __restrict__ a, int ca, const uint4* __restrict__ b, int cb,
                                  int64_t pixels, uint4* __restrict__ y) {
  pdl_wait();
  pdl_launch_dependents();
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int c = ca + cb;
  if (idx >= pixels * c) return;
  const int64_t p = idx / c;
  const int ch = (int)(idx % c);
  y[idx] = ch < ca ? a[p * ca + ch] : b[p * cb + (ch - ca)];
}

inline int grid1d(int64_t total, int block) { return (int)((total + block - 1) / block); }



}  // namespace

#define SN_DISPATCH(dtype, T, ...)                    \
  switch (dtype) {                                    \
    case SWAPNET_F32: { using T = float; __VA_ARGS__; break; }          \
    case SWAPNET_F16: { using T = __half; __VA_ARGS__; break; }         \
    case SWAPNET_BF16: { using T = __nv_bfloat16; __VA_ARGS__; break; } \
    default: return SWAPNET_ERR_INVALID_ARG;          \
  }

static int last_launch() {
  const cudaError_t err = cudaGetLastError();
  if (err != cudaSuccess) {
    set_error(std::string("kernel launch: ") + cudaGetErrorString(err));
    return SWAPNET_ERR_CUDA;
  }
  return SWAPNET_OK;
}

int launch_linear_skinny(int dtype, const void* x, int M, int K, const void* W, int N, const Epi& e, void* y,
                         int64_t ldy, cudaStream_t s) {
  const int es = dtype_size(dtype);
  if (M < 1 || M > 16 || K < 1 || N < 1) SN_FAIL(SWAPNET_ERR_UNSUPPORTED, "skinny linear: M must be in [1, 16]");
  if ((K * es) % 16 || ((uintptr_t)x | (uintptr_t)W) % 16)
    SN_FAIL(SWAPNET_ERR_MISALIGNED, "skinny linear: rows must be 16-byte aligned");
  SN_DISPATCH(dtype, T, return skinny_dispatch<T>(x, M, K, W, N, e, y, ldy, s));
  return SWAPNET_OK;
}

int launch_linear_tiled(int dtype, const void* x, int M, int K, const void* W, int N, const Epi& e, void* y,
                        int64_t ldy, cudaStream_t s) {
  if (M < 1 || K < 1 || N < 1) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "tiled linear: empty shape");
  const dim3 grid((N + 63) / 64, (M + 63) / 64);
  SN_DISPATCH(dtype, T,
              launch_pdl(linear_tiled_kernel<T>, grid, dim3(256), 0, s, static_cast<const T*>(x), M, K,
                         static_cast<const T*>(W), N, e, static_cast<T*>(y), ldy));
  return last_launch();
}

int launch_conv_direct(int dtype, const void* x, int n, int h, int w, int cin, const void* W, int cout, int kh,
                       int kw, int stride, int pad, int oh, int ow, const Epi& e, void* y, cudaStream_t s) {
  const int64_t npix = (int64_t)n * oh * ow;
  const size_t smem = (size_t)kh * kw * cin * kDcCo * sizeof(float);
  if (smem > 200 * 1024) SN_FAIL(SWAPNET_ERR_UNSUPPORTED, "direct conv: filter too large for shared memory");
  const dim3 grid(grid1d(npix, 128), (cout + kDcCo - 1) / kDcCo);
  SN_DISPATCH(dtype, T, {
    auto kern = conv_direct_kernel<T>;
    if (smem > 48 * 1024 &&
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
      SN_FAIL(SWAPNET_ERR_CUDA, "cudaFuncSetAttribute failed");
    launch_pdl(kern, grid, dim3(128), smem, s, static_cast<const T*>(x), n, h, w, cin, static_cast<const T*>(W), cout,
               kh, kw, stride, pad, oh, ow, e, static_cast<T*>(y));
  });
  return last_launch();
}

int launch_maxpool(int dtype, const void* x, int n, int h, int w, int c, int kh, int kw, int stride, int pad,
                   int oh, int ow, void* y, cudaStream_t s) {
  SN_DISPATCH(dtype, T, {
    constexpr int V = Vec16<T>::N;
    if (c % V == 0 && ((uintptr_t)x | (uintptr_t)y) % 16 == 0) {
      const int64_t tv = (int64_t)n * oh * ow * (c / V);
      launch_pdl(maxpool_vec_kernel<T>, dim3(grid1d(tv, 256)), dim3(256), 0, s, static_cast<const uint4*>(x), n, h,
                 w, c / V, kh, kw, stride, pad, oh, ow, static_cast<uint4*>(y));
      return last_launch();
    }
  });
  const int64_t total = (int64_t)n * oh * ow * c;
  SN_DISPATCH(dtype, T,
              launch_pdl(maxpool_kernel<T>, dim3(grid1d(total, 256)), dim3(256), 0, s, static_cast<const T*>(x), n, h,
                         w, c, kh, kw, stride, pad, oh, ow, static_cast<T*>(y)));
  return last_launch();
}

int launch_gap(int dtype, const void* x, int n, int h, int w, int c, void* y, cudaStream_t s) {
  SN_DISPATCH(dtype, T,
              launch_pdl(gap_kernel<T>, dim3(grid1d((int64_t)n * c, 256)), dim3(256), 0, s, static_cast<const T*>(x),
                         n, h * w, c, static_cast<T*>(y)));
  return last_launch();
}

int launch_upsample2x(int dtype, const void* x, int n, int h, int w, int c, void* y, cudaStream_t s) {
  {
    const int es = dtype == SWAPNET_F32 ? 4 : 2;
    if ((c * es) % 16 == 0 && ((uintptr_t)x | (uintptr_t)y) % 16 == 0) {
      const int cv = c * es / 16;
      launch_pdl(upsample2x_vec_kernel, dim3(grid1d((int64_t)n * 4 * h * w * cv, 256)), dim3(256), 0, s,
                 static_cast<const uint4*>(x), n, h, w, cv, static_cast<uint4*>(y));
      return last_launch();
    }
  }
  const int64_t total = (int64_t)n * 4 * h * w * c;
  SN_DISPATCH(dtype, T,
              launch_pdl(upsample2x_kernel<T>, dim3(grid1d(total, 256)), dim3(256), 0, s, static_cast<const T*>(x), n,
                         h, w, c, static_cast<T*>(y)));
  return last_launch();
}

int launch_concat(int dtype, const void* a, int ca, const void* b, int cb, int64_t pixels, void* y,
                  cudaStream_t s) {
  {
    const int es = dtype == SWAPNET_F32 ? 4 : 2;
    if ((ca * es) % 16 == 0 && (cb * es) % 16 == 0 && ((uintptr_t)a | (uintptr_t)b | (uintptr_t)y) % 16 == 0) {
      const int av = ca * es / 16, bv = cb * es / 16;
      launch_pdl(concat_vec_kernel, dim3(grid1d(pixels * (av + bv), 256)), dim3(256), 0, s,
                 static_cast<const uint4*>(a), av, static_cast<const uint4*>(b), bv, pixels,
                 static_cast<uint4*>(y));
      return last_launch();
    }
  }
  const int64_t total = pixels * (ca + cb);
  SN_DISPATCH(dtype, T,
              launch_pdl(concat_kernel<T>, dim3(grid1d(total, 256)), dim3(256), 0, s, static_cast<const T*>(a), ca,
                         static_cast<const T*>(b), cb, pixels, static_cast<T*>(y)));
  return last_launch();
}

}  // namespace swapnet
