// Decoder-layer kernels: embedding gather (zero-copy from the host-resident
// table), RMSNorm, RoPE + KV-cache append, causal attention with an online
// softmax, row argmax, and the device-side advance of the cache position.
// bf16 / fp16 storage, fp32 arithmetic, fixed reduction orders.
#include <cstring>

#include "device.cuh"
#include "internal.h"
#include "kernels.h"

namespace swapnet {

namespace {

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

int done(cudaError_t e, const char* what) {
  if (e == cudaSuccess) e = cudaGetLastError();
  if (e != cudaSuccess) SN_FAIL(SWAPNET_ERR_CUDA, std::string(what) + ": " + cudaGetErrorString(e));
  return SWAPNET_OK;
}

// ------------------------------------------------------------ embedding
// Row t of the output is row ids[t] of the table, read straight from the
// page-locked host table (device alias) with 16-byte loads.
template <typename T>
__global__ void __launch_bounds__(256) embed_kernel(const T* __restrict__ table, const int* __restrict__ ids,
                                                    int vocab, int d, T* __restrict__ out, int* err) {
  pdl_wait();
  pdl_launch_dependents();
  const int t = blockIdx.x;
  const int id = ids[t];
  const bool ok = id >= 0 && id < vocab;
  if (!ok && threadIdx.x == 0) atomicExch(err, kDevErrBounds);
  const uint4* src = reinterpret_cast<const uint4*>(table + (int64_t)(ok ? id : 0) * d);
  uint4* dst = reinterpret_cast<uint4*>(out + (int64_t)t * d);
  const int n16 = d * (int)sizeof(T) / 16;
  for (int i = threadIdx.x; i < n16; i += blockDim.x) dst[i] = ok ? src[i] : make_uint4(0, 0, 0, 0);
}

// ------------------------------------------------------------ RMSNorm
// One CTA per row; the sum of squares is reduced in a fixed order (each
// thread's elements in index order, warp butterfly, warps in index order).
// Rows of whole 16-byte chunks are read once into registers (up to
// kNormKeep chunks per thread, the rest read again for the scaling pass).
constexpr int kNormThreads = 256;
constexpr int kNormKeep = 4;

template <typename T> struct Chunk8 {
  static_assert(sizeof(T) == 2, "16-bit element types");
  __device__ static void unpack(const uint4& v, float* f) {
    const T* e = reinterpret_cast<const T*>(&v);
#pragma unroll
    for (int i = 0; i < 8; ++i) f[i] = to_f<T>(e[i]);
  }
  __device__ static uint4 pack(const float* f) {
    uint4 v;
    T* e = reinterpret_cast<T*>(&v);
#pragma unroll
    for (int i = 0; i < 8; ++i) e[i] = from_f<T>(f[i]);
    return v;
  }
};

template <typename T>
__global__ void __launch_bounds__(kNormThreads) rmsnorm_kernel(const T* __restrict__ x, const T* __restrict__ g,
                                                               int d, float eps, T* __restrict__ y, int vec) {
  __shared__ float wsum[kNormThreads / 32];
  pdl_wait();
  pdl_launch_dependents();
  const T* xr = x + (int64_t)blockIdx.x * d;
  T* yr = y + (int64_t)blockIdx.x * d;
  const int t = threadIdx.x;
  float s = 0.f;
  uint4 keep[kNormKeep];
  const int nc = d / 8;
  if (vec) {
    const uint4* xv = reinterpret_cast<const uint4*>(xr);
#pragma unroll
    for (int j = 0; j < kNormKeep; ++j) {
      const int c = t + j * kNormThreads;
      keep[j] = c < nc ? xv[c] : make_uint4(0u, 0u, 0u, 0u);
    }
#pragma unroll
    for (int j = 0; j < kNormKeep; ++j) {
      float f[8];
      Chunk8<T>::unpack(keep[j], f);
#pragma unroll
      for (int i = 0; i < 8; ++i) s = fmaf(f[i], f[i], s);
    }
    for (int c = t + kNormKeep * kNormThreads; c < nc; c += kNormThreads) {
      float f[8];
      Chunk8<T>::unpack(xv[c], f);
#pragma unroll
      for (int i = 0; i < 8; ++i) s = fmaf(f[i], f[i], s);
    }
  } else {
    for (int i = t; i < d; i += kNormThreads) {
      const float v = to_f<T>(xr[i]);
      s = fmaf(v, v, s);
    }
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
  if ((t & 31) == 0) wsum[t >> 5] = s;
  __syncthreads();
  float tot = 0.f;
#pragma unroll
  for (int w = 0; w < kNormThreads / 32; ++w) tot += wsum[w];
  const float r = 1.0f / sqrtf(tot / (float)d + eps);
  if (vec) {
    const uint4* xv = reinterpret_cast<const uint4*>(xr);
    const uint4* gv = reinterpret_cast<const uint4*>(g);
    uint4* yv = reinterpret_cast<uint4*>(yr);
    auto scale = [&](int c, const uint4& xc) {
      float f[8], gf[8], o[8];
      Chunk8<T>::unpack(xc, f);
      Chunk8<T>::unpack(gv[c], gf);
#pragma unroll
      for (int i = 0; i < 8; ++i) o[i] = f[i] * r * gf[i];
      yv[c] = Chunk8<T>::pack(o);
    };
#pragma unroll
    for (int j = 0; j < kNormKeep; ++j)
      if (t + j * kNormThreads < nc) scale(t + j * kNormThreads, keep[j]);
    for (int c = t + kNormKeep * kNormThreads; c < nc; c += kNormThreads) scale(c, xv[c]);
  } else {
    for (int i = t; i < d; i += kNormThreads) yr[i] = from_f<T>(to_f<T>(xr[i]) * r * to_f<T>(g[i]));
  }
}

// ------------------------------------------------------------ RoPE + cache
// Thread = one adjacent pair (2i, 2i+1) of one head of one token: rotates
// q in place and k into the key cache at the state position, copies v into
// the value cache.  Angles: position * theta^(-2i/Dh), computed in fp32.
template <typename T>
__global__ void __launch_bounds__(256) rope_append_kernel(T* __restrict__ q, const T* __restrict__ k,
                                                          const T* __restrict__ v, T* __restrict__ kc,
                                                          T* __restrict__ vc, const int* __restrict__ pos_ptr,
                                                          int width, int dh, float theta, int max_seq, int* err) {
  pdl_wait();
  pdl_launch_dependents();
  const int t = blockIdx.y;
  const int pair = blockIdx.x * blockDim.x + threadIdx.x;  // over width / 2
  if (pair >= width / 2) return;
  const int pos = *pos_ptr + t;
  if (pos >= max_seq) {
    if (pair == 0) atomicExch(err, kDevErrBounds);
    return;
  }
  const int col = 2 * pair;
  const int i = (col % dh) / 2;
  const float inv = powf(theta, -2.0f * (float)i / (float)dh);
  float sn, cs;
  sincosf((float)pos * inv, &sn, &cs);
  T* qp = q + (int64_t)t * width + col;
  const float q0 = to_f<T>(qp[0]), q1 = to_f<T>(qp[1]);
  qp[0] = from_f<T>(q0 * cs - q1 * sn);
  qp[1] = from_f<T>(q0 * sn + q1 * cs);
  const T* kp = k + (int64_t)t * width + col;
  const float k0 = to_f<T>(kp[0]), k1 = to_f<T>(kp[1]);
  T* kd = kc + (int64_t)pos * width + col;
  kd[0] = from_f<T>(k0 * cs - k1 * sn);
  kd[1] = from_f<T>(k0 * sn + k1 * cs);
  const T* vp = v + (int64_t)t * width + col;
  T* vd = vc + (int64_t)pos * width + col;
  vd[0] = vp[0];
  vd[1] = vp[1];
}

// ------------------------------------------------------------ attention
// Runs of at least 64 queries (the prefill) take the tcgen05 kernel
// (k_attn_tc.cu).  Shorter runs take one of two SIMT kernels with the same
// arithmetic definition: fewer than kRowsMinWarps (query, head) pairs (a
// decode step) the CTA kernel, more the warp kernel.
//
// Short query runs: CTA = one (query t, head h), 512 threads; the scores of all visible keys
// live in shared memory, so the softmax is exact two-pass (max, then
// exponentials and their sum) rather than online:
//   phase 1: thread j computes key j's score (the whole 128-wide dot product
//            from 16 independent 16-byte loads of its cache row);
//   phase 2: block max, p_j = exp(s_j - max), block sum l in a fixed order;
//   phase 3: thread (pair d, group g) accumulates p_j * v_j[2d..2d+1] over
//            keys j = g, g + 8, ... (coalesced 4-byte loads along the row);
//            the 8 groups are added in index order and divided by l.
// Every key load of a phase is independent of the others, so a decode step
// (one query, keys in HBM) is bound by a few memory round trips, not by a
// chain of one round trip per key.
constexpr int kDh = 128;
constexpr int kAttThreads = 512;
constexpr int kAttGroups = kAttThreads / (kDh / 2);
constexpr int kRowsMinWarps = 1024;

__device__ __forceinline__ float block_reduce(float v, float* red, bool is_max) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const float o = __shfl_xor_sync(0xffffffffu, v, off);
    v = is_max ? fmaxf(v, o) : v + o;
  }
  __syncthreads();  // red is reused between calls
  if (lane == 0) red[warp] = v;
  __syncthreads();
  float r = red[0];
  for (int w = 1; w < kAttThreads / 32; ++w) r = is_max ? fmaxf(r, red[w]) : r + red[w];
  return r;
}

template <typename T>
__global__ void __launch_bounds__(kAttThreads) attention_kernel(const T* __restrict__ q, const T* __restrict__ kc,
                                                                const T* __restrict__ vc,
                                                                const int* __restrict__ pos_ptr, int heads,
                                                                int width, int max_seq, T* __restrict__ out) {
  extern __shared__ float att_smem[];
  float2* part = reinterpret_cast<float2*>(att_smem);          // kAttGroups x kDh/2 partial sums
  float* red = att_smem + 2 * kAttGroups * (kDh / 2);          // kAttThreads / 32 partials
  float* qs = red + kAttThreads / 32;                          // kDh query values
  float* sc = qs + kDh;                                        // max_seq scores
  pdl_wait();
  pdl_launch_dependents();
  const int h = blockIdx.x, t = blockIdx.y;
  const int tid = threadIdx.x;
  const int n = min(*pos_ptr + t + 1, max_seq);
  const int64_t col = (int64_t)h * kDh;
  if (tid < kDh) qs[tid] = to_f<T>(q[(int64_t)t * width + col + tid]);
  __syncthreads();
  const float scale = rsqrtf((float)kDh);
  float mx = -INFINITY;
  for (int j = tid; j < n; j += kAttThreads) {
    const uint4* kr = reinterpret_cast<const uint4*>(kc + (int64_t)j * width + col);
    uint4 u[kDh / 8];
#pragma unroll
    for (int i = 0; i < kDh / 8; ++i) u[i] = kr[i];
    float s = 0.f;
#pragma unroll
    for (int i = 0; i < kDh / 8; ++i) {
      const T* e = reinterpret_cast<const T*>(&u[i]);
#pragma unroll
      for (int k = 0; k < 8; ++k) s = fmaf(qs[i * 8 + k], to_f<T>(e[k]), s);
    }
    s *= scale;
    sc[j] = s;
    mx = fmaxf(mx, s);
  }
  mx = block_reduce(mx, red, true);
  float l = 0.f;
  for (int j = tid; j < n; j += kAttThreads) {
    const float p = expf(sc[j] - mx);
    sc[j] = p;
    l += p;
  }
  l = block_reduce(l, red, false);  // the barriers inside also publish sc[]
  const int d2 = tid % (kDh / 2), g = tid / (kDh / 2);
  const T* vcol = vc + col + 2 * d2;
  float a0 = 0.f, a1 = 0.f;
  int j = g;
#pragma unroll 1
  for (; j + 3 * kAttGroups < n; j += 4 * kAttGroups) {
    uint32_t w[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) w[i] = *reinterpret_cast<const uint32_t*>(vcol + (int64_t)(j + i * kAttGroups) * width);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const T* e = reinterpret_cast<const T*>(&w[i]);
      const float p = sc[j + i * kAttGroups];
      a0 = fmaf(p, to_f<T>(e[0]), a0);
      a1 = fmaf(p, to_f<T>(e[1]), a1);
    }
  }
  for (; j < n; j += kAttGroups) {
    const uint32_t w = *reinterpret_cast<const uint32_t*>(vcol + (int64_t)j * width);
    const T* e = reinterpret_cast<const T*>(&w);
    const float p = sc[j];
    a0 = fmaf(p, to_f<T>(e[0]), a0);
    a1 = fmaf(p, to_f<T>(e[1]), a1);
  }
  part[g * (kDh / 2) + d2] = make_float2(a0, a1);
  __syncthreads();
  if (tid < kDh / 2) {
    float o0 = 0.f, o1 = 0.f;
    for (int gg = 0; gg < kAttGroups; ++gg) {
      const float2 v = part[gg * (kDh / 2) + tid];
      o0 += v.x;
      o1 += v.y;
    }
    const float inv = 1.0f / l;
    T* o = out + (int64_t)t * width + col + 2 * tid;
    o[0] = from_f<T>(o0 * inv);
    o[1] = from_f<T>(o1 * inv);
  }
}

// Long query runs (prefill): warp = one (query, head), each lane holding 4
// of the 128 head dimensions; keys are visited in position order with an
// online softmax in fp32 (m running max, l running denominator, acc running
// numerator).  With hundreds of queries per head there are enough warps to
// hide each warp's chain of one memory round trip per key.
template <typename T>
__device__ __forceinline__ void load4(const T* p, float* f) {
  const uint2 u = *reinterpret_cast<const uint2*>(p);
  const T* e = reinterpret_cast<const T*>(&u);
#pragma unroll
  for (int j = 0; j < 4; ++j) f[j] = to_f<T>(e[j]);
}

template <typename T>
__global__ void __launch_bounds__(256) attention_rows_kernel(const T* __restrict__ q, const T* __restrict__ kc,
                                                             const T* __restrict__ vc,
                                                             const int* __restrict__ pos_ptr, int T_, int heads,
                                                             int width, int max_seq, T* __restrict__ out) {
  pdl_wait();
  pdl_launch_dependents();
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (warp >= T_ * heads) return;
  const int t = warp / heads, h = warp % heads;
  const int n = min(*pos_ptr + t + 1, max_seq);
  const int c0 = h * kDh + lane * 4;
  float qv[4];
  load4<T>(q + (int64_t)t * width + c0, qv);
  const float scale = rsqrtf((float)kDh);
  float m = -INFINITY, l = 0.f, acc[4] = {0.f, 0.f, 0.f, 0.f};
  for (int j = 0; j < n; ++j) {
    float kv[4];
    load4<T>(kc + (int64_t)j * width + c0, kv);
    float s = qv[0] * kv[0] + qv[1] * kv[1] + qv[2] * kv[2] + qv[3] * kv[3];
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
    s *= scale;
    const float mn = fmaxf(m, s);
    const float a = expf(m - mn);   // 0 on the first key (m = -inf)
    const float p = expf(s - mn);
    float vv[4];
    load4<T>(vc + (int64_t)j * width + c0, vv);
    l = l * a + p;
#pragma unroll
    for (int d = 0; d < 4; ++d) acc[d] = acc[d] * a + p * vv[d];
    m = mn;
  }
  const float inv = 1.0f / l;
  T* o = out + (int64_t)t * width + c0;
#pragma unroll
  for (int d = 0; d < 4; ++d) o[d] = from_f<T>(acc[d] * inv);
}

size_t attention_smem_bytes(int max_seq) {
  return sizeof(float) * ((size_t)max_seq + kDh + kAttThreads / 32) + sizeof(float2) * kAttGroups * (kDh / 2);
}

// ------------------------------------------------------------ argmax
// One CTA per row.  Each thread scans its elements in index order keeping
// the first maximum; threads, then warps, are combined by (larger value,
// then smaller index), an order-independent rule, so ties go to the
// lowest index.  Rows of whole 16-byte chunks are read kArgBatch chunks
// per thread at a time.
constexpr int kArgThreads = 1024;
constexpr int kArgBatch = 4;

__device__ __forceinline__ void arg_take(float& best, int& bi, float ov, int oi) {
  if (ov > best || (ov == best && oi < bi)) {
    best = ov;
    bi = oi;
  }
}

template <typename T>
__global__ void __launch_bounds__(kArgThreads) argmax_kernel(const T* __restrict__ x, int n, int* __restrict__ out,
                                                             int vec) {
  __shared__ float sv[kArgThreads / 32];
  __shared__ int si[kArgThreads / 32];
  pdl_wait();
  pdl_launch_dependents();
  const T* row = x + (int64_t)blockIdx.x * n;
  const int t = threadIdx.x;
  float best = -INFINITY;
  int bi = 0x7fffffff;
  if (vec) {
    const uint4* rv = reinterpret_cast<const uint4*>(row);
    const int nc = n / 8;
    for (int c0 = t; c0 < nc; c0 += kArgBatch * kArgThreads) {
      uint4 v[kArgBatch];
#pragma unroll
      for (int u = 0; u < kArgBatch; ++u) {
        const int c = c0 + u * kArgThreads;
        v[u] = c < nc ? rv[c] : make_uint4(0u, 0u, 0u, 0u);
      }
#pragma unroll
      for (int u = 0; u < kArgBatch; ++u) {
        const int c = c0 + u * kArgThreads;
        if (c < nc) {
          float f[8];
          Chunk8<T>::unpack(v[u], f);
#pragma unroll
          for (int i = 0; i < 8; ++i)
            if (f[i] > best) {  // strictly greater: the first index wins
              best = f[i];
              bi = c * 8 + i;
            }
        }
      }
    }
  } else {
    for (int j = t; j < n; j += kArgThreads) {
      const float v = to_f<T>(row[j]);
      if (v > best) {
        best = v;
        bi = j;
      }
    }
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1)
    arg_take(best, bi, __shfl_xor_sync(0xffffffffu, best, off), __shfl_xor_sync(0xffffffffu, bi, off));
  if ((t & 31) == 0) {
    sv[t >> 5] = best;
    si[t >> 5] = bi;
  }
  __syncthreads();
  if (t < 32) {
    best = sv[t];
    bi = si[t];
#pragma unroll
    for (int off = 16; off > 0; off >>= 1)
      arg_take(best, bi, __shfl_xor_sync(0xffffffffu, best, off), __shfl_xor_sync(0xffffffffu, bi, off));
    if (t == 0) out[blockIdx.x] = bi == 0x7fffffff ? 0 : bi;
  }
}

__global__ void advance_kernel(int* pos_ptr, int n) {
  pdl_wait();
  pdl_launch_dependents();
  *pos_ptr += n;
}

}  // namespace

#define SN_DISPATCH16(dtype, T, ...)                                     \
  switch (dtype) {                                                       \
    case SWAPNET_F16: { using T = __half; __VA_ARGS__; break; }          \
    case SWAPNET_BF16: { using T = __nv_bfloat16; __VA_ARGS__; break; }  \
    default: SN_FAIL(SWAPNET_ERR_UNSUPPORTED, "decoder kernels: fp16 / bf16 only"); \
  }

int launch_embed(int dtype, const void* table, const int* ids, int tokens, int vocab, int d, void* out, int* err,
                 cudaStream_t s) {
  if ((d * 2) % 16 || ((uintptr_t)table | (uintptr_t)out) % 16)
    SN_FAIL(SWAPNET_ERR_MISALIGNED, "embedding rows must be 16-byte aligned");
  SN_DISPATCH16(dtype, T, return done(launch_pdl(embed_kernel<T>, dim3(tokens), dim3(256), 0, s,
                                                 static_cast<const T*>(table), ids, vocab, d,
                                                 static_cast<T*>(out), err), "embedding launch"));
  return SWAPNET_OK;
}

int launch_rmsnorm(int dtype, const void* x, const void* g, int rows, int d, float eps, void* y, cudaStream_t s) {
  const int vec = d % 8 == 0 && (((uintptr_t)x | (uintptr_t)g | (uintptr_t)y) & 15) == 0;
  SN_DISPATCH16(dtype, T, return done(launch_pdl(rmsnorm_kernel<T>, dim3(rows), dim3(kNormThreads), 0, s,
                                                 static_cast<const T*>(x), static_cast<const T*>(g), d, eps,
                                                 static_cast<T*>(y), vec), "rmsnorm launch"));
  return SWAPNET_OK;
}

int launch_attention(int dtype, void* q, const void* k, const void* v, void* kc, void* vc, const int* pos_ptr,
                     int tokens, int heads, int width, float theta, int max_seq, void* out, int* err,
                     cudaStream_t s) {
  if (width % heads || width / heads != kDh) SN_FAIL(SWAPNET_ERR_UNSUPPORTED, "attention: head width must be 128");
  SN_DISPATCH16(dtype, T, {
    const dim3 g1((width / 2 + 255) / 256, tokens);
    int rc = done(launch_pdl(rope_append_kernel<T>, g1, dim3(256), 0, s, static_cast<T*>(q),
                             static_cast<const T*>(k), static_cast<const T*>(v), static_cast<T*>(kc),
                             static_cast<T*>(vc), pos_ptr, width, kDh, theta, max_seq, err),
                  "rope launch");
    if (rc) return rc;
    if (attention_tc_supported(dtype, tokens, heads, width))  // prefill: both contractions on the tensor cores
      return launch_attention_tc(dtype, q, kc, vc, pos_ptr, tokens, heads, width, max_seq, out, err, s);
    if (tokens * heads >= kRowsMinWarps) {
      const int warps = tokens * heads;
      return done(launch_pdl(attention_rows_kernel<T>, dim3((warps * 32 + 255) / 256), dim3(256), 0, s,
                             static_cast<const T*>(q), static_cast<const T*>(kc), static_cast<const T*>(vc),
                             pos_ptr, tokens, heads, width, max_seq, static_cast<T*>(out)),
                  "attention launch");
    }
    const size_t smem = attention_smem_bytes(max_seq);
    if (smem > 48 * 1024) {
      cudaError_t e = cudaFuncSetAttribute(attention_kernel<T>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           (int)smem);
      if (e != cudaSuccess) return done(e, "attention shared memory");
    }
    return done(launch_pdl(attention_kernel<T>, dim3(heads, tokens), dim3(kAttThreads), smem, s,
                           static_cast<const T*>(q), static_cast<const T*>(kc), static_cast<const T*>(vc),
                           pos_ptr, heads, width, max_seq, static_cast<T*>(out)),
                "attention launch");
  });
  return SWAPNET_OK;
}

int launch_argmax(int dtype, const void* x, int rows, int n, int* out, cudaStream_t s) {
  const int vec = n % 8 == 0 && ((uintptr_t)x & 15) == 0;
  SN_DISPATCH16(dtype, T, return done(launch_pdl(argmax_kernel<T>, dim3(rows), dim3(kArgThreads), 0, s,
                                                 static_cast<const T*>(x), n, out, vec), "argmax launch"));
  return SWAPNET_OK;
}

int launch_advance(int* pos_ptr, int n, cudaStream_t s) {
  return done(launch_pdl(advance_kernel, dim3(1), dim3(1), 0, s, pos_ptr, n), "position advance launch");
}

}  // namespace swapnet
