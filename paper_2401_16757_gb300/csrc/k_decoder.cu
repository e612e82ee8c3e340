// Decoder-layer kernels: embedding gather (zero-copy from the host-resident
// table), RMSNorm, RoPE + KV-cache append, causal attention for short query
// runs (the decode step: keys split over a thread-block cluster) and for
// long runs the tensor cores do not take (warp per query, online softmax),
// row argmax, and the device-side advance of the cache position.
// bf16 / fp16 storage, fp32 arithmetic, fixed reduction orders.
#include <cooperative_groups.h>

#include <algorithm>
#include <cstring>

#include "device.cuh"
#include "internal.h"
#include "kernels.h"

namespace swapnet {

namespace cg = cooperative_groups;

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
// Short query runs (a decode step): the visible keys of one (query t,
// head h) are split into S consecutive chunks of `chunk` keys, one CTA per
// chunk, and the S CTAs of a (t, h) form a thread-block cluster.  Each CTA
// computes, over its chunk only (256 threads):
//   phase 1: scores s_j = q . k_j / sqrt(128): 16 threads per key, one
//            16-byte load each (8 head dims), summed over the 16 lanes in a
//            fixed butterfly order; 16 keys per pass, the loads of four
//            passes issued before their arithmetic;
//   phase 2: the chunk's max m_c, p_j = exp(s_j - m_c) and l_c = sum p_j
//            (block reductions in a fixed order);
//   phase 3: a_c[d] = sum_j p_j v_j[d]: thread (key group g, 8-dim slice)
//            over keys g, g + 16, ... with 16-byte loads (the first eight of
//            them issued before phase 1, so that they arrive during it),
//            then the 16 groups added in index order.
// After a cluster barrier the cluster's first CTA reads every chunk's
// (m_c, l_c, a_c) through distributed shared memory and combines them in
// chunk order: M = max m_c, L = sum l_c e^(m_c - M),
// out[d] = sum a_c[d] e^(m_c - M) / L  (chunks past the visible keys hold
// l_c = 0 and are skipped).  The result is that of one exact softmax over
// all visible keys, with every sum in a fixed order.
constexpr int kDh = 128;
constexpr int kSpThreads = 256;
constexpr int kSpMaxSplit = 8;      // portable cluster size
constexpr int kSpKeysPerPass = kSpThreads / 16;
constexpr int kSpVPre = 8;          // value rows per thread requested with the keys
constexpr int kRowsMinWarps = 1024;

struct SplitPlan {
  int split, chunk;
};

// Chunks of at least 64 keys (a multiple of 16), at most kSpMaxSplit of them.
inline SplitPlan split_plan(int max_seq) {
  int split = std::min(kSpMaxSplit, std::max(1, (max_seq + 63) / 64));
  int chunk = ((max_seq + split - 1) / split + 15) / 16 * 16;
  return SplitPlan{split, chunk};
}

__device__ __forceinline__ float sp_block_reduce(float v, float* red, bool is_max) {
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
  for (int w = 1; w < kSpThreads / 32; ++w) r = is_max ? fmaxf(r, red[w]) : r + red[w];
  return r;
}

template <typename T>
__global__ void __launch_bounds__(kSpThreads) attention_split_kernel(const T* __restrict__ q,
                                                                     const T* __restrict__ kc,
                                                                     const T* __restrict__ vc,
                                                                     const int* __restrict__ pos_ptr, int width,
                                                                     int max_seq, int chunk, T* __restrict__ out) {
  extern __shared__ float sp_smem[];
  float* part = sp_smem;                         // 16 groups x kDh partial sums
  float* acc = part + 16 * kDh;                  // kDh: this chunk's a_c
  float* ml = acc + kDh;                         // m_c, l_c
  float* red = ml + 2;                           // kSpThreads / 32 partials
  float* sc = red + kSpThreads / 32;             // chunk scores
  cg::cluster_group cluster = cg::this_cluster();
  pdl_wait();
  pdl_launch_dependents();
  const int c = (int)cluster.block_rank();
  const int split = (int)cluster.num_blocks();
  const int h = blockIdx.y, t = blockIdx.z;
  const int tid = threadIdx.x;
  const int n = min(*pos_ptr + t + 1, max_seq);
  const int j0 = c * chunk, j1 = min(j0 + chunk, n);
  const int64_t col = (int64_t)h * kDh;
  const float scale = rsqrtf((float)kDh);
  float m_c = -INFINITY, l_c = 0.f;
  if (j0 < j1) {
    const int sl = tid & 15, kq = tid >> 4;
    // the first kSpVPre value rows this thread sums in phase 3 (keys
    // kq, kq + 16, ... of the chunk), requested now so that they arrive
    // while the scores and the softmax are computed
    uint4 vpre[kSpVPre];
#pragma unroll
    for (int r = 0; r < kSpVPre; ++r) {
      const int j = j0 + kq + r * 16;
      vpre[r] = j < j1 ? *reinterpret_cast<const uint4*>(vc + (int64_t)j * width + col + sl * 8)
                       : make_uint4(0u, 0u, 0u, 0u);
    }
    // phase 1: lane group of 16 per key, 8 dims per thread
    float qv[8];
    {
      const uint4 u = *reinterpret_cast<const uint4*>(q + (int64_t)t * width + col + sl * 8);
      const T* e = reinterpret_cast<const T*>(&u);
#pragma unroll
      for (int i = 0; i < 8; ++i) qv[i] = to_f<T>(e[i]);
    }
    float mx = -INFINITY;
    for (int jb = j0; jb < j1; jb += 4 * kSpKeysPerPass) {
      uint4 ku[4];
#pragma unroll
      for (int r = 0; r < 4; ++r) {
        const int j = jb + r * kSpKeysPerPass + kq;
        ku[r] = j < j1 ? *reinterpret_cast<const uint4*>(kc + (int64_t)j * width + col + sl * 8)
                       : make_uint4(0u, 0u, 0u, 0u);
      }
#pragma unroll
      for (int r = 0; r < 4; ++r) {
        const int j = jb + r * kSpKeysPerPass + kq;
        const T* e = reinterpret_cast<const T*>(&ku[r]);
        float sdot = 0.f;
#pragma unroll
        for (int i = 0; i < 8; ++i) sdot = fmaf(qv[i], to_f<T>(e[i]), sdot);
#pragma unroll
        for (int off = 8; off > 0; off >>= 1) sdot += __shfl_xor_sync(0xffffffffu, sdot, off);
        sdot *= scale;
        if (j < j1) {
          if (sl == 0) sc[j - j0] = sdot;
          mx = fmaxf(mx, sdot);
        }
      }
    }
    // phase 2
    m_c = sp_block_reduce(mx, red, true);
    float l = 0.f;
    for (int j = tid; j < j1 - j0; j += kSpThreads) {
      const float pj = expf(sc[j] - m_c);
      sc[j] = pj;
      l += pj;
    }
    l_c = sp_block_reduce(l, red, false);  // the barriers inside also publish sc[]
    // phase 3: key group g = tid / 16, dims 8 * (tid % 16) .. + 7
    const int g = tid >> 4;
    float a[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) a[i] = 0.f;
    const T* vcol = vc + col + sl * 8;
#pragma unroll
    for (int r = 0; r < kSpVPre; ++r) {
      const int j = j0 + g + r * 16;
      if (j < j1) {
        const float pj = sc[j - j0];
        const T* e = reinterpret_cast<const T*>(&vpre[r]);
#pragma unroll
        for (int i = 0; i < 8; ++i) a[i] = fmaf(pj, to_f<T>(e[i]), a[i]);
      }
    }
    for (int jb = j0 + g + kSpVPre * 16; jb < j1; jb += 4 * 16) {
      uint4 vu[4];
#pragma unroll
      for (int r = 0; r < 4; ++r) {
        const int j = jb + r * 16;
        vu[r] = j < j1 ? *reinterpret_cast<const uint4*>(vcol + (int64_t)j * width) : make_uint4(0u, 0u, 0u, 0u);
      }
#pragma unroll
      for (int r = 0; r < 4; ++r) {
        const int j = jb + r * 16;
        if (j < j1) {
          const float pj = sc[j - j0];
          const T* e = reinterpret_cast<const T*>(&vu[r]);
#pragma unroll
          for (int i = 0; i < 8; ++i) a[i] = fmaf(pj, to_f<T>(e[i]), a[i]);
        }
      }
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) part[g * kDh + sl * 8 + i] = a[i];
    __syncthreads();
    if (tid < kDh) {
      float sum = 0.f;
      for (int gg = 0; gg < 16; ++gg) sum += part[gg * kDh + tid];
      acc[tid] = sum;
    }
  } else if (tid < kDh) {
    acc[tid] = 0.f;
  }
  if (tid == 0) {
    ml[0] = m_c;
    ml[1] = l_c;
  }
  cluster.sync();  // every chunk's (m_c, l_c, a_c) is visible to the cluster
  if (c == 0 && tid < kDh) {
    float M = -INFINITY;
    for (int r = 0; r < split; ++r) {
      const float* rml = cluster.map_shared_rank(ml, r);
      if (rml[1] > 0.f) M = fmaxf(M, rml[0]);
    }
    float L = 0.f, o = 0.f;
    for (int r = 0; r < split; ++r) {
      const float* rml = cluster.map_shared_rank(ml, r);
      if (rml[1] > 0.f) {
        const float w = expf(rml[0] - M);
        L += rml[1] * w;
        o += cluster.map_shared_rank(acc, r)[tid] * w;
      }
    }
    out[(int64_t)t * width + col + tid] = from_f<T>(o / L);
  }
  cluster.sync();  // the first CTA has read every chunk before any CTA exits
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

size_t attention_split_smem_bytes(int chunk) {
  return sizeof(float) * (16 * kDh + kDh + 2 + kSpThreads / 32 + (size_t)chunk);
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
    // decode: the visible keys split over a cluster of CTAs per (query, head)
    const SplitPlan sp = split_plan(max_seq);
    const size_t smem = attention_split_smem_bytes(sp.chunk);
    if (smem > 48 * 1024) {
      cudaError_t e = cudaFuncSetAttribute(attention_split_kernel<T>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           (int)smem);
      if (e != cudaSuccess) return done(e, "attention shared memory");
    }
    cudaLaunchConfig_t cfg;
    std::memset(&cfg, 0, sizeof(cfg));
    cfg.gridDim = dim3(sp.split, heads, tokens);
    cfg.blockDim = dim3(kSpThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = sp.split;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    return done(cudaLaunchKernelEx(&cfg, attention_split_kernel<T>, static_cast<const T*>(q),
                                   static_cast<const T*>(kc), static_cast<const T*>(vc), pos_ptr, width, max_seq,
                                   sp.chunk, static_cast<T*>(out)),
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
