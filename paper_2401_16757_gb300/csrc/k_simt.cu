// SIMT layer kernels: skinny linear (M <= 16, HBM-bound GEMV family),
// direct convolution for channel counts the tensor-core path cannot tile,
// pooling, upsampling and channel concatenation.  NHWC everywhere.
#include <algorithm>
#include <atomic>
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
//
// One launch may serve several layers that read the same input (SkJob
// segments, e.g. the q, k, v projections): the warps are dealt to the
// segments' features in order.  In pair mode (a gate and the layer whose
// epilogue takes the gate's output as its residual, e.g. SwiGLU) one warp
// computes feature o of both: it stores the gate's rounded output and uses
// that same rounded value as the second layer's residual.  Every feature is
// computed by the same per-row routine as in a one-layer launch, so the
// results are bit-identical to launching the layers one by one.
constexpr int kSkWarps = 8;
constexpr int kSkBatch = 8;

template <typename T, int MT>
__device__ __forceinline__ void sk_row(const T* __restrict__ x, int M, int K, const T* __restrict__ wrow, int lane,
                                       uint4 (&wv)[kSkBatch], bool preloaded, float (&acc)[MT]) {
  constexpr int V = Vec16<T>::N;
  const int kchunks = K / V;  // K % V == 0 (checked on the host)
  auto load_batch = [&](int c0) {
#pragma unroll
    for (int u = 0; u < kSkBatch; ++u) {
      const int ch = c0 + u * 32;
      wv[u] = ch < kchunks ? ld_stream16(wrow + (int64_t)ch * V) : make_uint4(0u, 0u, 0u, 0u);
    }
  };
#pragma unroll
  for (int m = 0; m < MT; ++m) acc[m] = 0.f;
  for (int c0 = lane; c0 < kchunks; c0 += 32 * kSkBatch) {
    if (c0 != lane || !preloaded) load_batch(c0);
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
#pragma unroll
  for (int m = 0; m < MT; ++m) {
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) acc[m] += __shfl_xor_sync(0xffffffffu, acc[m], off);
  }
}

template <typename T, int MT>
__global__ void __launch_bounds__(kSkWarps * 32) linear_skinny_kernel(const SkJob j) {
  constexpr int V = Vec16<T>::N;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  int o = blockIdx.x * kSkWarps + warp;
  // this warp's segment (pair mode: both segments, feature o)
  int si = 0;
  if (!j.pair)
    for (int i = 0; i + 1 < j.nseg && o >= j.seg[i].N; ++i) {
      o -= j.seg[i].N;
      si = i + 1;
    }
  SkSeg S = j.seg[0];
#pragma unroll
  for (int i = 1; i < kSkMaxSeg; ++i)
    if (i == si) S = j.seg[i];
  const bool active = o < S.N;
  const T* x = static_cast<const T*>(j.x);
  uint4 wv[kSkBatch];
  if (active) {
    const T* wrow = static_cast<const T*>(S.W) + (int64_t)o * j.K;
#pragma unroll
    for (int u = 0; u < kSkBatch; ++u) {
      const int ch = lane + u * 32;
      wv[u] = ch < j.K / V ? ld_stream16(wrow + (int64_t)ch * V) : make_uint4(0u, 0u, 0u, 0u);
    }
  }
  pdl_wait();
  pdl_launch_dependents();
  if (!active) return;
  float acc[MT];
  float gate[MT];
  const int passes = j.pair ? 2 : 1;
  for (int p = 0; p < passes; ++p) {
    if (p == 1) S = j.seg[1];
    sk_row<T, MT>(x, j.M, j.K, static_cast<const T*>(S.W) + (int64_t)o * j.K, lane, wv, p == 0, acc);
    const float b = S.e.bias ? to_f<T>(static_cast<const T*>(S.e.bias)[o]) : 0.f;
#pragma unroll
    for (int m = 0; m < MT; ++m) {
      if (m < j.M) {
        float r = 0.f;
        bool has_r = S.e.res != nullptr;
        if (p == 1) {
          r = gate[m];
          has_r = true;
        } else if (has_r) {
          r = to_f<T>(static_cast<const T*>(S.e.res)[(int64_t)m * S.e.ldr + o]);
        }
        const T out = from_f<T>(epilogue(acc[m], b, r, has_r, S.e.act, S.e.res_post));
        gate[m] = to_f<T>(out);  // the stored value, as the paired layer would read it
        if (lane == m) static_cast<T*>(S.y)[(int64_t)m * S.ldy + o] = out;
      }
    }
  }
}

// ------------------------------------------------------------ streamed skinny linear
// The same per-feature arithmetic as linear_skinny_kernel (lane l takes the
// 16-byte chunks l, l + 32, ... of the weight row in order, one fp32 sum per
// row of x, the same butterfly and epilogue), so its outputs are
// bit-identical; only the way the weight rows reach the lanes differs.  For
// weights in device memory each warp streams its rows into its own ring of
// D shared-memory slots with bulk copies (cp.async.bulk, completion counted
// on one mbarrier per slot), issued by lane 0 up to D rows ahead of the
// row being summed, so each SM keeps D x row bytes per warp in flight
// (about 100-200 KB) with a handful of registers.  x (M rows of K) is read
// once per CTA into shared memory.  The first D rows of every warp are
// requested before the programmatic wait (weights never depend on the
// previous kernel), so the weight stream starts while that kernel drains.
// One CTA per SM (grid = number of SMs, or fewer when there are fewer
// features); warp g of the grid takes features g, g + G, ... (G = warps in
// the grid); in pair mode a feature's two rows (gate, then its paired
// layer) take two consecutive slots.  Every slot wait is bounded: on
// timeout the warp records the error, stops, and waits (bounded) for the
// copies it still has in flight before the CTA exits.
constexpr int kStXMax = 64 * 1024;        // x staged in shared memory: at most this many bytes
constexpr int kStSmem = 227 * 1024;       // dynamic shared memory of the streamed kernel's CTA
constexpr int kStMaxWarps = 8;

struct StLayout {
  int warps, depth, slot_bytes, x_bytes, smem;
};

inline StLayout st_layout(int M, int K, int es, bool pair) {
  StLayout L{0, 0, 0, 0, 0};
  const int row = K * es;
  L.x_bytes = (M * row + 127) / 128 * 128;
  if (M * row > kStXMax) return L;
  L.slot_bytes = (row + 127) / 128 * 128;
  L.depth = row <= 8192 ? 4 : (row <= 16384 && !pair ? 3 : 2);
  const int fixed = L.x_bytes + 256;  // + abort flag, alignment slack
  const int per_warp = L.depth * (L.slot_bytes + 8);
  L.warps = std::min(kStMaxWarps, (kStSmem - fixed) / per_warp);
  L.smem = fixed + L.warps * per_warp;
  return L;
}

__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
               ::"r"(dst), "l"(src), "r"(bytes), "r"(bar) : "memory");
}

template <typename T, int MT>
__global__ void __launch_bounds__(kStMaxWarps * 32, 1) linear_stream_kernel(const SkJob j, int depth, int slot_bytes,
                                                                             int x_bytes) {
  constexpr int V = Vec16<T>::N;
  extern __shared__ __align__(128) uint8_t st_smem[];
  const int warps = blockDim.x >> 5;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  T* xs = reinterpret_cast<T*>(st_smem);
  uint8_t* ring = st_smem + x_bytes + (size_t)warp * depth * slot_bytes;
  uint64_t* bars = reinterpret_cast<uint64_t*>(st_smem + x_bytes + (size_t)warps * depth * slot_bytes) + warp * depth;
  volatile int* abort_flag =
      reinterpret_cast<volatile int*>(st_smem + x_bytes + (size_t)warps * depth * (slot_bytes + 8));
  const int row_bytes = j.K * (int)sizeof(T);
  const int kchunks = j.K / V;
  const int rows_per_item = j.pair ? 2 : 1;
  int features = j.seg[0].N;
  if (!j.pair)
    for (int i = 1; i < j.nseg; ++i) features += j.seg[i].N;
  const int gw = blockIdx.x * warps + warp, G = gridDim.x * warps;
  const int my_items = gw < features ? (features - 1 - gw) / G + 1 : 0;
  const int my_rows = my_items * rows_per_item;
  // weight row q of this warp's stream
  auto row_ptr = [&](int q) -> const T* {
    int o = gw + (q / rows_per_item) * G;
    int si = j.pair ? (q % 2) : 0;
    if (!j.pair)
      for (int i = 0; i + 1 < j.nseg && o >= j.seg[i].N; ++i) {
        o -= j.seg[i].N;
        si = i + 1;
      }
    const T* W = static_cast<const T*>(j.seg[0].W);
#pragma unroll
    for (int i = 1; i < kSkMaxSeg; ++i)
      if (i == si) W = static_cast<const T*>(j.seg[i].W);
    return W + (int64_t)o * j.K;
  };
  auto issue = [&](int q) {
    const int slot = q % depth;
    const uint32_t bar = smem_u32(bars + slot);
    mbar_arrive_expect_tx(bar, (uint32_t)row_bytes);
    bulk_g2s(smem_u32(ring + (size_t)slot * slot_bytes), row_ptr(q), (uint32_t)row_bytes, bar);
  };
  if (lane == 0)
    for (int i = 0; i < depth; ++i) mbar_init(smem_u32(bars + i), 1);
  if (threadIdx.x == 0) *abort_flag = 0;
  fence_barrier_init();
  __syncthreads();
  int issued = 0;
  if (lane == 0)
    for (; issued < depth && issued < my_rows; ++issued) issue(issued);
  pdl_wait();
  pdl_launch_dependents();
  {  // x into shared memory, 16 bytes per access
    const uint4* src = static_cast<const uint4*>(j.x);
    uint4* dst = reinterpret_cast<uint4*>(xs);
    const int n16 = j.M * row_bytes / 16;
    for (int i = threadIdx.x; i < n16; i += blockDim.x) dst[i] = src[i];
  }
  __syncthreads();
  int q = 0;
  bool ok = true;
  for (int it = 0; it < my_items && ok; ++it) {
    const int o_global = gw + it * G;
    int o = o_global, si = 0;
    if (!j.pair)
      for (int i = 0; i + 1 < j.nseg && o >= j.seg[i].N; ++i) {
        o -= j.seg[i].N;
        si = i + 1;
      }
    float gate[MT];
    for (int p = 0; p < rows_per_item; ++p, ++q) {
      SkSeg S = j.seg[0];
#pragma unroll
      for (int i = 1; i < kSkMaxSeg; ++i)
        if (i == (j.pair ? p : si)) S = j.seg[i];
      const int slot = q % depth;
      if (!mbar_wait_bounded(smem_u32(bars + slot), (uint32_t)((q / depth) & 1), abort_flag, j.err)) {
        ok = false;
        break;
      }
      const uint4* wrow = reinterpret_cast<const uint4*>(ring + (size_t)slot * slot_bytes);
      float acc[MT];
#pragma unroll
      for (int m = 0; m < MT; ++m) acc[m] = 0.f;
      for (int ch = lane; ch < kchunks; ch += 32) {
        float wf[V];
        unpack16<T>(wrow[ch], wf);
#pragma unroll
        for (int m = 0; m < MT; ++m) {
          if (m < j.M) {
            float xv[V];
            unpack16<T>(*reinterpret_cast<const uint4*>(xs + (int64_t)m * j.K + (int64_t)ch * V), xv);
#pragma unroll
            for (int i = 0; i < V; ++i) acc[m] = fmaf(wf[i], xv[i], acc[m]);
          }
        }
      }
#pragma unroll
      for (int m = 0; m < MT; ++m) {
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) acc[m] += __shfl_xor_sync(0xffffffffu, acc[m], off);
      }
      // every lane has read the slot (its sums are complete): refill it
      __syncwarp();
      if (lane == 0 && issued < my_rows) {
        fence_proxy_async_smem();
        issue(issued);
        ++issued;
      }
      const float b = S.e.bias ? to_f<T>(static_cast<const T*>(S.e.bias)[o]) : 0.f;
#pragma unroll
      for (int m = 0; m < MT; ++m) {
        if (m < j.M) {
          float r = 0.f;
          bool has_r = S.e.res != nullptr;
          if (p == 1) {
            r = gate[m];
            has_r = true;
          } else if (has_r) {
            r = to_f<T>(static_cast<const T*>(S.e.res)[(int64_t)m * S.e.ldr + o]);
          }
          const T out = from_f<T>(epilogue(acc[m], b, r, has_r, S.e.act, S.e.res_post));
          gate[m] = to_f<T>(out);  // the stored value, as the paired layer reads it
          if (lane == m) static_cast<T*>(S.y)[(int64_t)m * S.ldy + o] = out;
        }
      }
    }
  }
  if (!ok && lane == 0) {
    // copies still in flight land in this warp's slots: wait for them
    // (bounded) before the CTA's shared memory goes away
    volatile int drain = 0;
    for (int r = q; r < issued; ++r)
      mbar_wait_bounded(smem_u32(bars + r % depth), (uint32_t)((r / depth) & 1), &drain, nullptr);
  }
}

template <typename T, int MT>
int stream_launch(const SkJob& j, const StLayout& L, int grid, cudaStream_t s) {
  static std::atomic<uint64_t> attr_done{0};  // per instantiation, one bit per device
  auto kern = linear_stream_kernel<T, MT>;
  if (attr_needed(attr_done)) {
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kStSmem) != cudaSuccess)
      SN_FAIL(SWAPNET_ERR_CUDA, "cudaFuncSetAttribute failed");
    attr_set(attr_done);
  }
  const cudaError_t e = launch_pdl(kern, dim3(grid), dim3(L.warps * 32), (size_t)L.smem, s, j, L.depth,
                                   L.slot_bytes, L.x_bytes);
  return e == cudaSuccess ? SWAPNET_OK : SWAPNET_ERR_CUDA;
}

template <typename T> int stream_dispatch(const SkJob& j, const StLayout& L, cudaStream_t s) {
  int features = j.seg[0].N;
  if (!j.pair)
    for (int i = 1; i < j.nseg; ++i) features += j.seg[i].N;
  const int grid = std::max(1, std::min(j.num_sms, (features + L.warps - 1) / L.warps));
  if (j.M <= 1) return stream_launch<T, 1>(j, L, grid, s);
  if (j.M <= 2) return stream_launch<T, 2>(j, L, grid, s);
  if (j.M <= 4) return stream_launch<T, 4>(j, L, grid, s);
  if (j.M <= 8) return stream_launch<T, 8>(j, L, grid, s);
  return stream_launch<T, 16>(j, L, grid, s);
}

// Rows of x from which the streamed kernel is used.  Measured on the GB300
// box: with 8 rows (the fp32 MLP, K = 1024) it took a layer from 11.9 to
// 6.3 us, x being read once per CTA instead of once per warp; with one row
// (the 7B decode projections) it was slower than the plain-load kernel
// (20.6 against 12.2 us per launch): one CTA of 4-8 warps per SM sums its
// rows one after another and cannot hide each row's shared-memory, reduction
// and epilogue latency the way 32 resident warps with loads in flight do.
constexpr int kStMinRows = 8;

template <typename T> int skinny_dispatch(const SkJob& j, cudaStream_t s) {
  if (j.device_weights && j.num_sms > 0 && j.M >= kStMinRows) {
    const StLayout L = st_layout(j.M, j.K, (int)sizeof(T), j.pair != 0);
    if (L.warps >= 1) return stream_dispatch<T>(j, L, s);
  }
  int rows = j.seg[0].N;
  if (!j.pair)
    for (int i = 1; i < j.nseg; ++i) rows += j.seg[i].N;
  const dim3 grid((rows + kSkWarps - 1) / kSkWarps), block(kSkWarps * 32);
  cudaError_t e;
  if (j.M <= 1) e = launch_pdl(linear_skinny_kernel<T, 1>, grid, block, 0, s, j);
  else if (j.M <= 2) e = launch_pdl(linear_skinny_kernel<T, 2>, grid, block, 0, s, j);
  else if (j.M <= 4) e = launch_pdl(linear_skinny_kernel<T, 4>, grid, block, 0, s, j);
  else if (j.M <= 8) e = launch_pdl(linear_skinny_kernel<T, 8>, grid, block, 0, s, j);
  else e = launch_pdl(linear_skinny_kernel<T, 16>, grid, block, 0, s, j);
  return e == cudaSuccess ? SWAPNET_OK : SWAPNET_ERR_CUDA;
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

int launch_linear_skinny_job(int dtype, const SkJob& j, cudaStream_t s) {
  const int es = dtype_size(dtype);
  if (j.M < 1 || j.M > 16 || j.K < 1 || j.nseg < 1 || j.nseg > kSkMaxSeg || (j.pair && j.nseg != 2))
    SN_FAIL(SWAPNET_ERR_UNSUPPORTED, "skinny linear: M must be in [1, 16], 1 to 3 layers");
  if ((j.K * es) % 16 || (uintptr_t)j.x % 16) SN_FAIL(SWAPNET_ERR_MISALIGNED, "skinny linear: rows must be 16-byte aligned");
  for (int i = 0; i < j.nseg; ++i) {
    if (j.seg[i].N < 1) SN_FAIL(SWAPNET_ERR_UNSUPPORTED, "skinny linear: no output features");
    if ((uintptr_t)j.seg[i].W % 16) SN_FAIL(SWAPNET_ERR_MISALIGNED, "skinny linear: rows must be 16-byte aligned");
  }
  if (j.pair && j.seg[0].N != j.seg[1].N) SN_FAIL(SWAPNET_ERR_UNSUPPORTED, "skinny linear: paired layers differ in width");
  SN_DISPATCH(dtype, T, return skinny_dispatch<T>(j, s));
  return SWAPNET_OK;
}

int launch_linear_skinny(int dtype, const void* x, int M, int K, const void* W, int N, const Epi& e, void* y,
                         int64_t ldy, cudaStream_t s, int device_weights, int num_sms, int* err) {
  SkJob j{};
  j.x = x;
  j.M = M;
  j.K = K;
  j.nseg = 1;
  j.seg[0] = SkSeg{W, e, N, y, ldy};
  j.device_weights = device_weights;
  j.num_sms = num_sms;
  j.err = err;
  return launch_linear_skinny_job(dtype, j, s);
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
