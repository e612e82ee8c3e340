// tcgen05 convolution for inputs with few channels (C % 8 != 0: the RGB
// stems), where neither TMA nor 16-byte cp.async can fetch the im2col rows:
//
//   y[m, n] = epi( sum_k A[m, k] * W[n, k] ),  K = kh * kw * C <= 64 * kSmMaxKB
//
// One CTA of 128 threads is persistent over 128-row output tiles of one
// 64-column slice of N.  The weights of that slice are built once in shared
// memory, zero-padded to whole 64-wide k-blocks, in the 128-byte-swizzled
// K-major layout the MMA reads.  For every tile, thread t gathers im2col row
// t element by element (zero for padding and for k >= K) into one of two A
// buffers; one elected thread issues the MMAs into one of two TMEM
// accumulators and commits them to that buffer's mbarrier; then all threads
// run the epilogue of the PREVIOUS tile, which overlaps the tensor-core work
// of the current one.  Waits are bounded; a timeout is recorded in the error
// word and every CTA leaves the loop together.
#include <algorithm>
#include <cstring>
#include <type_traits>

#include "device.cuh"
#include "internal.h"
#include "kernels.h"

namespace swapnet {


namespace {

constexpr int kSmBM = 128;
constexpr int kSmBN = 64;
constexpr int kSmMaxKB = 3;
constexpr int kSmThreads = 128;
constexpr int kSmATile = kSmBM * 128;   // one k-block of A: 128 rows x 128 bytes
constexpr int kSmBTile = kSmBN * 128;   // one k-block of B: 64 rows x 128 bytes
constexpr int kInvalidTap = 0x4000;     // a row offset no image reaches

struct SmallArgs {
  const void* x;
  const void* w;
  int M, N, K, H, Wd, C, Ho, Wo, kh, kw, stride, pad;
  Epi e;
  void* y;
  int64_t ldy;
  int* err;
  int nkb, tiles;
};

__host__ __device__ constexpr int small_smem_bytes(int nkb) {
  return nkb * kSmBTile + 2 * nkb * kSmATile + kSmBN * 4 + 64 + nkb * 64 * 8 + 1024;
}

__device__ __forceinline__ void st_shared_v4(uint32_t addr, const uint4& v) {
  asm volatile("st.shared.v4.u32 [%0], {%1,%2,%3,%4};" ::"r"(addr), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
               : "memory");
}

template <typename T>
__device__ __forceinline__ uint32_t bits2(T lo, T hi) {
  uint16_t a, b;
  std::memcpy(&a, &lo, 2);
  std::memcpy(&b, &hi, 2);
  return (uint32_t)a | ((uint32_t)b << 16);
}

// Epilogue of one finished tile: thread t owns row t (TMEM lane t).  With no
// residual and 32 or 64 columns left in the slice, each warp passes its 32
// rows through `stage` (4 KB per warp of the idle A buffer, 16-byte chunks
// swizzled by row) so that every store instruction writes whole rows (four
// of 128 bytes, or eight of 64) instead of one 16-byte piece of 32 rows.
template <typename T>
__device__ __forceinline__ void small_epilogue(const SmallArgs& p, uint32_t tmem_buf, const float* sbias, int tile,
                                               int n0, uint32_t stage) {
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int m = tile * kSmBM + tid;
  const T* res = static_cast<const T*>(p.e.res);
  const int ncols = p.N - n0 >= kSmBN ? kSmBN : (p.N - n0 == 32 ? 32 : 0);
  if (!res && ncols && ((p.ldy | n0) % 8 == 0)) {
    const uint32_t wst = stage + (uint32_t)(warp * 32 * 128);
#pragma unroll 1
    for (int c0 = 0; c0 < ncols; c0 += 32) {
      uint32_t r[32];
      tmem_ld_32x32b_x32(tmem_buf + ((uint32_t)(warp * 32) << 16) + (uint32_t)c0, r);
      tmem_ld_wait();
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        uint32_t o[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int j = 8 * q + 2 * i;
          const T lo = from_f<T>(epilogue(__uint_as_float(r[j]), sbias[c0 + j], 0.f, 0, p.e.act, p.e.res_post));
          const T hi = from_f<T>(epilogue(__uint_as_float(r[j + 1]), sbias[c0 + j + 1], 0.f, 0, p.e.act, p.e.res_post));
          o[i] = bits2<T>(lo, hi);
        }
        const uint32_t chunk = (uint32_t)(c0 / 8 + q);
        st_shared_v4(wst + (uint32_t)lane * 128 + ((chunk ^ (uint32_t)(lane & 7)) << 4),
                     make_uint4(o[0], o[1], o[2], o[3]));
      }
    }
    __syncwarp();
    const int m_base = tile * kSmBM + warp * 32;
    const int cpr_log2 = ncols == kSmBN ? 3 : 2;  // 16-byte chunks per row: 8 or 4
#pragma unroll 1
    for (int i = 0; i < (1 << cpr_log2); ++i) {
      const int row = (i << (5 - cpr_log2)) + (lane >> cpr_log2), chunk = lane & ((1 << cpr_log2) - 1);
      uint4 v;
      asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];"
                   : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                   : "r"(wst + (uint32_t)row * 128 + (((uint32_t)chunk ^ (uint32_t)(row & 7)) << 4)));
      if (m_base + row < p.M)
        *reinterpret_cast<uint4*>(static_cast<T*>(p.y) + (int64_t)(m_base + row) * p.ldy + n0 + chunk * 8) = v;
    }
    __syncwarp();
    return;
  }
#pragma unroll 1
  for (int c0 = 0; c0 < kSmBN; c0 += 32) {
    uint32_t r[32];
    tmem_ld_32x32b_x32(tmem_buf + ((uint32_t)(warp * 32) << 16) + (uint32_t)c0, r);
    tmem_ld_wait();
    if (m >= p.M) continue;
    T* yrow = static_cast<T*>(p.y) + (int64_t)m * p.ldy;
    const T* rrow = res ? res + (int64_t)m * p.e.ldr : nullptr;
    const bool vec = n0 + c0 + 32 <= p.N && ((p.ldy | n0) % 8 == 0) && (!rrow || (p.e.ldr % 8 == 0));
    if (vec) {
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        uint32_t o[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int j = 8 * q + 2 * i, n = n0 + c0 + j;
          const float r0 = rrow ? to_f<T>(rrow[n]) : 0.f, r1 = rrow ? to_f<T>(rrow[n + 1]) : 0.f;
          const T lo = from_f<T>(epilogue(__uint_as_float(r[j]), sbias[c0 + j], r0, rrow != nullptr, p.e.act,
                                          p.e.res_post));
          const T hi = from_f<T>(epilogue(__uint_as_float(r[j + 1]), sbias[c0 + j + 1], r1, rrow != nullptr,
                                          p.e.act, p.e.res_post));
          o[i] = bits2<T>(lo, hi);
        }
        *reinterpret_cast<uint4*>(yrow + n0 + c0 + 8 * q) = make_uint4(o[0], o[1], o[2], o[3]);
      }
      continue;
    }
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      const int n = n0 + c0 + j;
      if (n < p.N) {
        const float rv = rrow ? to_f<T>(rrow[n]) : 0.f;
        yrow[n] = from_f<T>(epilogue(__uint_as_float(r[j]), sbias[c0 + j], rv, rrow != nullptr, p.e.act,
                                     p.e.res_post));
      }
    }
  }
}

template <typename T>
__global__ void __launch_bounds__(kSmThreads, 4) tc_conv_small_kernel(const SmallArgs p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int nkb = p.nkb;
  uint8_t* sB = smem;
  uint8_t* sA = smem + nkb * kSmBTile;
  float* sbias = reinterpret_cast<float*>(sA + 2 * nkb * kSmATile);
  uint64_t* bars = reinterpret_cast<uint64_t*>(sbias + kSmBN);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  // per k: element offset inside the receptive window and the tap (dy, dx);
  // k >= K gets dy = kInvalidTap, which fails the bounds test
  int2* tab = reinterpret_cast<int2*>(reinterpret_cast<uint8_t*>(bars) + 64);
  const int tid = threadIdx.x, warp = tid >> 5;
  const int n0 = blockIdx.y * kSmBN;
  const uint32_t bar0 = smem_u32(bars);

  if (tid == 0) {
    mbar_init(bar0, 1);
    mbar_init(bar0 + 8, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0) {
    tmem_alloc(smem_u32(tmem_slot), 2 * kSmBN);
    tmem_relinquish();
  }
  // weights of this N slice -> swizzled B tiles (zero-padded), bias -> smem
  const T* W = static_cast<const T*>(p.w);
  const T zero = from_f<T>(0.f);
  for (int q = tid; q < nkb * kSmBN * 8; q += kSmThreads) {
    const int kb = q / (kSmBN * 8), r = q % (kSmBN * 8);
    const int n = r >> 3, j = r & 7;
    const bool nv = n0 + n < p.N;
    uint32_t v[4];
#pragma unroll
    for (int h = 0; h < 4; ++h) {
      const int k = kb * 64 + j * 8 + 2 * h;
      const T lo = (nv && k < p.K) ? W[(int64_t)(n0 + n) * p.K + k] : zero;
      const T hi = (nv && k + 1 < p.K) ? W[(int64_t)(n0 + n) * p.K + k + 1] : zero;
      v[h] = bits2<T>(lo, hi);
    }
    st_shared_v4(smem_u32(sB + kb * kSmBTile + (n >> 3) * 1024 + (n & 7) * 128 + ((j ^ (n & 7)) << 4)),
                 make_uint4(v[0], v[1], v[2], v[3]));
  }
  if (tid < kSmBN) {
    const T* bias = static_cast<const T*>(p.e.bias);
    sbias[tid] = (bias && n0 + tid < p.N) ? to_f<T>(bias[n0 + tid]) : 0.f;
  }
  for (int k = tid; k < nkb * 64; k += kSmThreads) {
    if (k < p.K) {
      const int tap = k / p.C, c = k - tap * p.C;
      const int dy = tap / p.kw, dx = tap - dy * p.kw;
      tab[k] = make_int2((dy * p.Wd + dx) * p.C + c, (dy << 16) | dx);
    } else {
      tab[k] = make_int2(0, kInvalidTap << 16);
    }
  }
  fence_proxy_async_smem();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_wait();  // the input is the previous kernel's output
  pdl_launch_dependents();

  constexpr uint32_t idesc = idesc_f16(std::is_same<T, __nv_bfloat16>::value ? 1 : 0, kSmBM, kSmBN);
  const T* X = static_cast<const T*>(p.x);
  const int hw = p.Ho * p.Wo;
  const uint32_t row_off = (uint32_t)((tid >> 3) * 1024 + (tid & 7) * 128);
  const uint32_t sw = (uint32_t)(tid & 7);
  int it = 0;
  int pending = -1;  // buffer whose MMAs were committed and not yet waited for
  for (int tile = blockIdx.x; tile < p.tiles; tile += gridDim.x, ++it) {
    if (__syncthreads_or(*abort_flag)) break;
    const int buf = it & 1;
    // ---- gather row tid of this tile (A buffer `buf` is free: its previous
    // MMAs were waited for in the epilogue of the last iteration)
    const int m = tile * kSmBM + tid;
    const bool mv = m < p.M;
    int img = 0, oy = 0, ox = 0;
    if (mv) {
      img = m / hw;
      const int rem = m - img * hw;
      oy = rem / p.Wo;
      ox = rem - oy * p.Wo;
    }
    const int iy0 = oy * p.stride - p.pad, ix0 = ox * p.stride - p.pad;
    // window origin (may lie outside the image; only valid taps are read)
    const T* xw = X + (((int64_t)img * p.H + iy0) * p.Wd + ix0) * p.C;
    const uint32_t abase = smem_u32(sA + buf * nkb * kSmATile) + row_off;
    for (int kb = 0; kb < nkb; ++kb) {
      uint32_t e2[32];  // packed pairs: up to 64 independent loads in flight
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        // 16 k per chunk; a chunk wholly past K (e.g. k 32..63 of a 27-deep
        // RGB 3x3 stem) is zero without touching the table or the input
        if (kb * 64 + q * 16 < p.K) {
#pragma unroll
          for (int h = q * 16; h < q * 16 + 16; h += 2) {
            T e[2];
#pragma unroll
            for (int u = 0; u < 2; ++u) {
              const int2 t = tab[kb * 64 + h + u];
              const int iy = iy0 + (t.y >> 16), ix = ix0 + (t.y & 0xffff);
              const bool valid = mv && (unsigned)iy < (unsigned)p.H && (unsigned)ix < (unsigned)p.Wd;
              e[u] = valid ? __ldg(xw + t.x) : zero;
            }
            e2[h >> 1] = bits2<T>(e[0], e[1]);
          }
        } else {
#pragma unroll
          for (int h = q * 16; h < q * 16 + 16; h += 2) e2[h >> 1] = 0u;
        }
      }
#pragma unroll
      for (int j = 0; j < 8; ++j)
        st_shared_v4(abase + kb * kSmATile + (((uint32_t)j ^ sw) << 4),
                     make_uint4(e2[4 * j], e2[4 * j + 1], e2[4 * j + 2], e2[4 * j + 3]));
    }
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    if (tid == 0) {
      tc_fence_after();
      const uint32_t d = tmem + (uint32_t)(buf * kSmBN);
      for (int kb = 0; kb < nkb; ++kb) {
        const uint64_t ad = smem_desc_sw128(smem_u32(sA + (buf * nkb + kb) * kSmATile));
        const uint64_t bd = smem_desc_sw128(smem_u32(sB + kb * kSmBTile));
#pragma unroll
        for (int k = 0; k < 4; ++k) tc_mma_f16(d, ad + 2ull * k, bd + 2ull * k, idesc, (kb | k) != 0);
      }
      tc_commit(bar0 + 8u * buf);
    }
    // ---- epilogue of the previous tile (its MMAs ran while we gathered)
    if (it > 0) {
      const int pb = buf ^ 1;
      const bool got = mbar_wait_bounded(bar0 + 8u * pb, ((it - 1) >> 1) & 1, abort_flag, p.err);
      if (__all_sync(0xffffffffu, got)) {  // tcgen05.ld is warp-collective
        tc_fence_after();
        small_epilogue<T>(p, tmem + (uint32_t)(pb * kSmBN), sbias, tile - (int)gridDim.x, n0,
                          smem_u32(sA + pb * nkb * kSmATile));
      }
      tc_fence_before();
    }
    pending = buf;
  }
  // ---- last tile (or drain after an abort)
  if (pending >= 0) {
    volatile int no_abort = 0;
    const int last = it - 1;
    const bool ok = !*abort_flag;
    const bool got = mbar_wait_bounded(bar0 + 8u * pending, (last >> 1) & 1, ok ? abort_flag : &no_abort, p.err);
    if (__all_sync(0xffffffffu, got && ok)) {
      tc_fence_after();
      small_epilogue<T>(p, tmem + (uint32_t)(pending * kSmBN), sbias, blockIdx.x + last * (int)gridDim.x, n0,
                        smem_u32(sA + pending * nkb * kSmATile));
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, 2 * kSmBN);
  }
}

// CTAs per SM for a given k-block count, per element type and device (0
// until known); computed outside stream capture (tc_small_prepare), where
// the occupancy query is allowed, together with the kernel's attributes on
// that device.  An unknown device index shares the last slot.
template <typename T>
std::atomic<int>& small_occ(int nkb) {
  static std::atomic<int> occ[65][kSmMaxKB + 1];
  const int dev = device_index();
  return occ[dev >= 0 ? dev : 64][nkb];
}

template <typename T>
int small_prepare_t(int nkb) {
  auto kern = tc_conv_small_kernel<T>;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, small_smem_bytes(kSmMaxKB)) !=
      cudaSuccess)
    SN_FAIL(SWAPNET_ERR_CUDA, "cudaFuncSetAttribute failed");
  // several CTAs share an SM: ask for the whole carveout as shared memory
  // (without a preference the occupancy query assumes room for one CTA)
  if (cudaFuncSetAttribute(kern, cudaFuncAttributePreferredSharedMemoryCarveout, cudaSharedmemCarveoutMaxShared) !=
      cudaSuccess)
    cudaGetLastError();
  // CTAs per SM from the kernel's registers and shared memory
  cudaFuncAttributes fa;
  int dev = 0, regs_sm = 0, smem_sm = 0, reserved = 0, blocks_sm = 0;
  if (cudaFuncGetAttributes(&fa, kern) != cudaSuccess || cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&regs_sm, cudaDevAttrMaxRegistersPerMultiprocessor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&smem_sm, cudaDevAttrMaxSharedMemoryPerMultiprocessor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&reserved, cudaDevAttrReservedSharedMemoryPerBlock, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&blocks_sm, cudaDevAttrMaxBlocksPerMultiprocessor, dev) != cudaSuccess)
    SN_FAIL(SWAPNET_ERR_CUDA, "small-channel conv: kernel attributes unavailable");
  const int warp_regs = (fa.numRegs * 32 + 255) / 256 * 256;
  const int by_regs = regs_sm / std::max(1, warp_regs * (kSmThreads / 32));
  const int by_smem = smem_sm / std::max(1, small_smem_bytes(nkb) + (int)fa.sharedSizeBytes + reserved);
  const int n = std::min(std::min(by_regs, by_smem), blocks_sm);
  small_occ<T>(nkb).store(std::max(1, std::min(n, 512 / (2 * kSmBN))));  // TMEM: 128 columns per CTA
  return SWAPNET_OK;
}

template <typename T>
int launch_small(const TcSmallConv& g, int* err, cudaStream_t s) {
  auto kern = tc_conv_small_kernel<T>;
  const int nkb = (g.K + 63) / 64;
  const int smem = small_smem_bytes(nkb);
  if (small_occ<T>(nkb).load() == 0) {
    const int rc = small_prepare_t<T>(nkb);
    if (rc) return rc;
  }
  const int occ = small_occ<T>(nkb).load();
  SmallArgs a;
  std::memset(&a, 0, sizeof(a));
  a.x = g.x; a.w = g.W;
  a.M = g.M; a.N = g.N; a.K = g.K;
  a.H = g.H; a.Wd = g.Wd; a.C = g.C; a.Ho = g.Ho; a.Wo = g.Wo;
  a.kh = g.kh; a.kw = g.kw; a.stride = g.stride; a.pad = g.pad;
  a.e = g.e; a.y = g.y; a.ldy = g.ldy; a.err = err;
  a.nkb = nkb;
  a.tiles = (g.M + kSmBM - 1) / kSmBM;
  const int sms = g.num_sms > 0 ? g.num_sms : 148;
  const dim3 grid(std::min(a.tiles, sms * occ), (g.N + kSmBN - 1) / kSmBN);
  cudaLaunchConfig_t cfg;
  std::memset(&cfg, 0, sizeof(cfg));
  cfg.gridDim = grid;
  cfg.blockDim = dim3(kSmThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const cudaError_t le = cudaLaunchKernelEx(&cfg, kern, a);
  if (le != cudaSuccess) SN_FAIL(SWAPNET_ERR_CUDA, std::string("small-channel conv launch: ") + cudaGetErrorString(le));
  return SWAPNET_OK;
}

}  // namespace

bool tc_small_supported(int dtype, int K) {
  return (dtype == SWAPNET_F16 || dtype == SWAPNET_BF16) && K >= 1 && K <= 64 * kSmMaxKB;
}

int tc_small_prepare(int dtype, int K) {
  if (!tc_small_supported(dtype, K)) SN_FAIL(SWAPNET_ERR_UNSUPPORTED, "small-channel conv: K out of range");
  const int nkb = (K + 63) / 64;
  return dtype == SWAPNET_BF16 ? small_prepare_t<__nv_bfloat16>(nkb) : small_prepare_t<__half>(nkb);
}

int launch_tc_conv_small(const TcSmallConv& g, int* err, cudaStream_t s) {
  if (!tc_small_supported(g.dtype, g.K)) SN_FAIL(SWAPNET_ERR_UNSUPPORTED, "small-channel conv: K out of range");
  if (g.M < 1 || g.N < 1) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "small-channel conv: empty problem");
  if (g.dtype == SWAPNET_BF16) return launch_small<__nv_bfloat16>(g, err, s);
  return launch_small<__half>(g, err, s);
}

}  // namespace swapnet
