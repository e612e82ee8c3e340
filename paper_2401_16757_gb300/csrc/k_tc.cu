// tcgen05 tensor-core GEMM and implicit-GEMM convolution for sm_103a.
//
//   C[m, n] = sum_k A[m, k] * B[n, k],  fp16/bf16 operands, fp32 accumulate
//   in TMEM, fused epilogue (bias, residual, activation) on the way out.
//
// B is a weight matrix [N][K] (K contiguous) that lives in the arena slot of
// the block being executed; it is staged by TMA (128-byte swizzle).  A is
// either a row-major activation matrix (linear layers, 1x1 stride-1 convs),
// also staged by TMA, or the implicit im2col of an NHWC input for general
// convolutions, gathered by four warps with cp.async (zero fill for padding)
// into the same swizzled layout.  One CTA computes one 128 x BN tile:
//   warp 0      TMA producer (one elected lane)
//   warp 1      TMEM allocation and MMA issue (one elected lane)
//   warps 2..5  im2col gather (conv) and the epilogue (TMEM -> registers ->
//               global), warp w reading TMEM lanes 32*(w % 4) .. +31.
// Every wait is bounded; on timeout the kernel records kDevErrTimeout in
// the error word, drains what it started, frees TMEM and returns.
#include <cudaTypedefs.h>

#include <algorithm>
#include <cstring>
#include <mutex>
#include <type_traits>

#include "device.cuh"
#include "internal.h"
#include "kernels.h"

namespace swapnet {

__device__ int g_tc_err;

namespace {

constexpr int kBM = 128;
constexpr int kBK = 64;  // 64 x 2 bytes = one 128-byte swizzle row
constexpr int kThreads = 192;
constexpr int kABytes = kBM * kBK * 2;

template <int BN> struct Cfg {
  static constexpr int kStages = BN == 64 ? 6 : 4;
  static constexpr int kLag = kStages - 2;  // gather: cp.async groups in flight per thread
  static constexpr int kBBytes = BN * kBK * 2;
  static constexpr int kSmem = kStages * (kABytes + kBBytes) + 1024 + 256;
};

struct TcArgs {
  int M, N, K;
  const void* x;  // conv input (gather)
  int H, Wd, C, Ho, Wo, kh, kw, stride, pad;
  Epi e;
  void* y;
  int64_t ldy;
  int* err;
  int kb_per_split;  // k-blocks per split; gridDim.z splits
  float* partial;    // [splits][M][N] fp32 partial sums (split-K only)
  int* counters;     // per output tile, zero between launches (split-K only)
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

// 8 consecutive outputs (16 bytes): acc -> bias, residual, activation -> T.
template <typename T>
__device__ __forceinline__ void epi8(const float (&a)[8], const T* bias, const T* res, T* out, int act,
                                     int res_post) {
  const uint4 b = *reinterpret_cast<const uint4*>(bias);
  uint4 r = make_uint4(0, 0, 0, 0);
  if (res) r = *reinterpret_cast<const uint4*>(res);
  const uint32_t bw[4] = {b.x, b.y, b.z, b.w};
  const uint32_t rw[4] = {r.x, r.y, r.z, r.w};
  uint32_t o[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float v0 = epilogue(a[2 * i], lo_f<T>(bw[i]), lo_f<T>(rw[i]), res != nullptr, act, res_post);
    const float v1 = epilogue(a[2 * i + 1], hi_f<T>(bw[i]), hi_f<T>(rw[i]), res != nullptr, act, res_post);
    o[i] = pack2<T>(v0, v1);
  }
  *reinterpret_cast<uint4*>(out) = make_uint4(o[0], o[1], o[2], o[3]);
}

// Final epilogue of 32 columns [n, n+32) of row m from fp32 values v.
template <typename T>
__device__ __forceinline__ void finish32(const float (&v)[32], const TcArgs& p, int m, int n, bool vec_ok) {
  const T* bias = static_cast<const T*>(p.e.bias);
  const T* res = static_cast<const T*>(p.e.res);
  T* y = static_cast<T*>(p.y) + (int64_t)m * p.ldy;
  const T* rrow = res ? res + (int64_t)m * p.e.ldr : nullptr;
  if (vec_ok && n + 32 <= p.N) {
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      float a[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) a[j] = v[8 * q + j];
      epi8<T>(a, bias + n + 8 * q, rrow ? rrow + n + 8 * q : nullptr, y + n + 8 * q, p.e.act, p.e.res_post);
    }
  } else {
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      if (n + j < p.N) {
        const float rv = rrow ? to_f<T>(rrow[n + j]) : 0.f;
        y[n + j] = from_f<T>(epilogue(v[j], to_f<T>(bias[n + j]), rv, rrow != nullptr, p.e.act, p.e.res_post));
      }
    }
  }
}

__device__ __forceinline__ void epi_bar() { asm volatile("bar.sync 1, 128;" ::: "memory"); }

template <typename T, int BN, bool GATHER>
__global__ void __launch_bounds__(kThreads, 1)
    tc_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB, const TcArgs p) {
  constexpr int kStages = Cfg<BN>::kStages;
  constexpr int kLag = Cfg<BN>::kLag;
  constexpr int kBBytes = Cfg<BN>::kBBytes;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + kStages * kABytes;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sB + kStages * kBBytes);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * kStages + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  volatile int* last_flag = reinterpret_cast<volatile int*>(tmem_slot + 2);
  const uint32_t full0 = smem_u32(bars), empty0 = smem_u32(bars + kStages);
  const uint32_t accum_bar = smem_u32(bars + 2 * kStages);
  auto full_bar = [&](int s) { return full0 + 8u * s; };
  auto empty_bar = [&](int s) { return empty0 + 8u * s; };

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int m0 = blockIdx.x * kBM, n0 = blockIdx.y * BN;
  const int KB = (p.K + kBK - 1) / kBK;
  const int kb0 = blockIdx.z * p.kb_per_split;
  const int nk = min(KB, kb0 + p.kb_per_split) - kb0;  // >= 1 by construction
  const int splits = gridDim.z;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(full_bar(s), GATHER ? 1 + 128 : 1);
      mbar_init(empty_bar(s), 1);
    }
    mbar_init(accum_bar, 1);
    *abort_flag = 0;
    *last_flag = 0;
    fence_barrier_init();
    fence_proxy_async_smem();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), BN);
    tmem_relinquish();
  }
  if (threadIdx.x == 0) {
    prefetch_tmap(&tmB);
    if (!GATHER) prefetch_tmap(&tmA);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer
      int i = 0;
      for (; i < nk; ++i) {
        const int s = i % kStages, r = i / kStages, kb = kb0 + i;
        if (!mbar_wait_bounded(empty_bar(s), (r & 1) ^ 1, abort_flag, p.err)) break;
        mbar_arrive_expect_tx(full_bar(s), kBBytes + (GATHER ? 0 : kABytes));
        tma_load_2d(smem_u32(sB + s * kBBytes), &tmB, full_bar(s), kb * kBK, n0);
        if (!GATHER) tma_load_2d(smem_u32(sA + s * kABytes), &tmA, full_bar(s), kb * kBK, m0);
      }
      if (i < nk) {
        // aborted: let the loads already issued land before the CTA exits
        volatile int no_abort = 0;
        for (int j = (i > kStages ? i - kStages : 0); j < i; ++j)
          mbar_wait_bounded(full_bar(j % kStages), (j / kStages) & 1, &no_abort, nullptr);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer
      constexpr uint32_t idesc = idesc_f16(std::is_same<T, __nv_bfloat16>::value ? 1 : 0, kBM, BN);
      for (int i = 0; i < nk; ++i) {
        const int s = i % kStages, r = i / kStages;
        if (!mbar_wait_bounded(full_bar(s), r & 1, abort_flag, p.err)) break;
        tc_fence_after();
        const uint64_t ad = smem_desc_sw128(smem_u32(sA + s * kABytes));
        const uint64_t bd = smem_desc_sw128(smem_u32(sB + s * kBBytes));
#pragma unroll
        for (int k = 0; k < kBK / 16; ++k) tc_mma_f16(tmem, ad + 2ull * k, bd + 2ull * k, idesc, (i | k) != 0);
        tc_commit(empty_bar(s));
      }
      tc_commit(accum_bar);  // fires once every MMA issued above has completed
    }
  } else {
    const int t = threadIdx.x - 64;  // 0..127
    if (GATHER) {
      // ---------------- implicit im2col gather of A (row t of the tile)
      const int m = m0 + t;
      const bool mvalid = m < p.M;
      int img = 0, oy = 0, ox = 0;
      if (mvalid) {
        const int hw = p.Ho * p.Wo;
        img = m / hw;
        const int rem = m - img * hw;
        oy = rem / p.Wo;
        ox = rem - oy * p.Wo;
      }
      const int iy0 = oy * p.stride - p.pad, ix0 = ox * p.stride - p.pad;
      const T* xb = static_cast<const T*>(p.x) + (int64_t)img * p.H * p.Wd * p.C;
      const uint32_t row_off = (uint32_t)((t >> 3) * 1024 + (t & 7) * 128);
      int i = 0;
      for (; i < nk; ++i) {
        const int s = i % kStages, r = i / kStages, kb = kb0 + i;
        if (!mbar_wait_bounded(empty_bar(s), (r & 1) ^ 1, abort_flag, p.err)) break;
        const uint32_t dst_row = smem_u32(sA + s * kABytes) + row_off;
        // the 64-wide K block starts at tap kb*64 / C (C is a multiple of 8)
        int k = kb * kBK;
        int tap = k / p.C;
        int c = k - tap * p.C;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          bool valid = mvalid && k < p.K;
          const T* src = static_cast<const T*>(p.x);
          if (valid) {
            const int ry = tap / p.kw;
            const int rx = tap - ry * p.kw;
            const int iy = iy0 + ry, ix = ix0 + rx;
            valid = (unsigned)iy < (unsigned)p.H && (unsigned)ix < (unsigned)p.Wd;
            if (valid) src = xb + ((int64_t)iy * p.Wd + ix) * p.C + c;
          }
          cp_async_16(dst_row + (uint32_t)((j ^ (t & 7)) << 4), src, valid);
          k += 8;
          c += 8;
          if (c == p.C) { c = 0; ++tap; }
        }
        cp_async_commit();
        if (i >= kLag) {
          cp_async_wait<kLag>();
          fence_proxy_async_smem();
          mbar_arrive(full_bar((i - kLag) % kStages));
        }
      }
      cp_async_wait<0>();
      fence_proxy_async_smem();
      for (int j = (i > kLag ? i - kLag : 0); j < i; ++j) mbar_arrive(full_bar(j % kStages));
    }
    // ---------------- epilogue
    const int q = warp & 3;
    const int m = m0 + q * 32 + lane;
    const bool ok = mbar_wait_bounded(accum_bar, 0, abort_flag, p.err);
    tc_fence_after();
    const bool vec_ok = ((p.ldy | n0) % 8 == 0) && (!p.e.res || ((p.e.ldr | n0) % 8 == 0));
    if (ok && splits == 1) {
#pragma unroll 1
      for (int c0 = 0; c0 < BN; c0 += 32) {
        uint32_t r[32];
        tmem_ld_32x32b_x32(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)c0, r);
        tmem_ld_wait();
        if (m < p.M && n0 + c0 < p.N) {
          float v[32];
#pragma unroll
          for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(r[j]);
          finish32<T>(v, p, m, n0 + c0, vec_ok);
        }
      }
    } else if (ok) {
      // split-K: publish the fp32 partial tile, then the last CTA of this
      // tile sums all partials in split order and applies the epilogue.
      float* part = p.partial + ((int64_t)blockIdx.z * p.M) * p.N;
      const bool pvec = (p.N % 4 == 0);
#pragma unroll 1
      for (int c0 = 0; c0 < BN; c0 += 32) {
        uint32_t r[32];
        tmem_ld_32x32b_x32(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)c0, r);
        tmem_ld_wait();
        const int n = n0 + c0;
        if (m < p.M && n < p.N) {
          float* dst = part + (int64_t)m * p.N + n;
          if (pvec && n + 32 <= p.N) {
#pragma unroll
            for (int j = 0; j < 32; j += 4)
              __stcg(reinterpret_cast<float4*>(dst + j), make_float4(__uint_as_float(r[j]), __uint_as_float(r[j + 1]),
                                                                       __uint_as_float(r[j + 2]), __uint_as_float(r[j + 3])));
          } else {
#pragma unroll
            for (int j = 0; j < 32; ++j)
              if (n + j < p.N) __stcg(dst + j, __uint_as_float(r[j]));
          }
        }
      }
      __threadfence();
      epi_bar();
      if (t == 0) {
        int* ctr = p.counters + blockIdx.y * gridDim.x + blockIdx.x;
        const int old = atomicAdd(ctr, 1);
        if (old == splits - 1) {
          *ctr = 0;  // ready for the next launch
          *last_flag = 1;
        }
      }
      epi_bar();
      if (*last_flag) {
        __threadfence();
#pragma unroll 1
        for (int c0 = 0; c0 < BN; c0 += 32) {
          const int n = n0 + c0;
          if (m >= p.M || n >= p.N) continue;
          float v[32];
#pragma unroll
          for (int j = 0; j < 32; ++j) v[j] = 0.f;
          for (int z = 0; z < splits; ++z) {
            const float* src = p.partial + ((int64_t)z * p.M + m) * p.N + n;
            if (pvec && n + 32 <= p.N) {
#pragma unroll
              for (int j = 0; j < 32; j += 4) {
                const float4 f = __ldcg(reinterpret_cast<const float4*>(src + j));
                v[j] += f.x; v[j + 1] += f.y; v[j + 2] += f.z; v[j + 3] += f.w;
              }
            } else {
#pragma unroll
              for (int j = 0; j < 32; ++j)
                if (n + j < p.N) v[j] += __ldcg(src + j);
            }
          }
          finish32<T>(v, p, m, n, vec_ok);
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, BN);
  }
}

// ------------------------------------------------------------ host side
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  });
  return fn;
}

int make_tmap(CUtensorMap* m, int dtype, const void* base, uint64_t inner, uint64_t rows, uint64_t row_stride_bytes,
              uint32_t box_rows) {
  auto fn = encode_fn();
  if (!fn) SN_FAIL(SWAPNET_ERR_CUDA, "cuTensorMapEncodeTiled unavailable");
  if (((uintptr_t)base & 15) || (row_stride_bytes & 15))
    SN_FAIL(SWAPNET_ERR_MISALIGNED, "TMA operand must be 16-byte aligned with a 16-byte multiple row stride");
  const cuuint64_t dims[2] = {inner, rows};
  const cuuint64_t strides[1] = {row_stride_bytes};
  const cuuint32_t box[2] = {(cuuint32_t)kBK, box_rows};
  const cuuint32_t estr[2] = {1, 1};
  const CUresult r = fn(m, dtype == SWAPNET_BF16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT16,
                        2, const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) SN_FAIL(SWAPNET_ERR_CUDA, "cuTensorMapEncodeTiled failed (" + std::to_string((int)r) + ")");
  return SWAPNET_OK;
}

template <typename T, int BN, bool GATHER>
int launch_inst(const TcGemm& g, const TcPlan& pl, int* err, cudaStream_t s) {
  static bool attr_done = false;  // per instantiation
  auto kern = tc_gemm_kernel<T, BN, GATHER>;
  if (!attr_done) {
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg<BN>::kSmem) != cudaSuccess)
      SN_FAIL(SWAPNET_ERR_CUDA, "cudaFuncSetAttribute failed");
    attr_done = true;
  }
  TcArgs a;
  std::memset(&a, 0, sizeof(a));
  a.M = g.M; a.N = g.N; a.K = g.K;
  a.x = g.A;
  a.H = g.H; a.Wd = g.Wd; a.C = g.C; a.Ho = g.Ho; a.Wo = g.Wo;
  a.kh = g.kh; a.kw = g.kw; a.stride = g.stride; a.pad = g.pad;
  a.e = g.e; a.y = g.y; a.ldy = g.ldy; a.err = err;
  a.kb_per_split = pl.kb_per_split;
  a.partial = g.partial;
  a.counters = g.counters;
  if (pl.splits > 1 && (!g.partial || !g.counters)) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "split-K needs scratch");
  const dim3 grid((g.M + kBM - 1) / kBM, (g.N + BN - 1) / BN, pl.splits);
  kern<<<grid, kThreads, Cfg<BN>::kSmem, s>>>(pl.tmA, pl.tmB, a);
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) SN_FAIL(SWAPNET_ERR_CUDA, std::string("tcgen05 GEMM launch: ") + cudaGetErrorString(e));
  return SWAPNET_OK;
}

}  // namespace

int tc_prepare(const TcGemm& g, TcPlan* p) {
  std::memset(p, 0, sizeof(*p));
  if (g.dtype != SWAPNET_F16 && g.dtype != SWAPNET_BF16) SN_FAIL(SWAPNET_ERR_UNSUPPORTED, "tcgen05 path: fp16/bf16 only");
  if (g.K % 8) SN_FAIL(SWAPNET_ERR_UNSUPPORTED, "tcgen05 path: K must be a multiple of 8");
  if (g.conv && g.C % 8) SN_FAIL(SWAPNET_ERR_UNSUPPORTED, "tcgen05 conv: channels must be a multiple of 8");
  if ((uintptr_t)g.y % 2) SN_FAIL(SWAPNET_ERR_MISALIGNED, "unaligned output");
  const int sms = g.num_sms > 0 ? g.num_sms : 148;
  if (g.N <= 64) {
    p->bn = 64;
  } else {
    const int64_t tiles128 = (int64_t)((g.M + kBM - 1) / kBM) * ((g.N + 127) / 128);
    p->bn = tiles128 < sms ? 64 : 128;
  }
  // deterministic split-K: enough CTAs to cover the SMs, >= 2 k-blocks each
  const int64_t tiles = (int64_t)((g.M + kBM - 1) / kBM) * ((g.N + p->bn - 1) / p->bn);
  const int KB = (g.K + kBK - 1) / kBK;
  int64_t splits = tiles >= sms ? 1 : std::min<int64_t>(sms / tiles, std::max(1, KB / 2));
  splits = std::max<int64_t>(1, std::min<int64_t>(splits, 32));
  p->kb_per_split = (KB + (int)splits - 1) / (int)splits;
  p->splits = (KB + p->kb_per_split - 1) / p->kb_per_split;
  p->tiles = tiles;
  p->scratch_bytes = p->splits > 1 ? (uint64_t)p->splits * g.M * g.N * sizeof(float) : 0;
  int rc = make_tmap(&p->tmB, g.dtype, g.W, (uint64_t)g.K, (uint64_t)g.N, (uint64_t)g.K * 2, (uint32_t)p->bn);
  if (rc) return rc;
  if (!g.conv && g.A) {
    rc = make_tmap(&p->tmA, g.dtype, g.A, (uint64_t)g.K, (uint64_t)g.M, (uint64_t)g.lda * 2, (uint32_t)kBM);
    if (rc) return rc;
  }
  p->ready = 1;
  return SWAPNET_OK;
}

int launch_tc_gemm(const TcGemm& g, const TcPlan& pl, int* err, cudaStream_t s) {
  if (!pl.ready) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "tcgen05 GEMM not prepared");
  const bool bf = g.dtype == SWAPNET_BF16;
  if (g.conv) {
    if (pl.bn == 64) return bf ? launch_inst<__nv_bfloat16, 64, true>(g, pl, err, s) : launch_inst<__half, 64, true>(g, pl, err, s);
    return bf ? launch_inst<__nv_bfloat16, 128, true>(g, pl, err, s) : launch_inst<__half, 128, true>(g, pl, err, s);
  }
  if (pl.bn == 64) return bf ? launch_inst<__nv_bfloat16, 64, false>(g, pl, err, s) : launch_inst<__half, 64, false>(g, pl, err, s);
  return bf ? launch_inst<__nv_bfloat16, 128, false>(g, pl, err, s) : launch_inst<__half, 128, false>(g, pl, err, s);
}

// ------------------------------------------------------------ allocation-free GEMM
// Scratch of swapnet_gemm_noalloc: tile counters (first kNoAllocCounterBytes)
// then fp32 split-K partials.  Zero-initialised when the module loads.
constexpr uint64_t kNoAllocBytes = SWAPNET_NOALLOC_SCRATCH_BYTES;
constexpr uint64_t kNoAllocCounterBytes = 64 * 1024;
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocBytes];

namespace {
struct NoAllocDevice {
  unsigned char* scratch = nullptr;  // device address of g_noalloc_scratch
  int* err = nullptr;                // device address of g_tc_err
  int sms = 0;
};
std::mutex g_noalloc_mu;
NoAllocDevice g_noalloc_dev[64];
}  // namespace

int tc_error_word(int** ptr) {
  void* p = nullptr;
  if (cudaGetSymbolAddress(&p, g_tc_err) != cudaSuccess) SN_FAIL(SWAPNET_ERR_CUDA, "cudaGetSymbolAddress failed");
  *ptr = static_cast<int*>(p);
  return SWAPNET_OK;
}

}  // namespace swapnet

extern "C" int swapnet_gemm_noalloc(int32_t dtype, const void* A, const void* W, const void* bias, void* Y,
                                    int32_t M, int32_t N, int32_t K, int32_t act, swapnet_stream stream) {
  using namespace swapnet;
  if (dtype != SWAPNET_F16 && dtype != SWAPNET_BF16) SN_FAIL(SWAPNET_ERR_UNSUPPORTED, "fp16 or bf16 only");
  if (!A || !W || !bias || !Y || M < 1 || N < 1 || K < 1) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null pointer or empty shape");
  if (act < SWAPNET_ACT_NONE || act > SWAPNET_ACT_LEAKY) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "bad activation");
  if (K % 8) SN_FAIL(SWAPNET_ERR_UNSUPPORTED, "K must be a multiple of 8");
  if (((uintptr_t)A | (uintptr_t)W | (uintptr_t)bias | (uintptr_t)Y) & 15)
    SN_FAIL(SWAPNET_ERR_MISALIGNED, "pointers must be 16-byte aligned");
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
    cudaGetLastError();
    SN_FAIL(SWAPNET_ERR_CUDA, "no current CUDA device");
  }
  NoAllocDevice d;
  {
    std::lock_guard<std::mutex> lk(g_noalloc_mu);
    NoAllocDevice& c = g_noalloc_dev[dev];
    if (!c.scratch) {  // once per device, with that device current
      void* p = nullptr;
      cudaError_t r = cudaGetSymbolAddress(&p, g_noalloc_scratch);
      if (r != cudaSuccess || !p) {
        cudaGetLastError();
        SN_FAIL(SWAPNET_ERR_CUDA, std::string("cudaGetSymbolAddress(scratch): ") + cudaGetErrorString(r));
      }
      void* e = nullptr;
      r = cudaGetSymbolAddress(&e, g_tc_err);
      if (r != cudaSuccess || !e) {
        cudaGetLastError();
        SN_FAIL(SWAPNET_ERR_CUDA, std::string("cudaGetSymbolAddress(error word): ") + cudaGetErrorString(r));
      }
      int sms = 0;
      if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
        cudaGetLastError();
        SN_FAIL(SWAPNET_ERR_CUDA, "device attribute query failed");
      }
      c.scratch = static_cast<unsigned char*>(p);
      c.err = static_cast<int*>(e);
      c.sms = sms;
    }
    d = c;
  }
  TcGemm g;
  std::memset(&g, 0, sizeof(g));
  g.dtype = dtype;
  g.M = M; g.N = N; g.K = K;
  g.W = W;
  g.A = A; g.lda = K; g.conv = 0;
  g.e.bias = bias; g.e.res = nullptr; g.e.ldr = N; g.e.act = act; g.e.res_post = 0;
  g.y = Y; g.ldy = N;
  g.num_sms = d.sms;
  TcPlan pl;
  int rc = tc_prepare(g, &pl);
  if (rc) return rc;
  if (pl.splits > 1) {
    const uint64_t counters = (uint64_t)pl.tiles * sizeof(int);
    if (counters > kNoAllocCounterBytes || kNoAllocCounterBytes + pl.scratch_bytes > kNoAllocBytes)
      SN_FAIL(SWAPNET_ERR_INVALID_ARG, "problem needs " + std::to_string(kNoAllocCounterBytes + pl.scratch_bytes) +
                                           " bytes of split-K scratch; the static scratch holds " +
                                           std::to_string(kNoAllocBytes));
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    if (cudaMemsetAsync(d.scratch, 0, counters, s) != cudaSuccess) {
      cudaGetLastError();
      SN_FAIL(SWAPNET_ERR_CUDA, "clearing the split-K counters failed");
    }
    g.counters = reinterpret_cast<int*>(d.scratch);
    g.partial = reinterpret_cast<float*>(d.scratch + kNoAllocCounterBytes);
  }
  return launch_tc_gemm(g, pl, d.err, reinterpret_cast<cudaStream_t>(stream));
}
