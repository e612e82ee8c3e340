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
// into the same swizzled layout.  One CTA computes one 128 x BN tile (BN 64
// or 128; 256 for linear layers of at most kFewRows rows, whose work is
// streaming the weight matrix):
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
#include "tc_epi.cuh"

namespace swapnet {

__device__ int g_tc_err;

namespace {

constexpr int kBM = 128;
constexpr int kBK = 64;  // 64 x 2 bytes = one 128-byte swizzle row
constexpr int kThreads = 192;
constexpr int kABytes = kBM * kBK * 2;

// N tile 256 serves GEMMs of at most kFewRows rows (one partly filled M
// tile) that stream a large weight matrix: their cluster split-K partials
// are distributed by column, so the receive buffer holds kFewRows rows.
constexpr int kFewRows = 16;

template <int BN> struct Cfg {
  static constexpr int kStages = BN == 64 ? 6 : 4;
  static constexpr int kLag = kStages - 2;  // gather: cp.async groups in flight per thread
  static constexpr int kBBytes = BN * kBK * 2;
  static constexpr int kStageBytes = kStages * (kABytes + kBBytes);
  // cluster split-K receive buffer.  BN 64/128 (row owners): up to 16 splits
  // x ceil(128/splits) rows.  BN 256 (column owners): splits x kFewRows rows
  // x (columns per owner + 4), at most kFewRows x (256 + 8 x 8) floats.
  static constexpr int kRecvBytes = BN == 256 ? kFewRows * (BN + 64) * 4 : (kBM + 15) * (BN + 4) * 4;
  static constexpr int kBiasBytes = BN * 4;
  static constexpr int kSmem = kStageBytes + kRecvBytes + kBiasBytes + 256 + 1024;
};

// A operand: kA2d (2-D TMA of a row-major matrix: linear layers, 1x1
// stride-1 convs), kAGather (cp.async im2col gather by warps 2..5), kATap
// (convs whose taps are whole 64-channel k-blocks: one 4-D TMA per k-block
// of the tap's 64 channels over a wt x ht patch of output pixels, zero fill
// for the padding; the CTA's 128 rows are that patch, rows >= wt * ht unused)
constexpr int kA2d = 0, kAGather = 1, kATap = 2;

template <typename T, int BN, int AMODE>
__global__ void __launch_bounds__(kThreads, 1)
    tc_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB, const TcArgs p) {
  constexpr bool GATHER = AMODE == kAGather;
  constexpr bool TAP = AMODE == kATap;
  constexpr int kStages = Cfg<BN>::kStages;
  constexpr int kLag = Cfg<BN>::kLag;
  constexpr int kBBytes = Cfg<BN>::kBBytes;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + kStages * kABytes;
  float* recv = reinterpret_cast<float*>(smem + Cfg<BN>::kStageBytes);
  float* sbias = reinterpret_cast<float*>(smem + Cfg<BN>::kStageBytes + Cfg<BN>::kRecvBytes);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + Cfg<BN>::kStageBytes + Cfg<BN>::kRecvBytes + Cfg<BN>::kBiasBytes);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * kStages + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  volatile int* last_flag = reinterpret_cast<volatile int*>(tmem_slot + 2);
  const uint32_t full0 = smem_u32(bars), empty0 = smem_u32(bars + kStages);
  const uint32_t accum_bar = smem_u32(bars + 2 * kStages);
  auto full_bar = [&](int s) { return full0 + 8u * s; };
  auto empty_bar = [&](int s) { return empty0 + 8u * s; };

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int m0 = TAP ? 0 : blockIdx.x * kBM, n0 = blockIdx.y * BN;
  // tap mode: this CTA's patch (image, patch row th, patch column tw)
  int pimg = 0, pth = 0, ptw = 0;
  if (TAP) {
    const int patches = p.tiles_w * p.tiles_h;
    pimg = blockIdx.x / patches;
    const int rem = blockIdx.x - pimg * patches;
    pth = rem / p.tiles_w;
    ptw = rem - pth * p.tiles_w;
  }
  const uint32_t a_bytes = TAP ? (uint32_t)(p.wt * p.ht * 128) : (GATHER ? 0u : (uint32_t)kABytes);
  // output row of tile row r (-1: no output)
  auto row_m = [&](int r) -> int {
    if (TAP) {
      if (r >= p.wt * p.ht) return -1;
      const int oy = pth * p.ht + r / p.wt, ox = ptw * p.wt + r % p.wt;
      return (oy < p.Ho && ox < p.Wo) ? (pimg * p.Ho + oy) * p.Wo + ox : -1;
    }
    return m0 + r < p.M ? m0 + r : -1;
  };
  // A tile of k-block kb into stage buffer dst (TMA modes)
  auto load_a = [&](uint32_t dst, uint32_t bar, int kb) {
    if (TAP) {
      const int k0 = kb * kBK, tap = k0 / p.C, c0 = k0 - tap * p.C;
      const int ry = tap / p.kw, rx = tap - ry * p.kw;
      tma_load_4d(dst, &tmA, bar, c0, ptw * p.wt * p.stride - p.pad + rx, pth * p.ht * p.stride - p.pad + ry, pimg);
    } else {
      tma_load_2d(dst, &tmA, bar, kb * kBK, m0);
    }
  };
  const int KB = (p.K + kBK - 1) / kBK;
  const int kb0 = blockIdx.z * p.kb_per_split;
  const int nk = min(KB, kb0 + p.kb_per_split) - kb0;  // >= 1 by construction
  const int splits = gridDim.z;
  const bool csplit = splits > 1 && p.cluster;

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
  // bias of this tile to shared memory (weights: ready before the kernel)
  if (threadIdx.x >= 64) {
    const T* bias = static_cast<const T*>(p.e.bias);
    for (int j = threadIdx.x - 64; j < BN; j += 128) sbias[j] = (bias && n0 + j < p.N) ? to_f<T>(bias[n0 + j]) : 0.f;
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_launch_dependents();
  if (csplit) asm volatile("barrier.cluster.arrive.relaxed;" ::: "memory");  // peers started (waited before DSMEM use)

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer: weight tiles of the first stages go
      // out before waiting for the previous kernel (they do not depend on it)
      const int early = min(nk, kStages);
      for (int i = 0; i < early; ++i) {
        mbar_arrive_expect_tx(full_bar(i), kBBytes + a_bytes);
        tma_load_2d(smem_u32(sB + i * kBBytes), &tmB, full_bar(i), (kb0 + i) * kBK, n0);
      }
      pdl_wait();
      if (!GATHER)
        for (int i = 0; i < early; ++i) load_a(smem_u32(sA + i * kABytes), full_bar(i), kb0 + i);
      int i = early;
      for (; i < nk; ++i) {
        const int s = i % kStages, r = i / kStages, kb = kb0 + i;
        if (!mbar_wait_bounded(empty_bar(s), (r & 1) ^ 1, abort_flag, p.err)) break;
        mbar_arrive_expect_tx(full_bar(s), kBBytes + a_bytes);
        tma_load_2d(smem_u32(sB + s * kBBytes), &tmB, full_bar(s), kb * kBK, n0);
        if (!GATHER) load_a(smem_u32(sA + s * kABytes), full_bar(s), kb);
      }
      if (i < nk) {
        // aborted: let the loads already issued land before the CTA exits
        volatile int no_abort = 0;
        for (int j = (i > kStages ? i - kStages : 0); j < i; ++j)
          mbar_wait_bounded(full_bar(j % kStages), (j / kStages) & 1, &no_abort, nullptr);
      }
    } else {
      pdl_wait();
    }
  } else if (warp == 1) {
    pdl_wait();
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
    pdl_wait();
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
      const uint32_t sw = (uint32_t)(t & 7);
      // position of the first K element of this split: tap (ry, rx), channel c
      int k = kb0 * kBK;
      int tap = k / p.C;
      int c = k - tap * p.C;
      int ry = tap / p.kw, rx = tap - (tap / p.kw) * p.kw;
      const bool whole_tap = (p.C % kBK) == 0;  // a 64-wide K block never straddles taps
      int i = 0;
      for (; i < nk; ++i) {
        const int s = i % kStages, r = i / kStages;
        if (!mbar_wait_bounded(empty_bar(s), (r & 1) ^ 1, abort_flag, p.err)) break;
        const uint32_t dst_row = smem_u32(sA + s * kABytes) + row_off;
        if (whole_tap) {
          const int iy = iy0 + ry, ix = ix0 + rx;
          const bool valid = mvalid && k < p.K && (unsigned)iy < (unsigned)p.H && (unsigned)ix < (unsigned)p.Wd;
          const T* src = valid ? xb + ((int64_t)iy * p.Wd + ix) * p.C + c : static_cast<const T*>(p.x);
#pragma unroll
          for (int j = 0; j < 8; ++j) cp_async_16(dst_row + (((uint32_t)j ^ sw) << 4), src + (valid ? 8 * j : 0), valid);
          k += kBK;
          c += kBK;
          if (c == p.C) {
            c = 0;
            if (++rx == p.kw) { rx = 0; ++ry; }
          }
        } else {
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            const int iy = iy0 + ry, ix = ix0 + rx;
            const bool valid =
                mvalid && k < p.K && (unsigned)iy < (unsigned)p.H && (unsigned)ix < (unsigned)p.Wd;
            const T* src = valid ? xb + ((int64_t)iy * p.Wd + ix) * p.C + c : static_cast<const T*>(p.x);
            cp_async_16(dst_row + (((uint32_t)j ^ sw) << 4), src, valid);
            k += 8;
            c += 8;
            if (c == p.C) {
              c = 0;
              if (++rx == p.kw) { rx = 0; ++ry; }
            }
          }
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
    const int row = q * 32 + lane;
    const int m = row_m(row);  // -1: this row has no output
    const bool vec_ok = ((p.ldy | n0) % 8 == 0) && (!p.e.res || ((p.e.ldr | n0) % 8 == 0));
    // without a split, the residual of the first 32 columns is requested
    // while the MMAs run, each later chunk's one chunk ahead of its use (zeros
    // for layers without one: one loop for both measured faster than two)
    const bool has_res = splits == 1;
    uint4 rnext[4];
    if (has_res) res_prefetch32<T>(rnext, p, m, n0, vec_ok);
    const bool ok = mbar_wait_bounded(accum_bar, 0, abort_flag, p.err);
    tc_fence_after();
    if (ok && splits == 1) {
#pragma unroll 1
      for (int c0 = 0; c0 < BN; c0 += 32) {
        uint4 rcur[4];
        if (has_res) {
#pragma unroll
          for (int i = 0; i < 4; ++i) rcur[i] = rnext[i];
          if (c0 + 32 < BN) res_prefetch32<T>(rnext, p, m, n0 + c0 + 32, vec_ok);
        }
        uint32_t r[32];
        tmem_ld_32x32b_x32(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)c0, r);
        tmem_ld_wait();
        if (m >= 0 && n0 + c0 < p.N) {
          float v[32];
#pragma unroll
          for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(r[j]);
          if (has_res) finish32r<T>(v, sbias + c0, p, m, n0 + c0, vec_ok, rcur);
          else finish32<T>(v, sbias + c0, p, m, n0 + c0, vec_ok);
        }
      }
    } else if (csplit && BN == 256) {
      // cluster split-K over columns (at most kFewRows rows): columns
      // [o * cpo, (o + 1) * cpo) of the tile belong to CTA o of the cluster;
      // this split's partial goes to slot blockIdx.z of each owner
      const int cpo = (((BN + splits - 1) / splits) + 3) & ~3;
      const int rs = cpo + 4;  // row stride of a slot, floats
      const bool mine = ok && m >= 0 && row < kFewRows;
      asm volatile("barrier.cluster.wait;" ::: "memory");  // every peer is running
#pragma unroll 1
      for (int c0 = 0; c0 < BN; c0 += 32) {
        uint32_t r[32];
        tmem_ld_32x32b_x32(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)c0, r);
        tmem_ld_wait();
        if (mine) {
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            const int c = c0 + 4 * j;
            const uint32_t owner = (uint32_t)(c / cpo);
            const int cl = c - (int)owner * cpo;
            const uint32_t la = smem_u32(recv) + (uint32_t)((((int)blockIdx.z * kFewRows + row) * rs + cl) * 4);
            uint32_t ra;
            asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(ra) : "r"(la), "r"(owner));
            asm volatile("st.shared::cluster.v4.f32 [%0], {%1,%2,%3,%4};" ::"r"(ra), "f"(__uint_as_float(r[4 * j])),
                         "f"(__uint_as_float(r[4 * j + 1])), "f"(__uint_as_float(r[4 * j + 2])),
                         "f"(__uint_as_float(r[4 * j + 3]))
                         : "memory");
          }
        }
      }
    } else if (csplit) {
      // cluster split-K: push this split's rows to the CTA that owns them
      // (owner of row w = w / rows_per_owner), slot = this split's index
      const int rpo = (kBM + splits - 1) / splits;
      const uint32_t owner = (uint32_t)(row / rpo);
      const int rr = row - (int)owner * rpo;
      const uint32_t base = smem_u32(recv) + (uint32_t)(((blockIdx.z * rpo + rr) * (BN + 4)) * 4);
      asm volatile("barrier.cluster.wait;" ::: "memory");  // every peer is running
#pragma unroll 1
      for (int c0 = 0; c0 < BN; c0 += 32) {
        uint32_t r[32];
        tmem_ld_32x32b_x32(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)c0, r);
        tmem_ld_wait();
        if (ok && m >= 0) {
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            uint32_t ra;
            asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(ra) : "r"(base + (uint32_t)((c0 + 4 * j) * 4)), "r"(owner));
            asm volatile("st.shared::cluster.v4.f32 [%0], {%1,%2,%3,%4};" ::"r"(ra), "f"(__uint_as_float(r[4 * j])),
                         "f"(__uint_as_float(r[4 * j + 1])), "f"(__uint_as_float(r[4 * j + 2])),
                         "f"(__uint_as_float(r[4 * j + 3]))
                         : "memory");
          }
        }
      }
    } else if (ok) {
      // global split-K: publish the fp32 partial tile, then the last CTA of
      // this tile sums all partials in split order and applies the epilogue.
      float* part = p.partial + ((int64_t)blockIdx.z * p.M) * p.N;
      const bool pvec = (p.N % 4 == 0);
#pragma unroll 1
      for (int c0 = 0; c0 < BN; c0 += 32) {
        uint32_t r[32];
        tmem_ld_32x32b_x32(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)c0, r);
        tmem_ld_wait();
        const int n = n0 + c0;
        if (m >= 0 && n < p.N) {
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
          if (m < 0 || n >= p.N) continue;
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
          finish32<T>(v, sbias + c0, p, m, n, vec_ok);
        }
      }
    }
  }
  if (csplit) {
    if (threadIdx.x < 64) asm volatile("barrier.cluster.wait;" ::: "memory");  // pairs the early arrive
    // all pushes are visible after this barrier; each CTA reduces the rows
    // it owns from its own receive buffer, in split order 0..S-1
    asm volatile("barrier.cluster.arrive.release;\n\tbarrier.cluster.wait.acquire;" ::: "memory");
    if constexpr (BN == 256) {
      // this CTA owns columns [c_lo, c_hi) of the tile, every row
      const int cpo = (((BN + splits - 1) / splits) + 3) & ~3;
      const int rs = cpo + 4;
      const int c_lo = (int)blockIdx.z * cpo, c_hi = min(BN, c_lo + cpo);
      const int rows = max(0, min(kFewRows, p.M - m0));
      const int w4 = max(0, c_hi - c_lo) / 4;
      const int groups = rows * w4;
      for (int g = threadIdx.x; g < groups; g += kThreads) {
        const int rr = g / w4, c4 = g % w4;
        const int n = n0 + c_lo + 4 * c4;
        const float* src = recv + rr * rs + 4 * c4;
        float4 acc = *reinterpret_cast<const float4*>(src);
        for (int z = 1; z < splits; ++z) {
          const float4 v = *reinterpret_cast<const float4*>(src + z * kFewRows * rs);
          acc.x += v.x; acc.y += v.y; acc.z += v.z; acc.w += v.w;
        }
        if (n < p.N) finish4<T>(acc, sbias + c_lo + 4 * c4, p, m0 + rr, n);
      }
    } else {
      const int rpo = (kBM + splits - 1) / splits;
      const int r0 = (int)blockIdx.z * rpo;
      const int rows = TAP ? max(0, min(rpo, kBM - r0)) : max(0, min(min(rpo, kBM - r0), p.M - m0 - r0));
      const int groups = rows * (BN / 4);
      for (int g = threadIdx.x; g < groups; g += kThreads) {
        const int rr = g / (BN / 4), c4 = g % (BN / 4);
        const int n = n0 + 4 * c4;
        const int mm = row_m(r0 + rr);
        if (mm < 0) continue;
        const float* src = recv + rr * (BN + 4) + 4 * c4;
        float4 acc = *reinterpret_cast<const float4*>(src);
        for (int z = 1; z < splits; ++z) {
          const float4 v = *reinterpret_cast<const float4*>(src + z * rpo * (BN + 4));
          acc.x += v.x; acc.y += v.y; acc.z += v.z; acc.w += v.w;
        }
        if (n < p.N) finish4<T>(acc, sbias + 4 * c4, p, mm, n);
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

// 4-D map of an NHWC activation tensor for per-tap im2col loads: box of 64
// channels x wt columns x ht rows of one image, every s-th column and row
// (the conv stride), zero fill outside the image (the conv padding).
int make_tmap_conv4d(CUtensorMap* m, int dtype, const void* base, int n, int h, int w, int c, int wt, int ht,
                     int stride) {
  auto fn = encode_fn();
  if (!fn) SN_FAIL(SWAPNET_ERR_CUDA, "cuTensorMapEncodeTiled unavailable");
  if (((uintptr_t)base & 15) || (c * 2) % 16)
    SN_FAIL(SWAPNET_ERR_MISALIGNED, "TMA conv operand must be 16-byte aligned");
  const cuuint64_t dims[4] = {(cuuint64_t)c, (cuuint64_t)w, (cuuint64_t)h, (cuuint64_t)n};
  const cuuint64_t strides[3] = {(cuuint64_t)c * 2, (cuuint64_t)w * c * 2, (cuuint64_t)h * w * c * 2};
  const cuuint32_t box[4] = {(cuuint32_t)kBK, (cuuint32_t)(wt * stride), (cuuint32_t)(ht * stride), 1};
  const cuuint32_t estr[4] = {1, (cuuint32_t)stride, (cuuint32_t)stride, 1};
  const CUresult r = fn(m, dtype == SWAPNET_BF16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT16,
                        4, const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS)
    SN_FAIL(SWAPNET_ERR_CUDA, "cuTensorMapEncodeTiled (conv) failed (" + std::to_string((int)r) + ")");
  return SWAPNET_OK;
}

// Output patch (wt x ht pixels, wt * ht <= 128) for per-tap TMA loads that
// wastes the fewest of the 128 MMA rows; returns the used fraction.
double conv_patch(int ho, int wo, int stride, int* wt, int* ht) {
  double best = 0.0;
  *wt = *ht = 0;
  for (int cand : {wo, 128, 64, 32, 16, 8, 4}) {
    if (cand < 1 || cand > 128 || cand * stride > 256) continue;
    const int w_ = cand, h_ = std::min(128 / w_, ho);
    if (h_ < 1 || h_ * stride > 256) continue;
    const double tiles = (double)((wo + w_ - 1) / w_) * ((ho + h_ - 1) / h_);
    const double util = (double)ho * wo / (tiles * kBM);
    if (util > best + 1e-9) {
      best = util;
      *wt = w_;
      *ht = h_;
    }
  }
  return best;
}

template <typename T, int BN, int AMODE>
int launch_inst(const TcGemm& g, const TcPlan& pl, int* err, cudaStream_t s) {
  static std::atomic<uint64_t> attr_done{0};  // per instantiation, one bit per device
  auto kern = tc_gemm_kernel<T, BN, AMODE>;
  if (attr_needed(attr_done)) {
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg<BN>::kSmem) != cudaSuccess)
      SN_FAIL(SWAPNET_ERR_CUDA, "cudaFuncSetAttribute failed");
    attr_set(attr_done);
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
  if (pl.splits > 1 && !pl.cluster && (!g.partial || !g.counters))
    SN_FAIL(SWAPNET_ERR_INVALID_ARG, "split-K needs scratch");
  a.wt = pl.wt; a.ht = pl.ht; a.tiles_w = pl.tiles_w; a.tiles_h = pl.tiles_h;
  const int64_t mtiles = AMODE == kATap ? (int64_t)g.M / ((int64_t)g.Ho * g.Wo) * pl.tiles_w * pl.tiles_h
                                        : (g.M + kBM - 1) / kBM;
  if (AMODE == kATap && (pl.splits > 1 && !pl.cluster)) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "tap mode needs cluster split-K");
  const dim3 grid((unsigned)mtiles, (g.N + BN - 1) / BN, pl.splits);
  a.cluster = pl.cluster;
  const bool csplit = pl.splits > 1 && pl.cluster;
  if (csplit) {
    static std::atomic<uint64_t> np_done{0};  // per instantiation, one bit per device
    if (attr_needed(np_done)) {
      if (cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) != cudaSuccess)
        SN_FAIL(SWAPNET_ERR_CUDA, "non-portable cluster attribute failed");
      attr_set(np_done);
    }
  }
  cudaLaunchConfig_t cfg;
  std::memset(&cfg, 0, sizeof(cfg));
  cfg.gridDim = grid;
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = Cfg<BN>::kSmem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  int na = 0;
  if (!g.no_pdl) {
    attr[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[na].val.programmaticStreamSerializationAllowed = 1;
    ++na;
  }
  if (csplit) {
    attr[na].id = cudaLaunchAttributeClusterDimension;
    attr[na].val.clusterDim.x = 1;
    attr[na].val.clusterDim.y = 1;
    attr[na].val.clusterDim.z = pl.splits;
    ++na;
  }
  cfg.attrs = attr;
  cfg.numAttrs = na;
  const cudaError_t le = cudaLaunchKernelEx(&cfg, kern, pl.tmA, pl.tmB, a);
  if (le != cudaSuccess) SN_FAIL(SWAPNET_ERR_CUDA, std::string("tcgen05 GEMM launch: ") + cudaGetErrorString(le));
  return SWAPNET_OK;
}


// Largest cluster (along the split dimension) that the device can co-schedule
// for this kernel instance: 16, 8, 4 or 2 (cached per instance and device).
template <typename T, int BN, int AMODE>
int max_cluster_inst() {
  static std::atomic<int> cached[64];  // 0 until known
  const int dev = device_index();
  if (dev >= 0) {
    const int c = cached[dev].load(std::memory_order_relaxed);
    if (c > 0) return c;
  }
  auto kern = tc_gemm_kernel<T, BN, AMODE>;
  cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg<BN>::kSmem);
  cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  int best = 1;
  for (int c : {16, 8, 4, 2}) {
    cudaLaunchConfig_t cfg;
    std::memset(&cfg, 0, sizeof(cfg));
    cfg.gridDim = dim3(1, 1, c);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = Cfg<BN>::kSmem;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 1;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = c;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) == cudaSuccess && n > 0) {
      best = c;
      break;
    }
    cudaGetLastError();
  }
  if (dev >= 0) cached[dev].store(best, std::memory_order_relaxed);
  return best;
}

// Clusters of c CTAs of the N-tile-256 instance that the device runs at
// once (cudaOccupancyMaxActiveClusters; cached per dtype, size and device).
template <typename T>
int active_clusters_inst(int c) {
  static std::atomic<int> cached[64][9];  // the count + 1, 0 until known
  if (c < 1 || c > 8) return 0;
  const int dev = device_index();
  if (dev >= 0) {
    const int v = cached[dev][c].load(std::memory_order_relaxed);
    if (v > 0) return v - 1;
  }
  auto kern = tc_gemm_kernel<T, 256, kA2d>;
  cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg<256>::kSmem);
  cudaLaunchConfig_t cfg;
  std::memset(&cfg, 0, sizeof(cfg));
  cfg.gridDim = dim3(1, 1, c);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = Cfg<256>::kSmem;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 1;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = c;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess) {
    cudaGetLastError();
    n = 0;
  }
  if (dev >= 0) cached[dev][c].store(n + 1, std::memory_order_relaxed);
  return n;
}

int active_clusters(int dtype, int c) {
  return dtype == SWAPNET_BF16 ? active_clusters_inst<__nv_bfloat16>(c) : active_clusters_inst<__half>(c);
}

int max_cluster(int dtype, int bn, bool gather) {
  const bool bf = dtype == SWAPNET_BF16;
  if (bn == 256) return bf ? max_cluster_inst<__nv_bfloat16, 256, kA2d>() : max_cluster_inst<__half, 256, kA2d>();
  if (bn == 64)
    return gather ? (bf ? max_cluster_inst<__nv_bfloat16, 64, kAGather>() : max_cluster_inst<__half, 64, kAGather>())
                  : (bf ? max_cluster_inst<__nv_bfloat16, 64, kA2d>() : max_cluster_inst<__half, 64, kA2d>());
  return gather ? (bf ? max_cluster_inst<__nv_bfloat16, 128, kAGather>() : max_cluster_inst<__half, 128, kAGather>())
                : (bf ? max_cluster_inst<__nv_bfloat16, 128, kA2d>() : max_cluster_inst<__half, 128, kA2d>());
}

}  // namespace

int tc_prepare(const TcGemm& g, TcPlan* p) {
  std::memset(p, 0, sizeof(*p));
  if (g.dtype != SWAPNET_F16 && g.dtype != SWAPNET_BF16) SN_FAIL(SWAPNET_ERR_UNSUPPORTED, "tcgen05 path: fp16/bf16 only");
  if (g.K % 8) SN_FAIL(SWAPNET_ERR_UNSUPPORTED, "tcgen05 path: K must be a multiple of 8");
  if (g.conv && g.C % 8) SN_FAIL(SWAPNET_ERR_UNSUPPORTED, "tcgen05 conv: channels must be a multiple of 8");
  if ((uintptr_t)g.y % 2) SN_FAIL(SWAPNET_ERR_MISALIGNED, "unaligned output");
  const int sms = g.num_sms > 0 ? g.num_sms : 148;
  const int Nd = g.N_layer > 0 ? g.N_layer : g.N;  // decisions follow the whole layer
  const int64_t mtiles = (g.M + kBM - 1) / kBM;
  if (g.allow_persist) {
    // at least one output tile per SM: the persistent kernel, no split.
    // Convolutions whose taps are whole 64-channel k-blocks load A by 4-D TMA
    // when a pixel patch fills the 128 MMA rows well enough.
    int wt = 0, ht = 0;
    const bool tmac = g.conv && g.C % kBK == 0 && conv_patch(g.Ho, g.Wo, g.stride, &wt, &ht) >= 0.75;
    const int64_t sp_tiles = tmac ? (int64_t)g.M / ((int64_t)g.Ho * g.Wo) * ((g.Wo + wt - 1) / wt) *
                                        ((g.Ho + ht - 1) / ht)
                                  : mtiles;
    // the widest useful N tile.  Measured on this kernel, a pipeline stage
    // costs about the same (~0.5 us) whatever the tile width, so the time is
    // about waves x k-blocks and wider tiles mean fewer waves; a third of the
    // SMs busy with one wide tile each still beats splitting K across them
    int pbn = Nd <= 64 ? 64 : (Nd <= 128 ? 128 : 256);
    // with at most half as many 256-wide tiles as SMs, 128-wide tiles (twice
    // the CTAs) were measured faster: the 512-token decoder projections
    // 25.8 -> 23.4 us (q, k, v), 32.3 -> 26.7 us (o), 74.1 -> 57.1 us (down),
    // VGG-16 b16's 14x14 convolutions 27.8 -> 25.1 us
    if (pbn == 256 && sp_tiles * ((Nd + 255) / 256) * 2 <= sms) pbn = 128;
    if (sp_tiles * ((Nd + pbn - 1) / pbn) * 3 >= sms) {
      p->persist = 1;
      if (tmac) {
        p->tma_conv = 1;
        p->wt = wt;
        p->ht = ht;
        p->tiles_w = (g.Wo + wt - 1) / wt;
        p->tiles_h = (g.Ho + ht - 1) / ht;
      }
      p->bn = pbn;
      p->splits = 1;
      p->kb_per_split = (g.K + kBK - 1) / kBK;
      // N tiles of 64 with A by TMA: four (else two) 128-row sub-tiles per
      // tile share each weight stage when that still leaves a tile per SM.
      // Their MMAs go to independent accumulators, which the tensor pipe
      // overlaps: a single 128x64x16 MMA chain leaves it mostly idle
      p->msub = 1;
      if (pbn == 64 && (!g.conv || tmac)) {
        const int64_t nt64 = (Nd + 63) / 64;
        if ((sp_tiles + 3) / 4 * nt64 >= sms) p->msub = 4;
        else if ((sp_tiles + 1) / 2 * nt64 >= sms) p->msub = 2;
      }
      p->tiles = (sp_tiles + p->msub - 1) / p->msub * ((g.N + pbn - 1) / pbn);
      int rc = make_tmap(&p->tmB, g.dtype, g.W, (uint64_t)g.K, (uint64_t)g.N, (uint64_t)g.K * 2, (uint32_t)pbn);
      if (rc) return rc;
      if (!g.conv && g.A) {
        rc = make_tmap(&p->tmA, g.dtype, g.A, (uint64_t)g.K, (uint64_t)g.M, (uint64_t)g.lda * 2, (uint32_t)kBM);
        if (rc) return rc;
      }
      if (tmac && g.A) {
        const int n_img = (int)((int64_t)g.M / ((int64_t)g.Ho * g.Wo));
        rc = make_tmap_conv4d(&p->tmA, g.dtype, g.A, n_img, g.H, g.Wd, g.C, wt, ht, g.stride);
        if (rc) return rc;
      }
      p->ready = 1;
      return SWAPNET_OK;
    }
  }
  const int KB = (g.K + kBK - 1) / kBK;
  if (g.cluster_max > 0 && !g.conv && g.M <= kFewRows && KB >= 16) {
    // a few rows against a large weight matrix: streaming the weights is the
    // work.  A 128xNx16 MMA costs about the same for N = 64 and 256, so the
    // widest tile moves 4x the weight bytes per MMA; K is split across a
    // cluster (column-owner reduction).  The split count minimises
    // waves x k-blocks per CTA, a wave being the clusters of that size the
    // device co-schedules: clusters of 7-8 CTAs of this kernel do not all
    // fit at once, and the second wave costs more than the wider split saves
    p->bn = 256;
    const int64_t tiles_d = (Nd + 255) / 256;
    const int smax = std::max(1, std::min(std::min(8, KB / 8), std::min(g.cluster_max, max_cluster(g.dtype, 256, false))));
    int64_t splits = 1, best = -1;
    for (int c = 1; c <= smax; ++c) {
      const int64_t act = c == 1 ? sms : active_clusters(g.dtype, c);
      if (act < 1) continue;
      const int64_t cost = (tiles_d + act - 1) / act * ((KB + c - 1) / c);
      if (best < 0 || cost < best) {
        best = cost;
        splits = c;
      }
    }
    p->cluster = 1;
    p->kb_per_split = (KB + (int)splits - 1) / (int)splits;
    p->splits = (KB + p->kb_per_split - 1) / p->kb_per_split;
    p->tiles = (g.N + 255) / 256;
    int rc = make_tmap(&p->tmB, g.dtype, g.W, (uint64_t)g.K, (uint64_t)g.N, (uint64_t)g.K * 2, 256u);
    if (rc) return rc;
    if (g.A) {
      rc = make_tmap(&p->tmA, g.dtype, g.A, (uint64_t)g.K, (uint64_t)g.M, (uint64_t)g.lda * 2, (uint32_t)kBM);
      if (rc) return rc;
    }
    p->ready = 1;
    return SWAPNET_OK;
  }
  // convolutions whose taps are whole 64-channel k-blocks: A by one 4-D TMA
  // per tap over a pixel patch (as in the persistent kernel) instead of the
  // cp.async gather, when the patches fill the 128 rows well enough or need
  // no more CTAs than 128-row tiles would (these layers are latency-bound:
  // unused MMA rows cost nothing, the gather's address work does); the CTA
  // grid then runs over patches
  int twt = 0, tht = 0;
  bool tap = false;
  int64_t mt = (int64_t)((g.M + kBM - 1) / kBM);
  if (g.conv && g.cluster_max > 0 && g.C % kBK == 0) {
    const double util = conv_patch(g.Ho, g.Wo, g.stride, &twt, &tht);
    const int64_t patches = twt > 0 ? (int64_t)g.M / ((int64_t)g.Ho * g.Wo) * ((g.Wo + twt - 1) / twt) *
                                          ((g.Ho + tht - 1) / tht)
                                    : 0;
    if (twt > 0 && (util >= 0.75 || patches <= mt)) {
      tap = true;
      mt = patches;
    }
  }
  if (Nd <= 64) {
    p->bn = 64;
  } else {
    const int64_t tiles128 = mt * ((Nd + 127) / 128);
    p->bn = tiles128 < sms ? 64 : 128;
  }
  // deterministic split-K: enough CTAs to cover the SMs, >= 2 k-blocks each
  const int64_t tiles_d = mt * ((Nd + p->bn - 1) / p->bn);
  const int64_t tiles = mt * ((g.N + p->bn - 1) / p->bn);
  int64_t splits = tiles_d >= sms ? 1 : std::min<int64_t>(sms / tiles_d, std::max(1, KB / 2));
  if (g.cluster_max > 0) {
    // cluster split-K, from sweeps of the split count on the batch-1 CNN
    // layers: the cluster reduction costs more than it saves below nine
    // k-blocks; clusters above 8 CTAs, or more than ~96 CTAs in clusters of
    // 5-8, wait longer to be scheduled than the split saves, while clusters
    // of up to 4 filling up to one wave of SMs pay off from 16 k-blocks
    // (YOLOv3's 26x26 and 13x13 3x3 convs: 15.7 -> 12.8 us, 13.1 -> 11.0 us)
    const int64_t s96 = std::min<int64_t>(splits, std::min<int64_t>(8, std::max<int64_t>(1, 96 / tiles_d)));
    if (KB <= 8) splits = 1;
    else if (KB < 16) splits = s96;
    else splits = std::max<int64_t>(s96, std::min<int64_t>(splits, 4));
  }
  const int cap = g.cluster_max > 0 ? std::min(g.cluster_max, max_cluster(g.dtype, p->bn, g.conv && !tap)) : 32;
  splits = std::max<int64_t>(1, std::min<int64_t>(splits, cap));
  p->cluster = g.cluster_max > 0 ? 1 : 0;
  p->kb_per_split = (KB + (int)splits - 1) / (int)splits;
  p->splits = (KB + p->kb_per_split - 1) / p->kb_per_split;
  p->tiles = tiles;
  p->scratch_bytes = (p->splits > 1 && !p->cluster) ? (uint64_t)p->splits * g.M * g.N * sizeof(float) : 0;
  int rc = make_tmap(&p->tmB, g.dtype, g.W, (uint64_t)g.K, (uint64_t)g.N, (uint64_t)g.K * 2, (uint32_t)p->bn);
  if (rc) return rc;
  if (!g.conv && g.A) {
    rc = make_tmap(&p->tmA, g.dtype, g.A, (uint64_t)g.K, (uint64_t)g.M, (uint64_t)g.lda * 2, (uint32_t)kBM);
    if (rc) return rc;
  }
  if (tap) {
    p->tma_conv = 1;
    p->wt = twt;
    p->ht = tht;
    p->tiles_w = (g.Wo + twt - 1) / twt;
    p->tiles_h = (g.Ho + tht - 1) / tht;
    if (g.A) {
      const int n_img = (int)((int64_t)g.M / ((int64_t)g.Ho * g.Wo));
      rc = make_tmap_conv4d(&p->tmA, g.dtype, g.A, n_img, g.H, g.Wd, g.C, twt, tht, g.stride);
      if (rc) return rc;
    }
  }
  p->ready = 1;
  return SWAPNET_OK;
}

int launch_tc_gemm(const TcGemm& g, const TcPlan& pl, int* err, cudaStream_t s) {
  if (!pl.ready) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "tcgen05 GEMM not prepared");
  if (pl.persist) return launch_tc_persist(g, pl, err, s);
  const bool bf = g.dtype == SWAPNET_BF16;
  if (g.conv && pl.tma_conv) {
    if (pl.bn == 64) return bf ? launch_inst<__nv_bfloat16, 64, kATap>(g, pl, err, s) : launch_inst<__half, 64, kATap>(g, pl, err, s);
    return bf ? launch_inst<__nv_bfloat16, 128, kATap>(g, pl, err, s) : launch_inst<__half, 128, kATap>(g, pl, err, s);
  }
  if (g.conv) {
    if (pl.bn == 64) return bf ? launch_inst<__nv_bfloat16, 64, kAGather>(g, pl, err, s) : launch_inst<__half, 64, kAGather>(g, pl, err, s);
    return bf ? launch_inst<__nv_bfloat16, 128, kAGather>(g, pl, err, s) : launch_inst<__half, 128, kAGather>(g, pl, err, s);
  }
  if (pl.bn == 64) return bf ? launch_inst<__nv_bfloat16, 64, kA2d>(g, pl, err, s) : launch_inst<__half, 64, kA2d>(g, pl, err, s);
  if (pl.bn == 256) return bf ? launch_inst<__nv_bfloat16, 256, kA2d>(g, pl, err, s) : launch_inst<__half, 256, kA2d>(g, pl, err, s);
  return bf ? launch_inst<__nv_bfloat16, 128, kA2d>(g, pl, err, s) : launch_inst<__half, 128, kA2d>(g, pl, err, s);
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

int make_tmap_2d(CUtensorMap* m, int dtype, const void* base, uint64_t inner, uint64_t rows, uint64_t row_stride_bytes,
                 uint32_t box_inner, uint32_t box_rows) {
  auto fn = encode_fn();
  if (!fn) SN_FAIL(SWAPNET_ERR_CUDA, "cuTensorMapEncodeTiled unavailable");
  if (((uintptr_t)base & 15) || (row_stride_bytes & 15) || (box_inner * 2) % 16)
    SN_FAIL(SWAPNET_ERR_MISALIGNED, "TMA operand must be 16-byte aligned with a 16-byte multiple row stride");
  const cuuint64_t dims[2] = {inner, rows};
  const cuuint64_t strides[1] = {row_stride_bytes};
  const cuuint32_t box[2] = {box_inner, box_rows};
  const cuuint32_t estr[2] = {1, 1};
  const CUresult r = fn(m, dtype == SWAPNET_BF16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT16,
                        2, const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) SN_FAIL(SWAPNET_ERR_CUDA, "cuTensorMapEncodeTiled failed (" + std::to_string((int)r) + ")");
  return SWAPNET_OK;
}

int tc_error_word(int** ptr) {
  void* p = nullptr;
  if (cudaGetSymbolAddress(&p, g_tc_err) != cudaSuccess) SN_FAIL(SWAPNET_ERR_CUDA, "cudaGetSymbolAddress failed");
  *ptr = static_cast<int*>(p);
  return SWAPNET_OK;
}

}  // namespace swapnet

extern "C" int swapnet_gemm_noalloc(int32_t dtype, const void* A, const void* W, const void* bias, void* Y,
                                    int32_t M, int32_t N, int32_t K, int32_t act, swapnet_stream stream) {
  return swapnet::guard_abi([&]() -> int {
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
    // W and bias are caller memory that the previous work on the stream (an
    // earlier call, say) may have written: no early start before it completes
    g.no_pdl = 1;
    TcPlan pl;
    int rc = tc_prepare(g, &pl);
    if (rc) return rc;
    if (pl.splits > 1) {  // cluster_max == 0: global split-K scratch
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
  });
}
