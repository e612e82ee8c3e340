// Persistent tcgen05 GEMM / implicit-GEMM convolution for problems with at
// least one 128-row output tile per SM (no split-K):
//
//   C[m, n] = sum_k A[m, k] * B[n, k],  fp16/bf16 in, fp32 accumulate in TMEM
//
// One CTA per SM loops over 128 x BN output tiles; tile t is (m-tile t % mt,
// n-tile t / mt), so the CTAs running together share one weight tile in L2.
// Warp roles:
//   warp 0       TMA producer: the weight tile B of every k-block, and A too
//                for plain GEMMs (linear layers, 1x1 stride-1 convs)
//   warp 1       TMEM owner and MMA issuer (one elected lane)
//   warps 2..5   epilogue: TMEM -> registers -> bias / residual / activation
//                -> global, warp w reading TMEM lanes 32 * (w % 4) .. + 31
//   warps 6..9   (convolutions without whole-tap TMA) implicit im2col gather of
//                A with cp.async
// A-operand modes: kAT2d (row-major A by 2-D TMA), kAGather (cp.async im2col
// gather), kATap (convolution A by one 4-D TMA per k-block: the 64 channels
// of one filter tap at a wt x ht patch of output pixels, the image border
// and the stride handled by the copy engine's zero fill and element stride;
// the output tile is then that patch, rows >= wt * ht unused).
// A ring of shared-memory stages (full / empty mbarriers) feeds the MMAs,
// continuous across tiles.  The accumulator is double-buffered in TMEM
// (2 x BN columns, tfull / tempty mbarriers): the MMAs of the next tile run
// while the epilogue drains the last one.  Every wait is bounded; on timeout
// the kernel records the error, every role leaves its loop, in-flight copies
// and MMAs are drained, and TMEM is freed.
#include <cudaTypedefs.h>

#include <algorithm>
#include <cstring>
#include <type_traits>

#include "device.cuh"
#include "internal.h"
#include "kernels.h"
#include "tc_epi.cuh"

namespace swapnet {

namespace {

constexpr int kPBM = 128;
constexpr int kPBK = 64;  // one 128-byte swizzle row of 16-bit elements
constexpr int kPA = kPBM * kPBK * 2;

// MS: 128-row sub-tiles per tile sharing each weight stage (1, or 2 or 4
// for N tiles of 64, where one 128x64 MMA chain per k16 step is too little
// work per stage): a tile is then MS*128 x BN, MS accumulators side by side
// in TMEM (2 x MS x BN columns with the double buffer: 512 for MS = 4).
template <int BN, int MS> struct PCfg {
  static constexpr int kStages = BN == 256 ? 4 : (BN == 128 ? 6 : (MS == 4 ? 3 : (MS == 2 ? 5 : 8)));
  static constexpr int kLag = kStages - 2;  // gather: cp.async groups in flight per thread
  static constexpr int kB = BN * kPBK * 2;
  static constexpr int kSA = MS * kPA;      // A bytes per stage
  static constexpr int kStageBytes = kStages * (kSA + kB);
  static constexpr int kBias = 2 * 4 * BN * 4;  // [buffer][epilogue warp][BN] fp32
  static constexpr int kSmem = kStageBytes + kBias + 256 + 1024;
  static_assert(kSmem <= 232448, "dynamic shared memory above the 227 KB per-CTA limit");
  static_assert(2 * MS * BN <= 512, "TMEM holds 512 fp32 columns");
};

constexpr int kAT2d = 0, kAGather = 1, kATap = 2;

template <int AMODE> constexpr int persist_threads() { return AMODE == kAGather ? 320 : 192; }

template <typename T, int BN, int AMODE, int MS>
__global__ void __launch_bounds__(persist_threads<AMODE>(), 1)
    tc_persist_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                      const TcArgs p) {
  constexpr bool GATHER = AMODE == kAGather;
  static_assert(MS == 1 || !GATHER, "the gather threads cover one 128-row sub-tile");
  using Cfg = PCfg<BN, MS>;
  constexpr int kStages = Cfg::kStages;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + kStages * Cfg::kSA;
  float* sbias = reinterpret_cast<float*>(smem + Cfg::kStageBytes);  // [2][4][BN]
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + Cfg::kStageBytes + Cfg::kBias);
  // bars: full[kStages], empty[kStages], tfull[2], tempty[2], drain
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * kStages + 5);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  const uint32_t full0 = smem_u32(bars), empty0 = smem_u32(bars + kStages);
  const uint32_t tfull0 = smem_u32(bars + 2 * kStages), tempty0 = smem_u32(bars + 2 * kStages + 2);
  const uint32_t drain_bar = smem_u32(bars + 2 * kStages + 4);
  auto full_bar = [&](int s) { return full0 + 8u * s; };
  auto empty_bar = [&](int s) { return empty0 + 8u * s; };

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // m-tiles: 128-row blocks of the output matrix, or pixel patches (kATap)
  const int hw = p.Ho * p.Wo;
  const int patches = p.tiles_w * p.tiles_h;
  const int mt = AMODE == kATap ? (p.M / hw) * patches : (p.M + kPBM - 1) / kPBM;
  const int nt = (p.N + BN - 1) / BN;
  const uint32_t a_bytes = AMODE == kATap ? (uint32_t)(p.wt * p.ht * 128) : (AMODE == kAT2d ? kPA : 0);
  const int mtp = (mt + MS - 1) / MS;  // tiles along M (MS sub-tiles each)
  const int tiles = mtp * nt;
  const int KB = (p.K + kPBK - 1) / kPBK;
  const int my_tiles = blockIdx.x < tiles ? (tiles - 1 - (int)blockIdx.x) / (int)gridDim.x + 1 : 0;
  const int work = my_tiles * KB;  // (tile, k-block) items of this CTA
  auto tile_of = [&](int lt) { return (int)blockIdx.x + lt * (int)gridDim.x; };

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(full_bar(s), GATHER ? 1 + 128 : 1);
      mbar_init(empty_bar(s), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(tfull0 + 8u * b, 1);
      mbar_init(tempty0 + 8u * b, 4);  // one arrival per epilogue warp
    }
    mbar_init(drain_bar, 1);
    *abort_flag = 0;
    fence_barrier_init();
    fence_proxy_async_smem();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), 2 * MS * BN);
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
  pdl_launch_dependents();

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer.  The weight tiles of the first stages
      // go out before waiting for the previous kernel (they do not depend on it).
      auto coords = [&](int g, int* kx, int* m0, int* n0) {
        const int tile = tile_of(g / KB);
        *kx = (g % KB) * kPBK;
        *m0 = (tile % mtp) * MS * kPBM;
        *n0 = (tile / mtp) * BN;
      };
      auto load_a = [&](int s, int g) {
        const int tile = tile_of(g / KB);
        const int k0 = (g % KB) * kPBK;
#pragma unroll
        for (int sub = 0; sub < MS; ++sub) {
          // a sub-tile past the last one reads only out-of-range coordinates (zero fill)
          const int idx = (tile % mtp) * MS + sub;
          const uint32_t dst = smem_u32(sA + s * Cfg::kSA + sub * kPA);
          if (AMODE == kAT2d) {
            tma_load_2d(dst, &tmA, full_bar(s), k0, idx * kPBM);
          } else if (AMODE == kATap) {
            const int img = idx / patches, rem = idx - img * patches;
            const int th = rem / p.tiles_w, tw = rem - th * p.tiles_w;
            const int tap = k0 / p.C, c0 = k0 - tap * p.C;
            const int ry = tap / p.kw, rx = tap - ry * p.kw;
            tma_load_4d(dst, &tmA, full_bar(s), c0, tw * p.wt * p.stride - p.pad + rx,
                        th * p.ht * p.stride - p.pad + ry, img);
          }
        }
      };
      const int early = min(work, kStages);
      for (int g = 0; g < early; ++g) {
        int kx, m0, n0;
        coords(g, &kx, &m0, &n0);
        mbar_arrive_expect_tx(full_bar(g), Cfg::kB + MS * a_bytes);
        tma_load_2d(smem_u32(sB + g * Cfg::kB), &tmB, full_bar(g), kx, n0);
      }
      pdl_wait();
      if (!GATHER)
        for (int g = 0; g < early; ++g) load_a(g, g);
      // steady state: coordinates advance incrementally (divisions only when
      // a new tile starts), so the single producer thread keeps ahead
      int g = early;
      if (g < work) {
        int lt = g / KB, kb = g % KB;
        int s = g % kStages, par = ((g / kStages) & 1) ^ 1;
        int n0 = 0, ay[MS], az[MS], aw[MS];
        int c0 = 0, rx = 0, ry = 0;
        auto start_tile = [&]() {
          const int tile = tile_of(lt);
          n0 = (tile / mtp) * BN;
#pragma unroll
          for (int sub = 0; sub < MS; ++sub) {
            const int idx = (tile % mtp) * MS + sub;
            if (AMODE == kATap) {
              const int img = idx / patches, rem = idx - img * patches;
              const int th = rem / p.tiles_w, tw = rem - th * p.tiles_w;
              ay[sub] = tw * p.wt * p.stride - p.pad;
              az[sub] = th * p.ht * p.stride - p.pad;
              aw[sub] = img;
            } else {
              ay[sub] = idx * kPBM;
              az[sub] = aw[sub] = 0;
            }
          }
        };
        start_tile();
        if (AMODE == kATap) {  // position of k-block kb inside the filter
          const int k0 = kb * kPBK, tap = k0 / p.C;
          c0 = k0 - tap * p.C;
          ry = tap / p.kw;
          rx = tap - ry * p.kw;
        }
        for (; g < work; ++g) {
          if (!mbar_wait_bounded(empty_bar(s), par, abort_flag, p.err)) break;
          mbar_arrive_expect_tx(full_bar(s), Cfg::kB + MS * a_bytes);
          tma_load_2d(smem_u32(sB + s * Cfg::kB), &tmB, full_bar(s), kb * kPBK, n0);
          if (!GATHER) {
#pragma unroll
            for (int sub = 0; sub < MS; ++sub) {
              const uint32_t dst = smem_u32(sA + s * Cfg::kSA + sub * kPA);
              if (AMODE == kAT2d) tma_load_2d(dst, &tmA, full_bar(s), kb * kPBK, ay[sub]);
              else tma_load_4d(dst, &tmA, full_bar(s), c0, ay[sub] + rx, az[sub] + ry, aw[sub]);
            }
          }
          if (++s == kStages) { s = 0; par ^= 1; }
          if (++kb == KB) {
            kb = 0;
            c0 = rx = ry = 0;
            if (++lt < my_tiles) start_tile();
          } else if (AMODE == kATap) {
            c0 += kPBK;
            if (c0 == p.C) {
              c0 = 0;
              if (++rx == p.kw) { rx = 0; ++ry; }
            }
          }
        }
      }
      if (g < work) {
        // aborted: let the loads already issued land before the CTA exits
        volatile int no_abort = 0;
        for (int j = (g > kStages ? g - kStages : 0); j < g; ++j)
          mbar_wait_bounded(full_bar(j % kStages), (j / kStages) & 1, &no_abort, nullptr);
      }
    } else {
      pdl_wait();
    }
  } else if (warp == 1) {
    pdl_wait();
    if (lane == 0) {
      // ---------------- MMA issuer
      constexpr uint32_t idesc = idesc_f16(std::is_same<T, __nv_bfloat16>::value ? 1 : 0, kPBM, BN);
      int g = 0;
      bool ok = true;
      for (int lt = 0; lt < my_tiles && ok; ++lt) {
        const int buf = lt & 1, use = lt >> 1;
        if (!mbar_wait_bounded(tempty0 + 8u * buf, (use & 1) ^ 1, abort_flag, p.err)) break;
        tc_fence_after();
        const uint32_t d = tmem + (uint32_t)(buf * MS * BN);
        for (int kb = 0; kb < KB; ++kb, ++g) {
          const int s = g % kStages, r = g / kStages;
          if (!mbar_wait_bounded(full_bar(s), r & 1, abort_flag, p.err)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t bd = smem_desc_sw128(smem_u32(sB + s * Cfg::kB));
#pragma unroll
          for (int sub = 0; sub < MS; ++sub) {
            const uint64_t ad = smem_desc_sw128(smem_u32(sA + s * Cfg::kSA + sub * kPA));
#pragma unroll
            for (int k = 0; k < kPBK / 16; ++k)
              tc_mma_f16(d + (uint32_t)(sub * BN), ad + 2ull * k, bd + 2ull * k, idesc, (kb | k) != 0);
          }
          tc_commit(empty_bar(s));
        }
        if (ok) tc_commit(tfull0 + 8u * buf);
      }
      // every MMA issued above has completed once this arrives
      tc_commit(drain_bar);
      volatile int no_abort = 0;
      mbar_wait_bounded(drain_bar, 0, &no_abort, p.err);
    }
  } else if (warp < 6) {
    // ---------------- epilogue
    pdl_wait();
    const int q = warp & 3;
    const int row = q * 32 + lane;
    for (int lt = 0; lt < my_tiles; ++lt) {
      const int buf = lt & 1, use = lt >> 1;
      const int tile = tile_of(lt);
      const int n0 = (tile / mtp) * BN;
      // each warp stages its own copy of the tile's bias: no cross-warp barrier
      float* sb = sbias + (buf * 4 + q) * BN;
      const T* bias = static_cast<const T*>(p.e.bias);
      for (int j = lane; j < BN; j += 32) sb[j] = (bias && n0 + j < p.N) ? to_f<T>(bias[n0 + j]) : 0.f;
      __syncwarp();
      // output row of this thread's TMEM lane in sub-tile sub, -1 when unused
      auto row_of = [&](int sub) {
        const int idx = (tile % mtp) * MS + sub;  // m-tile (or pixel patch) of this sub-tile
        int m = -1;
        if (idx < mt) {
          if (AMODE == kATap) {
            const int img = idx / patches, rem = idx - img * patches;
            const int th = rem / p.tiles_w, tw = rem - th * p.tiles_w;
            if (row < p.wt * p.ht) {
              const int oy = th * p.ht + row / p.wt, ox = tw * p.wt + row % p.wt;
              if (oy < p.Ho && ox < p.Wo) m = (img * p.Ho + oy) * p.Wo + ox;
            }
          } else {
            m = idx * kPBM + row;
            if (m >= p.M) m = -1;
          }
        }
        return m;
      };
      const bool vec_ok = ((p.ldy | n0) % 8 == 0) && (!p.e.res || ((p.e.ldr | n0) % 8 == 0));
      // the residual of the first 32 columns is requested while the
      // accumulator is still being computed, each later chunk's one chunk
      // ahead of its use.  The same loop serves layers without a residual
      // (zeros): skipping it for them measured slower on whole networks
      // (YOLOv3 resident 0.742 -> 0.788 ms, ResNet-50 0.330 -> 0.345 ms)
      const bool has_res = true;
      uint4 rnext[4];
      if (has_res) res_prefetch32<T>(rnext, p, row_of(0), n0, vec_ok);
      const bool got = mbar_wait_bounded(tfull0 + 8u * buf, use & 1, abort_flag, p.err);
      if (!__all_sync(0xffffffffu, got)) break;  // tcgen05.ld is warp-collective
      tc_fence_after();
#pragma unroll 1
      for (int sub = 0; sub < MS; ++sub) {
        const int m = row_of(sub);
#pragma unroll 1
        for (int c0 = 0; c0 < BN; c0 += 32) {
          uint4 rcur[4];
          if (has_res) {
#pragma unroll
            for (int i = 0; i < 4; ++i) rcur[i] = rnext[i];
            if (c0 + 32 < BN) res_prefetch32<T>(rnext, p, m, n0 + c0 + 32, vec_ok);
            else if (sub + 1 < MS) res_prefetch32<T>(rnext, p, row_of(sub + 1), n0, vec_ok);
          }
          uint32_t r[32];
          tmem_ld_32x32b_x32(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)((buf * MS + sub) * BN + c0), r);
          tmem_ld_wait();
          if (m >= 0 && n0 + c0 < p.N) {
            float v[32];
#pragma unroll
            for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(r[j]);
            if (has_res) finish32r<T>(v, sb + c0, p, m, n0 + c0, vec_ok, rcur);
            else finish32<T>(v, sb + c0, p, m, n0 + c0, vec_ok);
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(tempty0 + 8u * buf);
    }
  } else if (GATHER) {
    // ---------------- implicit im2col gather of A (row t of every tile)
    pdl_wait();
    const int t = threadIdx.x - 192;  // 0..127
    const uint32_t row_off = (uint32_t)((t >> 3) * 1024 + (t & 7) * 128);
    const uint32_t sw = (uint32_t)(t & 7);
    const bool whole_tap = (p.C % kPBK) == 0;  // a 64-wide k-block never straddles taps
    constexpr int kLag = Cfg::kLag;
    int g = 0;
    bool ok = true;
    for (int lt = 0; lt < my_tiles && ok; ++lt) {
      const int tile = tile_of(lt);
      const int m = (tile % mtp) * kPBM + t;  // MS == 1 here
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
      int k = 0, c = 0, ry = 0, rx = 0;
      for (int kb = 0; kb < KB; ++kb, ++g) {
        const int s = g % kStages, r = g / kStages;
        if (!mbar_wait_bounded(empty_bar(s), (r & 1) ^ 1, abort_flag, p.err)) {
          ok = false;
          break;
        }
        const uint32_t dst_row = smem_u32(sA + s * kPA) + row_off;
        if (whole_tap) {
          const int iy = iy0 + ry, ix = ix0 + rx;
          const bool valid = mvalid && k < p.K && (unsigned)iy < (unsigned)p.H && (unsigned)ix < (unsigned)p.Wd;
          const T* src = valid ? xb + ((int64_t)iy * p.Wd + ix) * p.C + c : static_cast<const T*>(p.x);
#pragma unroll
          for (int j = 0; j < 8; ++j) cp_async_16(dst_row + (((uint32_t)j ^ sw) << 4), src + (valid ? 8 * j : 0), valid);
          k += kPBK;
          c += kPBK;
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
        if (g >= kLag) {
          cp_async_wait<kLag>();
          fence_proxy_async_smem();
          mbar_arrive(full_bar((g - kLag) % kStages));
        }
      }
    }
    cp_async_wait<0>();
    fence_proxy_async_smem();
    for (int j = (g > kLag ? g - kLag : 0); j < g; ++j) mbar_arrive(full_bar(j % kStages));
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 2 * MS * BN);
  }
}

template <typename T, int BN, int AMODE, int MS>
int launch_persist_inst(const TcGemm& g, const TcPlan& pl, int* err, cudaStream_t s) {
  static std::atomic<uint64_t> attr_done{0};  // per instantiation, one bit per device
  auto kern = tc_persist_kernel<T, BN, AMODE, MS>;
  if (attr_needed(attr_done)) {
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, PCfg<BN, MS>::kSmem) != cudaSuccess)
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
  a.wt = pl.wt; a.ht = pl.ht; a.tiles_w = pl.tiles_w; a.tiles_h = pl.tiles_h;
  const int64_t mt = AMODE == kATap ? (int64_t)g.M / ((int64_t)g.Ho * g.Wo) * pl.tiles_w * pl.tiles_h
                                    : (g.M + kPBM - 1) / kPBM;
  const int64_t tiles = (mt + MS - 1) / MS * ((g.N + BN - 1) / BN);
  const int sms = g.num_sms > 0 ? g.num_sms : 148;
  cudaLaunchConfig_t cfg;
  std::memset(&cfg, 0, sizeof(cfg));
  cfg.gridDim = dim3((unsigned)std::min<int64_t>(tiles, sms));
  cfg.blockDim = dim3(persist_threads<AMODE>());
  cfg.dynamicSmemBytes = PCfg<BN, MS>::kSmem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = g.no_pdl ? 0 : 1;
  const cudaError_t le = cudaLaunchKernelEx(&cfg, kern, pl.tmA, pl.tmB, a);
  if (le != cudaSuccess) SN_FAIL(SWAPNET_ERR_CUDA, std::string("persistent GEMM launch: ") + cudaGetErrorString(le));
  return SWAPNET_OK;
}

template <typename T, int BN>
int launch_persist_bn(const TcGemm& g, const TcPlan& pl, int* err, cudaStream_t s) {
  if constexpr (BN == 64) {  // sub-tiles only with N tiles of 64
    if (pl.msub == 4) {
      if (!g.conv) return launch_persist_inst<T, BN, kAT2d, 4>(g, pl, err, s);
      if (pl.tma_conv) return launch_persist_inst<T, BN, kATap, 4>(g, pl, err, s);
      SN_FAIL(SWAPNET_ERR_INVALID_ARG, "persistent GEMM: four sub-tiles need A by TMA");
    }
    if (pl.msub == 2) {
      if (!g.conv) return launch_persist_inst<T, BN, kAT2d, 2>(g, pl, err, s);
      if (pl.tma_conv) return launch_persist_inst<T, BN, kATap, 2>(g, pl, err, s);
      SN_FAIL(SWAPNET_ERR_INVALID_ARG, "persistent GEMM: two sub-tiles need A by TMA");
    }
  }
  if (pl.msub != 1) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "persistent GEMM: sub-tiles need N tiles of 64");
  if (!g.conv) return launch_persist_inst<T, BN, kAT2d, 1>(g, pl, err, s);
  if (pl.tma_conv) return launch_persist_inst<T, BN, kATap, 1>(g, pl, err, s);
  return launch_persist_inst<T, BN, kAGather, 1>(g, pl, err, s);
}

template <typename T>
int launch_persist_t(const TcGemm& g, const TcPlan& pl, int* err, cudaStream_t s) {
  switch (pl.bn) {
    case 64: return launch_persist_bn<T, 64>(g, pl, err, s);
    case 128: return launch_persist_bn<T, 128>(g, pl, err, s);
    case 256: return launch_persist_bn<T, 256>(g, pl, err, s);
    default: SN_FAIL(SWAPNET_ERR_INVALID_ARG, "persistent GEMM: bad N tile");
  }
}

}  // namespace

int launch_tc_persist(const TcGemm& g, const TcPlan& pl, int* err, cudaStream_t s) {
  if (g.dtype == SWAPNET_BF16) return launch_persist_t<__nv_bfloat16>(g, pl, err, s);
  return launch_persist_t<__half>(g, pl, err, s);
}

}  // namespace swapnet
