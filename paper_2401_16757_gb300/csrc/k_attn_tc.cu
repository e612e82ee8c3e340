// Causal attention of a long query run (the decoder prefill) on the tcgen05
// tensor cores, for head width 128 (fp16 / bf16 storage, fp32 arithmetic).
//
// Per head h, query t (position pos0 + t) attends to cache positions
// 0 .. pos0 + t:  out[t] = sum_j softmax_j(q_t . k_j / sqrt(128)) v_j.  Both
// contractions are dense and run on the tensor cores; the softmax is exact,
// computed online over key tiles in fp32.
//
// One CTA owns 128 queries of one head.  For each tile of 128 keys:
//   S = Q K^T   tcgen05.mma kind::f16, M 128 (queries) x N 128 (keys) x K 128
//               (head dims); Q and the key tile by TMA (128-byte swizzle,
//               K-major), S in TMEM columns [0, 128)
//   P           warps 2..5, one query row per thread: the row of S from TMEM,
//               causal mask, running max m and denominator l, p = e^(s - m)
//               written to shared memory as two bf16/fp16 parts p_hi + p_lo
//               (p_lo = round(p - p_hi)), so the product with V keeps about
//               16 significant bits of p instead of 8
//   O_t = P V   tcgen05.mma, M 128 x N 128 x K 16 steps for each part; V
//               is the value tile as loaded by TMA (two 64-dim boxes),
//               [keys][dims] with the dims contiguous, i.e. the B operand in
//               MN-major layout; O_t in TMEM columns [128, 256)
//   O           the softmax warps keep the row's 128 outputs in registers:
//               O = O * e^(m_old - m_new) + O_t
// and at the end write O / l.  Warp 0 issues the TMA loads (key and value
// tiles double-buffered), warp 1 owns TMEM and issues the MMAs.  Every wait
// is bounded: on timeout the kernel records kDevErrTimeout, drains the loads
// and MMAs it started, frees TMEM and returns.
#include <cudaTypedefs.h>

#include <cstring>
#include <type_traits>

#include "device.cuh"
#include "internal.h"
#include "kernels.h"

namespace swapnet {

namespace {

constexpr int kAQ = 128;        // queries per CTA (MMA M)
constexpr int kAK = 128;        // keys per tile
constexpr int kAD = 128;        // head width
constexpr int kAThreads = 192;  // warp 0 TMA, warp 1 MMA, warps 2..5 softmax
constexpr int kHalf = 128 * 64 * 2;  // one 128-row x 64-column swizzled half tile (16 KB)
constexpr int kTile = 2 * kHalf;     // 128 x 128 elements
// shared memory: Q | K stage 0, 1 | V stage 0, 1 | P_hi | P_lo | barriers
constexpr int kOffQ = 0;
constexpr int kOffK = kOffQ + kTile;
constexpr int kOffV = kOffK + 2 * kTile;
constexpr int kOffPh = kOffV + 2 * kTile;
constexpr int kOffPl = kOffPh + kTile;
constexpr int kOffBar = kOffPl + kTile;
constexpr int kASmem = kOffBar + 128 + 1024;  // + barriers, TMEM slot, flags; + alignment slack
static_assert(kASmem <= 232448, "attention tile set exceeds the shared memory of a CTA");
constexpr uint32_t kTmemCols = 256;  // S: [0, 128), O_t: [128, 256)

// Shared-memory descriptor of a B operand stored MN-major with the 128-byte
// swizzle (the layout TMA gives a [K rows][64 N] box): 8-row K groups are
// 1024 bytes apart (stride byte offset); the two 64-column N blocks of the
// value tile (the two TMA boxes) are kHalf bytes apart (leading byte
// offset), so one N = 128 MMA covers all head dims.
__device__ __forceinline__ uint64_t smem_desc_sw128_mn(uint32_t addr) {
  uint64_t d = 0;
  d |= (uint64_t)((addr & 0x3FFFFu) >> 4);
  d |= (uint64_t)(kHalf >> 4) << 16;
  d |= (uint64_t)(1024 >> 4) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
}

struct AttnArgs {
  void* out;
  const int* pos_ptr;
  int tokens, heads, width, max_seq;
  float scale_log2;  // log2(e) / sqrt(head width)
  int* err;
};

template <typename T>
__device__ __forceinline__ uint32_t pack2(float a, float b) {
  const T x = from_f<T>(a), y = from_f<T>(b);
  return (uint32_t)(*reinterpret_cast<const uint16_t*>(&x)) |
         ((uint32_t)(*reinterpret_cast<const uint16_t*>(&y)) << 16);
}

template <typename T>
__global__ void __launch_bounds__(kAThreads, 1)
    attention_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                        const __grid_constant__ CUtensorMap tmV, const AttnArgs p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kOffBar);
  const uint32_t q_full = smem_u32(bars + 0);
  auto kv_full = [&](int s) { return smem_u32(bars + 1 + s); };
  auto kv_empty = [&](int s) { return smem_u32(bars + 3 + s); };
  const uint32_t s_full = smem_u32(bars + 5);
  const uint32_t p_full = smem_u32(bars + 6);
  const uint32_t o_full = smem_u32(bars + 7);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 8);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(bars + 9);
  const uint32_t done_bar = smem_u32(bars + 10);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int t0 = blockIdx.x * kAQ, h = blockIdx.y;
  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int s = 0; s < 2; ++s) {
      mbar_init(kv_full(s), 1);
      mbar_init(kv_empty(s), 1);
    }
    mbar_init(s_full, 1);
    mbar_init(p_full, 128);
    mbar_init(o_full, 1);
    mbar_init(done_bar, 1);
    *abort_flag = 0;
    fence_barrier_init();
    prefetch_tmap(&tmQ);
    prefetch_tmap(&tmK);
    prefetch_tmap(&tmV);
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t tS = tmem, tO = tmem + 128;
  // q, the caches and the position are written by the kernel before
  pdl_wait();
  pdl_launch_dependents();
  const int pos0 = *p.pos_ptr;
  const int last_q = min(t0 + kAQ, p.tokens) - 1;
  const int n_keys = max(0, min(pos0 + last_q + 1, p.max_seq));
  const int nkt = (n_keys + kAK - 1) / kAK;
  const int col0 = h * kAD;

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer
      mbar_arrive_expect_tx(q_full, kTile);
      tma_load_2d(smem_u32(smem + kOffQ), &tmQ, q_full, col0, t0);
      tma_load_2d(smem_u32(smem + kOffQ + kHalf), &tmQ, q_full, col0 + 64, t0);
      int kt = 0;
      for (; kt < nkt; ++kt) {
        const int s = kt & 1;
        if (kt >= 2 && !mbar_wait_bounded(kv_empty(s), ((kt >> 1) - 1) & 1, abort_flag, p.err)) break;
        mbar_arrive_expect_tx(kv_full(s), 2 * kTile);
        const uint32_t ks = smem_u32(smem + kOffK + s * kTile), vs = smem_u32(smem + kOffV + s * kTile);
        tma_load_2d(ks, &tmK, kv_full(s), col0, kt * kAK);
        tma_load_2d(ks + kHalf, &tmK, kv_full(s), col0 + 64, kt * kAK);
        tma_load_2d(vs, &tmV, kv_full(s), col0, kt * kAK);
        tma_load_2d(vs + kHalf, &tmV, kv_full(s), col0 + 64, kt * kAK);
      }
      // let every load issued land before the CTA can exit
      volatile int no_abort = 0;
      mbar_wait_bounded(q_full, 0, &no_abort, nullptr);
      for (int j = (kt > 2 ? kt - 2 : 0); j < kt; ++j)
        mbar_wait_bounded(kv_full(j & 1), (j >> 1) & 1, &no_abort, nullptr);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer
      constexpr int bf = std::is_same<T, __nv_bfloat16>::value ? 1 : 0;
      constexpr uint32_t idesc_s = idesc_f16(bf, kAQ, kAK);
      constexpr uint32_t idesc_pv = idesc_f16(bf, kAQ, kAD) | (1u << 16);  // B (values) MN-major, N = 128
      bool ok = mbar_wait_bounded(q_full, 0, abort_flag, p.err);
      for (int kt = 0; ok && kt < nkt; ++kt) {
        const int s = kt & 1;
        if (!mbar_wait_bounded(kv_full(s), (kt >> 1) & 1, abort_flag, p.err)) break;
        tc_fence_after();
        const uint32_t qa = smem_u32(smem + kOffQ), ka = smem_u32(smem + kOffK + s * kTile);
#pragma unroll
        for (int kb = 0; kb < 2; ++kb)
#pragma unroll
          for (int k = 0; k < 4; ++k)
            tc_mma_f16(tS, smem_desc_sw128(qa + kb * kHalf) + 2ull * k, smem_desc_sw128(ka + kb * kHalf) + 2ull * k,
                       idesc_s, (kb | k) != 0);
        tc_commit(s_full);
        if (!mbar_wait_bounded(p_full, kt & 1, abort_flag, p.err)) break;
        tc_fence_after();
        const uint32_t va = smem_u32(smem + kOffV + s * kTile);
#pragma unroll
        for (int part = 0; part < 2; ++part) {
          const uint32_t pa = smem_u32(smem + (part ? kOffPl : kOffPh));
#pragma unroll
          for (int ks = 0; ks < 8; ++ks)  // 16 keys per step, all 128 head dims (both 64-wide halves)
            tc_mma_f16(tO, smem_desc_sw128(pa + (ks >> 2) * kHalf) + 2ull * (ks & 3),
                       smem_desc_sw128_mn(va + ks * 2048), idesc_pv, (part | ks) != 0);
        }
        tc_commit(o_full);
        tc_commit(kv_empty(s));
      }
      // every MMA issued must have finished before TMEM is freed (on the
      // normal path the softmax warps have already waited for the last one)
      tc_commit(done_bar);
      volatile int no_abort = 0;
      mbar_wait_bounded(done_bar, 0, &no_abort, nullptr);
    }
  } else {
    // ---------------- softmax and output: warps 2..5, query row per thread
    const int q4 = warp & 3;
    const int row = q4 * 32 + lane;
    const int tq = t0 + row;
    // last visible key: padding rows reuse the last query's horizon; never
    // past the cache (a position beyond it is reported by the RoPE kernel)
    const int qpos = min(pos0 + min(tq, p.tokens - 1), p.max_seq - 1);
    const uint32_t lane_off = (uint32_t)(q4 * 32) << 16;
    const uint32_t prow = (uint32_t)((row >> 3) * 1024 + (row & 7) * 128);
    const uint32_t psw = (uint32_t)(row & 7);
    float m = -INFINITY, l = 0.f;
    float o[kAD];
#pragma unroll
    for (int d = 0; d < kAD; ++d) o[d] = 0.f;
    bool ok = true;
    for (int kt = 0; kt < nkt; ++kt) {
      if (!mbar_wait_bounded(s_full, kt & 1, abort_flag, p.err)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const int kbase = kt * kAK;
      // pass 1: the row maximum over this tile's visible keys
      float mx = m;
#pragma unroll 1
      for (int c0 = 0; c0 < kAK; c0 += 32) {
        uint32_t r[32];
        tmem_ld_32x32b_x32(tS + lane_off + (uint32_t)c0, r);
        tmem_ld_wait();
#pragma unroll
        for (int i = 0; i < 32; ++i)
          if (kbase + c0 + i <= qpos) mx = fmaxf(mx, __uint_as_float(r[i]));
      }
      const float alpha = exp2f((m - mx) * p.scale_log2);  // 0 on the first tile (m = -inf)
      // pass 2: p = e^(s - mx), split into two parts, to shared memory
      float lt = 0.f;
#pragma unroll 1
      for (int c0 = 0; c0 < kAK; c0 += 32) {
        uint32_t r[32];
        tmem_ld_32x32b_x32(tS + lane_off + (uint32_t)c0, r);
        tmem_ld_wait();
        uint32_t hi[16], lo[16];
#pragma unroll
        for (int i = 0; i < 32; i += 2) {
          float pv[2];
#pragma unroll
          for (int u = 0; u < 2; ++u) {
            const bool vis = kbase + c0 + i + u <= qpos;
            pv[u] = vis ? exp2f((__uint_as_float(r[i + u]) - mx) * p.scale_log2) : 0.f;
            lt += pv[u];
          }
          const T h0 = from_f<T>(pv[0]), h1 = from_f<T>(pv[1]);
          hi[i / 2] = (uint32_t)(*reinterpret_cast<const uint16_t*>(&h0)) |
                      ((uint32_t)(*reinterpret_cast<const uint16_t*>(&h1)) << 16);
          lo[i / 2] = pack2<T>(pv[0] - to_f<T>(h0), pv[1] - to_f<T>(h1));
        }
        // keys c0..c0+31 of the row: k-block c0 / 64, 16-byte chunks (c0 % 64) / 8 + 0..3
        const uint32_t kb = (uint32_t)(c0 >> 6), ch0 = (uint32_t)((c0 & 63) >> 3);
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          const uint32_t off = kb * kHalf + prow + (((ch0 + c) ^ psw) << 4);
          asm volatile("st.shared.v4.b32 [%0], {%1,%2,%3,%4};" ::"r"(smem_u32(smem + kOffPh) + off), "r"(hi[4 * c]),
                       "r"(hi[4 * c + 1]), "r"(hi[4 * c + 2]), "r"(hi[4 * c + 3])
                       : "memory");
          asm volatile("st.shared.v4.b32 [%0], {%1,%2,%3,%4};" ::"r"(smem_u32(smem + kOffPl) + off), "r"(lo[4 * c]),
                       "r"(lo[4 * c + 1]), "r"(lo[4 * c + 2]), "r"(lo[4 * c + 3])
                       : "memory");
        }
      }
      l = l * alpha + lt;
      m = mx;
      fence_proxy_async_smem();  // P is read by the tensor cores (async proxy)
      tc_fence_before();
      mbar_arrive(p_full);
      if (!mbar_wait_bounded(o_full, kt & 1, abort_flag, p.err)) {
        ok = false;
        break;
      }
      tc_fence_after();
#pragma unroll
      for (int c0 = 0; c0 < kAD; c0 += 32) {
        uint32_t r[32];
        tmem_ld_32x32b_x32(tO + lane_off + (uint32_t)c0, r);
        tmem_ld_wait();
#pragma unroll
        for (int i = 0; i < 32; ++i) o[c0 + i] = fmaf(o[c0 + i], alpha, __uint_as_float(r[i]));
      }
      tc_fence_before();
    }
    if (ok && tq < p.tokens && nkt > 0) {
      const float inv = 1.0f / l;
      uint4* dst = reinterpret_cast<uint4*>(static_cast<T*>(p.out) + (int64_t)tq * p.width + col0);
#pragma unroll
      for (int c = 0; c < kAD / 8; ++c) {
        uint4 v;
        v.x = pack2<T>(o[8 * c] * inv, o[8 * c + 1] * inv);
        v.y = pack2<T>(o[8 * c + 2] * inv, o[8 * c + 3] * inv);
        v.z = pack2<T>(o[8 * c + 4] * inv, o[8 * c + 5] * inv);
        v.w = pack2<T>(o[8 * c + 6] * inv, o[8 * c + 7] * inv);
        dst[c] = v;
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

int done(cudaError_t e, const char* what) {
  if (e == cudaSuccess) e = cudaGetLastError();
  if (e != cudaSuccess) SN_FAIL(SWAPNET_ERR_CUDA, std::string(what) + ": " + cudaGetErrorString(e));
  return SWAPNET_OK;
}

template <typename T>
int launch_t(const void* q, const void* kc, const void* vc, const int* pos_ptr, int tokens, int heads, int width,
             int max_seq, void* out, int* err, cudaStream_t s) {
  static std::atomic<uint64_t> attr_done{0};
  auto kern = attention_tc_kernel<T>;
  if (attr_needed(attr_done)) {
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kASmem) != cudaSuccess)
      return done(cudaGetLastError(), "attention shared memory");
    attr_set(attr_done);
  }
  const int dt = std::is_same<T, __nv_bfloat16>::value ? SWAPNET_BF16 : SWAPNET_F16;
  CUtensorMap tq, tk, tv;
  int rc = make_tmap_2d(&tq, dt, q, (uint64_t)width, (uint64_t)tokens, (uint64_t)width * 2, 64, kAQ);
  if (!rc) rc = make_tmap_2d(&tk, dt, kc, (uint64_t)width, (uint64_t)max_seq, (uint64_t)width * 2, 64, kAK);
  if (!rc) rc = make_tmap_2d(&tv, dt, vc, (uint64_t)width, (uint64_t)max_seq, (uint64_t)width * 2, 64, kAK);
  if (rc) return rc;
  AttnArgs a;
  std::memset(&a, 0, sizeof(a));
  a.out = out;
  a.pos_ptr = pos_ptr;
  a.tokens = tokens;
  a.heads = heads;
  a.width = width;
  a.max_seq = max_seq;
  a.scale_log2 = 1.4426950408889634f / sqrtf((float)kAD);
  a.err = err;
  cudaLaunchConfig_t cfg;
  std::memset(&cfg, 0, sizeof(cfg));
  cfg.gridDim = dim3((tokens + kAQ - 1) / kAQ, heads);
  cfg.blockDim = dim3(kAThreads);
  cfg.dynamicSmemBytes = kASmem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return done(cudaLaunchKernelEx(&cfg, kern, tq, tk, tv, a), "tensor-core attention launch");
}

}  // namespace

bool attention_tc_supported(int dtype, int tokens, int heads, int width) {
  return (dtype == SWAPNET_F16 || dtype == SWAPNET_BF16) && heads > 0 && width == heads * kAD && tokens >= 64;
}

int launch_attention_tc(int dtype, const void* q, const void* kc, const void* vc, const int* pos_ptr, int tokens,
                        int heads, int width, int max_seq, void* out, int* err, cudaStream_t s) {
  if (!attention_tc_supported(dtype, tokens, heads, width))
    SN_FAIL(SWAPNET_ERR_UNSUPPORTED, "tensor-core attention: fp16/bf16, head width 128, at least 64 queries");
  if (((uintptr_t)q | (uintptr_t)kc | (uintptr_t)vc | (uintptr_t)out) & 15)
    SN_FAIL(SWAPNET_ERR_MISALIGNED, "tensor-core attention: operands must be 16-byte aligned");
  if (dtype == SWAPNET_BF16)
    return launch_t<__nv_bfloat16>(q, kc, vc, pos_ptr, tokens, heads, width, max_seq, out, err, s);
  return launch_t<__half>(q, kc, vc, pos_ptr, tokens, heads, width, max_seq, out, err, s);
}

}  // namespace swapnet
