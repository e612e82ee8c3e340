// Host-side launchers of the layer and swap kernels (internal interface).
// Every launcher validates what its kernel assumes (alignment, sizes) and
// returns a swapnet_status; it never synchronises.
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>
#include <atomic>
#include <cstdint>

namespace swapnet {

// Kernel attributes (dynamic shared memory size, cluster permissions) are
// set per function and per device.  A launcher keeps one bit per device in
// `done`: attr_needed() says whether the current device still lacks the
// attribute, attr_set() records it once cudaFuncSetAttribute succeeded.
// Two threads racing on a first launch may both set it, which is harmless.
inline uint64_t device_bit() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
    cudaGetLastError();
    return 0;  // unknown device: always set the attribute
  }
  return 1ull << dev;
}
// The current device's index for per-device caches (static arrays of 64),
// or -1 when it is unknown or beyond them (then nothing is cached).
inline int device_index() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
    cudaGetLastError();
    return -1;
  }
  return dev;
}
inline bool attr_needed(const std::atomic<uint64_t>& done) {
  const uint64_t b = device_bit();
  return b == 0 || (done.load(std::memory_order_acquire) & b) == 0;
}
inline void attr_set(std::atomic<uint64_t>& done) { done.fetch_or(device_bit(), std::memory_order_acq_rel); }

// Epilogue operands shared by linear and conv layers.
struct Epi {
  const void* bias;  // [n] (a piece's own slice for split linear layers)
  const void* res;   // residual, row stride ldr elements, or nullptr
  int64_t ldr;
  int act;
  int res_post;
};

// y[m, col0 + o] (row stride ldy) = epi(sum_k x[m,k] W[o,k]) for o < N,
// M <= 16.  fp32 / fp16 / bf16; fixed-order reduction (deterministic).
int launch_linear_skinny(int dtype, const void* x, int M, int K, const void* W, int N, const Epi& e, void* y,
                         int64_t ldy, cudaStream_t s, int device_weights = 0, int num_sms = 0,
                         int* err = nullptr);

// Several skinny linear layers reading the same x (M rows, K columns) in one
// launch: segment i computes y_i[m, o] = epi_i(sum_k x[m,k] W_i[o,k]) for
// o < N_i.  pair = 1 (two segments of equal N): segment 1's residual is
// segment 0's stored output (its own res is ignored).  Bit-identical to
// launching the segments one by one.
constexpr int kSkMaxSeg = 3;
struct SkSeg {
  const void* W;
  Epi e;
  int N;
  void* y;
  int64_t ldy;
};
struct SkJob {
  const void* x;
  int M, K;
  int nseg, pair;
  SkSeg seg[kSkMaxSeg];
  // weights in device memory (an arena slot or a resident arena): the
  // rows may be streamed into shared memory by bulk copies; 0 for weights
  // read in place in mapped host memory (plain loads only)
  int device_weights;
  int num_sms;  // grid of the streamed kernel (0: plain-load kernel)
  int* err;     // device error word for the streamed kernel's bounded waits
};
int launch_linear_skinny_job(int dtype, const SkJob& j, cudaStream_t s);

// General tiled SIMT linear (any M, K, N): the fallback when neither the
// tensor-core nor the skinny kernel applies.
int launch_linear_tiled(int dtype, const void* x, int M, int K, const void* W, int N, const Epi& e, void* y,
                        int64_t ldy, cudaStream_t s);

// Direct convolution (SIMT) for any channel count; NHWC in, NHWC out.
int launch_conv_direct(int dtype, const void* x, int n, int h, int w, int cin, const void* W, int cout, int kh,
                       int kw, int stride, int pad, int oh, int ow, const Epi& e, void* y, cudaStream_t s);

int launch_maxpool(int dtype, const void* x, int n, int h, int w, int c, int kh, int kw, int stride, int pad,
                   int oh, int ow, void* y, cudaStream_t s);
int launch_gap(int dtype, const void* x, int n, int h, int w, int c, void* y, cudaStream_t s);
int launch_upsample2x(int dtype, const void* x, int n, int h, int w, int c, void* y, cudaStream_t s);
int launch_concat(int dtype, const void* a, int ca, const void* b, int cb, int64_t pixels, void* y,
                  cudaStream_t s);

// Decoder kernels (fp16 / bf16).  The embedding table pointer is the device
// alias of the page-locked host table.  The attention launcher runs the RoPE
// + cache-append kernel (q rotated in place) and then the attention kernel;
// pos_ptr is the device-side position of the decoder state.
int launch_embed(int dtype, const void* table, const int* ids, int tokens, int vocab, int d, void* out, int* err,
                 cudaStream_t s);
int launch_rmsnorm(int dtype, const void* x, const void* g, int rows, int d, float eps, void* y, cudaStream_t s);
int launch_attention(int dtype, void* q, const void* k, const void* v, void* kc, void* vc, const int* pos_ptr,
                     int tokens, int heads, int width, float theta, int max_seq, void* out, int* err,
                     cudaStream_t s);
int launch_argmax(int dtype, const void* x, int rows, int n, int* out, cudaStream_t s);
int launch_advance(int* pos_ptr, int n, cudaStream_t s);

// Zero-copy swap: copy segments from mapped host memory (device aliases)
// into the arena with 16-byte vector loads/stores.
struct ZcSeg {
  const void* src;  // device alias of page-locked host memory, 16-byte aligned
  void* dst;        // arena, 16-byte aligned
  uint64_t bytes;
};
int launch_zerocopy(const ZcSeg* segs, int nseg, int ctas, cudaStream_t s);

// tcgen05 GEMM / implicit-GEMM convolution (fp16 or bf16, fp32 accumulate).
struct TcGemm {
  int dtype;          // SWAPNET_F16 or SWAPNET_BF16
  int M, N, K;
  // B operand: weights [N][K] row-major (K contiguous)
  const void* W;
  // A operand: either a row-major [M][K] matrix (conv == 0) ...
  const void* A;
  int64_t lda;
  // ... or the implicit im2col of an NHWC input (conv == 1)
  int conv;
  int H, Wd, C, Ho, Wo, kh, kw, stride, pad;
  Epi e;
  void* y;
  int64_t ldy;
  int num_sms;          // used by tc_prepare to size the grid
  int allow_persist;    // 1: problems with a tile per SM take the persistent kernel
  int N_layer;          // > 0: N of the whole layer this GEMM is a column piece
                        // of; tiling and split-K follow it, so every piece sums
                        // each output in the same order as the unsplit layer
  int cluster_max;      // > 0: split K across a thread-block cluster of at most
                        // this many CTAs (DSMEM reduction); 0: global scratch
  float* partial;       // split-K scratch (TcPlan::scratch_bytes), set per launch
  int* counters;        // split-K tile counters (TcPlan::tiles ints, zeroed once)
  int no_pdl;           // 1: launch without programmatic dependent launch.  The
                        // kernel reads its bias and issues its first weight
                        // loads before waiting on the previous kernel, which
                        // is safe only when nothing earlier on the stream
                        // writes them (the engine's arena); callers whose W or
                        // bias may come from the kernel just before set this.
};
// Pre-encoded descriptors of one GEMM (built once per layer at load time).
struct TcPlan {
  CUtensorMap tmA;  // valid when conv == 0
  CUtensorMap tmB;
  int bn;           // N tile
  int splits;       // K splits (grid z); 1 = no split
  int cluster;      // splits reduce through a cluster (no global scratch)
  int kb_per_split; // 64-wide k-blocks per split
  int64_t tiles;    // output tiles (split-K counters needed)
  uint64_t scratch_bytes;  // fp32 partials of all splits
  int persist;      // persistent kernel (one CTA per SM looping over tiles)
  int tma_conv;     // convolution A by 4-D TMA per filter tap (tmA is then 4-D)
  int msub;         // persistent: 128-row sub-tiles per tile (2 for N tiles of 64 with A by TMA)
  int wt, ht, tiles_w, tiles_h;  // its output patch and patch counts per image
  int ready;
};
int tc_prepare(const TcGemm& g, TcPlan* p);
int launch_tc_gemm(const TcGemm& g, const TcPlan& p, int* dev_err, cudaStream_t s);
int launch_tc_persist(const TcGemm& g, const TcPlan& p, int* dev_err, cudaStream_t s);

// tcgen05 convolution for channel counts the gather cannot fetch in 16-byte
// pieces (C % 8 != 0), K = kh*kw*C <= 192: weights built in shared memory,
// im2col gathered element by element, persistent over output tiles.
struct TcSmallConv {
  int dtype;  // SWAPNET_F16 or SWAPNET_BF16
  const void* x;  // NHWC input
  const void* W;  // [N][kh][kw][C]
  int M, N, K;    // M = n*Ho*Wo, N = cout, K = kh*kw*C
  int H, Wd, C, Ho, Wo, kh, kw, stride, pad;
  Epi e;
  void* y;
  int64_t ldy;
  int num_sms;
};
bool tc_small_supported(int dtype, int K);
int tc_small_prepare(int dtype, int K);  // once per shape class, outside stream capture
int launch_tc_conv_small(const TcSmallConv& g, int* dev_err, cudaStream_t s);

// Device error word of the tcgen05 kernels (bounded waits).
int tc_error_word(int** ptr);

// 2-D TMA map of a row-major fp16/bf16 matrix (inner x rows elements, row
// stride in bytes), box of box_inner x box_rows elements, 128-byte swizzle,
// zero fill outside the matrix.  box_inner * 2 bytes must be <= 128.
int make_tmap_2d(CUtensorMap* m, int dtype, const void* base, uint64_t inner, uint64_t rows, uint64_t row_stride_bytes,
                 uint32_t box_inner, uint32_t box_rows);

// tcgen05 causal attention for long query runs (prefill): q [tokens][width]
// (already rotated), key and value caches [max_seq][width], head width 128,
// query t at position *pos_ptr + t attends to positions 0..*pos_ptr + t.
bool attention_tc_supported(int dtype, int tokens, int heads, int width);
int launch_attention_tc(int dtype, const void* q, const void* kc, const void* vc, const int* pos_ptr, int tokens,
                        int heads, int width, int max_seq, void* out, int* err, cudaStream_t s);

}  // namespace swapnet
