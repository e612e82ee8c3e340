/*
 * swapnet.h — C ABI of libswapnet: block-swapped DNN inference under a
 * device-memory budget on one GPU (SwapNet, arXiv 2401.16757).
 *
 * The problem the calls solve is the paper's (Sec. 3 "Basic Idea", Sec.
 * 6.2.2 "Partition Blocks within DNN"): given a memory budget b for a model
 * of size s > b, cut the layer sequence into n blocks and execute them in
 * order, swapping each block's parameters into device memory before it runs
 * and releasing them after.  Sec. 6.2.2 ("Allocate Memory Budget across
 * DNNs", Eq. 1) shares one budget among several models.
 *
 * Conventions for every call:
 *   - Status: int, SWAPNET_OK (0) on success, a negative swapnet_status
 *     otherwise.  No C++ exception crosses this boundary (a failed host
 *     allocation is SWAPNET_ERR_OOM, any other one SWAPNET_ERR_INTERNAL).  Output handles
 *     and output arrays are written only on success.  swapnet_last_error()
 *     returns a message for the calling thread's most recent failure.
 *   - Ownership: plans and engines are opaque, library-owned and freed with
 *     swapnet_plan_free / swapnet_engine_free.  Host weight buffers, model
 *     descriptors, and caller-provided device buffers stay caller-owned.
 *   - Layout: activations are NHWC in the model's storage dtype; conv
 *     weights are [cout][kh][kw][cin]; linear weights are [out][in]; a
 *     linear layer flattens its input per batch item in (h, w, c) order.
 *   - Threads: a plan is immutable after creation and may be shared; an
 *     engine is used by one host thread at a time.
 */
#ifndef SWAPNET_H
#define SWAPNET_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ------------------------------------------------------------------ status */
typedef enum swapnet_status {
  SWAPNET_OK = 0,
  SWAPNET_ERR_INVALID_ARG = -1, /* malformed descriptor, option or argument */
  SWAPNET_ERR_INFEASIBLE = -2,  /* no partition fits the budget            */
  SWAPNET_ERR_OOM = -3,         /* host or device allocation failed        */
  SWAPNET_ERR_CUDA = -4,        /* a CUDA runtime/driver call failed       */
  SWAPNET_ERR_TIMEOUT = -5,     /* a bounded device-side wait gave up      */
  SWAPNET_ERR_MISALIGNED = -6,  /* a pointer or size breaks an alignment rule */
  SWAPNET_ERR_UNSUPPORTED = -7, /* shape/dtype combination not implemented */
  SWAPNET_ERR_IO = -8,          /* a weights-file read or write failed      */
  SWAPNET_ERR_INTERNAL = -9     /* an unexpected host-side exception, caught
                                   before it could cross the C ABI          */
} swapnet_status;

/* ------------------------------------------------------------ descriptors */
typedef enum swapnet_dtype {
  SWAPNET_F32 = 0,
  SWAPNET_F16 = 1,
  SWAPNET_BF16 = 2,
  SWAPNET_I32 = 3 /* model input only: token ids */
} swapnet_dtype;

typedef enum swapnet_op {
  SWAPNET_OP_LINEAR = 1,     /* y[m,o] = act(sum_i x[m,i] W[o,i] + b[o] (+res)) */
  SWAPNET_OP_CONV2D = 2,     /* zero-padded 2-D convolution, + bias (+res), act  */
  SWAPNET_OP_MAXPOOL = 3,    /* window max; padding never wins                  */
  SWAPNET_OP_GAP = 4,        /* global average over H and W                     */
  SWAPNET_OP_UPSAMPLE2X = 5, /* nearest neighbour, factor 2 in H and W          */
  SWAPNET_OP_CONCAT = 6,     /* channels of src0 followed by channels of src1   */
  SWAPNET_OP_EMBED = 7,      /* rows of a [cin = vocab][cout = d] table picked by the
                                int32 token ids of the model input; the table
                                stays in host memory and its rows are read there
                                (never swapped)                                  */
  SWAPNET_OP_RMSNORM = 8,    /* x / sqrt(mean(x^2) + eps) * g over cout = d      */
  SWAPNET_OP_ATTENTION = 9,  /* RoPE on q = src0 and k = src1, both stored rounded;
                                k and v = src2 appended to this layer's cache at
                                the state position; query t attends causally to
                                positions 0..pos+t: softmax(q k^T / sqrt(Dh)) v  */
  SWAPNET_OP_ARGMAX = 10     /* int32 index of each row's maximum (ties: lowest) */
} swapnet_op;

typedef enum swapnet_act {
  SWAPNET_ACT_NONE = 0,
  SWAPNET_ACT_RELU = 1,
  SWAPNET_ACT_LEAKY = 2,  /* slope 0.1 */
  SWAPNET_ACT_SWIGLU = 3  /* silu(res) * (acc + b), res = the gate layer */
} swapnet_act;

#define SWAPNET_LAYER_NO_BIAS 1 /* flags: a linear layer without bias tensor */

#define SWAPNET_SRC_INPUT (-1) /* the model input                       */
#define SWAPNET_SRC_NONE (-2)  /* unused producer / no residual operand */

/* One layer of the model information table (Sec. 6.1, Table 2: per layer
 * size, parameter depth and FLOPs — derived here from the shapes).  Layers
 * are listed in execution order; producers precede consumers. */
typedef struct swapnet_layer {
  int32_t op;       /* swapnet_op                                             */
  int32_t src0;     /* producer of the input (layer index or SWAPNET_SRC_INPUT) */
  int32_t src1;     /* second input of CONCAT, else SWAPNET_SRC_NONE           */
  int32_t res;      /* residual operand (layer index) or SWAPNET_SRC_NONE      */
  int32_t act;      /* swapnet_act                                             */
  int32_t res_post; /* 0: act(acc + b + res); 1: act(acc + b) + res            */
  int32_t cin;      /* conv: input channels;  linear: input features            */
  int32_t cout;     /* conv: output channels; linear: output features           */
  int32_t kh, kw, stride, pad; /* conv and maxpool window                      */
  int32_t is_output;/* nonzero: a model output, written to the output buffer   */
  int32_t flags;    /* SWAPNET_LAYER_NO_BIAS                                   */
  int64_t t_ex_ns;  /* measured execution delay; 0 = gamma * FLOPs (Sec. 6.1)  */
  int32_t src2;     /* ATTENTION: the values layer                             */
  int32_t heads;    /* ATTENTION: heads (head width = cout / heads)            */
  int32_t max_seq;  /* ATTENTION: positions the KV cache holds                 */
  float eps;        /* RMSNORM epsilon                                         */
  float theta;      /* ATTENTION: RoPE base (angle = pos * theta^(-2i/Dh))     */
  int32_t reserved;
} swapnet_layer;

/* Parameter tensors of a layer, in this order, are what swapnet_load's
 * host_weights lists: CONV2D and LINEAR have two (weights, bias; one with
 * SWAPNET_LAYER_NO_BIAS), EMBED one (the table), RMSNORM one (the gains);
 * the other ops none.  Model outputs are written to the output buffer in
 * increasing layer order, each at a 256-byte aligned offset (ARGMAX outputs
 * are int32, everything else the model dtype).  ATTENTION uses cout = the
 * width of q, k and v (heads x head width, head width 128). */
typedef struct swapnet_model_desc {
  int32_t dtype;    /* swapnet_dtype of weights and activations          */
  int32_t n_layers;
  const swapnet_layer* layers;
  int32_t in_n, in_h, in_w, in_c; /* model input, NHWC (a matrix is n x 1 x 1 x c) */
  int32_t in_dtype; /* dtype of the model input: the model dtype or SWAPNET_I32 (token ids) */
  int32_t reserved;
} swapnet_model_desc;

typedef enum swapnet_swap_variant {
  SWAPNET_SWAP_AUTO = 0,     /* pick per block by measured time at load        */
  SWAPNET_SWAP_MEMCPY = 1,   /* copy engine: cudaMemcpyAsync from pinned memory */
  SWAPNET_SWAP_ZEROCOPY = 2, /* SM kernel reading mapped host memory           */
  SWAPNET_SWAP_DIRECT = 3,   /* no swap-in: the block's kernels read their
                                parameters in mapped host memory themselves
                                (copy-free dispatch, Sec. 4.2.2, taken to the
                                kernels); for blocks whose units all run SIMT
                                kernels (GEMV, norms, attention, pools), other
                                blocks take ZEROCOPY (MEMCPY when a tensor is
                                not 16-byte aligned), so copy-engine and SM
                                reads of the host weights are not mixed.
                                Never chosen by AUTO.                         */
  SWAPNET_SWAP_PACKED = 4    /* an extension the paper has no counterpart
                                for: bf16 models only.  At load each swapped
                                bf16 tensor whose size is a multiple of 8192
                                bytes is packed losslessly (swapnet_pack_bf16)
                                into engine-held page-locked memory, and an SM
                                kernel reads the packed form over the host
                                link and unpacks it into the arena, so fewer
                                bytes cross the link for the same arena
                                contents.  Pieces that do not pack, and blocks
                                with none that do, take ZEROCOPY.  Packed
                                images are shared by the engines over the same
                                host tensors; the host weights must not change
                                while one of those engines exists.  Not for
                                pageable weights or weights files (a file
                                engine ignores it).  Never chosen by AUTO.     */
} swapnet_swap_variant;

/* Options.  Delay coefficients follow Sec. 6.1: t_in = alpha*s + beta*d,
 * t_ex = gamma*f, t_out = eta*d, in integer units (attoseconds per byte or
 * FLOP; nanoseconds per tensor). */
typedef struct swapnet_options {
  int32_t slots;                 /* arena slots: 2 (swap overlaps compute) or 1 */
  int32_t activations_in_budget; /* 1: the budget also covers the activation workspace */
  int32_t swap_variant;          /* swapnet_swap_variant                         */
  int32_t objective;             /* 0: m-slot pipeline completion; 1: Eq. 4 sum  */
  uint64_t alpha_as_per_byte;
  uint64_t beta_ns_per_tensor;
  uint64_t gamma_as_per_flop;
  uint64_t eta_ns_per_tensor;
  int32_t zc_ctas;               /* CTAs of the zero-copy swap kernel (and of the
                                    unpack kernel of SWAPNET_SWAP_PACKED), 0 =
                                    default (32; one per SM for unpacking)     */
  int32_t graphs;                /* 1 (default): each (input, output) binding of an
                                    engine is captured once as a CUDA graph and
                                    replayed; 0: launch eagerly every call      */
  int32_t preloaded;             /* resident plans only: the caller's arena already
                                    holds this layout (loaded by another engine of
                                    the same layers); swapnet_load skips the upload */
  int32_t branches;              /* 1 (default): a conv / linear layer whose inputs
                                     were all produced before the previous layer runs
                                     on a second stream beside the layers in between
                                     (e.g. a ResNet projection shortcut), when it, its
                                     last producer and its consumers share a block;
                                     0: every layer in order on one stream.  Results
                                     are identical either way. */
  int32_t resident_prefix;       /* 0 (default, the paper's method): every block is
                                     swapped in for every inference.  1 (an extension
                                     the paper has no counterpart for): the planner may
                                     keep the first units' weights in the arena across
                                     inferences (uploaded once at load, never swapped)
                                     and swap the rest through the remaining region;
                                     the prefix length is chosen by the objective among
                                     0, the longest prefix that leaves room for the
                                     rest, and the longest within 1/4, 1/2, 3/4 of its
                                     bytes.  Objective 0 only. */
  int32_t split_cap;             /* 0 (default): the kernels choose how many ways to
                                     split K for layers with fewer output tiles than
                                     SMs; n > 0: at most n (1 = never split).  A
                                     tuning knob; results differ in the last bits
                                     between split counts (each count is
                                     deterministic). */
  int32_t prefetch;              /* 0 (default): every inference is self-contained and
                                     starts by swapping in its first block.  1: steady-
                                     state back-to-back inferences (Sec. 4.3 pipeline
                                     carried across inferences): each inference ends by
                                     swapping the next inference's first block into its
                                     place, overlapped with its own last layers, and the
                                     next one starts with it present (the engine swaps it
                                     in once at load).  The planner minimises that cyclic
                                     schedule: first block ready at t = 0; its next copy
                                     starts once the copy engine is free and the last
                                     block sharing its place (the last even-indexed
                                     block) has executed; with an even number of blocks
                                     the last block and the first must fit the region
                                     together.  Objective 0, two slots, no resident
                                     prefix.  Consecutive inferences of one engine must
                                     be issued on one stream (as for any engine). */
  int32_t merge;                 /* 1 (default): GEMV layers of one block that read
                                     the same input (e.g. q, k, v; a SwiGLU gate and
                                     up projection) run as one launch; 0: one launch
                                     per layer.  Results are identical either way;
                                     profiling gives every layer of a merged launch
                                     that launch's start and end. */
  int32_t pageable;              /* 0 (default): the host weights are page-locked
                                     (registered at load unless CUDA already pinned
                                     them).  1 (the paper's w/o-uni-add ablation): they
                                     stay in pageable memory and every swap-in is a
                                     copy-engine copy the driver stages through its own
                                     page-locked buffer; launches are eager (no graphs),
                                     the swap variant is MEMCPY (AUTO resolves to it;
                                     ZEROCOPY and DIRECT are refused), and models whose
                                     layers read a table in host memory (EMBED) are
                                     refused (UNSUPPORTED) at load.  Ignored by engines
                                     loaded from a weights file. */
  int32_t reserved[1];
} swapnet_options;

/* Fills the defaults: 2 slots, activations outside the budget, AUTO swap,
 * pipeline objective, alpha = 2.5e6 as/B (400 GB/s), beta = 2000 ns,
 * gamma = 2000 as/FLOP (500 TFLOP/s), eta = 0, CUDA graphs on. */
void swapnet_default_options(swapnet_options* opt);

/* ------------------------------------------------------------------ plans */
typedef struct swapnet_plan swapnet_plan;

typedef struct swapnet_plan_info {
  uint32_t n_blocks;
  uint32_t n_units;        /* layers, with oversize linear layers split      */
  uint32_t slots;          /* 0 for a resident (all weights in HBM) plan     */
  uint32_t n_layers;
  uint64_t budget_bytes;
  uint64_t arena_bytes;    /* device bytes for weights                       */
  uint64_t slot_bytes;     /* largest piece of a split linear layer          */
  uint64_t workspace_bytes;/* intermediate activations (liveness-planned)    */
  uint64_t input_bytes;    /* model input                                    */
  uint64_t output_bytes;   /* all model outputs, 256-byte aligned each       */
  uint64_t weight_bytes;   /* sum of 256-aligned parameter tensor sizes      */
  uint64_t plan_bytes;     /* host bytes of the plan (the resident skeleton) */
  int64_t predicted_ns;    /* objective value of the chosen partition        */
  uint64_t state_bytes;    /* decoder state (position + KV caches), 0 if none */
  int32_t exact;           /* 1: the search proved the plan optimal; 0: its
                              frontier was capped and the plan is the best found */
  int32_t reserved;
  uint32_t prefix_units;   /* resident_prefix: units kept in the arena (block 0) */
  uint32_t reserved2;
  uint64_t prefix_bytes;   /* their bytes at the bottom of the arena; the swap
                              region follows them                             */
} swapnet_plan_info;

typedef struct swapnet_unit_info {
  int32_t layer;   /* layer index                                            */
  int32_t row0;    /* first output feature (linear pieces), else 0           */
  int32_t rows;    /* output features in this unit (linear), else 0          */
  int32_t depth;   /* parameter tensors                                      */
  uint64_t bytes;  /* 256-aligned parameter bytes                            */
  uint64_t flops;
  int64_t t_ex_ns;
} swapnet_unit_info;

typedef struct swapnet_block_info {
  uint32_t unit0, unit1; /* units [unit0, unit1)                             */
  uint32_t slot;         /* block parity: which co-resident position it takes;
                            UINT32_MAX for a resident prefix block           */
  uint32_t depth;
  uint64_t bytes;
  int64_t t_in_ns, t_ex_ns, t_out_ns;
  uint64_t offset;       /* byte offset of the block in the arena            */
} swapnet_block_info;

/* Partition the model for a budget (Sec. 6.2.2, Eq. 2-3; objective per
 * opt->objective).  The arena is the budget (minus the workspace when
 * activations_in_budget), rounded down to 256 bytes.  With two co-resident
 * blocks every pair of consecutive blocks must fit the arena together
 * (Eq. 3: s_i + s_{i+1} <= b): even blocks are placed at the bottom of the
 * arena and odd blocks against its top.  With one slot each block must fit
 * the arena alone.  A linear layer larger than slot_bytes (half the arena
 * with two blocks) is split along output features into pieces of a
 * multiple of 128 features.  Ties: fewer blocks, then the
 * lexicographically smallest cut vector.  Host only; no device work.
 * Errors: INVALID_ARG (descriptor/options), INFEASIBLE (no partition). */
int swapnet_partition(const swapnet_model_desc* desc, uint64_t budget_bytes,
                      const swapnet_options* opt /* nullable: defaults */,
                      swapnet_plan** out_plan);

/* Build a plan from explicit cut points (Sec. 6.2.2 "create_blocks"): cut c
 * places a block boundary before unit c; cuts strictly increasing in
 * [1, n_units).  Units are computed for the budget as in swapnet_partition.
 * Errors: INVALID_ARG (bad cuts), INFEASIBLE (a block exceeds a slot). */
int swapnet_plan_from_cuts(const swapnet_model_desc* desc, const uint32_t* cuts, uint32_t n_cuts,
                           uint64_t budget_bytes, const swapnet_options* opt,
                           swapnet_plan** out_plan);

/* The sufficient-memory reference (DInf): one block holding every weight,
 * loaded once and kept resident; the same kernels run the same units. */
int swapnet_plan_resident(const swapnet_model_desc* desc, const swapnet_options* opt,
                          swapnet_plan** out_plan);

int swapnet_plan_info_get(const swapnet_plan* plan, swapnet_plan_info* info);
/* Copy up to `cap` entries; return the number available in *n (nullable). */
int swapnet_plan_cuts(const swapnet_plan* plan, uint32_t* cuts, uint32_t cap, uint32_t* n);
int swapnet_plan_units(const swapnet_plan* plan, swapnet_unit_info* units, uint32_t cap, uint32_t* n);
int swapnet_plan_blocks(const swapnet_plan* plan, swapnet_block_info* blocks, uint32_t cap, uint32_t* n);
/* Byte offset of each model output inside the output buffer (in layer order). */
int swapnet_plan_output_offsets(const swapnet_plan* plan, uint64_t* offs, uint32_t cap, uint32_t* n);
void swapnet_plan_free(swapnet_plan* plan);

/* Multi-DNN budget split (Sec. 6.2.2, Eq. 1): with demands M_i (weight
 * bytes) and performance scores PS_i = u_i * latency_i / M_i (latency_i =
 * predicted all-resident latency), model i receives
 *   A_i = M_i/sum(M) (1 - 1/n) M + PS_i/sum(PS) (1/n) M,
 * floored to 256 bytes, when sum(M) > M (else A_i = M_i); each model is
 * then partitioned for A_i.  budgets_out[n] and plans_out[n] are written on
 * success only; the caller frees each plan. */
int swapnet_schedule(const swapnet_model_desc* const* models, const float* urgency, uint32_t n,
                     uint64_t arena_bytes, const swapnet_options* opt,
                     uint64_t* budgets_out, swapnet_plan** plans_out);

/* ---------------------------------------------------------------- engines */
typedef struct swapnet_engine swapnet_engine;
typedef struct CUstream_st* swapnet_stream; /* a cudaStream_t; NULL = legacy default stream */

/* Bind a plan to host weights and device memory (Sec. 4.2 zero-copy
 * swap-in, Sec. 5.2 assembly by reference).
 *   host_weights: n_tensors pointers, one per parameter tensor in layer
 *     order; caller-owned, must outlive the engine and must not change.
 *     They are page-locked and mapped in place (cudaHostRegister), never
 *     copied on the host; memory already pinned by CUDA is used as is.
 *   d_arena: device buffer of >= arena_bytes for the weight slots, 256-byte
 *     aligned; NULL = the library allocates it.  d_workspace likewise for
 *     the activation workspace.
 * The plan is copied; it may be freed after this call.  Creates a copy
 * stream and per-slot events; resolves every layer's parameter address to
 * slot base + offset and builds its TMA descriptors once (the skeleton).
 * With SWAPNET_SWAP_AUTO it times both swap variants per block, then whole
 * inferences with that per-block choice, with every block on the copy
 * engine and with every block on the zero-copy kernel, and keeps the
 * fastest; decoder models (attention layers, a bound state) take the
 * zero-copy kernel for every block, so that the engines of one model never
 * mix copy-engine and SM reads of their shared host weights.  With
 * SWAPNET_SWAP_PACKED it packs every swapped bf16 tensor that packs (or
 * takes the packed image another engine made of the same host tensor) and
 * keeps a device table of the unpack jobs of each block.  A resident plan
 * copies all weights to the arena here.
 * Errors: INVALID_ARG, MISALIGNED, OOM, CUDA, UNSUPPORTED, INTERNAL. */
int swapnet_load(const swapnet_plan* plan, const void* const* host_weights, uint32_t n_tensors,
                 void* d_arena, uint64_t arena_bytes, void* d_workspace, uint64_t workspace_bytes,
                 swapnet_engine** out_engine);

/* ----------------------------------------------------------- storage tier
 * Sec. 4.2.1 "Direct Block Fetch": the blocks live in external storage and
 * are fetched with direct I/O (O_DIRECT, bypassing the page cache, so no
 * second copy of a block sits in host memory) into a dedicated swap-in
 * channel.  Here the channel is two page-locked staging buffers per engine:
 * block k is read from the file into staging buffer k mod 2 by a host
 * function on the engine's read stream, then copied by the copy engine into
 * its arena slot, so the read of block k+1 overlaps the copy of block k and
 * the execution of block k-1.
 *
 * Weights file layout (little-endian), written by swapnet_weights_file_write:
 *   bytes 0..7     magic "SWNWGT01"
 *   uint32         version = 1
 *   uint32         n_tensors
 *   uint64         data_offset (first tensor; a multiple of 4096)
 *   n_tensors x {uint64 offset, uint64 bytes}: tensor t in layer order, as
 *                  in swapnet_load's host_weights; offset a multiple of 4096
 *   zero padding; the file length is a multiple of 4096.
 */
typedef struct swapnet_weights_file swapnet_weights_file;

enum { SWAPNET_FILE_ALLOW_BUFFERED = 1 }; /* open flag: no O_DIRECT -> page cache */

/* Write every parameter tensor of `desc` (n_tensors host pointers in layer
 * order, tensor sizes from the descriptor) to `path` in the layout above,
 * then fsync.  Errors: INVALID_ARG, IO (errno text in swapnet_last_error). */
int swapnet_weights_file_write(const char* path, const swapnet_model_desc* desc, const void* const* host_weights,
                               uint32_t n_tensors);

/* Open and validate a weights file for reading with O_DIRECT.  Where the
 * file system refuses O_DIRECT, fails with IO unless flags has
 * SWAPNET_FILE_ALLOW_BUFFERED (then reads go through the page cache and
 * swapnet_weights_file_info reports direct = 0).  Errors: INVALID_ARG (bad
 * header), IO, OOM. */
int swapnet_weights_file_open(const char* path, uint32_t flags, swapnet_weights_file** out);
int swapnet_weights_file_info(const swapnet_weights_file* f, uint32_t* n_tensors, int32_t* direct);
/* Host read of bytes [offset, offset + bytes) of tensor t into dst through
 * the file's read path (an aligned bounce buffer).  Errors: INVALID_ARG
 * (range outside the tensor), IO. */
int swapnet_weights_file_read(swapnet_weights_file* f, uint32_t tensor, uint64_t offset, uint64_t bytes, void* dst);
/* The file must outlive every engine loaded from it. */
void swapnet_weights_file_close(swapnet_weights_file* f);

/* As swapnet_load, with the parameters in a weights file instead of host
 * memory: swapped blocks are fetched from the file for every inference
 * (staging, read stream and host functions as above); a resident plan or a
 * resident prefix is read once here.  Swap variant: copy engine (AUTO and
 * ZEROCOPY are taken as MEMCPY).  Models with host-resident parameters
 * (EMBED) are not supported.  A failed read inside an inference is reported
 * by the next swapnet_engine_sync as IO.  Errors: as swapnet_load, plus IO,
 * UNSUPPORTED. */
int swapnet_load_file(const swapnet_plan* plan, swapnet_weights_file* file, void* d_arena, uint64_t arena_bytes,
                      void* d_workspace, uint64_t workspace_bytes, swapnet_engine** out_engine);

/* One inference, asynchronous on `stream` (Sec. 4.3, Sec. 6.2.2 with m
 * slots): block k is swapped into slot k mod m on the engine's copy stream
 * once the slot's previous block has finished executing, and its layers run
 * on `stream` once the swap is done; block k+1's swap overlaps block k's
 * execution.  d_input / d_output are device pointers of input_bytes and
 * output_bytes (plan info), 16-byte aligned.  Device faults surface at the
 * next synchronising call; bounded device waits report through
 * swapnet_engine_sync.  Errors: INVALID_ARG, MISALIGNED, CUDA. */
int swapnet_infer(swapnet_engine* eng, const void* d_input, void* d_output, swapnet_stream stream);

/* As swapnet_infer, from and to host buffers: the input is copied to an
 * engine-owned device buffer and the outputs back, all on `stream` (copies
 * are asynchronous when the host buffers are pinned).  The host output is
 * valid after the stream has been synchronised. */
int swapnet_infer_host(swapnet_engine* eng, const void* h_input, void* h_output, swapnet_stream stream);

/* Waits for the engine's streams; returns TIMEOUT if a kernel's bounded
 * wait gave up since the last call (the error word is then cleared), CUDA
 * on a device error, IO if a weights-file read failed (then cleared). */
int swapnet_engine_sync(swapnet_engine* eng);

/* Runtime budget adaptation (Sec. 6.2.2 "adaptively partition and exchange
 * blocks"; the dynamic-budget case study of Sec. 8): switch a loaded engine,
 * between inferences, to another plan of the same model, e.g. one of several
 * plans made ahead with swapnet_partition for different budgets (the
 * paper's look-up table of partitions).  Waits for the engine's work in
 * flight; keeps the host registration, streams, workspace and bound decoder
 * state; re-derives blocks, copy segments, unit pointers and descriptors
 * (the paper's "repeat steps 2 and 3"); re-allocates an engine-owned arena
 * at the new plan's size, releasing the old one first, so a smaller budget
 * gives memory back.  A caller-provided arena stays and must hold the new
 * plan.  The plan is copied; the caller may free it after the call.
 * Errors: INVALID_ARG (a plan for another model, resident <-> swapped, or
 * a different `pageable` option), OOM, CUDA. */
int swapnet_engine_adapt(swapnet_engine* eng, const swapnet_plan* plan);

/* Decoder state of a model with ATTENTION layers: a device buffer of
 * state_bytes (plan info), caller-owned, 256-byte aligned.  Layout: an int32
 * position (tokens already cached) in the first 256 bytes, then for every
 * ATTENTION layer in layer order its key cache and value cache
 * [max_seq][cout] in the model dtype, each 256-byte aligned.  Zero the
 * buffer to start a new sequence.  Each inference reads the position on the
 * device, appends its tokens at that position and advances it by the number
 * of input tokens, so a prefill engine and a decode engine built from the
 * same layers can share one state buffer, and a decode step replays the same
 * CUDA graph every time.  A position that would pass max_seq is not written;
 * swapnet_engine_sync then reports SWAPNET_ERR_INVALID_ARG.
 * Must be bound before the first swapnet_infer of such a model. */
int swapnet_engine_bind_state(swapnet_engine* eng, void* d_state, uint64_t state_bytes);

typedef struct swapnet_engine_block {
  int32_t variant;       /* swapnet_swap_variant chosen for the block     */
  int32_t n_segments;    /* contiguous host->arena copies per swap-in     */
  float memcpy_us;       /* measured at load (AUTO), else 0               */
  float zerocopy_us;
} swapnet_engine_block;

int swapnet_engine_blocks(const swapnet_engine* eng, swapnet_engine_block* blocks, uint32_t cap,
                          uint32_t* n);
/* Counters of the inferences since load: kernel launches include the layer
 * kernels and the swap kernels (zero-copy, unpack); memcpy_calls counts copy-engine
 * transfers and bytes_swapped the bytes moved into the arena (uploads at
 * load time excluded; a block read in place, SWAPNET_SWAP_DIRECT, adds
 * nothing). */
typedef struct swapnet_engine_stats {
  uint64_t infer_calls;
  uint64_t kernel_launches;
  uint64_t memcpy_calls;
  uint64_t bytes_swapped;
  uint64_t link_bytes;   /* bytes the swaps read over the host link: the
                            packed form for SWAPNET_SWAP_PACKED blocks, the
                            bytes swapped for the others */
} swapnet_engine_stats;
int swapnet_engine_stats_get(const swapnet_engine* eng, swapnet_engine_stats* stats);

/* Kernel family that runs each unit. */
typedef enum swapnet_kernel_kind {
  SWAPNET_KERNEL_TC_GEMM = 1,     /* tcgen05 GEMM, A and B by TMA             */
  SWAPNET_KERNEL_TC_CONV = 2,     /* tcgen05 implicit-GEMM conv (A gathered)  */
  SWAPNET_KERNEL_SKINNY = 3,      /* SIMT GEMV family: fp32 <= 16 rows, fp16/bf16 <= 4 rows */
  SWAPNET_KERNEL_DIRECT_CONV = 4, /* SIMT direct convolution                  */
  SWAPNET_KERNEL_MAXPOOL = 5,
  SWAPNET_KERNEL_GAP = 6,
  SWAPNET_KERNEL_UPSAMPLE = 7,
  SWAPNET_KERNEL_CONCAT = 8,
  SWAPNET_KERNEL_TILED = 9,       /* SIMT tiled linear (general fallback)     */
  SWAPNET_KERNEL_EMBED = 10,      /* zero-copy embedding gather               */
  SWAPNET_KERNEL_RMSNORM = 11,
  SWAPNET_KERNEL_ATTENTION = 12,  /* two launches: RoPE + cache append, attention */
  SWAPNET_KERNEL_ARGMAX = 13,
  SWAPNET_KERNEL_TC_CONV_SMALL = 14 /* tcgen05 conv for C % 8 != 0 (RGB stems)  */
} swapnet_kernel_kind;
int swapnet_engine_unit_kernels(const swapnet_engine* eng, int32_t* kinds, uint32_t cap, uint32_t* n);

/* How each tensor-core unit is tiled (introspection for measurement; the
 * paper has no counterpart).  For unit i, tiling[i] gets: n_tile (N columns
 * per output tile), splits (K splits; 1 = none), cluster (1: the splits of a
 * tile reduce through a thread-block cluster), persistent (1: one CTA per SM
 * loops over the tiles), tap_tma (1: convolution A loaded by one 4-D TMA per
 * filter tap).  Units off the tensor cores get all zeros.  Same count
 * protocol as swapnet_engine_unit_kernels. */
typedef struct swapnet_unit_tiling {
  int32_t n_tile, splits, cluster, persistent, tap_tma, reserved[3];
} swapnet_unit_tiling;
int swapnet_engine_unit_tiling(const swapnet_engine* eng, swapnet_unit_tiling* tiling, uint32_t cap,
                               uint32_t* n);

/* Device timing for measurement: while enabled, every swapnet_infer records
 * a CUDA event pair around each unit's kernel (on the inference stream) and
 * around each block's swap-in (on the copy stream).  The events add a small
 * gap between launches; leave profiling off for latency measurements.
 * swapnet_engine_last_times synchronises and returns, for the most recent
 * profiled inference, microseconds per unit and per block swap-in. */
int swapnet_engine_set_profiling(swapnet_engine* eng, int enable);

/* Offline profiling of the execution delays (Sec. 6.1: the paper fits its
 * coefficients once per device).  Times every unit's kernel on the engine's
 * device as a graph of `reps` back-to-back launches (so consecutive launches
 * overlap as they do inside an inference) and writes microseconds per launch
 * to unit_us[0..n_units).  The values a unit reads are whatever its buffers
 * hold; the kernels' timing does not depend on them.  Synchronous.
 * Errors: INVALID_ARG, OOM (staging buffers), CUDA. */
int swapnet_engine_measure_units(swapnet_engine* eng, int32_t reps, float* unit_us, uint32_t n_units);
int swapnet_engine_last_times(swapnet_engine* eng, float* unit_us, uint32_t n_units, float* swap_us,
                              uint32_t n_blocks);

/* Swap-in time of each block as it runs inside the inference graph that
 * swapnet_infer replays (Sec. 4.2's t^in, measured in place rather than
 * with the eager, event-instrumented launches of profiling).  With swap
 * timing on, the engine captures (and caches) a graph variant that records
 * an event on the copy stream right before and right after each block's
 * swap-in; layer launches are unchanged, so the replay is the inference
 * that swapnet_infer times, plus 2 event-record nodes per swapped block.
 * swapnet_engine_last_swap_times waits for the most recent inference's last
 * swap events and writes microseconds per block to swap_us[0..n_blocks)
 * (0 for blocks that are not swapped: a resident prefix, blocks read in
 * place, every block of a resident plan).
 * Errors: INVALID_ARG (null engine or output, timing never enabled), CUDA. */
int swapnet_engine_set_swap_timing(swapnet_engine* eng, int enable);
int swapnet_engine_last_swap_times(swapnet_engine* eng, float* swap_us, uint32_t n_blocks);

/* The pipeline of Sec. 4.3 as it runs inside the replayed inference graph:
 * with the timeline on, the engine captures (and caches) a graph variant
 * that also records an event on the caller's stream at the start of the
 * inference and right before and after each block's layers, besides the
 * swap-in events above.  swapnet_engine_last_graph_timeline waits for the
 * most recent inference's last block and writes 4 floats per block to
 * t_us[4 * k .. 4 * k + 3], microseconds since the start of that inference:
 * swap-in start, swap-in end (both -1 for blocks that are not swapped in
 * during the inference: a resident prefix, blocks read in place, the first
 * block under first-block prefetch, every block of a resident plan), start
 * and end of the block's layers on the caller's stream.  The extra nodes
 * sit between the last layer of one block and the first of the next, so
 * they can add the cost of a dependent launch at each block boundary; the
 * timeline explains a replay, swapnet_infer without it is the one to time.
 * Errors: INVALID_ARG (null engine or output, timeline never enabled), CUDA. */
int swapnet_engine_set_graph_timeline(swapnet_engine* eng, int enable);
int swapnet_engine_last_graph_timeline(swapnet_engine* eng, float* t_us, uint32_t n_blocks);

/* The offline fit of the delay model on this device (Sec. 6.1: the paper
 * profiles each device once and fits t_ex = gamma * f and t_in = alpha * s +
 * beta * d by linear regression).  Here the execution delays are measured
 * per layer instead of fitted per FLOP:
 *   t_ex_ns[l] (n_layers entries, the model's layer count) = the summed
 *     swapnet_engine_measure_units time of layer l's units (reps launches
 *     each), at least 1 ns; when resident_ns > 0 (the measured latency of
 *     the same model with every weight resident), every t_ex is scaled so
 *     that they add up to it, since units timed alone miss the launch and
 *     cache effects of the whole dependent chain;
 *   alpha_as_per_byte = the copy-engine swap-in times measured at load
 *     (SWAPNET_SWAP_AUTO engines) over those blocks' bytes, in attoseconds
 *     per byte; 0 when the engine measured none.
 * The results are meant for swapnet_layer.t_ex_ns and
 * swapnet_options.alpha_as_per_byte of the next swapnet_partition (with
 * beta_ns_per_tensor 0: the per-block times already contain it).
 * Synchronous.  Errors: INVALID_ARG (n_layers other than the model's), OOM,
 * CUDA. */
int swapnet_engine_calibrate(swapnet_engine* eng, int32_t reps, int64_t resident_ns, int64_t* t_ex_ns,
                             uint32_t n_layers, uint64_t* alpha_as_per_byte);
/* Start and end of every unit kernel and block swap-in of the most recent
 * profiled inference, in microseconds after the first of those events
 * (arrays of n_units and n_blocks entries; swap entries are 0 for a
 * resident plan).  Synchronises. */
int swapnet_engine_last_timeline(swapnet_engine* eng, float* unit_start, float* unit_end, uint32_t n_units,
                                 float* swap_start, float* swap_end, uint32_t n_blocks);

/* Waits for the device to finish the engine's work (inferences may still be
 * queued on the caller's stream), then releases its streams, events,
 * graphs, staging buffers and engine-owned device memory, and unregisters
 * the host ranges it registered.  NULL is ignored. */
void swapnet_engine_free(swapnet_engine* eng);

/* ------------------------------------------------- allocation-free GEMM */
/* Y[m][n] = act(sum_k A[m][k] * W[n][k] + bias[n]) for fp16 or bf16 data,
 * computed by the same tcgen05 split-K GEMM kernel the engine uses for
 * linear layers, but with its split-K scratch (fp32 partial sums and tile
 * counters) in a fixed device array inside the library instead of memory
 * the engine allocates.  The paper has no counterpart to this call.
 *
 * It is for callers that must not allocate device memory: code running
 * under a hard device-memory budget in which every byte is already
 * assigned (the situation this library is about), or hosts whose own
 * allocator has reserved the whole GPU so that cudaMalloc would fail.
 * The call allocates nothing: no cudaMalloc, no cudaFree, no allocating
 * library routine.
 *
 *   dtype   SWAPNET_F16 or SWAPNET_BF16
 *   A       device, [M][K] row-major; W device, [N][K] row-major;
 *           bias device, [N]; Y device, [M][N] row-major, written
 *   act     swapnet_act applied after the bias
 *   stream  the call is asynchronous on it
 * Pointers must be 16-byte aligned and K a multiple of 8.
 *
 * Limits and sharing: the scratch array holds SWAPNET_NOALLOC_SCRATCH_BYTES
 * (4 MiB) on every GPU that loads the library, until the process exits.  A
 * problem whose split-K scratch exceeds it is rejected with
 * SWAPNET_ERR_INVALID_ARG before anything is launched.  Every call shares
 * the array and it keeps the last call's contents; each call clears the
 * counters it needs on `stream` first.  Calls that overlap on the GPU (on
 * different streams, or on the same device from several threads) race on
 * the array and must be serialised by the caller.
 *
 * Ordering: the kernel starts only after the work queued before it on
 * `stream` has completed (no programmatic early start), so A, W and bias may
 * be the output of the previous call or kernel on the stream.
 *
 * Set-up: the first call on a device looks up the array's device address
 * (cudaGetSymbolAddress) with that device current and caches it; make that
 * first call before any stream capture.
 * Errors: INVALID_ARG, MISALIGNED, UNSUPPORTED, CUDA.  Device-side failures
 * are not returned by this call, which does not wait for its kernel: if a
 * bounded wait inside the kernel gives up (one second), Y is incomplete and
 * the timeout is recorded in the library's device error word, which the
 * next swapnet_engine_sync (of any engine on the device) reports as
 * SWAPNET_ERR_TIMEOUT and clears. */
#define SWAPNET_NOALLOC_SCRATCH_BYTES (4u << 20)
int swapnet_gemm_noalloc(int32_t dtype, const void* A, const void* W, const void* bias, void* Y, int32_t M,
                         int32_t N, int32_t K, int32_t act, swapnet_stream stream);

/* --------------------------------------------------------- host weights */
/* Page-locked, device-mapped host memory for weight storage (the pinned
 * host copy that Sec. 4.2's swap-in reads): allocated by the CUDA driver in
 * large physically contiguous pieces, so the copy engines and the zero-copy
 * kernel stream it at full link rate however large it is; swapnet_load uses
 * it in place (no registration).  Caller-owned: release with
 * swapnet_host_free after every engine using it is freed.
 * Errors: INVALID_ARG (null out or zero bytes), OOM. */
int swapnet_host_alloc(uint64_t bytes, void** out);
int swapnet_host_free(void* p);

/* The lossless packed form of n_elems bf16 values (SWAPNET_SWAP_PACKED; an
 * extension the paper has no counterpart for).  Each value is split into
 * its exponent and a sign-mantissa byte; the exponent x is stored as the
 * 4-bit code x - x0, where x0 .. x0 + 14 (x0 <= 240) is the window of 15
 * consecutive exponents holding most of the tensor, code 15 marking an
 * exception; up to 4 exceptions per chunk of 4096 values are listed in the
 * chunk's header and chunks with more are stored unpacked.  Layout
 * (little-endian): 16 bytes (x0, then zeros); a 16-byte header per chunk
 * ([0] exception count or 0xff for an unpacked chunk, [4,12) positions as
 * uint16 (for 0xff: the overflow index as uint32 in [4,8)), [12,16) their
 * exponents); zeros up to a multiple of 128 bytes; a 6144-byte body per
 * chunk (2048 bytes of codes, two per byte, low nibble first, then 4096
 * sign-mantissa bytes (w >> 8 & 0x80) | (w & 0x7f); zeros for an unpacked
 * chunk); then the unpacked chunks, 8192 bytes
 * each.  A value is rebuilt as ((s & 0x80) << 8) | (x << 7) | (s & 0x7f)
 * with x = x0 + code, or the listed exponent for code 15.
 * With dst NULL only *used_bytes (the packed size) is written; otherwise
 * dst (dst_bytes long, any alignment) receives the packed form.  Host only,
 * multithreaded.  Errors: INVALID_ARG (null src or used_bytes, dst too
 * small), UNSUPPORTED (n_elems not a positive multiple of 4096), OOM (host
 * memory or threads). */
int swapnet_pack_bf16(const void* src, uint64_t n_elems, void* dst, uint64_t dst_bytes, uint64_t* used_bytes);

/* ------------------------------------------------------------------- misc */
const char* swapnet_strerror(int status);
const char* swapnet_last_error(void);

/* Host-side fault injection for tests: the next `count` calls of the named
 * step fail as if the CUDA call had failed.  what: 1 = cudaHostRegister,
 * 2 = device allocation, 3 = event/stream creation.  count 0 disarms. */
int swapnet_debug_fail_next(int what, int count);

/* Failure-detection check for tests: launches on `stream` one kernel whose
 * bounded device wait (the wait every kernel of the library uses on its
 * mbarriers) waits on an mbarrier that nothing completes, so it gives up
 * after the wait limit (one second), records the timeout in the library's
 * device error word and returns; no trap, no fault, the context stays
 * usable.  Synchronises the stream, reads and clears the error word, and
 * returns what swapnet_engine_sync would: SWAPNET_ERR_TIMEOUT. */
int swapnet_debug_wait_timeout(swapnet_stream stream);

#ifdef __cplusplus
}
#endif
#endif /* SWAPNET_H */
