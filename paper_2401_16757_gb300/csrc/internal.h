// Internal structures shared by the host-side translation units of libswapnet.
#pragma once
#include <cstdint>
#include <exception>
#include <new>
#include <string>
#include <vector>

#include "../../include/swapnet.h"

namespace swapnet {

constexpr uint64_t kAlign = 256;
inline uint64_t align_up(uint64_t x, uint64_t a = kAlign) { return (x + a - 1) / a * a; }
inline uint64_t ceil_div_u(uint64_t a, uint64_t b) { return (a + b - 1) / b; }

// Thread-local error message for swapnet_last_error().
void set_error(const std::string& msg);

struct Status {
  int code = SWAPNET_OK;
  static Status ok() { return Status{}; }
};

#define SN_FAIL(code, msg)   \
  do {                       \
    ::swapnet::set_error(msg); \
    return (code);           \
  } while (0)

// Runs the body of a C entry point so that no C++ exception crosses the C
// ABI: a failed host allocation becomes SWAPNET_ERR_OOM, anything else
// SWAPNET_ERR_INTERNAL, with the message in swapnet_last_error().
template <typename F>
inline int guard_abi(F&& body) noexcept {
  try {
    return body();
  } catch (const std::bad_alloc&) {
    set_error("host allocation failed");
    return SWAPNET_ERR_OOM;
  } catch (const std::exception& ex) {
    set_error(ex.what());
    return SWAPNET_ERR_INTERNAL;
  } catch (...) {
    set_error("unexpected host-side exception");
    return SWAPNET_ERR_INTERNAL;
  }
}

int dtype_size(int dtype);

// One analysed layer: descriptor plus derived shapes, sizes and liveness.
struct Layer {
  swapnet_layer d;
  int n, h, w, c;        // dims of src0 (the main input)
  int on, oh, ow, oc;    // output dims
  int c1;                // channels of src1 (concat)
  int n_tensors;
  uint64_t tbytes[2];    // raw bytes of each parameter tensor
  int first_tensor;      // global index of the first parameter tensor
  uint64_t flops;
  int last_use;          // last layer reading this output (inclusive)
  int start;             // first layer step at which this output may be written:
                         // i, or (conv / linear whose producers all precede
                         // i - 1) one step after its last producer, so the
                         // engine may run it beside the layers in between
  int64_t ws_off;        // workspace offset, -1 when the output is a model output
  int64_t out_off;       // offset in the output buffer, -1 if not an output
  uint64_t out_bytes;    // raw bytes of the output tensor
  bool host_resident;    // parameters read in host memory, never swapped (EMBED)
  int64_t state_off;     // ATTENTION: offset of its key cache in the decoder state
};

struct Model {
  int dtype = 0, es = 0, in_dtype = 0;
  uint64_t state_bytes = 0;  // decoder state: 256-byte position header + KV caches
  bool has_attention = false;
  int in_n = 0, in_h = 0, in_w = 0, in_c = 0;
  std::vector<Layer> L;
  int n_tensors = 0;
  uint64_t ws_bytes = 0, out_bytes = 0, in_bytes = 0, weight_bytes = 0;
  std::vector<uint64_t> tensor_raw;  // raw bytes per global tensor
};

// Partition unit: a layer, or a piece of an oversize linear layer.
struct Unit {
  int layer, row0, rows, depth;
  uint64_t bytes, flops;
  int64_t t_ex;
  // parameter tensors of the unit: global tensor index, byte offset in that
  // tensor, bytes to copy, offset inside the block's slot
  int nt;
  int tidx[2];
  uint64_t toff[2], tlen[2], slot_off[2];
  bool host;  // host-resident parameters: not swapped, read through the mapped alias
};

struct Block {
  int u0, u1, slot, depth;
  uint64_t bytes;
  uint64_t base;  // offset of the block in the arena
  int64_t t_in, t_ex, t_out;
};

}  // namespace swapnet

struct swapnet_plan {
  swapnet::Model model;
  swapnet_options opt;
  bool resident = false;
  // arena: bytes the blocks share; region: the 256-aligned part blocks use;
  // slot: largest piece of a split linear layer (half the region for two
  // co-resident blocks), also the bound for one block with one slot
  uint64_t budget = 0, arena = 0, region = 0, slot = 0;
  std::vector<swapnet::Unit> units;
  std::vector<swapnet::Block> blocks;
  std::vector<uint32_t> cuts;
  int64_t predicted = 0;
  bool exact = true;  // the search proved the plan optimal for its objective
  int prefix_units = 0;       // resident prefix: units [0, prefix_units) are block 0,
  uint64_t prefix_bytes = 0;  // kept at arena offset 0; the swap region follows
};

// An open weights file (storage tier): descriptor, O_DIRECT or not, and the
// validated offset and length of every tensor.
struct swapnet_weights_file {
  int fd = -1;
  bool direct = false;
  uint32_t n = 0;
  uint64_t file_bytes = 0;
  std::vector<uint64_t> off, bytes;
};

namespace swapnet {
constexpr uint64_t kFileAlign = 4096;  // O_DIRECT offset / length / buffer alignment
// One aligned read of a block's swap-in: file bytes [file_off, file_off +
// len) into staging + stage_off.
struct FileRun {
  uint64_t file_off, len, stage_off;
};
// Reads every run; 0, or the errno of the first failure (EIO at end of file).
int file_read_runs(const swapnet_weights_file* f, const FileRun* runs, size_t n, char* stage);

int analyse_model(const swapnet_model_desc* desc, Model* m);
int make_units(const Model& m, const swapnet_options& opt, uint64_t slot, uint64_t region, std::vector<Unit>* out);
void finalize_blocks(swapnet_plan* p, const std::vector<uint32_t>& cuts);
int64_t pipeline_ns(const std::vector<Block>& b, int slots, bool prefix = false);
int64_t cyclic_ns(const std::vector<Block>& b);
int64_t eq4_ns(const std::vector<Block>& b);
uint64_t resident_latency_ns(const Model& m, const swapnet_options& opt);
}  // namespace swapnet
