// Engine: binds a plan to host weights (or a weights file, Sec. 4.2.1) and
// device memory, and runs the block pipeline (Sec. 4 swapping, Sec. 5
// assembly by reference, Sec. 6.2.2 with m = slots blocks co-resident).
#include <cuda_runtime.h>
#include <unistd.h>

#include <algorithm>
#include <atomic>
#include <chrono>
#include <cstring>
#include <map>
#include <memory>
#include <mutex>
#include <new>
#include <thread>
#include <utility>

#include "internal.h"
#include "kernels.h"
#include "pack.h"

namespace swapnet {

int g_fail_next[4] = {0, 0, 0, 0};

// Host ranges this library page-locked, shared by every engine that uses
// them: (base, length) -> number of engines.  A range is unregistered when
// its last engine is freed.
static std::mutex g_reg_mu;
static std::map<std::pair<uintptr_t, size_t>, int> g_reg;

static void unregister_range(uintptr_t base, size_t len) {
  std::lock_guard<std::mutex> lk(g_reg_mu);
  auto it = g_reg.find({base, len});
  if (it == g_reg.end()) return;
  if (--it->second == 0) {
    cudaHostUnregister(reinterpret_cast<void*>(base));
    g_reg.erase(it);
  }
}

static bool injected(int what) {
  if (what < 1 || what > 3 || g_fail_next[what] <= 0) return false;
  --g_fail_next[what];
  return true;
}

#define CU(call, what)                                                                         \
  do {                                                                                         \
    cudaError_t e_ = (call);                                                                   \
    if (e_ != cudaSuccess) {                                                                   \
      set_error(std::string(what) + ": " + cudaGetErrorString(e_));                          \
      return SWAPNET_ERR_CUDA;                                                                 \
    }                                                                                          \
  } while (0)

struct Segment {
  const char* src;  // device alias of host memory
  char* dst;
  uint64_t bytes;
};

struct EngBlock {
  std::vector<Segment> segs;
  int variant = SWAPNET_SWAP_MEMCPY;
  float memcpy_us = 0.f, zerocopy_us = 0.f;
};

struct UnitExec {
  const void* w = nullptr;
  const void* b = nullptr;
  bool use_tc = false;
  TcGemm g{};
  TcPlan tc{};
  const void* tmA_for = nullptr;  // A pointer the TMA map was encoded for
  bool in_place = false;          // parameters read in mapped host memory
};

struct HostRange {
  uintptr_t base;
  size_t len;
  bool registered_by_us;
  char* dev;
};

// The packed form of one host tensor (pack.h), made at load by the first
// engine that swaps it with SWAPNET_SWAP_PACKED and shared by every engine
// over the same host tensor (same address and size) until the last is freed.
struct PackedImage {
  uint8_t* host = nullptr;       // page-locked, mapped
  const uint8_t* dev = nullptr;  // its device alias
  uint64_t bytes = 0, chunks = 0, body_off = 0, overflow_off = 0;
  uint32_t x0 = 0;  // exponent window start
  std::vector<uint32_t> raw_before;  // overflow chunks before chunk c (chunks + 1 entries)
  int refs = 0;
};

static std::mutex g_pk_mu;
static std::map<std::pair<uintptr_t, uint64_t>, PackedImage*> g_pk;

static void release_packed(PackedImage* im) {
  std::lock_guard<std::mutex> lk(g_pk_mu);
  if (--im->refs > 0) return;
  for (auto it = g_pk.begin(); it != g_pk.end(); ++it)
    if (it->second == im) {
      g_pk.erase(it);
      break;
    }
  if (im->host) cudaFreeHost(im->host);
  delete im;
}

// Up to 1024 unpack jobs of a block launched together (first: their index
// in the engine's device job array).
struct PkLaunch {
  size_t first;
  int njobs;
  uint32_t chunks;
};

}  // namespace swapnet

using namespace swapnet;

struct swapnet_engine {
  swapnet_plan plan;
  int device = 0;
  int num_sms = 0;
  char* d_arena = nullptr;
  bool own_arena = false;
  uint64_t arena_bytes = 0;
  char* d_ws = nullptr;
  bool own_ws = false;
  char* d_in_stage = nullptr;
  char* d_out_stage = nullptr;
  std::vector<HostRange> ranges;
  std::vector<const char*> tensor_dev;  // device alias per tensor
  std::vector<const char*> tensor_host;  // the caller's pointer per tensor
  // packed swap variant: the packed image of each swapped tensor that packs
  // (null otherwise), and per block the unpack launches, the segments that
  // are not packed (zero-copy kernel) and the bytes read over the host link
  std::vector<PackedImage*> packed;
  PkJob* d_pkjobs = nullptr;
  std::vector<std::vector<PkLaunch>> pk_launch;
  std::vector<std::vector<Segment>> pk_rest;
  std::vector<uint64_t> link_bytes;
  cudaStream_t copy = nullptr;
  cudaEvent_t slot_free[2] = {nullptr, nullptr};
  cudaEvent_t ready[2] = {nullptr, nullptr};
  std::vector<EngBlock> blocks;
  std::vector<UnitExec> ux;
  int* err_word = nullptr;
  int zc_ctas = 32;
  bool weights_loaded = false;  // resident plan: copied once at load
  std::vector<int> unit_kind;   // swapnet_kernel_kind per unit
  swapnet_engine_stats stats{};
  bool profiling = false;
  std::vector<cudaEvent_t> ev_unit;  // 2 per unit
  std::vector<cudaEvent_t> ev_swap;  // 2 per block
  // swap timing inside the replayed graph: event-record nodes around each
  // block's swap-in on the copy stream (swapnet_engine_set_swap_timing)
  bool swap_timing = false;
  std::vector<cudaEvent_t> ev_gswap;  // 2 per block
  // block timeline inside the replayed graph (swapnet_engine_set_graph_timeline):
  // also an event at the start of the inference on the caller's stream and
  // around each block's layers
  bool timeline = false;
  std::vector<cudaEvent_t> ev_gexec;  // 2 per block
  cudaEvent_t ev_g0 = nullptr;
  cudaStream_t cap = nullptr;        // capture origin stream
  cudaEvent_t fork = nullptr, join = nullptr;
  // per (input, output, profiling) binding
  std::map<std::pair<std::pair<const void*, void*>, int>, cudaGraphExec_t> graphs;
  char* d_state = nullptr;           // decoder state (position + KV caches), caller-owned
  // concurrent branches: side units run on `side`, forked after their last
  // producer's unit and joined before their first consumer's
  cudaStream_t side = nullptr;
  cudaEvent_t side_fork = nullptr;
  std::vector<cudaEvent_t> side_done;        // per unit (side units only)
  std::vector<std::vector<int>> side_after;  // per unit: side units forked after it
  std::vector<std::vector<int>> side_wait;   // per unit: side units it waits for
  std::vector<char> is_side;
  // merged GEMV launches: unit u launches itself and the merge_n[u] units
  // after it (merge_pair: as a gate and its paired layer); merged_into[v]:
  // v is launched by an earlier unit
  std::vector<int> merge_n;
  std::vector<char> merge_pair, merged_into;
  char* d_splitk = nullptr;          // split-K scratch: tile counters, then fp32 partials
  uint64_t splitk_bytes = 0;
  uint64_t splitk_counter_bytes = 0;
  // storage tier: blocks fetched from a weights file into staging buffer
  // k mod 2 by a host function on `rd`, then copied into their slot
  swapnet_weights_file* file = nullptr;
  char* stage[2] = {nullptr, nullptr};  // page-locked, kFileAlign aligned
  uint64_t stage_bytes = 0;
  cudaStream_t rd = nullptr;
  cudaEvent_t staged[2] = {nullptr, nullptr}, stage_free[2] = {nullptr, nullptr};
  std::vector<std::vector<FileRun>> fruns;  // per block
  struct ReadJob {
    swapnet_engine* e;
    int k;
  };
  std::vector<ReadJob> jobs;  // host-function arguments, one per block
  std::atomic<int> io_errno{0};
};

namespace swapnet {

static int release(swapnet_engine* e) {
  if (!e) return SWAPNET_OK;
  cudaSetDevice(e->device);
  // a graph replay may still be queued on the caller's stream, and the read
  // host functions of a file engine dereference this engine
  cudaDeviceSynchronize();
  if (e->copy) cudaStreamSynchronize(e->copy);
  for (cudaEvent_t ev : {e->slot_free[0], e->slot_free[1], e->ready[0], e->ready[1]})
    if (ev) cudaEventDestroy(ev);
  for (auto& kv : e->graphs) cudaGraphExecDestroy(kv.second);
  if (e->side) cudaStreamSynchronize(e->side);
  for (cudaEvent_t ev : e->side_done)
    if (ev) cudaEventDestroy(ev);
  if (e->side_fork) cudaEventDestroy(e->side_fork);
  if (e->side) cudaStreamDestroy(e->side);
  if (e->fork) cudaEventDestroy(e->fork);
  if (e->join) cudaEventDestroy(e->join);
  if (e->cap) cudaStreamDestroy(e->cap);
  for (cudaEvent_t ev : e->ev_unit) cudaEventDestroy(ev);
  for (cudaEvent_t ev : e->ev_swap) cudaEventDestroy(ev);
  for (cudaEvent_t ev : e->ev_gswap) cudaEventDestroy(ev);
  for (cudaEvent_t ev : e->ev_gexec) cudaEventDestroy(ev);
  if (e->ev_g0) cudaEventDestroy(e->ev_g0);
  if (e->copy) cudaStreamDestroy(e->copy);
  if (e->rd) {
    cudaStreamSynchronize(e->rd);
    cudaStreamDestroy(e->rd);
  }
  for (cudaEvent_t ev : {e->staged[0], e->staged[1], e->stage_free[0], e->stage_free[1]})
    if (ev) cudaEventDestroy(ev);
  for (char* p : e->stage)
    if (p) cudaFreeHost(p);
  if (e->own_arena && e->d_arena) cudaFree(e->d_arena);
  if (e->own_ws && e->d_ws) cudaFree(e->d_ws);
  if (e->d_splitk) cudaFree(e->d_splitk);
  if (e->d_pkjobs) cudaFree(e->d_pkjobs);
  for (PackedImage* im : e->packed)
    if (im) release_packed(im);
  if (e->d_in_stage) cudaFree(e->d_in_stage);
  if (e->d_out_stage) cudaFree(e->d_out_stage);
  for (const HostRange& r : e->ranges)
    if (r.registered_by_us) unregister_range(r.base, r.len);
  delete e;
  return SWAPNET_OK;
}

// Page-lock and map the caller's weight buffers in place; record the device
// alias of every tensor.
static int register_host(swapnet_engine* e, const void* const* hw, uint32_t nt) {
  const Model& m = e->plan.model;
  if (e->plan.opt.pageable) {  // never registered: every copy is staged by the driver
    for (const Unit& U : e->plan.units)
      if (U.host) SN_FAIL(SWAPNET_ERR_UNSUPPORTED, "pageable weights: a layer reads its table in host memory");
    e->tensor_dev.assign(nt, nullptr);
    for (uint32_t t = 0; t < nt; ++t) {
      if (!hw[t]) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null host weight pointer");
      e->tensor_dev[t] = static_cast<const char*>(hw[t]);
    }
    return SWAPNET_OK;
  }
  const uintptr_t page = (uintptr_t)sysconf(_SC_PAGESIZE);
  struct R { uintptr_t lo, hi; };
  std::vector<R> rs;
  for (uint32_t t = 0; t < nt; ++t) {
    if (!hw[t]) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null host weight pointer");
    const uintptr_t p = reinterpret_cast<uintptr_t>(hw[t]);
    if (m.tensor_raw[t] == 0) continue;
    rs.push_back(R{p / page * page, (p + m.tensor_raw[t] + page - 1) / page * page});
  }
  std::sort(rs.begin(), rs.end(), [](const R& a, const R& b) { return a.lo < b.lo; });
  std::vector<R> merged;
  for (const R& r : rs) {
    if (!merged.empty() && r.lo <= merged.back().hi) merged.back().hi = std::max(merged.back().hi, r.hi);
    else merged.push_back(r);
  }
  for (const R& r : merged) {
    HostRange hr{r.lo, (size_t)(r.hi - r.lo), false, nullptr};
    void* base = reinterpret_cast<void*>(r.lo);
    {  // memory CUDA already page-locked (cudaHostAlloc / cudaMallocHost) is used as is
      uintptr_t probe = r.hi - 1;
      for (uint32_t t = 0; t < nt; ++t) {
        const uintptr_t p = reinterpret_cast<uintptr_t>(hw[t]);
        if (m.tensor_raw[t] && p >= r.lo && p < r.hi) { probe = p; break; }
      }
      cudaPointerAttributes pa;
      if (cudaPointerGetAttributes(&pa, reinterpret_cast<void*>(probe)) == cudaSuccess &&
          pa.type == cudaMemoryTypeHost && g_reg.find({hr.base, hr.len}) == g_reg.end()) {
        e->ranges.push_back(hr);
        continue;
      }
      cudaGetLastError();
    }
    std::lock_guard<std::mutex> lk(g_reg_mu);
    auto it = g_reg.find({hr.base, hr.len});
    if (it != g_reg.end()) {
      ++it->second;
      hr.registered_by_us = true;
      e->ranges.push_back(hr);
      continue;
    }
    cudaError_t err = injected(1) ? cudaErrorMemoryAllocation
                                  : cudaHostRegister(base, hr.len, cudaHostRegisterMapped | cudaHostRegisterReadOnly);
    if (err == cudaErrorNotSupported || err == cudaErrorInvalidValue) {
      cudaGetLastError();
      err = cudaHostRegister(base, hr.len, cudaHostRegisterMapped);
    }
    if (err == cudaSuccess) {
      hr.registered_by_us = true;
      g_reg[{hr.base, hr.len}] = 1;
    } else if (err == cudaErrorHostMemoryAlreadyRegistered) {
      cudaGetLastError();  // pinned by its owner (e.g. cudaHostAlloc): used as is
    } else {
      cudaGetLastError();
      set_error(std::string("cudaHostRegister: ") + cudaGetErrorString(err));
      return SWAPNET_ERR_CUDA;  // ranges registered so far are released with the engine
    }
    e->ranges.push_back(hr);
  }
  e->tensor_dev.assign(nt, nullptr);
  e->tensor_host.assign(nt, nullptr);
  for (uint32_t t = 0; t < nt; ++t) e->tensor_host[t] = static_cast<const char*>(hw[t]);
  for (uint32_t t = 0; t < nt; ++t) {
    if (m.tensor_raw[t] == 0) continue;
    void* dptr = nullptr;
    cudaError_t err = cudaHostGetDevicePointer(&dptr, const_cast<void*>(hw[t]), 0);
    if (err != cudaSuccess || !dptr) {
      cudaGetLastError();
      SN_FAIL(SWAPNET_ERR_CUDA, std::string("cudaHostGetDevicePointer: ") + cudaGetErrorString(err));
    }
    e->tensor_dev[t] = static_cast<const char*>(dptr);
  }
  return SWAPNET_OK;
}

static char* block_base(swapnet_engine* e, const Block& B) { return e->d_arena + B.base; }

// Storage tier: each block's parameter pieces become aligned file runs
// (pieces closer than kRunGap share a run), packed one after another in the
// block's staging buffer, and copy segments from staging to the slot.
// Grows the two staging buffers to the largest block.
static int build_file_blocks(swapnet_engine* e) {
  constexpr uint64_t kRunGap = 256 * 1024;
  const swapnet_plan& p = e->plan;
  const swapnet_weights_file* f = e->file;
  e->blocks.assign(p.blocks.size(), EngBlock{});
  e->fruns.assign(p.blocks.size(), {});
  struct Piece {
    uint64_t file_off, len, slot_off;
  };
  std::vector<std::vector<Piece>> pieces(p.blocks.size());
  uint64_t need = kFileAlign;
  for (size_t k = 0; k < p.blocks.size(); ++k) {
    const Block& B = p.blocks[k];
    std::vector<Piece>& pc = pieces[k];
    for (int u = B.u0; u < B.u1; ++u) {
      const Unit& U = p.units[u];
      if (U.host) SN_FAIL(SWAPNET_ERR_UNSUPPORTED, "host-resident parameters cannot be read from a weights file");
      for (int t = 0; t < U.nt; ++t) {
        if (U.tlen[t] == 0) continue;
        const int ti = U.tidx[t];
        if (U.toff[t] + U.tlen[t] > f->bytes[ti]) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "weights file tensor too short");
        pc.push_back(Piece{f->off[ti] + U.toff[t], U.tlen[t], U.slot_off[t]});
      }
    }
    std::sort(pc.begin(), pc.end(), [](const Piece& a, const Piece& b) { return a.file_off < b.file_off; });
    std::vector<FileRun>& runs = e->fruns[k];
    uint64_t staged = 0;
    for (const Piece& q : pc) {
      const uint64_t lo = q.file_off / kFileAlign * kFileAlign, hi = align_up(q.file_off + q.len, kFileAlign);
      if (!runs.empty() && lo <= runs.back().file_off + runs.back().len + kRunGap) {
        FileRun& r = runs.back();
        const uint64_t end = std::max(r.file_off + r.len, hi);
        staged += end - (r.file_off + r.len);
        r.len = end - r.file_off;
      } else {
        runs.push_back(FileRun{lo, hi - lo, staged});
        staged += hi - lo;
      }
    }
    need = std::max(need, staged);
  }
  if (need > e->stage_bytes) {
    for (char*& b : e->stage) {
      if (b) cudaFreeHost(b);
      b = nullptr;
    }
    e->stage_bytes = 0;
    for (char*& b : e->stage) {
      void* q = nullptr;
      if (injected(1) || cudaHostAlloc(&q, need, cudaHostAllocPortable) != cudaSuccess) {
        cudaGetLastError();
        SN_FAIL(SWAPNET_ERR_OOM, "page-locked staging allocation failed");
      }
      b = static_cast<char*>(q);
    }
    e->stage_bytes = need;
  }
  for (size_t k = 0; k < p.blocks.size(); ++k) {
    const std::vector<FileRun>& runs = e->fruns[k];
    char* stage = e->stage[k % 2];
    char* base = block_base(e, p.blocks[k]);
    std::vector<Segment>& segs = e->blocks[k].segs;
    size_t r = 0;
    for (const Piece& q : pieces[k]) {
      while (q.file_off >= runs[r].file_off + runs[r].len) ++r;  // pieces and runs are both sorted
      Segment g{stage + runs[r].stage_off + (q.file_off - runs[r].file_off), base + q.slot_off, q.len};
      if (!segs.empty()) {
        Segment& b = segs.back();
        if (g.src == b.src + b.bytes && g.dst == b.dst + b.bytes) {
          b.bytes += g.bytes;
          continue;
        }
      }
      segs.push_back(g);
    }
  }
  e->jobs.assign(p.blocks.size(), swapnet_engine::ReadJob{e, 0});
  for (size_t k = 0; k < p.blocks.size(); ++k) e->jobs[k].k = (int)k;
  return SWAPNET_OK;
}

// Host function on the read stream: fetch block k's runs into its staging
// buffer.  Calls no CUDA API; a failure is kept for swapnet_engine_sync.
static void CUDART_CB read_block_host(void* arg) {
  const swapnet_engine::ReadJob* j = static_cast<const swapnet_engine::ReadJob*>(arg);
  swapnet_engine* e = j->e;
  const std::vector<FileRun>& runs = e->fruns[j->k];
  const int err = file_read_runs(e->file, runs.data(), runs.size(), e->stage[j->k % 2]);
  if (err) {
    int none = 0;
    e->io_errno.compare_exchange_strong(none, err);
  }
}

// Synchronous fetch of block k (load-time uploads and calibration).
static int fetch_block_sync(swapnet_engine* e, size_t k, float* read_us) {
  const auto t0 = std::chrono::steady_clock::now();
  const int err = file_read_runs(e->file, e->fruns[k].data(), e->fruns[k].size(), e->stage[k % 2]);
  if (read_us)
    *read_us = std::chrono::duration<float, std::micro>(std::chrono::steady_clock::now() - t0).count();
  if (err) SN_FAIL(SWAPNET_ERR_IO, std::string("weights file read: ") + std::strerror(err));
  return SWAPNET_OK;
}

static int swap_block(swapnet_engine* e, size_t k, int variant, cudaStream_t s);

static int upload_file_block(swapnet_engine* e, size_t k, float* us) {
  float read_us = 0.f;
  int rc = fetch_block_sync(e, k, &read_us);
  if (rc) return rc;
  cudaEvent_t a = nullptr, b = nullptr;
  if (us) {
    CU(cudaEventCreate(&a), "event");
    CU(cudaEventCreate(&b), "event");
    cudaEventRecord(a, e->copy);
  }
  rc = swap_block(e, k, SWAPNET_SWAP_MEMCPY, e->copy);
  if (us) cudaEventRecord(b, e->copy);
  const cudaError_t se = cudaStreamSynchronize(e->copy);
  if (us) {
    float ms = 0.f;
    cudaEventElapsedTime(&ms, a, b);
    *us = read_us + ms * 1000.f;
    cudaEventDestroy(a);
    cudaEventDestroy(b);
  }
  if (rc) return rc;
  if (se != cudaSuccess) {
    cudaGetLastError();
    SN_FAIL(SWAPNET_ERR_CUDA, "staging to arena copy failed");
  }
  return SWAPNET_OK;
}

// Per-block swap cost of a file engine, read plus copy, each block alone
// (best of 3): the measured counterpart of t_in for the planner.
static int calibrate_file(swapnet_engine* e) {
  for (size_t k = 0; k < e->blocks.size(); ++k) {
    EngBlock& B = e->blocks[k];
    B.variant = SWAPNET_SWAP_MEMCPY;
    B.zerocopy_us = 0.f;
    if (e->plan.blocks[k].slot < 0) continue;
    float best = 1e30f;
    for (int rep = 0; rep < 3; ++rep) {
      float us = 0.f;
      int rc = upload_file_block(e, k, &us);
      if (rc) return rc;
      best = std::min(best, us);
    }
    B.memcpy_us = best;
  }
  return SWAPNET_OK;
}

static int build_segments(swapnet_engine* e) {
  e->link_bytes.assign(e->plan.blocks.size(), 0);
  for (size_t k = 0; k < e->plan.blocks.size(); ++k) e->link_bytes[k] = e->plan.blocks[k].bytes;
  if (e->file) return build_file_blocks(e);
  const swapnet_plan& p = e->plan;
  e->blocks.assign(p.blocks.size(), EngBlock{});
  for (size_t k = 0; k < p.blocks.size(); ++k) {
    const Block& B = p.blocks[k];
    std::vector<Segment>& segs = e->blocks[k].segs;
    char* base = block_base(e, B);
    for (int u = B.u0; u < B.u1; ++u) {
      const Unit& U = p.units[u];
      if (U.host) continue;  // host-resident parameters are never swapped
      for (int t = 0; t < U.nt; ++t) {
        if (U.tlen[t] == 0) continue;
        Segment s{e->tensor_dev[U.tidx[t]] + U.toff[t], base + U.slot_off[t], U.tlen[t]};
        if (!segs.empty()) {
          Segment& q = segs.back();
          // coalesce when host and slot offsets advance together
          if (s.src > q.src && s.dst > q.dst && (uint64_t)(s.src - q.src) == (uint64_t)(s.dst - q.dst) &&
              (uint64_t)(s.dst - q.dst) <= align_up(q.bytes)) {
            q.bytes = (uint64_t)(s.dst - q.dst) + s.bytes;
            continue;
          }
        }
        segs.push_back(s);
      }
    }
  }
  return SWAPNET_OK;
}

static bool zerocopy_ok(const EngBlock& b);

// The packed image of host tensor t: the one another engine made for the
// same host tensor, or a new one packed from the caller's buffer now.
static int acquire_packed(swapnet_engine* e, int t) {
  const uint64_t raw = e->plan.model.tensor_raw[t];
  const uintptr_t key = reinterpret_cast<uintptr_t>(e->tensor_host[t]);
  std::lock_guard<std::mutex> lk(g_pk_mu);
  auto it = g_pk.find({key, raw});
  if (it != g_pk.end()) {
    ++it->second->refs;
    e->packed[t] = it->second;
    return SWAPNET_OK;
  }
  const int threads = (int)std::min(32u, std::max(1u, std::thread::hardware_concurrency()));
  const uint16_t* src = reinterpret_cast<const uint16_t*>(e->tensor_host[t]);
  const uint64_t n = raw / 2;
  PackInfo info;
  try {
    info = pack_prepare(src, n, threads);
  } catch (...) {  // allocation or thread creation
    SN_FAIL(SWAPNET_ERR_OOM, "packing: host resources exhausted");
  }
  std::unique_ptr<PackedImage> im(new (std::nothrow) PackedImage());
  if (!im) SN_FAIL(SWAPNET_ERR_OOM, "host allocation failed");
  void* h = nullptr;
  if (cudaHostAlloc(&h, info.bytes, cudaHostAllocMapped | cudaHostAllocPortable) != cudaSuccess) {
    cudaGetLastError();
    SN_FAIL(SWAPNET_ERR_OOM, "page-locked allocation of packed weights failed");
  }
  im->host = static_cast<uint8_t*>(h);
  try {
    pack_write(src, n, info, im->host, threads);
  } catch (...) {
    cudaFreeHost(h);
    SN_FAIL(SWAPNET_ERR_OOM, "packing: host resources exhausted");
  }
  void* d = nullptr;
  if (cudaHostGetDevicePointer(&d, h, 0) != cudaSuccess || !d) {
    cudaGetLastError();
    cudaFreeHost(h);
    SN_FAIL(SWAPNET_ERR_CUDA, "device alias of packed weights");
  }
  im->dev = static_cast<const uint8_t*>(d);
  im->bytes = info.bytes;
  im->chunks = n / kPkChunk;
  im->body_off = pk_body_off(im->chunks);
  im->overflow_off = im->body_off + im->chunks * (uint64_t)kPkBody;
  im->x0 = info.exp[0];
  im->raw_before.assign(im->chunks + 1, 0);
  for (uint64_t c = 0; c < im->chunks; ++c)
    im->raw_before[c + 1] = im->raw_before[c] + (info.overflow[c] != UINT32_MAX ? 1u : 0u);
  im->refs = 1;
  e->packed[t] = im.get();
  g_pk[{key, raw}] = im.release();
  return SWAPNET_OK;
}

// Packed swap variant: every piece of a bf16 tensor that starts and ends on
// a chunk boundary is unpacked from its packed image; the other pieces
// (other types, ragged tensors) are copied by the zero-copy kernel.  A
// block with no packed piece takes the zero-copy kernel (the copy engine
// when a piece is not 16-byte aligned).
static int build_packed(swapnet_engine* e) {
  const swapnet_plan& p = e->plan;
  const Model& m = p.model;
  e->packed.resize(m.n_tensors, nullptr);
  e->pk_launch.assign(p.blocks.size(), {});
  e->pk_rest.assign(p.blocks.size(), {});
  std::vector<PkJob> jobs;
  for (size_t k = 0; k < p.blocks.size(); ++k) {
    const Block& B = p.blocks[k];
    EngBlock& EB = e->blocks[k];
    if (B.slot < 0) continue;  // a resident prefix is uploaded once
    uint64_t link = 0;
    std::vector<PkJob> bj;
    for (int u = B.u0; u < B.u1; ++u) {
      const Unit& U = p.units[u];
      if (U.host) continue;
      for (int t = 0; t < U.nt; ++t) {
        if (U.tlen[t] == 0) continue;
        const int ti = U.tidx[t];
        char* dst = e->d_arena + B.base + U.slot_off[t];
        const bool packs = m.dtype == SWAPNET_BF16 && m.tensor_raw[ti] % kPkChunkBytes == 0 &&
                           U.toff[t] % kPkChunkBytes == 0 && U.tlen[t] % kPkChunkBytes == 0 &&
                           ((uintptr_t)dst & 15) == 0;
        if (!packs) {
          e->pk_rest[k].push_back(Segment{e->tensor_dev[ti] + U.toff[t], dst, U.tlen[t]});
          link += U.tlen[t];
          continue;
        }
        if (!e->packed[ti]) {
          int rc = acquire_packed(e, ti);
          if (rc) return rc;
        }
        const PackedImage* im = e->packed[ti];
        PkJob j;
        std::memset(&j, 0, sizeof(j));
        j.base = im->dev;
        j.dst = reinterpret_cast<uint16_t*>(dst);
        j.body_off = im->body_off;
        j.overflow_off = im->overflow_off;
        j.c0 = (uint32_t)(U.toff[t] / kPkChunkBytes);
        j.nchunks = (uint32_t)(U.tlen[t] / kPkChunkBytes);
        j.x0 = im->x0;
        bj.push_back(j);
        link += (uint64_t)j.nchunks * (kPkBody + kPkHeader) +
                (uint64_t)(im->raw_before[j.c0 + j.nchunks] - im->raw_before[j.c0]) * kPkChunkBytes;
      }
    }
    if (bj.empty()) {  // nothing packs: the block is copied as it is
      e->pk_rest[k].clear();
      EB.variant = zerocopy_ok(EB) ? SWAPNET_SWAP_ZEROCOPY : SWAPNET_SWAP_MEMCPY;
      continue;
    }
    for (const Segment& g : e->pk_rest[k])
      if (((uintptr_t)g.src | (uintptr_t)g.dst) & 15)
        SN_FAIL(SWAPNET_ERR_MISALIGNED, "packed swaps: an unpacked piece is not 16-byte aligned");
    for (size_t i = 0; i < bj.size(); i += 1024) {
      PkLaunch L{jobs.size(), (int)std::min<size_t>(1024, bj.size() - i), 0};
      for (int q = 0; q < L.njobs; ++q) {
        PkJob j = bj[i + q];
        j.first = L.chunks;
        L.chunks += j.nchunks;
        jobs.push_back(j);
      }
      e->pk_launch[k].push_back(L);
    }
    EB.variant = SWAPNET_SWAP_PACKED;
    e->link_bytes[k] = link;
  }
  if (!jobs.empty()) {
    if (cudaMalloc(&e->d_pkjobs, jobs.size() * sizeof(PkJob)) != cudaSuccess) {
      cudaGetLastError();
      e->d_pkjobs = nullptr;
      SN_FAIL(SWAPNET_ERR_OOM, "unpack job table allocation failed");
    }
    CU(cudaMemcpy(e->d_pkjobs, jobs.data(), jobs.size() * sizeof(PkJob), cudaMemcpyHostToDevice), "unpack jobs");
  }
  return SWAPNET_OK;
}

static int swap_block(swapnet_engine* e, size_t k, int variant, cudaStream_t s) {
  const EngBlock& b = e->blocks[k];
  if (variant == SWAPNET_SWAP_PACKED) {
    for (const PkLaunch& L : e->pk_launch[k]) {
      // one CTA per SM unless the options fix the swap kernels' CTA count
      const int ctas = e->plan.opt.zc_ctas > 0 ? e->plan.opt.zc_ctas : e->num_sms;
      int rc = launch_unpack(e->d_pkjobs + L.first, L.njobs, L.chunks, ctas, s);
      if (rc) return rc;
    }
    std::vector<ZcSeg> z;
    for (const Segment& g : e->pk_rest[k]) z.push_back(ZcSeg{g.src, g.dst, g.bytes});
    return launch_zerocopy(z.data(), (int)z.size(), e->zc_ctas, s);
  }
  if (variant == SWAPNET_SWAP_ZEROCOPY) {
    std::vector<ZcSeg> z;
    z.reserve(b.segs.size());
    for (const Segment& g : b.segs) z.push_back(ZcSeg{g.src, g.dst, g.bytes});
    return launch_zerocopy(z.data(), (int)z.size(), e->zc_ctas, s);
  }
  for (const Segment& g : b.segs) CU(cudaMemcpyAsync(g.dst, g.src, g.bytes, cudaMemcpyDefault, s), "swap-in copy");
  return SWAPNET_OK;
}

static bool wants_tc(const Model& m, const Layer& L);
static bool small_conv_ok(const Model& m, const Layer& L);

// A block runs without a swap-in (SWAPNET_SWAP_DIRECT) when every unit
// with parameters runs a SIMT kernel, which takes plain 16-byte global loads
// that reach mapped host memory as well as the arena; tensor-core units read
// their weights by TMA from device memory and keep the swap.
static bool direct_ok(const swapnet_engine* e, size_t k) {
  const swapnet_plan& p = e->plan;
  const Block& B = p.blocks[k];
  for (int u = B.u0; u < B.u1; ++u) {
    const Unit& U = p.units[u];
    if (U.host) continue;
    const Layer& L = p.model.L[U.layer];
    if (U.nt > 0 && (wants_tc(p.model, L) || small_conv_ok(p.model, L))) return false;
    for (int t = 0; t < U.nt; ++t)
      if ((uintptr_t)(e->tensor_dev[U.tidx[t]] + U.toff[t]) & 15) return false;
  }
  return true;
}

static bool zerocopy_ok(const EngBlock& b) {
  for (const Segment& g : b.segs)
    if (((uintptr_t)g.src | (uintptr_t)g.dst) & 15) return false;
  return true;
}

// Time both swap variants per block (best of 3 each) and keep the faster
// (the zero-copy kernel on a near tie).
static int calibrate(swapnet_engine* e) {
  cudaEvent_t a, b;
  CU(cudaEventCreate(&a), "event");
  CU(cudaEventCreate(&b), "event");
  int rc = SWAPNET_OK;
  for (size_t k = 0; k < e->blocks.size() && rc == SWAPNET_OK; ++k) {
    EngBlock& B = e->blocks[k];
    if (e->plan.blocks[k].slot < 0) continue;  // resident prefix: never swapped
    float best[3] = {1e30f, 1e30f, 1e30f};
    for (int v : {SWAPNET_SWAP_MEMCPY, SWAPNET_SWAP_ZEROCOPY}) {
      if (v == SWAPNET_SWAP_ZEROCOPY && !zerocopy_ok(B)) continue;
      for (int rep = 0; rep < 3 && rc == SWAPNET_OK; ++rep) {
        cudaEventRecord(a, e->copy);
        rc = swap_block(e, k, v, e->copy);
        cudaEventRecord(b, e->copy);
        if (cudaEventSynchronize(b) != cudaSuccess) { rc = SWAPNET_ERR_CUDA; break; }
        float ms = 0;
        cudaEventElapsedTime(&ms, a, b);
        best[v] = std::min(best[v], ms * 1000.f);
      }
    }
    B.memcpy_us = best[SWAPNET_SWAP_MEMCPY];
    B.zerocopy_us = best[SWAPNET_SWAP_ZEROCOPY] < 1e29f ? best[SWAPNET_SWAP_ZEROCOPY] : 0.f;
    // SM loads win ties (within 3 %): on multi-GB blocks both reach the link
    // rate, but copy-engine transfers were measured to stall now and then
    // (single decode passes of the 7B model taking 2x) while SM loads did not
    B.variant = (B.zerocopy_us > 0.f && B.zerocopy_us <= 1.03f * B.memcpy_us) ? SWAPNET_SWAP_ZEROCOPY
                                                                             : SWAPNET_SWAP_MEMCPY;
  }
  cudaEventDestroy(a);
  cudaEventDestroy(b);
  return rc;
}

static int capture(swapnet_engine* e, const void* din, void* dout, cudaGraphExec_t* out);

// Second stage of the AUTO choice.  The first stage times each block's copy
// alone; inside the pipeline a zero-copy swap shares the SMs with the layers
// while a copy-engine swap does not, and their start-up latencies differ.
// So whole inferences (CUDA graph replays on scratch input and output
// buffers) are timed with the per-block choice, with every block on the copy
// engine and with every block zero-copy, and the fastest assignment is kept.
// Unless the options fix the zero-copy kernel's CTA count, every-block
// zero-copy is also timed with 24 and 16 CTAs: fewer CTAs leave more SMs to
// the layers while still keeping ahead of them (measured on ResNet-50 and
// YOLOv3: 1-2 % faster inferences than 32).
// Decoder models (which need a bound state) are not timed whole: their
// blocks all take the zero-copy kernel when every block allows it.  Their
// prefill and decode engines read the same multi-GB host weights, and on
// the GB300 machine copy-engine reads of a 13 GB page-locked region that SM
// loads had just read ran about 9x below the link rate (a prefill pass of
// the 7B decoder at 120 instead of 63 ms when one of its nine blocks took
// the copy engine after decode passes on the zero-copy kernel), while SM
// loads keep the link rate in every order.
static int calibrate_in_situ(swapnet_engine* e) {
  const Model& m = e->plan.model;
  if (e->blocks.empty()) return SWAPNET_OK;
  if (m.has_attention) {
    bool zc_all = true;
    for (size_t k = 0; k < e->blocks.size(); ++k)
      zc_all = zc_all && (e->plan.blocks[k].slot < 0 || zerocopy_ok(e->blocks[k]));
    if (zc_all)
      for (EngBlock& b : e->blocks) b.variant = SWAPNET_SWAP_ZEROCOPY;
    return SWAPNET_OK;
  }
  void* din = nullptr;
  void* dout = nullptr;
  if (cudaMalloc(&din, align_up(m.in_bytes)) != cudaSuccess ||
      cudaMalloc(&dout, align_up(m.out_bytes)) != cudaSuccess) {
    cudaGetLastError();
    if (din) cudaFree(din);
    return SWAPNET_OK;  // no room for scratch buffers: keep the per-block choice
  }
  cudaMemset(din, 0, align_up(m.in_bytes));
  std::vector<std::vector<int>> cand(1);
  std::vector<int> ctas(1, e->zc_ctas);  // zero-copy CTAs of each candidate
  for (const EngBlock& b : e->blocks) cand[0].push_back(b.variant);
  cand.push_back(std::vector<int>(e->blocks.size(), SWAPNET_SWAP_MEMCPY));
  ctas.push_back(e->zc_ctas);
  bool zc_all = true;
  for (size_t k = 0; k < e->blocks.size(); ++k)
    zc_all = zc_all && (e->plan.blocks[k].slot < 0 || zerocopy_ok(e->blocks[k]));
  if (zc_all) {
    std::vector<int> n_ctas{e->zc_ctas};
    if (e->plan.opt.zc_ctas == 0) n_ctas = {e->zc_ctas, 24, 16};
    for (int c : n_ctas) {
      cand.push_back(std::vector<int>(e->blocks.size(), SWAPNET_SWAP_ZEROCOPY));
      ctas.push_back(c);
    }
  }
  cudaEvent_t a = nullptr, b = nullptr;
  int rc = SWAPNET_OK;
  if (cudaEventCreate(&a) != cudaSuccess || cudaEventCreate(&b) != cudaSuccess) rc = SWAPNET_ERR_CUDA;
  float best = 1e30f;
  size_t best_i = 0;
  const int zc0 = e->zc_ctas;
  for (size_t c = 0; c < cand.size() && rc == SWAPNET_OK; ++c) {
    for (size_t k = 0; k < e->blocks.size(); ++k) e->blocks[k].variant = cand[c][k];
    e->zc_ctas = ctas[c];
    cudaGraphExec_t ge = nullptr;
    rc = capture(e, din, dout, &ge);
    if (rc) break;
    std::vector<float> t;
    for (int rep = 0; rep < 7 && rc == SWAPNET_OK; ++rep) {
      cudaEventRecord(a, e->cap);
      if (cudaGraphLaunch(ge, e->cap) != cudaSuccess) rc = SWAPNET_ERR_CUDA;
      cudaEventRecord(b, e->cap);
      if (cudaEventSynchronize(b) != cudaSuccess) rc = SWAPNET_ERR_CUDA;
      float ms = 0.f;
      cudaEventElapsedTime(&ms, a, b);
      if (rep >= 2) t.push_back(ms);  // two warm-up replays
    }
    cudaGraphExecDestroy(ge);
    if (rc) break;
    std::sort(t.begin(), t.end());
    const float med = t[t.size() / 2];
    if (med < best * 0.98f) {  // prefer the earlier candidate unless clearly faster
      best = med;
      best_i = c;
    }
  }
  if (rc == SWAPNET_OK) {
    for (size_t k = 0; k < e->blocks.size(); ++k) e->blocks[k].variant = cand[best_i][k];
    e->zc_ctas = ctas[best_i];
  } else {
    e->zc_ctas = zc0;
    set_error("swap variant calibration failed");
  }
  if (a) cudaEventDestroy(a);
  if (b) cudaEventDestroy(b);
  cudaFree(din);
  cudaFree(dout);
  return rc;
}

static const char* act_ptr(const swapnet_engine* e, int src, const void* din, const void* dout) {
  if (src == SWAPNET_SRC_INPUT) return static_cast<const char*>(din);
  const Layer& L = e->plan.model.L[src];
  if (L.out_off >= 0) return static_cast<const char*>(dout) + L.out_off;
  return e->d_ws + L.ws_off;
}

static char* out_ptr(const swapnet_engine* e, int li, void* dout) {
  const Layer& L = e->plan.model.L[li];
  if (L.out_off >= 0) return static_cast<char*>(dout) + L.out_off;
  return e->d_ws + L.ws_off;
}

// Fill the GEMM description of a unit for the given activation pointers.
static bool unit_gemm(const swapnet_engine* e, const Unit& U, const UnitExec& X, const char* x, const char* r,
                      char* y, TcGemm* g) {
  const Model& m = e->plan.model;
  const Layer& L = m.L[U.layer];
  const int es = m.es;
  std::memset(g, 0, sizeof(*g));
  g->dtype = m.dtype;
  g->num_sms = e->num_sms;
  g->cluster_max = e->plan.opt.split_cap > 0 ? std::min(16, (int)e->plan.opt.split_cap) : 16;
  g->allow_persist = 1;
  g->W = X.w;
  g->e.bias = X.b;
  g->e.act = L.d.act;
  g->e.res_post = L.d.res_post;
  if (L.d.op == SWAPNET_OP_LINEAR) {
    g->M = L.n; g->N = U.rows; g->K = L.d.cin;
    g->N_layer = L.d.cout;
    g->A = x; g->lda = L.d.cin; g->conv = 0;
    g->y = y + (int64_t)U.row0 * es; g->ldy = L.d.cout;
    g->e.res = r ? r + (int64_t)U.row0 * es : nullptr; g->e.ldr = L.d.cout;
    return true;
  }
  // conv
  g->N = L.d.cout;
  g->K = L.d.kh * L.d.kw * L.d.cin;
  g->M = L.on * L.oh * L.ow;
  g->y = y; g->ldy = L.d.cout;
  g->e.res = r; g->e.ldr = L.d.cout;
  g->A = x;
  const bool pointwise = L.d.kh == 1 && L.d.kw == 1 && L.d.stride == 1 && L.d.pad == 0;
  g->conv = pointwise ? 0 : 1;
  g->lda = L.d.cin;
  g->H = L.h; g->Wd = L.w; g->C = L.d.cin; g->Ho = L.oh; g->Wo = L.ow;
  g->kh = L.d.kh; g->kw = L.d.kw; g->stride = L.d.stride; g->pad = L.d.pad;
  return true;
}

static bool skinny_ok(const Model& m, const Layer& L) {
  return L.n <= 16 && ((uint64_t)L.d.cin * m.es) % 16 == 0;
}

// Rows above which a linear layer goes to the tensor cores: the SIMT GEMV
// does 2 * rows FLOPs per weight byte, which outruns HBM only for a few rows
// (fp32 FMA rate / HBM bandwidth ~ 6 FLOP/byte on this part).
constexpr int kSkinnyMaxRows = 4;

static bool wants_tc(const Model& m, const Layer& L) {
  if (m.dtype == SWAPNET_F32) return false;
  if (L.d.op == SWAPNET_OP_LINEAR) return L.n > kSkinnyMaxRows && L.d.cin % 8 == 0;
  if (L.d.op == SWAPNET_OP_CONV2D) return L.d.cin % 8 == 0;
  return false;
}

static bool small_conv_ok(const Model& m, const Layer& L) {
  return L.d.op == SWAPNET_OP_CONV2D && L.d.cin % 8 != 0 &&
         tc_small_supported(m.dtype, L.d.kh * L.d.kw * L.d.cin);
}

static int plan_side(swapnet_engine* e);

// A whole (unsplit) linear layer on the GEMV kernel, its weights in the arena
// or read in place.
static bool whole_skinny(const swapnet_engine* e, int u) {
  const Unit& U = e->plan.units[u];
  return e->unit_kind[u] == SWAPNET_KERNEL_SKINNY && !U.host && U.row0 == 0 &&
         U.rows == e->plan.model.L[U.layer].d.cout;
}

// Merged GEMV launches (option merge): inside one block, consecutive whole
// GEMV layers that read the same input with the same K and rows run as one
// launch: up to kSkMaxSeg siblings none of which reads another's output
// (e.g. the q, k, v projections), or a pair whose second layer takes the
// first's output as its residual and nothing else of it (e.g. gate and up
// of a SwiGLU feed-forward).  Results are bit-identical to separate
// launches.
static void plan_merges(swapnet_engine* e) {
  const swapnet_plan& p = e->plan;
  const Model& m = p.model;
  const int n = (int)p.units.size();
  e->merge_n.assign(n, 0);
  e->merge_pair.assign(n, 0);
  e->merged_into.assign(n, 0);
  if (!p.opt.merge) return;
  for (const Block& B : p.blocks) {
    for (int u = B.u0; u < B.u1; ++u) {
      if (!whole_skinny(e, u)) continue;
      const Layer& L0 = m.L[p.units[u].layer];
      auto same_input = [&](int v) {
        const Layer& L = m.L[p.units[v].layer];
        return v < B.u1 && whole_skinny(e, v) && L.d.src0 == L0.d.src0 && L.d.cin == L0.d.cin && L.n == L0.n;
      };
      if (same_input(u + 1)) {
        const Layer& L1 = m.L[p.units[u + 1].layer];
        if (L1.d.res == p.units[u].layer && L1.d.cout == L0.d.cout) {
          e->merge_n[u] = 1;
          e->merge_pair[u] = 1;
          e->merged_into[u + 1] = 1;
          ++u;
          continue;
        }
      }
      int k = 1;
      for (; k < kSkMaxSeg && same_input(u + k); ++k) {
        const Layer& L = m.L[p.units[u + k].layer];
        bool reads_group = false;
        for (int i = 0; i < k; ++i) {
          const int li = p.units[u + i].layer;
          reads_group = reads_group || L.d.res == li || L.d.src0 == li;
        }
        if (reads_group) break;
      }
      if (k == 1) continue;
      e->merge_n[u] = k - 1;
      for (int i = 1; i < k; ++i) e->merged_into[u + i] = 1;
      u += k - 1;
    }
  }
}

// Launch unit u with the merge_n[u] units after it as one GEMV launch.
static int run_group(swapnet_engine* e, int u, const void* din, void* dout, cudaStream_t s) {
  const swapnet_plan& p = e->plan;
  const Model& m = p.model;
  const Layer& L0 = m.L[p.units[u].layer];
  SkJob j{};
  j.x = act_ptr(e, L0.d.src0, din, dout);
  j.M = L0.n;
  j.K = L0.d.cin;
  j.nseg = 1 + e->merge_n[u];
  j.pair = e->merge_pair[u];
  for (int i = 0; i < j.nseg; ++i) {
    const int v = u + i;
    const Layer& L = m.L[p.units[v].layer];
    const UnitExec& X = e->ux[v];
    const char* r = L.d.res == SWAPNET_SRC_NONE ? nullptr : act_ptr(e, L.d.res, din, dout);
    j.seg[i] = SkSeg{X.w, Epi{X.b, r, L.d.cout, L.d.act, L.d.res_post}, L.d.cout,
                     out_ptr(e, p.units[v].layer, dout), L.d.cout};
  }
  j.device_weights = 1;
  for (int i = 0; i < j.nseg; ++i)
    if (e->ux[u + i].in_place) j.device_weights = 0;
  j.num_sms = e->num_sms;
  j.err = e->err_word;
  return launch_linear_skinny_job(m.dtype, j, s);
}

static int prepare_units(swapnet_engine* e) {
  const swapnet_plan& p = e->plan;
  const Model& m = p.model;
  e->ux.assign(p.units.size(), UnitExec{});
  e->unit_kind.assign(p.units.size(), 0);
  for (size_t u = 0; u < p.units.size(); ++u) {
    const Layer& L = m.L[p.units[u].layer];
    int k = 0;
    switch (L.d.op) {
      case SWAPNET_OP_LINEAR:
        k = wants_tc(m, L) ? SWAPNET_KERNEL_TC_GEMM : skinny_ok(m, L) ? SWAPNET_KERNEL_SKINNY : SWAPNET_KERNEL_TILED;
        break;
      case SWAPNET_OP_CONV2D:
        if (!wants_tc(m, L))
          k = small_conv_ok(m, L) ? SWAPNET_KERNEL_TC_CONV_SMALL : SWAPNET_KERNEL_DIRECT_CONV;
        else if (L.d.kh == 1 && L.d.kw == 1 && L.d.stride == 1 && L.d.pad == 0) k = SWAPNET_KERNEL_TC_GEMM;
        else k = SWAPNET_KERNEL_TC_CONV;
        break;
      case SWAPNET_OP_MAXPOOL: k = SWAPNET_KERNEL_MAXPOOL; break;
      case SWAPNET_OP_GAP: k = SWAPNET_KERNEL_GAP; break;
      case SWAPNET_OP_UPSAMPLE2X: k = SWAPNET_KERNEL_UPSAMPLE; break;
      case SWAPNET_OP_CONCAT: k = SWAPNET_KERNEL_CONCAT; break;
      case SWAPNET_OP_EMBED: k = SWAPNET_KERNEL_EMBED; break;
      case SWAPNET_OP_RMSNORM: k = SWAPNET_KERNEL_RMSNORM; break;
      case SWAPNET_OP_ATTENTION: k = SWAPNET_KERNEL_ATTENTION; break;
      case SWAPNET_OP_ARGMAX: k = SWAPNET_KERNEL_ARGMAX; break;
    }
    e->unit_kind[u] = k;
  }
  for (const Block& B : p.blocks) {
    char* base = block_base(e, B);
    for (int u = B.u0; u < B.u1; ++u) {
      const Unit& U = p.units[u];
      UnitExec& X = e->ux[u];
      if (U.host) {
        X.w = e->tensor_dev[U.tidx[0]];  // device alias of the page-locked host table
        X.in_place = true;
      } else if (e->blocks[&B - p.blocks.data()].variant == SWAPNET_SWAP_DIRECT) {
        // read in place in page-locked host memory (device aliases)
        if (U.nt >= 1) X.w = e->tensor_dev[U.tidx[0]] + U.toff[0];
        if (U.nt == 2) X.b = e->tensor_dev[U.tidx[1]] + U.toff[1];
        X.in_place = true;
      } else {
        if (U.nt >= 1) X.w = base + U.slot_off[0];
        if (U.nt == 2) X.b = base + U.slot_off[1];
      }
      const Layer& L = m.L[U.layer];
      if (small_conv_ok(m, L)) {
        int rc = tc_small_prepare(m.dtype, L.d.kh * L.d.kw * L.d.cin);
        if (rc) return rc;
      }
      if (!wants_tc(m, L)) continue;
      X.use_tc = true;
      // A pointers in the workspace are fixed; the model input and outputs
      // are bound per call (the map is re-encoded when they change).
      const char* x = (L.d.src0 == SWAPNET_SRC_INPUT || m.L[L.d.src0].out_off >= 0)
                          ? nullptr
                          : act_ptr(e, L.d.src0, nullptr, nullptr);
      TcGemm g;
      unit_gemm(e, U, X, x, nullptr, nullptr, &g);
      if (!g.conv && !x) g.A = nullptr;
      int rc = tc_prepare(g, &X.tc);
      if (rc) return rc;
      X.tmA_for = g.A;
    }
  }
  plan_merges(e);
  return SWAPNET_OK;
}

static int run_unit(swapnet_engine* e, int u, const void* din, void* dout, cudaStream_t s) {
  const swapnet_plan& p = e->plan;
  const Model& m = p.model;
  const Unit& U = p.units[u];
  UnitExec& X = e->ux[u];
  const Layer& L = m.L[U.layer];
  const char* x = act_ptr(e, L.d.src0, din, dout);
  const char* r = L.d.res == SWAPNET_SRC_NONE ? nullptr : act_ptr(e, L.d.res, din, dout);
  char* y = out_ptr(e, U.layer, dout);
  const int es = m.es;
  switch (L.d.op) {
    case SWAPNET_OP_LINEAR:
    case SWAPNET_OP_CONV2D: {
      if (X.use_tc) {
        TcGemm g;
        unit_gemm(e, U, X, x, r, y, &g);
        if ((!g.conv || X.tc.tma_conv) && g.A != X.tmA_for) {
          int rc = tc_prepare(g, &X.tc);
          if (rc) return rc;
          X.tmA_for = g.A;
        }
        if (X.tc.splits > 1) {
          g.counters = reinterpret_cast<int*>(e->d_splitk);
          g.partial = reinterpret_cast<float*>(e->d_splitk + e->splitk_counter_bytes);
        }
        return launch_tc_gemm(g, X.tc, e->err_word, s);
      }
      Epi ep{X.b, nullptr, L.d.cout, L.d.act, L.d.res_post};
      if (L.d.op == SWAPNET_OP_LINEAR) {
        ep.res = r ? r + (int64_t)U.row0 * es : nullptr;
        if (skinny_ok(m, L))
          return launch_linear_skinny(m.dtype, x, L.n, L.d.cin, X.w, U.rows, ep, y + (int64_t)U.row0 * es,
                                      L.d.cout, s, X.in_place ? 0 : 1, e->num_sms, e->err_word);
        return launch_linear_tiled(m.dtype, x, L.n, L.d.cin, X.w, U.rows, ep, y + (int64_t)U.row0 * es, L.d.cout,
                                   s);
      }
      ep.res = r;
      if (small_conv_ok(m, L)) {
        TcSmallConv g;
        g.dtype = m.dtype; g.x = x; g.W = X.w;
        g.M = L.on * L.oh * L.ow; g.N = L.d.cout; g.K = L.d.kh * L.d.kw * L.d.cin;
        g.H = L.h; g.Wd = L.w; g.C = L.d.cin; g.Ho = L.oh; g.Wo = L.ow;
        g.kh = L.d.kh; g.kw = L.d.kw; g.stride = L.d.stride; g.pad = L.d.pad;
        g.e = ep; g.y = y; g.ldy = L.d.cout; g.num_sms = e->num_sms;
        return launch_tc_conv_small(g, e->err_word, s);
      }
      return launch_conv_direct(m.dtype, x, L.n, L.h, L.w, L.d.cin, X.w, L.d.cout, L.d.kh, L.d.kw, L.d.stride,
                                L.d.pad, L.oh, L.ow, ep, y, s);
    }
    case SWAPNET_OP_MAXPOOL:
      return launch_maxpool(m.dtype, x, L.n, L.h, L.w, L.c, L.d.kh, L.d.kw, L.d.stride, L.d.pad, L.oh, L.ow, y, s);
    case SWAPNET_OP_GAP:
      return launch_gap(m.dtype, x, L.n, L.h, L.w, L.c, y, s);
    case SWAPNET_OP_UPSAMPLE2X:
      return launch_upsample2x(m.dtype, x, L.n, L.h, L.w, L.c, y, s);
    case SWAPNET_OP_CONCAT:
      return launch_concat(m.dtype, x, L.c, act_ptr(e, L.d.src1, din, dout), L.c1, (int64_t)L.n * L.h * L.w, y, s);
    case SWAPNET_OP_EMBED:
      return launch_embed(m.dtype, X.w, reinterpret_cast<const int*>(x), L.on, L.d.cin, L.d.cout, y, e->err_word, s);
    case SWAPNET_OP_RMSNORM:
      return launch_rmsnorm(m.dtype, x, X.w, L.n, L.c, L.d.eps, y, s);
    case SWAPNET_OP_ATTENTION: {
      if (!e->d_state) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "decoder state not bound (swapnet_engine_bind_state)");
      char* kc = e->d_state + L.state_off;
      char* vc = kc + align_up((uint64_t)L.d.max_seq * L.c * es);
      return launch_attention(m.dtype, const_cast<char*>(x), act_ptr(e, L.d.src1, din, dout),
                              act_ptr(e, L.d.src2, din, dout), kc, vc, reinterpret_cast<const int*>(e->d_state),
                              L.n, L.d.heads, L.c, L.d.theta, L.d.max_seq, y, e->err_word, s);
    }
    case SWAPNET_OP_ARGMAX:
      return launch_argmax(m.dtype, x, L.n, L.c1, reinterpret_cast<int*>(y), s);
    default:
      SN_FAIL(SWAPNET_ERR_INVALID_ARG, "unknown op");
  }
}

// Everything an engine derives from its plan: arena (allocated when the
// engine owns it), copy segments, unit pointers and TMA descriptors, side
// branches, split-K scratch, the resident upload or prefix upload, and the
// swap variants.  Used by swapnet_load and again by swapnet_engine_adapt.
static bool prefetch_on(const swapnet_engine* e);

static int bind_plan(swapnet_engine* e, void* d_arena_user, uint64_t arena_bytes_user, bool preloaded_arena) {
  const swapnet_plan* plan = &e->plan;
  e->zc_ctas = plan->opt.zc_ctas > 0 ? plan->opt.zc_ctas : 32;  // the AUTO choice may lower it
  const uint64_t arena_need = plan->prefix_bytes + plan->region;  // resident prefix, then the swap region
  if (d_arena_user && arena_bytes_user < arena_need) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "arena buffer too small");
  for (const Block& B : plan->blocks)  // every block lies inside the arena
    if (B.base + B.bytes > arena_need) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "plan places a block outside the arena");
  if (d_arena_user) {
    e->d_arena = static_cast<char*>(d_arena_user);
    e->arena_bytes = arena_bytes_user;
  } else if (!e->own_arena || e->arena_bytes != std::max<uint64_t>(arena_need, kAlign)) {
    if (e->own_arena && e->d_arena) cudaFree(e->d_arena);  // a new budget: give the old arena back
    e->d_arena = nullptr;
    e->own_arena = false;
    if (injected(2)) SN_FAIL(SWAPNET_ERR_OOM, "arena allocation failed (injected)");
    const uint64_t bytes = std::max<uint64_t>(arena_need, kAlign);
    if (cudaMalloc(&e->d_arena, bytes) != cudaSuccess) {
      cudaGetLastError();
      e->d_arena = nullptr;
      SN_FAIL(SWAPNET_ERR_OOM, "arena allocation failed");
    }
    e->own_arena = true;
    e->arena_bytes = bytes;
    // touch every page now, so that the first inference does not pay for
    // the driver backing fresh allocations
    CU(cudaMemset(e->d_arena, 0, bytes), "arena first touch");
  }
  int rc = build_segments(e);
  if (rc) return rc;
  if (!plan->resident && !e->file && plan->opt.swap_variant == SWAPNET_SWAP_DIRECT)
    for (size_t k = 0; k < e->blocks.size(); ++k)
      if (plan->blocks[k].slot >= 0 && direct_ok(e, k)) e->blocks[k].variant = SWAPNET_SWAP_DIRECT;
  rc = prepare_units(e);
  if (rc) return rc;
  rc = plan_side(e);
  if (rc) return rc;
  {
    uint64_t part = 0;
    int64_t tiles = 0;
    for (const UnitExec& X : e->ux)
      if (X.use_tc && X.tc.splits > 1) {
        part = std::max(part, X.tc.scratch_bytes);
        tiles = std::max(tiles, X.tc.tiles);
      }
    if (part) {
      e->splitk_counter_bytes = align_up((uint64_t)tiles * sizeof(int));
      e->splitk_bytes = e->splitk_counter_bytes + part;
      if (injected(2) || cudaMalloc(&e->d_splitk, e->splitk_bytes) != cudaSuccess) {
        cudaGetLastError();
        e->d_splitk = nullptr;
        SN_FAIL(SWAPNET_ERR_OOM, "split-K scratch allocation failed");
      }
      CU(cudaMemset(e->d_splitk, 0, e->splitk_counter_bytes), "split-K counters");
    }
  }
  const int variant = (plan->opt.pageable && plan->opt.swap_variant == SWAPNET_SWAP_AUTO) ? SWAPNET_SWAP_MEMCPY
                                                                                        : plan->opt.swap_variant;
  if (plan->resident) {
    if (!preloaded_arena) {
      for (size_t k = 0; k < e->blocks.size() && !rc; ++k)
        rc = e->file ? upload_file_block(e, k, nullptr) : swap_block(e, k, SWAPNET_SWAP_MEMCPY, e->copy);
      if (rc) return rc;
      CU(cudaStreamSynchronize(e->copy), "resident upload");
    }
    e->weights_loaded = true;
  } else if (plan->prefix_units > 0 && !plan->blocks.empty() && plan->blocks[0].slot < 0) {
    // resident prefix: uploaded once, then only the other blocks are swapped
    rc = e->file ? upload_file_block(e, 0, nullptr) : swap_block(e, 0, SWAPNET_SWAP_MEMCPY, e->copy);
    if (rc) return rc;
    CU(cudaStreamSynchronize(e->copy), "prefix upload");
  }
  if (e->file) {
    if (!plan->resident) {
      rc = calibrate_file(e);
      if (rc) return rc;
      if (prefetch_on(e)) return upload_file_block(e, 0, nullptr);  // present for the first inference
    }
    return SWAPNET_OK;
  }
  if (!plan->resident && variant == SWAPNET_SWAP_AUTO) {
    rc = calibrate(e);
    if (rc) return rc;
    rc = calibrate_in_situ(e);
    if (rc) return rc;
  } else if (!plan->resident && variant == SWAPNET_SWAP_PACKED) {
    for (EngBlock& b : e->blocks) b.variant = SWAPNET_SWAP_ZEROCOPY;  // until build_packed says otherwise
    rc = build_packed(e);
    if (rc) return rc;
  } else if (!plan->resident) {
    for (size_t k = 0; k < e->blocks.size(); ++k) {
      EngBlock& b = e->blocks[k];
      if (variant == SWAPNET_SWAP_DIRECT) {
        // the blocks direct_ok refused are copied by SM loads too: on the
        // GB300 machine, copy-engine reads of a large page-locked region right
        // after SM loads had read it ran about 9x slower (24 instead of
        // 210 GB/s over the 13.2 GB of the 7B decoder), while SM loads
        // after SM loads keep the link rate
        if (b.variant != SWAPNET_SWAP_DIRECT) b.variant = zerocopy_ok(b) ? SWAPNET_SWAP_ZEROCOPY : SWAPNET_SWAP_MEMCPY;
        continue;
      }
      b.variant = variant;
      if (plan->blocks[k].slot >= 0 && variant == SWAPNET_SWAP_ZEROCOPY && !zerocopy_ok(b))
        SN_FAIL(SWAPNET_ERR_MISALIGNED, "zero-copy needs 16-byte aligned host tensors");
    }
  }
  if (prefetch_on(e)) {  // the first block is present for the first inference
    rc = swap_block(e, 0, e->blocks[0].variant, e->copy);
    if (rc) return rc;
    CU(cudaStreamSynchronize(e->copy), "first block upload");
  }
  return SWAPNET_OK;
}

// Drop what bind_plan derived from the previous plan (the arena stays
// allocated until bind_plan knows the new size).
static void unbind_plan(swapnet_engine* e) {
  for (auto& kv : e->graphs) cudaGraphExecDestroy(kv.second);
  e->graphs.clear();
  for (cudaEvent_t& ev : e->side_done)
    if (ev) cudaEventDestroy(ev);
  e->side_done.clear();
  for (cudaEvent_t ev : e->ev_unit) cudaEventDestroy(ev);
  for (cudaEvent_t ev : e->ev_swap) cudaEventDestroy(ev);
  for (cudaEvent_t ev : e->ev_gswap) cudaEventDestroy(ev);
  for (cudaEvent_t ev : e->ev_gexec) cudaEventDestroy(ev);
  e->ev_unit.clear();
  e->ev_swap.clear();
  e->ev_gswap.clear();
  e->ev_gexec.clear();
  if (e->d_pkjobs) cudaFree(e->d_pkjobs);
  e->d_pkjobs = nullptr;
  e->pk_launch.clear();
  e->pk_rest.clear();
  if (e->d_splitk) cudaFree(e->d_splitk);
  e->d_splitk = nullptr;
  e->splitk_bytes = e->splitk_counter_bytes = 0;
  e->weights_loaded = false;
}

// swapnet_load and swapnet_load_file: parameters from host memory
// (host_weights) or from a weights file (file).
static int load_engine(const swapnet_plan* plan, const void* const* host_weights, uint32_t n_tensors,
                       swapnet_weights_file* file, void* d_arena, uint64_t arena_bytes, void* d_workspace,
                       uint64_t workspace_bytes, swapnet_engine** out) {
  if ((int)n_tensors != plan->model.n_tensors)
    SN_FAIL(SWAPNET_ERR_INVALID_ARG, "expected " + std::to_string(plan->model.n_tensors) + " tensors, got " +
                                         std::to_string(n_tensors));
  if (((uintptr_t)d_arena | (uintptr_t)d_workspace) % kAlign)
    SN_FAIL(SWAPNET_ERR_MISALIGNED, "device buffers must be 256-byte aligned");
  if (d_workspace && workspace_bytes < plan->model.ws_bytes)
    SN_FAIL(SWAPNET_ERR_INVALID_ARG, "workspace buffer too small");
  swapnet_engine* e = new (std::nothrow) swapnet_engine();
  if (!e) SN_FAIL(SWAPNET_ERR_OOM, "host allocation failed");
  std::unique_ptr<swapnet_engine, int (*)(swapnet_engine*)> guard(e, release);
  try {
    e->plan = *plan;
  } catch (const std::bad_alloc&) {
    SN_FAIL(SWAPNET_ERR_OOM, "host allocation failed");
  }
  CU(cudaGetDevice(&e->device), "cudaGetDevice");
  CU(cudaDeviceGetAttribute(&e->num_sms, cudaDevAttrMultiProcessorCount, e->device), "device attribute");
  e->zc_ctas = plan->opt.zc_ctas > 0 ? plan->opt.zc_ctas : 32;
  int rc = tc_error_word(&e->err_word);
  if (rc) return rc;
  if (d_workspace || plan->model.ws_bytes == 0) {
    e->d_ws = static_cast<char*>(d_workspace);
  } else {
    if (injected(2)) SN_FAIL(SWAPNET_ERR_OOM, "workspace allocation failed (injected)");
    if (cudaMalloc(&e->d_ws, plan->model.ws_bytes) != cudaSuccess) {
      cudaGetLastError();
      SN_FAIL(SWAPNET_ERR_OOM, "workspace allocation failed");
    }
    e->own_ws = true;
    CU(cudaMemset(e->d_ws, 0, plan->model.ws_bytes), "workspace first touch");
  }
  if (injected(3)) SN_FAIL(SWAPNET_ERR_CUDA, "stream creation failed (injected)");
  int lo = 0, hi = 0;
  CU(cudaDeviceGetStreamPriorityRange(&lo, &hi), "stream priority range");
  CU(cudaStreamCreateWithPriority(&e->copy, cudaStreamNonBlocking, hi), "copy stream");
  for (int s = 0; s < 2; ++s) {
    CU(cudaEventCreateWithFlags(&e->slot_free[s], cudaEventDisableTiming), "event");
    CU(cudaEventCreateWithFlags(&e->ready[s], cudaEventDisableTiming), "event");
  }
  CU(cudaStreamCreateWithFlags(&e->cap, cudaStreamNonBlocking), "capture stream");
  CU(cudaEventCreateWithFlags(&e->fork, cudaEventDisableTiming), "event");
  CU(cudaEventCreateWithFlags(&e->join, cudaEventDisableTiming), "event");
  if (file) {
    e->file = file;
    CU(cudaStreamCreateWithPriority(&e->rd, cudaStreamNonBlocking, hi), "read stream");
    for (int s = 0; s < 2; ++s) {
      CU(cudaEventCreateWithFlags(&e->staged[s], cudaEventDisableTiming), "event");
      CU(cudaEventCreateWithFlags(&e->stage_free[s], cudaEventDisableTiming), "event");
    }
  } else {
    rc = register_host(e, host_weights, n_tensors);
    if (rc) return rc;
  }
  rc = bind_plan(e, d_arena, arena_bytes, plan->resident && plan->opt.preloaded && d_arena);
  if (rc) return rc;
  e->stats = swapnet_engine_stats{};
  *out = guard.release();
  return SWAPNET_OK;
}

}  // namespace swapnet

extern "C" {

int swapnet_load(const swapnet_plan* plan, const void* const* host_weights, uint32_t n_tensors, void* d_arena,
                 uint64_t arena_bytes, void* d_workspace, uint64_t workspace_bytes, swapnet_engine** out) {
  return swapnet::guard_abi([&]() -> int {
    if (!plan || !out || (n_tensors && !host_weights)) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null argument");
    return swapnet::load_engine(plan, host_weights, n_tensors, nullptr, d_arena, arena_bytes, d_workspace,
                                workspace_bytes, out);
  });
}

int swapnet_load_file(const swapnet_plan* plan, swapnet_weights_file* file, void* d_arena, uint64_t arena_bytes,
                      void* d_workspace, uint64_t workspace_bytes, swapnet_engine** out) {
  return swapnet::guard_abi([&]() -> int {
    if (!plan || !file || !out) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null argument");
    return swapnet::load_engine(plan, nullptr, file->n, file, d_arena, arena_bytes, d_workspace, workspace_bytes,
                                out);
  });
}

int swapnet_engine_adapt(swapnet_engine* e, const swapnet_plan* plan) {
  return swapnet::guard_abi([&]() -> int {
    if (!e || !plan) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null argument");
    const Model& a = e->plan.model;
    const Model& b = plan->model;
    bool same = a.L.size() == b.L.size() && a.n_tensors == b.n_tensors && a.dtype == b.dtype &&
                a.weight_bytes == b.weight_bytes && a.in_bytes == b.in_bytes && a.ws_bytes == b.ws_bytes;
    for (size_t i = 0; same && i < a.L.size(); ++i)
      same = std::memcmp(&a.L[i].d, &b.L[i].d, sizeof(swapnet_layer)) == 0 ||
             (a.L[i].d.op == b.L[i].d.op && a.L[i].d.cin == b.L[i].d.cin && a.L[i].d.cout == b.L[i].d.cout &&
              a.L[i].tbytes[0] == b.L[i].tbytes[0] && a.L[i].tbytes[1] == b.L[i].tbytes[1]);
    if (!same) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "the plan is for a different model");
    if (plan->resident != e->plan.resident) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "cannot switch between resident and swapped plans");
    if (!e->file && plan->opt.pageable != e->plan.opt.pageable)
      SN_FAIL(SWAPNET_ERR_INVALID_ARG, "cannot switch between pageable and page-locked host weights");
    CU(cudaSetDevice(e->device), "cudaSetDevice");
    CU(cudaStreamSynchronize(e->copy), "drain copies");
    if (e->side) CU(cudaStreamSynchronize(e->side), "drain side stream");
    CU(cudaDeviceSynchronize(), "drain inferences");
    swapnet::unbind_plan(e);
    try {
      e->plan = *plan;
    } catch (const std::bad_alloc&) {
      SN_FAIL(SWAPNET_ERR_OOM, "host allocation failed");
    }
    // per-unit and per-block events were sized for the old plan: they are
    // made again for the new one after binding it (whose swap-variant
    // calibration captures inferences without them)
    const bool prof = e->profiling, st = e->swap_timing, tl = e->timeline;
    e->profiling = e->swap_timing = e->timeline = false;
    // an engine given a caller arena keeps it (the new plan must fit it)
    int rc = swapnet::bind_plan(e, e->own_arena ? nullptr : e->d_arena, e->own_arena ? 0 : e->arena_bytes, false);
    if (rc) return rc;
    if (prof) rc = swapnet_engine_set_profiling(e, 1);
    if (!rc && st) rc = swapnet_engine_set_swap_timing(e, 1);
    if (!rc && tl) rc = swapnet_engine_set_graph_timeline(e, 1);
    return rc;
  });
}

}  // extern "C"

namespace swapnet {

// Enqueue one inference: swaps on the copy stream, layers on `s`.
// Enqueue one inference: swaps on the copy stream, layers on `s`.  Each
// inference is self-contained: the copy stream forks from `s` (so swaps
// start after everything already queued on `s`, which also orders them
// after the previous inference's use of the slots), a slot's later reuse
// waits for the block that last used it in this inference, and the copy
// stream joins `s` again at the end.  The same sequence is captured as a
// graph, where the fork, the slot gating and the join become graph edges.
// Units that may run on the side stream: a whole-layer conv / linear unit
// whose layer may start early (Layer::start < layer), whose last producer's
// unit is on the main stream in the same block, and whose consumers are all
// in that block (they wait for it; the block's slot is released after them).
static int plan_side(swapnet_engine* e) {
  const swapnet_plan& p = e->plan;
  const Model& m = p.model;
  const int n = (int)p.units.size(), nl = (int)m.L.size();
  e->is_side.assign(n, 0);
  e->side_after.assign(n, {});
  e->side_wait.assign(n, {});
  e->side_done.assign(n, nullptr);
  if (!p.opt.branches) return SWAPNET_OK;
  std::vector<int> lfirst(nl, -1), llast(nl, -1), ublock(n, -1);
  for (size_t b = 0; b < p.blocks.size(); ++b)
    for (int u = p.blocks[b].u0; u < p.blocks[b].u1; ++u) ublock[u] = (int)b;
  for (int u = 0; u < n; ++u) {
    const int l = p.units[u].layer;
    if (lfirst[l] < 0) lfirst[l] = u;
    llast[l] = u;
  }
  auto reads = [&](const Layer& L, int l) {
    const swapnet_layer& d = L.d;
    return d.src0 == l || d.src1 == l || d.res == l || (d.op == SWAPNET_OP_ATTENTION && d.src2 == l);
  };
  for (int u = 0; u < n; ++u) {
    const Unit& U = p.units[u];
    const Layer& L = m.L[U.layer];
    if (L.start >= U.layer || U.host || lfirst[U.layer] != u || llast[U.layer] != u) continue;
    if (e->merge_n[u] || e->merged_into[u]) continue;  // one launch with its siblings
    const UnitExec& X = e->ux[u];
    if (X.use_tc && X.tc.splits > 1 && !X.tc.cluster) continue;  // global split-K scratch is shared
    const int du = llast[L.start - 1];
    if (du < 0 || ublock[du] != ublock[u] || e->is_side[du]) continue;
    bool ok = true;
    for (int s : {L.d.src0, L.d.src1, L.d.res})
      if (s >= 0 && e->is_side[llast[s]]) ok = false;
    std::vector<int> cons;
    for (int v = u + 1; v < n && ok; ++v)
      if (reads(m.L[p.units[v].layer], U.layer)) {
        if (ublock[v] != ublock[u] || e->is_side[v]) ok = false;
        cons.push_back(v);
      }
    if (!ok || cons.empty()) continue;
    e->is_side[u] = 1;
    e->side_after[du].push_back(u);
    for (int v : cons) e->side_wait[v].push_back(u);
    CU(cudaEventCreateWithFlags(&e->side_done[u], cudaEventDisableTiming), "event");
  }
  if (!e->side) {
    int lo = 0, hi = 0;
    CU(cudaDeviceGetStreamPriorityRange(&lo, &hi), "stream priority range");
    CU(cudaStreamCreateWithPriority(&e->side, cudaStreamNonBlocking, lo), "side stream");
    CU(cudaEventCreateWithFlags(&e->side_fork, cudaEventDisableTiming), "event");
  }
  return SWAPNET_OK;
}

// First-block prefetch is on for swapped plans made with option prefetch
// (the planner allows it only with two slots and no resident prefix).
// Block k is copied into its slot for every inference (not resident, not
// part of a resident prefix, not read in place in host memory).
static bool swapped(const swapnet_engine* e, size_t k) {
  return !e->plan.resident && e->plan.blocks[k].slot >= 0 &&
         (k >= e->blocks.size() || e->blocks[k].variant != SWAPNET_SWAP_DIRECT);
}

static bool prefetch_on(const swapnet_engine* e) {
  return e->plan.opt.prefetch && !e->plan.blocks.empty() && e->plan.blocks[0].slot == 0 && swapped(e, 0);
}

static int enqueue(swapnet_engine* e, const void* din, void* dout, cudaStream_t s, bool capturing = false) {
  const swapnet_plan& p = e->plan;
  const bool prof = e->profiling && !capturing;
  const bool pf = prefetch_on(e);
  bool used[2] = {false, false};
  bool stage_used[2] = {false, false};
  // in a captured graph an event-record node (external event), eagerly a
  // plain record
  const unsigned gflag = capturing ? cudaEventRecordExternal : cudaEventRecordDefault;
  const bool swap_ev = e->swap_timing || e->timeline;
  if (e->timeline) CU(cudaEventRecordWithFlags(e->ev_g0, s, gflag), "timeline event");
  if (!p.resident) {
    CU(cudaEventRecord(e->fork, s), "record fork");
    CU(cudaStreamWaitEvent(e->copy, e->fork, 0), "wait fork");
    if (e->file) CU(cudaStreamWaitEvent(e->rd, e->fork, 0), "wait fork");
  }
  // swap block k in once its place is free (the last block released in its
  // slot); gate_compute: the layers on `s` wait for it
  auto swap_in = [&](size_t k, bool gate_compute) -> int {
    const Block& B = p.blocks[k];
    const int j = (int)(k % 2);  // staging buffer of a file engine
    if (e->file) {
      // fetch into staging j once the copies of its previous block are done;
      // this overlaps the copy of the block before and the layers running
      if (stage_used[j]) CU(cudaStreamWaitEvent(e->rd, e->stage_free[j], 0), "wait staging");
      if (prof) CU(cudaEventRecord(e->ev_swap[2 * k], e->rd), "profile event");
      CU(cudaLaunchHostFunc(e->rd, read_block_host, &e->jobs[k]), "read host function");
      CU(cudaEventRecord(e->staged[j], e->rd), "record staged");
    }
    if (used[B.slot]) CU(cudaStreamWaitEvent(e->copy, e->slot_free[B.slot], 0), "wait slot");
    used[B.slot] = true;
    if (e->file) {
      CU(cudaStreamWaitEvent(e->copy, e->staged[j], 0), "wait staged");
    } else if (prof) {
      CU(cudaEventRecord(e->ev_swap[2 * k], e->copy), "profile event");
    }
    // the copy stream's own time for this swap
    if (swap_ev) CU(cudaEventRecordWithFlags(e->ev_gswap[2 * k], e->copy, gflag), "swap timing event");
    int rc = swap_block(e, k, e->blocks[k].variant, e->copy);
    if (rc) return rc;
    if (swap_ev) CU(cudaEventRecordWithFlags(e->ev_gswap[2 * k + 1], e->copy, gflag), "swap timing event");
    if (e->file) {
      CU(cudaEventRecord(e->stage_free[j], e->copy), "record staging free");
      stage_used[j] = true;
    }
    if (prof) CU(cudaEventRecord(e->ev_swap[2 * k + 1], e->copy), "profile event");
    if (gate_compute) {
      CU(cudaEventRecord(e->ready[B.slot], e->copy), "record ready");
      CU(cudaStreamWaitEvent(s, e->ready[B.slot], 0), "wait ready");
    }
    return SWAPNET_OK;
  };
  for (size_t k = 0; k < p.blocks.size(); ++k) {
    const Block& B = p.blocks[k];
    const bool swap_k = swapped(e, k);  // a resident prefix stays in the arena
    if (swap_k) {
      if (pf && k == 0) {
        used[B.slot] = true;  // swapped in at the end of the previous inference (or at load)
      } else {
        int rc = swap_in(k, true);
        if (rc) return rc;
      }
    }
    if (e->timeline) CU(cudaEventRecordWithFlags(e->ev_gexec[2 * k], s, gflag), "timeline event");
    for (int u = B.u0; u < B.u1; ++u) {
      if (e->is_side[u]) continue;  // launched on the side stream after its producer
      if (e->merged_into[u]) continue;  // launched with an earlier unit
      const int g1 = u + e->merge_n[u];  // last unit of this launch
      for (int v = u; v <= g1; ++v)
        for (int w : e->side_wait[v]) CU(cudaStreamWaitEvent(s, e->side_done[w], 0), "wait side");
      if (prof)
        for (int v = u; v <= g1; ++v) CU(cudaEventRecord(e->ev_unit[2 * v], s), "profile event");
      int rc = g1 > u ? run_group(e, u, din, dout, s) : run_unit(e, u, din, dout, s);
      if (rc) return rc;
      if (prof)
        for (int v = u; v <= g1; ++v) CU(cudaEventRecord(e->ev_unit[2 * v + 1], s), "profile event");
      for (int v = u; v <= g1; ++v) {
        for (int w : e->side_after[v]) {
          CU(cudaEventRecord(e->side_fork, s), "record side fork");
          CU(cudaStreamWaitEvent(e->side, e->side_fork, 0), "wait side fork");
          if (prof) CU(cudaEventRecord(e->ev_unit[2 * w], e->side), "profile event");
          rc = run_unit(e, w, din, dout, e->side);
          if (rc) return rc;
          if (prof) CU(cudaEventRecord(e->ev_unit[2 * w + 1], e->side), "profile event");
          CU(cudaEventRecord(e->side_done[w], e->side), "record side done");
        }
      }
    }
    if (e->timeline) CU(cudaEventRecordWithFlags(e->ev_gexec[2 * k + 1], s, gflag), "timeline event");
    if (swap_k) CU(cudaEventRecord(e->slot_free[B.slot], s), "record slot free");
  }
  if (p.model.has_attention) {
    if (!e->d_state) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "decoder state not bound (swapnet_engine_bind_state)");
    const Model& m = p.model;
    int rc = launch_advance(reinterpret_cast<int*>(e->d_state), m.in_n * m.in_h * m.in_w * m.in_c, s);
    if (rc) return rc;
  }
  if (pf) {
    // the next inference's first block, into its place once the last block
    // placed there has executed; overlaps this inference's last layers (the
    // plan keeps the last block clear of it)
    int rc = swap_in(0, false);
    if (rc) return rc;
  }
  if (!p.resident) {
    if (e->file) {  // the read stream's last fetch is waited for by the copy stream
      CU(cudaEventRecord(e->staged[0], e->rd), "record read join");
      CU(cudaStreamWaitEvent(e->copy, e->staged[0], 0), "wait read join");
    }
    CU(cudaEventRecord(e->join, e->copy), "record join");
    CU(cudaStreamWaitEvent(s, e->join, 0), "wait join");
  }
  return SWAPNET_OK;
}

static uint64_t launches_per_infer(const swapnet_engine* e) {
  uint64_t n = e->plan.units.size() + (e->plan.model.has_attention ? 1 : 0);
  for (int k : e->unit_kind) n += (k == SWAPNET_KERNEL_ATTENTION) ? 1 : 0;
  for (char c : e->merged_into) n -= c ? 1 : 0;
  if (!e->plan.resident)
    for (size_t k = 0; k < e->blocks.size(); ++k)
      if (e->plan.blocks[k].slot >= 0 && e->blocks[k].variant == SWAPNET_SWAP_ZEROCOPY)
        n += (e->blocks[k].segs.size() + 47) / 48;
      else if (e->plan.blocks[k].slot >= 0 && e->blocks[k].variant == SWAPNET_SWAP_PACKED)
        n += e->pk_launch[k].size() + (e->pk_rest[k].size() + 47) / 48;
  return n;
}

// Capture one inference for this binding as a graph: the capture starts on
// the engine's own stream, the copy stream joins through an event (fork) and
// rejoins at the end, so slot gating becomes graph edges.
static int capture(swapnet_engine* e, const void* din, void* dout, cudaGraphExec_t* out) {
  const swapnet_engine_stats saved = e->stats;
  CU(cudaStreamBeginCapture(e->cap, cudaStreamCaptureModeThreadLocal), "begin capture");
  cudaGraph_t g = nullptr;
  const int rc = enqueue(e, din, dout, e->cap, true);
  const cudaError_t ee = cudaStreamEndCapture(e->cap, &g);
  e->stats = saved;
  if (rc || ee != cudaSuccess || !g) {
    if (g) cudaGraphDestroy(g);
    cudaGetLastError();
    SN_FAIL(rc ? rc : SWAPNET_ERR_CUDA, "graph capture failed");
  }
  const cudaError_t ie = cudaGraphInstantiate(out, g, 0);
  cudaGraphDestroy(g);
  if (ie != cudaSuccess) {
    cudaGetLastError();
    SN_FAIL(SWAPNET_ERR_CUDA, std::string("graph instantiate: ") + cudaGetErrorString(ie));
  }
  return SWAPNET_OK;
}

}  // namespace swapnet

extern "C" {

int swapnet_infer(swapnet_engine* e, const void* din, void* dout, swapnet_stream stream) {
  return swapnet::guard_abi([&]() -> int {
    if (!e || !din || !dout) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null argument");
    if (((uintptr_t)din | (uintptr_t)dout) & 15) SN_FAIL(SWAPNET_ERR_MISALIGNED, "input/output must be 16-byte aligned");
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    CU(cudaSetDevice(e->device), "cudaSetDevice");
    // event timing needs eager launches; stream capture takes no copy from pageable memory
    if (e->plan.opt.graphs && !e->profiling && !(e->plan.opt.pageable && !e->file)) {
      const auto key = std::make_pair(std::make_pair(din, dout), (e->swap_timing ? 1 : 0) | (e->timeline ? 2 : 0));
      auto it = e->graphs.find(key);
      if (it == e->graphs.end()) {
        if (e->graphs.size() >= 8) {
          for (auto& kv : e->graphs) cudaGraphExecDestroy(kv.second);
          e->graphs.clear();
        }
        cudaGraphExec_t ge = nullptr;
        int rc = capture(e, din, dout, &ge);
        if (rc) return rc;
        it = e->graphs.emplace(key, ge).first;
      }
      CU(cudaGraphLaunch(it->second, s), "graph launch");
    } else {
      int rc = enqueue(e, din, dout, s);
      if (rc) return rc;
    }
    e->stats.kernel_launches += launches_per_infer(e);
    e->stats.infer_calls += 1;
    for (size_t k = 0; k < e->blocks.size(); ++k) {  // every swapped block once per inference
      if (!swapped(e, k)) continue;
      for (const Segment& g : e->blocks[k].segs) e->stats.bytes_swapped += g.bytes;
      e->stats.link_bytes += e->link_bytes[k];
      if (e->blocks[k].variant == SWAPNET_SWAP_MEMCPY) e->stats.memcpy_calls += e->blocks[k].segs.size();
    }
    return SWAPNET_OK;
  });
}

int swapnet_infer_host(swapnet_engine* e, const void* hin, void* hout, swapnet_stream stream) {
  return swapnet::guard_abi([&]() -> int {
    if (!e || !hin || !hout) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null argument");
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    CU(cudaSetDevice(e->device), "cudaSetDevice");
    const Model& m = e->plan.model;
    if (!e->d_in_stage) {
      if (cudaMalloc(&e->d_in_stage, align_up(m.in_bytes)) != cudaSuccess ||
          cudaMalloc(&e->d_out_stage, align_up(m.out_bytes)) != cudaSuccess) {
        cudaGetLastError();
        SN_FAIL(SWAPNET_ERR_OOM, "staging allocation failed");
      }
    }
    CU(cudaMemcpyAsync(e->d_in_stage, hin, m.in_bytes, cudaMemcpyHostToDevice, s), "input copy");
    int rc = swapnet_infer(e, e->d_in_stage, e->d_out_stage, stream);
    if (rc) return rc;
    CU(cudaMemcpyAsync(hout, e->d_out_stage, m.out_bytes, cudaMemcpyDeviceToHost, s), "output copy");
    return SWAPNET_OK;
  });
}

int swapnet_engine_sync(swapnet_engine* e) {
  return swapnet::guard_abi([&]() -> int {
    if (!e) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null engine");
    CU(cudaSetDevice(e->device), "cudaSetDevice");
    if (e->rd) CU(cudaStreamSynchronize(e->rd), "read stream");
    CU(cudaStreamSynchronize(e->copy), "copy stream");
    CU(cudaDeviceSynchronize(), "device synchronize");
    if (const int io = e->io_errno.exchange(0))
      SN_FAIL(SWAPNET_ERR_IO, std::string("weights file read during an inference: ") + std::strerror(io));
    int w = 0;
    CU(cudaMemcpy(&w, e->err_word, sizeof(int), cudaMemcpyDeviceToHost), "error word");
    if (w) {
      const int zero = 0;
      cudaMemcpy(e->err_word, &zero, sizeof(int), cudaMemcpyHostToDevice);
      if (e->d_splitk) cudaMemset(e->d_splitk, 0, e->splitk_counter_bytes);  // an aborted kernel may leave counts
      if (w == 2) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "a token id or a cache position was out of range");
      SN_FAIL(SWAPNET_ERR_TIMEOUT, "a device-side wait gave up");
    }
    return SWAPNET_OK;
  });
}

int swapnet_engine_blocks(const swapnet_engine* e, swapnet_engine_block* b, uint32_t cap, uint32_t* n) {
  return swapnet::guard_abi([&]() -> int {
    if (!e) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null engine");
    if (n) *n = (uint32_t)e->blocks.size();
    for (uint32_t i = 0; b && i < cap && i < e->blocks.size(); ++i) {
      const EngBlock& B = e->blocks[i];
      b[i] = swapnet_engine_block{B.variant, (int32_t)B.segs.size(), B.memcpy_us, B.zerocopy_us};
    }
    return SWAPNET_OK;
  });
}

int swapnet_engine_measure_units(swapnet_engine* e, int32_t reps, float* unit_us, uint32_t n_units) {
  return swapnet::guard_abi([&]() -> int {
    if (!e || !unit_us || reps < 1 || reps > 10000) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "bad argument");
    CU(cudaSetDevice(e->device), "cudaSetDevice");
    const Model& m = e->plan.model;
    if (!e->d_in_stage) {
      if (cudaMalloc(&e->d_in_stage, align_up(m.in_bytes)) != cudaSuccess ||
          cudaMalloc(&e->d_out_stage, align_up(m.out_bytes)) != cudaSuccess) {
        cudaGetLastError();
        SN_FAIL(SWAPNET_ERR_OOM, "staging allocation failed");
      }
      CU(cudaMemset(e->d_in_stage, 0, align_up(m.in_bytes)), "clear staging");
    }
    cudaEvent_t a, b;
    CU(cudaEventCreate(&a), "event");
    CU(cudaEventCreate(&b), "event");
    int rc = SWAPNET_OK;
    const bool prof = e->profiling;
    e->profiling = false;
    for (uint32_t u = 0; u < n_units && u < e->plan.units.size() && rc == SWAPNET_OK; ++u) {
      cudaGraph_t g = nullptr;
      cudaGraphExec_t ge = nullptr;
      if (cudaStreamBeginCapture(e->cap, cudaStreamCaptureModeThreadLocal) != cudaSuccess) { rc = SWAPNET_ERR_CUDA; break; }
      for (int r = 0; r < reps && rc == SWAPNET_OK; ++r) rc = run_unit(e, (int)u, e->d_in_stage, e->d_out_stage, e->cap);
      const cudaError_t ce = cudaStreamEndCapture(e->cap, &g);
      if (rc || ce != cudaSuccess || cudaGraphInstantiate(&ge, g, 0) != cudaSuccess) {
        if (g) cudaGraphDestroy(g);
        cudaGetLastError();
        rc = rc ? rc : SWAPNET_ERR_CUDA;
        break;
      }
      cudaGraphDestroy(g);
      float best = 1e30f;
      for (int t = 0; t < 3; ++t) {
        cudaEventRecord(a, e->cap);
        cudaGraphLaunch(ge, e->cap);
        cudaEventRecord(b, e->cap);
        if (cudaEventSynchronize(b) != cudaSuccess) { rc = SWAPNET_ERR_CUDA; break; }
        float ms = 0.f;
        cudaEventElapsedTime(&ms, a, b);
        if (t > 0) best = std::min(best, ms);  // the first replay warms caches
      }
      cudaGraphExecDestroy(ge);
      unit_us[u] = best * 1000.f / (float)reps;
    }
    e->profiling = prof;
    cudaEventDestroy(a);
    cudaEventDestroy(b);
    if (rc) SN_FAIL(rc, "unit measurement failed");
    return SWAPNET_OK;
  });
}

int swapnet_engine_calibrate(swapnet_engine* e, int32_t reps, int64_t resident_ns, int64_t* t_ex_ns,
                             uint32_t n_layers, uint64_t* alpha_as_per_byte) {
  return swapnet::guard_abi([&]() -> int {
    if (!e || !t_ex_ns || !alpha_as_per_byte || resident_ns < 0) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "bad argument");
    const swapnet_plan& p = e->plan;
    if (n_layers != p.model.L.size()) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "t_ex_ns needs one entry per layer");
    std::vector<float> us(p.units.size(), 0.f);
    int rc = swapnet_engine_measure_units(e, reps, us.data(), (uint32_t)us.size());
    if (rc) return rc;
    // t_ex per layer: the sum of its units' launch times (a split linear
    // layer's pieces run one after another)
    std::vector<int64_t> t(n_layers, 0);
    for (size_t u = 0; u < p.units.size(); ++u) t[p.units[u].layer] += (int64_t)llround((double)us[u] * 1000.0);
    for (auto& v : t) v = std::max<int64_t>(1, v);
    if (resident_ns > 0) {
      // a unit timed alone runs faster than inside the dependent chain of a
      // whole inference: scale the t_ex so they add up to the measured
      // all-resident latency
      double sum = 0.0;
      for (int64_t v : t) sum += (double)v;
      const double f = (double)resident_ns / sum;
      for (auto& v : t) v = std::max<int64_t>(1, (int64_t)llround((double)v * f));
    }
    // alpha: the copy-engine time of every block measured at load over its bytes
    double bytes = 0.0, copy_us = 0.0;
    for (size_t k = 0; k < e->blocks.size() && k < p.blocks.size(); ++k) {
      if (e->blocks[k].memcpy_us <= 0.f) continue;
      bytes += (double)p.blocks[k].bytes;
      copy_us += (double)e->blocks[k].memcpy_us;
    }
    const uint64_t alpha = (bytes > 0.0 && copy_us > 0.0) ? (uint64_t)llround(copy_us * 1e12 / bytes) : 0;
    std::copy(t.begin(), t.end(), t_ex_ns);
    *alpha_as_per_byte = alpha;
    return SWAPNET_OK;
  });
}

int swapnet_engine_bind_state(swapnet_engine* e, void* d_state, uint64_t bytes) {
  return swapnet::guard_abi([&]() -> int {
    if (!e) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null engine");
    if (!e->plan.model.has_attention) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "the model has no decoder state");
    if (!d_state || bytes < e->plan.model.state_bytes) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "state buffer too small");
    if ((uintptr_t)d_state % kAlign) SN_FAIL(SWAPNET_ERR_MISALIGNED, "state buffer must be 256-byte aligned");
    e->d_state = static_cast<char*>(d_state);
    for (auto& kv : e->graphs) cudaGraphExecDestroy(kv.second);  // captured with the old state
    e->graphs.clear();
    return SWAPNET_OK;
  });
}

int swapnet_engine_stats_get(const swapnet_engine* e, swapnet_engine_stats* st) {
  return swapnet::guard_abi([&]() -> int {
    if (!e || !st) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null argument");
    *st = e->stats;
    return SWAPNET_OK;
  });
}

int swapnet_engine_unit_kernels(const swapnet_engine* e, int32_t* kinds, uint32_t cap, uint32_t* n) {
  return swapnet::guard_abi([&]() -> int {
    if (!e) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null engine");
    if (n) *n = (uint32_t)e->unit_kind.size();
    for (uint32_t i = 0; kinds && i < cap && i < e->unit_kind.size(); ++i) kinds[i] = e->unit_kind[i];
    return SWAPNET_OK;
  });
}

int swapnet_engine_unit_tiling(const swapnet_engine* e, swapnet_unit_tiling* t, uint32_t cap, uint32_t* n) {
  return swapnet::guard_abi([&]() -> int {
    if (!e) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null engine");
    if (n) *n = (uint32_t)e->ux.size();
    for (uint32_t i = 0; t && i < cap && i < e->ux.size(); ++i) {
      const UnitExec& X = e->ux[i];
      swapnet_unit_tiling r;
      std::memset(&r, 0, sizeof(r));
      if (X.use_tc) {
        r.n_tile = X.tc.bn;
        r.splits = X.tc.splits;
        r.cluster = X.tc.splits > 1 && X.tc.cluster;
        r.persistent = X.tc.persist;
        r.tap_tma = X.tc.tma_conv;
      }
      t[i] = r;
    }
    return SWAPNET_OK;
  });
}

int swapnet_engine_set_profiling(swapnet_engine* e, int enable) {
  return swapnet::guard_abi([&]() -> int {
    if (!e) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null engine");
    CU(cudaSetDevice(e->device), "cudaSetDevice");
    if (enable && e->ev_unit.empty()) {
      e->ev_unit.assign(2 * e->plan.units.size(), nullptr);
      e->ev_swap.assign(2 * e->plan.blocks.size(), nullptr);
      for (cudaEvent_t& ev : e->ev_unit) CU(cudaEventCreate(&ev), "event");
      for (cudaEvent_t& ev : e->ev_swap) CU(cudaEventCreate(&ev), "event");
    }
    e->profiling = enable != 0;
    return SWAPNET_OK;
  });
}

int swapnet_engine_set_swap_timing(swapnet_engine* e, int enable) {
  return swapnet::guard_abi([&]() -> int {
    if (!e) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null engine");
    CU(cudaSetDevice(e->device), "cudaSetDevice");
    if (enable && e->ev_gswap.empty()) {
      e->ev_gswap.assign(2 * e->plan.blocks.size(), nullptr);
      for (cudaEvent_t& ev : e->ev_gswap) CU(cudaEventCreate(&ev), "event");
    }
    e->swap_timing = enable != 0;
    return SWAPNET_OK;
  });
}

int swapnet_engine_last_swap_times(swapnet_engine* e, float* swap_us, uint32_t nb) {
  return swapnet::guard_abi([&]() -> int {
    if (!e || !swap_us) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null argument");
    if (e->ev_gswap.empty()) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "swap timing was never enabled");
    CU(cudaSetDevice(e->device), "cudaSetDevice");
    for (uint32_t k = 0; k < nb && k < e->plan.blocks.size(); ++k) {
      float ms = 0.f;
      if (swapped(e, k)) {
        CU(cudaEventSynchronize(e->ev_gswap[2 * k + 1]), "event synchronize");
        CU(cudaEventElapsedTime(&ms, e->ev_gswap[2 * k], e->ev_gswap[2 * k + 1]), "elapsed");
      }
      swap_us[k] = ms * 1000.f;
    }
    return SWAPNET_OK;
  });
}

int swapnet_engine_set_graph_timeline(swapnet_engine* e, int enable) {
  return swapnet::guard_abi([&]() -> int {
    if (!e) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null engine");
    CU(cudaSetDevice(e->device), "cudaSetDevice");
    if (enable && e->ev_gswap.empty()) {
      e->ev_gswap.assign(2 * e->plan.blocks.size(), nullptr);
      for (cudaEvent_t& ev : e->ev_gswap) CU(cudaEventCreate(&ev), "event");
    }
    if (enable && e->ev_gexec.empty()) {
      e->ev_gexec.assign(2 * e->plan.blocks.size(), nullptr);
      for (cudaEvent_t& ev : e->ev_gexec) CU(cudaEventCreate(&ev), "event");
      if (!e->ev_g0) CU(cudaEventCreate(&e->ev_g0), "event");
    }
    e->timeline = enable != 0;
    return SWAPNET_OK;
  });
}

int swapnet_engine_last_graph_timeline(swapnet_engine* e, float* t_us, uint32_t nb) {
  return swapnet::guard_abi([&]() -> int {
    if (!e || !t_us) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null argument");
    if (e->ev_gexec.empty()) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "the timeline was never enabled");
    CU(cudaSetDevice(e->device), "cudaSetDevice");
    const uint32_t n = std::min<uint32_t>(nb, (uint32_t)e->plan.blocks.size());
    if (n) CU(cudaEventSynchronize(e->ev_gexec[2 * (n - 1) + 1]), "event synchronize");
    auto since = [&](cudaEvent_t ev, float* out) -> int {
      float ms = 0.f;
      CU(cudaEventSynchronize(ev), "event synchronize");
      CU(cudaEventElapsedTime(&ms, e->ev_g0, ev), "elapsed");
      *out = ms * 1000.f;
      return SWAPNET_OK;
    };
    for (uint32_t k = 0; k < n; ++k) {
      float* o = t_us + 4 * k;
      o[0] = o[1] = -1.f;
      const bool pf_first = k == 0 && prefetch_on(e);
      if (swapped(e, k) && !pf_first) {
        int rc = since(e->ev_gswap[2 * k], o);
        if (!rc) rc = since(e->ev_gswap[2 * k + 1], o + 1);
        if (rc) return rc;
      }
      int rc = since(e->ev_gexec[2 * k], o + 2);
      if (!rc) rc = since(e->ev_gexec[2 * k + 1], o + 3);
      if (rc) return rc;
    }
    return SWAPNET_OK;
  });
}

int swapnet_engine_last_times(swapnet_engine* e, float* unit_us, uint32_t nu, float* swap_us, uint32_t nb) {
  return swapnet::guard_abi([&]() -> int {
    if (!e) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null engine");
    if (e->ev_unit.empty()) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "profiling was never enabled");
    CU(cudaSetDevice(e->device), "cudaSetDevice");
    CU(cudaDeviceSynchronize(), "device synchronize");
    for (uint32_t u = 0; unit_us && u < nu && u < e->plan.units.size(); ++u) {
      float ms = 0.f;
      CU(cudaEventElapsedTime(&ms, e->ev_unit[2 * u], e->ev_unit[2 * u + 1]), "elapsed");
      unit_us[u] = ms * 1000.f;
    }
    for (uint32_t k = 0; swap_us && k < nb && k < e->plan.blocks.size(); ++k) {
      float ms = 0.f;
      if (swapped(e, k))  // a resident prefix and a block read in host memory are never swapped
        CU(cudaEventElapsedTime(&ms, e->ev_swap[2 * k], e->ev_swap[2 * k + 1]), "elapsed");
      swap_us[k] = ms * 1000.f;
    }
    return SWAPNET_OK;
  });
}

int swapnet_engine_last_timeline(swapnet_engine* e, float* us0, float* us1, uint32_t nu, float* ss0, float* ss1,
                                 uint32_t nb) {
  return swapnet::guard_abi([&]() -> int {
    if (!e) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null engine");
    if (e->ev_unit.empty()) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "profiling was never enabled");
    CU(cudaSetDevice(e->device), "cudaSetDevice");
    CU(cudaDeviceSynchronize(), "device synchronize");
    // first block swapped at the start (a resident prefix has no swap events;
    // with first-block prefetch block 0's swap comes at the end)
    size_t k0 = swapnet::prefetch_on(e) ? 1 : 0;
    while (k0 < e->plan.blocks.size() && !swapnet::swapped(e, k0)) ++k0;
    const bool sw = !e->plan.resident && !e->ev_swap.empty() && k0 < e->plan.blocks.size();
    cudaEvent_t origin = sw ? e->ev_swap[2 * k0] : e->ev_unit[0];
    float first = 0.f;
    if (sw) {  // the first kernel may start before the first swap event on another stream
      float d = 0.f;
      CU(cudaEventElapsedTime(&d, e->ev_swap[2 * k0], e->ev_unit[0]), "elapsed");
      first = std::min(0.f, d);
    }
    auto rel = [&](cudaEvent_t ev, float* out) -> int {
      float ms = 0.f;
      CU(cudaEventElapsedTime(&ms, origin, ev), "elapsed");
      *out = (ms - first) * 1000.f;
      return SWAPNET_OK;
    };
    for (uint32_t u = 0; u < nu && u < e->plan.units.size(); ++u) {
      if (us0 && rel(e->ev_unit[2 * u], &us0[u])) return SWAPNET_ERR_CUDA;
      if (us1 && rel(e->ev_unit[2 * u + 1], &us1[u])) return SWAPNET_ERR_CUDA;
    }
    for (uint32_t k = 0; k < nb && k < e->plan.blocks.size(); ++k) {
      if (!sw || !swapnet::swapped(e, k)) {
        if (ss0) ss0[k] = 0.f;
        if (ss1) ss1[k] = 0.f;
        continue;
      }
      if (ss0 && rel(e->ev_swap[2 * k], &ss0[k])) return SWAPNET_ERR_CUDA;
      if (ss1 && rel(e->ev_swap[2 * k + 1], &ss1[k])) return SWAPNET_ERR_CUDA;
    }
    return SWAPNET_OK;
  });
}

void swapnet_engine_free(swapnet_engine* e) { release(e); }

int swapnet_host_alloc(uint64_t bytes, void** out) {
  return swapnet::guard_abi([&]() -> int {
    if (!out || bytes == 0) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null out or zero bytes");
    *out = nullptr;
    if (injected(1) || cudaHostAlloc(out, bytes, cudaHostAllocPortable | cudaHostAllocMapped) != cudaSuccess) {
      cudaGetLastError();
      *out = nullptr;
      SN_FAIL(SWAPNET_ERR_OOM, "page-locked host allocation failed");
    }
    return SWAPNET_OK;
  });
}

int swapnet_host_free(void* p) {
  return swapnet::guard_abi([&]() -> int {
    if (!p) return SWAPNET_OK;
    CU(cudaFreeHost(p), "cudaFreeHost");
    return SWAPNET_OK;
  });
}

int swapnet_debug_fail_next(int what, int count) {
  return swapnet::guard_abi([&]() -> int {
    if (what < 1 || what > 3 || count < 0) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "bad fault-injection request");
    g_fail_next[what] = count;
    return SWAPNET_OK;
  });
}

}  // extern "C"
