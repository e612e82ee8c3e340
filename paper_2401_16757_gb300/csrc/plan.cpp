// Host-side planning: model analysis (Sec. 6.1 model information table),
// activation workspace, partition units, the delay model (Sec. 6.1), the
// partition search (Sec. 6.2.2, Eq. 2-4) and the multi-DNN split (Eq. 1).
// No device work happens here.
#include <algorithm>
#include <cmath>
#include <cstring>
#include <memory>
#include <new>

#include "internal.h"

namespace swapnet {

int dtype_size(int dtype) {
  switch (dtype) {
    case SWAPNET_F32: return 4;
    case SWAPNET_F16: return 2;
    case SWAPNET_BF16: return 2;
    default: return 0;
  }
}

static uint64_t mul_div_ceil(uint64_t a, uint64_t b, uint64_t d) {
  unsigned __int128 p = (unsigned __int128)a * b;
  return (uint64_t)((p + d - 1) / d);
}

// ------------------------------------------------------------ model analysis
int analyse_model(const swapnet_model_desc* desc, Model* m) {
  if (!desc || !desc->layers || desc->n_layers <= 0) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "empty model descriptor");
  m->dtype = desc->dtype;
  m->es = dtype_size(desc->dtype);
  if (!m->es || desc->dtype == SWAPNET_I32) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "unknown dtype");
  m->in_dtype = desc->in_dtype;
  if (m->in_dtype != m->dtype && m->in_dtype != SWAPNET_I32)
    SN_FAIL(SWAPNET_ERR_INVALID_ARG, "input dtype must be the model dtype or int32 token ids");
  if (desc->in_n <= 0 || desc->in_h <= 0 || desc->in_w <= 0 || desc->in_c <= 0)
    SN_FAIL(SWAPNET_ERR_INVALID_ARG, "bad input shape");
  m->in_n = desc->in_n; m->in_h = desc->in_h; m->in_w = desc->in_w; m->in_c = desc->in_c;
  m->in_bytes = (uint64_t)m->in_n * m->in_h * m->in_w * m->in_c *
                (m->in_dtype == SWAPNET_I32 ? 4 : m->es);
  m->state_bytes = 0;
  m->has_attention = false;
  uint64_t state_cur = kAlign;  // position header
  const int nl = desc->n_layers;
  m->L.assign(nl, Layer{});
  m->n_tensors = 0;
  m->tensor_raw.clear();
  m->weight_bytes = 0;
  for (int i = 0; i < nl; ++i) {
    Layer& L = m->L[i];
    L.d = desc->layers[i];
    const swapnet_layer& d = L.d;
    auto dims_of = [&](int src, int* n, int* h, int* w, int* c) -> bool {
      if (src == SWAPNET_SRC_INPUT) { *n = m->in_n; *h = m->in_h; *w = m->in_w; *c = m->in_c; return true; }
      if (src < 0 || src >= i) return false;
      const Layer& P = m->L[src];
      *n = P.on; *h = P.oh; *w = P.ow; *c = P.oc;
      return true;
    };
    if (!dims_of(d.src0, &L.n, &L.h, &L.w, &L.c))
      SN_FAIL(SWAPNET_ERR_INVALID_ARG, "layer " + std::to_string(i) + ": bad src0");
    L.c1 = 0;
    L.n_tensors = 0;
    L.tbytes[0] = L.tbytes[1] = 0;
    L.flops = 0;
    L.host_resident = false;
    L.state_off = -1;
    const uint64_t es = m->es;
    const bool token_input = d.src0 == SWAPNET_SRC_INPUT && m->in_dtype == SWAPNET_I32;
    if (token_input && d.op != SWAPNET_OP_EMBED)
      SN_FAIL(SWAPNET_ERR_INVALID_ARG, "layer " + std::to_string(i) + ": only EMBED reads token ids");
    auto same_dims = [&](int src) -> bool {
      int n, h, w, c;
      return dims_of(src, &n, &h, &w, &c) && n == L.n && h == L.h && w == L.w && c == L.c;
    };
    switch (d.op) {
      case SWAPNET_OP_CONV2D: {
        if (d.cin != L.c || d.cout <= 0 || d.kh <= 0 || d.kw <= 0 || d.stride <= 0 || d.pad < 0)
          SN_FAIL(SWAPNET_ERR_INVALID_ARG, "layer " + std::to_string(i) + ": bad conv parameters");
        L.on = L.n;
        L.oh = (L.h + 2 * d.pad - d.kh) / d.stride + 1;
        L.ow = (L.w + 2 * d.pad - d.kw) / d.stride + 1;
        L.oc = d.cout;
        if (L.oh <= 0 || L.ow <= 0) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "layer " + std::to_string(i) + ": empty output");
        L.n_tensors = 2;
        L.tbytes[0] = (uint64_t)d.cout * d.kh * d.kw * d.cin * es;
        L.tbytes[1] = (uint64_t)d.cout * es;
        L.flops = 2ull * L.on * L.oh * L.ow * (uint64_t)d.cout * d.cin * d.kh * d.kw;
        break;
      }
      case SWAPNET_OP_LINEAR: {
        if ((int64_t)d.cin != (int64_t)L.h * L.w * L.c || d.cout <= 0)
          SN_FAIL(SWAPNET_ERR_INVALID_ARG, "layer " + std::to_string(i) + ": linear in-features mismatch");
        L.on = L.n; L.oh = 1; L.ow = 1; L.oc = d.cout;
        L.n_tensors = (d.flags & SWAPNET_LAYER_NO_BIAS) ? 1 : 2;
        L.tbytes[0] = (uint64_t)d.cout * d.cin * es;
        L.tbytes[1] = L.n_tensors == 2 ? (uint64_t)d.cout * es : 0;
        L.flops = 2ull * L.n * (uint64_t)d.cin * d.cout;
        break;
      }
      case SWAPNET_OP_MAXPOOL: {
        if (d.kh <= 0 || d.kw <= 0 || d.stride <= 0 || d.pad < 0 || 2 * d.pad >= d.kh + 1 + d.kh || d.pad >= d.kh || d.pad >= d.kw)
          SN_FAIL(SWAPNET_ERR_INVALID_ARG, "layer " + std::to_string(i) + ": bad pool window");
        L.on = L.n;
        L.oh = (L.h + 2 * d.pad - d.kh) / d.stride + 1;
        L.ow = (L.w + 2 * d.pad - d.kw) / d.stride + 1;
        L.oc = L.c;
        if (L.oh <= 0 || L.ow <= 0) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "layer " + std::to_string(i) + ": empty output");
        break;
      }
      case SWAPNET_OP_GAP:
        L.on = L.n; L.oh = 1; L.ow = 1; L.oc = L.c;
        break;
      case SWAPNET_OP_UPSAMPLE2X:
        L.on = L.n; L.oh = 2 * L.h; L.ow = 2 * L.w; L.oc = L.c;
        break;
      case SWAPNET_OP_CONCAT: {
        int n1, h1, w1, c1;
        if (!dims_of(d.src1, &n1, &h1, &w1, &c1) || n1 != L.n || h1 != L.h || w1 != L.w)
          SN_FAIL(SWAPNET_ERR_INVALID_ARG, "layer " + std::to_string(i) + ": concat operands mismatch");
        L.c1 = c1;
        L.on = L.n; L.oh = L.h; L.ow = L.w; L.oc = L.c + c1;
        break;
      }
      case SWAPNET_OP_EMBED: {
        if (!token_input || d.cin <= 0 || d.cout <= 0 || (d.cout * es) % 16)
          SN_FAIL(SWAPNET_ERR_INVALID_ARG, "layer " + std::to_string(i) + ": bad embedding");
        L.on = L.n * L.h * L.w * L.c; L.oh = 1; L.ow = 1; L.oc = d.cout;
        L.n_tensors = 1;
        L.tbytes[0] = (uint64_t)d.cin * d.cout * es;
        L.host_resident = true;
        break;
      }
      case SWAPNET_OP_RMSNORM:
        if (d.cout != L.c || L.h != 1 || L.w != 1 || !(d.eps >= 0.f))
          SN_FAIL(SWAPNET_ERR_INVALID_ARG, "layer " + std::to_string(i) + ": bad rmsnorm");
        L.on = L.n; L.oh = 1; L.ow = 1; L.oc = L.c;
        L.n_tensors = 1;
        L.tbytes[0] = (uint64_t)d.cout * es;
        break;
      case SWAPNET_OP_ATTENTION: {
        if (!same_dims(d.src1) || !same_dims(d.src2) || L.h != 1 || L.w != 1 || d.cout != L.c || d.heads <= 0 ||
            L.c % d.heads || d.max_seq <= 0 || !(d.theta > 0.f))
          SN_FAIL(SWAPNET_ERR_INVALID_ARG, "layer " + std::to_string(i) + ": bad attention");
        L.on = L.n; L.oh = 1; L.ow = 1; L.oc = L.c;
        L.flops = 4ull * L.n * (uint64_t)d.max_seq * L.c;
        L.state_off = (int64_t)state_cur;
        state_cur += 2 * align_up((uint64_t)d.max_seq * L.c * es);
        m->has_attention = true;
        break;
      }
      case SWAPNET_OP_ARGMAX:
        L.on = L.n; L.oh = 1; L.ow = 1; L.oc = 1;
        L.c1 = L.h * L.w * L.c;  // row length
        break;
      default:
        SN_FAIL(SWAPNET_ERR_INVALID_ARG, "layer " + std::to_string(i) + ": unknown op");
    }
    if (d.op != SWAPNET_OP_CONCAT && d.op != SWAPNET_OP_ATTENTION && d.src1 != SWAPNET_SRC_NONE)
      SN_FAIL(SWAPNET_ERR_INVALID_ARG, "layer " + std::to_string(i) + ": src1 only for concat and attention");
    if (d.op != SWAPNET_OP_ATTENTION && d.src2 != SWAPNET_SRC_NONE && d.src2 != 0)
      SN_FAIL(SWAPNET_ERR_INVALID_ARG, "layer " + std::to_string(i) + ": src2 only for attention");
    if (d.res != SWAPNET_SRC_NONE) {
      if (d.op != SWAPNET_OP_CONV2D && d.op != SWAPNET_OP_LINEAR)
        SN_FAIL(SWAPNET_ERR_INVALID_ARG, "layer " + std::to_string(i) + ": residual only on conv/linear");
      if (d.res < 0 || d.res >= i) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "layer " + std::to_string(i) + ": bad residual");
      const Layer& R = m->L[d.res];
      if (R.on != L.on || R.oh != L.oh || R.ow != L.ow || R.oc != L.oc)
        SN_FAIL(SWAPNET_ERR_INVALID_ARG, "layer " + std::to_string(i) + ": residual shape mismatch");
    }
    if (d.act < SWAPNET_ACT_NONE || d.act > SWAPNET_ACT_SWIGLU)
      SN_FAIL(SWAPNET_ERR_INVALID_ARG, "layer " + std::to_string(i) + ": bad activation");
    if (d.act == SWAPNET_ACT_SWIGLU && (d.op != SWAPNET_OP_LINEAR || d.res == SWAPNET_SRC_NONE))
      SN_FAIL(SWAPNET_ERR_INVALID_ARG, "layer " + std::to_string(i) + ": SWIGLU needs a linear layer and a gate");
    if (d.t_ex_ns < 0) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "negative t_ex_ns");
    L.first_tensor = m->n_tensors;
    for (int t = 0; t < L.n_tensors; ++t) {
      m->tensor_raw.push_back(L.tbytes[t]);
      m->weight_bytes += align_up(L.tbytes[t]);
    }
    m->n_tensors += L.n_tensors;
    L.out_bytes = (uint64_t)L.on * L.oh * L.ow * L.oc * (d.op == SWAPNET_OP_ARGMAX ? 4 : es);
  }
  m->state_bytes = m->has_attention ? state_cur : 0;
  // liveness: last reader of every output
  for (int i = 0; i < nl; ++i) m->L[i].last_use = i;
  for (int j = 0; j < nl; ++j) {
    const swapnet_layer& d = m->L[j].d;
    int last_producer = -1;
    for (int s : {d.src0, d.src1, d.res, d.op == SWAPNET_OP_ATTENTION ? d.src2 : -1})
      if (s >= 0) {
        m->L[s].last_use = std::max(m->L[s].last_use, j);
        last_producer = std::max(last_producer, s);
      }
    m->L[j].start = j;
    const bool weighted = d.op == SWAPNET_OP_CONV2D || d.op == SWAPNET_OP_LINEAR;
    if (weighted && last_producer >= 0 && last_producer + 1 < j) m->L[j].start = last_producer + 1;
  }
  // outputs go to the output buffer, in layer order
  uint64_t cur = 0;
  for (int i = 0; i < nl; ++i) {
    Layer& L = m->L[i];
    L.out_off = -1;
    if (L.d.is_output) { L.out_off = (int64_t)cur; cur += align_up(L.out_bytes); }
  }
  if (cur == 0) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "model has no output layer");
  m->out_bytes = cur;
  // workspace: first fit over live intervals
  struct Placed { int lo, hi; uint64_t off, size; };
  std::vector<Placed> placed;
  uint64_t ws = 0;
  for (int i = 0; i < nl; ++i) {
    Layer& L = m->L[i];
    L.ws_off = -1;
    if (L.d.is_output) continue;
    const uint64_t size = align_up(L.out_bytes);
    std::vector<const Placed*> conf;
    for (const Placed& p : placed)
      if (p.lo <= L.last_use && L.start <= p.hi) conf.push_back(&p);
    std::vector<uint64_t> cand{0};
    for (const Placed* p : conf) cand.push_back(p->off + p->size);
    std::sort(cand.begin(), cand.end());
    uint64_t chosen = 0;
    for (uint64_t o : cand) {
      bool ok = true;
      for (const Placed* p : conf)
        if (!(o + size <= p->off || p->off + p->size <= o)) { ok = false; break; }
      if (ok) { chosen = o; break; }
    }
    L.ws_off = (int64_t)chosen;
    placed.push_back(Placed{L.start, L.last_use, chosen, size});
    ws = std::max(ws, chosen + size);
  }
  m->ws_bytes = ws;
  return SWAPNET_OK;
}

static int64_t unit_tex(const Model& m, const swapnet_options& opt, const Layer& L, uint64_t flops, int rows) {
  if (L.d.t_ex_ns > 0) {
    if (L.d.op == SWAPNET_OP_LINEAR && rows != L.d.cout)
      return (int64_t)ceil_div_u((uint64_t)L.d.t_ex_ns * rows, (uint64_t)L.d.cout);
    return L.d.t_ex_ns;
  }
  (void)m;
  return (int64_t)mul_div_ceil(opt.gamma_as_per_flop, flops, 1000000000ull);
}

int make_units(const Model& m, const swapnet_options& opt, uint64_t slot, uint64_t region, std::vector<Unit>* out) {
  out->clear();
  const uint64_t es = m.es;
  for (int li = 0; li < (int)m.L.size(); ++li) {
    const Layer& L = m.L[li];
    uint64_t size = 0;
    for (int t = 0; t < L.n_tensors && !L.host_resident; ++t) size += align_up(L.tbytes[t]);
    if (size <= slot || (L.d.op != SWAPNET_OP_LINEAR && size <= region)) {
      Unit u{};
      u.host = L.host_resident;
      u.layer = li; u.row0 = 0; u.rows = (L.d.op == SWAPNET_OP_LINEAR) ? L.d.cout : 0;
      u.depth = L.n_tensors; u.bytes = size; u.flops = L.flops;
      u.t_ex = unit_tex(m, opt, L, L.flops, u.rows);
      u.nt = L.n_tensors;
      for (int t = 0; t < L.n_tensors; ++t) {
        u.tidx[t] = L.first_tensor + t; u.toff[t] = 0; u.tlen[t] = L.tbytes[t];
      }
      out->push_back(u);
      continue;
    }
    if (L.d.op != SWAPNET_OP_LINEAR)
      SN_FAIL(SWAPNET_ERR_INFEASIBLE, "layer " + std::to_string(li) + " (" + std::to_string(size) +
                                          " B) does not fit the arena of " + std::to_string(region) + " B");
    const uint64_t K = L.d.cin, N = L.d.cout;
    const bool has_bias = L.n_tensors == 2;
    auto piece_bytes = [&](uint64_t r) { return align_up(r * K * es) + (has_bias ? align_up(r * es) : 0); };
    uint64_t rmax = 0;
    for (uint64_t r = 128; r <= N + 127 && piece_bytes(r) <= slot; r += 128) rmax = r;
    if (rmax == 0)
      SN_FAIL(SWAPNET_ERR_INFEASIBLE, "layer " + std::to_string(li) + ": 128 output features exceed a slot");
    const uint64_t np = ceil_div_u(N, rmax);
    const uint64_t rr = ceil_div_u(ceil_div_u(N, np), 128) * 128;
    for (uint64_t r0 = 0; r0 < N; r0 += rr) {
      const uint64_t rows = std::min(rr, N - r0);
      Unit u{};
      u.layer = li; u.row0 = (int)r0; u.rows = (int)rows; u.depth = L.n_tensors;
      u.bytes = piece_bytes(rows);
      u.flops = 2ull * L.n * K * rows;
      u.t_ex = unit_tex(m, opt, L, u.flops, (int)rows);
      u.nt = L.n_tensors;
      u.tidx[0] = L.first_tensor; u.toff[0] = r0 * K * es; u.tlen[0] = rows * K * es;
      if (has_bias) { u.tidx[1] = L.first_tensor + 1; u.toff[1] = r0 * es; u.tlen[1] = rows * es; }
      out->push_back(u);
    }
  }
  return SWAPNET_OK;
}

static Block make_block(const std::vector<Unit>& us, int a, int b, const swapnet_options& opt) {
  Block B{};
  B.u0 = a; B.u1 = b;
  for (int u = a; u < b; ++u) { B.bytes += us[u].bytes; B.depth += us[u].depth; B.t_ex += us[u].t_ex; }
  B.t_in = (int64_t)mul_div_ceil(opt.alpha_as_per_byte, B.bytes, 1000000000ull) +
           (int64_t)(opt.beta_ns_per_tensor * B.depth);
  B.t_out = (int64_t)(opt.eta_ns_per_tensor * B.depth);
  return B;
}

// prefix: block 0 is the resident prefix (already in the arena: no copy,
// never released); the swapped blocks after it gate only on each other.
int64_t pipeline_ns(const std::vector<Block>& b, int slots, bool prefix) {
  int64_t C = 0, E = 0;
  std::vector<int64_t> R;
  const int64_t lo = prefix ? 1 : 0;
  for (size_t k = 0; k < b.size(); ++k) {
    if (prefix && k == 0) {
      E = b[0].t_ex;
      R.push_back(0);
      continue;
    }
    const int64_t gate = ((int64_t)k - slots >= lo) ? R[k - slots] : 0;
    C = std::max(C, gate) + b[k].t_in;
    E = std::max(E, C) + b[k].t_ex;
    R.push_back(E + b[k].t_out);
  }
  return E;
}

// Steady state of back-to-back inferences with first-block prefetch (two
// slots): block 0 was copied during the previous inference, so C_0 = 0;
// the copy of the next inference's block 0 follows the copy of block n-1
// (one copy engine) once the last block placed with it (the last even
// block) is released; the inference ends when that copy and the last
// execution have both finished.
int64_t cyclic_ns(const std::vector<Block>& b) {
  if (b.empty()) return 0;
  const size_t n = b.size();
  std::vector<int64_t> R(n);
  int64_t C = 0, E = b[0].t_ex;
  R[0] = E + b[0].t_out;
  for (size_t k = 1; k < n; ++k) {
    const int64_t gate = k >= 2 ? R[k - 2] : 0;
    C = std::max(C, gate) + b[k].t_in;
    E = std::max(E, C) + b[k].t_ex;
    R[k] = E + b[k].t_out;
  }
  const size_t g = (n % 2 == 1) ? n - 1 : n - 2;
  return std::max(E, std::max(C, R[g]) + b[0].t_in);
}

int64_t eq4_ns(const std::vector<Block>& b) {
  const size_t n = b.size();
  int64_t total = 0, ov_prev = 0;
  for (size_t i = 1; i < n; ++i) {
    const int64_t tin_next = (i + 1 < n) ? b[i + 1].t_in : 0;
    const int64_t ov = (b[i - 1].t_out + tin_next) - (b[i].t_ex + ov_prev);
    total += std::max<int64_t>(ov, 0);
    ov_prev = ov;
  }
  return total;
}

uint64_t resident_latency_ns(const Model& m, const swapnet_options& opt) {
  uint64_t t = 0;
  for (const Layer& L : m.L)
    t += (uint64_t)unit_tex(m, opt, L, L.flops, L.d.op == SWAPNET_OP_LINEAR ? L.d.cout : 0);
  return t;
}

void finalize_blocks(swapnet_plan* p, const std::vector<uint32_t>& cuts) {
  p->cuts = cuts;
  p->blocks.clear();
  std::vector<uint32_t> b{0};
  b.insert(b.end(), cuts.begin(), cuts.end());
  b.push_back((uint32_t)p->units.size());
  const int slots = p->resident ? 1 : p->opt.slots;
  const bool prefix = !p->resident && p->prefix_units > 0;
  for (size_t k = 0; k + 1 < b.size(); ++k) {
    Block B = make_block(p->units, (int)b[k], (int)b[k + 1], p->opt);
    if (prefix && k == 0) {  // resident prefix: bottom of the arena, never swapped
      B.slot = -1;
      B.base = 0;
      B.t_in = 0;
      B.t_out = 0;
    } else {
      const size_t s = prefix ? k - 1 : k;  // index among the swapped blocks
      B.slot = (int)(s % slots);
      // two co-resident blocks (Eq. 3): even blocks from the bottom of the
      // region, odd blocks against its top, so s_k + s_{k+1} <= region keeps
      // consecutive blocks apart
      B.base = p->prefix_bytes + ((slots == 2 && (s % 2) == 1) ? p->region - B.bytes : 0);
    }
    // slot layout: tensors in unit order, 256-byte aligned
    uint64_t off = 0;
    for (int u = B.u0; u < B.u1; ++u) {
      Unit& U = p->units[u];
      if (U.host) continue;  // read in host memory: no place in the slot
      for (int t = 0; t < U.nt; ++t) { U.slot_off[t] = off; off += align_up(U.tlen[t]); }
    }
    p->blocks.push_back(B);
  }
  if (p->resident) {
    int64_t t = 0;
    for (const Unit& u : p->units) t += u.t_ex;
    p->predicted = t;
  } else {
    p->predicted = p->opt.objective != 0 ? eq4_ns(p->blocks)
                   : p->opt.prefetch    ? cyclic_ns(p->blocks)
                                        : pipeline_ns(p->blocks, p->opt.slots, prefix);
  }
}

// ----------------------------------------------------------- partition search
// Feasibility of consecutive blocks: each fits the region; with two
// co-resident blocks every adjacent pair fits it together (Eq. 3).
static bool pair_ok(const swapnet_plan* p, uint64_t prev_bytes, uint64_t bytes) {
  if (bytes > p->region) return false;
  return p->opt.slots != 2 || prev_bytes + bytes <= p->region;
}

namespace {

struct State {
  // v[0] a: earliest start of the next copy (m = 2: max(C_k, R_{k-1});
  //         m = 1: R_k); v[1] E_k; v[2] R_k; v[3] bytes of the last block;
  // with first-block prefetch also v[4] bytes and v[5] t_in of block 0
  int64_t v[6];
  int nblocks;
  int prev_j;       // boundary of the previous state
  int prev_idx;     // index in the previous frontier
};

struct Search {
  const std::vector<Unit>& us;
  const swapnet_options& opt;
  uint64_t slot;
  int slots;
  bool cyclic = false;  // first-block prefetch: the finish depends on the block count's parity
  std::vector<std::vector<State>> front;

  Search(const std::vector<Unit>& u, const swapnet_options& o, uint64_t s)
      : us(u), opt(o), slot(s), slots(o.slots) {}

  std::vector<uint32_t> cuts_of(int j, int idx) const {
    std::vector<uint32_t> c;
    while (j > 0) {
      const State& s = front[j][idx];
      if (s.prev_j > 0) c.push_back((uint32_t)s.prev_j);
      const int pj = s.prev_j, pi = s.prev_idx;
      j = pj; idx = pi;
    }
    std::reverse(c.begin(), c.end());
    return c;
  }

  // a is preferred-or-equal to b on ties (fewer blocks, then lexicographic cuts)
  bool tie_le(int j, int ia, int ib) const {
    const State& a = front[j][ia];
    const State& b = front[j][ib];
    if (a.nblocks != b.nblocks) return a.nblocks < b.nblocks;
    return cuts_of(j, ia) <= cuts_of(j, ib);
  }

  bool le_all(const State& a, const State& b) const {
    if (cyclic && (a.nblocks & 1) != (b.nblocks & 1)) return false;
    for (int t = 0; t < (cyclic ? 6 : 4); ++t)
      if (a.v[t] > b.v[t]) return false;
    return true;
  }

  void insert(int j, const State& s) {
    std::vector<State>& F = front[j];
    F.push_back(s);
    const int is = (int)F.size() - 1;
    for (int t = 0; t < is; ++t)
      if (le_all(F[t], F[is]) && tie_le(j, t, is)) { F.pop_back(); return; }
    // drop the states the new one dominates (it stays last, at index w)
    int w = 0;
    for (int t = 0; t < is; ++t) {
      if (le_all(F[is], F[t]) && tie_le(j, is, t)) continue;
      if (w != t) F[w] = F[t];
      ++w;
    }
    F[w] = F[is];
    F.resize(w + 1);
  }

  State step(const State& s, const Block& B) const {
    State r{};
    const int64_t C = s.v[0] + B.t_in;
    const int64_t E = std::max(s.v[1], C) + B.t_ex;
    const int64_t R = E + B.t_out;
    r.v[0] = slots == 2 ? std::max(C, s.v[2]) : std::max(C, R);
    r.v[1] = E;
    r.v[2] = R;
    r.v[3] = slots == 2 ? (int64_t)B.bytes : 0;
    r.v[4] = s.v[4];
    r.v[5] = s.v[5];
    r.nblocks = s.nblocks + 1;
    return r;
  }
};

}  // namespace

// A feasible plan for an upper bound: consecutive units packed into blocks
// of at most half the arena (any two such neighbours fit together).
static int64_t greedy_upper_bound(const swapnet_plan* p, int start, int64_t e0) {
  const int U = (int)p->units.size();
  const uint64_t cap = p->opt.slots == 2 ? p->region / 2 : p->region;
  std::vector<Block> bl;
  if (start > 0) {  // the resident prefix as block 0
    Block P{};
    P.t_ex = e0;
    bl.push_back(P);
  }
  for (int j = start; j < U;) {
    uint64_t bytes = 0;
    int j2 = j;
    while (j2 < U && bytes + p->units[j2].bytes <= cap) bytes += p->units[j2++].bytes;
    if (j2 == j) j2 = j + 1;  // one unit larger than the cap: a block of its own
    Block B = make_block(p->units, j, j2, p->opt);
    const bool first = (int)bl.size() == (start > 0 ? 1 : 0);
    if (!pair_ok(p, first ? 0 : bl.back().bytes, B.bytes)) return INT64_MAX;
    bl.push_back(B);
    j = j2;
  }
  return pipeline_ns(bl, p->opt.slots, start > 0);
}

// Exact search over cut vectors: a Pareto front of pipeline states per unit
// boundary, pruned by dominance and by a bound.  A state at boundary j that
// next copies no earlier than a (and has executed up to E) finishes no
// earlier than max(E + remaining t_ex, a + remaining t_in + t_ex of the last
// unit), since copies and executions each form a chain; states whose bound
// exceeds the best finish found (or a greedy plan's) cannot win.
static int search_pipeline_capped(swapnet_plan* p, std::vector<uint32_t>* best_cuts, size_t cap,
                                  int64_t ub_in, int64_t* best_ns, bool* exact, int start, int64_t e0,
                                  bool cyclic = false, int head = 0) {
  const int U = (int)p->units.size();
  std::vector<int64_t> rem_ex(U + 1, 0), rem_in(U + 1, 0);
  {
    uint64_t bytes = 0, depth = 0;
    for (int j = U - 1; j >= 0; --j) {
      rem_ex[j] = rem_ex[j + 1] + p->units[j].t_ex;
      bytes += p->units[j].bytes;
      depth += p->units[j].depth;
      rem_in[j] = (int64_t)mul_div_ceil(p->opt.alpha_as_per_byte, bytes, 1000000000ull) +
                  (int64_t)(p->opt.beta_ns_per_tensor * depth);
    }
  }
  const int64_t last_ex = U ? p->units[U - 1].t_ex : 0;
  int64_t ub = std::min(ub_in, cyclic ? INT64_MAX : greedy_upper_bound(p, start, e0));
  auto bound = [&](const State& c, int j) -> int64_t {
    if (j == U) return c.v[1];
    return std::max(c.v[1] + rem_ex[j], c.v[0] + rem_in[j] + last_ex);
  };
  // finish of a complete state: E, or with first-block prefetch the later of
  // E and the next block 0's copy (INT64_MAX where the last block and the
  // next block 0 would overlap)
  auto finish = [&](const State& c) -> int64_t {
    if (!cyclic) return c.v[1];
    if (c.nblocks % 2 == 1) return std::max(c.v[1], c.v[2] + c.v[5]);  // block n-1 shares its place
    if ((uint64_t)(c.v[3] + c.v[4]) > p->region) return INT64_MAX;
    return std::max(c.v[1], c.v[0] + c.v[5]);
  };
  Search S(p->units, p->opt, p->slot);
  S.cyclic = cyclic;
  S.front.assign(U + 1, {});
  // initial state at boundary `start`: with a resident prefix, its layers
  // execute from t = 0 (E = e0) while the first copy starts at t = 0, and
  // no swapped block waits for the prefix to be released.  With first-block
  // prefetch, the first block [0, c1) (c1 = head, or every c1 whose block
  // fits the region when head is 0) gives a state at boundary c1: block 0
  // is present at t = 0, executes at once, and the copy engine is free for
  // block 1; states of different first blocks compete in the same fronts
  // (v[4], v[5] carry what the finish needs)
  if (cyclic) {
    Block B0{};
    for (int c1 = 1; c1 <= U; ++c1) {
      const Unit& un = p->units[c1 - 1];
      B0.bytes += un.bytes;
      B0.depth += un.depth;
      B0.t_ex += un.t_ex;
      if (B0.bytes > p->region) break;
      if (head > 0 && c1 != head) continue;
      State s0{};
      s0.v[1] = B0.t_ex;
      s0.v[2] = B0.t_ex + (int64_t)(p->opt.eta_ns_per_tensor * B0.depth);
      s0.v[3] = (int64_t)B0.bytes;
      s0.v[4] = (int64_t)B0.bytes;
      s0.v[5] = (int64_t)mul_div_ceil(p->opt.alpha_as_per_byte, B0.bytes, 1000000000ull) +
                (int64_t)(p->opt.beta_ns_per_tensor * B0.depth);
      s0.prev_j = -1; s0.prev_idx = -1; s0.nblocks = 1;
      if (c1 == U) {
        ub = std::min(ub, finish(s0));
        S.insert(U, s0);
      } else {
        S.insert(c1, s0);
      }
    }
    start = 1;
  } else {
    State s0{};
    s0.v[1] = e0;
    s0.prev_j = -1; s0.prev_idx = -1; s0.nblocks = start > 0 ? 1 : 0;
    S.front[start].push_back(s0);
  }
  // frontier states of boundary j only get children once j is final; a
  // frontier wider than kFrontCap keeps its kFrontCap states of smallest
  // bound (the result is then the best plan found, not a proven optimum)
  *exact = true;
  for (int j = start; j < U; ++j) {
    std::vector<State>& Fj = S.front[j];
    if (Fj.size() > cap) {
      std::vector<std::pair<std::pair<int64_t, int64_t>, size_t>> key(Fj.size());
      for (size_t i = 0; i < Fj.size(); ++i) key[i] = {{bound(Fj[i], j), Fj[i].v[1]}, i};
      std::nth_element(key.begin(), key.begin() + cap, key.end());
      std::sort(key.begin(), key.begin() + cap, [](const auto& x, const auto& y) { return x.second < y.second; });
      std::vector<State> kept;
      kept.reserve(cap);
      for (size_t i = 0; i < cap; ++i) kept.push_back(Fj[key[i].second]);
      Fj.swap(kept);
      *exact = false;
    }
    for (int idx = 0; idx < (int)S.front[j].size(); ++idx) {
      if (bound(S.front[j][idx], j) > ub) continue;
      const uint64_t prev = (uint64_t)S.front[j][idx].v[3];
      Block B{};  // grown one unit at a time: units [j, j2)
      B.u0 = j;
      for (int j2 = j + 1; j2 <= U; ++j2) {
        const Unit& un = p->units[j2 - 1];
        B.u1 = j2;
        B.bytes += un.bytes;
        B.depth += un.depth;
        B.t_ex += un.t_ex;
        if (!pair_ok(p, prev, B.bytes)) break;
        B.t_in = (int64_t)mul_div_ceil(p->opt.alpha_as_per_byte, B.bytes, 1000000000ull) +
                 (int64_t)(p->opt.beta_ns_per_tensor * B.depth);
        B.t_out = (int64_t)(p->opt.eta_ns_per_tensor * B.depth);
        State c = S.step(S.front[j][idx], B);
        c.prev_j = j; c.prev_idx = idx;
        if (bound(c, j2) > ub) continue;
        if (j2 == U) {
          const int64_t f = finish(c);
          if (f == INT64_MAX) continue;
          ub = std::min(ub, f);
        }
        S.insert(j2, c);
      }
    }
  }
  const std::vector<State>& F = S.front[U];
  if (F.empty()) SN_FAIL(SWAPNET_ERR_INFEASIBLE, "no feasible partition");
  int best = 0;
  for (int i = 1; i < (int)F.size(); ++i) {
    const int64_t fi = finish(F[i]), fb = finish(F[best]);
    if (fi < fb || (fi == fb && S.tie_le(U, i, best) && !S.tie_le(U, best, i))) best = i;
  }
  *best_cuts = S.cuts_of(U, best);  // includes `start` (the first block's boundary)
  *best_ns = finish(F[best]);
  return SWAPNET_OK;
}

// A narrow beam first finds a good plan; its finish time then bounds the
// full search, which prunes every state that cannot reach it.  States
// whose bound equals it are kept, so ties are still broken exactly.
static int search_pipeline(swapnet_plan* p, std::vector<uint32_t>* best_cuts, int64_t* best_ns = nullptr,
                           int start = 0, int64_t e0 = 0, bool cyclic = false, int head = 0,
                           int64_t ub = INT64_MAX) {
  std::vector<uint32_t> beam_cuts;
  int64_t beam_ns = INT64_MAX;
  bool beam_exact = false;
  int rc = search_pipeline_capped(p, &beam_cuts, 32, ub, &beam_ns, &beam_exact, start, e0, cyclic, head);
  if (rc) return rc;
  if (beam_exact) {
    p->exact = true;
    *best_cuts = beam_cuts;
    if (best_ns) *best_ns = beam_ns;
    return SWAPNET_OK;
  }
  int64_t ns = 0;
  bool exact = false;
  rc = search_pipeline_capped(p, best_cuts, 4096, std::min(ub, beam_ns), &ns, &exact, start, e0, cyclic, head);
  if (rc) return rc;
  p->exact = exact;
  if (best_ns) *best_ns = ns;
  return SWAPNET_OK;
}

// Resident prefix (option resident_prefix): the candidate prefix lengths are
// 0, the longest prefix that leaves a region every remaining unit (and with
// two co-resident blocks every adjacent pair of remaining units) fits, and
// the longest prefixes within 1/4, 1/2 and 3/4 of that one's bytes.  Each is
// searched exactly; the smallest predicted time wins (ties: shorter prefix).
static int search_with_prefix(swapnet_plan* p, std::vector<uint32_t>* best_cuts) {
  const int U = (int)p->units.size();
  const uint64_t region = p->region;
  std::vector<uint64_t> pb(U + 1, 0);
  std::vector<int64_t> pex(U + 1, 0);
  for (int j = 0; j < U; ++j) {
    pb[j + 1] = pb[j] + p->units[j].bytes;
    pex[j + 1] = pex[j] + p->units[j].t_ex;
  }
  std::vector<uint64_t> need(U + 1, 0);  // smallest region units [r, U) need
  for (int r = U - 1; r >= 0; --r) {
    uint64_t m = std::max(need[r + 1], p->units[r].bytes);
    if (p->opt.slots == 2 && r + 1 < U) m = std::max(m, p->units[r].bytes + p->units[r + 1].bytes);
    need[r] = m;
  }
  int rmax = 0;
  for (int r = 1; r <= U; ++r)
    if (align_up(pb[r]) + need[r] <= region) rmax = r;
  std::vector<int> cand{0};
  for (int q = 1; q <= 3; ++q) {
    int r = 0;
    for (int j = 1; j <= rmax; ++j)
      if (pb[j] * 4 <= pb[rmax] * (uint64_t)q) r = j;
    cand.push_back(r);
  }
  cand.push_back(rmax);
  std::sort(cand.begin(), cand.end());
  cand.erase(std::unique(cand.begin(), cand.end()), cand.end());
  int64_t best = INT64_MAX;
  int best_r = -1;
  bool best_exact = true;
  std::vector<uint32_t> cuts;
  for (int r : cand) {
    p->prefix_units = r;
    p->prefix_bytes = r > 0 ? align_up(pb[r]) : 0;
    p->region = region - p->prefix_bytes;
    std::vector<uint32_t> c;
    int64_t ns = 0;
    if (r == U) {  // everything fits: the prefix is the whole model
      c = {};
      ns = pex[U];
      p->exact = true;
    } else {
      const int rc = search_pipeline(p, &c, &ns, r, pex[r]);
      if (rc == SWAPNET_ERR_INFEASIBLE) continue;
      if (rc) return rc;
    }
    if (ns < best) {
      best = ns;
      best_r = r;
      best_exact = p->exact;
      cuts = c;
    }
  }
  if (best_r < 0) SN_FAIL(SWAPNET_ERR_INFEASIBLE, "no feasible partition");
  p->prefix_units = best_r;
  p->prefix_bytes = best_r > 0 ? align_up(pb[best_r]) : 0;
  p->region = region - p->prefix_bytes;
  p->exact = best_exact;
  *best_cuts = cuts;
  return SWAPNET_OK;
}

// First-block prefetch (option prefetch): for each first block [0, c1)
// an exact search of the rest, finishing with the next block 0's copy.  The
// plan without prefetch, timed as a cyclic schedule (when its last and first
// blocks may be co-resident), gives the first bound; the best finish so far
// bounds each next search.  Ties: smaller time, fewer blocks,
// lexicographically smaller cut vector.  When the region holds more than
// max_heads first blocks, the max_heads smallest and the first block of the
// plan without prefetch are tried (the plan then reports exact = 0); models
// of more than 128 units (each search takes seconds) try only the latter.
static int search_cyclic(swapnet_plan* p, std::vector<uint32_t>* best_cuts) {
  const int U = (int)p->units.size();
  const int max_heads = U > 128 ? 0 : 16;
  std::vector<int> heads;
  {
    uint64_t bytes = 0;
    for (int c1 = 1; c1 <= U; ++c1) {
      bytes += p->units[c1 - 1].bytes;
      if (bytes > p->region) break;
      heads.push_back(c1);
    }
  }
  int64_t best = INT64_MAX;
  int best_n = 0;
  bool found = false;
  std::vector<uint32_t> cuts;
  auto consider = [&](int64_t ns, const std::vector<uint32_t>& c) {
    const int n = (int)c.size() + 1;
    if (!found || ns < best || (ns == best && (n < best_n || (n == best_n && c < cuts)))) {
      best = ns;
      best_n = n;
      cuts = c;
      found = true;
    }
  };
  std::vector<uint32_t> cold;
  {
    swapnet_options o = p->opt;
    p->opt.prefetch = 0;
    const int rc = search_pipeline(p, &cold);
    p->opt = o;
    if (rc && rc != SWAPNET_ERR_INFEASIBLE) return rc;
    if (!rc) {
      std::vector<uint32_t> bnd{0};
      bnd.insert(bnd.end(), cold.begin(), cold.end());
      bnd.push_back((uint32_t)U);
      std::vector<Block> bl;
      for (size_t k = 0; k + 1 < bnd.size(); ++k) bl.push_back(make_block(p->units, (int)bnd[k], (int)bnd[k + 1], p->opt));
      const size_t n = bl.size();
      if (n % 2 == 1 || bl[0].bytes + bl[n - 1].bytes <= p->region) consider(cyclic_ns(bl), cold);
    }
  }
  bool all_exact = true;
  if ((int)heads.size() > max_heads) {
    const int c1 = cold.empty() ? U : (int)cold[0];
    heads.resize(max_heads);
    if (std::find(heads.begin(), heads.end(), c1) == heads.end()) heads.insert(heads.begin(), c1);
    all_exact = false;
  }
  for (int c1 : heads) {
    std::vector<uint32_t> c;
    int64_t ns = 0;
    p->exact = true;
    const int rc = search_pipeline(p, &c, &ns, 0, 0, true, c1, found ? best : INT64_MAX);
    if (rc == SWAPNET_ERR_INFEASIBLE) continue;
    if (rc) return rc;
    all_exact = all_exact && p->exact;
    consider(ns, c);
  }
  if (!found) SN_FAIL(SWAPNET_ERR_INFEASIBLE, "no feasible partition");
  p->exact = all_exact;
  *best_cuts = cuts;
  return SWAPNET_OK;
}

static int search_exhaustive_eq4(swapnet_plan* p, std::vector<uint32_t>* best_cuts) {
  const int U = (int)p->units.size();
  if (U > 24) SN_FAIL(SWAPNET_ERR_UNSUPPORTED, "objective 1 (Eq. 4) search is exhaustive: at most 24 units");
  bool found = false;
  int64_t bo = 0;
  std::vector<uint32_t> bc;
  for (uint64_t mask = 0; mask < (1ull << (U - 1)); ++mask) {
    std::vector<uint32_t> cuts;
    for (int c = 1; c < U; ++c)
      if ((mask >> (c - 1)) & 1) cuts.push_back((uint32_t)c);
    std::vector<uint32_t> b{0};
    b.insert(b.end(), cuts.begin(), cuts.end());
    b.push_back((uint32_t)U);
    std::vector<Block> blocks;
    bool ok = true;
    for (size_t k = 0; k + 1 < b.size(); ++k) {
      Block B = make_block(p->units, (int)b[k], (int)b[k + 1], p->opt);
      if (!pair_ok(p, blocks.empty() ? 0 : blocks.back().bytes, B.bytes)) { ok = false; break; }
      blocks.push_back(B);
    }
    if (!ok) continue;
    const int64_t o = eq4_ns(blocks);
    if (!found || o < bo || (o == bo && (cuts.size() < bc.size() || (cuts.size() == bc.size() && cuts < bc)))) {
      found = true; bo = o; bc = cuts;
    }
  }
  if (!found) SN_FAIL(SWAPNET_ERR_INFEASIBLE, "no feasible partition");
  *best_cuts = bc;
  return SWAPNET_OK;
}

static int check_options(const swapnet_options& o) {
  if (o.slots != 1 && o.slots != 2) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "slots must be 1 or 2");
  if (o.objective != 0 && o.objective != 1) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "objective must be 0 or 1");
  if (o.swap_variant < 0 || o.swap_variant > 4) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "bad swap_variant");
  if (o.zc_ctas < 0 || o.zc_ctas > 4096) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "bad zc_ctas");
  if (o.graphs != 0 && o.graphs != 1) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "graphs must be 0 or 1");
  if (o.preloaded != 0 && o.preloaded != 1) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "preloaded must be 0 or 1");
  if (o.branches != 0 && o.branches != 1) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "branches must be 0 or 1");
  if (o.merge != 0 && o.merge != 1) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "merge must be 0 or 1");
  if (o.pageable != 0 && o.pageable != 1) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "pageable must be 0 or 1");
  if (o.pageable && (o.swap_variant == SWAPNET_SWAP_ZEROCOPY || o.swap_variant == SWAPNET_SWAP_DIRECT ||
                     o.swap_variant == SWAPNET_SWAP_PACKED))
    SN_FAIL(SWAPNET_ERR_INVALID_ARG, "pageable weights are copied by the copy engine only");
  if (o.split_cap < 0 || o.split_cap > 64) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "split_cap must be in [0, 64]");
  if (o.resident_prefix != 0 && o.resident_prefix != 1)
    SN_FAIL(SWAPNET_ERR_INVALID_ARG, "resident_prefix must be 0 or 1");
  if (o.resident_prefix && o.objective != 0)
    SN_FAIL(SWAPNET_ERR_INVALID_ARG, "resident_prefix needs the pipeline objective (0)");
  if (o.prefetch != 0 && o.prefetch != 1) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "prefetch must be 0 or 1");
  if (o.prefetch && (o.objective != 0 || o.slots != 2 || o.resident_prefix))
    SN_FAIL(SWAPNET_ERR_INVALID_ARG, "prefetch needs objective 0, two slots and no resident prefix");
  return SWAPNET_OK;
}

static int prepare(const swapnet_model_desc* desc, uint64_t budget, const swapnet_options* opt,
                   std::unique_ptr<swapnet_plan>* out) {
  std::unique_ptr<swapnet_plan> p(new (std::nothrow) swapnet_plan());
  if (!p) SN_FAIL(SWAPNET_ERR_OOM, "host allocation failed");
  if (opt) p->opt = *opt; else swapnet_default_options(&p->opt);
  int rc = check_options(p->opt);
  if (rc) return rc;
  rc = analyse_model(desc, &p->model);
  if (rc) return rc;
  p->budget = budget;
  const uint64_t ws = p->model.ws_bytes;
  if (p->opt.activations_in_budget && budget <= ws)
    SN_FAIL(SWAPNET_ERR_INFEASIBLE, "budget does not cover the activation workspace");
  p->arena = p->opt.activations_in_budget ? budget - ws : budget;
  p->region = p->arena / kAlign * kAlign;
  p->slot = (p->arena / (uint64_t)p->opt.slots) / kAlign * kAlign;
  rc = make_units(p->model, p->opt, p->slot, p->region, &p->units);
  if (rc) return rc;
  *out = std::move(p);
  return SWAPNET_OK;
}

}  // namespace swapnet

using namespace swapnet;

extern "C" {

void swapnet_default_options(swapnet_options* o) {
  if (!o) return;
  std::memset(o, 0, sizeof(*o));
  o->slots = 2;
  o->activations_in_budget = 0;
  o->swap_variant = SWAPNET_SWAP_AUTO;
  o->objective = 0;
  o->alpha_as_per_byte = 2500000;  // 400 GB/s
  o->beta_ns_per_tensor = 2000;
  o->gamma_as_per_flop = 2000;     // 500 TFLOP/s
  o->eta_ns_per_tensor = 0;
  o->zc_ctas = 0;
  o->graphs = 1;
  o->branches = 1;
  o->merge = 1;
}

int swapnet_partition(const swapnet_model_desc* desc, uint64_t budget, const swapnet_options* opt,
                      swapnet_plan** out) {
  return swapnet::guard_abi([&]() -> int {
    if (!out) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null out_plan");
    try {
      std::unique_ptr<swapnet_plan> p;
      int rc = prepare(desc, budget, opt, &p);
      if (rc) return rc;
      std::vector<uint32_t> cuts;
      if (p->opt.objective != 0) rc = search_exhaustive_eq4(p.get(), &cuts);
      else if (p->opt.resident_prefix) rc = search_with_prefix(p.get(), &cuts);
      else if (p->opt.prefetch) rc = search_cyclic(p.get(), &cuts);
      else rc = search_pipeline(p.get(), &cuts);
      if (rc) return rc;
      finalize_blocks(p.get(), cuts);
      *out = p.release();
      return SWAPNET_OK;
    } catch (const std::bad_alloc&) {
      SN_FAIL(SWAPNET_ERR_OOM, "host allocation failed");
    }
  });
}

int swapnet_plan_from_cuts(const swapnet_model_desc* desc, const uint32_t* cuts, uint32_t n_cuts,
                           uint64_t budget, const swapnet_options* opt, swapnet_plan** out) {
  return swapnet::guard_abi([&]() -> int {
    if (!out || (n_cuts && !cuts)) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null argument");
    try {
      std::unique_ptr<swapnet_plan> p;
      int rc = prepare(desc, budget, opt, &p);
      if (rc) return rc;
      std::vector<uint32_t> c(cuts, cuts + n_cuts);
      uint32_t prev = 0;
      for (uint32_t v : c) {
        if (v <= prev || v >= p->units.size()) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "cuts must increase within [1, n_units)");
        prev = v;
      }
      finalize_blocks(p.get(), c);
      for (size_t k = 0; k < p->blocks.size(); ++k)
        if (!pair_ok(p.get(), k ? p->blocks[k - 1].bytes : 0, p->blocks[k].bytes))
          SN_FAIL(SWAPNET_ERR_INFEASIBLE, "a block (or two adjacent blocks) exceeds the arena");
      const size_t n = p->blocks.size();
      if (p->opt.prefetch && n >= 2 && n % 2 == 0 && p->blocks[0].bytes + p->blocks[n - 1].bytes > p->region)
        SN_FAIL(SWAPNET_ERR_INFEASIBLE, "the last block and the next inference's first block exceed the arena");
      *out = p.release();
      return SWAPNET_OK;
    } catch (const std::bad_alloc&) {
      SN_FAIL(SWAPNET_ERR_OOM, "host allocation failed");
    }
  });
}

int swapnet_plan_resident(const swapnet_model_desc* desc, const swapnet_options* opt, swapnet_plan** out) {
  return swapnet::guard_abi([&]() -> int {
    if (!out) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null out_plan");
    try {
      std::unique_ptr<swapnet_plan> p(new swapnet_plan());
      if (opt) p->opt = *opt; else swapnet_default_options(&p->opt);
      int rc = check_options(p->opt);
      if (rc) return rc;
      rc = analyse_model(desc, &p->model);
      if (rc) return rc;
      p->resident = true;
      p->arena = p->model.weight_bytes;
      p->region = p->arena;
      p->slot = p->arena;
      p->budget = p->arena;
      rc = make_units(p->model, p->opt, ~0ull, ~0ull, &p->units);
      if (rc) return rc;
      finalize_blocks(p.get(), {});
      *out = p.release();
      return SWAPNET_OK;
    } catch (const std::bad_alloc&) {
      SN_FAIL(SWAPNET_ERR_OOM, "host allocation failed");
    }
  });
}

int swapnet_plan_info_get(const swapnet_plan* p, swapnet_plan_info* info) {
  return swapnet::guard_abi([&]() -> int {
    if (!p || !info) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null argument");
    swapnet_plan_info r{};
    r.n_blocks = (uint32_t)p->blocks.size();
    r.n_units = (uint32_t)p->units.size();
    r.slots = p->resident ? 0 : (uint32_t)p->opt.slots;
    r.n_layers = (uint32_t)p->model.L.size();
    r.budget_bytes = p->budget;
    r.arena_bytes = p->arena;
    r.slot_bytes = p->slot;
    r.workspace_bytes = p->model.ws_bytes;
    r.input_bytes = p->model.in_bytes;
    r.output_bytes = p->model.out_bytes;
    r.weight_bytes = p->model.weight_bytes;
    r.plan_bytes = sizeof(swapnet_plan) + p->units.size() * sizeof(Unit) + p->blocks.size() * sizeof(Block) +
                   p->model.L.size() * sizeof(Layer) + p->cuts.size() * sizeof(uint32_t);
    r.predicted_ns = p->predicted;
    r.state_bytes = p->model.state_bytes;
    r.exact = p->exact ? 1 : 0;
    r.prefix_units = (uint32_t)p->prefix_units;
    r.prefix_bytes = p->prefix_bytes;
    *info = r;
    return SWAPNET_OK;
  });
}

int swapnet_plan_cuts(const swapnet_plan* p, uint32_t* cuts, uint32_t cap, uint32_t* n) {
  return swapnet::guard_abi([&]() -> int {
    if (!p) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null plan");
    if (n) *n = (uint32_t)p->cuts.size();
    for (uint32_t i = 0; cuts && i < cap && i < p->cuts.size(); ++i) cuts[i] = p->cuts[i];
    return SWAPNET_OK;
  });
}

int swapnet_plan_units(const swapnet_plan* p, swapnet_unit_info* u, uint32_t cap, uint32_t* n) {
  return swapnet::guard_abi([&]() -> int {
    if (!p) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null plan");
    if (n) *n = (uint32_t)p->units.size();
    for (uint32_t i = 0; u && i < cap && i < p->units.size(); ++i) {
      const Unit& U = p->units[i];
      u[i] = swapnet_unit_info{U.layer, U.row0, U.rows, U.depth, U.bytes, U.flops, U.t_ex};
    }
    return SWAPNET_OK;
  });
}

int swapnet_plan_blocks(const swapnet_plan* p, swapnet_block_info* b, uint32_t cap, uint32_t* n) {
  return swapnet::guard_abi([&]() -> int {
    if (!p) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null plan");
    if (n) *n = (uint32_t)p->blocks.size();
    for (uint32_t i = 0; b && i < cap && i < p->blocks.size(); ++i) {
      const Block& B = p->blocks[i];
      b[i] = swapnet_block_info{(uint32_t)B.u0, (uint32_t)B.u1, (uint32_t)B.slot, (uint32_t)B.depth, B.bytes,
                                B.t_in, B.t_ex, B.t_out, B.base};
    }
    return SWAPNET_OK;
  });
}

int swapnet_plan_output_offsets(const swapnet_plan* p, uint64_t* offs, uint32_t cap, uint32_t* n) {
  return swapnet::guard_abi([&]() -> int {
    if (!p) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null plan");
    uint32_t k = 0;
    for (const Layer& L : p->model.L) {
      if (L.out_off < 0) continue;
      if (offs && k < cap) offs[k] = (uint64_t)L.out_off;
      ++k;
    }
    if (n) *n = k;
    return SWAPNET_OK;
  });
}

void swapnet_plan_free(swapnet_plan* p) { delete p; }

int swapnet_schedule(const swapnet_model_desc* const* models, const float* urgency, uint32_t n,
                     uint64_t M, const swapnet_options* opt, uint64_t* budgets_out, swapnet_plan** plans_out) {
  return swapnet::guard_abi([&]() -> int {
    if (!models || !urgency || n == 0 || !plans_out) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null argument");
    try {
      swapnet_options o;
      if (opt) o = *opt; else swapnet_default_options(&o);
      std::vector<Model> ms(n);
      std::vector<long double> demand(n), ps(n);
      long double sumM = 0, sumPS = 0;
      for (uint32_t i = 0; i < n; ++i) {
        int rc = analyse_model(models[i], &ms[i]);
        if (rc) return rc;
        if (!(urgency[i] >= 0.0f) || !std::isfinite(urgency[i])) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "bad urgency");
        demand[i] = (long double)ms[i].weight_bytes;
        const long double lat = (long double)resident_latency_ns(ms[i], o);
        ps[i] = (long double)urgency[i] * lat / demand[i];
        sumM += demand[i];
        sumPS += ps[i];
      }
      std::vector<uint64_t> budgets(n);
      for (uint32_t i = 0; i < n; ++i) {
        if (sumM <= (long double)M) { budgets[i] = ms[i].weight_bytes; continue; }
        long double a = demand[i] / sumM * (1.0L - 1.0L / n) * (long double)M;
        if (sumPS > 0) a += ps[i] / sumPS * (1.0L / n) * (long double)M;
        budgets[i] = (uint64_t)floorl(a) / kAlign * kAlign;
      }
      std::vector<swapnet_plan*> plans(n, nullptr);
      for (uint32_t i = 0; i < n; ++i) {
        int rc = swapnet_partition(models[i], budgets[i], &o, &plans[i]);
        if (rc) {
          for (swapnet_plan* q : plans) delete q;
          return rc;
        }
      }
      for (uint32_t i = 0; i < n; ++i) {
        plans_out[i] = plans[i];
        if (budgets_out) budgets_out[i] = budgets[i];
      }
      return SWAPNET_OK;
    } catch (const std::bad_alloc&) {
      SN_FAIL(SWAPNET_ERR_OOM, "host allocation failed");
    }
  });
}

}  // extern "C"
