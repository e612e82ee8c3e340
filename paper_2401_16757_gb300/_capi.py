"""ctypes binding of libswapnet (include/swapnet.h): argument marshalling only.

Every step of the inference path runs in the library's CUDA kernels; this
module converts Python descriptions to the C structs, calls the C entry
points and raises SwapnetError on a non-zero status.  It fails loudly when
the shared library is missing.
"""
import ctypes as C
import mmap
import os

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libswapnet.so")

OK, ERR_INVALID_ARG, ERR_INFEASIBLE, ERR_OOM, ERR_CUDA, ERR_TIMEOUT, ERR_MISALIGNED, ERR_UNSUPPORTED, ERR_IO, \
    ERR_INTERNAL = 0, -1, -2, -3, -4, -5, -6, -7, -8, -9
F32, F16, BF16 = 0, 1, 2
I32 = 3
OP = {"linear": 1, "conv": 2, "maxpool": 3, "gap": 4, "upsample2x": 5, "concat": 6, "embed": 7, "rmsnorm": 8,
      "attention": 9, "argmax": 10}
ACT = {"none": 0, "relu": 1, "leaky": 2, "swiglu": 3}
DTYPE = {"f32": F32, "f16": F16, "bf16": BF16, "i32": I32}
LAYER_NO_BIAS = 1
SWAP_AUTO, SWAP_MEMCPY, SWAP_ZEROCOPY, SWAP_DIRECT, SWAP_PACKED = 0, 1, 2, 3, 4
SRC_INPUT, SRC_NONE = -1, -2


class Layer(C.Structure):
    _fields_ = [("op", C.c_int32), ("src0", C.c_int32), ("src1", C.c_int32), ("res", C.c_int32),
                ("act", C.c_int32), ("res_post", C.c_int32), ("cin", C.c_int32), ("cout", C.c_int32),
                ("kh", C.c_int32), ("kw", C.c_int32), ("stride", C.c_int32), ("pad", C.c_int32),
                ("is_output", C.c_int32), ("flags", C.c_int32), ("t_ex_ns", C.c_int64), ("src2", C.c_int32),
                ("heads", C.c_int32), ("max_seq", C.c_int32), ("eps", C.c_float), ("theta", C.c_float),
                ("reserved", C.c_int32)]


class ModelDesc(C.Structure):
    _fields_ = [("dtype", C.c_int32), ("n_layers", C.c_int32), ("layers", C.POINTER(Layer)),
                ("in_n", C.c_int32), ("in_h", C.c_int32), ("in_w", C.c_int32), ("in_c", C.c_int32),
                ("in_dtype", C.c_int32), ("reserved", C.c_int32)]


class Options(C.Structure):
    _fields_ = [("slots", C.c_int32), ("activations_in_budget", C.c_int32), ("swap_variant", C.c_int32),
                ("objective", C.c_int32), ("alpha_as_per_byte", C.c_uint64), ("beta_ns_per_tensor", C.c_uint64),
                ("gamma_as_per_flop", C.c_uint64), ("eta_ns_per_tensor", C.c_uint64), ("zc_ctas", C.c_int32),
                ("graphs", C.c_int32), ("preloaded", C.c_int32), ("branches", C.c_int32),
                ("resident_prefix", C.c_int32), ("split_cap", C.c_int32), ("prefetch", C.c_int32),
                ("merge", C.c_int32), ("pageable", C.c_int32), ("reserved", C.c_int32 * 1)]


class PlanInfo(C.Structure):
    _fields_ = [("n_blocks", C.c_uint32), ("n_units", C.c_uint32), ("slots", C.c_uint32),
                ("n_layers", C.c_uint32), ("budget_bytes", C.c_uint64), ("arena_bytes", C.c_uint64),
                ("slot_bytes", C.c_uint64), ("workspace_bytes", C.c_uint64), ("input_bytes", C.c_uint64),
                ("output_bytes", C.c_uint64), ("weight_bytes", C.c_uint64), ("plan_bytes", C.c_uint64),
                ("predicted_ns", C.c_int64), ("state_bytes", C.c_uint64), ("exact", C.c_int32),
                ("reserved", C.c_int32), ("prefix_units", C.c_uint32), ("reserved2", C.c_uint32),
                ("prefix_bytes", C.c_uint64)]


class UnitInfo(C.Structure):
    _fields_ = [("layer", C.c_int32), ("row0", C.c_int32), ("rows", C.c_int32), ("depth", C.c_int32),
                ("bytes", C.c_uint64), ("flops", C.c_uint64), ("t_ex_ns", C.c_int64)]


class BlockInfo(C.Structure):
    _fields_ = [("unit0", C.c_uint32), ("unit1", C.c_uint32), ("slot", C.c_uint32), ("depth", C.c_uint32),
                ("bytes", C.c_uint64), ("t_in_ns", C.c_int64), ("t_ex_ns", C.c_int64), ("t_out_ns", C.c_int64),
                ("offset", C.c_uint64)]


class EngineStats(C.Structure):
    _fields_ = [("infer_calls", C.c_uint64), ("kernel_launches", C.c_uint64), ("memcpy_calls", C.c_uint64),
                ("bytes_swapped", C.c_uint64), ("link_bytes", C.c_uint64)]


KERNEL_KIND = {1: "tc_gemm", 2: "tc_conv", 3: "skinny_linear", 4: "direct_conv", 5: "maxpool", 6: "gap",
               7: "upsample2x", 8: "concat", 9: "tiled_linear", 10: "embed", 11: "rmsnorm", 12: "attention",
               13: "argmax", 14: "tc_conv_small"}


class UnitTiling(C.Structure):
    _fields_ = [("n_tile", C.c_int32), ("splits", C.c_int32), ("cluster", C.c_int32), ("persistent", C.c_int32),
                ("tap_tma", C.c_int32), ("reserved", C.c_int32 * 3)]


class EngineBlock(C.Structure):
    _fields_ = [("variant", C.c_int32), ("n_segments", C.c_int32), ("memcpy_us", C.c_float),
                ("zerocopy_us", C.c_float)]


EXPORTS = ["swapnet_default_options", "swapnet_partition", "swapnet_plan_from_cuts", "swapnet_plan_resident",
           "swapnet_plan_info_get", "swapnet_plan_cuts", "swapnet_plan_units", "swapnet_plan_blocks",
           "swapnet_plan_output_offsets", "swapnet_plan_free", "swapnet_schedule", "swapnet_load",
           "swapnet_infer", "swapnet_infer_host", "swapnet_engine_sync", "swapnet_engine_blocks",
           "swapnet_engine_free", "swapnet_engine_stats_get", "swapnet_engine_unit_kernels", "swapnet_engine_unit_tiling", "swapnet_engine_adapt", "swapnet_host_alloc", "swapnet_host_free",
           "swapnet_engine_set_profiling", "swapnet_engine_last_times", "swapnet_engine_measure_units",
           "swapnet_engine_last_timeline", "swapnet_engine_calibrate",
           "swapnet_engine_set_swap_timing", "swapnet_engine_last_swap_times",
           "swapnet_engine_set_graph_timeline", "swapnet_engine_last_graph_timeline",
           "swapnet_engine_bind_state", "swapnet_strerror", "swapnet_last_error", "swapnet_debug_fail_next", "swapnet_gemm_noalloc",
           "swapnet_weights_file_write", "swapnet_weights_file_open", "swapnet_weights_file_info",
           "swapnet_weights_file_read", "swapnet_weights_file_close", "swapnet_load_file",
           "swapnet_debug_wait_timeout", "swapnet_pack_bf16"]

_lib = None


class SwapnetError(RuntimeError):
    def __init__(self, code, what):
        self.code = code
        super().__init__("%s: %s (%d): %s" % (what, lib().swapnet_strerror(code).decode(), code,
                                               lib().swapnet_last_error().decode()))


def lib():
    """The loaded libswapnet (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise ImportError("libswapnet.so is not built: run __graft_entry__.build() or "
                          "python paper_2401_16757_gb300/build.py")
    L = C.CDLL(LIB_PATH)
    P = C.c_void_p
    sig = {
        "swapnet_default_options": (None, [C.POINTER(Options)]),
        "swapnet_partition": (C.c_int, [C.POINTER(ModelDesc), C.c_uint64, C.POINTER(Options), C.POINTER(P)]),
        "swapnet_plan_from_cuts": (C.c_int, [C.POINTER(ModelDesc), C.POINTER(C.c_uint32), C.c_uint32, C.c_uint64,
                                             C.POINTER(Options), C.POINTER(P)]),
        "swapnet_plan_resident": (C.c_int, [C.POINTER(ModelDesc), C.POINTER(Options), C.POINTER(P)]),
        "swapnet_plan_info_get": (C.c_int, [P, C.POINTER(PlanInfo)]),
        "swapnet_plan_cuts": (C.c_int, [P, C.POINTER(C.c_uint32), C.c_uint32, C.POINTER(C.c_uint32)]),
        "swapnet_plan_units": (C.c_int, [P, C.POINTER(UnitInfo), C.c_uint32, C.POINTER(C.c_uint32)]),
        "swapnet_plan_blocks": (C.c_int, [P, C.POINTER(BlockInfo), C.c_uint32, C.POINTER(C.c_uint32)]),
        "swapnet_plan_output_offsets": (C.c_int, [P, C.POINTER(C.c_uint64), C.c_uint32, C.POINTER(C.c_uint32)]),
        "swapnet_plan_free": (None, [P]),
        "swapnet_schedule": (C.c_int, [C.POINTER(C.POINTER(ModelDesc)), C.POINTER(C.c_float), C.c_uint32,
                                       C.c_uint64, C.POINTER(Options), C.POINTER(C.c_uint64), C.POINTER(P)]),
        "swapnet_load": (C.c_int, [P, C.POINTER(P), C.c_uint32, P, C.c_uint64, P, C.c_uint64, C.POINTER(P)]),
        "swapnet_infer": (C.c_int, [P, P, P, P]),
        "swapnet_infer_host": (C.c_int, [P, P, P, P]),
        "swapnet_engine_sync": (C.c_int, [P]),
        "swapnet_engine_adapt": (C.c_int, [P, P]),
        "swapnet_host_alloc": (C.c_int, [C.c_uint64, C.POINTER(P)]),
        "swapnet_host_free": (C.c_int, [P]),
        "swapnet_pack_bf16": (C.c_int, [P, C.c_uint64, P, C.c_uint64, C.POINTER(C.c_uint64)]),
        "swapnet_engine_bind_state": (C.c_int, [P, P, C.c_uint64]),
        "swapnet_engine_blocks": (C.c_int, [P, C.POINTER(EngineBlock), C.c_uint32, C.POINTER(C.c_uint32)]),
        "swapnet_engine_free": (None, [P]),
        "swapnet_engine_stats_get": (C.c_int, [P, C.POINTER(EngineStats)]),
        "swapnet_engine_unit_kernels": (C.c_int, [P, C.POINTER(C.c_int32), C.c_uint32, C.POINTER(C.c_uint32)]),
        "swapnet_engine_unit_tiling": (C.c_int, [P, C.POINTER(UnitTiling), C.c_uint32, C.POINTER(C.c_uint32)]),
        "swapnet_engine_set_profiling": (C.c_int, [P, C.c_int]),
        "swapnet_engine_set_swap_timing": (C.c_int, [P, C.c_int]),
        "swapnet_engine_last_swap_times": (C.c_int, [P, C.POINTER(C.c_float), C.c_uint32]),
        "swapnet_engine_set_graph_timeline": (C.c_int, [P, C.c_int]),
        "swapnet_engine_last_graph_timeline": (C.c_int, [P, C.POINTER(C.c_float), C.c_uint32]),
        "swapnet_engine_measure_units": (C.c_int, [P, C.c_int32, C.POINTER(C.c_float), C.c_uint32]),
        "swapnet_engine_last_timeline": (C.c_int, [P, C.POINTER(C.c_float), C.POINTER(C.c_float), C.c_uint32,
                                                   C.POINTER(C.c_float), C.POINTER(C.c_float), C.c_uint32]),
        "swapnet_engine_last_times": (C.c_int, [P, C.POINTER(C.c_float), C.c_uint32, C.POINTER(C.c_float),
                                                C.c_uint32]),
        "swapnet_engine_calibrate": (C.c_int, [P, C.c_int32, C.c_int64, C.POINTER(C.c_int64), C.c_uint32,
                                               C.POINTER(C.c_uint64)]),
        "swapnet_strerror": (C.c_char_p, [C.c_int]),
        "swapnet_last_error": (C.c_char_p, []),
        "swapnet_debug_fail_next": (C.c_int, [C.c_int, C.c_int]),
        "swapnet_gemm_noalloc": (C.c_int, [C.c_int32, P, P, P, P, C.c_int32, C.c_int32, C.c_int32, C.c_int32, P]),
        "swapnet_weights_file_write": (C.c_int, [C.c_char_p, C.POINTER(ModelDesc), C.POINTER(P), C.c_uint32]),
        "swapnet_weights_file_open": (C.c_int, [C.c_char_p, C.c_uint32, C.POINTER(P)]),
        "swapnet_weights_file_info": (C.c_int, [P, C.POINTER(C.c_uint32), C.POINTER(C.c_int32)]),
        "swapnet_weights_file_read": (C.c_int, [P, C.c_uint32, C.c_uint64, C.c_uint64, P]),
        "swapnet_weights_file_close": (None, [P]),
        "swapnet_load_file": (C.c_int, [P, P, P, C.c_uint64, P, C.c_uint64, C.POINTER(P)]),
        "swapnet_debug_wait_timeout": (C.c_int, [P]),
    }
    for name, (res, args) in sig.items():
        f = getattr(L, name)
        f.restype, f.argtypes = res, args
    _lib = L
    return L


def check(rc, what):
    if rc != OK:
        raise SwapnetError(rc, what)


# ------------------------------------------------------------------ options
def options(**kw):
    o = Options()
    lib().swapnet_default_options(C.byref(o))
    for k, v in kw.items():
        if not hasattr(o, k):
            raise KeyError(k)
        setattr(o, k, v)
    return o


# ------------------------------------------------------------ descriptors
class Desc:
    """A C model descriptor built from a layer-sequence dict (see synth.arch)."""

    def __init__(self, model, t_ex_ns=None):
        layers = model["layers"]
        arr = (Layer * len(layers))()
        outs = set(model["outputs"])
        for i, L in enumerate(layers):
            c = arr[i]
            c.op = OP[L["op"]]
            c.src0 = L["src"][0]
            c.src1 = L["src"][1] if len(L["src"]) > 1 else SRC_NONE
            c.res = SRC_NONE if L.get("res") is None else L["res"]
            c.act = ACT[L.get("act", "none")]
            c.res_post = 1 if L.get("res_post") else 0
            if L["op"] == "conv":
                c.cin, c.cout, c.kh, c.kw, c.stride, c.pad = L["cin"], L["cout"], L["kh"], L["kw"], L["stride"], L["pad"]
            elif L["op"] == "linear":
                c.cin, c.cout = L["k"], L["n"]
            elif L["op"] == "maxpool":
                c.kh, c.kw, c.stride, c.pad = L["kh"], L["kw"], L["stride"], L["pad"]
            elif L["op"] == "embed":
                c.cin, c.cout = L["vocab"], L["d"]
            elif L["op"] == "rmsnorm":
                c.cout, c.eps = L["d"], L["eps"]
            elif L["op"] == "attention":
                c.src0, c.src1, c.src2 = L["src"]
                c.heads, c.max_seq, c.theta = L["heads"], L["max_seq"], L["theta"]
            if L["op"] == "attention":
                c.cout = 0  # filled below from the q width
            if L["op"] != "attention":
                c.src2 = SRC_NONE
            if L.get("bias") is False:
                c.flags |= LAYER_NO_BIAS
            c.is_output = 1 if i in outs else 0
            c.t_ex_ns = 0 if t_ex_ns is None else int(t_ex_ns[i])
        # attention width = width of its q input
        for i, L in enumerate(layers):
            if L["op"] == "attention":
                arr[i].cout = arr[L["src"][0]].cout
        n, h, w, ch = model["input"]
        self.layers = arr
        in_dt = DTYPE[model.get("input_dtype", model["dtype"])]
        self.c = ModelDesc(DTYPE[model["dtype"]], len(layers), arr, n, h, w, ch, in_dt, 0)
        self.model = model


class Plan:
    def __init__(self, handle):
        self.h = C.c_void_p(handle)

    @staticmethod
    def partition(desc, budget, opt=None):
        h = C.c_void_p()
        check(lib().swapnet_partition(C.byref(desc.c), budget, C.byref(opt) if opt else None, C.byref(h)),
              "swapnet_partition")
        return Plan(h.value)

    @staticmethod
    def from_cuts(desc, cuts, budget, opt=None):
        h = C.c_void_p()
        arr = (C.c_uint32 * max(1, len(cuts)))(*cuts)
        check(lib().swapnet_plan_from_cuts(C.byref(desc.c), arr, len(cuts), budget,
                                           C.byref(opt) if opt else None, C.byref(h)), "swapnet_plan_from_cuts")
        return Plan(h.value)

    @staticmethod
    def resident(desc, opt=None):
        h = C.c_void_p()
        check(lib().swapnet_plan_resident(C.byref(desc.c), C.byref(opt) if opt else None, C.byref(h)),
              "swapnet_plan_resident")
        return Plan(h.value)

    def info(self):
        i = PlanInfo()
        check(lib().swapnet_plan_info_get(self.h, C.byref(i)), "swapnet_plan_info_get")
        return {f: getattr(i, f) for f, _ in PlanInfo._fields_}

    def cuts(self):
        n = C.c_uint32()
        check(lib().swapnet_plan_cuts(self.h, None, 0, C.byref(n)), "swapnet_plan_cuts")
        arr = (C.c_uint32 * max(1, n.value))()
        check(lib().swapnet_plan_cuts(self.h, arr, n.value, None), "swapnet_plan_cuts")
        return list(arr[:n.value])

    def units(self):
        n = C.c_uint32()
        check(lib().swapnet_plan_units(self.h, None, 0, C.byref(n)), "swapnet_plan_units")
        arr = (UnitInfo * max(1, n.value))()
        check(lib().swapnet_plan_units(self.h, arr, n.value, None), "swapnet_plan_units")
        return [{f: getattr(u, f) for f, _ in UnitInfo._fields_} for u in arr[:n.value]]

    def blocks(self):
        n = C.c_uint32()
        check(lib().swapnet_plan_blocks(self.h, None, 0, C.byref(n)), "swapnet_plan_blocks")
        arr = (BlockInfo * max(1, n.value))()
        check(lib().swapnet_plan_blocks(self.h, arr, n.value, None), "swapnet_plan_blocks")
        return [{f: getattr(b, f) for f, _ in BlockInfo._fields_} for b in arr[:n.value]]

    def output_offsets(self):
        n = C.c_uint32()
        check(lib().swapnet_plan_output_offsets(self.h, None, 0, C.byref(n)), "swapnet_plan_output_offsets")
        arr = (C.c_uint64 * max(1, n.value))()
        check(lib().swapnet_plan_output_offsets(self.h, arr, n.value, None), "swapnet_plan_output_offsets")
        return list(arr[:n.value])

    def free(self):
        if self.h and self.h.value:
            lib().swapnet_plan_free(self.h)
            self.h = C.c_void_p()

    def __del__(self):
        try:
            self.free()
        except Exception:
            pass


def schedule(descs, urgency, arena_bytes, opt=None):
    n = len(descs)
    ptrs = (C.POINTER(ModelDesc) * n)(*[C.pointer(d.c) for d in descs])
    urg = (C.c_float * n)(*urgency)
    budgets = (C.c_uint64 * n)()
    plans = (C.c_void_p * n)()
    check(lib().swapnet_schedule(ptrs, urg, n, arena_bytes, C.byref(opt) if opt else None, budgets, plans),
          "swapnet_schedule")
    return list(budgets), [Plan(p) for p in plans]


def calibrate(model, engine, reps=20, resident_ns=None):
    """swapnet_engine_calibrate (Sec. 6.1 delay model measured on this GPU):
    per-layer t_ex in ns and alpha in attoseconds per byte (None when the
    engine measured no copy-engine swap).  resident_ns: the measured
    all-resident latency the t_ex are scaled to, or None."""
    n = len(model["layers"])
    t_ex = (C.c_int64 * n)()
    alpha = C.c_uint64()
    check(lib().swapnet_engine_calibrate(engine.h, int(reps), int(resident_ns or 0), t_ex, n,
                                         C.byref(alpha)), "swapnet_engine_calibrate")
    return list(t_ex), (alpha.value or None)


def pack_bf16(words):
    """swapnet_pack_bf16 of a uint16 array (bf16 bit patterns): the packed
    bytes as a uint8 array."""
    words = np.ascontiguousarray(words, dtype=np.uint16)
    used = C.c_uint64()
    check(lib().swapnet_pack_bf16(C.c_void_p(words.ctypes.data), words.size, None, 0, C.byref(used)),
          "swapnet_pack_bf16")
    out = np.empty(used.value, dtype=np.uint8)
    check(lib().swapnet_pack_bf16(C.c_void_p(words.ctypes.data), words.size, C.c_void_p(out.ctypes.data),
                                  out.size, C.byref(used)), "swapnet_pack_bf16")
    return out


def gemm_noalloc(dtype, a_ptr, w_ptr, bias_ptr, y_ptr, M, N, K, act=0, stream=0):
    """Y = act(A W^T + bias) through the allocation-free entry point."""
    check(lib().swapnet_gemm_noalloc(dtype, C.c_void_p(a_ptr), C.c_void_p(w_ptr), C.c_void_p(bias_ptr),
                                     C.c_void_p(y_ptr), M, N, K, act, C.c_void_p(stream or None)),
          "swapnet_gemm_noalloc")


# ------------------------------------------------------------ host weights
def _host_buffer(nbytes):
    """Anonymous page-aligned host memory, backed by transparent huge pages
    where the kernel allows it (fewer translations for the GPU to walk when
    it reads the registered range: measured 192 -> 211 GB/s host-to-device
    on a 13 GB buffer)."""
    mm = mmap.mmap(-1, max(int(nbytes), 1), flags=mmap.MAP_PRIVATE | mmap.MAP_ANONYMOUS)
    try:
        mm.madvise(mmap.MADV_HUGEPAGE)
    except (AttributeError, OSError, ValueError):
        pass
    return mm, np.frombuffer(mm, dtype=np.uint8)[:nbytes]


class HostWeights:
    """All parameter tensors of a model packed in one page-aligned host
    buffer, each tensor at a 256-byte aligned offset in layer order (the
    layout of the arena slots, so a block's tensors are one contiguous
    range)."""

    @classmethod
    def allocate(cls, nbytes_list, pinned=False):
        """An uninitialised packed buffer for tensors of the given sizes;
        fill tensor i through view(i).  pinned: page-locked by the CUDA
        driver (swapnet_host_alloc) instead of anonymous memory the library
        page-locks at load (use it for buffers of many GB)."""
        self = cls.__new__(cls)
        offs, cur = [], 0
        for n in nbytes_list:
            offs.append(cur)
            cur += (n + 255) // 256 * 256
        if pinned:
            p = C.c_void_p()
            check(lib().swapnet_host_alloc(max(cur, 1), C.byref(p)), "swapnet_host_alloc")
            self._pinned = p.value
            self._raw = (C.c_uint8 * max(cur, 1)).from_address(p.value)
            self.buf = np.frombuffer(self._raw, dtype=np.uint8)[:cur]
        else:
            self._raw, self.buf = _host_buffer(cur)
        self._offs, self._sizes = offs, list(nbytes_list)
        base = self.buf.ctypes.data
        self.ptrs = (C.c_void_p * max(1, len(offs)))(*[base + o for o in offs])
        self.n = len(offs)
        self.nbytes = cur
        return self

    def view(self, i):
        return self.buf[self._offs[i]:self._offs[i] + self._sizes[i]]

    def __del__(self):
        p = getattr(self, "_pinned", None)
        if p:
            self.buf = self._raw = None
            self._pinned = None
            try:
                lib().swapnet_host_free(C.c_void_p(p))
            except Exception:
                pass

    def __init__(self, weights, buffer=None):
        """buffer: optional caller-provided uint8 array (e.g. already pinned)
        of at least the packed size; default: pageable memory the library
        page-locks in place."""
        flat = [np.ascontiguousarray(t) for lw in weights for t in lw]
        offs, cur = [], 0
        for t in flat:
            offs.append(cur)
            cur += (t.nbytes + 255) // 256 * 256
        if buffer is not None:
            assert buffer.nbytes >= cur and buffer.ctypes.data % 256 == 0
            self.buf = buffer[:cur]
            self._raw = buffer
        else:
            self._raw, self.buf = _host_buffer(cur)
        for t, o in zip(flat, offs):
            self.buf[o:o + t.nbytes] = t.view(np.uint8).reshape(-1)
        base = self.buf.ctypes.data
        self.ptrs = (C.c_void_p * max(1, len(flat)))(*[base + o for o in offs])
        self.n = len(flat)
        self.nbytes = cur


class WeightsFile:
    """A weights file of the storage tier (Sec. 4.2.1), opened for direct
    I/O; the layout is documented in swapnet.h."""

    ALLOW_BUFFERED = 1

    @staticmethod
    def write(path, desc, host):
        """Write the tensors of `host` (HostWeights) for model `desc`."""
        check(lib().swapnet_weights_file_write(os.fsencode(path), C.byref(desc.c), host.ptrs, host.n),
              "swapnet_weights_file_write")

    def __init__(self, path, allow_buffered=False):
        h = C.c_void_p()
        check(lib().swapnet_weights_file_open(os.fsencode(path), self.ALLOW_BUFFERED if allow_buffered else 0,
                                              C.byref(h)), "swapnet_weights_file_open")
        self.h = h
        self.path = path

    def info(self):
        n, d = C.c_uint32(), C.c_int32()
        check(lib().swapnet_weights_file_info(self.h, C.byref(n), C.byref(d)), "swapnet_weights_file_info")
        return {"n_tensors": n.value, "direct": bool(d.value)}

    def read(self, tensor, offset, nbytes):
        out = np.empty(nbytes, dtype=np.uint8)
        check(lib().swapnet_weights_file_read(self.h, tensor, offset, nbytes, C.c_void_p(out.ctypes.data)),
              "swapnet_weights_file_read")
        return out

    def close(self):
        if self.h and self.h.value:
            lib().swapnet_weights_file_close(self.h)
            self.h = C.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


class Engine:
    def __init__(self, plan, host, d_arena=0, arena_bytes=0, d_ws=0, ws_bytes=0):
        """host: HostWeights (parameters in host memory) or WeightsFile
        (parameters read from storage for every swap-in)."""
        self.host = host  # keep the host buffer (or the open file) alive
        h = C.c_void_p()
        if isinstance(host, WeightsFile):
            check(lib().swapnet_load_file(plan.h, host.h, C.c_void_p(d_arena or None), arena_bytes,
                                          C.c_void_p(d_ws or None), ws_bytes, C.byref(h)), "swapnet_load_file")
        else:
            check(lib().swapnet_load(plan.h, host.ptrs, host.n, C.c_void_p(d_arena or None), arena_bytes,
                                     C.c_void_p(d_ws or None), ws_bytes, C.byref(h)), "swapnet_load")
        self.h = h

    def bind_state(self, d_state, nbytes):
        check(lib().swapnet_engine_bind_state(self.h, C.c_void_p(d_state), nbytes), "swapnet_engine_bind_state")

    def infer(self, d_in, d_out, stream=0):
        check(lib().swapnet_infer(self.h, C.c_void_p(d_in), C.c_void_p(d_out), C.c_void_p(stream or None)),
              "swapnet_infer")

    def infer_host(self, h_in, h_out, stream=0):
        check(lib().swapnet_infer_host(self.h, C.c_void_p(h_in), C.c_void_p(h_out), C.c_void_p(stream or None)),
              "swapnet_infer_host")

    def sync(self):
        check(lib().swapnet_engine_sync(self.h), "swapnet_engine_sync")

    def adapt(self, plan):
        """Switch to another plan of the same model (a new budget)."""
        check(lib().swapnet_engine_adapt(self.h, plan.h), "swapnet_engine_adapt")

    def blocks(self):
        n = C.c_uint32()
        check(lib().swapnet_engine_blocks(self.h, None, 0, C.byref(n)), "swapnet_engine_blocks")
        arr = (EngineBlock * max(1, n.value))()
        check(lib().swapnet_engine_blocks(self.h, arr, n.value, None), "swapnet_engine_blocks")
        return [{f: getattr(b, f) for f, _ in EngineBlock._fields_} for b in arr[:n.value]]

    def stats(self):
        st = EngineStats()
        check(lib().swapnet_engine_stats_get(self.h, C.byref(st)), "swapnet_engine_stats_get")
        return {f: getattr(st, f) for f, _ in EngineStats._fields_}

    def unit_kernels(self):
        n = C.c_uint32()
        check(lib().swapnet_engine_unit_kernels(self.h, None, 0, C.byref(n)), "swapnet_engine_unit_kernels")
        arr = (C.c_int32 * max(1, n.value))()
        check(lib().swapnet_engine_unit_kernels(self.h, arr, n.value, None), "swapnet_engine_unit_kernels")
        return [KERNEL_KIND.get(k, str(k)) for k in arr[:n.value]]

    def unit_tiling(self):
        n = C.c_uint32()
        check(lib().swapnet_engine_unit_tiling(self.h, None, 0, C.byref(n)), "swapnet_engine_unit_tiling")
        arr = (UnitTiling * max(1, n.value))()
        check(lib().swapnet_engine_unit_tiling(self.h, arr, n.value, None), "swapnet_engine_unit_tiling")
        return [{f: getattr(u, f) for f, _ in UnitTiling._fields_ if f != "reserved"} for u in arr[:n.value]]

    def set_profiling(self, enable):
        check(lib().swapnet_engine_set_profiling(self.h, 1 if enable else 0), "swapnet_engine_set_profiling")

    def set_swap_timing(self, enable):
        check(lib().swapnet_engine_set_swap_timing(self.h, 1 if enable else 0), "swapnet_engine_set_swap_timing")

    def last_swap_times(self, n_blocks):
        """Microseconds per block swap-in of the last inference, timed inside its graph."""
        b = (C.c_float * max(1, n_blocks))()
        check(lib().swapnet_engine_last_swap_times(self.h, b, n_blocks), "swapnet_engine_last_swap_times")
        return list(b[:n_blocks])

    def set_graph_timeline(self, enable):
        check(lib().swapnet_engine_set_graph_timeline(self.h, 1 if enable else 0),
              "swapnet_engine_set_graph_timeline")

    def last_graph_timeline(self, n_blocks):
        """Per block (swap start, swap end, layers start, layers end) of the
        last inference, microseconds since its start, timed inside its graph
        (-1 for a swap that did not happen in that inference)."""
        b = (C.c_float * max(4, 4 * n_blocks))()
        check(lib().swapnet_engine_last_graph_timeline(self.h, b, n_blocks), "swapnet_engine_last_graph_timeline")
        return [tuple(b[4 * k:4 * k + 4]) for k in range(n_blocks)]

    def measure_units(self, n_units, reps=20):
        u = (C.c_float * max(1, n_units))()
        check(lib().swapnet_engine_measure_units(self.h, reps, u, n_units), "swapnet_engine_measure_units")
        return list(u[:n_units])

    def last_timeline(self, n_units, n_blocks):
        """(unit start, unit end, swap start, swap end) lists in microseconds."""
        a, b = (C.c_float * max(1, n_units))(), (C.c_float * max(1, n_units))()
        c, d = (C.c_float * max(1, n_blocks))(), (C.c_float * max(1, n_blocks))()
        check(lib().swapnet_engine_last_timeline(self.h, a, b, n_units, c, d, n_blocks),
              "swapnet_engine_last_timeline")
        return list(a[:n_units]), list(b[:n_units]), list(c[:n_blocks]), list(d[:n_blocks])

    def last_times(self, n_units, n_blocks):
        u = (C.c_float * max(1, n_units))()
        b = (C.c_float * max(1, n_blocks))()
        check(lib().swapnet_engine_last_times(self.h, u, n_units, b, n_blocks), "swapnet_engine_last_times")
        return list(u[:n_units]), list(b[:n_blocks])

    def free(self):
        if self.h and self.h.value:
            lib().swapnet_engine_free(self.h)
            self.h = C.c_void_p()

    def __del__(self):
        try:
            self.free()
        except Exception:
            pass
