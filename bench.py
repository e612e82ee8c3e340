"""Benchmark of block-swapped inference on one GB300 (or N replicas).

A step is one swapped inference of the workload: every block's weights are
swapped from pinned host memory into the two-slot device arena and every
layer runs from the arena.  Default workload: the LLaMA-7B-shaped bf16
decoder (13.5 GB of weights) through a 4e9-byte weight arena, one step =
the prefill of 512 token ids plus 32 greedy decode passes; every other
workload (the MLP, ResNet-50, VGG-16 at batch 1 and 16, YOLOv3, the
multi-DNN mix) is measured after it in the same call and reported under
the line's `configs` key (--configs none skips them).

Reported (one JSON line, rank 0):
  value        whole-job inferences/s (device-timed, inputs resident in HBM)
  ms_per_step  swapped latency; dinf_ms the all-resident latency with the
               same kernels; ratio = swapped / DInf
  e2e          the same metric through swapnet_infer_host (host input and
               output buffers, copies inside the timed region)
  link         host-to-device bytes per swap-in over the swap time, against
               the measured pinned cudaMemcpy peak
  roofline     the dominant kernel's algorithmic FLOPs (or bytes) per launch
               over its CUDA-event launch duration, against MEASURED_PEAKS.json
  cpu_baseline the float64 CPU oracle on a bounded sample of the workload
L2 is flushed (a 512 MiB write) before every timed step; the flush is not
timed.  Replicas only: with torchrun each rank runs its own engine on its own
GPU with no collective on the data path.
"""
import argparse
import json
import mmap
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "swapped/DInf latency ratio and ms/inference at budget; host-link GB/s vs peak (1 GB300)"

CONFIGS = {
    # name: (builder, budget fraction of weight bytes, slots, activations in budget, workload text)
    "resnet50": ("resnet50", dict(batch=1), 0.40,
                 "ResNet-50-shaped CNN, fp16, batch 1, 1x3x224x224, budget 40% of weight bytes"),
    "mlp6": ("mlp6", dict(batch=8), None,
             "6-layer MLP width 1024 fp32 batch 8, budget = 2 layers of weights + 2 activation buffers"),
    "vgg16_b1": ("vgg16", dict(batch=1), 0.25, "VGG-16-shaped CNN, fp16, batch 1, budget 25% of weight bytes"),
    "vgg16_b16": ("vgg16", dict(batch=16), 0.25, "VGG-16-shaped CNN, fp16, batch 16, budget 25% of weight bytes"),
    "yolov3": ("yolov3", dict(batch=1), 0.30, "YOLOv3 (Darknet-53 + 3 heads), fp16, 1x3x416x416, budget 30%"),
    "multi": ("multi", {}, 0.30, "ResNet-50 + VGG-16 + YOLOv3 (fp16, batch 1), concurrent closed-loop request "
              "streams, one arena of 30% of the summed weight bytes split by Eq. 1"),
    "llm": ("llm", dict(tokens=512), None,
            "LLaMA-7B-shaped decoder bf16 (32 layers, d 4096, 32 heads, FFN 11008, vocab 32000); "
            "prefill 512 token ids + 32 greedy decode steps, batch 1; 4e9-byte weight arena"),
}


# swap variants by name (--variant); "direct" reads SIMT-only blocks in place
VARIANTS = ("auto", "memcpy", "zerocopy", "direct", "packed")


def variant_code(name):
    from paper_2401_16757_gb300 import capi
    return {"auto": capi.SWAP_AUTO, "memcpy": capi.SWAP_MEMCPY, "zerocopy": capi.SWAP_ZEROCOPY,
            "direct": capi.SWAP_DIRECT, "packed": capi.SWAP_PACKED}[name]

# DRAM traffic per launch of a kernel family, from ncu (dram__bytes_read.sum
# + dram__bytes_write.sum averaged over the launches of one swapped step of
# the named workload), valid only for the tensor-core sources it was taken on
# (traffic_sources_sha).
TRAFFIC = {
    ("resnet50", "tc_gemm"): ("1bb9110c06be", 1418599),
    ("resnet50", "tc_conv"): ("1bb9110c06be", 1807876),
    # zero-copy swap: bytes of a launch's output still in L2 when it ends
    # (DRAM writes = block bytes - this, from an ncu capture of two smaller launches)
    ("llm", "zerocopy_kernel"): ("d2d45db9fdff", 63_400_000),
}


class RankGroup:
    """Replicas under torchrun: each rank runs its own engine on its own GPU
    and nothing crosses ranks on the data path; the group only brackets the
    timed region with barriers and takes the slowest rank's time.  One rank:
    no process group, every call is a no-op."""

    def __init__(self, world, local=0, backend="nccl"):
        self.world = world
        self.dist = None
        self.backend = backend
        if world > 1:
            import torch
            import torch.distributed as dist
            if not dist.is_initialized():
                if backend == "nccl":
                    dist.init_process_group("nccl", device_id=torch.device("cuda", local))
                else:
                    dist.init_process_group(backend)
            self.dist = dist

    def barrier(self):
        if self.dist:
            self.dist.barrier()

    def max(self, x):
        """The largest x over the ranks (x on this rank)."""
        if not self.dist:
            return float(x)
        import torch
        t = torch.tensor([float(x)], dtype=torch.float64, device="cuda" if self.backend == "nccl" else "cpu")
        self.dist.all_reduce(t, op=self.dist.ReduceOp.MAX)
        return float(t.item())

    def close(self):
        if self.dist:
            self.dist.destroy_process_group()
            self.dist = None


def sources_sha(files):
    import hashlib
    h = hashlib.sha1()
    for f in files:
        with open(os.path.join(ROOT, "paper_2401_16757_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:12]


def kernel_sources_sha():
    """Tag of every layer-kernel source (names the sources a profile was taken on)."""
    return sources_sha(("k_tc.cu", "k_tc_persist.cu", "k_tc_small.cu", "tc_epi.cuh", "k_simt.cu", "k_decoder.cu",
                        "device.cuh"))


def traffic_sources_sha():
    """Tag of the sources the tensor-core GEMM family is compiled from: its
    TRAFFIC figures stay valid while these are unchanged."""
    return sources_sha(("k_tc.cu", "k_tc_persist.cu", "tc_epi.cuh", "device.cuh", "kernels.h", "internal.h"))


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            d = json.load(f)
        return d["hbm_gbs"], d["bf16_tflops"], d.get("bf16_tflops_sustained"), "measured"
    except Exception:
        return 6800.0, 1900.0, 1700.0, "fallback"


class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, index, interval_ms=100):
        # polling nvidia-smi itself disturbs the host link (measured: a
        # link-bound 7B decode pass went from 63 to 67-100 ms under 50 ms
        # polling), so poll no faster than needed to see the clocks
        self.index = index
        self.interval_ms = interval_ms
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), "--query-gpu=" + self.FIELDS,
                                          "--format=csv,noheader,nounits", "-lms", str(self.interval_ms)],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                mx.append(float(parts[1]))
            except ValueError:
                continue
            for nm, v in zip(names, parts[4:8]):
                if v.lower() == "active":
                    reasons.add(nm)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(sm)}


def cpu_oracle_baseline(model, weights, x, budget_s=12.0, max_runs=5):
    """The float64 oracle as it stands, timed on the host cores on a bounded
    sample (whole inferences until budget_s seconds of CPU work)."""
    from oracle import forward as F
    t0 = time.perf_counter()
    runs = 0
    while runs < max_runs:
        F.forward(model, weights, x)
        runs += 1
        if time.perf_counter() - t0 > budget_s:
            break
    dt = time.perf_counter() - t0
    cores = len(os.sched_getaffinity(0))
    return {"value": runs / dt, "unit": "inferences/s", "cores": cores, "kind": "oracle",
            "sample": "%d whole float64 inference(s) of the same workload (numpy, BLAS threads = %d cores)"
                      % (runs, cores)}


def build_workload(name, weight_bytes_fn):
    """The workload's structure, weights, input and budget.  weight_bytes_fn
    gives the 256-byte-aligned weight bytes (the library's plan query on the
    GPU leg; the oracle's count on the reference leg)."""
    import synth
    arch, kw, frac, text = CONFIGS[name]
    m = synth.arch.MODELS[arch](**kw)
    w = synth.gen.model_weights(m)
    x = synth.gen.model_input(m)
    wb = weight_bytes_fn(m)
    if frac is None:
        budget = 8_462_336
    else:
        budget = int(wb * frac) // 256 * 256
    return m, w, x, wb, budget, text


def capi_weight_bytes(m):
    from paper_2401_16757_gb300 import capi
    return capi.Plan.resident(capi.Desc(m)).info()["weight_bytes"]


def unit_algorithmic_bytes(m, units):
    """Bytes each unit must move at least once: its parameters, its inputs
    (every source and the residual) and its output, for a linear piece the
    share of the output it writes.  CNN and MLP layer types only."""
    es = {"f32": 4, "f16": 2, "bf16": 2}[m["dtype"]]
    shapes = []

    def shp(i):
        return tuple(m["input"]) if i == -1 else shapes[i]

    for L in m["layers"]:
        n, h, w, c = shp(L["src"][0])
        op = L["op"]
        if op in ("conv", "maxpool"):
            ho = (h + 2 * L["pad"] - L["kh"]) // L["stride"] + 1
            wo = (w + 2 * L["pad"] - L["kw"]) // L["stride"] + 1
            shapes.append((n, ho, wo, L["cout"] if op == "conv" else c))
        elif op == "linear":
            shapes.append((n, 1, 1, L["n"]))
        elif op == "gap":
            shapes.append((n, 1, 1, c))
        elif op == "upsample2x":
            shapes.append((n, 2 * h, 2 * w, c))
        elif op == "concat":
            shapes.append((n, h, w, c + shp(L["src"][1])[3]))
        else:
            return None
    out = []
    for u in units:
        L = m["layers"][u["layer"]]
        frac = u["rows"] / L["n"] if L["op"] == "linear" and u["rows"] else 1.0
        srcs = list(L["src"]) + ([L["res"]] if L.get("res") is not None else [])
        b = u["bytes"] + sum(int(np.prod(shp(s))) * es for s in srcs) + int(np.prod(shapes[u["layer"]])) * es * frac
        out.append(int(b))
    return out


def oracle_weight_bytes(m):
    from oracle import plan as OP
    return OP.weight_bytes(m)


def llm_host_weights(model, threads=16):
    """The 7B weights generated in parallel straight into the packed buffer."""
    import concurrent.futures as cf
    import synth
    from paper_2401_16757_gb300 import capi
    jobs, sizes = [], []
    for li, L in enumerate(model["layers"]):
        for ti, (_, shp) in enumerate(synth.arch.tensor_shapes(L)):
            jobs.append((li, ti, shp))
            sizes.append(int(np.prod(shp)) * 2)
    host = capi.HostWeights.allocate(sizes, pinned=True)

    def fill(k):
        li, ti, shp = jobs[k]
        host.view(k)[:] = synth.gen.llm_tensor(model, li, ti, shp).view(np.uint8).reshape(-1)

    with cf.ThreadPoolExecutor(threads) as ex:
        list(ex.map(fill, range(len(jobs))))
    return host


def llm_cpu_sample(n_dec_sample=2):
    """The float64 oracle on a bounded sample of the 7B workload: a model of
    the same widths with ONE decoder layer runs the 512-token prefill and
    n_dec_sample decode tokens; the embedding, layer and head parts are timed
    separately and scaled to 32 layers and 32 decode tokens.  Returns
    (seconds per whole inference, description)."""
    return llm_cpu_sampler()(n_dec_sample)


def llm_cpu_sampler():
    """The one-layer model and its weights of llm_cpu_sample, generated once
    (untimed); returns the sample function, which runs on a fresh KV state
    at every call."""
    import synth
    from oracle import forward as F
    m1 = synth.arch.llm(layers=1, tokens=512)
    w = synth.gen.model_weights(m1)
    ids = synth.gen.model_input(m1)
    nl = len(m1["layers"])
    return lambda n_dec_sample=2: _llm_cpu_run(F, m1, w, ids, nl, n_dec_sample)


def _llm_cpu_run(F, m1, w, ids, nl, n_dec_sample):
    state = F.new_state()

    def parts(x):
        acts, t = {}, []
        for lo, hi in ((0, 1), (1, nl - 3), (nl - 3, nl)):
            t0 = time.perf_counter()
            F.forward_range(m1, w, acts, np.asarray(x), lo, hi, state)
            t.append(time.perf_counter() - t0)
        state["pos"] += int(np.asarray(x).shape[0])
        return t, int(acts[nl - 1].reshape(-1)[-1])

    tp, tok = parts(ids)
    td = [0.0, 0.0, 0.0]
    for _ in range(n_dec_sample):
        t, tok = parts(np.array([[[[tok]]]], dtype=np.int32))
        td = [a + b for a, b in zip(td, t)]
    per_dec = [v / n_dec_sample for v in td]
    total = (tp[0] + 32 * tp[1] + tp[2]) + 32 * (per_dec[0] + 32 * per_dec[1] + per_dec[2])
    return total, ("float64 oracle, one 4096-wide decoder layer (+ embedding and LM head) over the 512-token "
                   "prefill and %d decode tokens, scaled to 32 layers and 32 decode tokens" % n_dec_sample)


def decoder_unit_bytes(model, units, positions):
    """Algorithmic bytes of each unit of a decoder pass over `positions`
    cached positions after it: parameters, every input read and the output
    written, each once (the attention layer reads the cached keys and values
    of all positions once)."""
    es = 2
    rows = model["input"][0]
    width = {}
    out = []
    for u in units:
        L = model["layers"][u["layer"]]
        op = L["op"]
        if op == "embed":
            b = 2 * rows * L["d"] * es            # rows gathered from the host table, written
            width[u["layer"]] = L["d"]
        elif op == "rmsnorm":
            b = u["bytes"] + 2 * rows * L["d"] * es
            width[u["layer"]] = L["d"]
        elif op == "linear":
            frac = u["rows"] / L["n"] if u["rows"] else 1.0
            # input rows, output rows, and the residual (or SwiGLU gate) rows
            outs = 2 if L.get("res") is not None else 1
            b = u["bytes"] + rows * L["k"] * es + outs * rows * L["n"] * es * frac
            width[u["layer"]] = L["n"]
        elif op == "attention":
            d = width[L["src"][0]]
            b = 4 * rows * d * es + 2 * positions * d * es   # q, k, v in, out; the whole cache read
            width[u["layer"]] = d
        elif op == "argmax":
            b = rows * width[L["src"][0]] * es + rows * 4
        else:
            b = u["bytes"]
        out.append(int(b))
    return out


def run_llm(args, rank, world, group):
    """Config 5: prefill of 512 ids then 32 greedy decode steps per step."""
    import torch
    import synth
    from paper_2401_16757_gb300 import capi
    text = CONFIGS["llm"][3]
    t0 = time.perf_counter()
    mp, md = synth.arch.llm(tokens=512), synth.arch.llm(tokens=1)
    host = llm_host_weights(mp)
    t_gen = time.perf_counter() - t0
    stream = torch.cuda.current_stream()
    sp = stream.cuda_stream
    placement = {}
    link_peak = measure_link_peak(stream, placement)
    alpha = int(round(1e18 / (link_peak * 1e9)))
    budget = 4_000_000_000
    variant = variant_code(args.variant)
    opt = capi.options(swap_variant=variant, alpha_as_per_byte=alpha, beta_ns_per_tensor=0, merge=args.merge)
    dp, dd = capi.Desc(mp), capi.Desc(md)
    t1 = time.perf_counter()
    pp, pd = capi.Plan.partition(dp, budget, opt), capi.Plan.partition(dd, budget, opt)
    t_plan = time.perf_counter() - t1
    ip, idd = pp.info(), pd.info()
    ep, ed = capi.Engine(pp, host), capi.Engine(pd, host)
    rpp = capi.Plan.resident(dp, capi.options(merge=args.merge))
    rdp = capi.Plan.resident(dd, capi.options(preloaded=1, merge=args.merge))
    arena = torch.empty(rpp.info()["arena_bytes"], dtype=torch.uint8, device="cuda")
    rp = capi.Engine(rpp, host, d_arena=arena.data_ptr(), arena_bytes=arena.numel())
    rd = capi.Engine(rdp, host, d_arena=arena.data_ptr(), arena_bytes=arena.numel())
    state = torch.zeros(ip["state_bytes"], dtype=torch.uint8, device="cuda")
    for e in (ep, ed, rp, rd):
        e.bind_state(state.data_ptr(), ip["state_bytes"])
    ids = synth.gen.model_input(mp).reshape(-1)
    in_p = torch.from_numpy(ids.view(np.uint8).copy()).cuda()
    out_p = torch.zeros(ip["output_bytes"], dtype=torch.uint8, device="cuda")
    tok = torch.zeros(16, dtype=torch.uint8, device="cuda")
    out_d = torch.zeros(idd["output_bytes"], dtype=torch.uint8, device="cuda")
    offs_p, offs_d = pp.output_offsets(), pd.output_offsets()
    n_dec = 32

    def one(eng_p, eng_d, evs=None, after_pass=None):
        state[:256].zero_()
        if evs: evs[0].record(stream)
        eng_p.infer(in_p.data_ptr(), out_p.data_ptr(), sp)
        if after_pass: after_pass(0)
        if evs: evs[1].record(stream)
        tok[:4].copy_(out_p[offs_p[1] + 511 * 4:offs_p[1] + 512 * 4])
        for _ in range(n_dec):
            eng_d.infer(tok.data_ptr(), out_d.data_ptr(), sp)
            if after_pass: after_pass(1)
            tok[:4].copy_(out_d[offs_d[1]:offs_d[1] + 4])
        if evs: evs[2].record(stream)

    def timed(eng_p, eng_d, steps):
        res = []
        for _ in range(steps):
            evs = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
            one(eng_p, eng_d, evs)
            torch.cuda.synchronize()
            res.append((evs[0].elapsed_time(evs[1]), evs[1].elapsed_time(evs[2]) / n_dec))
        return res

    # the link check and the clock sampler start before the warm-up: a fresh
    # page-locked allocation right before the timed steps made the next
    # prefill pass 5x slower (the host mappings are walked again)
    link_before = measure_link_peak(stream)
    clocks = ClockSampler(int(os.environ.get("LOCAL_RANK", "0")), interval_ms=500)
    clocks.start()
    for _ in range(max(1, args.warmup)):
        one(ep, ed)
        one(rp, rd)
    torch.cuda.synchronize()
    for e in (ep, ed, rp, rd):
        e.sync()
    launches0 = ep.stats()["kernel_launches"] + ed.stats()["kernel_launches"]
    group.barrier()
    torch.cuda.nvtx.range_push("swapped_steps")  # ncu --nvtx --nvtx-include swapped_steps/
    sw = timed(ep, ed, args.steps)
    torch.cuda.nvtx.range_pop()
    group.barrier()
    launches = ep.stats()["kernel_launches"] + ed.stats()["kernel_launches"] - launches0
    di = timed(rp, rd, args.steps)
    clk = clocks.stop()
    link_after = measure_link_peak(stream)
    # greedy tokens agree between swapped and resident runs
    one(ep, ed); torch.cuda.synchronize(); sw_tok = int(tok[:4].cpu().numpy().view(np.int32)[0])
    one(rp, rd); torch.cuda.synchronize(); rs_tok = int(tok[:4].cpu().numpy().view(np.int32)[0])

    # ---- the dominant kernel: one step with profiling on (eager launches,
    # events around every unit kernel and every block's swap-in on the copy
    # stream); per pass, per-block swap times and per-unit kernel times
    units_p, units_d = pp.units(), pd.units()
    kinds_p, kinds_d = ep.unit_kernels(), ed.unit_kernels()
    blocks_p, blocks_d = pp.blocks(), pd.blocks()
    var_p = [b["variant"] for b in ep.blocks()]
    var_d = [b["variant"] for b in ed.blocks()]
    prof = {"swap": [], "kern": {}}

    def collect(which):
        eng, units, blocks, kinds, var = ((ep, units_p, blocks_p, kinds_p, var_p) if which == 0
                                          else (ed, units_d, blocks_d, kinds_d, var_d))
        u_us, s_us = eng.last_times(len(units), len(blocks))
        for b, t, v in zip(blocks, s_us, var):
            prof["swap"].append((b["bytes"], t, v))
        for k, t in zip(kinds, u_us):
            prof["kern"][k] = prof["kern"].get(k, 0.0) + t

    for e in (ep, ed):
        e.set_profiling(True)
    one(ep, ed, after_pass=collect)
    torch.cuda.synchronize()
    for e in (ep, ed):
        e.set_profiling(False)
    # the swap kernel's own time inside the replayed graphs: one more step
    # whose graphs carry an event-record node before and after every block's
    # swap-in on the copy stream (the layer launches are those of the timed
    # steps)
    gswap = []

    def collect_graph(which):
        eng, blocks, var = (ep, blocks_p, var_p) if which == 0 else (ed, blocks_d, var_d)
        for b, t, v in zip(blocks, eng.last_swap_times(len(blocks)), var):
            gswap.append((b["bytes"], t, v))

    for e in (ep, ed):
        e.set_swap_timing(True)
    one(ep, ed)
    torch.cuda.synchronize()
    one(ep, ed, after_pass=collect_graph)
    torch.cuda.synchronize()
    for e in (ep, ed):
        e.set_swap_timing(False)
    zc = [(b, t) for b, t, v in gswap if v == capi.SWAP_ZEROCOPY and t > 0]
    swap_us_step = sum(t for _, t, _ in gswap)
    step_us = (statistics.mean(r[0] for r in sw) + n_dec * statistics.mean(r[1] for r in sw)) * 1e3
    if zc:
        zb, zt = sum(b for b, _ in zc), sum(t for _, t in zc)
        zc_us_step = zt
        ach = zb / (zt * 1e-6) / 1e9
        roofline = {
            "bound": "host_link", "kernel": "zerocopy_kernel", "achieved": ach, "peak": link_peak, "unit": "GB/s",
            "frac": ach / link_peak,
            "peak_source": "pinned cudaMemcpy H2D of 256 MiB measured in this run (MEASURED_PEAKS.json has no "
                           "host-link figure)",
            "launches_per_step": len(zc), "algorithmic_bytes_per_launch": zb // len(zc),
            "us_per_launch": zt / len(zc), "us_per_step": zt, "step_us": step_us,
            "timing": "CUDA events recorded inside the replayed inference graphs (event-record nodes on the copy "
                      "stream around each block's swap-in), one step after the timed steps; step_us is the timed "
                      "steps' mean",
            "share_of_step": zt / step_us,
            "eager_profiled_us_per_step": sum(t for b, t, v in prof["swap"] if v == capi.SWAP_ZEROCOPY),
            "kernel_time_share_eager": {k: round(v / (zt + sum(prof["kern"].values())), 4)
                                        for k, v in list(prof["kern"].items()) + [("zerocopy_kernel", zt)]},
            "traffic": None}
        tr = TRAFFIC.get(("llm", "zerocopy_kernel"))
        if tr and tr[0] == sources_sha(("k_swap.cu",)):
            roofline["traffic"] = int(zb // len(zc) - tr[1])
            roofline["traffic_note"] = ("ncu DRAM bytes of two smaller launches (224 and 315 MB blocks): reads ~0, "
                                        "writes = block bytes minus ~63 MB still in L2 at the kernel's end; "
                                        "applied to this line's mean launch")
    else:
        roofline = None

    # ---- the resident (DInf) kernels: every unit timed as a graph of 20
    # back-to-back launches, grouped by kernel family, per decoder step.
    # The units read the state's position: the prefill's units are timed at
    # position 0, the decode pass's at 512 (the attention over 513 keys,
    # near the middle of the 32 decode passes)
    hbm, tf_burst, tf_sust, peak_src = load_peaks()
    torch.cuda.synchronize()
    state[:256].zero_()
    us_rp = np.array(rp.measure_units(len(rpp.units()), 20))
    state[:4].copy_(torch.tensor([512], dtype=torch.int32).view(torch.uint8))
    us_rd = np.array(rd.measure_units(len(rdp.units()), 20))
    torch.cuda.synchronize()
    rp.sync()
    rd.sync()
    fam_p = kernel_rooflines(rp.unit_kernels(), rpp.units(), us_rp, decoder_unit_bytes(mp, rpp.units(), 512),
                             hbm, tf_burst, peak_src)
    fam_d = kernel_rooflines(rd.unit_kernels(), rdp.units(), us_rd, decoder_unit_bytes(md, rdp.units(), 528),
                             hbm, tf_burst, peak_src)

    # e2e through swapnet_infer_host: the token ids from pinned host memory,
    # every pass's output back to the host, and each greedy token taken from
    # the host copy for the next decode pass
    h_ids = torch.from_numpy(ids.view(np.uint8).copy()).pin_memory()
    h_out_p = torch.empty(ip["output_bytes"], dtype=torch.uint8).pin_memory()
    h_tok = torch.zeros(16, dtype=torch.uint8).pin_memory()
    h_out_d = torch.empty(idd["output_bytes"], dtype=torch.uint8).pin_memory()

    def one_host():
        state[:256].zero_()
        ep.infer_host(h_ids.data_ptr(), h_out_p.data_ptr(), sp)
        stream.synchronize()
        h_tok[:4].copy_(h_out_p[offs_p[1] + 511 * 4:offs_p[1] + 512 * 4])
        for _ in range(n_dec):
            ed.infer_host(h_tok.data_ptr(), h_out_d.data_ptr(), sp)
            stream.synchronize()
            h_tok[:4].copy_(h_out_d[offs_d[1]:offs_d[1] + 4])

    one_host()
    e2e_steps = min(args.steps, 5)
    e2e_ms = []
    for _ in range(e2e_steps):
        t0 = time.perf_counter()
        one_host()
        e2e_ms.append((time.perf_counter() - t0) * 1e3)
    e2e_step_ms = group.max(statistics.mean(e2e_ms))
    e2e_tok_equal = int(h_tok[:4].numpy().view(np.int32)[0]) == sw_tok
    # extension (not the paper's method): resident-prefix plans in the same budget
    opt_rp = capi.options(swap_variant=variant, alpha_as_per_byte=alpha, beta_ns_per_tensor=0, resident_prefix=1,
                          merge=args.merge)
    pp_rp, pd_rp = capi.Plan.partition(dp, budget, opt_rp), capi.Plan.partition(dd, budget, opt_rp)
    ep.free(); ed.free()
    ep_rp, ed_rp = capi.Engine(pp_rp, host), capi.Engine(pd_rp, host)
    for e_ in (ep_rp, ed_rp):
        e_.bind_state(state.data_ptr(), ip["state_bytes"])
    one(ep_rp, ed_rp)
    torch.cuda.synchronize()
    rp_t = timed(ep_rp, ed_rp, min(args.steps, 3))
    ext_rp = {"prefill_ms": statistics.mean(r[0] for r in rp_t),
              "decode_ms_per_token": statistics.mean(r[1] for r in rp_t),
              "prefix_units": [pp_rp.info()["prefix_units"], pd_rp.info()["prefix_units"]],
              "prefix_bytes": [pp_rp.info()["prefix_bytes"], pd_rp.info()["prefix_bytes"]], "steps": len(rp_t)}
    ext_rp["ms_per_step"] = ext_rp["prefill_ms"] + n_dec * ext_rp["decode_ms_per_token"]
    one(ep_rp, ed_rp); torch.cuda.synchronize()
    ext_rp["greedy_token_equals_resident"] = int(tok[:4].cpu().numpy().view(np.int32)[0]) == rs_tok
    ep_rp.free(); ed_rp.free()
    # extension (not the paper's method): the packed swap variant on the same
    # plans (bf16 tensors packed losslessly at load, unpacked into the arena
    # by an SM kernel, so fewer bytes cross the host link)
    opt_pk = capi.options(swap_variant=capi.SWAP_PACKED, alpha_as_per_byte=alpha, beta_ns_per_tensor=0,
                          merge=args.merge)
    pp_pk, pd_pk = capi.Plan.partition(dp, budget, opt_pk), capi.Plan.partition(dd, budget, opt_pk)
    t_pk = time.perf_counter()
    ep_pk, ed_pk = capi.Engine(pp_pk, host), capi.Engine(pd_pk, host)
    pack_s = time.perf_counter() - t_pk
    for e_ in (ep_pk, ed_pk):
        e_.bind_state(state.data_ptr(), ip["state_bytes"])
    one(ep_pk, ed_pk)
    torch.cuda.synchronize()
    st0 = [ep_pk.stats(), ed_pk.stats()]
    pk_t = timed(ep_pk, ed_pk, min(args.steps, 3))
    st1 = [ep_pk.stats(), ed_pk.stats()]
    pk_link = sum(b["link_bytes"] - a["link_bytes"] for a, b in zip(st0, st1)) / len(pk_t)
    pk_swapped = sum(b["bytes_swapped"] - a["bytes_swapped"] for a, b in zip(st0, st1)) / len(pk_t)
    ext_pk = {"prefill_ms": statistics.mean(r[0] for r in pk_t),
              "decode_ms_per_token": statistics.mean(r[1] for r in pk_t), "steps": len(pk_t),
              "load_s_with_packing": pack_s,
              "link_bytes_per_step": pk_link, "bytes_swapped_per_step": pk_swapped,
              "packed_fraction": pk_link / pk_swapped if pk_swapped else None,
              "variants": [[b["variant"] for b in ep_pk.blocks()], [b["variant"] for b in ed_pk.blocks()]]}
    ext_pk["ms_per_step"] = ext_pk["prefill_ms"] + n_dec * ext_pk["decode_ms_per_token"]
    ext_pk["link_gbs"] = pk_link / (ext_pk["ms_per_step"] * 1e-3) / 1e9
    ext_pk["link_frac"] = ext_pk["link_gbs"] / link_peak
    one(ep_pk, ed_pk); torch.cuda.synchronize()
    ext_pk["greedy_token_equals_resident"] = int(tok[:4].cpu().numpy().view(np.int32)[0]) == rs_tok
    # both extensions together: a resident prefix, the rest swapped packed
    # (the packed images are shared with the engines above)
    opt_pp = capi.options(swap_variant=capi.SWAP_PACKED, alpha_as_per_byte=alpha, beta_ns_per_tensor=0,
                          resident_prefix=1, merge=args.merge)
    ep_pp, ed_pp = capi.Engine(capi.Plan.partition(dp, budget, opt_pp), host), \
        capi.Engine(capi.Plan.partition(dd, budget, opt_pp), host)
    ep_pk.free(); ed_pk.free()
    for e_ in (ep_pp, ed_pp):
        e_.bind_state(state.data_ptr(), ip["state_bytes"])
    one(ep_pp, ed_pp)
    torch.cuda.synchronize()
    pp_t = timed(ep_pp, ed_pp, min(args.steps, 3))
    ext_pk["with_resident_prefix"] = {"prefill_ms": statistics.mean(r[0] for r in pp_t),
                                      "decode_ms_per_token": statistics.mean(r[1] for r in pp_t),
                                      "steps": len(pp_t)}
    ext_pk["with_resident_prefix"]["ms_per_step"] = (ext_pk["with_resident_prefix"]["prefill_ms"] +
                                                     n_dec * ext_pk["with_resident_prefix"]["decode_ms_per_token"])
    one(ep_pp, ed_pp); torch.cuda.synchronize()
    ext_pk["with_resident_prefix"]["greedy_token_equals_resident"] = \
        int(tok[:4].cpu().numpy().view(np.int32)[0]) == rs_tok
    ep_pp.free(); ed_pp.free()
    pre_ms = statistics.mean(r[0] for r in sw)
    dec_ms = statistics.mean(r[1] for r in sw)
    pre_d = statistics.mean(r[0] for r in di)
    dec_d = statistics.mean(r[1] for r in di)
    step_ms = group.max(pre_ms + n_dec * dec_ms)  # the slowest rank
    dinf_ms = pre_d + n_dec * dec_d
    swap_bytes_p = sum(b["bytes"] for b in blocks_p)
    swap_bytes_d = sum(b["bytes"] for b in blocks_d)
    bytes_step = swap_bytes_p + n_dec * swap_bytes_d
    bound_ms = bytes_step / (link_peak * 1e9) * 1e3
    unit = "inferences/s (prefill 512 + 32 decode)"
    line = {
        "metric": METRIC, "value": world * 1000.0 / step_ms, "unit": unit,
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup, "ms_per_step": step_ms,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": text, "budget_bytes": budget, "weight_bytes": ip["weight_bytes"],
                   "prefill_blocks": ip["n_blocks"], "decode_blocks": idd["n_blocks"],
                   "plans_exact": [ip["exact"], idd["exact"]], "l2": "inputs (13.2 GB of weights) larger than L2",
                   "swap_variant": args.variant, "swap_variants_prefill": var_p, "swap_variants_decode": var_d,
                   "merged_gemv_launches": args.merge, "state_bytes": ip["state_bytes"]},
        "prefill_ms": pre_ms, "decode_ms_per_token": dec_ms, "dinf_prefill_ms": pre_d,
        "dinf_decode_ms_per_token": dec_d, "dinf_ms": dinf_ms, "ratio": step_ms / dinf_ms,
        "greedy_token_swapped_equals_resident": sw_tok == rs_tok,
        "e2e": {"value": world * 1000.0 / e2e_step_ms, "unit": unit, "steps": e2e_steps,
                "h2d_bytes_per_step": ip["input_bytes"] + n_dec * idd["input_bytes"],
                "d2h_bytes_per_step": ip["output_bytes"] + n_dec * idd["output_bytes"],
                "greedy_token_equals_device_run": e2e_tok_equal},
        "link": {"achieved_gbs": bytes_step / (step_ms * 1e-3) / 1e9, "peak_gbs": link_peak,
                 "peak_source": "pinned cudaMemcpy H2D 256 MiB", "bytes_per_step": bytes_step,
                 "swap_busy_gbs": bytes_step / (swap_us_step * 1e-6) / 1e9 if swap_us_step > 0 else None,
                 "peak_before_after_gbs": [link_before, link_after], "host_placement": placement},
        "per_step": {"prefill_ms": [r[0] for r in sw], "decode_ms_per_token": [r[1] for r in sw],
                     "dinf_prefill_ms": [r[0] for r in di], "dinf_decode_ms_per_token": [r[1] for r in di]},
        "step_roofline": {"bound": "host link", "bound_ms": bound_ms, "frac": bound_ms / step_ms},
        "roofline": roofline,
        "kernel_rooflines": {"dinf_prefill_pass": fam_p, "dinf_decode_pass": fam_d,
                             "timing": "unit graphs of 20 back-to-back launches (swapnet_engine_measure_units)"},
        "gpu_launches": launches, "clocks": clk,
        "setup_s": {"weights": t_gen, "plans": t_plan},
        "extension_resident_prefix": ext_rp,
        "extension_packed_swap": ext_pk,
    }
    rp.free(); rd.free()
    del arena
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        tot, sample = llm_cpu_sample()
        line["cpu_baseline"] = {"value": 1.0 / tot, "unit": unit, "cores": len(os.sched_getaffinity(0)),
                                "kind": "oracle", "sample": sample}
    return line if rank == 0 else {}


def run_multi(args, rank, world, group):
    """Config 4: three models at batch 1, each with its own closed-loop request
    stream on its own CUDA stream, sharing one arena split by Eq. 1
    (swapnet_schedule); DInf is the same concurrent run with every model
    resident."""
    import torch
    import synth
    from paper_2401_16757_gb300 import capi
    names = ("resnet50", "vgg16", "yolov3")
    ms = [synth.arch.MODELS[n]() for n in names]
    stream0 = torch.cuda.current_stream()
    link_peak = measure_link_peak(stream0)
    # the three pipelines share one host link: each model's delay model takes
    # its share of the measured bandwidth (--link-share 1 plans as if alone)
    alpha = int(round(1e18 / (link_peak * 1e9 / args.link_share)))
    variant = variant_code(args.variant)
    opt = capi.options(swap_variant=variant, alpha_as_per_byte=alpha, beta_ns_per_tensor=0, eta_ns_per_tensor=0)
    descs = [capi.Desc(m) for m in ms]
    wbs = [capi_weight_bytes(m) for m in ms]
    arena = int(sum(wbs) * 0.30) // 256 * 256
    budgets, plans = capi.schedule(descs, [1.0, 1.0, 1.0], arena, opt)
    hosts = [capi.HostWeights(synth.gen.model_weights(m)) for m in ms]
    engs = [capi.Engine(p, h) for p, h in zip(plans, hosts)]
    rengs = [capi.Engine(capi.Plan.resident(d), h) for d, h in zip(descs, hosts)]
    infos = [p.info() for p in plans]
    ins, outs = [], []
    for m, inf in zip(ms, infos):
        x = synth.gen.model_input(m)
        d_in = torch.empty(max(16, inf["input_bytes"]), dtype=torch.uint8, device="cuda")
        d_in[:inf["input_bytes"]].copy_(torch.from_numpy(x.view(np.uint8).reshape(-1)))
        ins.append(d_in)
        outs.append(torch.empty(inf["output_bytes"], dtype=torch.uint8, device="cuda"))
    streams = [torch.cuda.Stream() for _ in ms]

    def run(engines, steps):
        ev = lambda: torch.cuda.Event(enable_timing=True)
        evs = [[(ev(), ev()) for _ in range(steps)] for _ in engines]
        start = ev()
        start.record(stream0)
        for s in streams:
            s.wait_event(start)
        for i in range(steps):
            for k, e in enumerate(engines):
                a, b = evs[k][i]
                a.record(streams[k])
                e.infer(ins[k].data_ptr(), outs[k].data_ptr(), streams[k].cuda_stream)
                b.record(streams[k])
        ends = []
        for s in streams:
            e_ = ev()
            e_.record(s)
            ends.append(e_)
        torch.cuda.synchronize()
        lat = [[a.elapsed_time(b) for a, b in evs[k]] for k in range(len(engines))]
        wall = max(start.elapsed_time(e_) for e_ in ends)
        return lat, wall

    run(engs, args.warmup)
    run(rengs, args.warmup)
    for e in engs + rengs:
        e.sync()
    clocks = ClockSampler(int(os.environ.get("LOCAL_RANK", "0")))
    clocks.start()
    launches0 = sum(e.stats()["kernel_launches"] for e in engs)
    group.barrier()
    lat_sw, wall_sw = run(engs, args.steps)
    group.barrier()
    wall_sw = group.max(wall_sw)  # the slowest rank
    launches = sum(e.stats()["kernel_launches"] for e in engs) - launches0
    lat_di, wall_di = run(rengs, args.steps)
    # e2e through swapnet_infer_host: each request's input from pinned host
    # memory and its output back, the three models concurrently on their
    # streams; wall time of all requests
    h_ins, h_outs = [], []
    for m, inf in zip(ms, infos):
        x8 = synth.gen.model_input(m).view(np.uint8).reshape(-1)
        h_in = torch.empty(inf["input_bytes"], dtype=torch.uint8, pin_memory=True)
        h_in.copy_(torch.from_numpy(x8[:inf["input_bytes"]]))
        h_ins.append(h_in)
        h_outs.append(torch.empty(inf["output_bytes"], dtype=torch.uint8, pin_memory=True))

    def run_host(steps):
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        for _ in range(steps):
            for k, e in enumerate(engs):
                e.infer_host(h_ins[k].data_ptr(), h_outs[k].data_ptr(), streams[k].cuda_stream)
        torch.cuda.synchronize()
        return (time.perf_counter() - t0) * 1e3

    run_host(args.warmup)
    wall_e2e = group.max(run_host(args.steps))
    clk = clocks.stop()
    for e in engs:
        e.sync()
    n_req = len(ms) * args.steps
    swap_bytes = sum(sum(b["bytes"] for b in p.blocks()) for p in plans)
    hbm, tf_burst, tf_sust, peak_src = load_peaks()
    flops = sum(sum(u["flops"] for u in p.units()) for p in plans)
    bound_ms = max(flops / (tf_burst * 1e12), swap_bytes / (link_peak * 1e9)) * 1e3  # one request of each model
    per_model = {}
    for k, n in enumerate(names):
        sw, di = statistics.mean(lat_sw[k]), statistics.mean(lat_di[k])
        per_model[n] = {"budget_bytes": budgets[k], "weight_bytes": wbs[k], "n_blocks": infos[k]["n_blocks"],
                        "ms_swapped": sw, "ms_dinf": di, "ratio": sw / di,
                        "p50_swapped": statistics.median(lat_sw[k]), "p50_dinf": statistics.median(lat_di[k])}
    line = {
        "metric": METRIC, "value": world * n_req / (wall_sw * 1e-3), "unit": "inferences/s (3 models, concurrent)",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup, "ms_per_step": wall_sw / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f16", "data": "synthetic",
        "config": {"workload": CONFIGS["multi"][3], "arena_bytes": arena, "weight_bytes": sum(wbs),
                   "link_share": args.link_share,
                   "l2": "no flush: 451.6 MB of weights stream through the arena every round"},
        "per_model": per_model,
        "dinf_ms_per_step": wall_di / args.steps, "throughput_ratio": wall_sw / wall_di,
        "e2e": {"value": world * n_req / (wall_e2e * 1e-3), "unit": "inferences/s (3 models, concurrent)",
                "h2d_bytes_per_step": sum(i["input_bytes"] for i in infos),
                "d2h_bytes_per_step": sum(i["output_bytes"] for i in infos)},
        "link": {"achieved_gbs": swap_bytes * args.steps / (wall_sw * 1e-3) / 1e9, "peak_gbs": link_peak,
                 "peak_source": "pinned cudaMemcpy H2D 256 MiB", "bytes_per_step": swap_bytes},
        "step_roofline": {"bound": "host link" if swap_bytes / (link_peak * 1e9) > flops / (tf_burst * 1e12)
                          else "tensor", "bound_ms": bound_ms, "frac": bound_ms / (wall_sw / args.steps)},
        "gpu_launches": launches, "clocks": clk,
    }
    for e in engs + rengs:
        e.free()
    return line if rank == 0 else {}


def host_placement(ptr):
    """Where page-locked host memory sits relative to the GPU (a host-side
    reading, no GPU setting): the online NUMA nodes, the GPU's node, and the
    node of the page at `ptr` (move_pages query)."""
    import ctypes
    import platform
    import torch

    def rd(path):
        try:
            with open(path) as f:
                return f.read().strip()
        except OSError:
            return None
    out = {"numa_nodes_online": rd("/sys/devices/system/node/online")}
    try:
        p = torch.cuda.get_device_properties(torch.cuda.current_device())
        bus = "%04x:%02x:%02x.0" % (p.pci_domain_id, p.pci_bus_id, p.pci_device_id)
    except Exception:
        bus = None
    if bus:
        out["gpu_pci"] = bus.lower()
        node = rd("/sys/bus/pci/devices/%s/numa_node" % bus.lower())
        out["gpu_numa_node"] = int(node) if node not in (None, "") else None
    nr = {"aarch64": 239, "x86_64": 279}.get(platform.machine())
    if nr is not None:
        libc = ctypes.CDLL(None, use_errno=True)
        pages = (ctypes.c_void_p * 1)(ptr & ~4095)
        status = (ctypes.c_int * 1)(-99)
        r = libc.syscall(ctypes.c_long(nr), 0, ctypes.c_ulong(1), pages, None, status, 0)
        out["pinned_page_node"] = status[0] if r == 0 else None
    return out


def measure_link_peak(stream, placement=None):
    import torch
    pk = torch.empty(256 << 20, dtype=torch.uint8, pin_memory=True)
    dv = torch.empty(256 << 20, dtype=torch.uint8, device="cuda")
    best = 1e9
    for _ in range(5):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        dv.copy_(pk, non_blocking=True)
        b.record(stream)
        b.synchronize()
        best = min(best, a.elapsed_time(b))
    if placement is not None:
        placement.update(host_placement(pk.data_ptr()))
    return (256 << 20) / (best / 1000.0) / 1e9


def run_ablation(args):
    import __graft_entry__
    __graft_entry__.build()
    print(json.dumps(ablation_line(args)))


def ablation_line(args):
    """Ablations of the partition (the shape of the paper's Sec. 8.4-8.5
    studies) on one single-model config: the planner's plan against
    equal-byte plans with the paper's block count ceil(2s/b) and the next
    four counts, the Eq. 4 objective, strictly sequential layers, and each
    swap variant forced.  Latency of each (median ms, with the 10th and 90th
    percentiles, CUDA events, L2 flushed)."""
    import torch
    from paper_2401_16757_gb300 import capi
    m, w, x, wb, budget, text = build_workload(args.config, capi_weight_bytes)
    act_in = 1 if args.config == "mlp6" else 0
    host = capi.HostWeights(w)
    d = capi.Desc(m)
    plan0 = capi.Plan.partition(d, budget, capi.options(activations_in_budget=act_in))
    eng0 = capi.Engine(plan0, host)
    t_ex, alpha = capi.calibrate(m, eng0)
    eng0.free()
    dc = capi.Desc(m, t_ex_ns=t_ex)
    base = dict(activations_in_budget=act_in, alpha_as_per_byte=alpha or 4_750_000, beta_ns_per_tensor=0,
                eta_ns_per_tensor=0, swap_variant=capi.SWAP_MEMCPY)
    stream = torch.cuda.current_stream()
    flush = torch.empty(512 << 20, dtype=torch.uint8, device="cuda")
    x8 = x.view(np.uint8).reshape(-1)

    def latency(plan):
        info = plan.info()
        eng = capi.Engine(plan, host)
        d_in = torch.empty(max(16, info["input_bytes"]), dtype=torch.uint8, device="cuda")
        d_in[:x8.size].copy_(torch.from_numpy(x8))
        d_out = torch.empty(info["output_bytes"], dtype=torch.uint8, device="cuda")
        for _ in range(3):
            eng.infer(d_in.data_ptr(), d_out.data_ptr(), stream.cuda_stream)
        ts = []
        for _ in range(args.steps):
            flush.zero_()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            eng.infer(d_in.data_ptr(), d_out.data_ptr(), stream.cuda_stream)
            b.record(stream)
            b.synchronize()
            ts.append(a.elapsed_time(b))
        eng.sync()
        eng.free()
        return {"ms": statistics.median(ts), "p10_p90_ms": [float(np.percentile(ts, 10)), float(np.percentile(ts, 90))],
                "n_blocks": info["n_blocks"], "predicted_ms": info["predicted_ns"] / 1e6}

    def try_plan(make):
        try:
            return latency(make())
        except capi.SwapnetError as ex:
            return {"infeasible": str(ex)}

    out = {"planner": try_plan(lambda: capi.Plan.partition(dc, budget, capi.options(**base)))}
    units = capi.Plan.partition(dc, budget, capi.options(**base)).units()
    ub = np.cumsum([u["bytes"] for u in units])
    n_min = int(np.ceil(2.0 * wb / budget))
    for n in range(n_min, n_min + 5):
        cuts = sorted({int(np.searchsorted(ub, ub[-1] * k / n, side="left")) + 1 for k in range(1, n)})
        cuts = [c for c in cuts if 0 < c < len(units)]
        out["equal_bytes_n%d" % n] = try_plan(lambda: capi.Plan.from_cuts(dc, cuts, budget, capi.options(**base)))
    if len(units) <= 24:
        out["objective_eq4"] = try_plan(lambda: capi.Plan.partition(dc, budget, capi.options(**dict(base, objective=1))))
    out["sequential_layers"] = try_plan(lambda: capi.Plan.partition(dc, budget, capi.options(**dict(base, branches=0))))
    out["zero_copy_swap"] = try_plan(
        lambda: capi.Plan.partition(dc, budget, capi.options(**dict(base, swap_variant=capi.SWAP_ZEROCOPY))))
    # weights left pageable: each swap staged by the driver (the paper's w/o-uni-add)
    out["pageable_staged_copy"] = try_plan(
        lambda: capi.Plan.partition(dc, budget, capi.options(**dict(base, pageable=1))))
    out["resident_dinf"] = try_plan(lambda: capi.Plan.resident(d))
    return {"ablation": args.config, "workload": text, "budget_bytes": budget, "weight_bytes": wb,
            "paper_block_count": n_min, "steps": args.steps, "results": out}


def run_adapt_study(args):
    import __graft_entry__
    __graft_entry__.build()
    print(json.dumps(adapt_line(args)))


def adapt_line(args):
    """Dynamic-budget case study (the paper's Sec. 8 adaptation experiment,
    on ResNet-50 here): plans for three budgets are made ahead; one engine
    runs `steps` inferences per phase and switches plan between phases with
    swapnet_engine_adapt.  Reports per phase the budget, blocks, latency
    (median, 10th and 90th percentiles), the planning time and the switch
    time."""
    import torch
    from paper_2401_16757_gb300 import capi
    name = args.config if args.config in ("resnet50", "vgg16_b1", "yolov3") else "resnet50"
    m, w, x, wb, _, text = build_workload(name, capi_weight_bytes)
    host = capi.HostWeights(w)
    d = capi.Desc(m)
    fracs = (0.80, 0.60, 0.40)
    # offline profiling once (Sec. 6.1), then the look-up table of plans
    plan0 = capi.Plan.partition(d, int(wb * fracs[-1]) // 256 * 256, capi.options())
    eng0 = capi.Engine(plan0, host)
    t_ex, alpha = capi.calibrate(m, eng0)
    eng0.free()
    dc = capi.Desc(m, t_ex_ns=t_ex)
    opt = capi.options(alpha_as_per_byte=alpha or 4_750_000, beta_ns_per_tensor=0, eta_ns_per_tensor=0)
    plans, t_plan = [], []
    for f in fracs:
        t0 = time.perf_counter()
        plans.append(capi.Plan.partition(dc, int(wb * f) // 256 * 256, opt))
        t_plan.append((time.perf_counter() - t0) * 1e3)
    stream = torch.cuda.current_stream()
    flush = torch.empty(512 << 20, dtype=torch.uint8, device="cuda")
    info = plans[0].info()
    d_in = torch.empty(max(16, info["input_bytes"]), dtype=torch.uint8, device="cuda")
    d_in[:info["input_bytes"]].copy_(torch.from_numpy(x.view(np.uint8).reshape(-1)))
    d_out = torch.empty(info["output_bytes"], dtype=torch.uint8, device="cuda")
    eng = capi.Engine(plans[0], host)
    phases = []
    for i, (f, p) in enumerate(zip(fracs, plans)):
        t_sw = None
        if i:
            torch.cuda.synchronize()
            t0 = time.perf_counter()
            eng.adapt(p)
            t_sw = (time.perf_counter() - t0) * 1e3
        for _ in range(3):
            eng.infer(d_in.data_ptr(), d_out.data_ptr(), stream.cuda_stream)
        ts = []
        for _ in range(args.steps):
            flush.zero_()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            eng.infer(d_in.data_ptr(), d_out.data_ptr(), stream.cuda_stream)
            b.record(stream)
            b.synchronize()
            ts.append(a.elapsed_time(b))
        pi = p.info()
        phases.append({"budget_frac": f, "budget_bytes": pi["budget_bytes"], "n_blocks": pi["n_blocks"],
                       "cuts": p.cuts(), "ms": statistics.median(ts),
                       "p10_p90_ms": [float(np.percentile(ts, 10)), float(np.percentile(ts, 90))],
                       "plan_ms": t_plan[i],
                       "switch_ms": t_sw, "free_device_bytes": torch.cuda.mem_get_info()[0]})
    eng.sync()
    eng.free()
    return {"adapt_study": name, "workload": text, "weight_bytes": wb, "steps": args.steps, "phases": phases}


def run_storage(args):
    """Storage tier (Sec. 4.2.1 direct block fetch): the weights of --config
    are written to a file in --storage and every inference reads its
    swapped blocks from there with O_DIRECT (staging ring, read stream,
    copy into the slot).  The delay model is calibrated on the file engine
    (its per-block read + copy cost becomes alpha), the plan made from it,
    and the swapped inference timed against DInf (resident, host memory).
    Prints one JSON line."""
    import torch
    import __graft_entry__
    __graft_entry__.build()
    from paper_2401_16757_gb300 import capi
    name = args.config if args.config in ("resnet50", "vgg16_b1", "vgg16_b16", "yolov3", "mlp6") else "resnet50"
    m, w, x, wb, budget, text = build_workload(name, capi_weight_bytes)
    d = capi.Desc(m)
    host = capi.HostWeights(w)
    path = os.path.join(args.storage, "%s_%d.swnw" % (name, os.getpid()))
    t0 = time.perf_counter()
    capi.WeightsFile.write(path, d, host)
    t_write = time.perf_counter() - t0
    try:
        wf = capi.WeightsFile(path, allow_buffered=True)
        file_bytes = os.path.getsize(path)
        # the file read alone, O_DIRECT into a page-aligned buffer (64 MiB reads)
        buf = mmap.mmap(-1, 64 << 20)
        fd = os.open(path, os.O_RDONLY | (os.O_DIRECT if wf.info()["direct"] else 0))
        best = 1e30
        for _ in range(3):
            t0, off = time.perf_counter(), 0
            while off < file_bytes:
                k = os.preadv(fd, [buf], off)
                if k <= 0:
                    break
                off += k
            best = min(best, time.perf_counter() - t0)
        os.close(fd)
        read_gbs = file_bytes / best / 1e9
        act_in = 1 if name == "mlp6" else 0
        opt0 = capi.options(slots=2, activations_in_budget=act_in)
        plan0 = capi.Plan.partition(d, budget, opt0)
        eng0 = capi.Engine(plan0, wf)
        t_ex, alpha = capi.calibrate(m, eng0)
        eng0.free()
        opt = capi.options(slots=2, activations_in_budget=act_in, alpha_as_per_byte=alpha or 4_750_000,
                           beta_ns_per_tensor=0, eta_ns_per_tensor=0)
        plan = capi.Plan.partition(capi.Desc(m, t_ex_ns=t_ex), budget, opt)
        info = plan.info()
        eng = capi.Engine(plan, wf)
        reng = capi.Engine(capi.Plan.resident(d), host)
        stream = torch.cuda.current_stream()
        flush = torch.empty(512 << 20, dtype=torch.uint8, device="cuda")
        d_in = torch.empty(max(16, info["input_bytes"]), dtype=torch.uint8, device="cuda")
        d_in[:info["input_bytes"]].copy_(torch.from_numpy(x.view(np.uint8).reshape(-1)))
        d_out = torch.empty(info["output_bytes"], dtype=torch.uint8, device="cuda")
        r_out = torch.empty_like(d_out)

        def timed(e, out, steps):
            for _ in range(args.warmup):
                e.infer(d_in.data_ptr(), out.data_ptr(), stream.cuda_stream)
            ts = []
            for _ in range(steps):
                flush.zero_()
                a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                a.record(stream)
                e.infer(d_in.data_ptr(), out.data_ptr(), stream.cuda_stream)
                b.record(stream)
                b.synchronize()
                ts.append(a.elapsed_time(b))
            e.sync()
            return ts

        ts = timed(eng, d_out, args.steps)
        tr = timed(reng, r_out, min(args.steps, 50))
        exact = bool(torch.equal(d_out, r_out))
        ms = sum(ts) / len(ts)
        swapped = sum(b["bytes"] for b in plan.blocks())
        hbm, tf_burst, _, peak_src = load_peaks()
        flops = sum(u["flops"] for u in plan.units())
        bound_ms = max(flops / (tf_burst * 1e12), swapped / (read_gbs * 1e9)) * 1e3
        print(json.dumps({
            "metric": "inferences_per_second", "value": 1000.0 / ms, "unit": "inferences/s", "n_gpus": 1,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "p50_ms": statistics.median(ts), "dinf_ms": sum(tr) / len(tr), "bit_exact_vs_resident": exact,
            "predicted_ms": info["predicted_ns"] / 1e6, "n_blocks": info["n_blocks"],
            "config": {"workload": text + "; swapped blocks read from a weights file for every inference",
                       "storage_dir": args.storage, "l2": "512 MiB flush before every step"},
            "storage": {"file_bytes": file_bytes, "direct_io": wf.info()["direct"], "write_s": t_write,
                        "read_gbs_file_alone": read_gbs, "swapped_bytes_per_step": swapped,
                        "alpha_as_per_byte": alpha,
                        "block_read_copy_us": [round(b["memcpy_us"], 1) for b in eng.blocks()]},
            "step_bound": {"ms": bound_ms, "what": "max(FLOPs / bf16 peak, swapped bytes / file read GB/s)",
                           "frac": bound_ms / ms},
        }))
        eng.free()
        reng.free()
        wf.close()
    finally:
        os.unlink(path)


def run_profile_once(args):
    """One resident inference of a single-model config (no timing)."""
    import torch
    import __graft_entry__
    __graft_entry__.build()
    from paper_2401_16757_gb300 import capi
    if args.config == "llm":  # one pass of --profile-tokens ids through a decoder of the 7B widths
        import synth                # with --profile-layers layers (1 token: a decode pass)
        m = synth.arch.llm(layers=args.profile_layers, tokens=args.profile_tokens)
        host = llm_host_weights(m)
        x = synth.gen.model_input(m).reshape(-1) if args.profile_tokens > 1 else np.array([7], dtype=np.int32)
    else:
        m, w, x, wb, budget, text = build_workload(args.config, capi_weight_bytes)
        host = capi.HostWeights(w)
    if args.profile_swapped:
        # one swapped pass through an arena of half the weight bytes, with
        # the swap variant of --variant (the zero-copy kernel's captures)
        wbytes = capi.Plan.resident(capi.Desc(m)).info()["weight_bytes"]
        plan = capi.Plan.partition(capi.Desc(m), wbytes // 2 // 256 * 256,
                                   capi.options(swap_variant=variant_code(args.variant)))
    else:
        plan = capi.Plan.resident(capi.Desc(m))
    info = plan.info()
    eng = capi.Engine(plan, host)
    if info["state_bytes"]:
        state = torch.zeros(info["state_bytes"], dtype=torch.uint8, device="cuda")
        if args.profile_pos:
            state[:4].copy_(torch.tensor([args.profile_pos], dtype=torch.int32).view(torch.uint8))
        eng.bind_state(state.data_ptr(), info["state_bytes"])
    d_in = torch.empty(max(16, info["input_bytes"]), dtype=torch.uint8, device="cuda")
    d_in[:info["input_bytes"]].copy_(torch.from_numpy(x.view(np.uint8).reshape(-1)))
    d_out = torch.empty(info["output_bytes"], dtype=torch.uint8, device="cuda")
    eng.infer(d_in.data_ptr(), d_out.data_ptr(), torch.cuda.current_stream().cuda_stream)
    eng.sync()
    print(json.dumps({"profile_once": args.config, "kernels": eng.unit_kernels(), "tiling": eng.unit_tiling(),
                      "blocks": [dict(b, bytes=pb["bytes"]) for b, pb in zip(eng.blocks(), plan.blocks())]
                      if args.profile_swapped else None}))


def run_reference(args, rank, world):
    """The reference arm: the CPU oracle, timed as it stands on the host cores."""
    if rank != 0:
        return
    if args.config == "multi":
        import synth
        from oracle import forward as F
        cores = len(os.sched_getaffinity(0))
        work = []
        for n in ("resnet50", "vgg16", "yolov3"):
            m = synth.arch.MODELS[n]()
            work.append((m, synth.gen.model_weights(m), synth.gen.model_input(m)))
        times = []
        for _ in range(args.steps):   # one request of each model per step
            t0 = time.perf_counter()
            for m, w, x in work:
                F.forward(m, w, x)
            times.append(time.perf_counter() - t0)
        ms = 1000.0 * sum(times) / len(times)
        val = 3000.0 / ms
        print(json.dumps({
            "impl": "reference", "metric": METRIC, "value": val, "unit": "inferences/s (3 models, concurrent)",
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": CONFIGS["multi"][3], "l2": "n/a (CPU)"},
            "cpu_baseline": {"value": val, "unit": "inferences/s", "cores": cores, "kind": "oracle",
                             "sample": "one float64 inference of each of the three models per step, in sequence"},
            "e2e": {"value": val, "unit": "inferences/s (3 models, concurrent)", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0},
        }))
        return
    if args.config == "llm":
        cores = len(os.sched_getaffinity(0))
        sampler = llm_cpu_sampler()   # weights generated once, outside the timed samples
        for _ in range(max(0, min(args.warmup, 1))):
            sampler(1)
        times, walls = [], []
        for _ in range(args.steps):
            t0 = time.perf_counter()
            times.append(sampler()[0])
            walls.append(time.perf_counter() - t0)
        # a step is one bounded sample (its own wall time is ms_per_step);
        # the value is the whole inference the sample is scaled to
        ms_inf = 1000.0 * sum(times) / len(times)
        ms = 1000.0 * sum(walls) / len(walls)
        val = 1000.0 / ms_inf
        sample = llm_cpu_sample.__doc__.split("Returns")[0].strip()
        unit = "inferences/s (prefill 512 + 32 decode)"
        print(json.dumps({
            "impl": "reference", "metric": METRIC, "value": val, "unit": unit, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": CONFIGS["llm"][3], "budget_bytes": 4_000_000_000, "l2": "n/a (CPU)"},
            "ms_per_inference_scaled": ms_inf,
            "cpu_baseline": {"value": val, "unit": unit, "cores": cores, "kind": "oracle",
                             "sample": " ".join(sample.split()) + " Each step times one such sample (ms_per_step); "
                                       "value is 1 / the whole inference it scales to (ms_per_inference_scaled)."},
            "e2e": {"value": val, "unit": unit, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        }))
        return
    m, w, x, wb, budget, text = build_workload(args.config, oracle_weight_bytes)
    from oracle import forward as F
    for _ in range(max(0, min(args.warmup, 1))):
        F.forward(m, w, x)
    times = []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        F.forward(m, w, x)
        times.append(time.perf_counter() - t0)
    ms = 1000.0 * sum(times) / len(times)
    cores = len(os.sched_getaffinity(0))
    val = 1000.0 / ms
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": val, "unit": "inferences/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": text, "budget_bytes": budget, "weight_bytes": wb, "l2": "n/a (CPU)"},
        "cpu_baseline": {"value": val, "unit": "inferences/s", "cores": cores, "kind": "oracle",
                         "sample": "one whole float64 inference per step"},
        "e2e": {"value": val, "unit": "inferences/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }))


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", default="swapnet", choices=["swapnet", "reference"])
    ap.add_argument("--config", default="llm", choices=sorted(CONFIGS))
    ap.add_argument("--configs", default="mlp6,resnet50,vgg16_b1,vgg16_b16,yolov3,multi",
                    help="other configs measured after the main line (N=1 only) and reported under its "
                         "'configs' key; 'none' to skip")
    ap.add_argument("--variant", default="auto", choices=VARIANTS)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--profile-layers", type=int, default=2,
                    help="--profile-once --config llm: decoder layers of the profiled decode pass")
    ap.add_argument("--profile-tokens", type=int, default=1,
                    help="--profile-once --config llm: token ids of the profiled pass (1: decode, 512: prefill)")
    ap.add_argument("--profile-pos", type=int, default=0,
                    help="--profile-once --config llm: cached positions before the profiled pass (the attention "
                         "reads that many cache entries)")
    ap.add_argument("--merge", type=int, default=1, choices=[0, 1],
                    help="decoder: GEMV layers sharing an input in one launch (1) or one launch each (0)")
    ap.add_argument("--link-share", type=float, default=1.0,
                    help="multi: models sharing the host link in each model's delay model")
    ap.add_argument("--ablation", action="store_true",
                    help="partition ablations of --config (planner vs equal-byte plans, Eq. 4, sequential "
                         "layers, zero-copy swap, DInf); prints one JSON line")
    ap.add_argument("--adapt-study", action="store_true",
                    help="dynamic-budget case study: one engine switched between plans for 80/60/40 % budgets")
    ap.add_argument("--storage", default=None, metavar="DIR",
                    help="storage tier: write --config's weights to a file in DIR and read every swapped block "
                         "from it with O_DIRECT; prints one JSON line")
    ap.add_argument("--profile-swapped", action="store_true",
                    help="with --profile-once: one swapped pass (arena of half the weight bytes, --variant) "
                         "instead of a resident one")
    ap.add_argument("--profile-once", action="store_true",
                    help="run one resident inference of --config through the C ABI and exit "
                         "(a driver for profiler captures of its kernels); prints one JSON line")
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        run_reference(args, rank, world)
        return
    if args.profile_once:
        run_profile_once(args)
        return
    if args.ablation:
        run_ablation(args)
        return
    if args.adapt_study:
        run_adapt_study(args)
        return
    if args.storage:
        run_storage(args)
        return
    import torch
    torch.cuda.set_device(local)
    group = RankGroup(world, local)
    import __graft_entry__
    __graft_entry__.build()
    if args.config == "llm":
        line = run_llm(args, rank, world, group)
    elif args.config == "multi":
        line = run_multi(args, rank, world, group)
    else:
        line = run_cnn(args, rank, world, group, args.config)
    extra = [c for c in args.configs.split(",") if c and c != "none" and c != args.config]
    if extra and world == 1:
        # every other config measured in the same call, after the main line's
        # engines and buffers are released
        torch.cuda.synchronize()
        torch.cuda.empty_cache()
        line["configs"] = {}
        for c in extra:
            sub = argparse.Namespace(**vars(args))
            sub.config = c
            sub.steps = min(args.steps, 30)
            sub.warmup = 3
            sub.no_cpu_baseline = True
            t0 = time.perf_counter()
            try:
                if c == "multi":
                    r = run_multi(sub, rank, world, group)
                else:
                    r = run_cnn(sub, rank, world, group, c, compact=True)
                r = compact_line(r)
            except Exception as ex:   # the main line is reported whatever happens here
                r = {"error": "%s: %s" % (type(ex).__name__, ex)}
            r["wall_s"] = time.perf_counter() - t0
            line["configs"][c] = r
            torch.cuda.synchronize()
            torch.cuda.empty_cache()
        # the partition ablations and the runtime budget adaptation study on
        # ResNet-50 (Sec. 8.4-8.5 and the adaptation experiment), same call
        for key, fn in (("ablation", ablation_line), ("adapt_study", adapt_line)):
            sub = argparse.Namespace(**vars(args))
            sub.config = "resnet50"
            sub.steps = min(args.steps, 30)
            t0 = time.perf_counter()
            try:
                r = fn(sub)
            except Exception as ex:
                r = {"error": "%s: %s" % (type(ex).__name__, ex)}
            r["wall_s"] = time.perf_counter() - t0
            line[key] = r
            torch.cuda.synchronize()
            torch.cuda.empty_cache()
    if rank == 0:
        print(json.dumps(line))
    group.close()


def compact_line(r):
    """The keys of a config's line kept under the main line's `configs`."""
    keep = ("value", "unit", "ms_per_step", "p50_ms", "dinf_ms", "ratio", "dinf_ms_per_step", "throughput_ratio",
            "per_model", "link", "step_roofline", "roofline", "strict_budget", "gpu_launches", "clocks", "steps",
            "config", "e2e")
    return {k: r[k] for k in keep if k in r}


def run_cnn(args, rank, world, group, name, compact=False):
    """One single-model config (the CNNs and the MLP): the plan is made on a
    delay model calibrated on this GPU (Sec. 6.1), then swapped and
    all-resident latency, e2e, link rate and rooflines; the strict budget
    reading (activations inside the budget) for the CNNs; and unless compact
    the uncalibrated plan, the extension and prefetch lines and the CPU
    baseline.  Returns the line (rank 0)."""
    import torch
    from paper_2401_16757_gb300 import capi
    local = int(os.environ.get("LOCAL_RANK", "0"))
    m, w, x, wb, budget, text = build_workload(name, capi_weight_bytes)
    d = capi.Desc(m)
    variant = variant_code(args.variant)
    act_in = 1 if name == "mlp6" else 0
    opt0 = capi.options(slots=2, activations_in_budget=act_in, swap_variant=variant)
    host = capi.HostWeights(w)
    rplan = capi.Plan.resident(d)
    reng = capi.Engine(rplan, host)
    stream = torch.cuda.current_stream()
    sp = stream.cuda_stream
    rinfo = rplan.info()
    d_in = torch.empty(max(16, rinfo["input_bytes"]), dtype=torch.uint8, device="cuda")
    d_in[:rinfo["input_bytes"]].copy_(torch.from_numpy(x.view(np.uint8).reshape(-1)))
    d_out = torch.empty(rinfo["output_bytes"], dtype=torch.uint8, device="cuda")
    flush = torch.empty(512 << 20, dtype=torch.uint8, device="cuda")

    def timed(engine, steps, flush_l2=True, out=None):
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
        for a, b in evs:
            if flush_l2:
                flush.zero_()
            a.record(stream)
            engine.infer(d_in.data_ptr(), (out if out is not None else d_out).data_ptr(), sp)
            b.record(stream)
        torch.cuda.synchronize()
        return [a.elapsed_time(b) for a, b in evs]

    # offline profiling (Sec. 6.1): plan with default coefficients, measure
    # every layer's execution delay (scaled to the resident latency measured
    # here) and the link on this GPU, then plan again
    for _ in range(3):
        reng.infer(d_in.data_ptr(), d_out.data_ptr(), sp)
    rts = timed(reng, 20)
    plan0 = capi.Plan.partition(d, budget, opt0)
    eng0 = capi.Engine(plan0, host)
    t_ex, alpha = capi.calibrate(m, eng0, resident_ns=statistics.median(rts) * 1e6)
    dc = capi.Desc(m, t_ex_ns=t_ex)
    coef = dict(alpha_as_per_byte=alpha or 4_750_000, beta_ns_per_tensor=0, eta_ns_per_tensor=0)
    opt = capi.options(slots=2, activations_in_budget=act_in, swap_variant=variant, **coef)
    plan = capi.Plan.partition(dc, budget, opt)
    info = plan.info()
    eng = capi.Engine(plan, host)

    # cold: the engine's first inference (CUDA graph capture and
    # instantiation included), host wall time to its completion
    torch.cuda.synchronize()
    t_cold = time.perf_counter()
    eng.infer(d_in.data_ptr(), d_out.data_ptr(), sp)
    torch.cuda.synchronize()
    cold_ms = (time.perf_counter() - t_cold) * 1e3
    for _ in range(args.warmup):
        eng.infer(d_in.data_ptr(), d_out.data_ptr(), sp)
        reng.infer(d_in.data_ptr(), d_out.data_ptr(), sp)
    eng.sync()
    reng.sync()

    # ---- timed region: swapped inference
    clocks = ClockSampler(local)
    clocks.start()
    group.barrier()
    torch.cuda.synchronize()
    launches0 = eng.stats()["kernel_launches"]
    t_wall0 = time.perf_counter()
    torch.cuda.nvtx.range_push("swapped_steps")  # ncu --nvtx --nvtx-include swapped_steps/
    ms_list = timed(eng, args.steps)
    torch.cuda.nvtx.range_pop()
    t_wall = time.perf_counter() - t_wall0
    launches = eng.stats()["kernel_launches"] - launches0
    group.barrier()
    eng.sync()
    ms_swapped = sum(ms_list) / len(ms_list)
    total_ms = group.max(sum(ms_list))  # the slowest rank
    value = world * args.steps / (total_ms / 1000.0)

    # ---- DInf: same kernels, weights resident
    ms_dinf_list = timed(reng, args.steps)
    ms_dinf = sum(ms_dinf_list) / len(ms_dinf_list)

    # ---- e2e: host buffers through swapnet_infer_host
    h_in = torch.empty(info["input_bytes"], dtype=torch.uint8, pin_memory=True)
    h_in.copy_(torch.from_numpy(x.view(np.uint8).reshape(-1)))
    h_out = torch.empty(info["output_bytes"], dtype=torch.uint8, pin_memory=True)
    for _ in range(3):
        eng.infer_host(h_in.data_ptr(), h_out.data_ptr(), sp)
    torch.cuda.synchronize()
    e2e_ms = []
    for _ in range(args.steps):
        flush.zero_()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        eng.infer_host(h_in.data_ptr(), h_out.data_ptr(), sp)
        b.record(stream)
        b.synchronize()
        e2e_ms.append(a.elapsed_time(b))
    e2e_val = 1000.0 / (sum(e2e_ms) / len(e2e_ms))
    clk = clocks.stop()

    line = {}
    if not compact:
        # ---- the plan made with the default (uncalibrated) coefficients
        for _ in range(3):
            eng0.infer(d_in.data_ptr(), d_out.data_ptr(), sp)
        ms_uncal_list = timed(eng0, min(args.steps, 50))
        line["uncalibrated_plan"] = {"cuts": plan0.cuts(), "ms": sum(ms_uncal_list) / len(ms_uncal_list)}
        # ---- extension (not the paper's method): the first units stay
        # resident in the arena between inferences, the rest swap through
        # the region left
        plan_rp = capi.Plan.partition(dc, budget, capi.options(slots=2, activations_in_budget=act_in,
                                                                swap_variant=variant, resident_prefix=1, **coef))
        eng_rp = capi.Engine(plan_rp, host)
        for _ in range(3):
            eng_rp.infer(d_in.data_ptr(), d_out.data_ptr(), sp)
        ms_rp_list = timed(eng_rp, min(args.steps, 50))
        ri = plan_rp.info()
        line["extension_resident_prefix"] = {
            "ms": sum(ms_rp_list) / len(ms_rp_list), "prefix_units": ri["prefix_units"],
            "prefix_bytes": ri["prefix_bytes"], "n_blocks": ri["n_blocks"],
            "swapped_bytes_per_step": sum(b["bytes"] for b in plan_rp.blocks()[1 if ri["prefix_units"] else 0:])}
        eng_rp.free()
        # ---- steady state with first-block prefetch: each inference swaps
        # the next one's first block in at its end (the cyclic objective)
        plan_pf = capi.Plan.partition(dc, budget, capi.options(slots=2, activations_in_budget=act_in,
                                                                swap_variant=variant, prefetch=1, **coef))
        eng_pf = capi.Engine(plan_pf, host)
        pf_out = torch.empty_like(d_out)
        for _ in range(3):
            eng_pf.infer(d_in.data_ptr(), pf_out.data_ptr(), sp)
        ms_pf_list = timed(eng_pf, args.steps, out=pf_out)
        eng_pf.sync()
        pi = plan_pf.info()
        line["first_block_prefetch"] = {
            "ms": sum(ms_pf_list) / len(ms_pf_list), "p50_ms": statistics.median(ms_pf_list),
            "n_blocks": pi["n_blocks"], "cuts": plan_pf.cuts(), "predicted_ms": pi["predicted_ns"] / 1e6,
            "exact": pi["exact"], "bit_exact_vs_cold": bool(torch.equal(pf_out, d_out))}
        eng_pf.free()
    eng0.free()

    # ---- stricter budget reading: the activation workspace inside the
    # budget as well (the same budget if a plan fits it, else the smallest
    # budget in steps of 5 % of the weight bytes that does)
    strict = None
    if name != "mlp6":
        opt_s = capi.options(slots=2, activations_in_budget=1, swap_variant=variant, **coef)
        b_s, plan_s = budget, None
        while plan_s is None and b_s <= wb + info["workspace_bytes"] + (1 << 20):
            try:
                plan_s = capi.Plan.partition(dc, b_s, opt_s)
            except capi.SwapnetError as e_:
                if e_.code != capi.ERR_INFEASIBLE:
                    raise
                b_s = (b_s + int(0.05 * wb)) // 256 * 256
        if plan_s is not None:
            eng_s = capi.Engine(plan_s, host)
            for _ in range(3):
                eng_s.infer(d_in.data_ptr(), d_out.data_ptr(), sp)
            ms_s = statistics.mean(timed(eng_s, args.steps))
            si = plan_s.info()
            strict = {"budget_bytes": b_s, "budget_frac_of_weights": b_s / wb, "arena_bytes": si["arena_bytes"],
                      "workspace_bytes": si["workspace_bytes"],
                      "arena_plus_workspace_bytes": si["arena_bytes"] + si["workspace_bytes"],
                      "n_blocks": si["n_blocks"], "ms": ms_s, "ratio": ms_s / ms_dinf,
                      "swapped_bytes_per_step": sum(b["bytes"] for b in plan_s.blocks())}
            eng_s.free()

    # ---- kernel rooflines: each unit's kernels timed as a CUDA graph of
    # back-to-back launches (the dependent-launch overlap of a real
    # inference, no events between launches), grouped by kernel family
    units = plan.units()
    blocks = plan.blocks()
    kinds = eng.unit_kernels()
    unit_us = np.array(eng.measure_units(len(units), 20))
    hbm, tf_burst, tf_sust, peak_src = load_peaks()
    ubytes = unit_algorithmic_bytes(m, units)
    fam = kernel_rooflines(kinds, units, unit_us, ubytes, hbm, tf_burst, peak_src)
    dom = max(fam, key=lambda k: fam[k]["us_per_step"])
    roofline = dict(fam[dom])
    roofline.update({"kernel": dom, "timing": "unit graphs of 20 back-to-back launches (swapnet_engine_measure_units)",
                     "family_us_per_step_vs_step_us": [roofline["us_per_step"], ms_swapped * 1e3],
                     "traffic": None, "kernel_sources_sha": kernel_sources_sha(),
                     "traffic_sources_sha": traffic_sources_sha(),
                     "kernel_time_share": {k: round(v["us_per_step"] / max(1e-9, unit_us.sum()), 4)
                                           for k, v in fam.items()}})
    tr = TRAFFIC.get((name, dom))
    if tr and tr[0] == roofline["traffic_sources_sha"]:
        roofline["traffic"] = tr[1]

    # ---- host link: each swap-in timed inside the replayed graph (event
    # nodes on the copy stream only), bytes per swap over swap time, against
    # the pinned memcpy peak
    prof_steps = min(10, args.steps)
    eng.set_swap_timing(True)
    for _ in range(2):
        eng.infer(d_in.data_ptr(), d_out.data_ptr(), sp)
    acc_s = np.zeros(len(blocks))
    for _ in range(prof_steps):
        flush.zero_()
        eng.infer(d_in.data_ptr(), d_out.data_ptr(), sp)
        acc_s += np.array(eng.last_swap_times(len(blocks)))
    eng.set_swap_timing(False)
    acc_s /= prof_steps
    # ---- where the swapped time goes: the block timeline of the replayed
    # graph (event nodes on both streams; those between blocks add a
    # dependent launch at every block boundary, so this replay runs slower
    # than the timed step and explains it rather than measures it)
    eng.set_graph_timeline(True)
    for _ in range(2):
        eng.infer(d_in.data_ptr(), d_out.data_ptr(), sp)
    tls, replay_us = [], []
    for _ in range(prof_steps):
        flush.zero_()
        a_, b_ = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a_.record(stream)
        eng.infer(d_in.data_ptr(), d_out.data_ptr(), sp)
        b_.record(stream)
        b_.synchronize()
        replay_us.append(a_.elapsed_time(b_) * 1e3)
        tls.append(eng.last_graph_timeline(len(blocks)))
    eng.set_graph_timeline(False)
    tl = [[statistics.median(t[k][j] for t in tls) for j in range(4)] for k in range(len(blocks))]
    # time the layers waited for a swap: a block's swap ending after the
    # previous block's layers (the start of the inference for block 0)
    waited = [max(0.0, b[1] - (tl[k - 1][3] if k else 0.0)) if b[1] >= 0 else 0.0 for k, b in enumerate(tl)]
    line["graph_timeline"] = {
        "replay_us": statistics.median(replay_us), "step_us": ms_swapped * 1e3,
        "blocks_us": [[round(v, 1) for v in b] for b in tl],
        "columns": ["swap start", "swap end", "layers start", "layers end"],
        "layers_waited_for_swap_us": [round(v, 1) for v in waited],
        "layers_us": round(sum(b[3] - b[2] for b in tl), 1)}
    swap_bytes = sum(b["bytes"] for b in blocks)
    swap_us = float(acc_s.sum())
    link_peak = measure_link_peak(stream)
    link_gbs = swap_bytes / (swap_us * 1e-6) / 1e9 if swap_us > 0 else None
    # roofline of the whole step (slower of tensor FLOPs and swapped bytes over the link)
    flops = sum(u["flops"] for u in units)
    step_bound_ms = max(flops / (tf_burst * 1e12), swap_bytes / (link_peak * 1e9)) * 1e3
    if strict is not None:
        sb = max(flops / (tf_burst * 1e12), strict["swapped_bytes_per_step"] / (link_peak * 1e9)) * 1e3
        strict["step_roofline"] = {"bound_ms": sb, "frac": sb / strict["ms"]}

    cpu = None
    if rank == 0 and not args.no_cpu_baseline and not compact:
        cpu = cpu_oracle_baseline(m, w, x)

    if rank != 0:
        return {}
    eb = eng.blocks()
    line.update({
        "metric": METRIC, "value": value, "unit": "inferences/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_swapped, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f32" if m["dtype"] == "f32" else m["dtype"], "data": "synthetic",
        "config": {"workload": text, "budget_bytes": budget, "weight_bytes": wb,
                   "n_blocks": info["n_blocks"], "cuts": plan.cuts(), "slot_bytes": info["slot_bytes"],
                   "workspace_bytes": info["workspace_bytes"], "l2": "flushed (512 MiB write) before each step",
                   "swap_variants": [b["variant"] for b in eb], "parallelism": "replicas" if world > 1 else "1 GPU"},
        "dinf_ms": ms_dinf, "ratio": ms_swapped / ms_dinf,
        "predicted_ms": info["predicted_ns"] / 1e6,
        "p50_ms": statistics.median(ms_list), "p99_ms": float(np.percentile(ms_list, 99)),
        "cold_first_inference_ms": cold_ms,
        "e2e": {"value": e2e_val, "unit": "inferences/s", "h2d_bytes_per_step": info["input_bytes"],
                "d2h_bytes_per_step": info["output_bytes"]},
        "link": {"achieved_gbs": link_gbs, "peak_gbs": link_peak, "peak_source": "pinned cudaMemcpy H2D 256 MiB",
                 "frac": (link_gbs / link_peak) if link_gbs else None, "bytes_per_step": swap_bytes},
        "step_roofline": {"bound_ms": step_bound_ms, "frac": step_bound_ms / ms_swapped},
        "strict_budget": strict,
        "roofline": roofline,
        "kernel_rooflines": fam,
        "gpu_launches": launches,
        "clocks": clk,
        "cpu_baseline": cpu,
        "wall_s_timed": t_wall,
    })
    eng.free()
    reng.free()
    return line


def kernel_rooflines(kinds, units, unit_us, ubytes, hbm, tf_burst, peak_src):
    """Per kernel family: launches, time per step, algorithmic FLOPs and bytes,
    and the roof that binds it.  The binding roof is the tensor pipe when the
    family's algorithmic FLOPs per byte reach the ridge point (peak FLOP/s
    over peak bytes/s), HBM bandwidth otherwise.  ubytes: algorithmic bytes
    per unit, or None where the workload's layer types have no count."""
    ridge = tf_burst * 1e12 / (hbm * 1e9)
    fam = {}
    for i, k in enumerate(kinds):
        f = fam.setdefault(k, {"launches_per_step": 0, "us_per_step": 0.0, "flops": 0, "bytes": 0})
        f["launches_per_step"] += 1
        f["us_per_step"] += float(unit_us[i])
        f["flops"] += units[i]["flops"]
        f["bytes"] += ubytes[i] if ubytes else 0
    out = {}
    for k, f in fam.items():
        us = f["us_per_step"]
        tensor = f["flops"] > 0 and (not f["bytes"] or f["flops"] / f["bytes"] >= ridge)
        if tensor:
            ach = f["flops"] / (us * 1e-6) / 1e12 if us > 0 else 0.0
            r = {"bound": "tensor", "achieved": ach, "peak": tf_burst, "unit": "TFLOP/s",
                 "peak_source": peak_src + " bf16 burst (fp16 has the same dense rate)"}
        else:
            ach = f["bytes"] / (us * 1e-6) / 1e9 if us > 0 else 0.0
            r = {"bound": "hbm", "achieved": ach, "peak": hbm, "unit": "GB/s", "peak_source": peak_src + " copy"}
        n = max(1, f["launches_per_step"])
        r.update({"frac": ach / r["peak"], "launches_per_step": f["launches_per_step"], "us_per_step": us,
                  "us_per_launch": us / n, "algorithmic_flops_per_launch": f["flops"] // n,
                  "algorithmic_bytes_per_launch": f["bytes"] // n,
                  "flops_per_byte": f["flops"] / f["bytes"] if f["bytes"] else None, "ridge_flops_per_byte": ridge})
        out[k] = r
    return out


if __name__ == "__main__":
    main()
