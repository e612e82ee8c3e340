"""Host-only checks of the C ABI (no GPU): exported symbols, the planner
against the exhaustive-search oracle (integer-identical), workspace and unit
bookkeeping against the oracle, Eq. 1 scheduling, and argument errors."""
import itertools
import os
import re
import subprocess

import numpy as np
import pytest

from oracle import plan as P
import synth
from paper_2401_16757_gb300 import capi

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared_functions():
    src = open(os.path.join(ROOT, "include", "swapnet.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(swapnet_[a-z0-9_]+)\s*\(", src)))


def test_library_exports_every_declared_symbol():
    capi.lib()
    out = subprocess.run(["nm", "-D", "--defined-only", capi.LIB_PATH], capture_output=True, text=True).stdout
    exported = set(re.findall(r"\bT (swapnet_\w+)", out))
    declared = _declared_functions()
    assert declared, "no declarations parsed"
    missing = [f for f in declared if f not in exported]
    assert not missing, missing
    assert set(capi.EXPORTS) <= set(declared)


def _coef(opt):
    return P.Coef(opt.alpha_as_per_byte, opt.beta_ns_per_tensor, opt.gamma_as_per_flop, opt.eta_ns_per_tensor)


def _random_model(r, nl):
    """Random chain of conv / pool / linear layers with random sizes."""
    dtype = ["f16", "bf16", "f32"][int(r.integers(0, 3))]
    n, h, c = 2, 8, int(r.choice([8, 16, 32]))
    inp = (n, h, h, c)
    layers = []
    for i in range(nl):
        kind = r.integers(0, 4)
        if kind == 0 and h >= 2:
            layers.append(dict(op="maxpool", src=[i - 1], kh=2, kw=2, stride=2, pad=0))
            h //= 2
        elif kind in (1, 2):
            co, k = int(r.choice([8, 16, 64, 128, 256])), int(r.choice([1, 3]))
            layers.append(dict(op="conv", src=[i - 1], cin=c, cout=co, kh=k, kw=k, stride=1, pad=k // 2,
                               act="relu", res=None, res_post=False))
            c = co
        else:
            co = int(r.choice([8, 64, 200, 512]))
            layers.append(dict(op="linear", src=[i - 1], k=h * h * c, n=co, act="relu", res=None, res_post=False))
            h, c = 1, co
    return dict(name="rand", model_id=77, dtype=dtype, input=inp, layers=layers, outputs=[nl - 1])


@pytest.mark.parametrize("slots", [1, 2])
@pytest.mark.parametrize("act_in_budget", [0, 1])
def test_partition_equals_exhaustive_oracle(slots, act_in_budget):
    r = np.random.default_rng(100 + slots * 10 + act_in_budget)
    checked = 0
    for trial in range(40):
        nl = int(r.integers(2, 9))
        m = _random_model(r, nl)
        opt = capi.options(slots=slots, activations_in_budget=act_in_budget,
                           alpha_as_per_byte=int(r.integers(1_000_000, 5_000_000)),
                           beta_ns_per_tensor=int(r.integers(0, 3000)),
                           gamma_as_per_flop=int(r.integers(100, 100_000)),
                           eta_ns_per_tensor=int(r.integers(0, 500)))
        wb = P.weight_bytes(m)
        if wb == 0:
            continue
        ws = P.workspace(m)[0]
        budget = int(r.integers(max(1, wb // 4), wb * 2 + 1)) + (ws if act_in_budget else 0)
        ref = P.exhaustive_partition(m, budget, _coef(opt), slots=slots, activations_in_budget=bool(act_in_budget))
        desc = capi.Desc(m)
        if ref is None:
            with pytest.raises(capi.SwapnetError) as ei:
                capi.Plan.partition(desc, budget, opt)
            assert ei.value.code == capi.ERR_INFEASIBLE
            continue
        plan = capi.Plan.partition(desc, budget, opt)
        info = plan.info()
        assert plan.cuts() == ref["cuts"]
        assert info["n_blocks"] == ref["n"]
        assert info["predicted_ns"] == ref["predicted_ns"]
        assert info["slot_bytes"] == ref["slot"] and info["arena_bytes"] == ref["arena"]
        assert info["workspace_bytes"] == ref["workspace"]
        checked += 1
    assert checked >= 10


@pytest.mark.parametrize("slots", [1, 2])
def test_resident_prefix_partition_equals_exhaustive_oracle(slots):
    """The resident-prefix extension: prefix length and cuts identical to
    the oracle's brute force over the same candidate prefixes."""
    r = np.random.default_rng(300 + slots)
    checked = with_prefix = 0
    for trial in range(40):
        m = _random_model(r, int(r.integers(2, 9)))
        opt = capi.options(slots=slots, resident_prefix=1,
                           alpha_as_per_byte=int(r.integers(1_000_000, 5_000_000)),
                           beta_ns_per_tensor=int(r.integers(0, 3000)),
                           gamma_as_per_flop=int(r.integers(100, 100_000)),
                           eta_ns_per_tensor=int(r.integers(0, 500)))
        wb = P.weight_bytes(m)
        if wb == 0:
            continue
        budget = int(r.integers(max(1, wb // 4), wb * 2 + 1))
        ref = P.exhaustive_partition(m, budget, _coef(opt), slots=slots, resident_prefix=True)
        desc = capi.Desc(m)
        if ref is None:
            with pytest.raises(capi.SwapnetError) as ei:
                capi.Plan.partition(desc, budget, opt)
            assert ei.value.code == capi.ERR_INFEASIBLE
            continue
        plan = capi.Plan.partition(desc, budget, opt)
        info = plan.info()
        assert info["prefix_units"] == ref["prefix_units"], (trial, info["prefix_units"], ref["prefix_units"])
        assert info["prefix_bytes"] == ref["prefix_bytes"]
        assert plan.cuts() == ref["cuts"]
        assert info["n_blocks"] == ref["n"]
        assert info["predicted_ns"] == ref["predicted_ns"]
        blocks = plan.blocks()
        if ref["prefix_units"]:
            with_prefix += 1
            assert blocks[0]["slot"] == 0xFFFFFFFF and blocks[0]["offset"] == 0
            assert blocks[0]["unit1"] == ref["prefix_units"]
            for b in blocks[1:]:  # swapped blocks sit in the region beside the prefix
                assert b["offset"] >= ref["prefix_bytes"]
                assert b["offset"] + b["bytes"] <= info["arena_bytes"] // 256 * 256
        checked += 1
    assert checked >= 10 and with_prefix >= 3


def test_prefetch_partition_equals_exhaustive_oracle():
    """First-block prefetch: the cyclic objective, the wrap pair and the
    cuts identical to the oracle's brute force."""
    r = np.random.default_rng(404)
    checked = 0
    for trial in range(50):
        m = _random_model(r, int(r.integers(2, 9)))
        opt = capi.options(slots=2, prefetch=1,
                           alpha_as_per_byte=int(r.integers(1_000_000, 5_000_000)),
                           beta_ns_per_tensor=int(r.integers(0, 3000)),
                           gamma_as_per_flop=int(r.integers(100, 100_000)),
                           eta_ns_per_tensor=int(r.integers(0, 500)))
        wb = P.weight_bytes(m)
        if wb == 0:
            continue
        budget = int(r.integers(max(1, wb // 4), wb * 2 + 1))
        ref = P.exhaustive_partition(m, budget, _coef(opt), slots=2, prefetch=True)
        desc = capi.Desc(m)
        if ref is None:
            with pytest.raises(capi.SwapnetError) as ei:
                capi.Plan.partition(desc, budget, opt)
            assert ei.value.code == capi.ERR_INFEASIBLE
            continue
        plan = capi.Plan.partition(desc, budget, opt)
        info = plan.info()
        assert plan.cuts() == ref["cuts"], (trial, plan.cuts(), ref["cuts"])
        assert info["n_blocks"] == ref["n"]
        assert info["predicted_ns"] == ref["predicted_ns"]
        # an explicit cut vector gets the same cyclic prediction
        again = capi.Plan.from_cuts(desc, ref["cuts"], budget, opt)
        assert again.info()["predicted_ns"] == ref["predicted_ns"]
        checked += 1
    assert checked >= 10


def test_swap_variant_range():
    """AUTO, MEMCPY, ZEROCOPY, DIRECT and PACKED are the variants a plan
    accepts; the variant changes what the engine does, not the partition.
    Pageable weights take the copy engine only."""
    m = _random_model(np.random.default_rng(4), 6)
    desc = capi.Desc(m)
    budget = P.weight_bytes(m) // 256 * 256
    cuts = None
    for v in (capi.SWAP_AUTO, capi.SWAP_MEMCPY, capi.SWAP_ZEROCOPY, capi.SWAP_DIRECT, capi.SWAP_PACKED):
        got = capi.Plan.partition(desc, budget, capi.options(swap_variant=v)).cuts()
        assert cuts is None or got == cuts
        cuts = got
    for v in (capi.SWAP_ZEROCOPY, capi.SWAP_DIRECT, capi.SWAP_PACKED):
        with pytest.raises(capi.SwapnetError) as ei:
            capi.Plan.partition(desc, budget, capi.options(swap_variant=v, pageable=1))
        assert ei.value.code == capi.ERR_INVALID_ARG
    for bad in (-1, 5):
        with pytest.raises(capi.SwapnetError) as ei:
            capi.Plan.partition(desc, budget, capi.options(swap_variant=bad))
        assert ei.value.code == capi.ERR_INVALID_ARG
    assert capi.options().merge == 1 and capi.options().pageable == 0
    capi.Plan.partition(desc, budget, capi.options(pageable=1))
    capi.Plan.partition(desc, budget, capi.options(pageable=1, swap_variant=capi.SWAP_MEMCPY))
    for bad in (dict(merge=2), dict(merge=-1), dict(pageable=2), dict(pageable=1, swap_variant=capi.SWAP_ZEROCOPY),
                dict(pageable=1, swap_variant=capi.SWAP_DIRECT)):
        with pytest.raises(capi.SwapnetError) as ei:
            capi.Plan.partition(desc, budget, capi.options(**bad))
        assert ei.value.code == capi.ERR_INVALID_ARG


def test_prefetch_options_and_wrap_pair_are_checked():
    m = _random_model(np.random.default_rng(9), 5)
    desc = capi.Desc(m)
    wb = P.weight_bytes(m)
    for bad in (dict(prefetch=2), dict(prefetch=1, slots=1), dict(prefetch=1, objective=1),
                dict(prefetch=1, resident_prefix=1)):
        with pytest.raises(capi.SwapnetError) as ei:
            capi.Plan.partition(desc, wb, capi.options(**bad))
        assert ei.value.code == capi.ERR_INVALID_ARG
    # eight equal layers of x bytes in blocks of 3, 1, 1, 3 layers in a
    # region of 4x: every adjacent pair fits (4x, 2x, 4x), the wrap pair
    # (last, first) needs 6x
    layers = [dict(op="linear", src=[i - 1], k=128, n=128, act="relu", res=None, res_post=False) for i in range(8)]
    mm = dict(name="rand", model_id=78, dtype="f16", input=(2, 1, 1, 128), layers=layers, outputs=[7])
    x = sum(P.align(b) for b in P.layer_tensor_bytes(mm, 0))
    d = capi.Desc(mm)
    plain = capi.Plan.from_cuts(d, [3, 4, 5], 4 * x, capi.options())
    assert [b["bytes"] for b in plain.blocks()] == [3 * x, x, x, 3 * x]
    with pytest.raises(capi.SwapnetError) as ei:
        capi.Plan.from_cuts(d, [3, 4, 5], 4 * x, capi.options(prefetch=1))
    assert ei.value.code == capi.ERR_INFEASIBLE
    capi.Plan.from_cuts(d, [3, 4, 5], 6 * x, capi.options(prefetch=1))


def test_resident_prefix_never_worse_than_swapping_everything():
    for name in ("mlp6", "resnet50", "vgg16"):
        m = synth.arch.MODELS[name]()
        wb = P.weight_bytes(m)
        budget = int(wb * 0.4) // 256 * 256 if name != "mlp6" else 8_462_336
        act = 1 if name == "mlp6" else 0
        a = capi.Plan.partition(capi.Desc(m), budget, capi.options(activations_in_budget=act)).info()
        b = capi.Plan.partition(capi.Desc(m), budget,
                                capi.options(activations_in_budget=act, resident_prefix=1)).info()
        assert b["predicted_ns"] <= a["predicted_ns"]


def test_partition_eq4_objective_equals_oracle():
    r = np.random.default_rng(5)
    for _ in range(20):
        m = _random_model(r, int(r.integers(2, 8)))
        opt = capi.options(objective=1, beta_ns_per_tensor=700, eta_ns_per_tensor=300)
        wb = P.weight_bytes(m)
        if wb == 0:
            continue
        budget = int(r.integers(wb // 3 + 1, wb * 2 + 2))
        ref = P.exhaustive_partition(m, budget, _coef(opt), objective=1)
        if ref is None:
            continue
        plan = capi.Plan.partition(capi.Desc(m), budget, opt)
        assert plan.cuts() == ref["cuts"] and plan.info()["predicted_ns"] == ref["predicted_ns"]


@pytest.mark.parametrize("name", ["mlp6", "resnet50", "vgg16", "yolov3", "llm_small", "llm"])
def test_units_workspace_match_oracle(name):
    if name == "llm_small":
        m = synth.arch.llm(layers=2, d=256, heads=2, ffn=688, vocab=1000, tokens=64, max_seq=80)
    else:
        m = synth.arch.MODELS[name]()
    wb = P.weight_bytes(m)
    opt = capi.options()
    budget = wb * 3 // 10 // 256 * 256
    a = P.arena_and_slot(m, budget, 2, False)
    region = a[0] // 256 * 256
    ref_units = P.units(m, a[1], None, region)
    plan = capi.Plan.partition(capi.Desc(m), budget, opt)
    info = plan.info()
    ws, offs, ob, oo = P.workspace(m)
    assert info["workspace_bytes"] == ws and info["output_bytes"] == ob
    assert plan.output_offsets() == [oo[i] for i in sorted(oo)]
    assert info["weight_bytes"] == wb
    got = plan.units()
    assert len(got) == len(ref_units)
    for g, u in zip(got, ref_units):
        assert (g["layer"], g["bytes"], g["depth"], g["flops"]) == (u["layer"], u["bytes"], u["depth"], u["flops"])
        assert g["t_ex_ns"] == P.unit_t_ex(u, _coef(opt))
    # Eq. 3: consecutive blocks fit the arena together; even blocks at the
    # bottom, odd blocks against the top, so neighbours never overlap
    blocks = plan.blocks()
    for k, b in enumerate(blocks):
        assert b["bytes"] <= region and b["slot"] == k % 2
        assert b["offset"] == (0 if k % 2 == 0 else region - b["bytes"])
        if k:
            assert blocks[k - 1]["bytes"] + b["bytes"] <= region


def test_plan_from_cuts_and_predicted():
    m = synth.arch.mlp6()
    opt = capi.options(slots=1, activations_in_budget=1)
    budget = 8_462_336  # one block of two layers + two activation buffers
    plan = capi.Plan.from_cuts(capi.Desc(m), [2, 4], budget, opt)
    assert plan.info()["n_blocks"] == 3
    assert plan.info()["predicted_ns"] == P.evaluate_cuts(m, budget, _coef(opt), [2, 4], slots=1,
                                                          activations_in_budget=True)
    with pytest.raises(capi.SwapnetError) as ei:
        capi.Plan.from_cuts(capi.Desc(m), [3], budget, opt)   # a 3-layer block exceeds the slot
    assert ei.value.code == capi.ERR_INFEASIBLE
    with pytest.raises(capi.SwapnetError) as ei:
        capi.Plan.from_cuts(capi.Desc(m), [4, 2], budget, opt)
    assert ei.value.code == capi.ERR_INVALID_ARG
    # the planner at the same budget picks the same 3 x 2 partition
    assert capi.Plan.partition(capi.Desc(m), budget, opt).cuts() == [2, 4]
    # two slots at the same budget: one layer per block
    p2 = capi.Plan.partition(capi.Desc(m), budget, capi.options(slots=2, activations_in_budget=1))
    assert p2.cuts() == [1, 2, 3, 4, 5]


def test_resident_plan():
    m = synth.arch.resnet50()
    plan = capi.Plan.resident(capi.Desc(m))
    info = plan.info()
    assert info["n_blocks"] == 1 and info["slots"] == 0
    assert info["arena_bytes"] == P.weight_bytes(m)
    assert info["predicted_ns"] == P.resident_latency_ns(m, _coef(capi.options()))


def test_schedule_matches_eq1_oracle():
    ms = [synth.arch.resnet50(), synth.arch.vgg16(), synth.arch.yolov3()]
    total = sum(P.weight_bytes(m) for m in ms)
    M = total * 3 // 10 // 256 * 256
    opt = capi.options()
    budgets, plans = capi.schedule([capi.Desc(m) for m in ms], [1.0, 1.0, 1.0], M, opt)
    ref = P.schedule(ms, [1.0, 1.0, 1.0], M, _coef(opt))
    assert budgets == ref
    assert sum(budgets) <= M
    for b, p in zip(budgets, plans):
        assert p.info()["budget_bytes"] == b
    # within budget: every model gets its demand
    budgets2, _ = capi.schedule([capi.Desc(m) for m in ms], [1.0, 2.0, 0.5], total + 4096, opt)
    assert budgets2 == [P.weight_bytes(m) for m in ms]


def test_schedule_urgency_moves_budget():
    ms = [synth.arch.resnet50(), synth.arch.yolov3()]
    M = sum(P.weight_bytes(m) for m in ms) // 2 // 256 * 256
    opt = capi.options()
    b1, _ = capi.schedule([capi.Desc(m) for m in ms], [1.0, 1.0], M, opt)
    b2, _ = capi.schedule([capi.Desc(m) for m in ms], [4.0, 1.0], M, opt)
    assert b2[0] > b1[0] and b2[1] < b1[1]
    assert b2 == P.schedule(ms, [4.0, 1.0], M, P.Coef(opt.alpha_as_per_byte, opt.beta_ns_per_tensor,
                                                      opt.gamma_as_per_flop, opt.eta_ns_per_tensor))


def test_argument_errors():
    m = synth.arch.mlp6()
    d = capi.Desc(m)
    with pytest.raises(capi.SwapnetError) as ei:
        capi.Plan.partition(d, 1 << 20, capi.options(slots=3))
    assert ei.value.code == capi.ERR_INVALID_ARG
    with pytest.raises(capi.SwapnetError) as ei:
        capi.Plan.partition(d, 1000, capi.options())
    assert ei.value.code == capi.ERR_INFEASIBLE
    bad = dict(m, layers=[dict(m["layers"][0], k=1000)] + m["layers"][1:])
    with pytest.raises(capi.SwapnetError) as ei:
        capi.Plan.partition(capi.Desc(bad), 1 << 30, capi.options())
    assert ei.value.code == capi.ERR_INVALID_ARG
    assert b"linear" in capi.lib().swapnet_last_error()
    assert capi.lib().swapnet_debug_fail_next(9, 1) == capi.ERR_INVALID_ARG


def test_partition_large_models_fast():
    import time
    for name in ("resnet50", "vgg16", "yolov3"):
        m = synth.arch.MODELS[name]()
        wb = P.weight_bytes(m)
        t0 = time.time()
        plan = capi.Plan.partition(capi.Desc(m), wb * 4 // 10 // 256 * 256, capi.options())
        assert time.time() - t0 < 5.0
        assert plan.info()["n_blocks"] >= P.block_count_rule(wb, wb * 4 // 10 // 256 * 256)


def test_calibrate_binding_only_marshals(monkeypatch):
    """capi.calibrate passes its arguments to swapnet_engine_calibrate and
    returns what the library wrote: the Sec. 6.1 arithmetic (summing unit
    times per layer, the rescaling to the resident latency, alpha from the
    copy times) lives behind the C ABI.  A fake library records the call."""
    seen = {}

    class FakeLib:
        def swapnet_engine_calibrate(self, h, reps, resident_ns, t_ex, n, alpha):
            seen.update(h=h, reps=reps, resident_ns=resident_ns, n=n)
            for i in range(n):
                t_ex[i] = 1000 + 7 * i
            alpha._obj.value = 4_750_123
            return 0

    class FakeEngine:
        h = "engine-handle"

    m = synth.arch.mlp6()
    monkeypatch.setattr(capi, "lib", lambda: FakeLib())
    t_ex, alpha = capi.calibrate(m, FakeEngine(), reps=5, resident_ns=123456)
    assert seen == dict(h="engine-handle", reps=5, resident_ns=123456, n=len(m["layers"]))
    assert t_ex == [1000 + 7 * i for i in range(len(m["layers"]))] and alpha == 4_750_123

    class ZeroAlpha(FakeLib):
        def swapnet_engine_calibrate(self, h, reps, resident_ns, t_ex, n, alpha):
            return 0

    monkeypatch.setattr(capi, "lib", lambda: ZeroAlpha())
    assert capi.calibrate(m, FakeEngine())[1] is None   # no copy-engine times measured


def test_calibrate_rejects_a_null_engine():
    t_ex = (capi.C.c_int64 * 3)()
    alpha = capi.C.c_uint64()
    assert capi.lib().swapnet_engine_calibrate(None, 5, 0, t_ex, 3, capi.C.byref(alpha)) == capi.ERR_INVALID_ARG


def test_swap_timing_calls_reject_a_null_engine_or_output():
    """The in-graph swap timing and timeline calls check their arguments
    before touching a device (no GPU needed)."""
    us = (capi.C.c_float * 4)()
    assert capi.lib().swapnet_engine_set_swap_timing(None, 1) == capi.ERR_INVALID_ARG
    assert capi.lib().swapnet_engine_last_swap_times(None, us, 4) == capi.ERR_INVALID_ARG
    assert b"null" in capi.lib().swapnet_last_error()
    assert capi.lib().swapnet_engine_set_graph_timeline(None, 1) == capi.ERR_INVALID_ARG
    assert capi.lib().swapnet_engine_last_graph_timeline(None, us, 1) == capi.ERR_INVALID_ARG
    assert b"null" in capi.lib().swapnet_last_error()


def test_status_strings_cover_every_code():
    """Every status code has its own message (no code falls to 'unknown')."""
    codes = [capi.OK, capi.ERR_INVALID_ARG, capi.ERR_INFEASIBLE, capi.ERR_OOM, capi.ERR_CUDA, capi.ERR_TIMEOUT,
             capi.ERR_MISALIGNED, capi.ERR_UNSUPPORTED, capi.ERR_IO, capi.ERR_INTERNAL]
    msgs = [capi.lib().swapnet_strerror(c) for c in codes]
    assert len(set(msgs)) == len(codes)
    assert capi.lib().swapnet_strerror(-100) == b"unknown status"
    assert all(m != b"unknown status" for m in msgs)
