"""GPU parity through the C ABI: every kernel and whole workloads against
the CPU oracle, and swapped against all-resident (bit-exact)."""
import numpy as np
import pytest

from oracle import forward as F
from oracle import plan as OP
import synth
from paper_2401_16757_gb300 import capi
from helpers import Runner, check_close, check_oracle, oracle_cached, oracle_outputs, rel_l2

pytestmark = pytest.mark.gpu


def _conv(src, cin, cout, k, stride=1, pad=None, act="relu", res=None, res_post=False):
    return dict(op="conv", src=[src], cin=cin, cout=cout, kh=k, kw=k, stride=stride,
                pad=k // 2 if pad is None else pad, act=act, res=res, res_post=res_post)


def _model(layers, inp, dtype="f16", outputs=None, mid=40):
    return dict(name="yolov3", model_id=mid, dtype=dtype, input=inp, layers=layers,
                outputs=outputs or [len(layers) - 1])


def _swap_and_resident(m, budget_frac=0.5, slots=2, variant=capi.SWAP_AUTO):
    w = synth.gen.model_weights(m)
    x = synth.gen.model_input(m)
    d = capi.Desc(m)
    wb = OP.weight_bytes(m)
    opt = capi.options(slots=slots, swap_variant=variant)
    biggest = max(sum(OP.align(b) for b in OP.layer_tensor_bytes(m, i)) for i in range(len(m["layers"])))
    budget = max(int(wb * budget_frac), 2 * biggest + 512) // 256 * 256
    host = capi.HostWeights(w)
    sw = Runner(m, w, capi.Plan.partition(d, budget, opt), host)
    rs = Runner(m, w, capi.Plan.resident(d), host)
    return w, x, sw, rs


def _check_model(m, budget_frac=0.5, slots=2, variant=capi.SWAP_AUTO):
    w, x, sw, rs = _swap_and_resident(m, budget_frac, slots, variant)
    ref = oracle_outputs(m, w, x)
    got_sw = sw.run(x)
    got_rs = rs.run(x)
    for a, b in zip(got_sw, got_rs):
        assert a.tobytes() == b.tobytes(), "swapped and resident differ"
    check_close(m, sw.decode(got_sw), ref)
    return sw


# ----------------------------------------------------------------- kernels
@pytest.mark.parametrize("dtype", ["f16", "bf16"])
@pytest.mark.parametrize("k,stride,cin,cout,hw", [
    (3, 1, 64, 64, 19),     # gather path, ragged M tile
    (3, 2, 32, 96, 23),     # Cin=32: K=288 not a multiple of 64; stride 2
    (1, 1, 64, 200, 17),    # pointwise: TMA A path, N not a multiple of 64
    (1, 2, 128, 256, 14),   # strided pointwise: gather path
    (7, 2, 3, 64, 40),      # ResNet stem: small-channel tcgen05 conv, K=147 (3 k-blocks)
    (3, 1, 3, 16, 12),      # small-channel conv, N=16
    (3, 1, 3, 96, 37),      # small-channel conv, two 64-column slices, ragged M
    (5, 1, 4, 32, 21),      # Cin=4, K=100 (2 k-blocks)
    (3, 1, 3, 32, 224),     # 784 tiles: more tiles than resident CTAs (persistent loop)
    (7, 1, 5, 40, 15),      # K=245 beyond the small-channel kernel: SIMT direct conv
    (3, 1, 64, 64, 112),    # 196 x 1 tiles >= one per SM: persistent kernel, N tile 64, gather
    (3, 1, 32, 128, 112),   # persistent, N tile 128, gather with k-blocks straddling taps
    (1, 1, 64, 300, 112),   # persistent, N tile 256 (ragged), A by TMA
    (3, 2, 64, 256, 224),   # persistent, N tile 256, strided gather
    (3, 1, 64, 64, 224),    # persistent, N tile 64, four 128-row patches per tile (784 patches)
    (1, 1, 64, 48, 220),    # persistent 2-D TMA, four sub-tiles per tile, ragged m-tile count, N 48
    (1, 1, 64, 48, 160),    # persistent 2-D TMA, two sub-tiles per tile (400 m-tiles)
    (3, 1, 64, 64, 150),    # persistent 4-D TMA, two 32 x 4 patches per tile (380 patches, ragged edge)
    (3, 1, 256, 256, 7),    # deep K, one M tile: split-K with last-CTA reduction
    (3, 1, 64, 24, 9),      # N below one 32-column chunk
    (3, 1, 64, 128, 14),    # few tiles, taps of 64 channels: A by 4-D TMA over 14 x 9 pixel patches
    (3, 2, 128, 128, 28),   # the same, strided
    (1, 2, 256, 256, 28),   # strided pointwise by 4-D TMA
    (3, 1, 64, 64, 26),     # 26 x 4 patches, last patch row ragged
    (3, 1, 256, 256, 14),   # 4-D TMA A with cluster split-K (36 k-blocks)
    (1, 2, 128, 256, 56),   # 28 x 4 patches
    (3, 1, 512, 128, 7),    # 7 x 7 patch (49 of 128 rows), as many CTAs as 128-row tiles
    (3, 2, 256, 64, 13),    # strided, 7 x 7 output, ragged against the 13-pixel input
])
def test_conv_layer(dtype, k, stride, cin, cout, hw):
    m = _model([_conv(-1, cin, cout, k, stride)], (2, hw, hw, cin), dtype)
    _check_model(m)


@pytest.mark.parametrize("res_post,act", [(False, "relu"), (True, "leaky"), (False, "none")])
def test_conv_residual_epilogue(res_post, act):
    layers = [_conv(-1, 64, 128, 1, act="none"),
              _conv(-1, 64, 64, 3),
              _conv(1, 64, 128, 3, act=act, res=0, res_post=res_post)]
    _check_model(_model(layers, (1, 30, 30, 64)))


@pytest.mark.parametrize("dtype", ["f16", "bf16", "f32"])
@pytest.mark.parametrize("rows,k,n", [(1, 2048, 1000), (16, 4096, 640), (8, 1024, 1024), (200, 512, 384),
                                      (300, 256, 64), (129, 1024, 136), (40, 512, 130),
                                      (16, 25088, 1000), (12, 2048, 520), (5, 1024, 296)])
def test_linear_layer(dtype, rows, k, n):
    layers = [dict(op="linear", src=[-1], k=k, n=n, act="relu", res=None, res_post=False),
              dict(op="linear", src=[0], k=n, n=n, act="none", res=0, res_post=False)]
    _check_model(_model(layers, (rows, 1, 1, k), dtype))


@pytest.mark.parametrize("dtype", ["f16", "bf16"])
@pytest.mark.parametrize("rows,k,n", [(1, 11008, 520), (3, 25088, 300), (4, 9000, 136), (2, 16384, 64)])
def test_linear_long_rows(dtype, rows, k, n):
    """GEMV rows of 9000 to 25088 elements (5 to 13 batches of loads per
    lane, the longest the VGG-16 FC1 row): against the oracle, swapped equal
    to resident bit for bit."""
    layers = [dict(op="linear", src=[-1], k=k, n=n, act="relu", res=None, res_post=False)]
    _check_model(_model(layers, (rows, 1, 1, k), dtype))


@pytest.mark.parametrize("k", [4096, 11008])
def test_swiglu_pair_long_rows(k):
    """A SwiGLU gate and its paired layer (one merged launch, the gate's
    stored output used as the pair's residual) at the 7B widths' K (4096)
    and at the FFN width (11008), one row of bf16 input: against the
    oracle, swapped (where the two layers may sit in different blocks and
    run as separate launches) equal to resident bit for bit."""
    layers = [dict(op="linear", src=[-1], k=k, n=192, act="none", res=None, res_post=False),
              dict(op="linear", src=[-1], k=k, n=192, act="swiglu", res=0, res_post=False)]
    _check_model(_model(layers, (1, 1, 1, k), "bf16"))


@pytest.mark.parametrize("dtype,ch", [("f16", 24), ("f32", 24), ("f16", 20), ("bf16", 8)])
def test_pool_upsample_concat(dtype, ch):
    layers = [dict(op="maxpool", src=[-1], kh=3, kw=3, stride=2, pad=1),
              dict(op="maxpool", src=[0], kh=2, kw=2, stride=2, pad=0),
              dict(op="upsample2x", src=[1]),
              dict(op="concat", src=[2, 0]),
              dict(op="gap", src=[3])]
    m = _model(layers, (2, 32, 32, ch), dtype, outputs=[3, 4])   # 16-byte vectors unless ch=20 (f16)
    # no weights: swapped plan has nothing to swap; compare to the oracle
    w = synth.gen.model_weights(m)
    x = synth.gen.model_input(m)
    r = Runner(m, w, capi.Plan.resident(capi.Desc(m)))
    got = r.decode(r.run(x))
    ref = oracle_outputs(m, w, x)
    np.testing.assert_array_equal(got[0], ref[0])      # max / copy ops are exact
    check_close(m, got[1:], ref[1:])


# ----------------------------------------------------------------- workloads
@pytest.mark.parametrize("variant", [capi.SWAP_MEMCPY, capi.SWAP_ZEROCOPY, capi.SWAP_AUTO])
def test_mlp_config(variant):
    """6-layer fp32 MLP: explicit 3 x 2 plan in one slot (budget = one block
    of weights + two activation buffers), the planner's 2-slot plan, and the
    resident reference; all equal bit for bit and within 1e-4 of the oracle."""
    m = synth.arch.mlp6()
    w = synth.gen.model_weights(m)
    x = synth.gen.model_input(m)
    d = capi.Desc(m)
    budget = 8_462_336
    host = capi.HostWeights(w)
    p1 = capi.Plan.from_cuts(d, [2, 4], budget, capi.options(slots=1, activations_in_budget=1,
                                                               swap_variant=variant))
    p2 = capi.Plan.partition(d, budget, capi.options(slots=2, activations_in_budget=1, swap_variant=variant))
    assert p2.cuts() == [1, 2, 3, 4, 5]
    outs = [Runner(m, w, p, host).run(x) for p in (p1, p2, capi.Plan.resident(d))]
    for o in outs[1:]:
        assert o[0].tobytes() == outs[0][0].tobytes()
    ref = oracle_outputs(m, w, x)
    check_close(m, [o.astype(np.float64) for o in outs[0]], ref)


def test_mlp_repeated_calls_stable():
    m = synth.arch.mlp6()
    w = synth.gen.model_weights(m)
    d = capi.Desc(m)
    r = Runner(m, w, capi.Plan.partition(d, 8_462_336, capi.options(activations_in_budget=1)))
    first = None
    for req in range(5):
        x = synth.gen.model_input(m, request=req % 2)
        o = r.run(x)[0].tobytes()
        if req == 0:
            first = o
        if req % 2 == 0:
            assert o == first


def test_every_partition_bit_exact_tiny():
    layers = [_conv(-1, 16, 32, 3), _conv(0, 32, 32, 3, stride=2), _conv(1, 32, 64, 1),
              dict(op="maxpool", src=[2], kh=2, kw=2, stride=2, pad=0),
              dict(op="gap", src=[3]),
              dict(op="linear", src=[4], k=64, n=40, act="none", res=None, res_post=False)]
    m = _model(layers, (1, 24, 24, 16))
    w = synth.gen.model_weights(m)
    x = synth.gen.model_input(m)
    d = capi.Desc(m)
    host = capi.HostWeights(w)
    base = Runner(m, w, capi.Plan.resident(d), host).run(x)[0].tobytes()
    budget = 2 * OP.weight_bytes(m)
    import itertools
    for k in range(0, 6):
        for cuts in itertools.combinations(range(1, 6), k):
            p = capi.Plan.from_cuts(d, list(cuts), budget, capi.options())
            assert Runner(m, w, p, host).run(x)[0].tobytes() == base, cuts


def test_resnet50_config():
    """ResNet-50 (BN folded), batch 1, budget 40 % of the weight bytes."""
    m = synth.arch.resnet50()
    sw = _check_model(m, budget_frac=0.4)
    assert sw.info["n_blocks"] >= OP.block_count_rule(sw.info["weight_bytes"], sw.info["budget_bytes"])


def test_swap_variants_bit_exact_resnet():
    m = synth.arch.resnet50()
    w = synth.gen.model_weights(m)
    x = synth.gen.model_input(m)
    d = capi.Desc(m)
    host = capi.HostWeights(w)
    budget = int(OP.weight_bytes(m) * 0.4) // 256 * 256
    outs = [Runner(m, w, capi.Plan.partition(d, budget, capi.options(swap_variant=v)), host).run(x)[0].tobytes()
            for v in (capi.SWAP_MEMCPY, capi.SWAP_ZEROCOPY)]
    assert outs[0] == outs[1]


def test_calibrated_plan_is_exact_and_feasible():
    """Offline profiling (measured per-layer t_ex and link alpha) changes the
    partition, never the result."""
    m = synth.arch.resnet50()
    w = synth.gen.model_weights(m)
    x = synth.gen.model_input(m)
    d = capi.Desc(m)
    host = capi.HostWeights(w)
    budget = int(OP.weight_bytes(m) * 0.4) // 256 * 256
    p0 = capi.Plan.partition(d, budget, capi.options())
    r0 = Runner(m, w, p0, host)
    t_ex, alpha = capi.calibrate(m, r0.engine)
    assert all(t > 0 for t in t_ex) and alpha and alpha > 0
    p1 = capi.Plan.partition(capi.Desc(m, t_ex_ns=t_ex), budget,
                             capi.options(alpha_as_per_byte=alpha, beta_ns_per_tensor=0))
    region = p1.info()["arena_bytes"] // 256 * 256
    bl = p1.blocks()
    assert all(b["bytes"] <= region for b in bl)
    assert all(bl[k - 1]["bytes"] + bl[k]["bytes"] <= region for k in range(1, len(bl)))
    base = Runner(m, w, capi.Plan.resident(d), host).run(x)[0].tobytes()
    assert r0.run(x)[0].tobytes() == base
    assert Runner(m, w, p1, host).run(x)[0].tobytes() == base


def test_vgg16_b1_config():
    """VGG-16, batch 1, budget 25 % of the weight bytes: FC1 (205 MB) is cut
    into output-feature pieces; swapped equals resident bit for bit."""
    m = synth.arch.vgg16(batch=1)
    w = synth.gen.model_weights(m)
    x = synth.gen.model_input(m)
    d = capi.Desc(m)
    budget = int(OP.weight_bytes(m) * 0.25) // 256 * 256
    host = capi.HostWeights(w)
    sw = Runner(m, w, capi.Plan.partition(d, budget, capi.options()), host)
    assert sum(1 for u in sw.plan.units() if u["layer"] == 18) > 1   # FC1 split
    got = sw.run(x)
    assert got[0].tobytes() == Runner(m, w, capi.Plan.resident(d), host).run(x)[0].tobytes()
    check_close(m, sw.decode(got), oracle_outputs(m, w, x))


def test_vgg16_b16_sampled_images():
    """VGG-16 at batch 16 (the bench launch configuration): images 0 and 15 of
    the GPU batch against the oracle run on those two images alone (the
    network treats images independently)."""
    m = synth.arch.vgg16(batch=16)
    w = synth.gen.model_weights(m)
    x = synth.gen.model_input(m)
    d = capi.Desc(m)
    budget = int(OP.weight_bytes(m) * 0.25) // 256 * 256
    host = capi.HostWeights(w)
    sw = Runner(m, w, capi.Plan.partition(d, budget, capi.options()), host)
    got = sw.run(x)[0]
    rs = Runner(m, w, capi.Plan.resident(d), host).run(x)[0]
    assert got.tobytes() == rs.tobytes()
    m2 = synth.arch.vgg16(batch=2)
    ref = oracle_outputs(m2, w, np.ascontiguousarray(x[[0, 15]]))[0]
    check_close(m2, [sw.decode([got[[0, 15]]])[0]], [ref])


def test_yolov3_config():
    """Darknet-53 + three YOLOv3 heads at 416x416: routes, upsample, concat,
    LeakyReLU and post-activation shortcuts; three output tensors."""
    m = synth.arch.yolov3()
    sw = _check_model(m, budget_frac=0.3)
    assert len(sw.offs) == 3


def test_multi_dnn_schedule_concurrent():
    """Eq. 1 split of one arena (30 % of the summed weight bytes) over
    ResNet-50, VGG-16 and YOLOv3; the three engines run concurrently on their
    own streams and each output equals its resident run bit for bit and the
    oracle within the fp16 bar."""
    import torch
    ms = [synth.arch.resnet50(), synth.arch.vgg16(), synth.arch.yolov3()]
    total = sum(OP.weight_bytes(m) for m in ms)
    M = int(total * 0.3) // 256 * 256
    descs = [capi.Desc(m) for m in ms]
    budgets, plans = capi.schedule(descs, [1.0, 1.0, 1.0], M, capi.options())
    assert sum(budgets) <= M
    runners, xs, refs = [], [], []
    for m, d, p in zip(ms, descs, plans):
        w = synth.gen.model_weights(m)
        host = capi.HostWeights(w)
        runners.append(Runner(m, w, p, host))
        xs.append(synth.gen.model_input(m))
        refs.append(Runner(m, w, capi.Plan.resident(d), host).run(xs[-1]))
    streams = [torch.cuda.Stream() for _ in ms]
    for r, x in zip(runners, xs):
        r.d_in[:x.nbytes].copy_(torch.from_numpy(np.ascontiguousarray(x).view(np.uint8).reshape(-1)))
    torch.cuda.synchronize()
    for _ in range(3):
        for r, s in zip(runners, streams):
            r.engine.infer(r.d_in.data_ptr(), r.d_out.data_ptr(), s.cuda_stream)
    torch.cuda.synchronize()
    for r, ref, x in zip(runners, refs, xs):
        r.engine.sync()
        got = r.outputs_raw()
        assert all(a.tobytes() == b.tobytes() for a, b in zip(got, ref))
        check_oracle(r, got, x)


@pytest.mark.parametrize("name", ["resnet50", "yolov3"])
def test_concurrent_branches_bit_exact(name):
    """Layers run beside their neighbours on the second stream (projection
    shortcuts, detection-head branches) give the same bits as strictly
    sequential execution, resident and swapped."""
    m = synth.arch.MODELS[name]()
    w = synth.gen.model_weights(m)
    x = synth.gen.model_input(m)
    d = capi.Desc(m)
    host = capi.HostWeights(w)
    seq = Runner(m, w, capi.Plan.resident(d, capi.options(branches=0)), host).run(x)
    par = Runner(m, w, capi.Plan.resident(d, capi.options(branches=1)), host).run(x)
    budget = int(OP.weight_bytes(m) * 0.4) // 256 * 256
    sw = Runner(m, w, capi.Plan.partition(d, budget, capi.options(branches=1)), host).run(x)
    for a, b, c in zip(seq, par, sw):
        assert a.tobytes() == b.tobytes() == c.tobytes()
    check_close(m, [F.decode(o, m["dtype"]) for o in sw], oracle_cached(m, w, x))


@pytest.mark.parametrize("name", ["resnet50", "yolov3"])
def test_resident_prefix_bit_exact_over_repeated_inferences(name):
    """Resident-prefix plans (an extension: the first units stay in the arena
    between inferences) give the resident plan's bits on every call, so the
    prefix is not disturbed by the blocks swapped beside it."""
    m = synth.arch.MODELS[name]()
    w = synth.gen.model_weights(m)
    d = capi.Desc(m)
    host = capi.HostWeights(w)
    budget = int(OP.weight_bytes(m) * 0.4) // 256 * 256
    plan = capi.Plan.partition(d, budget, capi.options(resident_prefix=1))
    info = plan.info()
    assert info["prefix_units"] > 0 and info["n_blocks"] > 1
    sw = Runner(m, w, plan, host)
    rs = Runner(m, w, capi.Plan.resident(d), host)
    for req in range(3):
        x = synth.gen.model_input(m, request=req)
        a, b = sw.run(x), rs.run(x)
        assert all(p.tobytes() == q.tobytes() for p, q in zip(a, b)), req
        if req == 0:
            check_oracle(sw, a, x)


@pytest.mark.parametrize("name,variant", [("resnet50", capi.SWAP_AUTO), ("yolov3", capi.SWAP_MEMCPY),
                                          ("resnet50", capi.SWAP_ZEROCOPY)])
def test_first_block_prefetch_bit_exact_over_repeated_inferences(name, variant):
    """First-block prefetch: each inference swaps the next one's first block
    in at its end; every call (the first one from the load-time upload) and
    every call after a switch to another prefetch plan gives the resident
    bits, on eager and graph launches alike."""
    m = synth.arch.MODELS[name]()
    w = synth.gen.model_weights(m)
    d = capi.Desc(m)
    host = capi.HostWeights(w)
    wb = OP.weight_bytes(m)
    opt = capi.options(prefetch=1, swap_variant=variant)
    plan = capi.Plan.partition(d, int(wb * 0.4) // 256 * 256, opt)
    assert plan.info()["n_blocks"] > 2
    sw = Runner(m, w, plan, host)
    rs = Runner(m, w, capi.Plan.resident(d), host)
    for req in range(3):
        x = synth.gen.model_input(m, request=req)
        a, b = sw.run(x), rs.run(x)
        assert all(p.tobytes() == q.tobytes() for p, q in zip(a, b)), req
        if req == 0:
            check_oracle(sw, a, x)
    sw.engine.set_profiling(True)  # eager launches
    x = synth.gen.model_input(m, request=7)
    assert all(p.tobytes() == q.tobytes() for p, q in zip(sw.run(x), rs.run(x)))
    sw.engine.set_profiling(False)
    sw.engine.adapt(capi.Plan.partition(d, int(wb * 0.3) // 256 * 256, opt))
    for req in range(2):
        x = synth.gen.model_input(m, request=10 + req)
        a, b = sw.run(x), rs.run(x)
        assert all(p.tobytes() == q.tobytes() for p, q in zip(a, b)), req


def test_engine_adapts_to_new_budgets_between_inferences():
    """Runtime budget adaptation: one engine switched through plans for
    shrinking and growing budgets (made ahead, like the paper's look-up
    table) gives the resident bits after every switch, and the oracle's
    outputs for each new request; a plan for another model is refused."""
    import torch
    m = synth.arch.resnet50()
    w = synth.gen.model_weights(m)
    d = capi.Desc(m)
    host = capi.HostWeights(w)
    wb = OP.weight_bytes(m)
    plans = {f: capi.Plan.partition(d, int(wb * f) // 256 * 256, capi.options()) for f in (0.8, 0.5, 0.3, 0.6)}
    sw = Runner(m, w, plans[0.8], host)
    rs = Runner(m, w, capi.Plan.resident(d), host)
    free0 = torch.cuda.mem_get_info()[0]
    for i, f in enumerate((0.8, 0.5, 0.3, 0.6)):
        if i:
            sw.engine.adapt(plans[f])
        x = synth.gen.model_input(m, request=i)
        a, b = sw.run(x), rs.run(x)
        assert all(p.tobytes() == q.tobytes() for p, q in zip(a, b)), f
        check_oracle(sw, a, x, request=i)
        assert sw.engine.stats()["infer_calls"] >= 1
    other = synth.arch.vgg16()
    with pytest.raises(capi.SwapnetError) as ei:
        sw.engine.adapt(capi.Plan.partition(capi.Desc(other), int(OP.weight_bytes(other) * 0.5), capi.options()))
    assert ei.value.code == capi.ERR_INVALID_ARG
    with pytest.raises(capi.SwapnetError):
        sw.engine.adapt(capi.Plan.resident(d))


def test_driver_pinned_host_weights():
    """Weights packed in swapnet_host_alloc memory are used in place."""
    m = synth.arch.resnet50()
    w = synth.gen.model_weights(m)
    flat = [np.ascontiguousarray(t) for lw in w for t in lw]
    host = capi.HostWeights.allocate([t.nbytes for t in flat], pinned=True)
    for i, t in enumerate(flat):
        host.view(i)[:] = t.view(np.uint8).reshape(-1)
    x = synth.gen.model_input(m)
    d = capi.Desc(m)
    budget = int(OP.weight_bytes(m) * 0.4) // 256 * 256
    a = Runner(m, w, capi.Plan.partition(d, budget, capi.options()), host).run(x)
    b = Runner(m, w, capi.Plan.resident(d), capi.HostWeights(w)).run(x)
    assert all(p.tobytes() == q.tobytes() for p, q in zip(a, b))


def test_device_wait_timeout_is_reported_and_the_context_stays_usable():
    """Failure detection on the GPU without a fault: a kernel's bounded wait
    on an mbarrier that nothing completes gives up after its limit, the
    library reports SWAPNET_ERR_TIMEOUT once, and inference afterwards gives
    the resident bits again."""
    import torch
    m = synth.arch.resnet50()
    w = synth.gen.model_weights(m)
    x = synth.gen.model_input(m)
    d = capi.Desc(m)
    host = capi.HostWeights(w)
    rs = Runner(m, w, capi.Plan.resident(d), host)
    before = rs.run(x)
    rc = capi.lib().swapnet_debug_wait_timeout(capi.C.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert rc == capi.ERR_TIMEOUT
    assert capi.lib().swapnet_debug_wait_timeout(None) == capi.ERR_TIMEOUT  # the legacy stream too
    budget = int(OP.weight_bytes(m) * 0.4) // 256 * 256
    sw = Runner(m, w, capi.Plan.partition(d, budget, capi.options()), host)
    for a, b in zip(sw.run(x), before):
        assert a.tobytes() == b.tobytes()
    rs.engine.sync()  # the error word was cleared: no stale timeout


@pytest.mark.parametrize("what,code", [(1, capi.ERR_CUDA), (2, capi.ERR_OOM), (3, capi.ERR_CUDA)])
def test_injected_load_failures_leave_nothing_behind(what, code):
    """Host-side fault injection at load (registration, device allocation,
    stream creation): swapnet_load fails with the matching status, releases
    what it had set up, and the next load of the same weights works."""
    m = synth.arch.resnet50()
    w = synth.gen.model_weights(m)
    x = synth.gen.model_input(m)
    d = capi.Desc(m)
    host = capi.HostWeights(w)
    plan = capi.Plan.partition(d, int(OP.weight_bytes(m) * 0.4) // 256 * 256, capi.options())
    assert capi.lib().swapnet_debug_fail_next(what, 1) == capi.OK
    with pytest.raises(capi.SwapnetError) as ei:
        capi.Engine(plan, host)
    assert ei.value.code == code, str(ei.value)
    assert capi.lib().swapnet_debug_fail_next(what, 0) == capi.OK
    got = Runner(m, w, plan, host).run(x)
    ref = Runner(m, w, capi.Plan.resident(d), host).run(x)
    assert all(a.tobytes() == b.tobytes() for a, b in zip(got, ref))


@pytest.mark.parametrize("variant", [capi.SWAP_MEMCPY, capi.SWAP_ZEROCOPY])
def test_swap_times_inside_the_replayed_graph(variant):
    """Swap timing in the graph (event-record nodes around each block's
    swap-in on the copy stream): the outputs stay the resident bits, every
    swapped block reports a positive time that is at least its bytes over a
    generous link ceiling, and the swaps of one inference add up to no more
    than the inference's own time on its stream."""
    import torch
    m = synth.arch.MODELS["resnet50"]()
    w = synth.gen.model_weights(m)
    d = capi.Desc(m)
    host = capi.HostWeights(w)
    wb = OP.weight_bytes(m)
    plan = capi.Plan.partition(d, int(wb * 0.4) // 256 * 256, capi.options(swap_variant=variant))
    nb = plan.info()["n_blocks"]
    sw = Runner(m, w, plan, host)
    rs = Runner(m, w, capi.Plan.resident(d), host)
    x = synth.gen.model_input(m, request=3)
    ref = rs.run(x)
    sw.engine.set_swap_timing(True)
    for _ in range(2):
        got = sw.run(x)
        assert all(p.tobytes() == q.tobytes() for p, q in zip(got, ref))
    s = torch.cuda.current_stream()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(s)
    sw.engine.infer(sw.d_in.data_ptr(), sw.d_out.data_ptr(), s.cuda_stream)
    b.record(s)
    b.synchronize()
    us = sw.engine.last_swap_times(nb)
    blocks = plan.blocks()
    for blk, t in zip(blocks, us):
        if blk["bytes"]:
            assert t > 0.0
            assert blk["bytes"] / (t * 1e-6) < 1e12   # under 1 TB/s: a real copy was timed
    assert sum(us) <= a.elapsed_time(b) * 1e3 * 1.01
    sw.engine.set_swap_timing(False)
    got = sw.run(x)
    assert all(p.tobytes() == q.tobytes() for p, q in zip(got, ref))
    sw.engine.sync()


def _min_feasible_budget(d, opt, hi):
    """Smallest multiple of 256 bytes the planner accepts (feasibility grows
    with the budget)."""
    lo = 0                       # infeasible
    while hi - lo > 256:
        mid = (lo + hi) // 2 // 256 * 256
        mid = max(mid, lo + 256)
        try:
            capi.Plan.partition(d, mid, opt)
            hi = mid
        except capi.SwapnetError as e:
            assert e.code == capi.ERR_INFEASIBLE
            lo = mid
    return hi


def test_degenerate_budgets_bit_exact():
    """The edge budgets run and equal resident bit for bit: the smallest
    budget the planner accepts (256 bytes less is refused as infeasible), and
    four times the weight bytes, where the paper's method still swaps every
    block while a resident prefix keeps the whole model in one block that is
    never swapped."""
    layers = [_conv(-1, 16, 32, 3), _conv(0, 32, 64, 3, stride=2), _conv(1, 64, 64, 1, res=1),
              dict(op="maxpool", src=[2], kh=2, kw=2, stride=2, pad=0),
              dict(op="gap", src=[3]),
              dict(op="linear", src=[4], k=64, n=40, act="none", res=None, res_post=False)]
    m = _model(layers, (1, 24, 24, 16))
    w = synth.gen.model_weights(m)
    x = synth.gen.model_input(m)
    d = capi.Desc(m)
    host = capi.HostWeights(w)
    wb = OP.weight_bytes(m)
    base = Runner(m, w, capi.Plan.resident(d), host).run(x)[0].tobytes()
    opt = capi.options()
    lo = _min_feasible_budget(d, opt, 4 * wb // 256 * 256)
    with pytest.raises(capi.SwapnetError) as ei:
        capi.Plan.partition(d, lo - 256, opt)
    assert ei.value.code == capi.ERR_INFEASIBLE
    tight = Runner(m, w, capi.Plan.partition(d, lo, opt), host)
    assert tight.info["n_blocks"] >= 3
    assert tight.run(x)[0].tobytes() == base
    big = 4 * wb // 256 * 256
    sw = Runner(m, w, capi.Plan.partition(d, big, opt), host)
    before = sw.engine.stats()["bytes_swapped"]
    assert sw.run(x)[0].tobytes() == base
    swapped = sw.engine.stats()["bytes_swapped"] - before    # every tensor, padding between them included
    n_tensors = sum(len(t) for t in w)
    assert wb - 256 * n_tensors < swapped <= wb, (swapped, wb)
    pre = Runner(m, w, capi.Plan.partition(d, big, capi.options(resident_prefix=1)), host)
    assert pre.info["n_blocks"] == 1 and pre.info["prefix_units"] == pre.info["n_units"]
    before = pre.engine.stats()["bytes_swapped"]
    for _ in range(2):
        got = pre.run(x)
        assert got[0].tobytes() == base
    assert pre.engine.stats()["bytes_swapped"] == before
    check_close(m, pre.decode(got), oracle_outputs(m, w, x))


def _check_pipeline_order(tl, total_us):
    """Swaps (those of this inference: start >= 0) one after another, each
    block's layers after its own swap and the previous block's layers, a
    swap after the layers of the block two back."""
    eps = 1.0                                   # event resolution, microseconds
    for k, (s0, s1, e0, e1) in enumerate(tl):
        assert 0.0 <= e0 <= e1 + eps, (k, tl[k])
        if k:
            assert tl[k - 1][3] <= e0 + eps, (k, tl[k - 1], tl[k])
        if s0 < 0:                              # not swapped in during this inference
            assert s1 < 0
            continue
        assert s0 <= s1 + eps and s1 <= e0 + eps, (k, tl[k])
        if k and tl[k - 1][1] >= 0:
            assert tl[k - 1][1] <= s0 + eps, (k, tl[k - 1], tl[k])
        if k >= 2:
            assert tl[k - 2][3] <= s0 + eps, (k, tl[k - 2], tl[k])
    assert tl[-1][3] <= total_us + eps


@pytest.mark.parametrize("variant", [capi.SWAP_MEMCPY, capi.SWAP_ZEROCOPY])
def test_graph_timeline_follows_the_pipeline_order(variant):
    """The block timeline of a replayed inference graph obeys the ordering
    of the Sec. 4.3 pipeline: swaps one after another on the copy stream,
    each block's layers after its own swap and after the previous block's
    layers, a block's swap after the layers of the block that last held
    its place (two blocks back); everything inside the inference's own time
    on its stream.  The outputs stay the resident bits."""
    import torch
    m = synth.arch.MODELS["resnet50"]()
    w = synth.gen.model_weights(m)
    d = capi.Desc(m)
    host = capi.HostWeights(w)
    wb = OP.weight_bytes(m)
    plan = capi.Plan.partition(d, int(wb * 0.4) // 256 * 256, capi.options(swap_variant=variant))
    nb = plan.info()["n_blocks"]
    assert nb >= 3
    sw = Runner(m, w, plan, host)
    ref = Runner(m, w, capi.Plan.resident(d), host).run(synth.gen.model_input(m))
    sw.engine.set_graph_timeline(True)
    got = sw.run(synth.gen.model_input(m))
    assert all(p.tobytes() == q.tobytes() for p, q in zip(got, ref))
    s = torch.cuda.current_stream()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(s)
    sw.engine.infer(sw.d_in.data_ptr(), sw.d_out.data_ptr(), s.cuda_stream)
    b.record(s)
    b.synchronize()
    _check_pipeline_order(sw.engine.last_graph_timeline(nb), a.elapsed_time(b) * 1e3)
    sw.engine.set_graph_timeline(False)
    got = sw.run(synth.gen.model_input(m))
    assert all(p.tobytes() == q.tobytes() for p, q in zip(got, ref))
    sw.engine.sync()


def test_timing_follows_an_adapted_plan():
    """Swap timing and the graph timeline stay on across
    swapnet_engine_adapt to a plan with more blocks: every block of the new
    plan is timed and the timeline keeps the pipeline order."""
    import torch
    m = synth.arch.MODELS["resnet50"]()
    w = synth.gen.model_weights(m)
    d = capi.Desc(m)
    host = capi.HostWeights(w)
    wb = OP.weight_bytes(m)
    p_big = capi.Plan.partition(d, int(wb * 0.8) // 256 * 256, capi.options())
    p_small = capi.Plan.partition(d, int(wb * 0.4) // 256 * 256, capi.options())
    nb = p_small.info()["n_blocks"]
    assert nb > p_big.info()["n_blocks"]
    sw = Runner(m, w, p_big, host)
    x = synth.gen.model_input(m)
    ref = Runner(m, w, capi.Plan.resident(d), host).run(x)
    sw.engine.set_swap_timing(True)
    sw.engine.set_graph_timeline(True)
    assert sw.run(x)[0].tobytes() == ref[0].tobytes()
    sw.engine.adapt(p_small)
    sw.plan = p_small
    sw.offs = p_small.output_offsets()
    s = torch.cuda.current_stream()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(s)
    sw.engine.infer(sw.d_in.data_ptr(), sw.d_out.data_ptr(), s.cuda_stream)
    b.record(s)
    b.synchronize()
    assert sw.outputs_raw()[0].tobytes() == ref[0].tobytes()
    us = sw.engine.last_swap_times(nb)
    assert all(t > 0.0 for t in us)
    _check_pipeline_order(sw.engine.last_graph_timeline(nb), a.elapsed_time(b) * 1e3)
    sw.engine.set_graph_timeline(False)
    sw.engine.set_swap_timing(False)
    sw.engine.sync()


def test_graph_timeline_with_first_block_prefetch():
    """First-block prefetch: the first block was swapped in by the previous
    inference, so the timeline reports no swap for it in this one (-1), and
    the other blocks keep the pipeline order; outputs stay the resident bits
    over back-to-back inferences."""
    import torch
    m = synth.arch.MODELS["resnet50"]()
    w = synth.gen.model_weights(m)
    d = capi.Desc(m)
    host = capi.HostWeights(w)
    plan = capi.Plan.partition(d, int(OP.weight_bytes(m) * 0.4) // 256 * 256, capi.options(prefetch=1))
    nb = plan.info()["n_blocks"]
    sw = Runner(m, w, plan, host)
    x = synth.gen.model_input(m)
    ref = Runner(m, w, capi.Plan.resident(d), host).run(x)
    sw.engine.set_graph_timeline(True)
    for _ in range(2):
        assert sw.run(x)[0].tobytes() == ref[0].tobytes()
    s = torch.cuda.current_stream()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(s)
    sw.engine.infer(sw.d_in.data_ptr(), sw.d_out.data_ptr(), s.cuda_stream)
    b.record(s)
    b.synchronize()
    tl = sw.engine.last_graph_timeline(nb)
    assert tl[0][0] < 0 and tl[0][1] < 0
    assert all(t[0] >= 0 for t in tl[1:])
    _check_pipeline_order(tl, a.elapsed_time(b) * 1e3)
    sw.engine.set_graph_timeline(False)
    assert sw.outputs_raw()[0].tobytes() == ref[0].tobytes()
    sw.engine.sync()
