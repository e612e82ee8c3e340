"""Pins of the CPU oracle's forward pass against brute force, library
routines, closed forms and invariants (no GPU)."""
import itertools

import numpy as np
import pytest
import torch

from oracle import forward as F
import synth


def brute_conv(x, w, b, s, p):
    """Seven nested loops straight from the conv definition (tiny shapes)."""
    n, ci, h, wd = x.shape
    co, kh, kw, _ = w.shape
    ho, wo = (h + 2 * p - kh) // s + 1, (wd + 2 * p - kw) // s + 1
    y = np.zeros((n, co, ho, wo))
    for a, c, oh, ow in itertools.product(range(n), range(co), range(ho), range(wo)):
        acc = b[c]
        for k, i, j in itertools.product(range(ci), range(kh), range(kw)):
            ih, iw = oh * s + i - p, ow * s + j - p
            if 0 <= ih < h and 0 <= iw < wd:
                acc += x[a, k, ih, iw] * w[c, i, j, k]
        y[a, c, oh, ow] = acc
    return y


@pytest.mark.parametrize("s,p,k", [(1, 0, 3), (1, 1, 3), (2, 1, 3), (2, 3, 7), (2, 0, 1), (1, 0, 1)])
def test_conv_vs_brute_force(s, p, k):
    r = np.random.default_rng(10 + s + p + k)
    x = r.normal(size=(2, 3, 9, 8))
    w = r.normal(size=(4, k, k, 3))
    b = r.normal(size=4)
    np.testing.assert_allclose(F.conv2d(x, w, b, s, p), brute_conv(x, w, b, s, p), rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("s,p,k", [(1, 1, 3), (2, 1, 3), (2, 3, 7), (2, 0, 1)])
def test_conv_vs_torch_f64(s, p, k):
    r = np.random.default_rng(7)
    x = r.normal(size=(2, 16, 20, 18))
    w = r.normal(size=(24, k, k, 16))
    b = r.normal(size=24)
    ref = torch.nn.functional.conv2d(torch.from_numpy(x), torch.from_numpy(w.transpose(0, 3, 1, 2).copy()),
                                     torch.from_numpy(b), stride=s, padding=p).numpy()
    np.testing.assert_allclose(F.conv2d(x, w, b, s, p), ref, rtol=1e-11, atol=1e-11)


def test_conv1x1_is_matmul():
    r = np.random.default_rng(3)
    x = r.normal(size=(1, 8, 5, 6))
    w = r.normal(size=(5, 1, 1, 8))
    y = F.conv2d(x, w, np.zeros(5), 1, 0)
    ref = np.einsum("oc,nchw->nohw", w[:, 0, 0, :], x)
    np.testing.assert_allclose(y, ref, rtol=1e-12)


def test_conv_delta_image_stride2():
    # A delta at (h0, w0) hits output (oh, ow) through tap (i, j) with
    # oh*2 + i - 1 = h0, ow*2 + j - 1 = w0; every output equals that weight.
    x = np.zeros((1, 1, 9, 9))
    h0, w0 = 4, 5
    x[0, 0, h0, w0] = 1.0
    w = np.arange(9, dtype=np.float64).reshape(1, 3, 3, 1) + 1.0
    y = F.conv2d(x, w, np.zeros(1), 2, 1)
    expect = np.zeros_like(y)
    for oh in range(y.shape[2]):
        for ow in range(y.shape[3]):
            i, j = h0 - 2 * oh + 1, w0 - 2 * ow + 1
            if 0 <= i < 3 and 0 <= j < 3:
                expect[0, 0, oh, ow] = w[0, i, j, 0]
    np.testing.assert_array_equal(y, expect)
    assert np.count_nonzero(y) == 2  # w0=5 is hit by two taps, h0=4 by one


def test_linear_vs_brute_and_identity():
    r = np.random.default_rng(5)
    x = r.normal(size=(3, 7))
    w = r.normal(size=(4, 7))
    b = r.normal(size=4)
    y = F.linear(x, w, b)
    for m in range(3):
        for o in range(4):
            assert abs(y[m, o] - (b[o] + sum(x[m, i] * w[o, i] for i in range(7)))) < 1e-12
    np.testing.assert_array_equal(F.linear(x, np.eye(7), np.zeros(7)), x)


def test_maxpool_vs_brute_and_padding():
    r = np.random.default_rng(6)
    x = r.normal(size=(1, 2, 7, 6)) - 10.0          # all negative: zero padding would win
    y = F.maxpool(x, 3, 3, 2, 1)
    ref = torch.nn.functional.max_pool2d(torch.from_numpy(x), 3, 2, 1).numpy()
    np.testing.assert_array_equal(y, ref)
    assert y.max() < -5.0
    y2 = F.maxpool(x, 2, 2, 2, 0)
    for c, i, j in itertools.product(range(2), range(3), range(3)):
        assert y2[0, c, i, j] == x[0, c, 2 * i:2 * i + 2, 2 * j:2 * j + 2].max()


def test_gap_upsample_concat():
    x = np.full((1, 3, 4, 5), 2.5)
    np.testing.assert_array_equal(F.gap(x), np.full((1, 3, 1, 1), 2.5))
    r = np.random.default_rng(1).normal(size=(1, 2, 3, 3))
    u = F.upsample2x(r)
    for i, j in itertools.product(range(6), range(6)):
        assert np.all(u[0, :, i, j] == r[0, :, i // 2, j // 2])
    c = F.concat(r, u[:, :, ::2, ::2])
    assert c.shape == (1, 4, 3, 3) and np.all(c[:, 2:] == r)


def test_activations_and_residual_order():
    y = np.array([-2.0, -0.5, 0.0, 3.0])
    np.testing.assert_array_equal(F.act_fn(y, "relu"), [0, 0, 0, 3])
    np.testing.assert_allclose(F.act_fn(y, "leaky"), [-0.2, -0.05, 0, 3])
    # pre-add: relu(acc + r); post-add: leaky(acc) + r -> differ on negative acc
    layer = dict(op="linear", src=[-1], k=1, n=1, act="relu", res=0, res_post=False)
    w = [np.array([[1.0]], dtype=np.float32), np.array([0.0], dtype=np.float32)]
    x = np.array([[[[-3.0]]]])
    acts = {0: np.array([[[[1.0]]]])}
    assert F.run_layer(layer, "f32", w, acts, x)[0, 0, 0, 0] == 0.0          # relu(-3 + 1)
    layer.update(res_post=True)
    assert F.run_layer(layer, "f32", w, acts, x)[0, 0, 0, 0] == 1.0          # relu(-3) + 1


def test_swiglu_branch_closed_forms():
    """SwiGLU layer (Sec. 10 names LLaMA-7B; its FFN is down(silu(gate x) *
    up x)): the layer with act swiglu is the up projection and its residual
    operand is the stored gate output r, so y = silu(r) * (acc + b).  One
    hand-worked case tells apart the plausible mistakes: acc = 1.5, b = 0.5,
    r = -1 gives silu(-1) * 2 = -2 / (1 + e) = -0.5378828427399902; swapping
    the gate and up roles would give silu(2) * (-1) = -1.7615941559557649,
    dropping the bias silu(-1) * 1.5 = -0.4034121320549927."""
    layer = dict(op="linear", src=[-1], k=1, n=1, act="swiglu", res=0, res_post=False)
    w = [np.array([[1.0]], dtype=np.float32), np.array([0.5], dtype=np.float32)]
    x = np.array([[[[1.5]]]])
    got = F.run_layer(layer, "f32", w, {0: np.array([[[[-1.0]]]])}, x)[0, 0, 0, 0]
    np.testing.assert_allclose(got, -0.5378828427399902, rtol=1e-7)
    # a zero gate closes the branch whatever the up projection gives
    assert F.run_layer(layer, "f32", w, {0: np.array([[[[0.0]]]])}, x)[0, 0, 0, 0] == 0.0
    # a large negative gate closes it too; a large positive one passes
    # r * (acc + b): silu(r) -> r as r grows
    assert abs(F.run_layer(layer, "f32", w, {0: np.array([[[[-60.0]]]])}, x)[0, 0, 0, 0]) < 1e-20
    np.testing.assert_allclose(F.run_layer(layer, "f32", w, {0: np.array([[[[40.0]]]])}, x)[0, 0, 0, 0],
                               80.0, rtol=1e-7)
    # the branch is elementwise over features: gate [0, -1] and acc + b [5, 2]
    layer2 = dict(layer, k=2, n=2)
    w2 = [np.array([[1.0, 0.0], [0.0, 1.0]], dtype=np.float32), np.array([0.5, 0.5], dtype=np.float32)]
    x2 = np.array([[[[4.5]], [[1.5]]]])
    got2 = F.run_layer(layer2, "f32", w2, {0: np.array([[[[0.0]], [[-1.0]]]])}, x2).reshape(-1)
    np.testing.assert_allclose(got2, [0.0, -0.5378828427399902], rtol=1e-7, atol=0)


def test_rounding_ties_and_values():
    # fp16: 1 + 2^-11 is a tie between 1 and 1 + 2^-10 -> even (1)
    assert F.round_as(1 + 2.0 ** -11, "f16") == 1.0
    assert F.round_as(1 + 3 * 2.0 ** -11, "f16") == 1 + 2.0 ** -9
    assert F.round_as(65520.0, "f16") == np.inf       # rounds past the largest finite half
    # bf16 keeps 8 significant bits
    assert F.round_as(1 + 2.0 ** -8, "bf16") == 1.0
    assert F.round_as(1 + 3 * 2.0 ** -8, "bf16") == 1 + 2.0 ** -6
    assert F.round_as(-3.0 * 2 ** 100 + 2.0 ** 93, "bf16") == -3.0 * 2 ** 100
    assert F.round_as(np.pi, "bf16") == 3.140625


def test_rounding_matches_generator_storage():
    # Two independent RNE implementations (oracle: frexp/rint; generator:
    # integer bit arithmetic) must agree on every value.
    r = np.random.default_rng(11)
    x = np.concatenate([r.normal(size=20000) * 10.0 ** r.integers(-6, 6, 20000),
                        (1 + (2 * np.arange(200) + 1) * 2.0 ** -9)])
    bits = synth.gen.round_to_storage(x, "bf16")
    np.testing.assert_array_equal(F.decode(bits, "bf16"), F.round_as(x, "bf16"))
    h = synth.gen.round_to_storage(x, "f16")
    np.testing.assert_array_equal(F.decode(h, "f16"), F.round_as(x, "f16"))


def _tiny_resnet():
    L = [dict(op="conv", src=[-1], cin=8, cout=16, kh=3, kw=3, stride=2, pad=1, act="relu", res=None, res_post=False),
         dict(op="maxpool", src=[0], kh=3, kw=3, stride=2, pad=1),
         dict(op="conv", src=[1], cin=16, cout=16, kh=1, kw=1, stride=1, pad=0, act="relu", res=None, res_post=False),
         dict(op="conv", src=[2], cin=16, cout=16, kh=3, kw=3, stride=1, pad=1, act="relu", res=1, res_post=False),
         dict(op="upsample2x", src=[3]),
         dict(op="conv", src=[4], cin=16, cout=8, kh=1, kw=1, stride=1, pad=0, act="leaky", res=None, res_post=True),
         dict(op="concat", src=[5, 4]),
         dict(op="gap", src=[6]),
         dict(op="linear", src=[7], k=24, n=10, act="none", res=None, res_post=False)]
    return dict(name="yolov3", model_id=9, dtype="f16", input=(2, 16, 16, 8), layers=L, outputs=[8])


def test_forward_is_composition_of_blocks():
    m = _tiny_resnet()
    w = synth.gen.model_weights(m)
    x = synth.gen.model_input(m)
    ref = F.forward(m, w, x)[0]
    x_in = F.nhwc_to_nchw(F.decode(x, m["dtype"]))
    for cuts in ([3], [1, 5], [2, 4, 6, 8], list(range(1, 9))):
        acts = {}
        b = [0] + cuts + [len(m["layers"])]
        for lo, hi in zip(b[:-1], b[1:]):
            F.forward_range(m, w, acts, x_in, lo, hi)
        np.testing.assert_array_equal(F.nchw_to_nhwc(acts[8]), ref)


def test_outputs_are_representable():
    m = _tiny_resnet()
    out = F.forward(m, synth.gen.model_weights(m), synth.gen.model_input(m))[0]
    np.testing.assert_array_equal(out.astype(np.float16).astype(np.float64), out)


@pytest.mark.parametrize("name", ["resnet50", "vgg16", "yolov3"])
def test_workload_activations_stay_in_fp16_range(name):
    # every layer output of the full-size workload is finite and well inside
    # the fp16 range (no overflow, no collapse to zero)
    m = synth.arch.MODELS[name]()
    w = synth.gen.model_weights(m)
    x = synth.gen.model_input(m)
    x_in = F.nhwc_to_nchw(F.decode(x, m["dtype"]))
    acts = F.forward_range(m, w, {}, x_in, 0, len(m["layers"]))
    for a in acts.values():
        assert np.all(np.isfinite(a)) and np.max(np.abs(a)) < 6e4
        assert np.sqrt(np.mean(a ** 2)) > 1e-2


# ----------------------------------------------------------------- decoder ops
def test_rmsnorm_closed_forms():
    g = np.array([0.5, 2.0, -1.0, 3.0])
    y = F.rmsnorm(np.full((1, 4), -7.0), g, 1e-12)          # constant row -> sign * g
    np.testing.assert_allclose(y[0], -g, rtol=1e-9)
    r = np.random.default_rng(3).normal(size=(3, 64))
    np.testing.assert_allclose(F.rmsnorm(5.0 * r, np.ones(64), 0.0), F.rmsnorm(r, np.ones(64), 0.0), rtol=1e-12)
    y = F.rmsnorm(r, np.ones(64), 0.0)
    np.testing.assert_allclose(np.mean(y * y, axis=1), 1.0, rtol=1e-12)   # unit mean square


def test_rope_identity_norm_composition():
    r = np.random.default_rng(4).normal(size=(3, 32))          # 2 heads x 16
    np.testing.assert_allclose(F.rope(r, [0, 0, 0], 2, 10000.0), r, rtol=0, atol=0)
    y = F.rope(r, [5, 17, 300], 2, 10000.0)
    pn = lambda a: np.hypot(a.reshape(3, 16, 2)[..., 0], a.reshape(3, 16, 2)[..., 1])
    np.testing.assert_allclose(pn(y), pn(r), rtol=1e-12)
    # one pair by hand: dims (2, 3) of head 1 use i = 1 -> angle = p * theta^(-2/16)
    p, ang = 17, 17 * 10000.0 ** (-2.0 / 16)
    x0, x1 = r[1, 16 + 2], r[1, 16 + 3]
    np.testing.assert_allclose(y[1, 16 + 2:16 + 4], [x0 * np.cos(ang) - x1 * np.sin(ang),
                                                     x0 * np.sin(ang) + x1 * np.cos(ang)], rtol=1e-12)
    # rotations compose: rope(rope(x, a), b) = rope(x, a + b)
    np.testing.assert_allclose(F.rope(F.rope(r, [3, 4, 5], 2, 10000.0), [7, 8, 9], 2, 10000.0),
                               F.rope(r, [10, 12, 14], 2, 10000.0), rtol=1e-10, atol=1e-12)


def test_attention_special_cases_and_brute_force():
    r = np.random.default_rng(5)
    v = r.normal(size=(6, 8))
    k = r.normal(size=(6, 8))
    # a single query at position 0 sees only itself: output = v[0]
    np.testing.assert_allclose(F.causal_attention(r.normal(size=(1, 8)), k, v, 0, 2), v[:1], rtol=1e-12)
    # zero query: uniform weights over the visible positions
    out = F.causal_attention(np.zeros((2, 8)), k, v, 3, 2)
    np.testing.assert_allclose(out[0], v[:4].mean(axis=0), rtol=1e-12)
    np.testing.assert_allclose(out[1], v[:5].mean(axis=0), rtol=1e-12)
    # brute force: explicit loops over heads, queries and keys
    q = r.normal(size=(3, 8))
    got = F.causal_attention(q, k, v, 2, 2)
    for h in range(2):
        for i in range(3):
            n = 2 + i + 1
            s = [sum(q[i, h * 4 + d] * k[j, h * 4 + d] for d in range(4)) / 2.0 for j in range(n)]
            e = [np.exp(x - max(s)) for x in s]
            for d in range(4):
                ref = sum(e[j] * v[j, h * 4 + d] for j in range(n)) / sum(e)
                assert abs(got[i, h * 4 + d] - ref) < 1e-12


def test_silu_and_argmax():
    assert F.silu(0.0) == 0.0
    np.testing.assert_allclose(F.silu(1.0), 1.0 / (1.0 + np.exp(-1.0)), rtol=1e-15)
    np.testing.assert_allclose(F.silu(40.0), 40.0, rtol=1e-15)
    assert abs(F.silu(-40.0)) < 1e-15
    layer = dict(op="argmax", src=[-1])
    x = np.array([[1.0, 3.0, 3.0, 2.0], [5.0, 5.0, 5.0, 5.0]]).reshape(2, 4, 1, 1)
    out = F.run_layer(layer, "bf16", [], {}, x)
    assert out.ravel().tolist() == [1.0, 0.0]      # ties -> lowest index


def _tiny_llm(tokens):
    return synth.arch.llm(layers=2, d=64, heads=2, ffn=160, vocab=300, tokens=tokens, max_seq=24)


def test_embedding_gathers_rows():
    m = _tiny_llm(5)
    w = synth.gen.model_weights(m)
    ids = np.array([3, 299, 0, 3, 17], dtype=np.int32).reshape(5, 1, 1, 1)
    out = F.run_layer(m["layers"][0], "bf16", w[0], {}, ids)
    np.testing.assert_array_equal(out.reshape(5, -1), F.decode(w[0][0], "bf16")[[3, 299, 0, 3, 17]])


def test_kv_cache_prefill_then_decode_equals_longer_prefill():
    # logits of token T from prefill(T) + one decode step equal the last row
    # of prefill(T + 1): the cache carries exactly the keys and values
    w = synth.gen.model_weights(_tiny_llm(9))
    ids = synth.gen.model_input(_tiny_llm(9))
    st = F.new_state()
    F.forward(_tiny_llm(8), w, ids[:8], state=st)
    step = F.forward(_tiny_llm(1), w, ids[8:9], state=st)[0]
    assert st["pos"] == 9
    full = F.forward(_tiny_llm(9), w, ids)[0]
    got, ref = step.ravel(), full[8].ravel()
    assert np.linalg.norm(got - ref) <= 1e-3 * np.linalg.norm(ref)
