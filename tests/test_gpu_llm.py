"""GPU parity of the LLM-shaped decoder through the C ABI: prefill and greedy
decode steps (teacher-forced) against the oracle, swapped against resident
bit for bit, and the KV-cache bound."""
import numpy as np
import pytest

import synth
from oracle import forward as F
from oracle import plan as OP
from paper_2401_16757_gb300 import capi
from helpers import rel_l2

pytestmark = pytest.mark.gpu

SMALL = dict(layers=2, d=256, heads=2, ffn=688, vocab=1000, max_seq=80)

# Relative-L2 bars.  Every layer, given the same stored inputs as the oracle
# (local parity), is held to 2e-3 per output tensor.  End to end, bf16
# chains saturate at the bf16 rounding noise: every stored bf16 tensor turns
# an input discrepancy e into about sqrt(e * ulp) of flipped roundings, so
# after a few chained rounding points GPU and oracle differ by about one bf16
# ulp per element however exact each kernel is.  One ulp is between 2^-8 and
# 2^-7 of the element it rounds, so whole decoders are held to 2^-7 (the
# small one-layer model happens to stay within 2e-3 and is held to that).
LOCAL_TOL = 2e-3
TOL = {1: 2e-3, 2: 2.0 ** -7}
CHAIN_TOL = 2.0 ** -7


class Decoder:
    """A prefill engine and a decode engine sharing weights and KV state."""

    def __init__(self, prefill_tokens, budget_frac=0.5, resident=False, host=None, weights=None, layers=2,
                 opts=None, **over):
        import torch
        self.torch = torch
        cfg = dict(SMALL, layers=layers, **over)
        self.vocab = cfg["vocab"]
        self.mp = synth.arch.llm(tokens=prefill_tokens, **cfg)
        self.md = synth.arch.llm(tokens=1, **cfg)
        self.w = weights or synth.gen.model_weights(self.mp)
        self.host = host or capi.HostWeights(self.w)
        budget = int(OP.weight_bytes(self.mp) * budget_frac) // 256 * 256
        self.engines, self.bufs = [], []
        for m in (self.mp, self.md):
            d = capi.Desc(m)
            o = capi.options(**(opts or {}))
            plan = capi.Plan.resident(d, o) if resident else capi.Plan.partition(d, budget, o)
            eng = capi.Engine(plan, self.host)
            info = plan.info()
            din = torch.zeros(max(16, info["input_bytes"]), dtype=torch.uint8, device="cuda")
            dout = torch.zeros(info["output_bytes"], dtype=torch.uint8, device="cuda")
            self.engines.append((plan, eng, info))
            self.bufs.append((din, dout, plan.output_offsets()))
        self.state_bytes = self.engines[0][2]["state_bytes"]
        assert self.state_bytes == self.engines[1][2]["state_bytes"] > 0
        self.state = torch.zeros(self.state_bytes, dtype=torch.uint8, device="cuda")
        for _, eng, _ in self.engines:
            eng.bind_state(self.state.data_ptr(), self.state_bytes)

    def run(self, which, ids):
        torch = self.torch
        plan, eng, info = self.engines[which]
        din, dout, offs = self.bufs[which]
        din[:ids.nbytes].copy_(torch.from_numpy(np.ascontiguousarray(ids, dtype=np.int32).view(np.uint8).reshape(-1)))
        eng.infer(din.data_ptr(), dout.data_ptr(), torch.cuda.current_stream().cuda_stream)
        eng.sync()
        host = dout.cpu().numpy()
        t = ids.size
        v = self.vocab
        logits = host[offs[0]:offs[0] + t * v * 2].view(np.uint16).reshape(t, v)
        tokens = host[offs[1]:offs[1] + t * 4].view(np.int32).copy()
        return logits, tokens


def _check_step(got_bits, got_tok, ref_logits, ref_tok, bar):
    got = F.decode(got_bits, "bf16")
    e = rel_l2(got, ref_logits)
    assert e <= bar, e
    tol = 3 * bar * np.max(np.abs(ref_logits))
    for row in range(got.shape[0]):
        g, r = int(got_tok[row]), int(ref_tok[row])
        assert g == int(np.argmax(got[row]))
        if g != r:   # a near-tie: several answers are right
            assert ref_logits[row, r] - ref_logits[row, g] <= tol


@pytest.mark.parametrize("layers", [1, 2])
def test_llm_prefill_and_greedy_decode_teacher_forced(layers):
    dec = Decoder(prefill_tokens=64, layers=layers)
    ids = synth.gen.model_input(dec.mp).reshape(-1)
    st = F.new_state()
    ref = F.forward(dec.mp, dec.w, ids.reshape(-1, 1, 1, 1), state=st)
    logits, toks = dec.run(0, ids)
    _check_step(logits, toks, ref[0].reshape(64, -1), ref[1].reshape(-1), TOL[layers])
    tok = int(toks[-1])
    for step in range(8):                      # the oracle consumes the GPU's token
        ref = F.forward(dec.md, dec.w, np.array([tok], dtype=np.int32).reshape(1, 1, 1, 1), state=st)
        logits, toks = dec.run(1, np.array([tok], dtype=np.int32))
        _check_step(logits, toks, ref[0].reshape(1, -1), ref[1].reshape(-1), TOL[layers])
        tok = int(toks[0])
    assert int(dec.state[:4].cpu().numpy().view(np.int32)[0]) == 64 + 8


WIDE = dict(layers=1, d=1024, heads=8, ffn=2752, max_seq=160)
# the 7B workload's widths (one decoder layer of the 32): d 4096, 32 heads,
# FFN 11008, vocabulary 32000, a 512-token prefill
FULL = dict(layers=1, d=4096, heads=32, ffn=11008, vocab=32000, max_seq=544)


def _weights_parallel(model):
    """synth.gen.model_weights, one tensor per thread (the same seeded
    streams; the generators release the GIL on large draws)."""
    import concurrent.futures as cf
    jobs = [(li, ti, shp) for li, L in enumerate(model["layers"])
            for ti, (_, shp) in enumerate(synth.arch.tensor_shapes(L))]
    with cf.ThreadPoolExecutor(max_workers=16) as ex:
        out = list(ex.map(lambda j: synth.gen.llm_tensor(model, *j), jobs))
    w = [[] for _ in model["layers"]]
    for (li, _, _), t in zip(jobs, out):
        w[li].append(t)
    return w


def test_llm_full_width_layer_prefill_512_and_decode():
    """The bench's launch configuration at full width on one decoder layer
    (the whole 32-layer model is tests/test_gpu_llm7b.py): 512-token prefill
    and two greedy decode passes, swapped through a budget of half the
    weight bytes, against the oracle teacher-forced."""
    mp = synth.arch.llm(tokens=512, **dict(SMALL, **FULL))
    dec = Decoder(prefill_tokens=512, budget_frac=0.5, weights=_weights_parallel(mp), **FULL)
    ids = synth.gen.model_input(dec.mp).reshape(-1)
    st = F.new_state()
    ref = F.forward(dec.mp, dec.w, ids.reshape(-1, 1, 1, 1), state=st)
    logits, toks = dec.run(0, ids)
    _check_step(logits, toks, ref[0].reshape(512, -1), ref[1].reshape(-1), CHAIN_TOL)
    tok = int(toks[-1])
    for step in range(2):
        ref = F.forward(dec.md, dec.w, np.array([tok], dtype=np.int32).reshape(1, 1, 1, 1), state=st)
        logits, toks = dec.run(1, np.array([tok], dtype=np.int32))
        _check_step(logits, toks, ref[0].reshape(1, -1), ref[1].reshape(-1), CHAIN_TOL)
        tok = int(toks[0])
    assert int(dec.state[:4].cpu().numpy().view(np.int32)[0]) == 512 + 2


def test_llm_long_prefill_many_heads():
    """128 queries x 8 heads: the prefill takes the tensor-core attention
    kernel, the decode steps after it the split-key cluster kernel."""
    dec = Decoder(prefill_tokens=128, **WIDE)
    ids = synth.gen.model_input(dec.mp).reshape(-1)
    st = F.new_state()
    ref = F.forward(dec.mp, dec.w, ids.reshape(-1, 1, 1, 1), state=st)
    logits, toks = dec.run(0, ids)
    _check_step(logits, toks, ref[0].reshape(128, -1), ref[1].reshape(-1), CHAIN_TOL)
    tok = int(toks[-1])
    for step in range(4):
        ref = F.forward(dec.md, dec.w, np.array([tok], dtype=np.int32).reshape(1, 1, 1, 1), state=st)
        logits, toks = dec.run(1, np.array([tok], dtype=np.int32))
        _check_step(logits, toks, ref[0].reshape(1, -1), ref[1].reshape(-1), CHAIN_TOL)
        tok = int(toks[0])


@pytest.mark.parametrize("prompt", [1, 17, 79])
def test_llm_short_and_ragged_prompts(prompt):
    """Prompt lengths at the edges of the small decoder (cache of 80): one
    token, so the prefill pass has the decode pass's shapes; 17, one row
    past a 16-row step; 79, one short of the cache, whose single decode
    step then fills it.  Teacher-forced against the oracle end to end at the
    chained bf16 bar (a single row's logits carry the rounding noise of
    every stored tensor before them, with no other rows to average it); the
    same passes are held layer by layer to 2e-3 in
    test_llm_every_layer_local_parity."""
    dec = Decoder(prefill_tokens=prompt, layers=1)
    ids = synth.gen.model_input(dec.mp).reshape(-1)
    st = F.new_state()
    ref = F.forward(dec.mp, dec.w, ids.reshape(-1, 1, 1, 1), state=st)
    logits, toks = dec.run(0, ids)
    _check_step(logits, toks, ref[0].reshape(prompt, -1), ref[1].reshape(-1), CHAIN_TOL)
    tok = int(toks[-1])
    steps = min(3, SMALL["max_seq"] - prompt)
    for _ in range(steps):
        ref = F.forward(dec.md, dec.w, np.array([tok], dtype=np.int32).reshape(1, 1, 1, 1), state=st)
        logits, toks = dec.run(1, np.array([tok], dtype=np.int32))
        _check_step(logits, toks, ref[0].reshape(1, -1), ref[1].reshape(-1), CHAIN_TOL)
        tok = int(toks[0])
    assert int(dec.state[:4].cpu().numpy().view(np.int32)[0]) == prompt + steps


@pytest.mark.parametrize("d,heads,chunk,max_seq", [
    (512, 4, 150, 400),    # tensor-core prefill: 2 query tiles (ragged), up to 3 key tiles, second chunk at pos 150
    (2560, 20, 60, 200),   # 60 queries x 20 heads: the SIMT warp-per-query kernel
])
def test_llm_prefill_in_chunks(d, heads, chunk, max_seq):
    """A prefill engine called twice in a row: the second call's queries
    start at the cache position the first left (pos0 > 0), so key tiles are
    not aligned with query tiles and the causal mask cuts tiles in the
    middle.  Both chunks and a decode step after them against the oracle
    (its state carried along), end to end at the decoder bar (the per-layer
    check of the same runs is test_llm_every_layer_local_parity)."""
    dec = Decoder(prefill_tokens=chunk, layers=1, d=d, heads=heads, max_seq=max_seq, ffn=688)
    st = F.new_state()
    tok = None
    for c in range(2):
        ids = synth.gen.model_input(dec.mp, request=c).reshape(-1)
        ref = F.forward(dec.mp, dec.w, ids.reshape(-1, 1, 1, 1), state=st)
        logits, toks = dec.run(0, ids)
        _check_step(logits, toks, ref[0].reshape(chunk, -1), ref[1].reshape(-1), CHAIN_TOL)
        tok = int(toks[-1])
    ref = F.forward(dec.md, dec.w, np.array([tok], dtype=np.int32).reshape(1, 1, 1, 1), state=st)
    logits, toks = dec.run(1, np.array([tok], dtype=np.int32))
    _check_step(logits, toks, ref[0].reshape(1, -1), ref[1].reshape(-1), CHAIN_TOL)
    assert int(dec.state[:4].cpu().numpy().view(np.int32)[0]) == 2 * chunk + 1


@pytest.mark.parametrize("cfg,passes", [
    (WIDE, (128, 1, 1)),                                               # tensor-core prefill, CTA decode
    (dict(layers=1, d=512, heads=4, ffn=688, max_seq=400), (150, 150, 1)),   # second prefill at pos0 150
    (dict(layers=1, d=2560, heads=20, ffn=688, max_seq=200), (60, 60, 1)),   # SIMT warp-per-query prefill
    (dict(layers=1, d=256, heads=2, ffn=688, max_seq=80), (1, 1, 1)),       # a one-token prompt at position 0
    (dict(layers=1, d=256, heads=2, ffn=688, max_seq=80), (17, 1)),         # one row past a 16-row step
    (dict(layers=1, d=256, heads=2, ffn=688, max_seq=80), (79, 1)),         # the decode step fills the cache
])
def test_llm_every_layer_local_parity(cfg, passes):
    """Each layer of a resident decoder whose every layer is a model output,
    against the oracle layer run on the GPU's own stored inputs, over
    consecutive passes of the given token counts (a second prefill starts at
    the position the first left), the oracle keeping its own KV cache built
    from the GPU's k and v.  The q projection is rotated in place by the
    attention layer, so attention takes the oracle's q computed from the
    GPU's normalised input."""
    import torch
    w = None
    st_or = F.new_state()
    state = None
    for pi, tokens in enumerate(passes):
        m = synth.arch.llm(tokens=tokens, vocab=SMALL["vocab"], **cfg)
        m = dict(m, outputs=list(range(len(m["layers"]))))
        if w is None:
            w = synth.gen.model_weights(m)
            host = capi.HostWeights(w)
        if tokens > 1 or pi == 0:
            x = synth.gen.model_input(m, request=pi)
        else:
            x = np.array([[[[next_tok]]]], dtype=np.int32)
        plan = capi.Plan.resident(capi.Desc(m))
        info = plan.info()
        eng = capi.Engine(plan, host)
        if state is None:
            state = torch.zeros(info["state_bytes"], dtype=torch.uint8, device="cuda")
        eng.bind_state(state.data_ptr(), info["state_bytes"])
        din = torch.zeros(max(16, info["input_bytes"]), dtype=torch.uint8, device="cuda")
        din[:x.nbytes].copy_(torch.from_numpy(x.view(np.uint8).reshape(-1)))
        dout = torch.zeros(info["output_bytes"], dtype=torch.uint8, device="cuda")
        eng.infer(din.data_ptr(), dout.data_ptr(), torch.cuda.current_stream().cuda_stream)
        eng.sync()
        hb = dout.cpu().numpy()
        shapes = OP.out_shapes(m)
        gpu = {}
        for li, off in enumerate(plan.output_offsets()):
            n = int(np.prod(shapes[li]))
            if m["layers"][li]["op"] == "argmax":
                gpu[li] = hb[off:off + 4 * n].view(np.int32).astype(np.float64).reshape(-1, 1, 1, 1)
            else:
                gpu[li] = F.decode(hb[off:off + 2 * n].view(np.uint16), "bf16").reshape(tokens, -1, 1, 1)
        local = {}
        for li, L in enumerate(m["layers"]):
            acts = gpu
            if L["op"] == "attention":
                acts = dict(gpu)
                acts[L["src"][0]] = local[L["src"][0]]
            local[li] = F.run_layer(L, "bf16", w[li], acts, np.asarray(x), st_or, li)
            att = [M for M in m["layers"] if M["op"] == "attention" and M["src"][0] == li]
            if att:   # the stored q was rotated in place: compare with the oracle's rotated q
                pos = np.arange(st_or["pos"], st_or["pos"] + tokens)
                qr = F.round_as(F.rope(local[li].reshape(tokens, -1), pos, att[0]["heads"], att[0]["theta"]), "bf16")
                e = rel_l2(gpu[li].ravel(), qr.ravel())
                assert e <= LOCAL_TOL, (tokens, li, "rotated q", e)
                continue
            if L["op"] == "argmax":   # the GPU's logits decide: exact, ties to the lowest index
                assert np.array_equal(gpu[li].ravel(), local[li].ravel()), li
                continue
            e = rel_l2(gpu[li].ravel(), local[li].ravel())
            assert e <= LOCAL_TOL, (tokens, li, L["op"], e)
        st_or["pos"] += tokens
        next_tok = int(gpu[len(m["layers"]) - 1].ravel()[-1])


def test_llm_swapped_equals_resident():
    sw = Decoder(prefill_tokens=32, budget_frac=0.4)
    rs = Decoder(prefill_tokens=32, resident=True, host=sw.host, weights=sw.w)
    assert sw.engines[0][2]["n_blocks"] > 1
    ids = synth.gen.model_input(sw.mp).reshape(-1)
    a, b = sw.run(0, ids), rs.run(0, ids)
    assert a[0].tobytes() == b[0].tobytes() and a[1].tobytes() == b[1].tobytes()
    tok = np.array([a[1][-1]], dtype=np.int32)
    for _ in range(4):
        a, b = sw.run(1, tok), rs.run(1, tok)
        assert a[0].tobytes() == b[0].tobytes()
        tok = np.array([a[1][0]], dtype=np.int32)


def test_llm_resident_prefix_equals_resident():
    """Decoder engines whose first units stay resident between passes."""
    import torch
    sw = Decoder(prefill_tokens=32, budget_frac=0.5)
    rs = Decoder(prefill_tokens=32, resident=True, host=sw.host, weights=sw.w)
    # rebuild the swapped engines with resident_prefix plans sharing sw's state
    for i, m in enumerate((sw.mp, sw.md)):
        budget = int(OP.weight_bytes(sw.mp) * 0.5) // 256 * 256
        plan = capi.Plan.partition(capi.Desc(m), budget, capi.options(resident_prefix=1))
        assert plan.info()["prefix_units"] > 0
        eng = capi.Engine(plan, sw.host)
        eng.bind_state(sw.state.data_ptr(), sw.state_bytes)
        info = plan.info()
        din = torch.zeros(max(16, info["input_bytes"]), dtype=torch.uint8, device="cuda")
        dout = torch.zeros(info["output_bytes"], dtype=torch.uint8, device="cuda")
        sw.engines[i] = (plan, eng, info)
        sw.bufs[i] = (din, dout, plan.output_offsets())
    ids = synth.gen.model_input(sw.mp).reshape(-1)
    a, b = sw.run(0, ids), rs.run(0, ids)
    assert a[0].tobytes() == b[0].tobytes() and a[1].tobytes() == b[1].tobytes()
    tok = np.array([a[1][-1]], dtype=np.int32)
    for _ in range(4):
        a, b = sw.run(1, tok), rs.run(1, tok)
        assert a[0].tobytes() == b[0].tobytes()
        tok = np.array([a[1][0]], dtype=np.int32)


def test_llm_cache_bound_reported_not_faulted():
    dec = Decoder(prefill_tokens=64)
    ids = synth.gen.model_input(dec.mp).reshape(-1)
    dec.run(0, ids)                            # positions 0..63 of 80
    plan, eng, info = dec.engines[0]
    din, dout, _ = dec.bufs[0]
    eng.infer(din.data_ptr(), dout.data_ptr(), dec.torch.cuda.current_stream().cuda_stream)   # would need 128
    with pytest.raises(capi.SwapnetError) as ei:
        eng.sync()
    assert ei.value.code == capi.ERR_INVALID_ARG


@pytest.mark.parametrize("vocab", [1000, 1003])
def test_argmax_ties_go_to_the_lowest_index(vocab):
    """A head whose second half of features repeats the first half gives
    every logit a twin: the argmax is the first of the two (and an all-zero
    head makes every logit equal: index 0).  1000 features take the
    16-byte-chunk scan, 1003 the element scan."""
    import torch
    m = synth.arch.llm(layers=0, d=256, heads=2, ffn=688, vocab=vocab, tokens=4, max_seq=16)
    w = synth.gen.model_weights(m)
    head = len(m["layers"]) - 2
    half = vocab // 2
    W = w[head][0]
    W[half:2 * half] = W[:half]
    x = synth.gen.model_input(m)
    for zero in (False, True):
        if zero:
            W[:] = 0
        plan = capi.Plan.resident(capi.Desc(m))
        info = plan.info()
        eng = capi.Engine(plan, capi.HostWeights(w))
        din = torch.zeros(max(16, info["input_bytes"]), dtype=torch.uint8, device="cuda")
        din[:x.nbytes].copy_(torch.from_numpy(x.view(np.uint8).reshape(-1)))
        dout = torch.zeros(info["output_bytes"], dtype=torch.uint8, device="cuda")
        eng.infer(din.data_ptr(), dout.data_ptr(), torch.cuda.current_stream().cuda_stream)
        eng.sync()
        hb = dout.cpu().numpy()
        offs = plan.output_offsets()
        logits = F.decode(hb[offs[0]:offs[0] + 4 * vocab * 2].view(np.uint16), "bf16").reshape(4, vocab)
        tok = hb[offs[1]:offs[1] + 16].view(np.int32)
        for t in range(4):
            assert tok[t] == int(np.argmax(logits[t])), (zero, t)
            assert tok[t] == 0 if zero else tok[t] < half or tok[t] == 2 * half
            if not zero and tok[t] < half:
                assert logits[t, tok[t]] == logits[t, tok[t] + half]


@pytest.mark.parametrize("resident", [True, False])
def test_merged_gemv_launches_equal_separate_launches(resident):
    """The decode pass launches q, k, v as one GEMV and gate, up as one
    paired GEMV (option merge, the default): bit-identical to one launch per
    layer, three launches fewer per decoder layer when the members share a
    block."""
    mg = Decoder(prefill_tokens=32, budget_frac=0.4, resident=resident)
    sp = Decoder(prefill_tokens=32, budget_frac=0.4, resident=resident, host=mg.host, weights=mg.w,
                 opts=dict(merge=0))
    ids = synth.gen.model_input(mg.mp).reshape(-1)
    a, b = mg.run(0, ids), sp.run(0, ids)
    assert a[0].tobytes() == b[0].tobytes() and a[1].tobytes() == b[1].tobytes()
    tok = np.array([a[1][-1]], dtype=np.int32)
    l0 = [d.engines[1][1].stats()["kernel_launches"] for d in (mg, sp)]
    for _ in range(4):
        a, b = mg.run(1, tok), sp.run(1, tok)
        assert a[0].tobytes() == b[0].tobytes() and a[1].tobytes() == b[1].tobytes()
        tok = np.array([a[1][0]], dtype=np.int32)
    per = [(d.engines[1][1].stats()["kernel_launches"] - x) // 4 for d, x in zip((mg, sp), l0)]
    if resident:
        assert per[1] - per[0] == 3 * SMALL["layers"]
    else:
        assert 0 <= per[1] - per[0] <= 3 * SMALL["layers"]


def test_llm_decode_to_the_end_of_the_cache_then_refused():
    """Greedy decode passes until the KV cache is full: the last pass
    attends over all max_seq positions, so the decode attention's last key
    chunk ends exactly at the end of the cache; every pass against the
    oracle (which consumes the GPU's token).  One pass more finds no place
    in the cache: the device reports the position as out of range and
    swapnet_engine_sync returns INVALID_ARG."""
    max_seq = 40
    dec = Decoder(prefill_tokens=32, layers=1, max_seq=max_seq)
    ids = synth.gen.model_input(dec.mp).reshape(-1)
    st = F.new_state()
    ref = F.forward(dec.mp, dec.w, ids.reshape(-1, 1, 1, 1), state=st)
    logits, toks = dec.run(0, ids)
    _check_step(logits, toks, ref[0].reshape(32, -1), ref[1].reshape(-1), TOL[1])
    tok = int(toks[-1])
    for step in range(max_seq - 32):
        ref = F.forward(dec.md, dec.w, np.array([tok], dtype=np.int32).reshape(1, 1, 1, 1), state=st)
        logits, toks = dec.run(1, np.array([tok], dtype=np.int32))
        _check_step(logits, toks, ref[0].reshape(1, -1), ref[1].reshape(-1), TOL[1])
        tok = int(toks[0])
    assert int(dec.state[:4].cpu().numpy().view(np.int32)[0]) == max_seq
    with pytest.raises(capi.SwapnetError) as ei:
        dec.run(1, np.array([tok], dtype=np.int32))
    assert ei.value.code == capi.ERR_INVALID_ARG


@pytest.mark.parametrize("prefix", [0, 1])
def test_llm_packed_swaps_equal_resident(prefix):
    """The packed swap variant (an extension: the bf16 tensors packed
    losslessly at load and unpacked into the arena by an SM kernel), alone
    and with a resident prefix: a prefill and decode steps equal the
    resident run bit for bit and the oracle at the decoder bar, the blocks
    that hold packable tensors take the unpack kernel, and fewer bytes cross
    the host link than are swapped."""
    sw = Decoder(prefill_tokens=32, budget_frac=0.6 if prefix else 0.4,
                 opts=dict(swap_variant=capi.SWAP_PACKED, resident_prefix=prefix))
    if prefix:
        assert all(info["prefix_units"] > 0 for _, _, info in sw.engines)
    rs = Decoder(prefill_tokens=32, resident=True, host=sw.host, weights=sw.w)
    for _, eng, info in sw.engines:
        assert info["n_blocks"] > 1
        assert any(b["variant"] == capi.SWAP_PACKED for b in eng.blocks())
    ids = synth.gen.model_input(sw.mp).reshape(-1)
    st = F.new_state()
    ref = F.forward(sw.mp, sw.w, ids.reshape(-1, 1, 1, 1), state=st)
    a, b = sw.run(0, ids), rs.run(0, ids)
    assert a[0].tobytes() == b[0].tobytes() and a[1].tobytes() == b[1].tobytes()
    _check_step(a[0], a[1], ref[0].reshape(32, -1), ref[1].reshape(-1), CHAIN_TOL)
    tok = np.array([a[1][-1]], dtype=np.int32)
    for _ in range(4):
        a, b = sw.run(1, tok), rs.run(1, tok)
        assert a[0].tobytes() == b[0].tobytes() and a[1].tobytes() == b[1].tobytes()
        tok = np.array([a[1][0]], dtype=np.int32)
    for _, eng, _ in sw.engines:
        s = eng.stats()
        assert 0 < s["link_bytes"] < 0.85 * s["bytes_swapped"], s


def test_packed_variant_falls_back_for_other_types():
    """An fp16 CNN under the packed variant: nothing packs, every block takes
    the zero-copy kernel, and the result is the resident one bit for bit."""
    import torch
    from helpers import Runner
    m = synth.arch.MODELS["resnet50"]()
    w = synth.gen.model_weights(m)
    d = capi.Desc(m)
    host = capi.HostWeights(w)
    plan = capi.Plan.partition(d, int(OP.weight_bytes(m) * 0.4) // 256 * 256,
                               capi.options(swap_variant=capi.SWAP_PACKED))
    sw = Runner(m, w, plan, host)
    assert all(b["variant"] == capi.SWAP_ZEROCOPY for b in sw.engine.blocks())
    x = synth.gen.model_input(m)
    assert sw.run(x)[0].tobytes() == Runner(m, w, capi.Plan.resident(d), host).run(x)[0].tobytes()
    s = sw.engine.stats()
    assert s["link_bytes"] == s["bytes_swapped"] or s["link_bytes"] >= 0.99 * s["bytes_swapped"]
    torch.cuda.synchronize()


def test_packed_engine_adapts_between_budgets():
    """A packed-swap decoder engine switched between two budgets with
    swapnet_engine_adapt keeps its packed images (no new packing) and equals
    the resident run bit for bit under both plans."""
    sw = Decoder(prefill_tokens=16, budget_frac=0.7, layers=2, opts=dict(swap_variant=capi.SWAP_PACKED))
    rs = Decoder(prefill_tokens=16, resident=True, host=sw.host, weights=sw.w, layers=2)
    ids = synth.gen.model_input(sw.mp).reshape(-1)
    base = rs.run(0, ids)
    a = sw.run(0, ids)
    assert a[0].tobytes() == base[0].tobytes()
    plan, eng, info = sw.engines[0]
    small = capi.Plan.partition(capi.Desc(sw.mp), int(OP.weight_bytes(sw.mp) * 0.35) // 256 * 256,
                                capi.options(swap_variant=capi.SWAP_PACKED))
    assert small.info()["n_blocks"] > info["n_blocks"]
    eng.adapt(small)
    sw.engines[0] = (small, eng, small.info())
    sw.bufs[0] = (sw.bufs[0][0], sw.bufs[0][1], small.output_offsets())
    assert any(b["variant"] == capi.SWAP_PACKED for b in eng.blocks())
    rs.state.zero_()
    sw.state.zero_()
    b = sw.run(0, ids)
    c = rs.run(0, ids)
    assert b[0].tobytes() == c[0].tobytes() == base[0].tobytes()
