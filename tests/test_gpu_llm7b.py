"""Parity of the whole LLaMA-7B-shaped decoder (32 layers, d 4096, 32 heads,
FFN 11008, vocabulary 32000) in the launch configuration the benchmark
times: weights in page-locked host memory, swapped through a 4e9-byte arena,
a 512-token prefill and two greedy decode passes.

Every layer of the GPU run is a model output, and the oracle takes the model
one decoder layer at a time (layer-streamed: one layer's parameters decoded
to float64, used, dropped), so the float64 model never has to sit in host
memory at once.  Two comparisons:

  local  every layer's output against the oracle's layer run on the GPU's
         own stored inputs (prefill and both decode passes), held to the
         fp16/bf16 bar of relative L2 2e-3 per output tensor;
  chain  the oracle's own forward pass of the prefill through all 32 layers
         against the GPU's residual stream after every decoder block and its
         logits, beside a second oracle chain whose every stored tensor has
         0.5 % of its elements moved by one bf16 ulp: rounding differences
         of that size grow with depth in this random-init model, and the GPU
         must drift from the oracle no farther than the flipped oracle does.
"""
import concurrent.futures as cf
import time

import numpy as np
import pytest

import synth
from oracle import forward as F
from paper_2401_16757_gb300 import capi
from helpers import rel_l2

pytestmark = pytest.mark.gpu

LOCAL_TOL = 2e-3
BUDGET = 4_000_000_000


def _packed_weights(model, threads=16):
    """The 7B parameters generated in parallel into one page-locked packed
    buffer; returns it and per-layer lists of storage views into it."""
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
    w = [[] for _ in model["layers"]]
    for k, (li, ti, shp) in enumerate(jobs):
        w[li].append(host.view(k).view(np.uint16).reshape(shp))
    return host, w


def _flip_ulps(x, rng, frac):
    """x (bf16 values held as float64) with a random `frac` of its nonzero
    elements moved to a neighbouring bf16 value (one step of the bit pattern
    up or down)."""
    flat = x.reshape(-1).copy()
    idx = np.nonzero(rng.random(flat.size) < frac)[0]
    idx = idx[flat[idx] != 0]
    bits = synth.gen.round_to_storage(flat[idx], "bf16").astype(np.int32)
    bits += rng.choice(np.array([-1, 1], dtype=np.int32), size=idx.size)
    flat[idx] = F.decode(bits.astype(np.uint16), "bf16")
    return flat.reshape(x.shape)


def _gpu_layers(model, plan, hb, tokens):
    """Per-layer outputs of one pass read from the host copy of the output
    buffer: float64 NCHW-shaped arrays ([tokens, width, 1, 1]); argmax rows
    as float64 indices."""
    out = {}
    for li, off in enumerate(plan.output_offsets()):
        L = model["layers"][li]
        if L["op"] == "argmax":
            out[li] = hb[off:off + 4 * tokens].view(np.int32).astype(np.float64).reshape(-1, 1, 1, 1)
            continue
        width = {"embed": L.get("d"), "rmsnorm": L.get("d"), "linear": L.get("n")}.get(L["op"])
        if L["op"] == "attention":
            width = model["layers"][L["src"][0]]["n"]
        n = tokens * width
        out[li] = F.decode(hb[off:off + 2 * n].view(np.uint16), "bf16").reshape(tokens, width, 1, 1)
    return out


def test_llm_7b_all_layers_local_parity_and_chained_prefill():
    import torch
    t_start = time.perf_counter()
    mp, md = synth.arch.llm(tokens=512), synth.arch.llm(tokens=1)
    n_layers = len(mp["layers"])
    every = list(range(n_layers))
    mp, md = dict(mp, outputs=every), dict(md, outputs=every)
    host, w = _packed_weights(mp)
    opt = capi.options()
    plans = [capi.Plan.partition(capi.Desc(m), BUDGET, opt) for m in (mp, md)]
    assert plans[0].info()["n_blocks"] > 3 and plans[1].info()["n_blocks"] > 3
    engines = [capi.Engine(p, host) for p in plans]
    state = torch.zeros(plans[0].info()["state_bytes"], dtype=torch.uint8, device="cuda")
    for e in engines:
        e.bind_state(state.data_ptr(), state.numel())
    stream = torch.cuda.current_stream().cuda_stream

    # ---- GPU: prefill of the bench's 512 ids, then two greedy decode passes
    ids = synth.gen.model_input(mp).reshape(-1)
    passes = []   # (token ids, position, per-layer GPU outputs)
    feed, pos = ids, 0
    for which in (0, 1, 1):
        info = plans[which].info()
        din = torch.zeros(max(16, info["input_bytes"]), dtype=torch.uint8, device="cuda")
        din[:feed.nbytes].copy_(torch.from_numpy(np.ascontiguousarray(feed, dtype=np.int32).view(np.uint8)))
        dout = torch.zeros(info["output_bytes"], dtype=torch.uint8, device="cuda")
        engines[which].infer(din.data_ptr(), dout.data_ptr(), stream)
        engines[which].sync()
        hb = dout.cpu().numpy()
        gpu = _gpu_layers(mp, plans[which], hb, feed.size)
        passes.append((np.asarray(feed, dtype=np.int32).reshape(-1, 1, 1, 1), pos, gpu))
        pos += feed.size
        feed = np.array([int(gpu[n_layers - 1].ravel()[-1])], dtype=np.int32)
        del hb, dout
    assert int(state[:4].cpu().numpy().view(np.int32)[0]) == 512 + 2
    for e in engines:
        e.free()
    t_gpu = time.perf_counter() - t_start

    # ---- oracle, one layer at a time
    gpu0_all = passes[0][2]
    st_local, st_chain, st_pert = F.new_state(), F.new_state(), F.new_state()
    chain, pert = {}, {}
    worst = {}
    growth = []     # (layer, GPU vs chain, perturbed chain vs chain) at each decoder layer's output
    rng = np.random.default_rng(12345)
    for li, L in enumerate(mp["layers"]):
        params = F.decode_params(w[li], "bf16") if w[li] else None
        att = [M for M in mp["layers"] if M["op"] == "attention" and M["src"][0] == li]
        for p_i, (x, pos0, gpu) in enumerate(passes):
            tokens = x.shape[0]
            acts = gpu
            if L["op"] == "attention":   # q was rotated in place on the GPU: take the oracle's q
                acts = dict(gpu)
                acts[L["src"][0]] = gpu["_q_local"]
            st_local["pos"] = pos0
            local = F.run_layer(L, "bf16", w[li], acts, x, st_local, li, params=params)
            if att:                      # the stored q is the rotated one
                gpu["_q_local"] = local
                qr = F.round_as(F.rope(local.reshape(tokens, -1), np.arange(pos0, pos0 + tokens),
                                       att[0]["heads"], att[0]["theta"]), "bf16")
                e = rel_l2(gpu[li].ravel(), qr.ravel())
            elif L["op"] == "argmax":    # decided by the GPU's logits: exact, ties to the lowest index
                assert np.array_equal(gpu[li].ravel(), local.ravel()), (li, p_i)
                e = 0.0
            else:
                e = rel_l2(gpu[li].ravel(), local.ravel())
            worst[(L["op"], p_i)] = max(worst.get((L["op"], p_i), 0.0), e)
            assert e <= LOCAL_TOL, (p_i, li, L["op"], e)
        # the oracle's own chain through the prefill, and a second chain whose
        # every stored tensor has 0.5 % of its elements moved by one bf16 ulp
        # (the size of the rounding flips a different summation order causes):
        # how far the model itself carries such flips to its logits
        x0 = passes[0][0]
        st_chain["pos"] = st_pert["pos"] = 0
        chain[li] = F.run_layer(L, "bf16", w[li], chain, x0, st_chain, li, params=params)
        pert[li] = F.run_layer(L, "bf16", w[li], pert, x0, st_pert, li, params=params)
        if L["op"] in ("rmsnorm", "linear", "attention"):
            pert[li] = _flip_ulps(pert[li], rng, 0.005)
        if L["op"] == "linear" and L.get("res") is not None and L.get("act", "none") == "none" \
                and mp["layers"][L["res"]]["op"] == "linear":   # a decoder layer's last output
            growth.append((li, rel_l2(gpu0_all[li].ravel(), chain[li].ravel()),
                           rel_l2(pert[li].ravel(), chain[li].ravel())))
        for d in (chain, pert):
            for dead in [j for j in d if j < li - 12 and j not in (n_layers - 2, n_layers - 1)]:
                del d[dead]             # nothing reads that far back (residual stream: <= 11 layers)
        del params
    gpu0 = passes[0][2]
    head = n_layers - 2
    e_chain = rel_l2(gpu0[head].ravel(), chain[head].ravel())
    tok_gpu = gpu0[n_layers - 1].ravel().astype(np.int64)
    tok_chain = chain[n_layers - 1].ravel().astype(np.int64)
    agree = float(np.mean(tok_gpu == tok_chain))
    e_self = rel_l2(pert[head].ravel(), chain[head].ravel())
    agree_self = float(np.mean(pert[n_layers - 1].ravel() == chain[n_layers - 1].ravel()))
    print("7B parity: worst local rel-L2 per op/pass %s; chained prefill logits rel-L2 %.3e (oracle with "
          "one-ulp flips: %.3e), greedy tokens agreeing %.4f (%.4f); GPU part %.1f s, total %.1f s" %
          ({"%s/%d" % k: float("%.2e" % v) for k, v in sorted(worst.items())}, e_chain, e_self, agree,
           agree_self, t_gpu, time.perf_counter() - t_start))
    print("divergence from the oracle's chain after each decoder layer (GPU, flipped oracle): " +
          " ".join("%d:%.1e/%.1e" % g for g in growth))
    # Chained through 32 random-init layers, any bf16 rounding difference
    # grows steadily with depth (measured: 4.8e-3 after the first attention
    # block to 4.5e-2 at the logits); the oracle itself, with 0.5 % of every
    # stored tensor's elements moved by one ulp, drifts farther from its own
    # chain.  The bar: after every decoder block, and at the logits, the GPU
    # stays within the flipped oracle's drift (25 % margin), and its greedy
    # tokens agree with the chain's at least as often, less 5 points.
    for li_, g, f in growth:
        assert g <= 1.25 * f, (li_, g, f)
    assert e_chain <= 1.25 * e_self, (e_chain, e_self)
    assert agree >= agree_self - 0.05, (agree, agree_self)
