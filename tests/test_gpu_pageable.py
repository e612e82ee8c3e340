"""Pageable host weights (option pageable, the counterpart of the paper's
w/o-uni-add ablation): the host tensors are never page-locked and every
swap-in is a copy the driver stages through its own page-locked buffer.
The arena receives the same bytes, so the outputs equal the resident run's
bit for bit (and the oracle's within the fp16 bar); the options that need
page-locked memory are refused."""
import pytest

from oracle import plan as OP
import synth
from paper_2401_16757_gb300 import capi
from helpers import Runner, check_oracle

pytestmark = pytest.mark.gpu


def test_pageable_swaps_equal_resident():
    m = synth.arch.resnet50(batch=1)
    w = synth.gen.model_weights(m)
    x = synth.gen.model_input(m)
    d = capi.Desc(m)
    budget = int(OP.weight_bytes(m) * 0.4) // 256 * 256
    ref = Runner(m, w, capi.Plan.resident(d), capi.HostWeights(w)).run(x)
    pg = Runner(m, w, capi.Plan.partition(d, budget, capi.options(pageable=1)), capi.HostWeights(w))
    assert pg.info["n_blocks"] > 2
    assert all(b["variant"] == capi.SWAP_MEMCPY for b in pg.engine.blocks())
    for _ in range(3):
        got = pg.run(x)
        assert all(a.tobytes() == b.tobytes() for a, b in zip(got, ref))
    check_oracle(pg, got, x)
    # a page-locked plan cannot be switched to on this engine
    with pytest.raises(capi.SwapnetError) as ei:
        pg.engine.adapt(capi.Plan.partition(d, budget, capi.options()))
    assert ei.value.code == capi.ERR_INVALID_ARG
    pg.engine.adapt(capi.Plan.partition(d, int(OP.weight_bytes(m) * 0.6) // 256 * 256, capi.options(pageable=1)))
    assert all(a.tobytes() == b.tobytes() for a, b in zip(pg.run(x), ref))


def test_pageable_refuses_host_read_tables():
    m = synth.arch.llm(layers=1, d=256, heads=2, ffn=688, vocab=1000, tokens=1, max_seq=16)
    d = capi.Desc(m)
    plan = capi.Plan.partition(d, OP.weight_bytes(m) // 256 * 256, capi.options(pageable=1))
    with pytest.raises(capi.SwapnetError) as ei:
        capi.Engine(plan, capi.HostWeights(synth.gen.model_weights(m)))
    assert ei.value.code == capi.ERR_UNSUPPORTED
