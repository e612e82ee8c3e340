"""Blocks read in place in host memory (SWAPNET_SWAP_DIRECT, the copy-free
dispatch of Sec. 4.2.2 carried into the kernels): blocks whose kernels are
all SIMT kernels skip the swap-in and read their parameters through the
device alias of the page-locked host tensors; tensor-core blocks keep the
copy.  Every output is bit-identical to the all-resident run, since the
kernels and their reduction order are the same and only the address of the
parameters differs."""
import numpy as np
import pytest

from oracle import plan as OP
import synth
from paper_2401_16757_gb300 import capi
from helpers import Runner, check_close, oracle_outputs
from test_gpu_llm import Decoder

pytestmark = pytest.mark.gpu


def _budget(m, frac):
    return int(OP.weight_bytes(m) * frac) // 256 * 256


def _pair(m, frac, **opt):
    w = synth.gen.model_weights(m)
    x = synth.gen.model_input(m)
    d = capi.Desc(m)
    host = capi.HostWeights(w)
    sw = Runner(m, w, capi.Plan.partition(d, _budget(m, frac), capi.options(swap_variant=capi.SWAP_DIRECT, **opt)),
                host)
    rs = Runner(m, w, capi.Plan.resident(d), host)
    return w, x, d, host, sw, rs


def test_mlp_reads_every_block_in_place():
    """The 6-layer fp32 MLP runs tiled SIMT GEMMs only: every swapped block
    is read in place, no byte is copied, the arena is never written."""
    m = synth.arch.mlp6(batch=8)
    w, x, d, host, sw, rs = _pair(m, 0.4)
    blocks = sw.engine.blocks()
    assert len(blocks) > 2
    assert all(b["variant"] == capi.SWAP_DIRECT for b in blocks)
    ref = rs.run(x)
    before = sw.engine.stats()
    for _ in range(3):
        got = sw.run(x)
        assert all(a.tobytes() == b.tobytes() for a, b in zip(got, ref))
    after = sw.engine.stats()
    assert after["bytes_swapped"] == before["bytes_swapped"] == 0
    assert after["memcpy_calls"] == 0 and after["infer_calls"] == before["infer_calls"] + 3
    check_close(m, sw.decode(got), oracle_outputs(m, w, x))


def test_mixed_blocks_vgg16():
    """VGG-16 at batch 1 under a quarter of its weights: the convolution
    blocks (tensor cores) are copied by the zero-copy kernel (so SM loads
    and copy-engine reads of the host weights are not mixed), the fully
    connected pieces (GEMV) are
    read in place; the swapped byte count is exactly that of the copied
    blocks."""
    m = synth.arch.vgg16(batch=1)
    w, x, d, host, sw, rs = _pair(m, 0.25)
    blocks = sw.engine.blocks()
    plan_blocks = sw.plan.blocks()
    kinds = sw.engine.unit_kernels()
    direct = [k for k, b in enumerate(blocks) if b["variant"] == capi.SWAP_DIRECT]
    copied = [k for k, b in enumerate(blocks) if b["variant"] == capi.SWAP_ZEROCOPY]
    assert direct and copied and len(direct) + len(copied) == len(blocks)
    for k in direct:
        pb = plan_blocks[k]
        assert all(kinds[u] not in ("tc_gemm", "tc_conv", "tc_conv_small") for u in range(pb["unit0"], pb["unit1"]))
    ref = rs.run(x)
    s0 = sw.engine.stats()["bytes_swapped"]
    got = sw.run(x)
    assert all(a.tobytes() == b.tobytes() for a, b in zip(got, ref))
    moved = sw.engine.stats()["bytes_swapped"] - s0
    assert 0 < moved < OP.weight_bytes(m) * 0.6
    check_close(m, sw.decode(got), oracle_outputs(m, w, x))


def test_profiling_and_prefetch_with_direct_blocks():
    """Per-unit and per-swap times and the timeline work with blocks that
    have no swap (their swap entries are 0); first-block prefetch is off
    when the first block is read in place."""
    m = synth.arch.mlp6(batch=8)
    w, x, d, host, sw, rs = _pair(m, 0.4, prefetch=1)
    ref = rs.run(x)
    sw.engine.set_profiling(True)
    got = sw.run(x)
    assert all(a.tobytes() == b.tobytes() for a, b in zip(got, ref))
    nu, nb = sw.info["n_units"], sw.info["n_blocks"]
    unit_us, swap_us = sw.engine.last_times(nu, nb)
    assert all(t > 0 for t in unit_us) and all(t == 0 for t in swap_us)
    s0, s1, b0, b1 = sw.engine.last_timeline(nu, nb)
    assert all(a <= b for a, b in zip(s0, s1)) and s0[0] >= 0
    sw.engine.set_profiling(False)
    for _ in range(2):
        assert all(a.tobytes() == b.tobytes() for a, b in zip(sw.run(x), ref))


def test_adapt_between_direct_and_copied_plans():
    m = synth.arch.vgg16(batch=1)
    w, x, d, host, sw, rs = _pair(m, 0.25)
    ref = rs.run(x)
    for frac, v in ((0.5, capi.SWAP_MEMCPY), (0.3, capi.SWAP_DIRECT), (0.6, capi.SWAP_AUTO)):
        sw.engine.adapt(capi.Plan.partition(d, _budget(m, frac), capi.options(swap_variant=v)))
        assert all(a.tobytes() == b.tobytes() for a, b in zip(sw.run(x), ref)), (frac, v)


def test_decoder_decode_pass_reads_in_place():
    """The LLM-shaped decoder: the prefill engine (tensor-core GEMMs) copies
    its blocks with the zero-copy kernel, the decode engine (GEMV, norms, attention) reads every block
    in place; prefill and four greedy decode passes equal the resident run
    bit for bit."""
    sw = Decoder(prefill_tokens=32, budget_frac=0.4, opts=dict(swap_variant=capi.SWAP_DIRECT))
    rs = Decoder(prefill_tokens=32, resident=True, host=sw.host, weights=sw.w)
    pre = sw.engines[0][1].blocks()
    dec = sw.engines[1][1].blocks()
    assert len(dec) > 1 and all(b["variant"] == capi.SWAP_DIRECT for b in dec)
    assert any(b["variant"] == capi.SWAP_ZEROCOPY for b in pre)
    ids = synth.gen.model_input(sw.mp).reshape(-1)
    a, b = sw.run(0, ids), rs.run(0, ids)
    assert a[0].tobytes() == b[0].tobytes() and a[1].tobytes() == b[1].tobytes()
    tok = np.array([a[1][-1]], dtype=np.int32)
    for _ in range(4):
        a, b = sw.run(1, tok), rs.run(1, tok)
        assert a[0].tobytes() == b[0].tobytes() and a[1].tobytes() == b[1].tobytes()
        tok = np.array([a[1][0]], dtype=np.int32)


def test_file_engine_ignores_direct(tmp_path):
    """Blocks read from a weights file have no host copy to read in place:
    a file engine copies every block whatever the variant asked for."""
    m = synth.arch.mlp6(batch=8)
    w = synth.gen.model_weights(m)
    x = synth.gen.model_input(m)
    d = capi.Desc(m)
    host = capi.HostWeights(w)
    path = str(tmp_path / "mlp6.swnw")
    capi.WeightsFile.write(path, d, host)
    wf = capi.WeightsFile(path, allow_buffered=True)
    rs = Runner(m, w, capi.Plan.resident(d), host).run(x)
    fr = Runner(m, w, capi.Plan.partition(d, _budget(m, 0.4), capi.options(swap_variant=capi.SWAP_DIRECT)), wf)
    assert all(b["variant"] == capi.SWAP_MEMCPY for b in fr.engine.blocks())
    assert all(a.tobytes() == b.tobytes() for a, b in zip(fr.run(x), rs))
