"""Storage tier on the GPU (Sec. 4.2.1 direct block fetch): engines whose
blocks are read from a weights file for every inference give the same bytes
as the all-resident run from host memory, and a read that fails inside an
inference is reported by swapnet_engine_sync."""
import os

import numpy as np
import pytest

from oracle import plan as OP
import synth
from paper_2401_16757_gb300 import capi
from helpers import Runner, check_close, check_oracle, oracle_outputs

pytestmark = pytest.mark.gpu


def _setup(name, kw, frac, tmp_path):
    m = synth.arch.MODELS[name](**kw)
    w = synth.gen.model_weights(m)
    x = synth.gen.model_input(m)
    d = capi.Desc(m)
    host = capi.HostWeights(w)
    path = str(tmp_path / (name + ".swnw"))
    capi.WeightsFile.write(path, d, host)
    wf = capi.WeightsFile(path, allow_buffered=True)
    budget = int(OP.weight_bytes(m) * frac) // 256 * 256
    return m, w, x, d, host, wf, budget, path


@pytest.mark.parametrize("name,kw,frac", [("resnet50", dict(batch=1), 0.40), ("vgg16", dict(batch=1), 0.25)])
def test_swapped_from_file_equals_resident(name, kw, frac, tmp_path):
    m, w, x, d, host, wf, budget, _ = _setup(name, kw, frac, tmp_path)
    rs = Runner(m, w, capi.Plan.resident(d), host).run(x)
    plan = capi.Plan.partition(d, budget, capi.options())
    assert plan.info()["n_blocks"] > 2
    fr = Runner(m, w, plan, wf)
    assert all(b["variant"] == capi.SWAP_MEMCPY for b in fr.engine.blocks())
    assert all(b["memcpy_us"] > 0 for b, pb in zip(fr.engine.blocks(), plan.blocks()) if pb["slot"] != 0xFFFFFFFF)
    for rep in range(3):  # every inference reads every block again
        got = fr.run(x)
        for a, b in zip(got, rs):
            assert a.tobytes() == b.tobytes(), "file-backed swapped run differs from the resident run"
    check_close(m, fr.decode(got), oracle_outputs(m, w, x))


def test_first_block_prefetch_from_file(tmp_path):
    m, w, x, d, host, wf, budget, _ = _setup("resnet50", dict(batch=1), 0.40, tmp_path)
    rs = Runner(m, w, capi.Plan.resident(d), host).run(x)
    fr = Runner(m, w, capi.Plan.partition(d, budget, capi.options(prefetch=1)), wf)
    for rep in range(3):
        got = fr.run(x)
        assert all(a.tobytes() == b.tobytes() for a, b in zip(got, rs)), rep
    check_oracle(fr, got, x)


def test_resident_prefix_from_file(tmp_path):
    """A resident-prefix plan (an extension) from a weights file: the
    prefix is read once at load, the rest for every inference."""
    m, w, x, d, host, wf, budget, _ = _setup("resnet50", dict(batch=1), 0.40, tmp_path)
    rs = Runner(m, w, capi.Plan.resident(d), host).run(x)
    plan = capi.Plan.partition(d, budget, capi.options(resident_prefix=1))
    assert plan.info()["prefix_units"] > 0
    fr = Runner(m, w, plan, wf)
    for rep in range(3):
        got = fr.run(x)
        assert all(a.tobytes() == b.tobytes() for a, b in zip(got, rs)), rep
    check_oracle(fr, got, x)


def test_resident_plan_and_adaptation_from_file(tmp_path):
    m, w, x, d, host, wf, budget, _ = _setup("resnet50", dict(batch=1), 0.40, tmp_path)
    ref = Runner(m, w, capi.Plan.resident(d), host).run(x)
    got = Runner(m, w, capi.Plan.resident(d), wf).run(x)
    assert all(a.tobytes() == b.tobytes() for a, b in zip(got, ref))
    r = Runner(m, w, capi.Plan.partition(d, budget, capi.options()), wf)
    for frac in (0.25, 0.6):
        r.engine.adapt(capi.Plan.partition(d, int(OP.weight_bytes(m) * frac) // 256 * 256, capi.options()))
        got = r.run(x)
        assert all(a.tobytes() == b.tobytes() for a, b in zip(got, ref))
        check_oracle(r, got, x)


def test_read_failure_inside_an_inference_is_reported(tmp_path):
    """The file shrinks under a loaded engine: the next inference's reads
    hit the end of the file, swapnet_engine_sync reports IO once, and with
    the file restored the engine gives the resident bytes again.  (A failed
    read leaves stale staging bytes; nothing on the device faults.)"""
    m, w, x, d, host, wf, budget, path = _setup("resnet50", dict(batch=1), 0.40, tmp_path)
    ref = Runner(m, w, capi.Plan.resident(d), host).run(x)
    r = Runner(m, w, capi.Plan.partition(d, budget, capi.options()), wf)
    assert all(a.tobytes() == b.tobytes() for a, b in zip(r.run(x), ref))
    full = open(path, "rb").read()
    os.truncate(path, 8192)
    with pytest.raises(capi.SwapnetError) as ei:
        r.run(x)
    assert ei.value.code == capi.ERR_IO
    with open(path, "r+b") as fh:
        fh.write(full)
    got = r.run(x)
    assert all(a.tobytes() == b.tobytes() for a, b in zip(got, ref))
