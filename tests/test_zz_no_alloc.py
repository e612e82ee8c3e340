"""swapnet_gemm_noalloc: the GEMM entry point that allocates no device
memory (its split-K scratch is a fixed array inside the library), for
callers that run under a device-memory budget with every byte already
assigned.  Its output must match the engine's own entry point
(swapnet_infer of the same one-layer model), call after call.

Kept in a file that pytest collects last, so a run that stops at the first
failure has run every other test before this one."""
import numpy as np
import pytest

import synth
from oracle import forward as F
from paper_2401_16757_gb300 import capi
from helpers import rel_l2

pytestmark = pytest.mark.gpu


def _layer_model(M, K, N, dtype):
    return dict(name="yolov3", model_id=61, dtype=dtype, input=(M, 1, 1, K),
                layers=[dict(op="linear", src=[-1], k=K, n=N, act="relu", res=None, res_post=False)],
                outputs=[0])


@pytest.mark.parametrize("dtype", ["f16", "bf16"])
def test_noalloc_gemm_matches_engine(dtype):
    import torch
    M, K, N = 64, 4096, 256          # one M tile, four N tiles, deep K: split-K with scratch
    m = _layer_model(M, K, N, dtype)
    w = synth.gen.model_weights(m)
    x = synth.gen.model_input(m)
    d = capi.Desc(m)
    plan = capi.Plan.resident(d)
    info = plan.info()
    eng = capi.Engine(plan, capi.HostWeights(w))
    assert eng.unit_kernels() == ["tc_gemm"]
    stream = torch.cuda.current_stream().cuda_stream
    d_x = torch.from_numpy(x.view(np.uint8).reshape(-1).copy()).cuda()
    d_ref = torch.zeros(info["output_bytes"], dtype=torch.uint8, device="cuda")
    eng.infer(d_x.data_ptr(), d_ref.data_ptr(), stream)
    eng.sync()
    ref = d_ref.cpu().numpy()[:M * N * 2].view(np.uint16 if dtype == "bf16" else np.float16)
    ref = F.decode(ref, dtype)
    d_w = torch.from_numpy(w[0][0].view(np.uint8).reshape(-1).copy()).cuda()
    d_b = torch.from_numpy(w[0][1].view(np.uint8).reshape(-1).copy()).cuda()
    d_y = torch.empty(M * N * 2, dtype=torch.uint8, device="cuda")
    dt = capi.DTYPE[dtype]
    for call in range(2):  # two calls in a row share the scratch array
        d_y.fill_(0xFF)
        capi.gemm_noalloc(dt, d_x.data_ptr(), d_w.data_ptr(), d_b.data_ptr(), d_y.data_ptr(), M, N, K,
                          act=capi.ACT["relu"], stream=stream)
        torch.cuda.synchronize()
        got = d_y.cpu().numpy().view(np.uint16 if dtype == "bf16" else np.float16)
        got = F.decode(got, dtype)
        assert np.all(np.isfinite(got))
        assert rel_l2(got, ref) <= 2e-3, (call, rel_l2(got, ref))
    eng.free()


def test_noalloc_gemm_rejects_oversize_scratch():
    import torch
    # M=128, N=4864, K=4096 splits K in two: 2 x 128 x 4864 fp32 partials
    # (~4.98 MB) exceed the 4 MiB array, so the call is refused before any
    # launch.  The buffers are sized for the full problem all the same.
    M, N, K = 128, 4864, 4096
    a = torch.zeros(M * K, dtype=torch.float16, device="cuda")
    w = torch.zeros(N * K, dtype=torch.float16, device="cuda")
    b = torch.zeros(N, dtype=torch.float16, device="cuda")
    y = torch.zeros(M * N, dtype=torch.float16, device="cuda")
    with pytest.raises(capi.SwapnetError) as ei:
        capi.gemm_noalloc(capi.F16, a.data_ptr(), w.data_ptr(), b.data_ptr(), y.data_ptr(), M, N, K)
    assert ei.value.code == capi.ERR_INVALID_ARG
    assert b"scratch" in capi.lib().swapnet_last_error()
    torch.cuda.synchronize()
    assert int(torch.count_nonzero(y)) == 0   # nothing ran
    # misaligned pointers are refused as well
    with pytest.raises(capi.SwapnetError) as ei:
        capi.gemm_noalloc(capi.F16, a.data_ptr() + 8, w.data_ptr(), b.data_ptr(), y.data_ptr(), 64, 64, 64)
    assert ei.value.code == capi.ERR_MISALIGNED
