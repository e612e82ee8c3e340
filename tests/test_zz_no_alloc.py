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
        # and the oracle: the same linear layer in float64, rounded once
        orc = F.forward(m, w, x)[0].reshape(-1)
        assert rel_l2(got, orc) <= 2e-3, (call, rel_l2(got, orc))
    eng.free()


def _oracle_linear(a, w, b, dtype):
    """relu(a w^T + b) in float64, rounded to the storage dtype (the oracle's
    linear layer and rounding)."""
    L = dict(op="linear", src=[-1], k=a.shape[1], n=w.shape[0], act="relu", res=None, res_post=False)
    acts = {}
    x_in = F.decode(a, dtype).reshape(a.shape[0], a.shape[1], 1, 1)
    return F.run_layer(L, dtype, [w, b], acts, x_in).reshape(a.shape[0], w.shape[0])


@pytest.mark.parametrize("dtype", ["f16", "bf16"])
def test_noalloc_chained_calls_against_oracle(dtype):
    """Two calls back to back on one stream where the second call's weight
    matrix is the first call's output: the second kernel must not read W
    before the first has written it.  Both results against the oracle (the
    second one fed the first call's stored output), and no device memory
    taken by the calls (free device bytes unchanged across a repeat of the
    pair, after a first pair has loaded the kernels)."""
    import torch
    npdt = np.uint16 if dtype == "bf16" else np.float16
    M1, K1, N1 = 64, 4096, 256     # split-K through the static scratch
    M2, K2, N2 = 96, 256, 64       # W2 = Y1 viewed as [64][256]: no split
    m1 = _layer_model(M1, K1, N1, dtype)
    w1 = synth.gen.model_weights(m1)
    a1 = synth.gen.model_input(m1).reshape(M1, K1)
    m2 = dict(_layer_model(M2, K2, N2, dtype), model_id=62)
    b2 = synth.gen.model_weights(m2)[0][1]
    a2 = synth.gen.model_input(m2).reshape(M2, K2)
    dev = lambda arr: torch.from_numpy(np.ascontiguousarray(arr).view(np.uint8).reshape(-1).copy()).cuda()
    d_a1, d_w1, d_b1, d_a2, d_b2 = dev(a1), dev(w1[0][0]), dev(w1[0][1]), dev(a2), dev(b2)
    d_y1 = torch.empty(M1 * N1 * 2, dtype=torch.uint8, device="cuda")
    d_y2 = torch.empty(M2 * N2 * 2, dtype=torch.uint8, device="cuda")
    stream = torch.cuda.current_stream().cuda_stream
    dt = capi.DTYPE[dtype]

    def pair():
        d_y1.fill_(0xFF)           # NaN bit patterns until the first call writes Y1
        d_y2.fill_(0xFF)
        capi.gemm_noalloc(dt, d_a1.data_ptr(), d_w1.data_ptr(), d_b1.data_ptr(), d_y1.data_ptr(), M1, N1, K1,
                          act=capi.ACT["relu"], stream=stream)
        capi.gemm_noalloc(dt, d_a2.data_ptr(), d_y1.data_ptr(), d_b2.data_ptr(), d_y2.data_ptr(), M2, N2, K2,
                          act=capi.ACT["relu"], stream=stream)

    pair()
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    pair()
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info()[0] == free0
    y1 = d_y1.cpu().numpy().view(npdt).reshape(M1, N1)
    y2 = d_y2.cpu().numpy().view(npdt).reshape(M2, N2)
    ref1 = _oracle_linear(a1, w1[0][0], w1[0][1], dtype)
    ref2 = _oracle_linear(a2, y1.reshape(N2, K2), b2, dtype)
    got1, got2 = F.decode(y1, dtype), F.decode(y2, dtype)
    assert np.all(np.isfinite(got1)) and np.all(np.isfinite(got2))
    assert rel_l2(got1, ref1) <= 2e-3, rel_l2(got1, ref1)
    assert rel_l2(got2, ref2) <= 2e-3, rel_l2(got2, ref2)


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
