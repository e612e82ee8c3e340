"""Shared helpers of the GPU tests: run a workload through the C ABI and
compare it with the CPU oracle."""
import numpy as np

from oracle import forward as F
from oracle import plan as OP
from paper_2401_16757_gb300 import capi

NP_STORAGE = {"f32": np.float32, "f16": np.float16, "bf16": np.uint16}


def rel_l2(got, ref):
    got = np.asarray(got, dtype=np.float64).ravel()
    ref = np.asarray(ref, dtype=np.float64).ravel()
    return float(np.linalg.norm(got - ref) / max(np.linalg.norm(ref), 1e-300))


def max_rel_normwise(got, ref):
    """max_i |g_i - o_i| / max_j |o_j| (the fp32 tolerance's reading)."""
    got = np.asarray(got, dtype=np.float64).ravel()
    ref = np.asarray(ref, dtype=np.float64).ravel()
    return float(np.max(np.abs(got - ref)) / max(np.max(np.abs(ref)), 1e-30))


def check_close(model, got_list, ref_list):
    """fp32: max normwise relative error <= 1e-4; fp16/bf16: relative L2
    error <= 2e-3 per output tensor."""
    for g, r in zip(got_list, ref_list):
        assert g.shape == r.shape, (g.shape, r.shape)
        assert np.all(np.isfinite(g))
        if model["dtype"] == "f32":
            e = max_rel_normwise(g, r)
            assert e <= 1e-4, e
        else:
            e = rel_l2(g, r)
            assert e <= 2e-3, e


class Runner:
    """Owns a plan, an engine and device buffers for one workload."""

    def __init__(self, model, weights, plan, host=None):
        import torch
        self.torch = torch
        self.model = model
        self.host_weights = weights
        self.plan = plan
        self.info = plan.info()
        self.host = host or capi.HostWeights(weights)
        self.engine = capi.Engine(plan, self.host)
        self.d_in = torch.empty(max(self.info["input_bytes"], 16), dtype=torch.uint8, device="cuda")
        self.d_out = torch.zeros(self.info["output_bytes"], dtype=torch.uint8, device="cuda")
        self.shapes = OP.out_shapes(model)
        self.offs = plan.output_offsets()

    def run(self, x_storage):
        torch = self.torch
        src = torch.from_numpy(np.ascontiguousarray(x_storage).view(np.uint8).reshape(-1))
        self.d_in[:src.numel()].copy_(src)
        s = torch.cuda.current_stream()
        self.engine.infer(self.d_in.data_ptr(), self.d_out.data_ptr(), s.cuda_stream)
        self.engine.sync()
        torch.cuda.synchronize()
        return self.outputs_raw()

    def outputs_raw(self):
        host = self.d_out.cpu().numpy()
        outs = []
        es = np.dtype(NP_STORAGE[self.model["dtype"]]).itemsize
        for li, off in zip(sorted(self.model["outputs"]), self.offs):
            shp = self.shapes[li]
            nb = int(np.prod(shp)) * es
            outs.append(host[off:off + nb].view(NP_STORAGE[self.model["dtype"]]).reshape(shp).copy())
        return outs

    def decode(self, raw):
        return [F.decode(r, self.model["dtype"]) for r in raw]


def oracle_outputs(model, weights, x):
    return F.forward(model, weights, x)


_ORACLE_CACHE = {}


def oracle_cached(model, weights, x, request=0):
    """oracle_outputs of a workload built by synth (seeded weights, input of
    `request`), kept for the rest of the session: several tests compare
    different engines of the same workload with the same oracle run."""
    key = (model["name"], model["model_id"], tuple(model["input"]), request, x.tobytes()[:64], x.nbytes)
    if key not in _ORACLE_CACHE:
        _ORACLE_CACHE[key] = F.forward(model, weights, x)
    return _ORACLE_CACHE[key]


def check_oracle(runner, got_raw, x, request=0):
    """The engine's raw outputs of input x against the (cached) oracle."""
    check_close(runner.model, runner.decode(got_raw), oracle_cached(runner.model, runner.host_weights, x, request))
