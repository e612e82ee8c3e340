"""Seeded generators for synthetic weights and inputs.

Both the CUDA path and the CPU oracle consume the tensors made here; this
module only draws random numbers and stores them in the storage dtype.

Reproducibility rules:
  * one PCG64 stream per tensor, keyed (seed, model_id, layer, tensor slot);
  * values are drawn in float64 and rounded once, round-to-nearest-even,
    to the storage dtype (fp32, fp16, or bf16 kept as uint16 bit patterns);
  * weights use seed 0, inputs seed 1 (request r of a stream: seed 1000*r+1).

Initialisation per workload:
  mlp6      W ~ N(0, 1/fan_in), b = 0
  resnet50  conv W ~ N(0, 2/fan_in) with an inference BatchNorm folded in:
            gamma ~ U(0.5, 1.5) (U(0, 0.2) for the last BN of each residual
            branch, which keeps fp16 activations finite through 16
            unnormalised residual adds), beta ~ N(0, 0.1), mean ~ N(0, 0.1),
            var ~ U(0.5, 1.5), eps = 1e-5; W' = W*g/sqrt(var+eps),
            b' = beta - mean*g/sqrt(var+eps) (folded in float64, rounded once);
            FC W ~ N(0, 1/fan_in), b ~ N(0, 0.01)
  vgg16     W ~ N(0, 2/fan_in) (He) for ReLU layers, N(0, 1/fan_in) for the
            last FC, b = 0
  yolov3    W ~ N(0, 1/fan_in), b ~ N(0, 0.01)
  llm       every matrix and the embedding N(0, 0.02) (drawn in float32,
            rounded to bf16), RMSNorm gains 1, no biases
  inputs    N(0, 1); token ids U[0, vocab) with seed 2
"""
import numpy as np

_NP_DTYPE = {"f32": np.float32, "f16": np.float16, "bf16": np.uint16}


def _rng(*key):
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence(list(key))))


def round_to_storage(x64, dtype):
    """float64 array -> storage array (RNE, one rounding)."""
    x64 = np.ascontiguousarray(x64, dtype=np.float64)
    if dtype == "f32":
        return x64.astype(np.float32)
    if dtype == "f16":
        return x64.astype(np.float16)
    if dtype == "bf16":
        # Round the float64 significand to 8 bits (RNE) by integer arithmetic
        # on the bit pattern, then the value is exact in float32 and its top
        # 16 bits are the bf16 pattern.
        b = x64.view(np.uint64)
        lsb = (b >> np.uint64(45)) & np.uint64(1)
        b = (b + np.uint64((1 << 44) - 1) + lsb) & ~np.uint64((1 << 45) - 1)
        f32 = b.view(np.float64).astype(np.float32)
        return (f32.view(np.uint32) >> np.uint32(16)).astype(np.uint16)
    raise ValueError(dtype)


def _fan_in(layer):
    if layer["op"] == "conv":
        return layer["cin"] * layer["kh"] * layer["kw"]
    return layer["k"]


def _bf16_from_f32(f):
    """float32 -> bf16 bit patterns, round-to-nearest-even."""
    u = f.view(np.uint32)
    lsb = (u >> np.uint32(16)) & np.uint32(1)
    return ((u + np.uint32(0x7FFF) + lsb) >> np.uint32(16)).astype(np.uint16)


def llm_tensor(model, li, ti, shape, seed=0):
    """LLM parameters: N(0, 0.02) drawn in float32 (the 7B tables are large),
    rounded once to bf16; RMSNorm gains are 1."""
    layer = model["layers"][li]
    if layer["op"] == "rmsnorm":
        return np.full(shape, 0x3F80, dtype=np.uint16)   # 1.0
    r = _rng(seed, model["model_id"], li, ti)
    f = r.standard_normal(int(np.prod(shape)), dtype=np.float32)
    f *= np.float32(0.02)
    return _bf16_from_f32(f).reshape(shape)


def layer_weights(model, li, seed=0):
    """Parameter tensors of layer li as storage arrays ([] for weightless ops)."""
    layer = model["layers"][li]
    if model["name"] == "llm":
        from .arch import tensor_shapes
        return [llm_tensor(model, li, ti, shp, seed) for ti, (_, shp) in enumerate(tensor_shapes(layer))]
    if layer["op"] == "rmsnorm":   # gains of a non-LLM test model: U(0.5, 1.5)
        return [round_to_storage(_rng(seed, model["model_id"], li, 0).uniform(0.5, 1.5, layer["d"]), model["dtype"])]
    if layer["op"] == "embed":
        return [round_to_storage(_rng(seed, model["model_id"], li, 0).normal(0.0, 1.0, (layer["vocab"], layer["d"])),
                                 model["dtype"])]
    if layer["op"] not in ("conv", "linear"):
        return []
    dt, mid, name = model["dtype"], model["model_id"], model["name"]
    fan = _fan_in(layer)
    if layer["op"] == "conv":
        wshape = (layer["cout"], layer["kh"], layer["kw"], layer["cin"])
        nout = layer["cout"]
    else:
        wshape = (layer["n"], layer["k"])
        nout = layer["n"]
    rw, rb = _rng(seed, mid, li, 0), _rng(seed, mid, li, 1)
    if layer.get("bias") is False:
        return [round_to_storage(rw.normal(0.0, np.sqrt(1.0 / fan), wshape), dt)]
    if name == "mlp6":
        w = rw.normal(0.0, np.sqrt(1.0 / fan), wshape)
        b = np.zeros(nout)
    elif name == "resnet50":
        if layer["op"] == "conv":
            w = rw.normal(0.0, np.sqrt(2.0 / fan), wshape)
            # the last BN of a residual branch: small gamma (zero-gamma style
            # residual init); elsewhere U(0.5, 1.5)
            last = layer.get("res") is not None
            gamma = rb.uniform(0.0, 0.2, nout) if last else rb.uniform(0.5, 1.5, nout)
            beta = rb.normal(0.0, 0.1, nout)
            mean = rb.normal(0.0, 0.1, nout)
            var = rb.uniform(0.5, 1.5, nout)
            scale = gamma / np.sqrt(var + 1e-5)
            w = w * scale[:, None, None, None]
            b = beta - mean * scale
        else:
            w = rw.normal(0.0, np.sqrt(1.0 / fan), wshape)
            b = rb.normal(0.0, 0.01, nout)
    elif name == "vgg16":
        gain = 2.0 if layer["act"] == "relu" else 1.0
        w = rw.normal(0.0, np.sqrt(gain / fan), wshape)
        b = np.zeros(nout)
    elif name == "yolov3":
        w = rw.normal(0.0, np.sqrt(1.0 / fan), wshape)
        b = rb.normal(0.0, 0.01, nout)
    else:
        raise ValueError(name)
    return [round_to_storage(w, dt), round_to_storage(b, dt)]


def model_weights(model, seed=0):
    """List (per layer) of lists of storage arrays."""
    return [layer_weights(model, li, seed) for li in range(len(model["layers"]))]


def model_input(model, seed=1, request=0):
    """Model input, NHWC storage array, N(0, 1); for token models, int32 ids
    U[0, vocab) with seed 2."""
    if model.get("input_dtype") == "i32":
        vocab = model["layers"][0]["vocab"]
        r = _rng(2 + 1000 * request, model["model_id"], 0xFFFF, 0)
        return r.integers(0, vocab, size=model["input"], dtype=np.int32)
    r = _rng(seed + 1000 * request, model["model_id"], 0xFFFF, 0)
    return round_to_storage(r.normal(0.0, 1.0, model["input"]), model["dtype"])


def storage_nbytes(dtype):
    return np.dtype(_NP_DTYPE[dtype]).itemsize
