"""Float64 forward pass of the synthetic workloads (test infrastructure only).

What is computed.  Swapping changes neither the parameters nor the
architecture (Sec. 3, "Design Scope": lossless), so the swapped result of any
partition is the plain forward pass; this module writes that forward pass out
from the textbook definition of each layer:

  linear   y[m, o] = b[o] + sum_i x[m, i] * W[o, i]          (W is [out, in])
  conv2d   y[n, c, h, w] = b[c] + sum_{ci, i, j}
               x[n, ci, h*s + i - p, w*s + j - p] * W[c, i, j, ci]
           (zero outside the image; W stored [cout][kh][kw][cin])
  maxpool  max over the window; padded positions never win
  gap      mean over H and W
  upsample nearest neighbour, factor 2
  concat   channels of src[0] followed by channels of src[1]
  act      relu(x) = max(x, 0); leaky(x) = x if x > 0 else 0.1 x;
           swiglu: silu(r) * (acc + b) with silu(z) = z / (1 + e^-z), r the
           gate layer's output
  residual res_post False: act(acc + b + r); True: act(acc + b) + r
  embed    rows of the table picked by the token ids
  rmsnorm  x / sqrt(mean(x^2) + eps) * g
  attention  RoPE (adjacent pairs, angle = position * theta^(-2i/Dh)) on q
           and k, both rounded to the storage dtype; k and v appended to the
           layer's cache at positions pos0..; query t attends to positions
           0..pos0+t: softmax(q k^T / sqrt(Dh)) v per head
  argmax   first index of the row maximum (int32 on the GPU)

Precision.  Arithmetic is float64.  The GPU path stores every layer output in
the model's storage dtype; the oracle rounds each layer output to that dtype
(round-to-nearest-even) at the same tensor boundaries and nowhere else, so
the two differ only by accumulation order inside a layer.

Layout.  Tensors are NCHW inside the oracle.  The model input and outputs are
NHWC (the storage layout of the workloads); a linear layer flattens its input
per batch item in (h, w, c) order.
"""
import numpy as np


# ----------------------------------------------------------------- dtypes
def decode(a, dtype):
    """Storage array -> float64 (exact)."""
    if dtype in ("f32", "f16"):
        return np.asarray(a).astype(np.float64)
    if dtype == "bf16":
        u = np.asarray(a, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
        return u.view(np.float32).astype(np.float64)
    raise ValueError(dtype)


def round_as(x, dtype):
    """Round float64 values to the nearest value of `dtype` (ties to even),
    returned as float64."""
    x = np.asarray(x, dtype=np.float64)
    if dtype == "f32":
        return x.astype(np.float32).astype(np.float64)
    if dtype == "f16":
        return x.astype(np.float16).astype(np.float64)
    if dtype == "bf16":
        # bf16 keeps 8 significant bits: x = m * 2^e with m in [0.5, 1);
        # round m * 2^8 to an integer, ties to even (np.rint), and rescale.
        m, e = np.frexp(x)
        return np.ldexp(np.rint(m * 256.0) / 256.0, e)
    raise ValueError(dtype)


# ----------------------------------------------------------------- layers
def silu(z):
    return z / (1.0 + np.exp(-z))


def rmsnorm(x2d, g, eps):
    """x / sqrt(mean(x^2) + eps) * g over the last axis."""
    return x2d / np.sqrt(np.mean(x2d * x2d, axis=-1, keepdims=True) + eps) * g[None, :]


def rope(x2d, positions, heads, theta):
    """Rotate adjacent pairs (2i, 2i+1) of every head by position * theta^(-2i/Dh)."""
    t, width = x2d.shape
    dh = width // heads
    x = x2d.reshape(t, heads, dh // 2, 2)
    inv = theta ** (-np.arange(0, dh, 2, dtype=np.float64) / dh)     # [Dh/2]
    ang = np.asarray(positions, dtype=np.float64)[:, None] * inv[None, :]   # [T, Dh/2]
    c, s = np.cos(ang)[:, None, :], np.sin(ang)[:, None, :]
    x0, x1 = x[..., 0], x[..., 1]
    out = np.stack([x0 * c - x1 * s, x0 * s + x1 * c], axis=-1)
    return out.reshape(t, width)


def causal_attention(q2d, keys, values, pos0, heads):
    """Query t (position pos0 + t) attends to cache positions 0..pos0+t:
    softmax(q k^T / sqrt(Dh)) v, per head."""
    t, width = q2d.shape
    dh = width // heads
    out = np.zeros((t, width))
    for h in range(heads):
        sl = slice(h * dh, (h + 1) * dh)
        for i in range(t):
            n = pos0 + i + 1
            sc = keys[:n, sl] @ q2d[i, sl] / np.sqrt(dh)
            p = np.exp(sc - sc.max())
            p /= p.sum()
            out[i, sl] = p @ values[:n, sl]
    return out


def act_fn(y, act):
    if act == "none":
        return y
    if act == "relu":
        return np.maximum(y, 0.0)
    if act == "leaky":
        return np.where(y > 0.0, y, 0.1 * y)
    raise ValueError(act)


def linear(x2d, w, b):
    """x2d [M, K], w [N, K], b [N] -> [M, N]."""
    return x2d @ w.T + b[None, :]


def conv2d(x, w_krsc, b, stride, pad):
    """x [N, Ci, H, W]; w [Co, kh, kw, Ci] -> [N, Co, Ho, Wo].

    The sum over (ci, i, j) is taken tap by tap: for each kernel tap (i, j)
    the strided window of the padded input is contracted with W[:, i, j, :]
    over ci (a matmul).
    """
    n, ci, h, wd = x.shape
    co, kh, kw, ci2 = w_krsc.shape
    assert ci == ci2
    ho = (h + 2 * pad - kh) // stride + 1
    wo = (wd + 2 * pad - kw) // stride + 1
    xp = np.zeros((n, ci, h + 2 * pad, wd + 2 * pad))
    xp[:, :, pad:pad + h, pad:pad + wd] = x
    y = np.zeros((n, co, ho, wo)) + b[None, :, None, None]
    for i in range(kh):
        for j in range(kw):
            win = xp[:, :, i:i + stride * (ho - 1) + 1:stride, j:j + stride * (wo - 1) + 1:stride]
            # [Co, Ci] x [N, Ci, Ho, Wo] -> [Co, N, Ho, Wo]
            y += np.tensordot(w_krsc[:, i, j, :], win, axes=([1], [1])).transpose(1, 0, 2, 3)
    return y


def maxpool(x, kh, kw, stride, pad):
    n, c, h, wd = x.shape
    ho = (h + 2 * pad - kh) // stride + 1
    wo = (wd + 2 * pad - kw) // stride + 1
    xp = np.full((n, c, h + 2 * pad, wd + 2 * pad), -np.inf)
    xp[:, :, pad:pad + h, pad:pad + wd] = x
    y = np.full((n, c, ho, wo), -np.inf)
    for i in range(kh):
        for j in range(kw):
            y = np.maximum(y, xp[:, :, i:i + stride * (ho - 1) + 1:stride,
                                 j:j + stride * (wo - 1) + 1:stride])
    return y


def gap(x):
    return x.mean(axis=(2, 3), keepdims=True)


def upsample2x(x):
    return x.repeat(2, axis=2).repeat(2, axis=3)


def concat(a, b):
    return np.concatenate([a, b], axis=1)


# ----------------------------------------------------------------- model
def nhwc_to_nchw(a):
    return np.ascontiguousarray(np.asarray(a).transpose(0, 3, 1, 2))


def nchw_to_nhwc(a):
    return np.ascontiguousarray(np.asarray(a).transpose(0, 2, 3, 1))


def _as2d(a):
    return a.reshape(a.shape[0], -1)


def decode_params(tensors, dtype):
    """A layer's parameter tensors as float64 (exact)."""
    return [decode(t, dtype) for t in tensors]


def run_layer(layer, dtype, tensors, acts, x_in, state=None, li=None, params=None):
    """Compute one layer (float64 in, rounded float64 out).

    tensors: the layer's storage arrays; acts: dict layer index -> NCHW
    float64 output; x_in: NCHW float64 model input (token ids for a token
    model); state: KV caches and position for attention layers; params:
    decode_params(tensors) when the caller already has them (a layer run
    several times is decoded once).
    """
    def get(i):
        return x_in if i == -1 else acts[i]

    def param(i):
        return params[i] if params is not None else decode(tensors[i], dtype)

    op = layer["op"]
    src = get(layer["src"][0])
    if op == "embed":
        table = param(0)
        ids = np.asarray(src).reshape(-1).astype(np.int64)
        return table[ids].reshape(len(ids), -1, 1, 1)          # a copy: no rounding needed
    if op == "rmsnorm":
        y = rmsnorm(_as2d(src), param(0), layer["eps"])
        return round_as(y, dtype).reshape(src.shape)
    if op == "attention":
        q, k, v = (_as2d(get(i)) for i in layer["src"])
        t = q.shape[0]
        pos0 = state["pos"]
        pos = np.arange(pos0, pos0 + t)
        qr = round_as(rope(q, pos, layer["heads"], layer["theta"]), dtype)
        kr = round_as(rope(k, pos, layer["heads"], layer["theta"]), dtype)
        cache = state["kv"].setdefault(li, (np.zeros((layer["max_seq"], q.shape[1])),
                                            np.zeros((layer["max_seq"], q.shape[1]))))
        cache[0][pos0:pos0 + t] = kr
        cache[1][pos0:pos0 + t] = v
        y = causal_attention(qr, cache[0], cache[1], pos0, layer["heads"])
        return round_as(y, dtype).reshape(t, -1, 1, 1)
    if op == "argmax":
        a = _as2d(src)
        return np.argmax(a, axis=1).astype(np.float64).reshape(-1, 1, 1, 1)
    if op in ("conv", "linear"):
        w = param(0)
        b = param(1) if len(tensors) > 1 else np.zeros(w.shape[0])
        if op == "conv":
            y = conv2d(src, w, b, layer["stride"], layer["pad"])
        else:
            n = src.shape[0]
            flat = nchw_to_nhwc(src).reshape(n, -1)          # (h, w, c) order
            assert flat.shape[1] == layer["k"], (flat.shape, layer["k"])
            y = linear(flat, w, b).reshape(n, layer["n"], 1, 1)
        r = None if layer.get("res") is None else get(layer["res"])
        if layer.get("act") == "swiglu":
            y = silu(r) * y
        elif r is not None and not layer["res_post"]:
            y = act_fn(y + r, layer["act"])
        elif r is not None:
            y = act_fn(y, layer["act"]) + r
        else:
            y = act_fn(y, layer["act"])
    elif op == "maxpool":
        y = maxpool(src, layer["kh"], layer["kw"], layer["stride"], layer["pad"])
    elif op == "gap":
        y = gap(src)
    elif op == "upsample2x":
        y = upsample2x(src)
    elif op == "concat":
        y = concat(src, get(layer["src"][1]))
    else:
        raise ValueError(op)
    return round_as(y, dtype)


def forward_range(model, weights, acts, x_in, lo, hi, state=None):
    """Run layers [lo, hi) in order, adding their outputs to `acts`."""
    dt = model["dtype"]
    for li in range(lo, hi):
        acts[li] = run_layer(model["layers"][li], dt, weights[li], acts, x_in, state, li)
    return acts


def new_state():
    """KV caches and the number of positions already cached."""
    return {"pos": 0, "kv": {}}


def _model_input(model, x_nhwc):
    if model.get("input_dtype") == "i32":
        return np.asarray(x_nhwc)
    return nhwc_to_nchw(decode(x_nhwc, model["dtype"]))


def forward(model, weights, x_nhwc, check_range=True, state=None):
    """Plain forward pass; returns the model outputs as NHWC float64 arrays
    (values exactly representable in the storage dtype).  Token models keep
    their KV caches and position in `state`, advanced by the tokens read."""
    x_in = _model_input(model, x_nhwc)
    if state is None:
        state = new_state()
    acts = forward_range(model, weights, {}, x_in, 0, len(model["layers"]), state)
    if model.get("input_dtype") == "i32":
        state["pos"] += int(np.asarray(x_nhwc).shape[0])
    outs = [nchw_to_nhwc(acts[i]) for i in model["outputs"]]
    if check_range:
        for o in outs:
            assert np.all(np.isfinite(o)), "non-finite activation in the oracle"
    return outs


def forward_all(model, weights, x_nhwc, state=None):
    """Every layer output, NHWC float64 (for per-layer parity checks)."""
    x_in = _model_input(model, x_nhwc)
    acts = forward_range(model, weights, {}, x_in, 0, len(model["layers"]), state or new_state())
    return {i: nchw_to_nhwc(a) for i, a in acts.items()}
