"""Layer-sequence descriptions of the synthetic workloads (structure only).

A model is a dict:
  name      short identifier
  model_id  small integer used to key the seeded generators
  dtype     storage dtype of weights and activations: 'f32' | 'f16' | 'bf16'
  input     (N, H, W, C) of the model input, NHWC.  A plain feature matrix
            [rows, features] is (rows, 1, 1, features).
  layers    list of layer dicts, in execution (topological) order
  outputs   indices of the layers whose outputs are model outputs

Layer dict keys (all integers unless noted):
  op        'linear' | 'conv' | 'maxpool' | 'gap' | 'upsample2x' | 'concat'
            | 'embed' | 'rmsnorm' | 'attention' | 'argmax'
  src       list of producer layer indices; -1 is the model input
  linear:   k (input features = H*W*C of the input, flattened in (h, w, c)
            order), n (output features), act, res, res_post
  conv:     cin, cout, kh, kw, stride, pad, act, res, res_post
            (zero padding, NHWC activations, weights stored [cout][kh][kw][cin])
  maxpool:  kh, kw, stride, pad (padding never wins the max)
  gap:      global average over H and W
  upsample2x: nearest-neighbour x2 in H and W
  concat:   channel concatenation of src[0] then src[1]
  embed:    vocab, d (rows of the table picked by int32 token ids)
  rmsnorm:  d, eps: x / sqrt(mean(x^2) + eps) * g
  attention: src = [q, k, v]; heads, max_seq, theta (RoPE base)
  argmax:   index of the largest value of each row (ties: lowest index)
  act       'none' | 'relu' | 'leaky' (slope 0.1) | 'swiglu' (silu(res) * y)
  bias      False: the linear layer has no bias tensor
  res       index of a layer whose output is added element-wise, or None
  res_post  False: out = act(acc + bias + res)   (ResNet bottleneck)
            True:  out = act(acc + bias) + res   (Darknet shortcut)

This module holds no arithmetic of the swapping method: it only states which
network each workload runs (sizes from the workload definitions: a 6-layer
MLP, ResNet-50, VGG-16, a Darknet-53 YOLOv3 backbone with three heads).
"""


def _conv(src, cin, cout, k, stride=1, pad=None, act="relu", res=None, res_post=False):
    return dict(op="conv", src=[src], cin=cin, cout=cout, kh=k, kw=k, stride=stride,
                pad=(k // 2 if pad is None else pad), act=act, res=res, res_post=res_post)


def _linear(src, k, n, act="none", res=None):
    return dict(op="linear", src=[src], k=k, n=n, act=act, res=res, res_post=False)


def mlp6(batch=8, width=1024):
    """Six fully connected layers of equal width, ReLU between layers, fp32."""
    layers = []
    for i in range(6):
        layers.append(_linear(i - 1, width, width, act=("relu" if i < 5 else "none")))
    return dict(name="mlp6", model_id=1, dtype="f32", input=(batch, 1, 1, width),
                layers=layers, outputs=[5])


def resnet50(batch=1, res=224, classes=1000):
    """ResNet-50 v1.5 (stride on the 3x3 conv), BN folded into each conv."""
    L = []
    L.append(_conv(-1, 3, 64, 7, stride=2, pad=3))                 # stem
    L.append(dict(op="maxpool", src=[0], kh=3, kw=3, stride=2, pad=1))
    x, cin = 1, 64
    for nblocks, mid, out, stride in ((3, 64, 256, 1), (4, 128, 512, 2),
                                      (6, 256, 1024, 2), (3, 512, 2048, 2)):
        for b in range(nblocks):
            s = stride if b == 0 else 1
            L.append(_conv(x, cin, mid, 1))
            c1 = len(L) - 1
            L.append(_conv(c1, mid, mid, 3, stride=s))
            c2 = len(L) - 1
            if b == 0:
                L.append(_conv(x, cin, out, 1, stride=s, act="none"))
                short = len(L) - 1
            else:
                short = x
            L.append(_conv(c2, mid, out, 1, act="relu", res=short, res_post=False))
            x, cin = len(L) - 1, out
    L.append(dict(op="gap", src=[x]))
    L.append(_linear(len(L) - 1, 2048, classes))
    return dict(name="resnet50", model_id=2, dtype="f16", input=(batch, res, res, 3),
                layers=L, outputs=[len(L) - 1])


def vgg16(batch=1, res=224, classes=1000):
    """VGG-16: 13 3x3 convs with ReLU, 5 max-pools, FC 25088-4096-4096-1000."""
    cfg = [64, 64, "M", 128, 128, "M", 256, 256, 256, "M", 512, 512, 512, "M",
           512, 512, 512, "M"]
    L, x, cin, hw = [], -1, 3, res
    for v in cfg:
        if v == "M":
            L.append(dict(op="maxpool", src=[x], kh=2, kw=2, stride=2, pad=0))
            hw //= 2
        else:
            L.append(_conv(x, cin, v, 3))
            cin = v
        x = len(L) - 1
    feat = hw * hw * cin
    L.append(_linear(x, feat, 4096, act="relu"))
    L.append(_linear(len(L) - 1, 4096, 4096, act="relu"))
    L.append(_linear(len(L) - 1, 4096, classes))
    return dict(name="vgg16", model_id=3, dtype="f16", input=(batch, res, res, 3),
                layers=L, outputs=[len(L) - 1])


def yolov3(batch=1, res=416, classes=80):
    """Darknet-53 backbone with the three YOLOv3 detection heads (raw outputs).

    Every conv is followed by LeakyReLU(0.1) except the three 1x1 detection
    convs (linear, with bias).  A Darknet shortcut adds the block input after
    the activation of the block's 3x3 conv.
    """
    L = []

    def conv(src, cin, cout, k, stride=1, act="leaky", res=None):
        L.append(_conv(src, cin, cout, k, stride=stride, act=act, res=res, res_post=True))
        return len(L) - 1

    x = conv(-1, 3, 32, 3)
    c = 32
    routes = {}
    for nres, cout in ((1, 64), (2, 128), (8, 256), (8, 512), (4, 1024)):
        x = conv(x, c, cout, 3, stride=2)
        c = cout
        for _ in range(nres):
            a = conv(x, c, c // 2, 1)
            x = conv(a, c // 2, c, 3, res=x)
        routes[c] = x
    head_out = 3 * (classes + 5)
    outs = []

    def head(x, cin, mid):
        a = conv(x, cin, mid, 1)
        a = conv(a, mid, mid * 2, 3)
        a = conv(a, mid * 2, mid, 1)
        a = conv(a, mid, mid * 2, 3)
        branch = conv(a, mid * 2, mid, 1)
        a = conv(branch, mid, mid * 2, 3)
        o = conv(a, mid * 2, head_out, 1, act="none")
        outs.append(o)
        return branch

    b = head(x, 1024, 512)
    u = conv(b, 512, 256, 1)
    L.append(dict(op="upsample2x", src=[u]))
    L.append(dict(op="concat", src=[len(L) - 1, routes[512]]))
    b = head(len(L) - 1, 256 + 512, 256)
    u = conv(b, 256, 128, 1)
    L.append(dict(op="upsample2x", src=[u]))
    L.append(dict(op="concat", src=[len(L) - 1, routes[256]]))
    head(len(L) - 1, 128 + 256, 128)
    return dict(name="yolov3", model_id=4, dtype="f16", input=(batch, res, res, 3),
                layers=L, outputs=outs)




def llm(layers=32, d=4096, heads=32, ffn=11008, vocab=32000, tokens=512, max_seq=544):
    """LLaMA-7B-shaped decoder (pre-norm, RMSNorm eps 1e-6 with gains, RoPE
    theta 10000 on adjacent pairs, causal attention with a KV cache of
    max_seq positions, SwiGLU FFN, untied LM head, no biases), bf16.

    The input is `tokens` int32 token ids; outputs are the logits of every
    position and their argmax (ties -> lowest index).  Decoder layer i:
      rmsnorm -> q, k, v -> attention -> o (+x) -> rmsnorm -> gate, up
      (silu(gate) * up) -> down (+h)
    """
    L = [dict(op="embed", src=[-1], vocab=vocab, d=d)]
    x = 0
    for _ in range(layers):
        L.append(dict(op="rmsnorm", src=[x], d=d, eps=1e-6))
        xn = len(L) - 1
        q = len(L); L.append(_linear(xn, d, d))
        k = len(L); L.append(_linear(xn, d, d))
        v = len(L); L.append(_linear(xn, d, d))
        L.append(dict(op="attention", src=[q, k, v], heads=heads, max_seq=max_seq, theta=10000.0))
        a = len(L) - 1
        L.append(_linear(a, d, d, res=x))
        h = len(L) - 1
        L.append(dict(op="rmsnorm", src=[h], d=d, eps=1e-6))
        hn = len(L) - 1
        g = len(L); L.append(_linear(hn, d, ffn))
        L.append(dict(_linear(hn, d, ffn), act="swiglu", res=g))
        u = len(L) - 1
        L.append(_linear(u, ffn, d, res=h))
        x = len(L) - 1
    L.append(dict(op="rmsnorm", src=[x], d=d, eps=1e-6))
    L.append(_linear(len(L) - 1, d, vocab))
    head = len(L) - 1
    L.append(dict(op="argmax", src=[head]))
    for l in L:
        if l["op"] == "linear":
            l["bias"] = False
    return dict(name="llm", model_id=5, dtype="bf16", input=(tokens, 1, 1, 1), input_dtype="i32",
                layers=L, outputs=[head, len(L) - 1])


def tensor_shapes(layer):
    """Names and shapes of a layer's parameter tensors, in storage order."""
    if layer["op"] == "conv":
        return [("w", (layer["cout"], layer["kh"], layer["kw"], layer["cin"])),
                ("b", (layer["cout"],))]
    if layer["op"] == "linear":
        t = [("w", (layer["n"], layer["k"]))]
        return t if layer.get("bias") is False else t + [("b", (layer["n"],))]
    if layer["op"] == "embed":
        return [("table", (layer["vocab"], layer["d"]))]
    if layer["op"] == "rmsnorm":
        return [("g", (layer["d"],))]
    return []


MODELS = {"mlp6": mlp6, "resnet50": resnet50, "vgg16": vgg16, "yolov3": yolov3, "llm": llm}
