"""Partitioning oracle: exhaustive search with the paper's delay model
(test infrastructure only).

Sec. 6.1 gives three delay abstractions for a block i of size s_i, parameter
depth d_i (number of tensors) and FLOPs f_i:
    t_in_i  = alpha * s_i + beta * d_i      (swap-in + assembly by reference)
    t_ex_i  = gamma * f_i                   (execution)
    t_out_i = eta * d_i                     (swap-out: pointer reset, no write-back)
All times here are integer nanoseconds; alpha and gamma are given in
attoseconds per byte / per FLOP and each product is rounded up to whole ns
per block (t_in) or per layer (t_ex).  A layer may carry a measured t_ex that
replaces gamma * f.

Sec. 6.2.2 partitions the layer sequence into n blocks, p = (p_1..p_{n-1}),
minimising t(p) (Eq. 2) subject to the block-size constraint (Eq. 3): with
m = 2 blocks co-resident, every two consecutive blocks fit the arena together,
s_i + s_{i+1} <= arena (the arena is the budget less the workspace when that
is counted, rounded down to 256 bytes); with one slot, every block fits the
arena alone.  The objective is either
  0: the completion time of the m-slot swap/execute pipeline,
       C_k = max(C_{k-1}, R_{k-m}) + t_in_k       (copy of block k ends)
       E_k = max(E_{k-1}, C_k) + t_ex_k           (execution of block k ends)
       R_k = E_k + t_out_k                        (slot of block k released)
     minimising E_n (C_0 = E_0 = 0, R_j = 0 for j <= 0); or
  1: Eq. 4 as printed, sum_{i=2..n} max(t_ov_i, 0) with
       t_ov_i = (t_out_{i-1} + t_in_{i+1}) - (t_ex_i + t_ov_{i-1}),
     taking t_ov_1 = 0 and t_in_{n+1} = 0 (the paper leaves both undefined).
Ties: smaller objective, then fewer blocks, then the lexicographically
smallest cut vector.  A cut c means "a block boundary before unit c".

Steady state with first-block prefetch (option prefetch, two slots; the
Sec. 4.3 pipeline carried across back-to-back inferences): block 1 of the
next inference (index 0 here) is copied at the end of the current one, so
C_0 = 0 and E_0 = t_ex_0; that copy starts when the copy engine is done
with block n-1 and the last block in block 0's place is released -- the
blocks alternate between the two ends of the region, so that is block n-1
when n is odd and block n-2 when n is even -- and the inference ends at
    max(E_{n-1}, max(C_{n-1}, R_g) + t_in_0).
With n even, block n-1 and the next block 0 are co-resident, so Eq. 3 also
holds for that pair: s_{n-1} + s_0 <= arena.

The search here enumerates all 2^(U-1) cut vectors, so it is only for small U.

Model bookkeeping (sizes, FLOPs, output shapes, the activation workspace and
the splitting of an oversize linear layer along its output features) is
restated here from the layer definitions, independently of the library.
"""
from fractions import Fraction
import math

ALIGN = 256
ES = {"f32": 4, "f16": 2, "bf16": 2}


def align(x, a=ALIGN):
    return (x + a - 1) // a * a


def ceil_div(a, b):
    return -(-a // b)


# ----------------------------------------------------------- model analysis
def out_shapes(model):
    """NHWC shape of each layer output."""
    shapes = []

    def shp(i):
        return tuple(model["input"]) if i == -1 else shapes[i]

    for L in model["layers"]:
        n, h, w, c = shp(L["src"][0])
        op = L["op"]
        if op == "conv":
            ho = (h + 2 * L["pad"] - L["kh"]) // L["stride"] + 1
            wo = (w + 2 * L["pad"] - L["kw"]) // L["stride"] + 1
            shapes.append((n, ho, wo, L["cout"]))
        elif op == "maxpool":
            ho = (h + 2 * L["pad"] - L["kh"]) // L["stride"] + 1
            wo = (w + 2 * L["pad"] - L["kw"]) // L["stride"] + 1
            shapes.append((n, ho, wo, c))
        elif op == "linear":
            shapes.append((n, 1, 1, L["n"]))
        elif op == "gap":
            shapes.append((n, 1, 1, c))
        elif op == "upsample2x":
            shapes.append((n, 2 * h, 2 * w, c))
        elif op == "concat":
            shapes.append((n, h, w, c + shp(L["src"][1])[3]))
        elif op == "embed":
            shapes.append((n * h * w * c, 1, 1, L["d"]))
        elif op in ("rmsnorm", "attention"):
            shapes.append((n, h, w, c))
        elif op == "argmax":
            shapes.append((n, 1, 1, 1))
        else:
            raise ValueError(op)
    return shapes


def out_elem_bytes(model, li):
    """Element size of a layer output (argmax writes int32 indices)."""
    return 4 if model["layers"][li]["op"] == "argmax" else ES[model["dtype"]]


def layer_tensor_bytes(model, li):
    L, es = model["layers"][li], ES[model["dtype"]]
    if L["op"] == "conv":
        return [L["cout"] * L["kh"] * L["kw"] * L["cin"] * es, L["cout"] * es]
    if L["op"] == "linear":
        w = [L["n"] * L["k"] * es]
        return w if L.get("bias") is False else w + [L["n"] * es]
    if L["op"] == "embed":
        return [L["vocab"] * L["d"] * es]
    if L["op"] == "rmsnorm":
        return [L["d"] * es]
    return []


def host_resident(model, li):
    """The embedding table stays in host memory: its rows are gathered
    (zero-copy) by the lookup, never swapped into the arena."""
    return model["layers"][li]["op"] == "embed"


def layer_flops(model, li, shapes):
    L = model["layers"][li]
    n, ho, wo, co = shapes[li]
    if L["op"] == "conv":
        return 2 * n * ho * wo * co * L["cin"] * L["kh"] * L["kw"]
    if L["op"] == "linear":
        return 2 * n * L["k"] * L["n"]
    if L["op"] == "attention":
        return 4 * n * L["max_seq"] * co
    return 0


def workspace(model):
    """Liveness-based placement of intermediate activations.

    A non-output layer output lives over [start, last reader] (inclusive),
    start = i, except for a conv / linear layer whose producers all come
    before i - 1: it may be computed beside the layers between its last
    producer and itself, so it lives from one step after that producer.  In
    layer order each output takes the lowest 256-byte-aligned offset where it
    overlaps no placed tensor whose live interval meets its own.  The lowest
    such offset is 0 or the end of one of those tensors (if an offset o > 0
    fits and o - 256 does not, some conflicting tensor ends in (o-256, o],
    i.e. at o since ends are aligned), so only those candidates are tried.

    Returns (workspace_bytes, {layer: offset}, output_bytes, {layer: offset
    in the output buffer}).
    """
    shapes = out_shapes(model)
    es = ES[model["dtype"]]
    nl = len(model["layers"])
    last, start = list(range(nl)), list(range(nl))
    for j, L in enumerate(model["layers"]):
        refs = [i for i in list(L["src"]) + ([L["res"]] if L.get("res") is not None else []) if i >= 0]
        for i in refs:
            last[i] = max(last[i], j)
        if L["op"] in ("conv", "linear") and refs and max(refs) + 1 < j:
            start[j] = max(refs) + 1
    outs = sorted(model["outputs"])
    placed = []  # (lo, hi, off, size)
    offs = {}
    for i in range(nl):
        if i in outs:
            continue
        size = align(math.prod(shapes[i]) * out_elem_bytes(model, i))
        conflict = [p for p in placed if p[0] <= last[i] and start[i] <= p[1]]
        cands = sorted({0} | {p[2] + p[3] for p in conflict})
        for o in cands:
            if all(o + size <= p[2] or p[2] + p[3] <= o for p in conflict):
                break
        offs[i] = o
        placed.append((start[i], last[i], o, size))
    ws = max([p[2] + p[3] for p in placed], default=0)
    out_off, cur = {}, 0
    for i in outs:
        out_off[i] = cur
        cur += align(math.prod(shapes[i]) * out_elem_bytes(model, i))
    return ws, offs, cur, out_off


# ----------------------------------------------------------- units and costs
class Coef:
    """Delay coefficients: alpha [as/byte], beta [ns/tensor], gamma [as/FLOP],
    eta [ns/tensor]."""

    def __init__(self, alpha_as=2_500_000, beta_ns=2_000, gamma_as=2_000, eta_ns=0):
        self.alpha_as, self.beta_ns, self.gamma_as, self.eta_ns = alpha_as, beta_ns, gamma_as, eta_ns


def units(model, slot, t_ex_override=None, region=None):
    """Partition units: layers in order, except that a linear layer larger
    than `slot` (half the arena when two blocks are co-resident) becomes
    pieces of whole output features (a multiple of 128 per piece, as equal
    as that allows).  Other layers may be as large as `region` (the whole
    arena).  Returns a list of dicts {layer, row0, rows, bytes, depth, flops,
    t_ex_ovr} or None when some layer cannot fit."""
    if region is None:
        region = slot
    shapes = out_shapes(model)
    es = ES[model["dtype"]]
    out = []
    for li, L in enumerate(model["layers"]):
        tb = layer_tensor_bytes(model, li)
        size = 0 if host_resident(model, li) else sum(align(b) for b in tb)
        f = layer_flops(model, li, shapes)
        ovr = 0 if t_ex_override is None else t_ex_override[li]
        if size <= slot or (L["op"] != "linear" and size <= region):
            out.append(dict(layer=li, row0=0, rows=L.get("n", 0), bytes=size, depth=len(tb),
                            flops=f, t_ex_ovr=ovr))
            continue
        if L["op"] != "linear":
            return None
        K, N = L["k"], L["n"]

        def piece_bytes(r):
            return align(r * K * es) + (0 if L.get("bias") is False else align(r * es))

        rmax = 0
        r = 128
        while r <= N + 127 and piece_bytes(r) <= slot:
            rmax = r
            r += 128
        if rmax == 0:
            return None
        npieces = ceil_div(N, rmax)
        rr = ceil_div(ceil_div(N, npieces), 128) * 128
        row0 = 0
        while row0 < N:
            rows = min(rr, N - row0)
            out.append(dict(layer=li, row0=row0, rows=rows, bytes=piece_bytes(rows), depth=len(tb),
                            flops=2 * shapes[li][0] * K * rows,
                            t_ex_ovr=(ceil_div(ovr * rows, N) if ovr else 0)))
            row0 += rows
    return out


def unit_t_ex(u, coef):
    if u["t_ex_ovr"] > 0:
        return u["t_ex_ovr"]
    return ceil_div(coef.gamma_as * u["flops"], 10**9)


def block_costs(us, cuts, coef):
    """Per-block (bytes, t_in, t_ex, t_out) for the cut vector."""
    bounds = [0] + list(cuts) + [len(us)]
    res = []
    for a, b in zip(bounds[:-1], bounds[1:]):
        s = sum(u["bytes"] for u in us[a:b])
        d = sum(u["depth"] for u in us[a:b])
        t_in = ceil_div(coef.alpha_as * s, 10**9) + coef.beta_ns * d
        t_ex = sum(unit_t_ex(u, coef) for u in us[a:b])
        t_out = coef.eta_ns * d
        res.append((s, t_in, t_ex, t_out))
    return res


def pipeline_time(blocks, slots, prefix=False):
    """Objective 0: completion time of the m-slot pipeline.  With prefix,
    blocks[0] is a resident prefix (an extension, not the paper's method):
    its layers start at t = 0 without a copy and it never frees room, so the
    swapped blocks after it gate only on each other."""
    C = E = 0
    R = []
    lo = 1 if prefix else 0
    for k, (_, t_in, t_ex, t_out) in enumerate(blocks):
        if prefix and k == 0:
            E = t_ex
            R.append(0)
            continue
        gate = R[k - slots] if k - slots >= lo else 0
        C = max(C, gate) + t_in
        E = max(E, C) + t_ex
        R.append(E + t_out)
    return E


def cyclic_time(blocks):
    """Steady-state time of one inference with first-block prefetch (two
    slots), blocks = [(bytes, t_in, t_ex, t_out), ...]."""
    n = len(blocks)
    C = [0] * n
    E = [0] * n
    R = [0] * n
    for k, (_, t_in, t_ex, t_out) in enumerate(blocks):
        if k == 0:
            C[0] = 0                      # copied during the previous inference
            E[0] = t_ex
        else:
            gate = R[k - 2] if k >= 2 else 0
            C[k] = max(C[k - 1], gate) + t_in
            E[k] = max(E[k - 1], C[k]) + t_ex
        R[k] = E[k] + t_out
    g = n - 1 if n % 2 == 1 else n - 2    # last block at the same end as block 0
    next_copy_done = max(C[n - 1], R[g]) + blocks[0][1]
    return max(E[n - 1], next_copy_done)


def feasible_cyclic(blocks, region):
    """Eq. 3 for two slots, plus the pair (block n-1, next block 0) when n is
    even (they sit at opposite ends of the region at the same time)."""
    if not feasible(blocks, region, 2):
        return False
    n = len(blocks)
    return n % 2 == 1 or blocks[-1][0] + blocks[0][0] <= region


def prefix_candidates(us, region, slots):
    """Resident-prefix lengths tried: 0; the longest prefix r whose bytes
    plus the smallest region the remaining units need (each unit, and with
    two co-resident blocks each adjacent pair) fit the region; and the
    longest prefixes within 1/4, 1/2 and 3/4 of that prefix's bytes."""
    U = len(us)
    pb = [0]
    for u in us:
        pb.append(pb[-1] + u["bytes"])

    def need(r):
        m = [u["bytes"] for u in us[r:]]
        if slots == 2:
            m += [us[i]["bytes"] + us[i + 1]["bytes"] for i in range(r, U - 1)]
        return max(m, default=0)

    rmax = max([r for r in range(1, U + 1) if align(pb[r]) + need(r) <= region], default=0)
    cands = {0, rmax}
    for q in (1, 2, 3):
        cands.add(max(r for r in range(0, rmax + 1) if 4 * pb[r] <= q * pb[rmax]))
    return sorted(cands), pb


def eq4_objective(blocks):
    """Objective 1: Eq. 4 as printed (t_ov_1 = 0, t_in_{n+1} = 0)."""
    n = len(blocks)
    t_in = [b[1] for b in blocks] + [0]
    t_ex = [b[2] for b in blocks]
    t_out = [b[3] for b in blocks]
    total, ov_prev = 0, 0
    for i in range(1, n):            # paper's i = 2..n (0-based block i)
        ov = (t_out[i - 1] + t_in[i + 1]) - (t_ex[i] + ov_prev)
        total += max(ov, 0)
        ov_prev = ov
    return total


def arena_and_slot(model, budget, slots, activations_in_budget):
    """(arena, slot, workspace): slot bounds a piece of a split linear layer."""
    ws = workspace(model)[0]
    arena = budget - ws if activations_in_budget else budget
    if arena <= 0:
        return None
    slot = (arena // slots) // ALIGN * ALIGN
    return arena, slot, ws


def feasible(blocks, region, slots):
    """Eq. 3: consecutive blocks fit the arena together (two co-resident
    blocks); every block fits it alone."""
    for k, b in enumerate(blocks):
        if b[0] > region:
            return False
        if slots == 2 and k > 0 and blocks[k - 1][0] + b[0] > region:
            return False
    return True


def exhaustive_partition(model, budget, coef, slots=2, activations_in_budget=False,
                         objective=0, t_ex_override=None, resident_prefix=False, prefetch=False):
    """Best cut vector by brute force over all 2^(U-1) candidates.

    With resident_prefix (objective 0 only) the first r units may stay in the
    arena across inferences, r among prefix_candidates(); for each r every
    cut vector of the remaining units is tried in the region left beside the
    prefix.  Ties: smaller objective, then shorter prefix, then fewer blocks,
    then the lexicographically smallest cut vector.

    With prefetch (objective 0, two slots, no prefix) the objective is
    cyclic_time() under feasible_cyclic().

    Returns dict(n, cuts, predicted_ns, slot, arena, workspace, units,
    prefix_units, prefix_bytes) or None when no partition is feasible."""
    a = arena_and_slot(model, budget, slots, activations_in_budget)
    if a is None:
        return None
    arena, slot, ws = a
    region = arena // ALIGN * ALIGN
    us = units(model, slot, t_ex_override, region)
    if us is None:
        return None
    U = len(us)
    if resident_prefix:
        cands, pb = prefix_candidates(us, region, slots)
    else:
        cands, pb = [0], [0]
    best = None
    for r in cands:
        reg = region - (align(pb[r]) if r else 0)
        rest = U - r
        masks = range(1 << (rest - 1)) if rest > 0 else [0]
        for mask in masks:
            inner = tuple(r + c for c in range(1, rest) if mask >> (c - 1) & 1)
            cuts = ((r,) if 0 < r < U else ()) + inner
            blocks = block_costs(us, cuts, coef)
            swapped = blocks[1:] if r else blocks
            if prefetch:
                if not feasible_cyclic(blocks, reg):
                    continue
                obj = cyclic_time(blocks)
            elif not feasible(swapped, reg, slots):
                continue
            elif objective == 0:
                obj = pipeline_time(blocks, slots, prefix=r > 0)
            else:
                obj = eq4_objective(blocks)
            key = (obj, r, len(blocks), cuts)
            if best is None or key < best:
                best = key
    if best is None:
        return None
    r = best[1]
    return dict(n=best[2], cuts=list(best[3]), predicted_ns=best[0], slot=slot, arena=arena,
                workspace=ws, units=us, prefix_units=r, prefix_bytes=align(pb[r]) if r else 0)


def evaluate_cuts(model, budget, coef, cuts, slots=2, activations_in_budget=False,
                  objective=0, t_ex_override=None):
    """Predicted objective of an explicit cut vector (None if infeasible)."""
    a = arena_and_slot(model, budget, slots, activations_in_budget)
    if a is None:
        return None
    arena, slot, ws = a
    region = arena // ALIGN * ALIGN
    us = units(model, slot, t_ex_override, region)
    if us is None:
        return None
    blocks = block_costs(us, cuts, coef)
    if not feasible(blocks, region, slots):
        return None
    return pipeline_time(blocks, slots) if objective == 0 else eq4_objective(blocks)


def resident_latency_ns(model, coef, t_ex_override=None):
    """Predicted all-resident (DInf) latency: the sum of the layers' t_ex."""
    us = units(model, 1 << 62, t_ex_override)
    return sum(unit_t_ex(u, coef) for u in us)


def weight_bytes(model):
    return sum(sum(align(b) for b in layer_tensor_bytes(model, li))
               for li in range(len(model["layers"])))


# ----------------------------------------------------------- rules of Sec. 6.2.2
def block_count_rule(s, b, m=2):
    """n = ceil(m * s / b), from m blocks of size s/n co-resident within b."""
    return ceil_div(m * s, b) if isinstance(s, int) and isinstance(b, int) \
        else math.ceil(Fraction(m) * Fraction(s) / Fraction(b))


def eq1_split(demands, perf_scores, M):
    """Eq. 1: A_i = (M_i / sum M)(1 - 1/n) M + (PS_i / sum PS)(1/n) M, exact.

    Applied only when sum M_i > M; otherwise every model gets its demand."""
    n = len(demands)
    SM = sum(Fraction(x) for x in demands)
    if SM <= M:
        return [Fraction(x) for x in demands]
    SP = sum(Fraction(p) for p in perf_scores)
    return [Fraction(Mi) / SM * (1 - Fraction(1, n)) * M + Fraction(Pi) / SP * Fraction(1, n) * M
            for Mi, Pi in zip(demands, perf_scores)]


def schedule(models, urgency, M, coef, slots=2, t_ex_overrides=None):
    """Multi-DNN budget split: PS_i = u_i * latency_i / memory_i with the
    predicted DInf latency and the weight bytes; A_i floored to 256 bytes."""
    demands = [weight_bytes(m) for m in models]
    lats = [resident_latency_ns(m, coef, None if t_ex_overrides is None else t_ex_overrides[i])
            for i, m in enumerate(models)]
    ps = [Fraction(u) * Fraction(lat) / Fraction(d) for u, lat, d in zip(urgency, lats, demands)]
    shares = eq1_split(demands, ps, M)
    return [int(math.floor(a)) // ALIGN * ALIGN for a in shares]
