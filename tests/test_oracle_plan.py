"""Pins of the partitioning oracle: the paper's printed block counts and
Eq. 1 example, closed forms of the pipeline recurrence, an independent
event simulation, and invariants of the workspace and unit splitting."""
import itertools
import os
from fractions import Fraction

import numpy as np
import pytest

from oracle import plan as P
import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _golden_lines(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return [l.split("#")[0].strip() for l in f if l.split("#")[0].strip()]


def test_block_count_rule_matches_paper():
    for line in _golden_lines("block_count.txt"):
        s, b, m, n = (int(v) for v in line.split())
        assert P.block_count_rule(s, b, m) == n


def test_eq1_worked_example():
    kv = dict(t.split("=") for t in _golden_lines("eq1_examples.txt")[0].split())
    sumM, M = Fraction(kv["sumM"]), Fraction(kv["M"])
    # proportional share of model i = M_i / sum M * M = (2/3) M_i
    assert M / sumM == Fraction(kv["proportional_fraction"])
    # With equal performance scores the second term is M/n each; the first
    # term is (1 - 1/n) of the proportional share.
    demands = [Fraction(1, 2), Fraction(1, 2), Fraction(1, 2)]
    A = P.eq1_split(demands, [1, 1, 1], M)
    assert sum(A) == M
    assert A[0] == Fraction(2, 3) * demands[0] * Fraction(2, 3) + M / 9


def test_eq1_selfdriving_budgets_consistent():
    kv = dict(t.split("=") for t in _golden_lines("eq1_examples.txt")[1].split())
    M = int(kv["M"])
    sizes = [int(v) for v in kv["sizes"].split(",")]
    budgets = [int(v) for v in kv["budgets"].split(",")]
    assert sum(budgets) == M
    n, S = len(sizes), sum(sizes)
    first = [Fraction(s, S) * (1 - Fraction(1, n)) * M for s in sizes]
    # every printed budget is at least its proportional term; the rest is the
    # performance-score term, whose shares must sum to one
    shares = [(b - f) / (Fraction(M) / n) for b, f in zip(budgets, first)]
    assert all(0 <= s <= 1 for s in shares)
    assert abs(float(sum(shares)) - 1.0) < 0.01
    # Eq. 1 with those shares as performance scores gives the printed budgets
    A = P.eq1_split(sizes, shares, M)
    assert all(abs(float(a) - b) < 1.0 for a, b in zip(A, budgets))


def _one_linear(mid, n):
    return dict(name="mlp6", model_id=mid, dtype="f32", input=(1, 1, 1, 256), outputs=[0],
                layers=[dict(op="linear", src=[-1], k=256, n=n, act="none", res=None, res_post=False,
                             bias=False)])


def test_schedule_performance_scores_hand_worked():
    """schedule(): PS_i = u_i * latency_i / M_i (Sec. 6.2.2 beside Eq. 1),
    hand-worked.  Model A holds 256 x 256 fp32 weights (262144 B), model B
    256 x 512 (524288 B); their DInf latencies are set to 1000 and 4000 ns;
    the budget is M = 393216 B, half the 786432 B demanded (n = 2).
      u = (1, 1): PS_A = 1000/262144, PS_B = 4000/524288 = 2 PS_A, so the
        score shares are 1/3 and 2/3 and
        A_A = (1/3)(1/2)M + (1/3)(1/2)M = 65536 + 65536 = 131072,
        A_B = (2/3)(1/2)M + (2/3)(1/2)M = 262144.
      u = (3, 1): score shares 3/5 and 2/5:
        A_A = 65536 + 117964.8 -> 183296 after flooring to 256 bytes,
        A_B = 131072 + 78643.2 -> 209664.
    PS = u * M / latency would give A_A = 196608 for u = (1, 1), and
    PS = u * latency (no division by the memory) 104857.6 -> 104704."""
    ms = [_one_linear(81, 256), _one_linear(82, 512)]
    assert [P.weight_bytes(m) for m in ms] == [262144, 524288]
    coef = P.Coef(2_500_000, 0, 2000, 0)
    ovr = [[1000], [4000]]
    assert P.schedule(ms, [1, 1], 393216, coef, t_ex_overrides=ovr) == [131072, 262144]
    assert P.schedule(ms, [3, 1], 393216, coef, t_ex_overrides=ovr) == [183296, 209664]


def test_eq1_within_budget_returns_demands():
    assert P.eq1_split([3, 4], [1, 1], 10) == [3, 4]


def _blocks(t_in, t_ex, t_out, n):
    return [(0, t_in, t_ex, t_out)] * n


@pytest.mark.parametrize("t_in,t_ex", [(5, 9), (9, 5), (7, 7), (1, 100), (100, 1)])
@pytest.mark.parametrize("n", [1, 2, 3, 7])
def test_pipeline_closed_forms(t_in, t_ex, n):
    # two slots, free release: one copy ahead of execution
    two = P.pipeline_time(_blocks(t_in, t_ex, 0, n), 2)
    assert two == (t_in + n * t_ex if t_ex >= t_in else n * t_in + t_ex)
    # one slot: strictly serial
    assert P.pipeline_time(_blocks(t_in, t_ex, 0, n), 1) == n * (t_in + t_ex)


def _simulate(blocks, slots):
    """Event simulation with explicit resources: a copy engine, a compute
    engine and `slots` arena slots, each with the time it becomes free."""
    copy_free = comp_free = 0
    slot_free = [0] * slots
    prev_exec_end = 0
    for k, (_, t_in, t_ex, t_out) in enumerate(blocks):
        s = k % slots
        start_copy = max(copy_free, slot_free[s])
        copy_free = start_copy + t_in
        start_exec = max(comp_free, copy_free, prev_exec_end)
        comp_free = prev_exec_end = start_exec + t_ex
        slot_free[s] = comp_free + t_out
    return comp_free


def test_pipeline_matches_event_simulation():
    r = np.random.default_rng(0)
    for _ in range(2000):
        n = int(r.integers(1, 9))
        blocks = [(0, int(r.integers(0, 50)), int(r.integers(0, 50)), int(r.integers(0, 20)))
                  for _ in range(n)]
        for slots in (1, 2):
            assert P.pipeline_time(blocks, slots) == _simulate(blocks, slots)


def test_eq4_hand_example():
    # three blocks (t_in, t_ex, t_out): (4,3,1), (6,2,1), (5,8,2)
    blocks = [(0, 4, 3, 1), (0, 6, 2, 1), (0, 5, 8, 2)]
    # i=2: ov = (1 + 5) - (2 + 0) = 4 ; i=3: ov = (1 + 0) - (8 + 4) = -11
    assert P.eq4_objective(blocks) == 4
    assert P.eq4_objective(blocks[:1]) == 0


def _uniform_model(nl, width, dtype="f16"):
    layers = [dict(op="linear", src=[i - 1], k=width, n=width, act="relu", res=None, res_post=False)
              for i in range(nl)]
    return dict(name="u", model_id=50, dtype=dtype, input=(4, 1, 1, width), layers=layers,
                outputs=[nl - 1])


def test_workspace_mlp_is_two_buffers():
    # the 6-layer MLP needs exactly two activation buffers (ping-pong)
    m = synth.arch.mlp6()
    ws, offs, ob, oo = P.workspace(m)
    assert ws == 2 * 8 * 1024 * 4
    assert sorted(set(offs.values())) == [0, 8 * 1024 * 4]
    assert ob == 8 * 1024 * 4 and oo == {5: 0}


@pytest.mark.parametrize("name", ["resnet50", "yolov3", "vgg16"])
def test_workspace_no_live_overlap_and_first_fit(name):
    m = synth.arch.MODELS[name]()
    ws, offs, _, _ = P.workspace(m)
    shapes = P.out_shapes(m)
    es = P.ES[m["dtype"]]
    nl = len(m["layers"])
    last = list(range(nl))
    first = list(range(nl))   # earliest step a layer may run: after its last producer
    for j, L in enumerate(m["layers"]):
        refs = [i for i in list(L["src"]) + ([L["res"]] if L.get("res") is not None else []) if i >= 0]
        for i in refs:
            last[i] = max(last[i], j)
        if L["op"] in ("conv", "linear") and refs:
            first[j] = min(j, max(refs) + 1)
    size = {i: P.align(int(np.prod(shapes[i])) * es) for i in offs}
    items = sorted(offs)
    for a, b in itertools.combinations(items, 2):
        live = first[a] <= last[b] and first[b] <= last[a]
        if live:
            assert offs[a] + size[a] <= offs[b] or offs[b] + size[b] <= offs[a]
    assert ws == max(offs[i] + size[i] for i in items)
    # first fit: no lower aligned offset was free when the tensor was placed
    for i in items:
        earlier = [j for j in items if j < i and first[j] <= last[i] and first[i] <= last[j]]
        for o in range(0, offs[i], 256 * max(1, offs[i] // 256 // 64)):
            clash = any(not (o + size[i] <= offs[j] or offs[j] + size[j] <= o) for j in earlier)
            assert clash


def test_units_split_vgg_fc1():
    m = synth.arch.vgg16()
    wb = P.weight_bytes(m)
    budget = wb // 4 // 256 * 256
    arena, slot, _ = P.arena_and_slot(m, budget, 2, False)
    us = P.units(m, slot, None, arena // 256 * 256)
    fc1 = [u for u in us if u["layer"] == 18]
    assert len(fc1) > 1
    assert sum(u["rows"] for u in fc1) == 4096
    assert all(u["rows"] % 128 == 0 for u in fc1)
    assert all(u["bytes"] <= slot for u in us)
    assert [u["row0"] for u in fc1] == list(np.cumsum([0] + [u["rows"] for u in fc1[:-1]]))
    assert sum(u["flops"] for u in fc1) == 2 * 25088 * 4096


def test_units_infeasible_when_conv_too_large():
    m = synth.arch.resnet50()
    assert P.units(m, 1 << 20) is None


def test_exhaustive_respects_rules():
    r = np.random.default_rng(1)
    coef = P.Coef(alpha_as=2_000_000, beta_ns=500, gamma_as=3000, eta_ns=50)
    for _ in range(20):
        nl = int(r.integers(2, 8))
        m = _uniform_model(nl, 256)
        s = P.weight_bytes(m)
        budget = int(r.integers(s // nl * 2, s * 2 + 1))
        res = P.exhaustive_partition(m, budget, coef)
        if res is None:
            us = P.units(m, budget // 2 // 256 * 256, None, budget // 256 * 256)
            assert us is None or max(u["bytes"] for u in us) > budget // 2
            continue
        # two co-resident blocks within the budget: summing s_i + s_{i+1} <= b
        # over the n-1 neighbour pairs gives 2s - s_1 - s_n <= (n-1) b, so
        # n >= ceil(2 s / b) - 1 (the paper's rule, less the two end blocks)
        assert res["n"] >= P.block_count_rule(s, budget) - 1
        # the optimum is no worse than every feasible alternative
        for cuts in itertools.combinations(range(1, nl), res["n"] - 1):
            v = P.evaluate_cuts(m, budget, coef, list(cuts))
            assert v is None or v >= res["predicted_ns"]


def test_rule_count_is_fewest_feasible_blocks():
    # balanced layers: the fewest blocks of any feasible partition equals the
    # paper's n = ceil(2 s / b); the exact objective may pick more blocks
    # (a smaller first block shortens the pipeline fill)
    coef = P.Coef(alpha_as=1000, beta_ns=100, gamma_as=100_000, eta_ns=0)
    m = _uniform_model(6, 512)
    s = P.weight_bytes(m)
    # the rule is for models larger than the budget (s > b); when the model
    # fits, one block suffices
    for per_block in (1, 2):
        budget = 2 * per_block * (s // 6)
        fewest = min(len(c) + 1 for k in range(6) for c in itertools.combinations(range(1, 6), k)
                     if P.evaluate_cuts(m, budget, coef, list(c)) is not None)
        assert fewest == P.block_count_rule(s, budget) == 6 // per_block
        assert P.exhaustive_partition(m, budget, coef)["n"] >= fewest
    assert P.evaluate_cuts(m, s, coef, []) is not None   # one block fits when s <= b


def test_pipeline_with_resident_prefix_hand_worked():
    """Resident prefix (extension): block 0 runs from t = 0 without a copy
    and never frees room, so block 2 may start copying as soon as block 1's
    copy ends.  Worked by hand: prefix t_ex 5; blocks (t_in, t_ex) = (3, 2),
    (4, 1), (2, 2); two slots.  Copies end at 3, 7, 9 (block 3 waits for
    block 1's release at 7); executions end at 7, 8, 11."""
    blocks = [(0, 0, 5, 0), (10, 3, 2, 0), (10, 4, 1, 0), (10, 2, 2, 0)]
    assert P.pipeline_time(blocks, 2, prefix=True) == 11
    # read as an ordinary first block the same numbers make block 2 wait for
    # block 0's release at 5: a different (later) finish
    assert P.pipeline_time(blocks, 2) == 13
    # one slot: every copy waits for the previous swapped block's release
    assert P.pipeline_time(blocks, 1, prefix=True) == max(5, 3) + 2 + 4 + 1 + 2 + 2


def test_prefix_candidates_rule():
    us = [dict(bytes=b) for b in (256, 512, 256, 1024, 512)]
    cands, pb = P.prefix_candidates(us, region=2048, slots=2)
    # the remaining units always include the pair 1024 + 512 = 1536 while
    # unit 3 is swapped: r = 1 (256 bytes) fits (1792), r = 2 (768) does not
    # (2304); r = 4 leaves 512 beside 2048 bytes of prefix: 2560 > 2048
    assert cands == [0, 1]
    assert pb == [0, 256, 768, 1024, 2048, 2560]
    cands1, _ = P.prefix_candidates(us, region=2048, slots=1)
    # one slot: the rest needs only its largest unit; r = 3 leaves 1024 beside
    # 1024 bytes of prefix (exactly 2048), r = 4 would need 2048 + 512
    assert max(cands1) == 3


def test_cyclic_pipeline_hand_worked():
    """First-block prefetch (steady state): blocks (t_in, t_ex) = (4, 2),
    (3, 5), (2, 1), (1, 3), t_out = 0, two slots.  Block 0 is present at
    t = 0 and ends at 2; copies of blocks 1-3 end at 3, 5 (block 2 waits
    for block 0's release at 2: no wait), 9 (block 3 waits for block 1's
    release at 8); executions end at 8, 9, 12.  Four blocks: the next
    block 0 shares block 2's place, so its copy starts at max(9, 9) and
    ends at 13, after the last execution: 13.  The same blocks run cold
    (block 0 copied first) finish at 16."""
    blocks = [(10, 4, 2, 0), (10, 3, 5, 0), (10, 2, 1, 0), (10, 1, 3, 0)]
    assert P.cyclic_time(blocks) == 13
    assert P.pipeline_time(blocks, 2) == 16
    # three blocks: block 2 shares block 0's place; its release at 9 plus 4
    assert P.cyclic_time(blocks[:3]) == 13
    # one block: execute, then copy it in again for the next inference
    assert P.cyclic_time(blocks[:1]) == 2 + 4


def test_cyclic_pipeline_invariants():
    r = np.random.default_rng(17)
    for _ in range(300):
        n = int(r.integers(1, 7))
        blocks = [(int(r.integers(1, 100)), int(r.integers(0, 50)), int(r.integers(0, 50)), 0) for _ in range(n)]
        t = P.cyclic_time(blocks)
        # one copy engine and one execution stream: both chains fit in a period
        assert t >= sum(b[1] for b in blocks) and t >= sum(b[2] for b in blocks)
        # a first block that costs nothing to copy: the cold pipeline exactly
        free0 = [(blocks[0][0], 0) + blocks[0][2:]] + blocks[1:]
        assert P.cyclic_time(free0) == P.pipeline_time(free0, 2)
        # prefetching never loses to running cold (the copy moves, it does not grow)
        assert t <= P.pipeline_time(blocks, 2) + blocks[0][1]


def test_cyclic_feasibility_adds_the_wrap_pair():
    # even count: the last block and the next first block are co-resident
    # (every adjacent pair fits; only the wrap pair 424 + 624 does not)
    wrap_fails = [(624, 0, 0, 0), (400, 0, 0, 0), (600, 0, 0, 0), (424, 0, 0, 0)]
    assert P.feasible(wrap_fails, 1024, 2) is True
    assert P.feasible_cyclic(wrap_fails, 1024) is False
    assert P.feasible_cyclic([(600, 0, 0, 0), (400, 0, 0, 0), (600, 0, 0, 0), (424, 0, 0, 0)], 1024) is True
    # odd count: the last block sits where the first does; only Eq. 3 applies
    assert P.feasible_cyclic([(600, 0, 0, 0), (400, 0, 0, 0), (600, 0, 0, 0)], 1024) is True
