"""Host-side pieces of bench.py's measurement (no GPU): the algorithmic byte
counts behind the roofline against the oracle's own shape bookkeeping, and
the reference arm's JSON line."""
import json
import os
import subprocess
import sys

import numpy as np
import pytest

import bench
import synth
from oracle import plan as OP

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.mark.parametrize("name,kw", [("resnet50", dict(batch=1)), ("vgg16", dict(batch=16)),
                                     ("yolov3", dict(batch=1)), ("mlp6", dict(batch=8))])
def test_algorithmic_bytes_match_the_oracle_shapes(name, kw):
    m = synth.arch.MODELS[name](**kw)
    shapes = OP.out_shapes(m)
    es = {"f32": 4, "f16": 2, "bf16": 2}[m["dtype"]]
    units = [dict(layer=i, rows=0, bytes=sum(OP.align(b) for b in OP.layer_tensor_bytes(m, i)))
             for i in range(len(m["layers"]))]
    got = bench.unit_algorithmic_bytes(m, units)

    def nbytes(i):
        return int(np.prod(tuple(m["input"]) if i == -1 else shapes[i])) * es

    for i, L in enumerate(m["layers"]):
        srcs = list(L["src"]) + ([L["res"]] if L.get("res") is not None else [])
        assert got[i] == units[i]["bytes"] + sum(nbytes(s) for s in srcs) + nbytes(i), i


def test_linear_pieces_count_their_share_of_the_output():
    m = synth.arch.vgg16(batch=1)
    fc1 = next(i for i, L in enumerate(m["layers"]) if L["op"] == "linear")
    n = m["layers"][fc1]["n"]
    whole = bench.unit_algorithmic_bytes(m, [dict(layer=fc1, rows=0, bytes=0)])[0]
    half = bench.unit_algorithmic_bytes(m, [dict(layer=fc1, rows=n // 2, bytes=0)])[0]
    out = n * 2  # batch 1, fp16
    assert whole - half == out // 2


def test_reference_arm_prints_one_oracle_line():
    """`--impl reference` times the oracle on the host: one JSON line with the
    reference fields (the 6-layer MLP: one step takes milliseconds)."""
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--config", "mlp6",
                        "--steps", "1", "--warmup", "0"], capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    line = json.loads(r.stdout.strip().splitlines()[-1])
    assert line["impl"] == "reference"
    assert line["cpu_baseline"]["kind"] == "oracle"
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["e2e"]["d2h_bytes_per_step"] == 0
    assert line["value"] > 0 and line["unit"] == line["e2e"]["unit"]


def _rank_group_worker(rank, port, out_dir):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE="2")
    sys.path.insert(0, ROOT)
    import bench as b
    g = b.RankGroup(2, backend="gloo")
    g.barrier()
    slowest = g.max(10.0 + 5.0 * rank)  # this rank's "timed" milliseconds
    g.barrier()
    g.close()
    with open(os.path.join(out_dir, "rank%d" % rank), "w") as fh:
        fh.write(repr(slowest))


def test_rank_group_takes_the_slowest_rank_over_gloo(tmp_path):
    """Replicas (N > 1): two ranks on the CPU (gloo) bracket the timed region
    with barriers and both see the slowest rank's time, from which bench.py
    computes the whole-job throughput; one rank needs no process group."""
    import socket
    import torch.multiprocessing as mp
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        port = s.getsockname()[1]
    mp.spawn(_rank_group_worker, args=(port, str(tmp_path)), nprocs=2, join=True)
    got = [float(open(os.path.join(str(tmp_path), "rank%d" % r)).read()) for r in range(2)]
    assert got == [15.0, 15.0]
    single = bench.RankGroup(1)
    assert single.max(3.5) == 3.5 and single.dist is None
    single.barrier()
    single.close()


def test_reference_arm_other_ranks_exit_quietly():
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--config", "mlp6",
                        "--steps", "1", "--warmup", "0"], capture_output=True, text=True, timeout=600, env=env)
    assert r.returncode == 0 and r.stdout.strip() == ""


def test_host_placement_reads_the_node_of_a_page():
    """The link record's placement reading (a host-side query, no GPU
    setting): the online NUMA nodes as the kernel lists them, and the node
    of a touched page of ordinary memory, which must be one of them."""
    import ctypes
    buf = (ctypes.c_uint8 * (1 << 16))()
    ctypes.memset(buf, 1, 1 << 16)
    got = bench.host_placement(ctypes.addressof(buf))
    online = got["numa_nodes_online"]
    if online is None:
        pytest.skip("no NUMA information on this host")
    nodes = set()
    for part in online.split(","):
        lo, _, hi = part.partition("-")
        nodes.update(range(int(lo), int(hi or lo) + 1))
    if "pinned_page_node" in got and got["pinned_page_node"] is not None:
        assert got["pinned_page_node"] in nodes
