"""Storage tier on the host (no GPU): the weights file written by the
library, parsed here independently from its documented layout; the
direct-I/O read path against the host tensors; malformed files and bad
arguments."""
import os
import struct

import numpy as np
import pytest

import synth
from paper_2401_16757_gb300 import capi


def _model():
    """Mixed sizes: a 3-channel conv (odd byte counts), a 4096 x 4096 fp16
    linear layer (32 MiB, wider than the 16 MiB read window) and a small
    tail layer."""
    layers = [dict(op="conv", src=[-1], cin=3, cout=24, kh=3, kw=3, stride=2, pad=1, act="relu", res=None,
                   res_post=False),
              dict(op="linear", src=[0], k=4 * 4 * 24, n=4096, act="relu", res=None, res_post=False),
              dict(op="linear", src=[1], k=4096, n=4096, act="relu", res=None, res_post=False),
              dict(op="linear", src=[2], k=4096, n=10, act="none", res=None, res_post=False)]
    return dict(name="vgg16", model_id=91, dtype="f16", input=(2, 8, 8, 3), layers=layers, outputs=[3])


@pytest.fixture(scope="module")
def written(tmp_path_factory):
    m = _model()
    w = synth.gen.model_weights(m)
    flat = [np.ascontiguousarray(t).view(np.uint8).reshape(-1) for lw in w for t in lw]
    path = str(tmp_path_factory.mktemp("wf") / "model.swnw")
    capi.WeightsFile.write(path, capi.Desc(m), capi.HostWeights(w))
    return m, flat, path


def _parse(path):
    raw = open(path, "rb").read()
    magic, version, n, data0 = struct.unpack_from("<8sIIQ", raw, 0)
    entries = [struct.unpack_from("<QQ", raw, 24 + 16 * t) for t in range(n)]
    return raw, magic, version, n, data0, entries


def test_layout_matches_the_documented_format(written):
    m, flat, path = written
    raw, magic, version, n, data0, entries = _parse(path)
    assert magic == b"SWNWGT01" and version == 1
    assert n == len(flat) == 8
    assert data0 % 4096 == 0 and data0 >= 24 + 16 * n
    assert len(raw) % 4096 == 0
    prev_end = data0
    covered = np.zeros(len(raw), dtype=bool)
    covered[:24 + 16 * n] = True
    for (off, nbytes), t in zip(entries, flat):
        assert off % 4096 == 0 and off >= prev_end
        assert nbytes == t.nbytes
        assert raw[off:off + nbytes] == t.tobytes()
        covered[off:off + nbytes] = True
        prev_end = off + nbytes
    # everything that is neither header nor tensor is zero padding
    pad = np.frombuffer(raw, dtype=np.uint8)[~covered]
    assert not pad.any()


def test_read_returns_the_host_bytes(written):
    m, flat, path = written
    f = capi.WeightsFile(path, allow_buffered=True)
    info = f.info()
    assert info["n_tensors"] == len(flat)
    r = np.random.default_rng(5)
    for t, ref in enumerate(flat):
        assert f.read(t, 0, ref.nbytes).tobytes() == ref.tobytes()
        for _ in range(4):
            a = int(r.integers(0, ref.nbytes))
            b = int(r.integers(a, ref.nbytes + 1))
            assert f.read(t, a, b - a).tobytes() == ref[a:b].tobytes()
    big = flat[4]  # the 32 MiB weight: reads that span the 16 MiB window
    a = (16 << 20) - 4097
    assert f.read(4, a, 3 * 4096 + 17).tobytes() == big[a:a + 3 * 4096 + 17].tobytes()
    assert f.read(2, 5, 0).nbytes == 0
    f.close()


def test_direct_io_where_the_file_system_allows_it(written):
    m, flat, path = written
    try:
        f = capi.WeightsFile(path)
    except capi.SwapnetError as e:
        assert e.code == capi.ERR_IO
        pytest.skip("this file system refuses O_DIRECT: %s" % e)
    assert f.info()["direct"]
    assert f.read(4, 123, 4096).tobytes() == flat[4][123:123 + 4096].tobytes()


def _expect(code, fn, *a):
    with pytest.raises(capi.SwapnetError) as ei:
        fn(*a)
    assert ei.value.code == code, str(ei.value)


def test_malformed_files_are_refused(written, tmp_path):
    m, flat, path = written
    raw = bytearray(open(path, "rb").read())

    def variant(name, data):
        p = str(tmp_path / name)
        with open(p, "wb") as fh:
            fh.write(bytes(data))
        return p

    bad = bytearray(raw)
    bad[0:8] = b"NOTSWNW!"
    _expect(capi.ERR_INVALID_ARG, capi.WeightsFile, variant("magic", bad), True)
    bad = bytearray(raw)
    struct.pack_into("<I", bad, 8, 2)
    _expect(capi.ERR_INVALID_ARG, capi.WeightsFile, variant("version", bad), True)
    _expect(capi.ERR_INVALID_ARG, capi.WeightsFile, variant("ragged", raw[:-100]), True)
    bad = bytearray(raw)
    off, nbytes = struct.unpack_from("<QQ", bad, 24 + 16 * 4)
    struct.pack_into("<Q", bad, 24 + 16 * 4 + 8, len(raw))            # runs past the end
    _expect(capi.ERR_INVALID_ARG, capi.WeightsFile, variant("long", bad), True)
    bad = bytearray(raw)
    struct.pack_into("<Q", bad, 24 + 16 * 4, off + 8)                 # unaligned offset
    _expect(capi.ERR_INVALID_ARG, capi.WeightsFile, variant("unaligned", bad), True)
    bad = bytearray(raw)
    o3 = struct.unpack_from("<Q", bad, 24 + 16 * 3)[0]
    struct.pack_into("<Q", bad, 24 + 16 * 4, o3)                      # overlaps the tensor before
    _expect(capi.ERR_INVALID_ARG, capi.WeightsFile, variant("overlap", bad), True)
    _expect(capi.ERR_IO, capi.WeightsFile, str(tmp_path / "missing.swnw"), True)


def test_argument_errors(written, tmp_path):
    m, flat, path = written
    f = capi.WeightsFile(path, allow_buffered=True)
    _expect(capi.ERR_INVALID_ARG, f.read, len(flat), 0, 1)
    _expect(capi.ERR_INVALID_ARG, f.read, 0, flat[0].nbytes, 1)
    _expect(capi.ERR_INVALID_ARG, f.read, 0, 1, flat[0].nbytes)
    h = capi.C.c_void_p()
    assert capi.lib().swapnet_weights_file_open(os.fsencode(path), 6, capi.C.byref(h)) == capi.ERR_INVALID_ARG
    # a weights list that does not match the descriptor
    m2 = _model()
    m2["layers"] = m2["layers"][:3]
    m2["outputs"] = [2]
    w = synth.gen.model_weights(_model())
    rc = capi.lib().swapnet_weights_file_write(os.fsencode(str(tmp_path / "x.swnw")),
                                               capi.C.byref(capi.Desc(m2).c), capi.HostWeights(w).ptrs, 8)
    assert rc == capi.ERR_INVALID_ARG
    # an unwritable path
    _expect(capi.ERR_IO, capi.WeightsFile.write, str(tmp_path / "no" / "dir" / "x.swnw"), capi.Desc(_model()),
            capi.HostWeights(w))
    f.close()
