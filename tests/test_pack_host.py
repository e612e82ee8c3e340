"""The host packer of the packed swap variant (swapnet_pack_bf16): its
output, read by a plain NumPy decoder of the documented layout, gives back
every input word; chunks with more exceptions than a record holds go to the
overflow area.  No GPU needed."""
import numpy as np
import pytest

from paper_2401_16757_gb300 import capi

CHUNK, BODY = 4096, 6144


def _bf16(x):
    """float32 -> bf16 bit patterns (round to nearest even)."""
    u = np.asarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    return ((u + 0x7FFF + ((u >> 16) & 1)) >> 16).astype(np.uint16)


def _body_off(chunks):
    return (16 + 16 * chunks + 127) // 128 * 128


def _unpack(buf, n):
    x0 = int(buf[0])
    assert x0 <= 240 and not buf[1:16].any()
    chunks = n // CHUNK
    hdrs = buf[16:16 + 16 * chunks].reshape(chunks, 16)
    off = _body_off(chunks)
    assert not buf[16 + 16 * chunks:off].any()
    bodies = buf[off:off + chunks * BODY].reshape(chunks, BODY)
    overflow = buf[off + chunks * BODY:]
    out = np.empty((chunks, CHUNK), dtype=np.uint16)
    raw = 0
    for c in range(chunks):
        h = hdrs[c]
        if h[0] == 0xFF:
            r = int(h[4:8].view(np.uint32)[0])
            out[c] = overflow[r * 2 * CHUNK:(r + 1) * 2 * CHUNK].view(np.uint16)
            assert not bodies[c].any()
            raw += 1
            continue
        codes = bodies[c, :CHUNK // 2]
        code = np.empty(CHUNK, dtype=np.uint8)
        code[0::2] = codes & 15
        code[1::2] = codes >> 4
        sm = bodies[c, CHUNK // 2:].astype(np.uint16)
        x = (x0 + code).astype(np.uint16)
        k = int(h[0])
        assert k <= 4
        pos = h[4:12].view(np.uint16)[:k]
        assert np.array_equal(np.flatnonzero(code == 15), pos)   # every escape listed, in order
        x[pos] = h[12:12 + k]
        out[c] = ((sm & 0x80) << 8) | (x << 7) | (sm & 0x7F)
    assert overflow.size == raw * 2 * CHUNK
    return out.reshape(-1), raw


def test_round_trip_of_llm_shaped_weights():
    """N(0, 0.02) weights (the decoder's initialisation): exact round trip,
    about (6144 + 16) / 8192 of the bytes."""
    r = np.random.default_rng(7)
    w = _bf16(r.normal(0.0, 0.02, size=CHUNK * 37))
    buf = capi.pack_bf16(w)
    back, raw = _unpack(buf, w.size)
    assert np.array_equal(back, w)
    assert buf.size == _body_off(37) + 37 * BODY + raw * 2 * CHUNK
    assert raw <= 2
    assert buf.size < 0.76 * w.nbytes


def test_escapes_up_to_four_per_chunk_then_overflow():
    """Exponents outside the table: zeros, huge values, infinities and NaN
    (exponent 255), negative zero.  A chunk with 4 of them keeps them in its
    header; one with 5 is stored unpacked."""
    r = np.random.default_rng(8)
    # fifteen exponents (108..122), the whole window, so only the planted
    # values escape
    n = CHUNK * 4
    w = ((r.integers(0, 2, n) << 15) | (r.integers(108, 123, n) << 7) | r.integers(0, 128, n)).astype(np.uint16)
    specials = np.array([0x0000, 0x8000, 0x7F80, 0x7FC1, 0x4700], dtype=np.uint16)
    w[[5, 700, 4095]] = specials[:3]                       # chunk 0: 3 escapes
    w[CHUNK + np.array([0, 1, 2, 4095])] = specials[1:]    # chunk 1: 4 escapes
    w[2 * CHUNK + np.array([9, 99, 999, 2000, 3000])] = specials   # chunk 2: 5 -> overflow
    buf = capi.pack_bf16(w)
    back, raw = _unpack(buf, w.size)
    assert np.array_equal(back, w)
    assert raw == 1
    assert list(buf[16:16 + 4 * 16].reshape(4, 16)[:, 0]) == [3, 4, 0xFF, 0]


def test_one_exponent_and_every_exponent():
    """A constant tensor (one exponent of the window used) and a tensor
    holding all 256 exponents (most of them escapes: chunks overflow)."""
    ones = np.full(CHUNK * 2, 0x3F80, dtype=np.uint16)
    back, raw = _unpack(capi.pack_bf16(ones), ones.size)
    assert np.array_equal(back, ones) and raw == 0
    every = (np.arange(CHUNK * 3, dtype=np.uint32) * 0x9E37 % 65536).astype(np.uint16)
    back, raw = _unpack(capi.pack_bf16(every), every.size)
    assert np.array_equal(back, every) and raw == 3


def test_argument_errors():
    w = np.zeros(CHUNK, dtype=np.uint16)
    used = capi.C.c_uint64()
    lib = capi.lib()
    assert lib.swapnet_pack_bf16(capi.C.c_void_p(w.ctypes.data), CHUNK + 8, None, 0,
                                 capi.C.byref(used)) == capi.ERR_UNSUPPORTED
    assert lib.swapnet_pack_bf16(capi.C.c_void_p(w.ctypes.data), 0, None, 0, capi.C.byref(used)) == \
        capi.ERR_UNSUPPORTED
    assert lib.swapnet_pack_bf16(None, CHUNK, None, 0, capi.C.byref(used)) == capi.ERR_INVALID_ARG
    assert lib.swapnet_pack_bf16(capi.C.c_void_p(w.ctypes.data), CHUNK, None, 0, capi.C.byref(used)) == capi.OK
    small = np.empty(used.value - 1, dtype=np.uint8)
    assert lib.swapnet_pack_bf16(capi.C.c_void_p(w.ctypes.data), CHUNK, capi.C.c_void_p(small.ctypes.data),
                                 small.size, capi.C.byref(used)) == capi.ERR_INVALID_ARG


def test_window_at_the_ends_of_the_exponent_range():
    """Exponents 241..255 only: the window starts at 240 (x0 + 15 must fit a
    byte), so exponent 255 escapes; exponents 0..14: the window starts at 0."""
    r = np.random.default_rng(9)
    n = CHUNK * 2
    top = ((r.integers(241, 256, n) << 7) | r.integers(0, 128, n)).astype(np.uint16)
    buf = capi.pack_bf16(top)
    assert buf[0] == 240
    back, _ = _unpack(buf, n)
    assert np.array_equal(back, top)
    low = ((r.integers(0, 2, n) << 15) | (r.integers(0, 15, n) << 7) | r.integers(0, 128, n)).astype(np.uint16)
    buf = capi.pack_bf16(low)
    assert buf[0] == 0
    back, raw = _unpack(buf, n)
    assert np.array_equal(back, low) and raw == 0


@pytest.mark.parametrize("seed", range(6))
def test_round_trip_of_mixed_distributions(seed):
    """Random mixtures: scaled normals of several widths, exact zeros,
    subnormals, infinities and NaNs, in random proportions and positions;
    every word comes back and the size matches the layout."""
    r = np.random.default_rng(100 + seed)
    chunks = int(r.integers(1, 9))
    n = CHUNK * chunks
    sigma = 10.0 ** r.uniform(-4, 1)
    w = _bf16(r.normal(0.0, sigma, n))
    for pattern, frac in ((0x0000, 1e-3), (0x8000, 1e-4), (0x0001, 1e-4), (0x7F80, 1e-5), (0x7FC1, 1e-5)):
        pick = r.random(n) < frac * 10 ** r.uniform(-1, 1)
        w[pick] = pattern
    buf = capi.pack_bf16(w)
    back, raw = _unpack(buf, n)
    assert np.array_equal(back, w)
    assert buf.size == _body_off(chunks) + chunks * BODY + raw * 2 * CHUNK
