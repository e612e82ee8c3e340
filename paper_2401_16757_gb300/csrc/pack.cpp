// Host side of the packed swap variant: building the packed form of a bf16
// tensor (the layout is described in pack.h) and the C ABI entry point that
// exposes it.
#include <algorithm>
#include <array>
#include <cstring>
#include <thread>

#include "internal.h"
#include "pack.h"

namespace swapnet {

namespace {

// f(lo, hi) over [0, n) in up to `threads` contiguous parts, one thread each
template <typename F>
void parallel_for(uint64_t n, int threads, F f) {
  const int t = (int)std::max<uint64_t>(1, std::min<uint64_t>((uint64_t)std::max(threads, 1), n));
  if (t == 1) {
    f(0, n);
    return;
  }
  std::vector<std::thread> pool;
  pool.reserve(t);
  for (int i = 0; i < t; ++i) pool.emplace_back([=, &f] { f(n * i / t, n * (i + 1) / t); });
  for (std::thread& th : pool) th.join();
}

inline uint32_t exponent(uint16_t w) { return (w >> 7) & 0xffu; }

}  // namespace

PackInfo pack_prepare(const uint16_t* src, uint64_t n, int threads) {
  PackInfo info;
  const uint64_t chunks = n / kPkChunk;
  // exponent histogram
  const int t = (int)std::max<uint64_t>(1, std::min<uint64_t>((uint64_t)std::max(threads, 1), chunks));
  std::vector<std::array<uint64_t, 256>> part(t);
  for (auto& h : part) h.fill(0);
  std::vector<std::thread> pool;
  for (int i = 0; i < t; ++i)
    pool.emplace_back([&, i] {
      const uint64_t lo = n * i / t, hi = n * (i + 1) / t;
      std::array<uint64_t, 256>& h = part[i];
      for (uint64_t e = lo; e < hi; ++e) ++h[exponent(src[e])];
    });
  for (std::thread& th : pool) th.join();
  std::array<uint64_t, 256> hist{};
  for (const auto& h : part)
    for (int x = 0; x < 256; ++x) hist[x] += h[x];
  // the window of 15 consecutive exponents x0 .. x0 + 14 that holds the
  // most elements (the smallest x0 among equals; x0 <= 240, so that x0 + 15
  // still fits a byte)
  int x0 = 0;
  uint64_t best = 0, run = 0;
  for (int x = 0; x < 15; ++x) run += hist[x];
  best = run;
  for (int b = 1; b <= 240; ++b) {
    run += hist[b + 14] - hist[b - 1];
    if (run > best) {
      best = run;
      x0 = b;
    }
  }
  std::memset(info.code, 15, sizeof(info.code));
  std::memset(info.exp, 0, sizeof(info.exp));
  info.exp[0] = (uint8_t)x0;
  for (int c = 0; c < 15; ++c) info.code[x0 + c] = (uint8_t)c;
  // chunks with more escapes than a record holds go to the overflow area
  std::vector<uint8_t> raw(chunks, 0);
  parallel_for(chunks, threads, [&](uint64_t lo, uint64_t hi) {
    for (uint64_t c = lo; c < hi; ++c) {
      const uint16_t* w = src + c * kPkChunk;
      int esc = 0;
      for (int e = 0; e < kPkChunk; ++e) esc += info.code[exponent(w[e])] == 15;
      raw[c] = esc > kPkMaxEsc;
    }
  });
  info.overflow.assign(chunks, UINT32_MAX);
  uint32_t r = 0;
  for (uint64_t c = 0; c < chunks; ++c)
    if (raw[c]) info.overflow[c] = r++;
  info.bytes = pk_body_off(chunks) + chunks * (uint64_t)kPkBody + r * kPkChunkBytes;
  return info;
}

void pack_write(const uint16_t* src, uint64_t n, const PackInfo& info, uint8_t* dst, int threads) {
  const uint64_t chunks = n / kPkChunk;
  const uint64_t body_off = pk_body_off(chunks);
  std::memset(dst, 0, body_off);
  std::memcpy(dst, info.exp, 16);
  uint8_t* bodies = dst + body_off;
  uint8_t* overflow = bodies + chunks * (uint64_t)kPkBody;
  parallel_for(chunks, threads, [&](uint64_t lo, uint64_t hi) {
    for (uint64_t c = lo; c < hi; ++c) {
      const uint16_t* w = src + c * kPkChunk;
      uint8_t* hdr = dst + 16 + kPkHeader * c;
      uint8_t* body = bodies + c * (uint64_t)kPkBody;
      std::memset(body, 0, kPkBody);
      if (info.overflow[c] != UINT32_MAX) {
        const uint32_t r = info.overflow[c];
        hdr[0] = (uint8_t)kPkRaw;
        std::memcpy(hdr + 4, &r, 4);
        std::memcpy(overflow + (uint64_t)r * kPkChunkBytes, w, kPkChunkBytes);
        continue;
      }
      uint8_t* codes = body;
      uint8_t* sm = body + kPkChunk / 2;
      int k = 0;
      for (int e = 0; e < kPkChunk; ++e) {
        const uint32_t x = exponent(w[e]);
        const uint8_t cd = info.code[x];
        codes[e >> 1] |= (uint8_t)(cd << ((e & 1) * 4));
        sm[e] = (uint8_t)(((w[e] >> 8) & 0x80u) | (w[e] & 0x7fu));
        if (cd == 15) {  // at most kPkMaxEsc here (pack_prepare sent the rest to the overflow area)
          const uint16_t pos = (uint16_t)e;
          std::memcpy(hdr + 4 + 2 * k, &pos, 2);
          hdr[12 + k] = (uint8_t)x;
          ++k;
        }
      }
      hdr[0] = (uint8_t)k;
    }
  });
}

}  // namespace swapnet

extern "C" int swapnet_pack_bf16(const void* src, uint64_t n_elems, void* dst, uint64_t dst_bytes,
                                 uint64_t* used_bytes) {
  return swapnet::guard_abi([&]() -> int {
    if (!src || !used_bytes) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null argument");
    if (n_elems == 0 || n_elems % swapnet::kPkChunk)
      SN_FAIL(SWAPNET_ERR_UNSUPPORTED, "packing: the element count must be a positive multiple of 4096");
    const int threads = (int)std::min(32u, std::max(1u, std::thread::hardware_concurrency()));
    try {
      const swapnet::PackInfo info = swapnet::pack_prepare(static_cast<const uint16_t*>(src), n_elems, threads);
      *used_bytes = info.bytes;
      if (!dst) return SWAPNET_OK;
      if (dst_bytes < info.bytes) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "packing: destination too small");
      swapnet::pack_write(static_cast<const uint16_t*>(src), n_elems, info, static_cast<uint8_t*>(dst), threads);
    } catch (...) {  // allocation or thread creation
      SN_FAIL(SWAPNET_ERR_OOM, "packing: host resources exhausted");
    }
    return SWAPNET_OK;
  });
}
