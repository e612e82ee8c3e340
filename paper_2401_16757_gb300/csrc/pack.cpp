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
  // the 15 most frequent exponents (ties: the smaller exponent first)
  std::array<int, 256> order;
  for (int x = 0; x < 256; ++x) order[x] = x;
  std::stable_sort(order.begin(), order.end(), [&](int a, int b) { return hist[a] > hist[b]; });
  std::memset(info.code, 15, sizeof(info.code));
  std::memset(info.exp, 0, sizeof(info.exp));
  for (int c = 0; c < 15; ++c) {
    info.exp[c] = (uint8_t)order[c];
    if (hist[order[c]]) info.code[order[c]] = (uint8_t)c;
  }
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
  info.bytes = kPkHeader + chunks * (uint64_t)kPkRecord + r * kPkChunkBytes;
  return info;
}

void pack_write(const uint16_t* src, uint64_t n, const PackInfo& info, uint8_t* dst, int threads) {
  const uint64_t chunks = n / kPkChunk;
  std::memcpy(dst, info.exp, 16);
  uint8_t* records = dst + kPkHeader;
  uint8_t* overflow = records + chunks * (uint64_t)kPkRecord;
  parallel_for(chunks, threads, [&](uint64_t lo, uint64_t hi) {
    for (uint64_t c = lo; c < hi; ++c) {
      const uint16_t* w = src + c * kPkChunk;
      uint8_t* rec = records + c * (uint64_t)kPkRecord;
      std::memset(rec, 0, kPkRecord);
      if (info.overflow[c] != UINT32_MAX) {
        const uint32_t r = info.overflow[c];
        rec[0] = (uint8_t)kPkRaw;
        std::memcpy(rec + 4, &r, 4);
        std::memcpy(overflow + (uint64_t)r * kPkChunkBytes, w, kPkChunkBytes);
        continue;
      }
      uint8_t* codes = rec + 16;
      uint8_t* sm = rec + 16 + kPkChunk / 2;
      int k = 0;
      for (int e = 0; e < kPkChunk; ++e) {
        const uint32_t x = exponent(w[e]);
        const uint8_t cd = info.code[x];
        codes[e >> 1] |= (uint8_t)(cd << ((e & 1) * 4));
        sm[e] = (uint8_t)(((w[e] >> 8) & 0x80u) | (w[e] & 0x7fu));
        if (cd == 15) {  // at most kPkMaxEsc here (pack_prepare sent the rest to the overflow area)
          const uint16_t pos = (uint16_t)e;
          std::memcpy(rec + 4 + 2 * k, &pos, 2);
          rec[12 + k] = (uint8_t)x;
          ++k;
        }
      }
      rec[0] = (uint8_t)k;
    }
  });
}

}  // namespace swapnet

extern "C" int swapnet_pack_bf16(const void* src, uint64_t n_elems, void* dst, uint64_t dst_bytes,
                                 uint64_t* used_bytes) {
  if (!src || !used_bytes) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null argument");
  if (n_elems == 0 || n_elems % swapnet::kPkChunk)
    SN_FAIL(SWAPNET_ERR_UNSUPPORTED, "packing: the element count must be a positive multiple of 4096");
  const int threads = (int)std::min(32u, std::max(1u, std::thread::hardware_concurrency()));
  const swapnet::PackInfo info = swapnet::pack_prepare(static_cast<const uint16_t*>(src), n_elems, threads);
  *used_bytes = info.bytes;
  if (!dst) return SWAPNET_OK;
  if (dst_bytes < info.bytes) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "packing: destination too small");
  swapnet::pack_write(static_cast<const uint16_t*>(src), n_elems, info, static_cast<uint8_t*>(dst), threads);
  return SWAPNET_OK;
}
