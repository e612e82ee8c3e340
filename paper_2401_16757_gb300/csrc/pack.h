// Lossless packing of bf16 parameter tensors for the packed swap variant
// (SWAPNET_SWAP_PACKED, an extension the paper has no counterpart for: the
// same parameters cross the host link in fewer bytes and are unpacked into
// the arena by an SM kernel).
//
// A bf16 value is sign (1 bit), exponent (8), mantissa (7).  Trained and
// initialised weights use few, neighbouring exponents, so each tensor gets
// the window of 15 consecutive exponents x0 .. x0 + 14 that holds most of
// its elements; an element stores its sign and mantissa in one byte and its
// exponent as a 4-bit code x - x0, 15 meaning "outside the window" (an
// escape).  Elements are grouped in chunks of 4096; a chunk with at most
// kPkMaxEsc escapes keeps their positions and exponents in its header, any
// other chunk is stored unpacked in an overflow area.  Every chunk body
// has the same size and starts on a 128-byte line, so a range of chunks (a
// piece of a tensor placed in a block) is a contiguous range of bodies
// that a warp reads in whole lines.
//
// Packed tensor of n elements (n a multiple of kPkChunk), C = n / kPkChunk:
//   [0, 16)                 x0 in byte 0, then zeros (x0 <= 240)
//   16 + 16 c               header of chunk c, c < C
//   B = pk_body_off(C)      (16 + 16 C rounded up to 128 bytes)
//   B + c * kPkBody         body of chunk c
//   B + C * kPkBody + 8192 r  overflow chunk r (4096 raw bf16 words)
// Header (16 bytes):
//   [0]       escapes k (0..kPkMaxEsc), or kPkRaw: stored in the overflow area
//   [4, 12)   k positions inside the chunk (uint16, ascending); for kPkRaw
//             bytes [4, 8) hold the overflow index r (uint32)
//   [12, 16)  the escaped elements' exponents, in the same order
// Body (kPkBody bytes; zeros for a chunk in the overflow area):
//   [0, 2048)      codes: byte b = element 2b (low nibble) and 2b + 1 (high)
//   [2048, 6144)   sign and mantissa: byte e = (w >> 8 & 0x80) | (w & 0x7f)
// Element e of the chunk is ((s & 0x80) << 8) | (x << 7) | (s & 0x7f) with
// s its sign-mantissa byte and x its exponent: x0 + its code, or for code
// 15 the exponent its header lists (little-endian throughout).
#pragma once

#include <cuda_runtime.h>

#include <cstdint>
#include <vector>

namespace swapnet {

constexpr int kPkChunk = 4096;                               // elements per chunk
constexpr int kPkMaxEsc = 4;                                 // escapes a record holds
constexpr int kPkRaw = 0xff;                                 // record kind: overflow
constexpr int kPkHeader = 16;                                // bytes of a chunk header
constexpr int kPkBody = kPkChunk / 2 + kPkChunk;             // 6144 bytes, 48 lines
constexpr uint64_t kPkChunkBytes = 2ull * kPkChunk;          // 8192 unpacked bytes

inline uint64_t pk_body_off(uint64_t chunks) { return (16 + kPkHeader * chunks + 127) / 128 * 128; }

// What packing n bf16 elements (n a multiple of kPkChunk) takes: the code
// table, which chunks go to the overflow area, and the packed bytes.
struct PackInfo {
  uint8_t exp[16];                // the tensor header: x0, then zeros
  uint8_t code[256];              // code of each exponent (15: escape)
  std::vector<uint32_t> overflow;  // per chunk: overflow index, or UINT32_MAX
  uint64_t bytes = 0;
};

// Both use up to `threads` worker threads (at least 1).
PackInfo pack_prepare(const uint16_t* src, uint64_t n, int threads);
void pack_write(const uint16_t* src, uint64_t n, const PackInfo& info, uint8_t* dst, int threads);

// One contiguous range of chunk records to unpack into the arena.
struct PkJob {
  const uint8_t* base;    // packed tensor (device alias of page-locked host memory)
  uint16_t* dst;          // arena address of chunk c0's first element
  uint64_t body_off;      // byte offsets of the bodies and the overflow area from base
  uint64_t overflow_off;
  uint32_t c0, nchunks;   // records c0 .. c0 + nchunks - 1
  uint32_t first;         // index of this job's first chunk among the launch's chunks
  uint32_t x0;            // the tensor's exponent window start
};

// Unpacks every chunk of jobs[0..njobs) (a device array, jobs in order of
// `first`, total chunks in all) with `ctas` CTAs of kUnpackThreads on s.
constexpr int kUnpackThreads = 256;
int launch_unpack(const PkJob* jobs, int njobs, uint32_t total, int ctas, cudaStream_t s);

}  // namespace swapnet
