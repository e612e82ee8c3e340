// Lossless packing of bf16 parameter tensors for the packed swap variant
// (SWAPNET_SWAP_PACKED, an extension the paper has no counterpart for: the
// same parameters cross the host link in fewer bytes and are unpacked into
// the arena by an SM kernel).
//
// A bf16 value is sign (1 bit), exponent (8), mantissa (7).  Trained and
// initialised weights use few exponents, so each tensor gets a table of its
// 15 most frequent exponents; an element stores its sign and mantissa in
// one byte and its exponent as a 4-bit code into that table, 15 meaning
// "not in the table" (an escape).  Elements are grouped in chunks of 4096;
// a chunk with at most kPkMaxEsc escapes keeps their positions and
// exponents in its header, any other chunk is stored unpacked in an
// overflow area.  Every chunk record has the same size, so a range of
// chunks (a piece of a tensor placed in a block) is a contiguous range of
// records.
//
// Packed tensor of n elements (n a multiple of kPkChunk), C = n / kPkChunk:
//   [0, 16)                      exponent of codes 0..14 (byte 15 unused)
//   16 + c * kPkRecord           record of chunk c, c < C
//   16 + C * kPkRecord + r * 8192  overflow chunk r (4096 raw bf16 words)
// Record (kPkRecord bytes, 16-byte aligned):
//   [0]       escapes k (0..kPkMaxEsc), or kPkRaw: stored in the overflow area
//   [4, 12)   k positions inside the chunk (uint16, ascending); for kPkRaw
//             bytes [4, 8) hold the overflow index r (uint32)
//   [12, 16)  the escaped elements' exponents, in the same order
//   [16, 16 + 2048)          codes: byte b = element 2b (low nibble) and
//                            element 2b + 1 (high nibble)
//   [16 + 2048, kPkRecord)   sign and mantissa: byte e = (w >> 8 & 0x80) | (w & 0x7f)
// Element e of the chunk is ((s & 0x80) << 8) | (x << 7) | (s & 0x7f) with
// s its sign-mantissa byte and x its exponent (little-endian throughout).
#pragma once

#include <cuda_runtime.h>

#include <cstdint>
#include <vector>

namespace swapnet {

constexpr int kPkChunk = 4096;                               // elements per chunk
constexpr int kPkMaxEsc = 4;                                 // escapes a record holds
constexpr int kPkRaw = 0xff;                                 // record kind: overflow
constexpr int kPkHeader = 16;                                // table bytes at the start
constexpr int kPkRecord = 16 + kPkChunk / 2 + kPkChunk;      // 6160 bytes
constexpr uint64_t kPkChunkBytes = 2ull * kPkChunk;          // 8192 unpacked bytes

// What packing n bf16 elements (n a multiple of kPkChunk) takes: the code
// table, which chunks go to the overflow area, and the packed bytes.
struct PackInfo {
  uint8_t exp[16];                // exponent of each code (15: escape)
  uint8_t code[256];              // code of each exponent
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
  uint64_t overflow_off;  // byte offset of the overflow area from base
  uint32_t c0, nchunks;   // records c0 .. c0 + nchunks - 1
  uint32_t first;         // index of this job's first chunk among the launch's chunks
  uint32_t pad;
  uint32_t table[4];      // the tensor's 16 table bytes
};

// Unpacks every chunk of jobs[0..njobs) (a device array, jobs in order of
// `first`, total chunks in all) with `ctas` CTAs on stream s.
int launch_unpack(const PkJob* jobs, int njobs, uint32_t total, int ctas, cudaStream_t s);

}  // namespace swapnet
