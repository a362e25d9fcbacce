// Packed device layout of one BitsMoE layer (library-internal).
//
// One contiguous image (the same bytes on the host as a "blob" and in HBM):
//
//   [ImageHeader][ExpertDesc 3 x E][K2 segment table 2 x E x (nseg+1)]
//   [basis_in  bf16 [2][n][D_pad]]  row j of projection h = phi_{h,j}  (gate, up)
//   [basis_out bf16 [D][n_pad]]     row d = Phi_dn[d, :]
//   [gate/up item table ItemRec 2 x E x nseg]
//   per (h, e), contiguous: [unit index int32 [nslots]][alpha f32 [nslots]]
//                           [scale/zero half2 [NG][nslots] over all slots][code stream]
//
// Units of one (h, e) are bucketed by bit-width b in {1,2,3,4,6,8,16} (0-bit
// units are dropped: they contribute nothing and move no bytes), stable in j.
// Every bucket is a uniform-bit stream of 512-byte warp chunks (16 bytes per
// lane), so each lane's load is one coalesced 128-bit access.
//
// gate/up ("row-lane" layout, RL): a lane owns 4 consecutive rows i of a
// 128-row block and a tile of U(b) units; word w of its 16-byte chunk is row w.
//   b in {1,2,4,8}: U = 32/b units per word; unit u = 4k + m sits at bit 8m + b*k,
//     so ((word >> b*k) & mask_bytes) yields 4 units of one row as 4 bytes.
//   b = 3: U = 32; chunks 0,1 = low 2-bit plane of units 0-15 / 16-31 (2-bit
//     format), chunk 2 = high 1-bit plane of units 0-31 (1-bit format).
//   b = 6: U = 16; chunks 0,1 = low 4-bit plane of units 0-7 / 8-15, chunk 2 =
//     high 2-bit plane of units 0-15.
//   b = 16: U = 4; chunk c, word w = fp16(unit 2c, row w) | fp16(unit 2c+1, row w) << 16.
//   Stream order: [row block][bucket][tile][chunk][lane] x 16 bytes.
//
// down ("unit-lane" layout, UL): a lane owns one unit (slot) of a 32-slot
// tile and streams its codes along the rows; per 128-row block a lane has
// b chunks of 16 bytes (16 for b = 16).
//   b in {1,2,4,8}: chunk c covers rows 128/b*c .. , word w of it 32/b rows,
//     row r' = 4k + m of a word at bit 8m + b*k.
//   b = 3: chunks 0,1 = low 2-bit plane rows 0-63 / 64-127; chunk 2 = high bit rows 0-127.
//   b = 6: chunks 0..3 = low 4-bit plane rows 32c ..; chunks 4,5 = high 2-bit plane rows 64(c-4) ..
//   b = 16: chunk c = rows 8c .. 8c+7, word w = fp16(row 2w) | fp16(row 2w+1) << 16.
//   Stream order: [bucket][tile][row block][chunk][lane] x 16 bytes.
//
// Every tile holds a multiple of 4 units, so every slot range of a bucket, a
// tile or a gate/up item starts on a 16-byte boundary of the slot arrays.
//
// Padding: slots beyond a bucket's unit count have alpha 0 and codes 0;
// rows beyond I (up to I_pad) have code 0 and scale/zero 0, so padded
// elements dequantise to exactly 0.
#pragma once
#include <stdint.h>

#ifndef __CUDACC__
#ifndef __host__
#define __host__
#endif
#ifndef __device__
#define __device__
#endif
#endif

namespace bmoe {

constexpr uint32_t kMagic = 0x454F4D42u;   // "BMOE"
constexpr uint32_t kVersion = 2;
constexpr int kNumBk = 7;
constexpr int kRows = 128;                 // rows per row block
constexpr int kChunkBytes = 512;           // one warp-wide 16-byte-per-lane load

__host__ __device__ constexpr int bk_bits(int k) {
  return k == 0 ? 1 : k == 1 ? 2 : k == 2 ? 3 : k == 3 ? 4 : k == 4 ? 6 : k == 5 ? 8 : 16;
}
__host__ __device__ constexpr int bk_of_bits(int b) {
  return b == 1 ? 0 : b == 2 ? 1 : b == 3 ? 2 : b == 4 ? 3 : b == 6 ? 4 : b == 8 ? 5 : b == 16 ? 6 : -1;
}
// gate/up tiles: units per tile and 16-byte chunks per lane per tile
__host__ __device__ constexpr int rl_units(int b) {
  return b == 1 ? 32 : b == 2 ? 16 : b == 3 ? 32 : b == 4 ? 8 : b == 6 ? 16 : 4;
}
__host__ __device__ constexpr int rl_chunks(int b) { return (b == 3 || b == 6) ? 3 : b == 16 ? 2 : 1; }
// down tiles: 32 units, chunks per lane per row block
__host__ __device__ constexpr int ul_chunks(int b) { return b; }

struct BucketDesc {
  int32_t bits;       // 1..16
  int32_t count;      // real units
  int32_t nslots;     // padded slots
  int32_t ntiles;     // RL: nslots / rl_units(b); UL: nslots / 32
  int32_t slot0;      // first slot of this bucket in the (h,e) slot arrays
  int32_t tile0;      // first flat tile index of this bucket within (h,e)
  uint64_t code_off;  // RL: byte offset inside one row-block stream; UL: inside the (h,e) stream
  uint64_t sz_off;    // image offset of this bucket's column 0 in the (h,e) scale/zero matrix
};

struct ExpertDesc {
  int32_t nbk;        // non-empty buckets (bk[0 .. nbk))
  int32_t ntiles;     // total tiles over buckets
  int32_t nslots;     // total slots over buckets
  int32_t nunits;     // units with b > 0
  uint64_t begin;     // image offset of this (h,e) block (for L2 prefetch)
  uint64_t end;
  uint64_t code_base; // image offset of the code stream
  uint64_t rb_stride; // RL: bytes per row block (stream = NRB * rb_stride); UL: stream bytes
  uint64_t unit_off;  // image offset of int32 [nslots]
  uint64_t alpha_off; // image offset of float [nslots]
  uint64_t sz_off;    // image offset of half2 (scale | zero << 16) [NG][nslots]; row stride nslots
  uint64_t moved;     // algorithmic bytes of this (h,e)
  BucketDesc bk[kNumBk];
};

// One gate/up work item: a segment of consecutive tiles of one (h, e) inside a
// row block.  Its code bytes are one contiguous run of the row-block stream and
// its slots one contiguous run of the slot arrays; its tiles cover nr
// consecutive buckets.
struct ItemRec {
  uint32_t byte0;     // first code byte inside the row-block stream
  uint32_t bytes;     // code bytes (16-byte multiple)
  uint32_t slot0;     // first slot (multiple of 4)
  uint16_t nslot;     // slots (multiple of 4)
  uint8_t nr;         // buckets touched (0: empty item)
  uint8_t bk0;        // index of the first one in ExpertDesc::bk
  uint8_t bits[kNumBk + 1];
  uint16_t ntl[kNumBk + 1];   // tiles per touched bucket
  uint32_t pad_[2];
};
static_assert(sizeof(ItemRec) == 48, "ItemRec layout");

struct ImageHeader {
  uint32_t magic, version;
  int32_t D, E, I, n, group;
  int32_t D_pad, n_pad, I_pad, NRB, NG;
  int32_t nseg;           // K2 (gate/up) segments per (h, e)
  int32_t seg_max_slots;  // most slots any K2 segment spans
  int32_t ul_max_tiles;   // most UL tiles of any expert
  int32_t reserved_;
  uint64_t total_bytes;
  uint64_t off_desc;      // ExpertDesc [3][E]
  uint64_t off_seg;       // int32 [2][E][nseg + 1], flat tile boundaries
  uint64_t off_basis_in;  // bf16 [2][n][D_pad]
  uint64_t off_basis_out; // bf16 [D][n_pad]
  uint64_t codes_bytes;   // code streams as stored
  uint64_t meta_bytes;    // unit/alpha/scale-zero arrays
  uint64_t off_items;     // ItemRec [2][E][nseg]
};

inline uint64_t align_up(uint64_t v, uint64_t a) { return (v + a - 1) / a * a; }

}  // namespace bmoe
