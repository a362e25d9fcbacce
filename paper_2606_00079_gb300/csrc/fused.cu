// Fused single-token decode forward: the whole quantized MoE layer in one
// persistent kernel (one block per SM), for a batch of one token.
//
// Same arithmetic as the kernel chain in forward.cu (Fig. 1 Stage 3; the
// association of Eq. app_normalized_decomposition), reorganised so that no
// phase waits for a kernel launch and every weight byte is requested at the
// start:
//
//   prologue   bulk copies of this block's rows of the input bases (Phi_g^T,
//              Phi_u^T) into shared memory; L2 prefetch of its rows of Phi_dn.
//              Weights only, so this overlaps the tail of the previous kernel
//              (programmatic dependent launch).
//   routing    every block routes the token itself (k largest logits, ties to
//              the lower index, softmax over the k), then stages its share of
//              the routed experts' gate/up items into shared memory and
//              prefetches its share of their down tiles into L2
//   B          z = Phi^T x for this block's rows                 -> grid barrier 1
//   C          gate/up items: dp2a over the staged codes, vector red.add into
//              gate/up; the last item of a (expert, 128-row block) computes
//              h = SiLU(gate) * up for those rows and quantises it to int16
//              with one scale per row block                      -> grid barrier 2
//   D          down tiles (staged into the freed projection buffer):
//              s += w_e * alpha * (P_dn^T h), fp32 atomics         -> grid barrier 3
//   E          y = Phi_dn s for this block's rows (staged after B)
//
// The grid barriers are counters in the workspace that a one-block prep
// kernel zeroes before each call; every wait is bounded (about one second of
// SM clock) and a timeout is reported in the workspace status word.
#include <algorithm>
#include <cstring>
#include <mutex>

#include "device.cuh"

namespace {

constexpr int kFWarps = 16;
constexpr int kFThreads = kFWarps * 32;
constexpr int kMaxBStages = 8;
constexpr int kFZ = 12;                 // slots per lane whose z values are gathered at once
constexpr long long kSpin = 2ll << 30;  // bounded waits: about one second of SM clock

__device__ __forceinline__ uint32_t ld_acquire_u32(const uint32_t* ptr) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(ptr) : "memory");
  return v;
}

// All blocks of the grid arrive on `cnt` (zeroed before the launch) and wait
// until every block has arrived.  Writes before the barrier are visible to
// loads after it (fence, then L2-coherent loads on the reading side).
__device__ __forceinline__ void grid_barrier(uint32_t* cnt, uint32_t nblocks, int* status) {
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    atomicAdd(cnt, 1u);
    const long long t0 = clock64();
    while (ld_acquire_u32(cnt) < nblocks) {
      if (clock64() - t0 > kSpin) {
        atomicCAS(status, 0, BITSMOE_ERR_TIMEOUT);
        break;
      }
    }
    __threadfence();
  }
  __syncthreads();
}

__device__ __forceinline__ void prefetch_run(const uint8_t* p, uint64_t bytes) {
  while (bytes > 0) {
    const uint32_t c = bytes > 65536 ? 65536u : (uint32_t)bytes;
    prefetch_l2(p, c);
    p += c;
    bytes -= c;
  }
}

// Issue `bytes` (16-byte multiple, 16-byte aligned) into shared memory on an
// already initialised mbarrier whose transaction count the caller has set.
__device__ __forceinline__ void bulk_run(void* dst, const uint8_t* src, uint32_t bytes, uint64_t* bar) {
  uint32_t o = 0;
  while (o < bytes) {
    const uint32_t c = bytes - o < 32768u ? bytes - o : 32768u;
    bulk_g2s(static_cast<uint8_t*>(dst) + o, src + o, c, bar);
    o += c;
  }
}

// gate/up work item i -> (routed-expert slot a, projection h, row block rb, segment sg)
struct CItem {
  int a, h, rb, sg;
};
__device__ __forceinline__ CItem c_item(const Fwd& p, int i) {
  const int per_e = 2 * p.NRB * p.nseg;
  CItem c;
  c.a = i / per_e;
  int r = i - c.a * per_e;
  c.h = r / (p.NRB * p.nseg);
  r -= c.h * p.NRB * p.nseg;
  c.rb = r / p.nseg;
  c.sg = r - c.rb * p.nseg;
  return c;
}

// Stage one gate/up item (codes of its row block, unit indices, alpha, the
// G scale/zero rows of its groups) into a slot.  Lane 0 only.
template <int G>
__device__ void c_stage(const Fwd& p, const FusedArgs& f, const CItem& ci, int e, const ItemRec& it, uint8_t* slot,
                        uint64_t* bar) {
  const ExpertDesc& xd = p.desc[ci.h * p.E + e];
  const uint64_t code_base = xd.code_base, rb_stride = xd.rb_stride, unit_off = xd.unit_off;
  const uint64_t alpha_off = xd.alpha_off, sz_off = xd.sz_off;
  const int nslots = xd.nslots;
  const uint32_t mb = (uint32_t)it.nslot * 4;
  uint8_t* codes = slot;
  uint8_t* su = slot + f.seg_al;
  uint8_t* sa = su + (size_t)f.smax * 4;
  uint8_t* ssz = sa + (size_t)f.smax * 4;
  const int g_base = (ci.rb * kRows) / p.group;
  mbar_expect_tx(bar, it.bytes + (2 + G) * mb);
  bulk_run(codes, p.img + code_base + (size_t)ci.rb * rb_stride + it.byte0, it.bytes, bar);
  bulk_g2s(su, p.img + unit_off + (size_t)it.slot0 * 4, mb, bar);
  bulk_g2s(sa, p.img + alpha_off + (size_t)it.slot0 * 4, mb, bar);
#pragma unroll
  for (int gl = 0; gl < G; ++gl)
    bulk_g2s(ssz + (size_t)gl * f.smax * 4, p.img + sz_off + ((size_t)(g_base + gl) * nslots + it.slot0) * 4, mb, bar);
}

// L2 prefetch of the bytes c_stage would copy (for items staged in a later round).
__device__ void c_prefetch(const Fwd& p, const CItem& ci, int e, const ItemRec& it) {
  const ExpertDesc& xd = p.desc[ci.h * p.E + e];
  prefetch_run(p.img + xd.code_base + (size_t)ci.rb * xd.rb_stride + it.byte0, it.bytes);
}

// One staged gate/up item for the single token: writes its partial rows of
// gate (h = 0) or up (h = 1) with vector reductions.
template <int G>
__device__ void c_compute(const Fwd& p, const FusedArgs& f, const CItem& ci, const ItemRec& it, const uint8_t* slot,
                          int16_t* cq, int pair, int lane) {
  const uint8_t* codes = slot;
  const int* su = reinterpret_cast<const int*>(slot + f.seg_al);
  const float* sa = reinterpret_cast<const float*>(su + f.smax);
  const uint32_t* ssz = reinterpret_cast<const uint32_t*>(sa + f.smax);
  const float* zrow = p.z + (size_t)ci.h * p.n_pad;   // one token: z[h][0][:]
  int nls = 0;
  for (int q = 0; q < it.nr; ++q)
    if (it.bits[q] < 16) nls += it.ntl[q] * rl_units(it.bits[q]);
  // c = alpha * z * scale per (slot, group), int16 with one scale per item
  const bool fast = nls <= 32 * kFZ;
  float mx = 0.f;
  float zr[kFZ];
  if (fast) {
#pragma unroll
    for (int m = 0; m < kFZ; ++m) {
      const int i = lane + 32 * m;
      zr[m] = i < nls ? __ldcg(zrow + su[i]) : 0.f;
    }
#pragma unroll
    for (int m = 0; m < kFZ; ++m) {
      const int i = lane + 32 * m;
      if (i < nls) {
        zr[m] *= sa[i];
#pragma unroll
        for (int gl = 0; gl < G; ++gl) {
          const float sc = __half2float(__ushort_as_half((unsigned short)(ssz[gl * f.smax + i] & 0xFFFFu)));
          mx = fmaxf(mx, fabsf(zr[m] * sc));
        }
      }
    }
  } else {
    for (int i = lane; i < nls; i += 32) {
      const float zv = sa[i] * __ldcg(zrow + su[i]);
#pragma unroll
      for (int gl = 0; gl < G; ++gl)
        mx = fmaxf(mx, fabsf(zv * __half2float(__ushort_as_half((unsigned short)(ssz[gl * f.smax + i] & 0xFFFFu)))));
    }
  }
  mx = warp_max(mx);
  const float inv = mx > 0.f ? 32767.f / mx : 0.f;
  const float scl = mx * (1.f / 32767.f);
  float corr[G];
#pragma unroll
  for (int gl = 0; gl < G; ++gl) corr[gl] = 0.f;
  if (fast) {
#pragma unroll
    for (int m = 0; m < kFZ; ++m) {
      const int i = lane + 32 * m;
      if (i < nls) {
#pragma unroll
        for (int gl = 0; gl < G; ++gl) {
          const uint32_t w = ssz[gl * f.smax + i];
          const float sc = __half2float(__ushort_as_half((unsigned short)(w & 0xFFFFu)));
          const float zp = __half2float(__ushort_as_half((unsigned short)(w >> 16)));
          const int ci2 = __float2int_rn(zr[m] * sc * inv);
          cq[(size_t)gl * f.s16 + i] = (int16_t)ci2;
          corr[gl] = fmaf((float)ci2, zp, corr[gl]);
        }
      }
    }
  } else {
    for (int i = lane; i < nls; i += 32) {
      const float zv = sa[i] * __ldcg(zrow + su[i]);
#pragma unroll
      for (int gl = 0; gl < G; ++gl) {
        const uint32_t w = ssz[gl * f.smax + i];
        const float sc = __half2float(__ushort_as_half((unsigned short)(w & 0xFFFFu)));
        const float zp = __half2float(__ushort_as_half((unsigned short)(w >> 16)));
        const int ci2 = __float2int_rn(zv * sc * inv);
        cq[(size_t)gl * f.s16 + i] = (int16_t)ci2;
        corr[gl] = fmaf((float)ci2, zp, corr[gl]);
      }
    }
  }
#pragma unroll
  for (int gl = 0; gl < G; ++gl) corr[gl] = warp_sum(corr[gl]);
  __syncwarp();
  float accf[4][1], acc16[4][1];
#pragma unroll
  for (int w = 0; w < 4; ++w) accf[w][0] = acc16[w][0] = 0.f;
  const int gl_lane = G == 1 ? 0 : (4 * lane) / p.group;
  const int* cq32 = reinterpret_cast<const int*>(cq + (size_t)gl_lane * f.s16);
  const float* const zrows[1] = {zrow};
  uint32_t boff = 0;
  int ls = 0;
  for (int q = 0; q < it.nr; ++q) {
    const int b = it.bits[q], ntl = it.ntl[q];
    const uint8_t* code = codes + boff + lane * 16;
    const int* cp = cq32 + ls / 2;
    switch (b) {
      case 1: rl_range<1, 1, true>(code, ntl, cp, 0, accf); break;
      case 2: rl_range<2, 1, true>(code, ntl, cp, 0, accf); break;
      case 3: rl_range<3, 1, true>(code, ntl, cp, 0, accf); break;
      case 4: rl_range<4, 1, true>(code, ntl, cp, 0, accf); break;
      case 6: rl_range<6, 1, true>(code, ntl, cp, 0, accf); break;
      case 8: rl_range<8, 1, true>(code, ntl, cp, 0, accf); break;
      default: rl_range16<1, true>(code, ntl, su + ls, sa + ls, zrows, acc16); break;
    }
    boff += (uint32_t)ntl * rl_chunks(b) * kChunkBytes;
    ls += ntl * rl_units(b);
  }
  float cl = corr[0];
#pragma unroll
  for (int gl = 1; gl < G; ++gl)
    if (gl == gl_lane) cl = corr[gl];
  float o[4];
#pragma unroll
  for (int w = 0; w < 4; ++w) o[w] = fmaf(scl, accf[w][0] - cl, acc16[w][0]);
  red_add_v4(p.gu + ((size_t)pair * 2 + ci.h) * p.I_pad + ci.rb * kRows + 4 * lane, o[0], o[1], o[2], o[3]);
}

// h = SiLU(gate) * up for the 128 rows of row block rb of one pair, quantised
// to int16 with one scale per row block; also the per-group sums of the codes.
// Called by the warp that finished the last gate/up item of (expert, rb).
template <int G>
__device__ void h_rows(const Fwd& p, const FusedArgs& f, int pair, int rb, int lane) {
  const int row = rb * kRows + 4 * lane;
  const float4 g = __ldcg(reinterpret_cast<const float4*>(p.gu + ((size_t)pair * 2) * p.I_pad + row));
  const float4 u = __ldcg(reinterpret_cast<const float4*>(p.gu + ((size_t)pair * 2 + 1) * p.I_pad + row));
  float hv[4] = {g.x / (1.f + __expf(-g.x)) * u.x, g.y / (1.f + __expf(-g.y)) * u.y,
                 g.z / (1.f + __expf(-g.z)) * u.z, g.w / (1.f + __expf(-g.w)) * u.w};
  float mx = fmaxf(fmaxf(fabsf(hv[0]), fabsf(hv[1])), fmaxf(fabsf(hv[2]), fabsf(hv[3])));
  mx = warp_max(mx);
  const float inv = mx > 0.f ? 32767.f / mx : 0.f;
  int q[4];
#pragma unroll
  for (int w = 0; w < 4; ++w) q[w] = __float2int_rn(hv[w] * inv);
  const uint32_t lo = (uint32_t)(q[0] & 0xFFFF) | ((uint32_t)q[1] << 16);
  const uint32_t hi = (uint32_t)(q[2] & 0xFFFF) | ((uint32_t)q[3] << 16);
  *reinterpret_cast<uint2*>(f.hq + (size_t)pair * p.I_pad + row) = make_uint2(lo, hi);
  int sq = q[0] + q[1] + q[2] + q[3];
  // group sums: lanes of one group are 8 (group 32), 16 (group 64) or all 32
  const int lanes_per_group = G == 1 ? 32 : p.group / 4;
#pragma unroll
  for (int o = 16; o; o >>= 1)
    if (o < lanes_per_group) sq += __shfl_xor_sync(0xFFFFFFFFu, sq, o);
  if ((lane & (lanes_per_group - 1)) == 0) f.hsum[((size_t)pair * p.NRB + rb) * G + lane / lanes_per_group] = sq;
  if (lane == 0) f.hsc[(size_t)pair * p.NRB + rb] = mx * (1.f / 32767.f);
}

// Down tile of the lane's unit over all row blocks, h quantised per row block:
//   accf = sum_rb hsc_rb * sum_g s_g (sum_{i in rb, g} q_i h_i - zero_g * sum_{i in rb, g} h_i)
template <int B, int G>
__device__ __forceinline__ float ul_tile_rb(const uint8_t* code, int NRB, int group, const int16_t* hq,
                                            const float* hsc, const int* hsum, const uint32_t* sz, int lane) {
  constexpr int C = ul_chunks(B);
  const int gshift = 31 - __clz(group);
  float accf = 0.f;
  for (int rb = 0; rb < NRB; ++rb) {
    const int* hq32 = reinterpret_cast<const int*>(hq + rb * kRows);
    const uint8_t* cb = code + (size_t)rb * C * kChunkBytes;
    if (B == 16) {
      float tmp = 0.f;
#pragma unroll 4
      for (int c = 0; c < 16; ++c) {
        const uint4 v = lds128(cb + (size_t)c * kChunkBytes);
        const uint32_t wv[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int w = 0; w < 4; ++w) {
          const int hp = hq32[(8 * c + 2 * w) / 2];
          tmp = fmaf((float)(int16_t)(hp & 0xFFFF), f16lo(wv[w]), fmaf((float)(hp >> 16), f16hi(wv[w]), tmp));
        }
      }
      accf = fmaf(hsc[rb], tmp, accf);
      continue;
    }
    int acc[G][1], acch[G][1];
#pragma unroll
    for (int g = 0; g < G; ++g) acc[g][0] = acch[g][0] = 0;
    uint4 v[C];
#pragma unroll
    for (int c = 0; c < C; ++c) v[c] = lds128(cb + (size_t)c * kChunkBytes);
    if (B == 3) {
      ul_chunk<2, G, 1>(v[0], 0, hq32, 0, gshift, acc);
      ul_chunk<2, G, 1>(v[1], 64, hq32, 0, gshift, acc);
      ul_chunk<1, G, 1>(v[2], 0, hq32, 0, gshift, acch);
    } else if (B == 6) {
#pragma unroll
      for (int c = 0; c < 4; ++c) ul_chunk<4, G, 1>(v[c], 32 * c, hq32, 0, gshift, acc);
      ul_chunk<2, G, 1>(v[4], 0, hq32, 0, gshift, acch);
      ul_chunk<2, G, 1>(v[5], 64, hq32, 0, gshift, acch);
    } else {
#pragma unroll
      for (int c = 0; c < C; ++c) ul_chunk<B, G, 1>(v[c], c * (kRows / B), hq32, 0, gshift, acc);
    }
    float d_rb = 0.f;
    const int gfirst = (rb * kRows) >> gshift;
#pragma unroll
    for (int g = 0; g < G; ++g) {
      const uint32_t szw = sz[(size_t)(gfirst + g) * 32 + lane];
      const float sc = __half2float(__ushort_as_half((unsigned short)(szw & 0xFFFFu)));
      const float zp = __half2float(__ushort_as_half((unsigned short)(szw >> 16)));
      const int tot = (B == 3 || B == 6) ? acc[g][0] + (acch[g][0] << (B == 3 ? 2 : 4)) : acc[g][0];
      d_rb = fmaf(sc, fmaf(-zp, (float)hsum[rb * G + g], (float)tot), d_rb);
    }
    accf = fmaf(hsc[rb], d_rb, accf);
  }
  return accf;
}

// down work item i -> (routed-expert slot a, UL tile)
struct DItem {
  int a, tile;
};
__device__ __forceinline__ DItem d_item(const FusedArgs& f, int i) {
  DItem d;
  d.a = i / f.ul_max_tiles;
  d.tile = i - d.a * f.ul_max_tiles;
  return d;
}

// Where a down tile lives: its bucket's bit-width, first slot, code run and
// scale/zero column.  bits = 0 when the tile index is past the expert's tiles.
struct DLoc {
  int bits, slot;       // slot of the tile's first unit in the (h=2, e) slot arrays
  int nslots;           // row stride of the scale/zero matrix
  uint64_t code, sz;    // image offsets: tile code run (NRB row blocks), scale/zero column of its first slot
  uint64_t unit, alpha; // image offsets of its 32 unit indices and alphas
};
__device__ DLoc d_loc(const Fwd& p, int e, int tile) {
  const ExpertDesc& xd = p.desc[2 * p.E + e];
  DLoc l;
  l.bits = 0;
  l.slot = 0;
  l.nslots = xd.nslots;
  l.code = l.sz = l.unit = l.alpha = 0;
  const int nbk = xd.nbk;
  for (int q = 0; q < nbk; ++q) {
    const int t0 = xd.bk[q].tile0, nt = xd.bk[q].ntiles;
    if (tile >= t0 && tile < t0 + nt) {
      const int b = xd.bk[q].bits;
      l.bits = b;
      l.slot = xd.bk[q].slot0 + (tile - t0) * 32;
      l.code = xd.code_base + xd.bk[q].code_off + (uint64_t)(tile - t0) * p.NRB * ul_chunks(b) * kChunkBytes;
      l.sz = xd.sz_off + (uint64_t)l.slot * 4;
      l.unit = xd.unit_off + (uint64_t)l.slot * 4;
      l.alpha = xd.alpha_off + (uint64_t)l.slot * 4;
    }
  }
  return l;
}

// D slot layout: [codes NRB * ul_max_chunks * 512][unit 32 x 4][alpha 32 x 4][scale/zero NG x 32 x 4]
__device__ void d_stage(const Fwd& p, const FusedArgs& f, const DLoc& l, uint8_t* slot, uint64_t* bar) {
  const uint32_t cb = (uint32_t)p.NRB * ul_chunks(l.bits) * kChunkBytes;
  uint8_t* su = slot + f.d_code_bytes;
  uint8_t* sa = su + 128;
  uint8_t* ssz = sa + 128;
  mbar_expect_tx(bar, cb + 256 + (uint32_t)p.NG * 128);
  bulk_run(slot, p.img + l.code, cb, bar);
  bulk_g2s(su, p.img + l.unit, 128, bar);
  bulk_g2s(sa, p.img + l.alpha, 128, bar);
  for (int g = 0; g < p.NG; ++g) bulk_g2s(ssz + g * 128, p.img + l.sz + (uint64_t)g * l.nslots * 4, 128, bar);
}

template <int G>
__device__ void d_compute(const Fwd& p, const FusedArgs& f, const DLoc& l, const uint8_t* slot,
                          const int16_t* hq, const float* hsc, const int* hsum, int pair, float wgt, int lane) {
  const uint8_t* code = slot + lane * 16;
  const int* su = reinterpret_cast<const int*>(slot + f.d_code_bytes);
  const float* sa = reinterpret_cast<const float*>(su + 32);
  const uint32_t* ssz = reinterpret_cast<const uint32_t*>(sa + 32);
  float acc = 0.f;
  switch (l.bits) {
    case 1: acc = ul_tile_rb<1, G>(code, p.NRB, p.group, hq, hsc, hsum, ssz, lane); break;
    case 2: acc = ul_tile_rb<2, G>(code, p.NRB, p.group, hq, hsc, hsum, ssz, lane); break;
    case 3: acc = ul_tile_rb<3, G>(code, p.NRB, p.group, hq, hsc, hsum, ssz, lane); break;
    case 4: acc = ul_tile_rb<4, G>(code, p.NRB, p.group, hq, hsc, hsum, ssz, lane); break;
    case 6: acc = ul_tile_rb<6, G>(code, p.NRB, p.group, hq, hsc, hsum, ssz, lane); break;
    case 8: acc = ul_tile_rb<8, G>(code, p.NRB, p.group, hq, hsc, hsum, ssz, lane); break;
    default: acc = ul_tile_rb<16, G>(code, p.NRB, p.group, hq, hsc, hsum, ssz, lane); break;
  }
  const float al = sa[lane];
  if (al != 0.f) atomicAdd(p.s + su[lane], wgt * al * acc);   // one token: s[0][j]
}

template <int G>
__global__ void __launch_bounds__(kFThreads, 1) k_fused(Fwd p, FusedArgs f) {
  extern __shared__ __align__(128) uint8_t fsm[];
  uint64_t* bar_b = reinterpret_cast<uint64_t*>(fsm);   // [kMaxBStages]
  uint64_t* bar_e = bar_b + kMaxBStages;                 // [1]
  uint64_t* bar_c = bar_e + 1;                           // [kFWarps]
  uint64_t* bar_d = bar_c + kFWarps;                     // [kFWarps]
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  const int nb = gridDim.x, blk = blockIdx.x;
  const uint32_t row_in = (uint32_t)p.D_pad * 2, row_out = (uint32_t)p.n_pad * 2;
  uint8_t* r1 = fsm + f.off_r1;
  uint8_t* rc = fsm + f.off_rc;
  const int nrows_b = 2 * p.n;
  const int b0 = min(nrows_b, blk * f.b_per), b1 = min(nrows_b, b0 + f.b_per);
  const int e0 = min(p.D, blk * f.e_per), e1 = min(p.D, e0 + f.e_per);

  // ---- prologue: weights only (may overlap the previous kernel)
  if (tid == 0) {
    for (int i = 0; i < kMaxBStages + 1 + 2 * kFWarps; ++i) mbar_init(bar_b + i);
    for (int st = 0; st < f.b_nst; ++st) {
      const int a = b0 + st * f.b_stage, b = min(b1, a + f.b_stage);
      if (b > a) {
        mbar_expect_tx(bar_b + st, (uint32_t)(b - a) * row_in);
        bulk_run(r1 + (size_t)st * f.b_stage * row_in, reinterpret_cast<const uint8_t*>(p.basis_in) + (size_t)a * row_in,
                 (uint32_t)(b - a) * row_in, bar_b + st);
      }
    }
    if (e1 > e0)
      prefetch_run(reinterpret_cast<const uint8_t*>(p.basis_out) + (size_t)e0 * row_out, (uint64_t)(e1 - e0) * row_out);
  }
  __syncthreads();
  pdl_wait();   // x, logits, y and the workspace belong to earlier kernels until here

  // ---- routing (every block), x into shared memory, zero gate/up and s
  const RouteView rv = route_block(p, reinterpret_cast<uint32_t*>(fsm + f.off_route));
  uint16_t* xs = reinterpret_cast<uint16_t*>(fsm + f.off_xs);
  for (int i = tid; i < p.D_pad; i += kFThreads) xs[i] = i < p.D ? p.x[i] : (uint16_t)0;
  {
    const size_t ng = (size_t)p.P * 2 * p.I_pad / 4, ns = (size_t)p.n_pad / 4;
    const float4 z4 = make_float4(0.f, 0.f, 0.f, 0.f);
    for (size_t i = (size_t)blk * kFThreads + tid; i < ng + ns; i += (size_t)nb * kFThreads) {
      if (i < ng) reinterpret_cast<float4*>(p.gu)[i] = z4;
      else reinterpret_cast<float4*>(p.s)[i - ng] = z4;
    }
  }
  const int A = rv.act[0];
  const int nci = A * 2 * p.NRB * p.nseg;   // gate/up items
  const int ndi = A * f.ul_max_tiles;        // down items (some past an expert's tiles)
  // this block's items: i = blk + m * nb; warp w < nslot works on m = w, w + nslot, ...
  const int mc = nci > blk ? (nci - blk + nb - 1) / nb : 0;
  const int md = ndi > blk ? (ndi - blk + nb - 1) / nb : 0;
  if (lane == 0) {
    if (wid < f.nslot_c) {
      for (int m = wid; m < mc; m += f.nslot_c) {
        const CItem ci = c_item(p, blk + m * nb);
        const int e = rv.act[1 + ci.a];
        const ItemRec it = p.items[((size_t)ci.h * p.E + e) * p.nseg + ci.sg];
        if (it.nr == 0) continue;
        if (m == wid) c_stage<G>(p, f, ci, e, it, fsm + f.off_rc + (size_t)wid * f.slot_c, bar_c + wid);
        else c_prefetch(p, ci, e, it);
      }
    }
    if (wid < f.nslot_d) {
      for (int m = wid; m < md; m += f.nslot_d) {
        const DItem di = d_item(f, blk + m * nb);
        const DLoc l = d_loc(p, rv.act[1 + di.a], di.tile);
        if (l.bits) prefetch_run(p.img + l.code, (uint64_t)p.NRB * ul_chunks(l.bits) * kChunkBytes);
      }
    }
  }

  __syncthreads();   // x is in shared memory

  // ---- B: z = Phi^T x for rows [b0, b1)
  for (int ri = wid; ri < b1 - b0; ri += kFWarps) {
    const int st = ri / f.b_stage;
    if (!mbar_wait(bar_b + st, 0)) {
      if (lane == 0) atomicCAS(p.status, 0, BITSMOE_ERR_TIMEOUT);
      continue;
    }
    const uint8_t* rp = r1 + (size_t)ri * row_in;
    float acc = 0.f;
    for (int c = lane; c < (p.D_pad >> 3); c += 32) {
      const uint4 v = lds128(rp + (size_t)c * 16);
      const uint4 xv = lds128(xs + c * 8);
      acc = fmaf(bf16lo(v.x), bf16lo(xv.x), acc);
      acc = fmaf(bf16hi(v.x), bf16hi(xv.x), acc);
      acc = fmaf(bf16lo(v.y), bf16lo(xv.y), acc);
      acc = fmaf(bf16hi(v.y), bf16hi(xv.y), acc);
      acc = fmaf(bf16lo(v.z), bf16lo(xv.z), acc);
      acc = fmaf(bf16hi(v.z), bf16hi(xv.z), acc);
      acc = fmaf(bf16lo(v.w), bf16lo(xv.w), acc);
      acc = fmaf(bf16hi(v.w), bf16hi(xv.w), acc);
    }
    acc = warp_sum(acc);
    if (lane == 0) {
      const int row = b0 + ri, h = row >= p.n, j = row - h * p.n;
      p.z[(size_t)h * p.n_pad + j] = acc;
    }
  }
  __syncthreads();   // the projection rows are consumed: stage Phi_dn rows and down tiles there
  uint8_t* ers = r1;                       // [e1 - e0][n_pad] bf16
  uint8_t* dslots = r1 + f.off_d;          // [nslot_d][slot_d]
  if (tid == 0) fence_proxy_async();   // generic reads of the rows above, then async writes
  if (tid == 0 && e1 > e0) {
    mbar_expect_tx(bar_e, (uint32_t)(e1 - e0) * row_out);
    bulk_run(ers, reinterpret_cast<const uint8_t*>(p.basis_out) + (size_t)e0 * row_out, (uint32_t)(e1 - e0) * row_out,
             bar_e);
  }
  if (lane == 0 && wid < f.nslot_d && wid < md) {
    const DItem di = d_item(f, blk + wid * nb);
    const DLoc l = d_loc(p, rv.act[1 + di.a], di.tile);
    if (l.bits) d_stage(p, f, l, dslots + (size_t)wid * f.slot_d, bar_d + wid);
  }
  grid_barrier(f.cnt + 0, nb, p.status);

  // ---- C: gate/up items
  if (wid < f.nslot_c) {
    uint8_t* slot = rc + (size_t)wid * f.slot_c;
    int16_t* cq = reinterpret_cast<int16_t*>(fsm + f.off_cq) + (size_t)wid * G * f.s16;
    int nst = 0;   // items staged into this slot so far (the mbarrier completes once per staging)
    for (int m = wid; m < mc; m += f.nslot_c) {
      const CItem ci = c_item(p, blk + m * nb);
      const int e = rv.act[1 + ci.a];
      const int pair = rv.plist[rv.start[e]];
      const ItemRec it = p.items[((size_t)ci.h * p.E + e) * p.nseg + ci.sg];
      if (it.nr != 0) {
        if (nst > 0 || m != wid) {   // not the prologue's staging: refill the slot (its last item is done)
          __syncwarp();
          if (lane == 0) {
            fence_proxy_async();
            c_stage<G>(p, f, ci, e, it, slot, bar_c + wid);
          }
        }
        if (mbar_wait(bar_c + wid, (uint32_t)nst & 1u)) {
          c_compute<G>(p, f, ci, it, slot, cq, pair, lane);
        } else if (lane == 0) {
          atomicCAS(p.status, 0, BITSMOE_ERR_TIMEOUT);
        }
        ++nst;
      }
      // completion of (expert slot a, row block rb): the last of its 2 * nseg items computes h
      __threadfence();
      __syncwarp();
      int last = 0;
      if (lane == 0) last = atomicAdd(f.ctr + ci.a * p.NRB + ci.rb, 1u) == (uint32_t)(2 * p.nseg - 1);
      last = __shfl_sync(0xFFFFFFFFu, last, 0);
      if (last) {
        __threadfence();
        h_rows<G>(p, f, pair, ci.rb, lane);
      }
    }
  }
  grid_barrier(f.cnt + 1, nb, p.status);

  // ---- D: down tiles, s += w * alpha * P_dn^T h
  if (wid < f.nslot_d) {
    uint8_t* slot = dslots + (size_t)wid * f.slot_d;
    int16_t* hqs = reinterpret_cast<int16_t*>(rc + (size_t)wid * f.d_h_bytes);   // C slots are free now
    float* hsc = reinterpret_cast<float*>(hqs + p.I_pad);
    int* hsum = reinterpret_cast<int*>(hsc + p.NRB);
    int staged = 0, cur_pair = -1;
    for (int m = wid; m < md; m += f.nslot_d) {
      const DItem di = d_item(f, blk + m * nb);
      const int e = rv.act[1 + di.a];
      const DLoc l = d_loc(p, e, di.tile);
      if (!l.bits) continue;
      if (m != wid) {
        __syncwarp();
        if (lane == 0) {
          fence_proxy_async();
          d_stage(p, f, l, slot, bar_d + wid);
        }
      }
      const int pair = rv.plist[rv.start[e]];
      if (pair != cur_pair) {   // h of this expert's token: int16 rows, scales, group sums
        __syncwarp();
        for (int i = lane; i < p.I_pad / 8; i += 32)
          reinterpret_cast<uint4*>(hqs)[i] = __ldcg(reinterpret_cast<const uint4*>(f.hq + (size_t)pair * p.I_pad) + i);
        for (int i = lane; i < p.NRB; i += 32) hsc[i] = __ldcg(f.hsc + (size_t)pair * p.NRB + i);
        for (int i = lane; i < p.NRB * G; i += 32) hsum[i] = __ldcg(f.hsum + (size_t)pair * p.NRB * G + i);
        __syncwarp();
        cur_pair = pair;
      }
      if (mbar_wait(bar_d + wid, (uint32_t)staged & 1u)) {
        d_compute<G>(p, f, l, slot, hqs, hsc, hsum, pair, rv.pw[pair], lane);
      } else if (lane == 0) {
        atomicCAS(p.status, 0, BITSMOE_ERR_TIMEOUT);
      }
      ++staged;
    }
  }
  grid_barrier(f.cnt + 2, nb, p.status);
  pdl_trigger();   // every block is past its last wait on other blocks

  // ---- E: y = Phi_dn s for rows [e0, e1)
  float* ss = reinterpret_cast<float*>(rc);
  for (int i = tid; i < p.n_pad / 4; i += kFThreads)
    reinterpret_cast<float4*>(ss)[i] = __ldcg(reinterpret_cast<const float4*>(p.s) + i);
  __syncthreads();
  if (e1 > e0) {
    bool ok = mbar_wait(bar_e, 0);
    if (!ok && tid == 0) atomicCAS(p.status, 0, BITSMOE_ERR_TIMEOUT);
    for (int ri = wid; ok && ri < e1 - e0; ri += kFWarps) {
      const uint8_t* rp = ers + (size_t)ri * row_out;
      float acc = 0.f;
      for (int c = lane; c < (p.n_pad >> 3); c += 32) {
        const uint4 v = lds128(rp + (size_t)c * 16);
        const float4 sa = *reinterpret_cast<const float4*>(ss + c * 8);
        const float4 sb = *reinterpret_cast<const float4*>(ss + c * 8 + 4);
        acc = fmaf(bf16lo(v.x), sa.x, acc);
        acc = fmaf(bf16hi(v.x), sa.y, acc);
        acc = fmaf(bf16lo(v.y), sa.z, acc);
        acc = fmaf(bf16hi(v.y), sa.w, acc);
        acc = fmaf(bf16lo(v.z), sb.x, acc);
        acc = fmaf(bf16hi(v.z), sb.y, acc);
        acc = fmaf(bf16lo(v.w), sb.z, acc);
        acc = fmaf(bf16hi(v.w), sb.w, acc);
      }
      acc = warp_sum(acc);
      if (lane == 0) {
        const int row = e0 + ri;
        p.y[row] = p.accum ? p.y[row] + acc : acc;
      }
    }
  }
}

// One block: clears the status word, the grid-barrier counters and the
// per-(expert, row block) completion counters before the fused kernel uses
// them.  It lets the fused kernel launch at once; the fused kernel waits for
// this grid (and so for the previous kernel) before touching the workspace.
__global__ void k_fused_prep(int* status, uint32_t* cnt, uint32_t* ctr, int nctr) {
  pdl_trigger();
  pdl_wait();
  if (threadIdx.x == 0) status[0] = 0;
  if (threadIdx.x < 4) cnt[threadIdx.x] = 0u;
  for (int i = threadIdx.x; i < nctr; i += blockDim.x) ctr[i] = 0u;
}

}  // namespace

namespace bmoe {

bool fused_plan(const ImageHeader& hd, int T, int top_k, int seg_bytes, int ul_max_chunks, int s16, int sms,
                FusedArgs* f) {
  if (T != 1 || sms < 1) return false;
  std::memset(f, 0, sizeof(*f));
  const int G = std::max(1, kRows / hd.group);
  const size_t row_in = (size_t)hd.D_pad * 2, row_out = (size_t)hd.n_pad * 2;
  const size_t budget = 227 * 1024;
  const int A = std::min(hd.E, top_k);
  f->b_per = (2 * hd.n + sms - 1) / sms;
  f->b_stage = std::max(1, (f->b_per + kMaxBStages - 1) / kMaxBStages);
  f->b_nst = (f->b_per + f->b_stage - 1) / f->b_stage;
  f->e_per = (hd.D + sms - 1) / sms;
  f->smax = s16 - 8;
  f->s16 = s16;
  f->seg_al = (int)align_up((uint64_t)std::max(seg_bytes, 16), 128);
  f->slot_c = (int)align_up((uint64_t)f->seg_al + (uint64_t)f->smax * 4 * (2 + G), 128);
  f->ul_max_tiles = hd.ul_max_tiles;
  f->d_code_bytes = hd.NRB * ul_max_chunks * kChunkBytes;
  f->slot_d = (int)align_up((uint64_t)f->d_code_bytes + 256 + (uint64_t)hd.NG * 128, 128);
  f->d_h_bytes = (int)align_up((uint64_t)hd.I_pad * 2 + (uint64_t)hd.NRB * 4 * (1 + G), 128);
  const int items_c = (A * 2 * hd.NRB * hd.nseg + sms - 1) / sms;
  const int items_d = (A * hd.ul_max_tiles + sms - 1) / sms;
  // fixed areas: mbarriers, routing, x, the per-warp int16 activation tables
  size_t off = 512;
  f->off_route = (int)off;
  off = align_up(off + (size_t)(T * hd.E + 3 * T * top_k + 3 * hd.E + 3) * 4, 128);
  f->off_xs = (int)off;
  off = align_up(off + row_in, 128);
  f->off_cq = (int)off;
  off = align_up(off + (size_t)kFWarps * G * s16 * 2, 128);
  const size_t r_b = (size_t)f->b_per * row_in;
  const size_t r_e = align_up((size_t)f->e_per * row_out, 128);
  f->off_d = (int)r_e;
  int nslot_d = std::min(std::max(items_d, 1), kFWarps);
  size_t r1 = std::max(r_b, r_e + (size_t)nslot_d * f->slot_d);
  while (nslot_d > 1 && off + r1 > budget) {
    --nslot_d;
    r1 = std::max(r_b, r_e + (size_t)nslot_d * f->slot_d);
  }
  f->off_r1 = (int)off;
  off = align_up(off + r1, 128);
  f->off_rc = (int)off;
  if (off >= budget) return false;
  int nslot_c = std::min(std::max(items_c, 1), kFWarps);
  while (nslot_c > 1 && off + (size_t)nslot_c * f->slot_c > budget) --nslot_c;
  size_t rc = std::max({(size_t)nslot_c * f->slot_c, (size_t)nslot_d * f->d_h_bytes, row_out * 2});
  if (off + rc > budget) return false;
  f->nslot_c = nslot_c;
  f->nslot_d = nslot_d;
  f->smem = (int)(off + rc);
  return true;
}

cudaError_t launch_fused(const Fwd& p, const FusedArgs& f, int nctr, int sms, cudaStream_t st, bool pdl) {
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(1);
  cfg.blockDim = dim3(256);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = st;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  cudaError_t e = cudaLaunchKernelEx(&cfg, k_fused_prep, p.status, f.cnt, f.ctr, nctr);
  if (e != cudaSuccess) return e;
  const int G = std::max(1, kRows / p.group);
  static std::mutex mu;
  static int done_smem[3] = {0, 0, 0};
  auto go = [&](void (*kernel)(Fwd, FusedArgs), int gi) -> cudaError_t {
    {
      std::lock_guard<std::mutex> lock(mu);
      if (f.smem > done_smem[gi]) {
        cudaError_t r = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, f.smem);
        if (r != cudaSuccess) return r;
        r = cudaFuncSetAttribute(kernel, cudaFuncAttributePreferredSharedMemoryCarveout, cudaSharedmemCarveoutMaxShared);
        if (r != cudaSuccess) return r;
        done_smem[gi] = f.smem;
      }
    }
    cudaLaunchConfig_t c2 = {};
    c2.gridDim = dim3(sms);
    c2.blockDim = dim3(kFThreads);
    c2.dynamicSmemBytes = f.smem;
    c2.stream = st;
    cudaLaunchAttribute a2[1];
    a2[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    a2[0].val.programmaticStreamSerializationAllowed = 1;
    c2.attrs = a2;
    c2.numAttrs = 1;   // always: the prep kernel triggers at once
    return cudaLaunchKernelEx(&c2, kernel, p, f);
  };
  if (G == 1) return go(k_fused<1>, 0);
  if (G == 2) return go(k_fused<2>, 1);
  return go(k_fused<4>, 2);
}

}  // namespace bmoe
