// Fused single-token decode forward: the whole quantized MoE layer in one
// persistent kernel (one block per SM), for a batch of one token.
//
// Same arithmetic as the kernel chain in forward.cu (Fig. 1 Stage 3; the
// association of Eq. app_normalized_decomposition), reorganised so that no
// phase waits for a kernel launch and every weight byte is requested early:
//
//   prologue   bulk copies of this block's rows of the input bases (Phi_g^T,
//              Phi_u^T) into shared memory.  Weights only, so this overlaps
//              the tail of the previous kernel (programmatic dependent launch).
//   routing    every block routes the token itself (k largest logits, ties to
//              the lower index, softmax over the k), then stages its share of
//              the routed experts' gate/up items into shared memory and
//              prefetches its down tiles and its rows of Phi_dn into L2
//   B          z = Phi^T x for this block's rows                 -> grid barrier 1
//   C          gate/up items: dp2a over the staged codes, vector red.add into
//              gate and up                                       -> grid barrier 2
//   D          down tiles (staged into the freed projection buffer):
//              h = SiLU(gate) * up of the tile's expert, quantised to int16
//              with one scale per 128-row block, then
//              s += w_e * alpha * (P_dn^T h), fp32 atomics         -> grid barrier 3
//   E          y = Phi_dn s for this block's rows (staged after B)
//
// Each work item's copies come from one staging record (CStage / DStage,
// derived from the image at upload), so a block issues them after a single
// vector load.  The grid barriers are counters at a fixed place in the
// workspace: zero when a call starts (the caller zero-fills the workspace once;
// the last block to finish a call resets them), checked on entry.  Every wait
// is bounded (about one second of SM clock) and a timeout is reported in the
// status word.
#include <algorithm>
#include <cstring>
#include <mutex>

#include "fused_common.cuh"

namespace {

// Phase timestamps of each block (%globaltimer), compiled in only with -DBITSMOE_F2_TRACE
// for timing studies; without it F1_MARK is empty.
#ifdef BITSMOE_F2_TRACE
__device__ unsigned long long g_f1_trace[1024][16];
#define F1_MARK(i)                                                                    \
  do {                                                                                \
    unsigned long long t_;                                                            \
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t_));                            \
    g_f1_trace[blockIdx.x & 1023][(i)] = t_;                                          \
  } while (0)
#else
#define F1_MARK(i) \
  do {             \
  } while (0)
#endif
// Copy of a gate/up staging record into shared memory (its per-bucket arrays
// are read with runtime indices, so it is used from there).
__device__ __forceinline__ void copy_crec(CStage* dst, const CStage* src) {
  static_assert(sizeof(CStage) % 16 == 0, "record size");
  uint4 v[sizeof(CStage) / 16];
#pragma unroll
  for (int i = 0; i < (int)(sizeof(CStage) / 16); ++i) v[i] = __ldg(reinterpret_cast<const uint4*>(src) + i);
#pragma unroll
  for (int i = 0; i < (int)(sizeof(CStage) / 16); ++i) reinterpret_cast<uint4*>(dst)[i] = v[i];
}
__device__ __forceinline__ uint64_t u64_of(uint32_t lo, uint32_t hi) { return (uint64_t)lo | ((uint64_t)hi << 32); }
// A down staging record, decoded field by field from three 16-byte loads.
__device__ __forceinline__ DStage load_drec(const DStage* src) {
  const uint4* q = reinterpret_cast<const uint4*>(src);
  const uint4 a = __ldg(q), b = __ldg(q + 1), c = __ldg(q + 2);
  DStage r;
  r.code = u64_of(a.x, a.y);
  r.unit = u64_of(a.z, a.w);
  r.alpha = u64_of(b.x, b.y);
  r.sz = u64_of(b.z, b.w);
  r.sz_row = c.x;
  r.bits = c.y;
  r.meta = c.z;
  r.pad_ = 0;
  return r;
}

// Down item m of block blk under the snake deal over nb blocks, and how many items of
// n a block gets.
__device__ __forceinline__ int d_item(int blk, int m, int nb) { return m * nb + ((m & 1) ? nb - 1 - blk : blk); }
__device__ __forceinline__ int d_count(int n, int blk, int nb) {
  const int full = n / nb, rem = n - full * nb;
  return full + (((full & 1) ? nb - 1 - blk : blk) < rem ? 1 : 0);
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

// Down tile of the lane's unit over row blocks rb = rb0, rb0 + step, ..., h
// quantised per row block:
//   sum_rb hsc_rb * sum_g s_g (sum_{i in rb, g} q_i h_i - zero_g * sum_{i in rb, g} h_i)
template <int G>
__device__ float ul_tile_rt(int b, const uint8_t* code, int NRB, int rb0, int step, int group, const int16_t* hq,
                            const float* hsc, const int* hsum, const uint32_t* sz, int lane) {
  const int gshift = 31 - __clz(group);
  const int C = ul_chunks(b);
  float accf = 0.f;
  for (int rb = rb0; rb < NRB; rb += step) {
    const int* hq32 = reinterpret_cast<const int*>(hq + rb * kRows);
    const uint8_t* cb = code + (size_t)rb * C * kChunkBytes;
    if (b == 16) {   // fp16 values: chunk c = rows 8c .. 8c + 7, two rows per word
      float tmp = 0.f;
#pragma unroll 1
      for (int c = 0; c < 16; ++c) {
        const uint4 v = lds128(cb + (size_t)c * kChunkBytes);
        const uint32_t wv[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int w = 0; w < 4; ++w) {
          const int hp = hq32[4 * c + w];
          tmp = fmaf((float)(int16_t)(hp & 0xFFFF), f16lo(wv[w]), fmaf((float)(hp >> 16), f16hi(wv[w]), tmp));
        }
      }
      accf = fmaf(hsc[rb], tmp, accf);
      continue;
    }
    int4 lo = make_int4(0, 0, 0, 0), hi = make_int4(0, 0, 0, 0);
    switch (b) {
      case 1: lo = ul_plane<1, G>(cb, 1, 0, hq32, gshift, lo); break;
      case 2: lo = ul_plane<2, G>(cb, 2, 0, hq32, gshift, lo); break;
      case 4: lo = ul_plane<4, G>(cb, 4, 0, hq32, gshift, lo); break;
      case 8: lo = ul_plane<8, G>(cb, 8, 0, hq32, gshift, lo); break;
      case 3:   // low 2-bit plane rows 0-63 / 64-127, then the high bit of rows 0-127
        lo = ul_plane<2, G>(cb, 2, 0, hq32, gshift, lo);
        hi = ul_plane<1, G>(cb + 2 * kChunkBytes, 1, 0, hq32, gshift, hi);
        break;
      default:  // 6: low 4-bit plane rows 32c .., then the high 2 bits of rows 0-63 / 64-127
        lo = ul_plane<4, G>(cb, 4, 0, hq32, gshift, lo);
        hi = ul_plane<2, G>(cb + 4 * kChunkBytes, 2, 0, hq32, gshift, hi);
        break;
    }
    const int hs = b == 3 ? 2 : 4;
    const int lo_g[4] = {lo.x, lo.y, lo.z, lo.w}, hi_g[4] = {hi.x, hi.y, hi.z, hi.w};
    float d_rb = 0.f;
    const int gfirst = (rb * kRows) >> gshift;
#pragma unroll
    for (int g = 0; g < G; ++g) {
      const uint32_t szw = sz[(size_t)(gfirst + g) * 32 + lane];
      const float sc = __half2float(__ushort_as_half((unsigned short)(szw & 0xFFFFu)));
      const float zp = __half2float(__ushort_as_half((unsigned short)(szw >> 16)));
      d_rb = fmaf(sc, fmaf(-zp, (float)hsum[rb * G + g], (float)(lo_g[g] + (hi_g[g] << hs))), d_rb);
    }
    accf = fmaf(hsc[rb], d_rb, accf);
  }
  return accf;
}

// The copies of a gate/up item of row block rb and of a down tile lie inside the image and
// the metadata mirror.
template <int G>
__device__ bool crec_ok(const Fwd& p, const FusedArgs& f, const CStage& r, int rb) {
  const uint64_t mrow = (uint64_t)(2 + G) * r.mb;
  return in_image(p, r.code0 + (uint64_t)rb * r.rb_stride, r.bytes) && r.meta0 + (rb + 1) * mrow <= f.meta_bytes;
}
__device__ bool drec_ok(const Fwd& p, const FusedArgs& f, const DStage& r) {
  return in_image(p, r.code, (uint64_t)p.NRB * ul_chunks((int)r.bits) * kChunkBytes) &&
         (uint64_t)r.meta + 256 + (uint64_t)p.NG * 128 <= f.meta_bytes;
}

// Copies of one gate/up item into a slot: [codes seg_al][unit mb][alpha mb][scale/zero G x mb]
// (mb = 4 bytes a slot of the item): the codes from the image, the rest from the metadata
// mirror, where they lie together, in one copy.
template <int G>
__device__ void c_stage(const Fwd& p, const FusedArgs& f, const CStage& r, int rb, uint8_t* slot, uint64_t* bar) {
  const uint32_t mrow = (2 + G) * r.mb;
  mbar_expect_tx(bar, r.bytes + mrow);
  bulk_run(slot, p.img + r.code0 + (uint64_t)rb * r.rb_stride, r.bytes, bar);
  bulk_g2s(slot + f.seg_al, f.meta + r.meta0 + (uint64_t)rb * mrow, mrow, bar);
}

// One staged gate/up item for the single token: adds its partial rows of gate
// (h = 0) or up (h = 1) with vector reductions.
template <int G>
__device__ void c_compute(const Fwd& p, const FusedArgs& f, const CStage& r, int h, int rb, const uint8_t* slot,
                          int16_t* cq, int pair, int lane) {
  const int ms = (int)(r.mb / 4);   // the item's slots
  const int* su = reinterpret_cast<const int*>(slot + f.seg_al);
  const float* sa = reinterpret_cast<const float*>(su + ms);
  const uint32_t* ssz = reinterpret_cast<const uint32_t*>(sa + ms);
  const float* zrow = p.z + (size_t)h * p.n_pad;   // one token: z[h][0][:]
  const int nls = r.nls;
  // c = alpha * z * scale per (slot, group), int16 with one scale per item.
  // Up to 32 * kFZ slots: one batch of z gathers, kept in registers for both
  // passes; larger items gather z again in the second pass.
  float mx = 0.f;
  float zr[kFZ];
#pragma unroll
  for (int m = 0; m < kFZ; ++m) {
    const int i = lane + 32 * m;
    zr[m] = i < nls ? __ldcg(zrow + su[i]) * sa[i] : 0.f;
  }
  const bool one_batch = nls <= 32 * kFZ;
  for (int i0 = 0; i0 < nls; i0 += 32 * kFZ) {
    if (i0 > 0) {
#pragma unroll
      for (int m = 0; m < kFZ; ++m) {
        const int i = i0 + lane + 32 * m;
        zr[m] = i < nls ? __ldcg(zrow + su[i]) * sa[i] : 0.f;
      }
    }
#pragma unroll
    for (int m = 0; m < kFZ; ++m) {
      const int i = i0 + lane + 32 * m;
      if (i < nls) {
#pragma unroll
        for (int gl = 0; gl < G; ++gl) {
          const float sc = __half2float(__ushort_as_half((unsigned short)(ssz[gl * ms + i] & 0xFFFFu)));
          mx = fmaxf(mx, fabsf(zr[m] * sc));
        }
      }
    }
  }
  mx = warp_max(mx);
  const float inv = mx > 0.f ? 32767.f / mx : 0.f;
  const float scl = mx * (1.f / 32767.f);
  float corr[G];
#pragma unroll
  for (int gl = 0; gl < G; ++gl) corr[gl] = 0.f;
  for (int i0 = 0; i0 < nls; i0 += 32 * kFZ) {
    if (!one_batch) {
#pragma unroll
      for (int m = 0; m < kFZ; ++m) {
        const int i = i0 + lane + 32 * m;
        zr[m] = i < nls ? __ldcg(zrow + su[i]) * sa[i] : 0.f;
      }
    }
#pragma unroll
    for (int m = 0; m < kFZ; ++m) {
      const int i = i0 + lane + 32 * m;
      if (i < nls) {
#pragma unroll
        for (int gl = 0; gl < G; ++gl) {
          const uint32_t w = ssz[gl * ms + i];
          const float sc = __half2float(__ushort_as_half((unsigned short)(w & 0xFFFFu)));
          const float zp = __half2float(__ushort_as_half((unsigned short)(w >> 16)));
          const int ci = __float2int_rn(zr[m] * sc * inv);
          cq[(size_t)gl * f.s16 + i] = (int16_t)ci;
          corr[gl] = fmaf((float)ci, zp, corr[gl]);
        }
      }
    }
  }
#pragma unroll
  for (int gl = 0; gl < G; ++gl) corr[gl] = warp_sum(corr[gl]);
  __syncwarp();
  float accf[4] = {0.f, 0.f, 0.f, 0.f};
  float acc16[4][1];
#pragma unroll
  for (int w = 0; w < 4; ++w) acc16[w][0] = 0.f;
  const int gl_lane = G == 1 ? 0 : (4 * lane) / p.group;
  const int* cq32 = reinterpret_cast<const int*>(cq + (size_t)gl_lane * f.s16);
  const float* const zrows[1] = {zrow};
  uint32_t boff = 0;
  int ls = 0;
  for (int q = 0; q < r.nr; ++q) {
    const int b = r.bits[q], ntl = r.ntl[q];
    const uint8_t* code = slot + boff + lane * 16;
    if (b < 16) rl_range_rt(b, code, ntl, cq32 + ls / 2, accf);
    else rl_range16<1, true>(code, ntl, su + ls, sa + ls, zrows, acc16);
    boff += (uint32_t)ntl * rl_chunks(b) * kChunkBytes;
    ls += ntl * rl_units(b);
  }
  float cl = corr[0];
#pragma unroll
  for (int gl = 1; gl < G; ++gl)
    if (gl == gl_lane) cl = corr[gl];
  float o[4];
#pragma unroll
  for (int w = 0; w < 4; ++w) o[w] = fmaf(scl, accf[w] - cl, acc16[w][0]);
  red_add_v4(p.gu + ((size_t)pair * 2 + h) * p.I_pad + rb * kRows + 4 * lane, o[0], o[1], o[2], o[3]);
}

// h = SiLU(gate) * up of one pair for row blocks rb0, rb0 + step, ... into the
// warp's area: int16 codes, one scale per 128-row block, sums of the codes per
// (row block, group).  The lane owns rows 4 * lane .. + 3 of a row block.
template <int G>
__device__ void h_rows(const Fwd& p, int pair, int rb0, int step, int16_t* hq, float* hsc, int* hsum, int lane) {
  const float* gp = p.gu + ((size_t)pair * 2) * p.I_pad + 4 * lane;
  const float* up = gp + p.I_pad;
  const int lanes_per_group = G == 1 ? 32 : p.group / 4;
  constexpr int kB = 4;   // row blocks whose gate/up loads are in flight together
  for (int rbb = rb0; rbb < p.NRB; rbb += kB * step) {
    float4 g4[kB], u4[kB];
#pragma unroll
    for (int i = 0; i < kB; ++i) {
      const int rb = rbb + i * step;
      const bool ok = rb < p.NRB;
      g4[i] = ok ? __ldcg(reinterpret_cast<const float4*>(gp + (size_t)rb * kRows)) : make_float4(0, 0, 0, 0);
      u4[i] = ok ? __ldcg(reinterpret_cast<const float4*>(up + (size_t)rb * kRows)) : make_float4(0, 0, 0, 0);
    }
#pragma unroll 1
    for (int i = 0; i < kB; ++i) {
      const int rb = rbb + i * step;
      if (rb >= p.NRB) break;
      const float4 g = g4[0], u = u4[0];   // the batch rotates through slot 0
      const float hv[4] = {__fdividef(g.x, 1.f + __expf(-g.x)) * u.x, __fdividef(g.y, 1.f + __expf(-g.y)) * u.y,
                           __fdividef(g.z, 1.f + __expf(-g.z)) * u.z, __fdividef(g.w, 1.f + __expf(-g.w)) * u.w};
#pragma unroll
      for (int j = 0; j + 1 < kB; ++j) {
        g4[j] = g4[j + 1];
        u4[j] = u4[j + 1];
      }
      float mx = fmaxf(fmaxf(fabsf(hv[0]), fabsf(hv[1])), fmaxf(fabsf(hv[2]), fabsf(hv[3])));
      mx = warp_max(mx);
      const float inv = mx > 0.f ? 32767.f / mx : 0.f;
      int q[4];
#pragma unroll
      for (int w = 0; w < 4; ++w) q[w] = __float2int_rn(hv[w] * inv);
      const uint32_t lo = (uint32_t)(q[0] & 0xFFFF) | ((uint32_t)q[1] << 16);
      const uint32_t hi = (uint32_t)(q[2] & 0xFFFF) | ((uint32_t)q[3] << 16);
      *reinterpret_cast<uint2*>(hq + rb * kRows + 4 * lane) = make_uint2(lo, hi);
      int sq = q[0] + q[1] + q[2] + q[3];
#pragma unroll
      for (int o = 16; o; o >>= 1)
        if (o < lanes_per_group) sq += __shfl_xor_sync(0xFFFFFFFFu, sq, o);
      if ((lane & (lanes_per_group - 1)) == 0) hsum[rb * G + lane / lanes_per_group] = sq;
      if (lane == 0) hsc[rb] = mx * (1.f / 32767.f);
    }
  }
}

// D slot layout: [codes NRB * ul_max_chunks * 512][unit 32 x 4][alpha 32 x 4][scale/zero NG x 32 x 4]:
// the codes from the image, the rest from the metadata mirror in one copy.
__device__ void d_stage(const Fwd& p, const FusedArgs& f, const DStage& r, uint8_t* slot, uint64_t* bar) {
  const uint32_t cb = (uint32_t)p.NRB * ul_chunks((int)r.bits) * kChunkBytes;
  const uint32_t mt = 256 + (uint32_t)p.NG * 128;
  mbar_expect_tx(bar, cb + mt);
  bulk_run(slot, p.img + r.code, cb, bar);
  bulk_g2s(slot + f.d_code_bytes, f.meta + r.meta, mt, bar);
}

template <int G>
__global__ void __launch_bounds__(kFThreads, 1) k_fused(Fwd p, FusedArgs f) {
  extern __shared__ __align__(128) uint8_t fsm[];
  uint64_t* bar_b = reinterpret_cast<uint64_t*>(fsm);   // [kMaxBStages]
  uint64_t* bar_e = bar_b + kMaxBStages;                 // [1]
  uint64_t* bar_c = bar_e + 1;                           // [kFWarps]
  uint64_t* bar_d = bar_c + kFWarps;                     // [kFWarps]
  CStage* crec = reinterpret_cast<CStage*>(fsm + f.off_rec);   // [kFWarps] first gate/up item of each slot
  DStage* drec = reinterpret_cast<DStage*>(crec + kFWarps);     // [kFWarps] first down item of each slot
  uint32_t* keys = reinterpret_cast<uint32_t*>(fsm + f.off_route);   // [E]
  int* sel_e = reinterpret_cast<int*>(keys + p.E);                     // [k] expert of routing rank a
  float* sel_w = reinterpret_cast<float*>(sel_e + p.k);                // [k] its gate weight
  float* part = reinterpret_cast<float*>(fsm + f.off_part);           // [kFWarps][32] down partial sums
  volatile int* seen = reinterpret_cast<volatile int*>(bar_d + kFWarps);   // [3] grid barriers passed
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  const int nb = gridDim.x, blk = blockIdx.x;
  const uint32_t row_in = (uint32_t)p.D_pad * 2, row_out = (uint32_t)p.n_pad * 2;
  uint8_t* r1 = fsm + f.off_r1;
  uint8_t* rc = fsm + f.off_rc;
  const int nrows_b = 2 * p.n;
  const int b0 = min(nrows_b, blk * f.b_per), b1 = min(nrows_b, b0 + f.b_per);
  const int e0 = min(p.D, blk * f.e_per), e1 = min(p.D, e0 + f.e_per);

  // ---- prologue: weights and the staging tables only (may overlap the previous kernel).
  // Half of this block's projection rows are requested now, the rest after the
  // logits and x loads, so that those small loads do not queue behind them.
  const int nst_pre = (f.b_nst + 1) / 2;
  auto issue_b = [&](int st0, int st1) {
    for (int st = st0; st < st1; ++st) {
      const int a = b0 + st * f.b_stage, b = min(b1, a + f.b_stage);
      if (b > a) {
        mbar_expect_tx(bar_b + st, (uint32_t)(b - a) * row_in);
        bulk_run(r1 + (size_t)st * f.b_stage * row_in, reinterpret_cast<const uint8_t*>(p.basis_in) + (size_t)a * row_in,
                 (uint32_t)(b - a) * row_in, bar_b + st);
      }
    }
  };
  if (tid == 0) {
    F1_MARK(0);
    for (int i = 0; i < kMaxBStages + 1 + 2 * kFWarps; ++i) mbar_init(bar_b + i);
    seen[0] = seen[1] = seen[2] = seen[3] = 0;
    issue_b(0, nst_pre);
  } else if (tid == 64 && f.norm) {   // this block's router rows (norm mode) into L2
    const int epb = (p.E + nb - 1) / nb, r0 = min(p.E, blk * epb), r1e = min(p.E, r0 + epb);
    if (r1e > r0) prefetch_run(reinterpret_cast<const uint8_t*>(f.wr + (size_t)r0 * p.D), (uint64_t)(r1e - r0) * p.D * 2);
  } else if (tid == 32) {   // this block's share of the staging tables into L2
    const uint64_t per = (f.tab_bytes / nb + 15) / 16 * 16;
    const uint64_t o = (uint64_t)blk * per;
    if (o < f.tab_bytes)
      prefetch_run(reinterpret_cast<const uint8_t*>(f.cst) + o, min(per, f.tab_bytes - o));
  }
  __syncthreads();
  pdl_trigger();   // the next call's blocks may take SMs as soon as this call's leave
  pdl_wait();      // x, logits, y and the workspace belong to earlier kernels until here
  if (threadIdx.x == 0) F1_MARK(1);
  const uint32_t epoch = __ldcg(f.sync);
  uint32_t* cnt = sync_set(f.sync, epoch);

  // counters 1 and 2 of this call's set must be zero (counters 0 and 3 can move before
  // every block has passed this check)
  {
    int* bad = reinterpret_cast<int*>(part);
    if (tid == 0) {
      const int v = (__ldcg(cnt + 1) | __ldcg(cnt + 2)) != 0u;
      *bad = v;
      if (v) {
        atomicExch(p.status, BITSMOE_ERR_WORKSPACE_STATE);
      } else if (blk == 0) {
        p.status[0] = 0;
        sync_clear_next(f.sync, epoch);
      }
    }
    __syncthreads();
    if (*bad) {   // compute nothing; the projection rows already requested land before the block exits
      if (tid == 0)
        for (int st = 0; st < nst_pre; ++st)
          if (b0 + st * f.b_stage < b1) mbar_wait(bar_b + st, 0);
      return;
    }
    __syncthreads();   // part[] is reused below
  }
  uint16_t* xs = reinterpret_cast<uint16_t*>(fsm + f.off_xs);
  if (f.norm) {
    // pre-norm of the block: x = bf16(h / sqrt(mean(h^2) + eps)) (unit weight), in the same
    // arithmetic order as the separate norm/router kernel: 256 strided partial sums, warp sums,
    // eight warp totals in order
    float* red = part;
    if (tid < 256) {
      float ss = 0.f;
      for (int d = tid; d < p.D; d += 256) {
        const float v = f.hn[d];
        ss = fmaf(v, v, ss);
      }
      ss = warp_sum(ss);
      if (lane == 0) red[wid] = ss;
    }
    __syncthreads();
    float sum = 0.f;
    for (int w = 0; w < 8; ++w) sum += red[w];
    const float iv = rsqrtf(sum / (float)p.D + f.eps);
    for (int d = tid; d < p.D_pad; d += kFThreads) {
      uint32_t u32 = 0;
      if (d < p.D) {   // round to bf16, nearest even
        u32 = __float_as_uint(f.hn[d] * iv);
        u32 = (u32 + 0x7FFFu + ((u32 >> 16) & 1u)) & 0xFFFF0000u;
      }
      xs[d] = (uint16_t)(u32 >> 16);
      // block 0 leaves x in the workspace, where the separate norm/router step would put it
      if (blk == 0 && d < p.D) const_cast<uint16_t*>(p.x)[d] = (uint16_t)(u32 >> 16);
    }
    __syncthreads();
  }

  // Down items of all blocks (some past an expert's tiles), ordered by descending tile
  // position -- later tiles hold the wider units -- with the k routed experts of a position
  // together, and dealt snake-wise over the blocks (round m even: block blk takes item
  // m nb + blk, odd: m nb + nb - 1 - blk), so heavy and light tiles pair up on every block.
  const int ndi = p.k * f.ul_max_tiles;
  const int md = d_count(ndi, blk, nb);
  if (wid < kBW) {
    // ---- x into shared memory (unless the block normalised h itself), zero gate/up and s
    // a token row inside a batch starts at 2*D*t bytes: 16-byte loads only when x is 16-byte aligned
    const bool x16 = (reinterpret_cast<uintptr_t>(p.x) & 15) == 0;
    for (int i = tid; i < (f.norm ? 0 : p.D_pad / 8); i += kBW * 32) {
      uint4 v = make_uint4(0, 0, 0, 0);
      if (x16 && 8 * i + 8 <= p.D) {
        v = *reinterpret_cast<const uint4*>(p.x + 8 * i);
      } else {
        uint16_t t[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) t[u] = 8 * i + u < p.D ? p.x[8 * i + u] : (uint16_t)0;
        v = make_uint4(t[0] | (uint32_t)t[1] << 16, t[2] | (uint32_t)t[3] << 16, t[4] | (uint32_t)t[5] << 16,
                       t[6] | (uint32_t)t[7] << 16);
      }
      reinterpret_cast<uint4*>(xs)[i] = v;
    }
    {
      const size_t ng = (size_t)p.P * 2 * p.I_pad / 4, ns = (size_t)p.n_pad / 4;
      const float4 z4 = make_float4(0.f, 0.f, 0.f, 0.f);
      for (size_t i = (size_t)blk * kBW * 32 + tid; i < ng + ns; i += (size_t)nb * kBW * 32) {
        if (i < ng) reinterpret_cast<float4*>(p.gu)[i] = z4;
        else reinterpret_cast<float4*>(p.s)[i - ng] = z4;
      }
    }
    if (tid == 0) issue_b(nst_pre, f.b_nst);
    asm volatile("bar.sync 1, %0;" ::"r"(kBW * 32) : "memory");   // x is in shared memory
    // ---- B: z = Phi^T x for rows [b0, b1)
    for (int ri = wid; ri < b1 - b0; ri += kBW) {
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
    // the block's z rows are written: arrive at barrier 1 without waiting for the control warps
    asm volatile("bar.sync 3, %0;" ::"r"(kBW * 32) : "memory");
    if (tid == 0) F1_MARK(5);
    if (tid == 0 && !((f.dbg & 1) && blk == 0)) grid_arrive(cnt + 0);
  } else {
    const int ct = tid - kBW * 32;
    if (f.norm) {
      // this block's router logits (rows blk * epb ..), one control warp per row, the lane's
      // 16-byte chunks in the same order as the separate norm/router kernel; then every
      // block's logits are published through grid counter 4
      const int epb = (p.E + nb - 1) / nb, cw = ct >> 5, nch = p.D >> 3;
      for (int j = cw; j < epb; j += kCT / 32) {
        const int e = blk * epb + j;
        if (e >= p.E) break;
        const uint4* rp = reinterpret_cast<const uint4*>(f.wr + (size_t)e * p.D);
        float acc = 0.f;
        for (int c0 = 0; c0 < nch; c0 += 256) {
#pragma unroll
          for (int u = 0; u < 8; ++u) {
            const int c = c0 + u * 32 + lane;
            if (c < nch) {
              const uint4 v = __ldg(rp + c), xv = *reinterpret_cast<const uint4*>(xs + c * 8);
              acc = fmaf(bf16lo(v.x), bf16lo(xv.x), acc);
              acc = fmaf(bf16hi(v.x), bf16hi(xv.x), acc);
              acc = fmaf(bf16lo(v.y), bf16lo(xv.y), acc);
              acc = fmaf(bf16hi(v.y), bf16hi(xv.y), acc);
              acc = fmaf(bf16lo(v.z), bf16lo(xv.z), acc);
              acc = fmaf(bf16hi(v.z), bf16hi(xv.z), acc);
              acc = fmaf(bf16lo(v.w), bf16lo(xv.w), acc);
              acc = fmaf(bf16hi(v.w), bf16hi(xv.w), acc);
            }
          }
        }
        acc = warp_sum(acc);
        if (lane == 0) const_cast<float*>(p.logits)[e] = acc;
      }
      asm volatile("bar.sync 2, %0;" ::"r"(kCT) : "memory");
      if (ct == 0) grid_arrive(cnt + 3);
      grid_wait_ctl(cnt + 3, nb, p.status, seen + 3, cw, kCT, f.spin);
    }
    // ---- routing of the token
    route_token(p.logits, p.E, p.k, keys, sel_e, sel_w, ct);
    if (ct == 0) F1_MARK(3);
    // ---- staging: control thread s < nslot_c stages gate/up slot s; 32 + s < 32 + nslot_d prefetches down slot s
    const int A = p.k;
    const int nci = A * 2 * p.NRB * p.nseg;
    const int mc = nci > blk ? (nci - blk + nb - 1) / nb : 0;
    if (ct < f.nslot_c) {
      for (int m = ct; m < mc; m += f.nslot_c) {
        const CItem ci = c_item(p, blk + m * nb);
        const CStage* g = f.cst + ((size_t)ci.h * p.E + sel_e[ci.a]) * p.nseg + ci.sg;
        if (m == ct) {
          copy_crec(crec + ct, g);
          if ((f.dbg & 2) && crec[ct].bytes && !crec_ok<G>(p, f, crec[ct], ci.rb)) {
            crec[ct].bytes = 0;
            report_bounds(p.status);
          }
          if (crec[ct].bytes) c_stage<G>(p, f, crec[ct], ci.rb, rc + (size_t)ct * f.slot_c, bar_c + ct);
        } else {
          const uint32_t bytes = __ldg(&g->bytes);
          const uint64_t o = __ldg(&g->code0) + (uint64_t)ci.rb * __ldg(&g->rb_stride);
          if (bytes && (!(f.dbg & 2) || in_image(p, o, bytes))) prefetch_run(p.img + o, bytes);
        }
      }
    } else if (ct >= 32 && ct < 32 + f.nslot_d) {
      const int s = ct - 32;
      for (int m = s; m < md; m += f.nslot_d) {
        const int i = d_item(blk, m, nb), a = i % p.k, tile = f.ul_max_tiles - 1 - i / p.k;
        DStage r = load_drec(f.dst + (size_t)sel_e[a] * f.ul_max_tiles + tile);
        if ((f.dbg & 2) && r.bits && !drec_ok(p, f, r)) {
          r.bits = 0;
          report_bounds(p.status);
        }
        if (m == s) drec[s] = r;
        else if (r.bits) prefetch_run(p.img + r.code, (uint64_t)p.NRB * ul_chunks((int)r.bits) * kChunkBytes);
      }
    }
  }
  if (tid == 0) F1_MARK(4);
  grid_wait(cnt + 0, nb, p.status, seen + 0, f.spin);
  if (tid == 0) F1_MARK(6);
  // The projection rows are consumed; their buffer receives the first down tiles
  // (each staged by its slot's warp once that warp's gate/up items are done, so
  // that the copies do not delay the latency-bound z gathers) and, once the
  // first down tiles are done, this block's rows of Phi_dn.
  uint8_t* ers = r1;                       // [e1 - e0][n_pad] bf16
  uint8_t* dslots = r1 + f.off_d;          // [nslot_d][slot_d]

  // ---- C: gate/up items
  if (wid < f.nslot_c) {
    const int A = p.k;
    const int nci = A * 2 * p.NRB * p.nseg;
    const int mc = nci > blk ? (nci - blk + nb - 1) / nb : 0;
    uint8_t* slot = rc + (size_t)wid * f.slot_c;
    int16_t* cq = reinterpret_cast<int16_t*>(fsm + f.off_cq) + (size_t)wid * G * f.s16;
    int nst = 0;   // items staged into this slot so far (the mbarrier completes once per staging)
    for (int m = wid; m < mc; m += f.nslot_c) {
      const CItem ci = c_item(p, blk + m * nb);
      const CStage& r = crec[wid];
      if (m != wid) {   // a later item of this slot: its record replaces the previous one
        __syncwarp();
        if (lane == 0) {
          copy_crec(crec + wid, f.cst + ((size_t)ci.h * p.E + sel_e[ci.a]) * p.nseg + ci.sg);
          if ((f.dbg & 2) && crec[wid].bytes && !crec_ok<G>(p, f, crec[wid], ci.rb)) {
            crec[wid].bytes = 0;
            report_bounds(p.status);
          }
        }
        __syncwarp();
      }
      if (!r.bytes) continue;
      if (m != wid && lane == 0) {   // refill the slot (its previous item is done)
        fence_proxy_async();
        c_stage<G>(p, f, r, ci.rb, slot, bar_c + wid);
      }
      if (mbar_wait(bar_c + wid, (uint32_t)nst & 1u)) {
        c_compute<G>(p, f, r, ci.h, ci.rb, slot, cq, ci.a, lane);
      } else if (lane == 0) {
        atomicCAS(p.status, 0, BITSMOE_ERR_TIMEOUT);
      }
      ++nst;
    }
  }
  if (lane == 0 && wid < f.nslot_d && wid < md && drec[wid].bits) {
    fence_proxy_async();   // generic reads of the projection rows (before barrier 1), then async writes
    d_stage(p, f, drec[wid], dslots + (size_t)wid * f.slot_d, bar_d + wid);
  }
  if (tid == 0) F1_MARK(7);
  grid_barrier(cnt + 1, nb, p.status, seen + 1, f.spin);
  if (tid == 0) F1_MARK(8);

  // ---- D: down tiles, s += w * alpha * P_dn^T h.  Warp w works on slot w % nslot_d
  // over row blocks w / nslot_d, + nsub, ...; the slot's partial sums meet in shared memory.
  {
    const int nsub = kFWarps / f.nslot_d;
    const int sl = wid % f.nslot_d, sub = wid / f.nslot_d;
    uint8_t* slot = dslots + (size_t)sl * f.slot_d;
    int16_t* hqs = reinterpret_cast<int16_t*>(rc + (size_t)wid * f.d_h_bytes);   // C slots are free now
    float* hsc = reinterpret_cast<float*>(hqs + p.I_pad);
    int* hsum = reinterpret_cast<int*>(hsc + p.NRB);
    const int rounds = (md + f.nslot_d - 1) / f.nslot_d;
    // this block's rows of Phi_dn: once the first down tiles have read h (or now, without down tiles)
    auto issue_e = [&]() {
      if (tid == 0 && e1 > e0) {
        fence_proxy_async();
        mbar_expect_tx(bar_e, (uint32_t)(e1 - e0) * row_out);
        bulk_run(ers, reinterpret_cast<const uint8_t*>(p.basis_out) + (size_t)e0 * row_out,
                 (uint32_t)(e1 - e0) * row_out, bar_e);
      }
    };
    if (rounds == 0) issue_e();
    int staged = 0, cur_a = -1;
    for (int rd = 0; rd < rounds; ++rd) {
      const int m = sl + rd * f.nslot_d;
      DStage r;
      r.bits = 0;
      int a = 0;
      if (m < md) {
        const int i = d_item(blk, m, nb), tile = f.ul_max_tiles - 1 - i / p.k;
        a = i % p.k;
        r = rd == 0 ? drec[sl] : load_drec(f.dst + (size_t)sel_e[a] * f.ul_max_tiles + tile);
        if (rd > 0 && (f.dbg & 2) && r.bits && !drec_ok(p, f, r)) {
          r.bits = 0;
          if (sub == 0 && lane == 0) report_bounds(p.status);
        }
      }
      if (r.bits && rd > 0 && sub == 0 && lane == 0) {   // refill: the slot's previous tile is done
        fence_proxy_async();
        d_stage(p, f, r, slot, bar_d + sl);
      }
      float acc = 0.f;
      if (r.bits) {
        if (a != cur_a) {   // h of this expert's token for this warp's row blocks
          h_rows<G>(p, a, sub, nsub, hqs, hsc, hsum, lane);
          __syncwarp();
          cur_a = a;
        }
        if (mbar_wait(bar_d + sl, (uint32_t)staged & 1u)) {
          acc = ul_tile_rt<G>((int)r.bits, slot + lane * 16, p.NRB, sub, nsub, p.group, hqs, hsc, hsum,
                              reinterpret_cast<const uint32_t*>(slot + f.d_code_bytes + 256), lane);
        } else if (lane == 0) {
          atomicCAS(p.status, 0, BITSMOE_ERR_TIMEOUT);
        }
        ++staged;
      }
      part[wid * 32 + lane] = acc;
      __syncthreads();
      if (rd == 0) issue_e();
      if (r.bits && sub == 0) {
        float t = 0.f;
        for (int q = 0; q < nsub; ++q) t += part[(sl + q * f.nslot_d) * 32 + lane];
        const int* su = reinterpret_cast<const int*>(slot + f.d_code_bytes);
        const float al = reinterpret_cast<const float*>(su + 32)[lane];
        if (al != 0.f) atomicAdd(p.s + su[lane], sel_w[a] * al * t);   // one token: s[0][j]
      }
      __syncthreads();
    }
  }
  if (tid == 0) F1_MARK(9);
  grid_barrier(cnt + 2, nb, p.status, seen + 2, f.spin);
  if (tid == 0) F1_MARK(10);
  if (tid == 0 && blk == 0) sync_finish(f.sync);   // every block has read the epoch

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
  if (tid == 0) F1_MARK(11);
}

}  // namespace

namespace bmoe {

bool build_stage_tables(const uint8_t* img, std::vector<CStage>& cst, std::vector<DStage>& dst,
                        std::vector<uint8_t>& meta) {
  const ImageHeader& hd = *header_of(img);
  const ExpertDesc* desc = desc_of(img);
  const ItemRec* items = reinterpret_cast<const ItemRec*>(img + hd.off_items);
  const int E = hd.E;
  const int G = std::max(1, kRows / hd.group);
  // the metadata mirror: per gate/up item and row block [unit | alpha | G scale/zero rows],
  // per down tile [unit 32 | alpha 32 | NG scale/zero rows of 32], 16-byte multiples
  meta.clear();
  bool fits = true;
  auto put = [&](uint64_t off, uint32_t bytes) { meta.insert(meta.end(), img + off, img + off + bytes); };
  auto at = [&]() -> uint32_t {
    if (meta.size() > 0xFFFFFFF0ull) fits = false;
    return (uint32_t)meta.size();
  };
  cst.assign(2 * (size_t)E * hd.nseg, CStage{});
  for (int pi = 0; pi < 2 * E; ++pi) {
    const ExpertDesc& x = desc[pi];
    for (int q = 0; q < hd.nseg; ++q) {
      const ItemRec& it = items[(size_t)pi * hd.nseg + q];
      CStage& r = cst[(size_t)pi * hd.nseg + q];
      if (it.nr == 0) continue;
      r.code0 = x.code_base + it.byte0;
      r.unit0 = x.unit_off + (uint64_t)it.slot0 * 4;
      r.alpha0 = x.alpha_off + (uint64_t)it.slot0 * 4;
      r.sz0 = x.sz_off + (uint64_t)it.slot0 * 4;
      r.rb_stride = (uint32_t)x.rb_stride;
      r.sz_row = (uint32_t)x.nslots * 4;
      r.bytes = it.bytes;
      r.mb = (uint32_t)it.nslot * 4;
      r.nr = it.nr;
      int nls = 0;
      for (int k = 0; k < it.nr && k < kNumBk; ++k) {
        r.bits[k] = it.bits[k];
        r.ntl[k] = it.ntl[k];
        if (it.bits[k] < 16) nls += it.ntl[k] * rl_units(it.bits[k]);
      }
      r.nls = (uint16_t)nls;
      r.meta0 = at();
      for (int rb = 0; rb < hd.NRB && fits; ++rb) {
        const int g_base = (rb * kRows) / hd.group;
        put(r.unit0, r.mb);
        put(r.alpha0, r.mb);
        for (int gl = 0; gl < G; ++gl) put(r.sz0 + (uint64_t)(g_base + gl) * r.sz_row, r.mb);
      }
    }
  }
  dst.assign((size_t)E * hd.ul_max_tiles, DStage{});
  for (int e = 0; e < E; ++e) {
    const ExpertDesc& x = desc[2 * E + e];
    for (int k = 0; k < x.nbk; ++k) {
      const BucketDesc& bd = x.bk[k];
      for (int t = 0; t < bd.ntiles; ++t) {
        const int tile = bd.tile0 + t;
        if (tile >= hd.ul_max_tiles) continue;
        DStage& r = dst[(size_t)e * hd.ul_max_tiles + tile];
        const uint64_t slot = (uint64_t)bd.slot0 + (uint64_t)t * 32;
        r.code = x.code_base + bd.code_off + (uint64_t)t * hd.NRB * ul_chunks(bd.bits) * kChunkBytes;
        r.unit = x.unit_off + slot * 4;
        r.alpha = x.alpha_off + slot * 4;
        r.sz = x.sz_off + slot * 4;
        r.sz_row = (uint32_t)x.nslots * 4;
        r.bits = (uint32_t)bd.bits;
        r.meta = at();
        if (fits) {
          put(r.unit, 128);
          put(r.alpha, 128);
          for (int g = 0; g < hd.NG; ++g) put(r.sz + (uint64_t)g * r.sz_row, 128);
        }
      }
    }
  }
  if (!fits) meta.clear();
  return fits;
}

bool fused_plan(const ImageHeader& hd, int T, int top_k, int seg_bytes, int ul_max_chunks, int s16, int sms,
                FusedArgs* f) {
  if (T != 1 || sms < 1 || top_k > 32) return false;
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
  if (hd.ul_max_tiles < 1) return false;
  const int items_c = (A * 2 * hd.NRB * hd.nseg + sms - 1) / sms;
  const int items_d = (A * hd.ul_max_tiles + sms - 1) / sms;
  // fixed areas: mbarriers, staging records, routing, x, per-warp int16 activation tables, down partial sums
  size_t off = 512;
  f->off_rec = (int)off;
  off = align_up(off + (size_t)kFWarps * (sizeof(CStage) + sizeof(DStage)), 128);
  f->off_route = (int)off;
  off = align_up(off + (size_t)(hd.E + 2 * top_k) * 4, 128);
  f->off_xs = (int)off;
  off = align_up(off + row_in, 128);
  f->off_cq = (int)off;
  off = align_up(off + (size_t)kFWarps * G * s16 * 2, 128);
  f->off_part = (int)off;
  off = align_up(off + (size_t)kFWarps * 32 * 4, 128);
  const size_t r_b = (size_t)f->b_per * row_in;
  const size_t r_e = align_up((size_t)f->e_per * row_out, 128);
  f->off_d = (int)r_e;
  int nslot_d = 1;   // a power of two: the warps split evenly over the down slots
  while (nslot_d * 2 <= std::min(items_d, kFWarps)) nslot_d *= 2;
  size_t r1 = std::max(r_b, r_e + (size_t)nslot_d * f->slot_d);
  while (nslot_d > 1 && off + r1 > budget) {
    nslot_d /= 2;
    r1 = std::max(r_b, r_e + (size_t)nslot_d * f->slot_d);
  }
  f->off_r1 = (int)off;
  off = align_up(off + r1, 128);
  f->off_rc = (int)off;
  if (off >= budget) return false;
  int nslot_c = std::min(std::max(items_c, 1), kFWarps);
  while (nslot_c > 1 && off + (size_t)nslot_c * f->slot_c > budget) --nslot_c;
  size_t rc = std::max({(size_t)nslot_c * f->slot_c, (size_t)kFWarps * f->d_h_bytes, row_out * 2});
  if (off + rc > budget) return false;
  f->nslot_c = nslot_c;
  f->nslot_d = nslot_d;
  f->spin = kSpin;
  f->smem = (int)(off + rc);
  return true;
}

cudaError_t launch_fused(const Fwd& p, const FusedArgs& f, int sms, cudaStream_t st, bool pdl) {
  static std::mutex mu;
  static int done_smem[3] = {0, 0, 0};
  const int G = std::max(1, kRows / p.group);
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
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cudaLaunchConfig_t c2 = {};
    c2.gridDim = dim3(sms);
    c2.blockDim = dim3(kFThreads);
    c2.dynamicSmemBytes = f.smem;
    c2.stream = st;
    c2.attrs = attr;
    c2.numAttrs = pdl ? 1 : 0;
    return cudaLaunchKernelEx(&c2, kernel, p, f);
  };
  if (G == 1) return go(k_fused<1>, 0);
  if (G == 2) return go(k_fused<2>, 1);
  return go(k_fused<4>, 2);
}

}  // namespace bmoe

#ifdef BITSMOE_F2_TRACE
extern "C" int bitsmoe_f1_trace_read(void* dst) {
  return (int)cudaMemcpyFromSymbol(dst, g_f1_trace, sizeof(g_f1_trace));
}
#endif
