// Tensor-core expert factors for calls with several tokens (Eq. 3's expert
// factors between the shared-basis projection and the output basis):
//
//   gate/up[t][h][i] = sum_j p_hat_{h,e}[i, j] alpha_{h,e,j} z_h[t][j]          (h = gate, up)
//   h_t[i]           = SiLU(gate[t][0][i]) up[t][1][i]
//   s[t][j']        += g_{t,e} alpha_{dn,e,j'} sum_i p_hat_{dn,e}[i, j'] h_t[i]
//   p_hat[i, j]      = scale_{j,g(i)} (q_ij - zero_{j,g(i)})                     (group g along i)
//
// The integer codes q enter the MMA unchanged: a code c, written as the bit
// pattern of an fp16 number, is the subnormal c * 2^-24 (exact for c < 1024), so a
// byte permute turns four unpacked codes into four A elements and no code is
// converted or scaled.  The other operand is carried as an fp16 pair hi + lo
// (hi = the value truncated to 11 significant bits, lo = the rounded remainder:
// about 22 bits), scaled by a power of two 2^S chosen so that it stays inside the
// fp16 range; hi and lo are stacked along N (one MMA of width 2N per K-step) and
// the two halves of the fp32 TMEM accumulator are added in the epilogue, which
// multiplies by 2^(24 - S).  Zero points enter as per-token corrections.
//
// k_zgather: z of every token tile gathered in unit-slot order (one contiguous
// block of 128 slots x N tokens per K-block), so that the gate/up kernel stages it
// with one bulk copy.
//
// k_gu16 (gate/up, fused with SiLU(gate) * up): one item = (token tile of a routed
// expert, 128-row block); its K-blocks are 128 unit slots of gate, then of up.
//   A[i][slot] = q as fp16 subnormal (row-lane streams decoded in shared memory),
//   B[t][slot] = scale_{j,g} alpha_j z_h[t][j] 2^S as an fp16 pair,
//   gate/up    = acc 2^(24-S) - sum_slot zero_{j,g} B[t][slot] 2^-S.
// The epilogue forms h = SiLU(gate) up for the tile's 128 rows and writes it as the
// down kernel's B operand: an fp16 pair, swizzled, scaled per (token, row block),
// with its sum over the rows (for the down zero points).
//
// k_dn16 (down): one item = (token tile, 128 down slots = four unit-lane tiles); its
// K-blocks are the row blocks.  A[slot][i] = q (unit-lane streams), B = the h tile
// copied as it is; the group scale varies along K, so each row block's partial sum
// is read out of TMEM and scaled in registers, overlapping the next row block's MMAs;
// the item's result goes into s with g alpha by fp32 reductions (experts meet in s).
//
// Both expert kernels are persistent (one CTA per SM) and warp-specialised: a
// producer warp streams each K-block's bytes (codes, slot metadata, gathered z or
// the h tile) by bulk copies into a byte ring of shared memory several K-blocks
// ahead, an MMA warp issues tcgen05.mma from double-buffered A/B tiles, and the
// compute warps decode A, build B and run the epilogues (named barrier 1 among
// them; mbarriers between the roles; every wait bounded).  Every CTA derives the
// same list of token tiles (at most 32 tokens) from the routing (full tiles first,
// then partial tiles by size) and takes its items in a snake order over the list.
// Requires: every unit below 16 bits and the group a multiple of 128 rows (checked
// at upload), z also stored token-fastest (zT) and max |z| per token (zmax).
#include <cuda_fp16.h>

#include <algorithm>
#include <cstring>
#include <mutex>

#include "device.cuh"
#include "tc.cuh"

namespace {

constexpr int kGuCW = 16;                      // compute warps of the gate/up kernel
constexpr int kDnCW = 16;                      // compute warps of the down kernel
constexpr int kGuThreads = kGuCW * 32 + 64;    // and a producer warp and an MMA warp
constexpr int kDnThreads = kDnCW * 32 + 64;
constexpr int kNI = 16;                        // K-block records in flight (copies issued ahead)
constexpr uint32_t kAHalf = 128u * 128u;       // one 64-wide K half of A: 128 rows x 128 bytes
constexpr uint32_t kAStage = 2u * kAHalf;      // one A buffer (K = 128)
constexpr int kMaxNT = 64;                     // largest token tile

// Per-K-block timestamps of block 0 (%globaltimer; compute thread 0, producer lane 0, MMA
// lane 0), compiled in only with -DBITSMOE_X_TRACE for timing studies; without it X_MARK
// is empty.
#ifdef BITSMOE_X_TRACE
__device__ unsigned long long g_x_trace[2][2048][12];
#define X_MARK(k, i, m)                                                             \
  do {                                                                              \
    if (blockIdx.x == 0 && (i) < 2048) {                                            \
      unsigned long long t_;                                                        \
      asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t_));                        \
      g_x_trace[(k)][(i)][(m)] = t_;                                                \
    }                                                                               \
  } while (0)
#else
#define X_MARK(k, i, m) \
  do {                  \
  } while (0)
#endif

// kind::f16 instruction descriptor: f16 A and B, fp32 accumulator, both K-major, M = 128.
__host__ __device__ constexpr uint32_t idesc_f16(int n) {
  return (1u << 4) | ((uint32_t)(n >> 3) << 17) | ((uint32_t)(128 >> 4) << 24);
}

// Four codes (the bytes of q4) -> four fp16 whose bit patterns are the codes.
__device__ __forceinline__ uint2 codes_f16(uint32_t q4) {
  return make_uint2(__byte_perm(q4, 0u, 0x4140), __byte_perm(q4, 0u, 0x4342));
}

__device__ __forceinline__ uint32_t lds32(const uint8_t* p) { return *reinterpret_cast<const uint32_t*>(p); }

__device__ __forceinline__ void sts64(uint8_t* p, uint2 v) { *reinterpret_cast<uint2*>(p) = v; }

// fp32 pair (a, b) -> fp16 pair hi (truncation to 11 significant bits, exact in fp16
// inside its normal range) and lo (the remainder, rounded)
__device__ __forceinline__ void split_f16(float a, float b, uint32_t& hi, uint32_t& lo) {
  const float ha = __uint_as_float(__float_as_uint(a) & 0xFFFFE000u);
  const float hb = __uint_as_float(__float_as_uint(b) & 0xFFFFE000u);
  const __half2 h2 = __floats2half2_rn(ha, hb);
  const __half2 l2 = __floats2half2_rn(a - ha, b - hb);
  hi = *reinterpret_cast<const uint32_t*>(&h2);
  lo = *reinterpret_cast<const uint32_t*>(&l2);
}

// Power-of-two exponent S with m 2^S in [2^13, 2^14) (0 for m = 0 or not finite).
__device__ __forceinline__ int scale_exp(float m) {
  if (!(m > 0.f) || !(m < 3.0e38f)) return 0;
  int ex;
  frexpf(m, &ex);   // m = f 2^ex, f in [0.5, 1)
  return max(-100, min(100, 14 - ex));
}

// MMA width of a tile of nt tokens, and the rows of the h buffers an expert with c
// tokens takes (its full tiles and the width of its partial one).
__host__ __device__ __forceinline__ int tile_n(int nt) { return nt <= 16 ? 16 : nt <= 32 ? 32 : 64; }
__host__ __device__ __forceinline__ int tile_rows(int c, int NT) {
  const int rem = c % NT;
  return (c / NT) * NT + (rem ? tile_n(rem) : 0);
}

// ---------------------------------------------------------------------------
// Token tiles of the call, derived by every CTA from the published routing:
// active expert a (its index in p.active) has cnt tokens, in tiles of NT rows; its
// rows of the h buffers start at a 16-row-aligned base (tile_rows per expert).  Tile list: the full tiles
// in (a, tile) order, then each expert's partial tile by decreasing size.
// ---------------------------------------------------------------------------
struct Tiles {
  int* a_e;      // [A_max] expert id
  int* a_cnt;    // tokens
  int* a_pst;    // first entry in pair_list
  int* a_row;    // first row of the h buffers
  int* a_full;   // first full tile in the list
  uint32_t* tl;  // [max_tiles] a | tile << 16
  int* cnt;      // [4]: active experts, tiles, full tiles, rows used
};

__device__ void build_tiles(const Fwd& p, const XArgs& x, const Tiles& t) {
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  const int na = min(p.active[0], x.A_max);
  for (int a = tid; a < na; a += (int)blockDim.x) {
    const int e = p.active[1 + a];
    t.a_e[a] = e;
    const int c = p.expert_count[e];
    t.a_cnt[a] = c >= x.tc_min ? c : 0;   // fewer tokens: the dp2a kernels' expert (no tiles)
    t.a_pst[a] = p.expert_start[e];
  }
  __syncthreads();
  if (wid == 0) {
    int row = 0, full = 0, part = 0;
    for (int a0 = 0; a0 < na; a0 += 32) {
      const int a = a0 + lane;
      const int c = a < na ? t.a_cnt[a] : 0;
      const int r = tile_rows(c, x.NT), f = c / x.NT, q = (c % x.NT) != 0;
      int ri = r, fi = f, qi = q;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int vr = __shfl_up_sync(0xFFFFFFFFu, ri, o), vf = __shfl_up_sync(0xFFFFFFFFu, fi, o);
        const int vq = __shfl_up_sync(0xFFFFFFFFu, qi, o);
        if (lane >= o) {
          ri += vr;
          fi += vf;
          qi += vq;
        }
      }
      if (a < na) {
        t.a_row[a] = row + ri - r;
        t.a_full[a] = full + fi - f;
      }
      row += __shfl_sync(0xFFFFFFFFu, ri, 31);
      full += __shfl_sync(0xFFFFFFFFu, fi, 31);
      part += __shfl_sync(0xFFFFFFFFu, qi, 31);
    }
    if (lane == 0) {
      t.cnt[0] = na;
      t.cnt[1] = full + part;
      t.cnt[2] = full;
      t.cnt[3] = row;
    }
  }
  __syncthreads();
  const int F = t.cnt[2];
  if (t.cnt[1] <= x.max_tiles) {
    for (int a = tid; a < na; a += (int)blockDim.x) {
      const int c = t.a_cnt[a], nf = c / x.NT, rem = c - nf * x.NT;
      for (int tt = 0; tt < nf; ++tt) t.tl[t.a_full[a] + tt] = (uint32_t)a | ((uint32_t)tt << 16);
      if (rem) {
        int rank = 0;
        for (int b = 0; b < na; ++b) {
          const int rb = t.a_cnt[b] % x.NT;
          rank += rb != 0 && (rb > rem || (rb == rem && b < a));
        }
        t.tl[F + rank] = (uint32_t)a | ((uint32_t)nf << 16);
      }
    }
  }
  __syncthreads();
}

// Per (h, tile) entry q = h * ntiles + tile of the gathered z: its first float (vo[q]) and
// its first K-block among all entries (kbase[q]); vo[2 ntiles] / kbase[2 ntiles] are the
// totals.  Warp 0 of the calling CTA; the tile list is built.
__device__ void zv_offsets(const Fwd& p, const XArgs& x, const Tiles& t, int* vo, int* kbase) {
  const int lane = threadIdx.x & 31, ntiles = t.cnt[1];
  int run_v = 0, run_k = 0;
  for (int q0 = 0; q0 < 2 * ntiles; q0 += 32) {
    const int q = q0 + lane;
    int nkb = 0, N = 0;
    if (q < 2 * ntiles) {
      const int h = q >= ntiles, tau = q - h * ntiles;
      const uint32_t tw = t.tl[tau];
      const int a = (int)(tw & 0xFFFFu), tt = (int)(tw >> 16);
      nkb = (p.desc[h * p.E + t.a_e[a]].nslots + 127) / 128;
      N = tile_n(min(x.NT, t.a_cnt[a] - tt * x.NT));
    }
    int v = nkb * 128 * N, k = nkb, vi = v, ki = k;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int a1 = __shfl_up_sync(0xFFFFFFFFu, vi, o), a2 = __shfl_up_sync(0xFFFFFFFFu, ki, o);
      if (lane >= o) {
        vi += a1;
        ki += a2;
      }
    }
    if (q < 2 * ntiles) {
      vo[q] = run_v + vi - v;
      kbase[q] = run_k + ki - k;
    }
    run_v += __shfl_sync(0xFFFFFFFFu, vi, 31);
    run_k += __shfl_sync(0xFFFFFFFFu, ki, 31);
  }
  if (lane == 0) {
    vo[2 * ntiles] = run_v;
    kbase[2 * ntiles] = run_k;
  }
}

// Copy of an expert descriptor into shared memory (one thread; its loads are independent).
__device__ __forceinline__ void desc_copy(ExpertDesc* dst, const ExpertDesc* src) {
  static_assert(sizeof(ExpertDesc) % 8 == 0, "descriptor size");
  constexpr int kW = (int)(sizeof(ExpertDesc) / 8);
  uint2 v[kW];
#pragma unroll
  for (int w = 0; w < kW; ++w) v[w] = __ldg(reinterpret_cast<const uint2*>(src) + w);
#pragma unroll
  for (int w = 0; w < kW; ++w) reinterpret_cast<uint2*>(dst)[w] = v[w];
}

// Item r of this CTA in the snake order over `nitems` items (-1 past the end).
__device__ __forceinline__ int snake_item(int r, int nitems) {
  const int G = gridDim.x, b = blockIdx.x;
  const int it = r * G + ((r & 1) ? G - 1 - b : b);
  return it < nitems ? it : -1;
}

// Byte ring of staged K-blocks (one thread): allocate `bytes` (multiple of `al`) for
// the next K-block, given the live range [tail, head) (empty when nlive == 0).
__device__ __forceinline__ bool ring_alloc(uint32_t cap, uint32_t& head, uint32_t tail, int nlive, uint32_t bytes,
                                           uint32_t& pos) {
  if (nlive == 0) {
    if (bytes > cap) return false;
    pos = 0;
  } else if (head > tail) {
    if (head + bytes <= cap) pos = head;
    else if (bytes <= tail) pos = 0;
    else return false;
  } else {
    if (head + bytes <= tail) pos = head;
    else return false;
  }
  head = pos + bytes;
  return true;
}

// ---------------------------------------------------------------------------
// Roles: warps 0 .. kCW - 1 compute (decode A, build B, epilogues; they meet at named
// barrier 1), warp kCW streams the K-blocks' bytes (lane 0), warp kCW + 1 issues the
// MMAs (lane 0).  Barriers: full[s] (copies of record slot s landed), cons[s] (its
// ring bytes are free), ready[b] (A/B buffer b written), mdone[b] (its MMAs done).
// ---------------------------------------------------------------------------
constexpr int kFlagEnd = 8;

template <int NT_>
__device__ __forceinline__ void cbar() { asm volatile("bar.sync 1, %0;" ::"n"(NT_) : "memory"); }

__device__ __forceinline__ void sts128(uint8_t* p, uint2 lo, uint2 hi) {
  *reinterpret_cast<uint4*>(p) = make_uint4(lo.x, lo.y, hi.x, hi.y);
}

// ---------------------------------------------------------------------------
// Gather of z per token tile (feeds the gate/up kernel's B operand)
// ---------------------------------------------------------------------------
// zv[vo(h, tile) + (kb * 128 + slot) * N + t] = z_h[token t of the tile][unit of slot 128 kb + slot]
// (0 past the projection's slots or the tile's tokens): one work item = (h, tile, K-block).
constexpr int kZgThreads = 256;

__global__ void __launch_bounds__(kZgThreads) k_zgather(Fwd p, XArgs x) {
  extern __shared__ uint8_t zsm_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(zsm_raw) + 15) & ~(uintptr_t)15);
  Tiles tb;
  tb.a_e = reinterpret_cast<int*>(sm);
  tb.a_cnt = tb.a_e + x.A_max;
  tb.a_pst = tb.a_cnt + x.A_max;
  tb.a_row = tb.a_pst + x.A_max;
  tb.a_full = tb.a_row + x.A_max;
  tb.cnt = tb.a_full + x.A_max;
  tb.tl = reinterpret_cast<uint32_t*>(tb.cnt + 4);
  int* vo = reinterpret_cast<int*>(tb.tl + x.max_tiles);   // [2 max_tiles + 1]
  int* kbase = vo + 2 * x.max_tiles + 1;                   // [2 max_tiles + 1]
  int* su = kbase + 2 * x.max_tiles + 1;                   // [128] units of the item's slots
  int* tk = su + 128;                                      // [kMaxNT] its tokens
  const int tid = threadIdx.x;

  pdl_trigger();
  pdl_wait();   // routing and zT come from earlier kernels
  build_tiles(p, x, tb);
  const int ntiles = tb.cnt[1];
  if (ntiles > x.max_tiles || tb.cnt[3] > x.Rtot) {
    if (tid == 0) atomicCAS(p.status, 0, BITSMOE_ERR_WORKSPACE_STATE);
    return;
  }
  if (tid < 32) zv_offsets(p, x, tb, vo, kbase);
  __syncthreads();
  if ((uint64_t)(uint32_t)vo[2 * ntiles] > x.zv_floats) {
    if (tid == 0) atomicCAS(p.status, 0, BITSMOE_ERR_WORKSPACE_STATE);
    return;
  }
  const int nwork = kbase[2 * ntiles];
  for (int w = blockIdx.x; w < nwork; w += gridDim.x) {
    int lo = 0, hi = 2 * ntiles;   // entry q with kbase[q] <= w < kbase[q + 1]
    while (hi - lo > 1) {
      const int md = (lo + hi) >> 1;
      if (kbase[md] <= w) lo = md;
      else hi = md;
    }
    const int q = lo, h = q >= ntiles, tau = q - h * ntiles, kb = w - kbase[q];
    const uint32_t tw = tb.tl[tau];
    const int a = (int)(tw & 0xFFFFu), tt = (int)(tw >> 16);
    const int nt = min(x.NT, tb.a_cnt[a] - tt * x.NT), N = tile_n(nt), lgN = 31 - __clz(N);
    const ExpertDesc& xd = p.desc[h * p.E + tb.a_e[a]];
    const int s0 = 128 * kb, nval = min(128, xd.nslots - s0);
    __syncthreads();   // the previous item's su / tk are read
    if (tid < 128) su[tid] = tid < nval ? min(max(reinterpret_cast<const int*>(p.img + xd.unit_off)[s0 + tid], 0), p.n - 1) : -1;
    if (tid < kMaxNT) tk[tid] = tid < nt ? p.pair_list[tb.a_pst[a] + tt * x.NT + tid] / p.k : -1;
    __syncthreads();
    const float* zTh = p.zT + (size_t)h * p.n_pad * p.T;
    float* dst = x.zv + (uint32_t)vo[q] + (size_t)kb * 128 * N;
    for (int idx = tid; idx < (128 << lgN); idx += kZgThreads) {
      const int sl = idx >> lgN, t = idx & (N - 1);
      const int j = su[sl], tok = tk[t];
      dst[idx] = (j >= 0 && tok >= 0) ? __ldcg(zTh + (size_t)j * p.T + tok) : 0.f;
    }
  }
}

// ---------------------------------------------------------------------------
// Gate/up kernel
// ---------------------------------------------------------------------------
struct GuRec {                 // one staged K-block
  int item, h, kb, s0, nval;
  int flags;                   // 1: first K-block of the item, 2: first of this h, 4: last of the item, 8: end
  uint32_t pos, cbytes;        // ring offset: [z N x 128 x 4][codes cbytes][alpha nval][scale|zero nval]
  uint32_t vbytes;             // N x 512: the gathered z of the K-block (128 slots x N tokens, fp32)
  int nseg;                    // bucket segments: bits, first tile's slot (relative to s0), tiles, offset
  int sbits[kNumBk], sslot[kNumBk], snt[kNumBk], soff[kNumBk];
};

struct MRec {                  // what the MMA warp needs of the K-block in an A/B buffer
  int h, nval, flags, N;
};

struct GuCur {                 // the producer's position in this CTA's K-block sequence
  int r, item, e, rb, h, kb, nkb0, nkb1, tau, N;
};

struct GuItem {                // the item in progress
  int item, tau, rb, a, e, nt, N, R0, cur_h;
  int has[2];                  // the projection has slots (else its accumulator is never written)
  float bs[2];                 // 2^S of B
  float f24[2];                // 2^(24 - S)
  float fS[2];                 // 2^-S
};

// Shared-memory plan of k_gu16 (offsets from the 1024-aligned base).
struct GuPlan {
  uint32_t a, b, b_stage, ring, rec, mrec, swf, szr, tabs, tl, vo, item, tok, corr, xdc, bars, slot, total;
};
__host__ __device__ inline GuPlan gu_plan(const XArgs& x) {
  GuPlan s;
  uint32_t o = 0;
  s.a = o;
  o += 2 * kAStage;
  s.b_stage = 512u * (uint32_t)x.NT;   // [half 2][piece 2][NT rows][128 bytes]
  s.b = o;
  o += 2 * s.b_stage;
  s.ring = o;
  o += x.ring;
  s.rec = o;
  o += kNI * (uint32_t)sizeof(GuRec);
  s.mrec = o;
  o += 2 * (uint32_t)sizeof(MRec);
  s.swf = o;
  o += 2 * 128 * 4;
  s.szr = o;
  o += 2 * 128 * 4;
  s.tabs = o;
  o += 5u * (uint32_t)x.A_max * 4 + 16;
  s.tl = o;
  o += ((uint32_t)x.max_tiles * 4 + 15) & ~15u;
  s.vo = o;
  o += (2u * (2u * (uint32_t)x.max_tiles + 1) * 4 + 15) & ~15u;
  s.item = o;
  o += ((uint32_t)sizeof(GuItem) + 15) & ~15u;
  s.tok = o;
  o += kMaxNT * 4;
  s.corr = o;
  o += 2 * kMaxNT * 4;
  s.xdc = o;
  o += (2 * (uint32_t)sizeof(ExpertDesc) + 15) & ~15u;
  s.bars = o;
  o += (2 * kNI + 4) * 8;
  s.slot = o;
  o += 16;
  s.total = o;
  return s;
}

// Fill record `g` for the cursor's K-block (no copies yet; g.pos = the stream offset
// of its first code byte); returns its ring bytes.
__device__ uint32_t gu_record(const ExpertDesc* xdc, const GuCur& c, GuRec& g) {
  const ExpertDesc& xd = xdc[c.h];
  const int s0 = c.kb * 128, s1 = min(s0 + 128, xd.nslots);
  g.item = c.item;
  g.h = c.h;
  g.kb = c.kb;
  g.s0 = s0;
  g.nval = max(0, s1 - s0);
  const bool first = c.kb == 0 && (c.h == 0 || c.nkb0 == 0);
  const bool last = (c.h == 1 && c.kb == c.nkb1 - 1) || (c.h == 0 && c.kb == c.nkb0 - 1 && c.nkb1 == 0);
  g.flags = (first ? 1 : 0) | (c.kb == 0 ? 2 : 0) | (last ? 4 : 0);
  int ns = 0;
  uint32_t start = 0, end = 0;
  for (int k = 0; k < xd.nbk && g.nval > 0; ++k) {
    const BucketDesc& bd = xd.bk[k];
    const int lo = max(s0, bd.slot0), hi = min(s1, bd.slot0 + bd.nslots);
    if (lo >= hi) continue;
    const int U = rl_units(bd.bits), C = rl_chunks(bd.bits);
    const int t0 = (lo - bd.slot0) / U, t1 = (hi - 1 - bd.slot0) / U;
    const uint32_t so = (uint32_t)bd.code_off + (uint32_t)t0 * C * kChunkBytes;
    if (ns == 0) start = so;
    end = so + (uint32_t)(t1 - t0 + 1) * C * kChunkBytes;
    g.sbits[ns] = bd.bits;
    g.sslot[ns] = bd.slot0 + t0 * U - s0;
    g.snt[ns] = t1 - t0 + 1;
    g.soff[ns] = (int)(so - start);
    ++ns;
  }
  g.nseg = ns;
  g.cbytes = end - start;
  g.vbytes = (uint32_t)c.N * 512u;
  g.pos = start;
  return g.nval > 0 ? g.vbytes + g.cbytes + 8u * (uint32_t)g.nval : 0u;   // a placeholder copies nothing
}

__device__ void gu_load(const Fwd& p, const Tiles& t, int nitems, int x_NT, GuCur& c, ExpertDesc* xdc) {
  c.item = snake_item(c.r, nitems);
  if (c.item < 0) return;
  const int tau = c.item / p.NRB;
  c.rb = c.item - tau * p.NRB;
  c.tau = tau;
  const uint32_t tw = t.tl[tau];
  c.N = tile_n(min(x_NT, t.a_cnt[tw & 0xFFFFu] - (int)(tw >> 16) * x_NT));
  const int e = t.a_e[tw & 0xFFFFu];
  if (e != c.e) {   // the expert's gate and up descriptors into shared memory
    desc_copy(xdc, p.desc + e);
    desc_copy(xdc + 1, p.desc + p.E + e);
    c.e = e;
  }
  c.nkb0 = (xdc[0].nslots + 127) / 128;
  c.nkb1 = (xdc[1].nslots + 127) / 128;
  if (c.nkb0 + c.nkb1 == 0) c.nkb0 = 1;   // an item without slots still ends in an epilogue (h = 0)
  c.h = c.nkb0 > 0 ? 0 : 1;
  c.kb = 0;
}

__device__ void gu_next(const Fwd& p, const Tiles& t, int nitems, int x_NT, GuCur& c, ExpertDesc* xdc) {
  ++c.kb;
  if (c.kb < (c.h ? c.nkb1 : c.nkb0)) return;
  if (c.h == 0 && c.nkb1 > 0) {
    c.h = 1;
    c.kb = 0;
    return;
  }
  ++c.r;
  gu_load(p, t, nitems, x_NT, c, xdc);
}

// Two rows of each lane of a row-lane tile of B-bit codes -> A (fp16 codes).  Lane L
// holds rows 4L .. 4L + 3 (word w of its 16-byte chunk of each plane is row 4L + w); for
// rotation rho it decodes row 4L + ((rho + L / 2 + L / 8) & 3): any eight consecutive lanes
// then store to eight different rows mod 8 (the eight 16-byte positions of the 128-byte
// swizzle) and lanes L, L + 8, L + 16, L + 24 load different words (different banks).
// Below 8 bits every tile starts on an 8-slot boundary: two groups of four units make one
// 16-byte store.
template <int B>
__device__ __forceinline__ void dec_rl(const uint8_t* tile, int slot, int nval, uint8_t* A, int lane, int rho0) {
  constexpr int U = rl_units(B), C = rl_chunks(B), NG = U / 4;
  constexpr uint32_t kMask = B == 1 ? 0x01010101u : B == 2 ? 0x03030303u : B == 4 ? 0x0F0F0F0Fu : 0xFFFFFFFFu;
  // two rows a lane (rotations rho0 and rho0 + 2): two independent chains
  uint32_t w0[2], w1[2], w2[2];
  uint8_t* rowp[2];
  int rx[2];
#pragma unroll
  for (int v = 0; v < 2; ++v) {
    const int w = (rho0 + 2 * v + (lane >> 1) + (lane >> 3)) & 3;
    const int r = 4 * lane + w;
    rx[v] = r & 7;
    const uint8_t* src = tile + lane * 16 + 4 * w;
    w0[v] = lds32(src);
    w1[v] = C > 1 ? lds32(src + kChunkBytes) : 0u;
    w2[v] = C > 2 ? lds32(src + 2 * kChunkBytes) : 0u;
    rowp[v] = A + (uint32_t)(r >> 3) * 1024u + (uint32_t)rx[v] * 128u;
  }
  auto group = [&](int v, int k) -> uint32_t {
    if (B == 3) return (((k < 4 ? w0[v] : w1[v]) >> (2 * (k & 3))) & 0x03030303u) | (((w2[v] >> k) & 0x01010101u) << 2);
    if (B == 6)
      return (((k < 2 ? w0[v] : w1[v]) >> (4 * (k & 1))) & 0x0F0F0F0Fu) | (((w2[v] >> (2 * k)) & 0x03030303u) << 4);
    return (w0[v] >> (B * k)) & kMask;
  };
  if (B == 8) {
    if (slot >= 0 && slot < nval) {
#pragma unroll
      for (int v = 0; v < 2; ++v)
        sts64(rowp[v] + (uint32_t)(slot >> 6) * kAHalf + ((uint32_t)(((slot & 63) >> 3) ^ rx[v]) << 4) +
                  ((uint32_t)((slot >> 2) & 1) << 3),
              codes_f16(w0[v]));
    }
  } else {
#pragma unroll
    for (int kp = 0; kp < NG / 2; ++kp) {
      const int sl = slot + 8 * kp;
      if (sl < 0 || sl >= nval) continue;
#pragma unroll
      for (int v = 0; v < 2; ++v)
        sts128(rowp[v] + (uint32_t)(sl >> 6) * kAHalf + ((uint32_t)(((sl & 63) >> 3) ^ rx[v]) << 4),
               codes_f16(group(v, 2 * kp)), codes_f16(group(v, 2 * kp + 1)));
    }
  }
}

__global__ void __launch_bounds__(kGuThreads, 1) k_gu16(Fwd p, XArgs x) {
  constexpr int kCW = kGuCW, kCT = kGuCW * 32;
  extern __shared__ uint8_t gsm_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(gsm_raw) + 1023) & ~(uintptr_t)1023);
  const GuPlan L = gu_plan(x);
  uint8_t* ring = sm + L.ring;
  GuRec* rec = reinterpret_cast<GuRec*>(sm + L.rec);
  MRec* mrec = reinterpret_cast<MRec*>(sm + L.mrec);
  float* swf = reinterpret_cast<float*>(sm + L.swf);   // [2][128] scale * alpha * 2^S per slot
  float* szr = reinterpret_cast<float*>(sm + L.szr);   // [2][128] zero point per slot
  Tiles tb;
  tb.a_e = reinterpret_cast<int*>(sm + L.tabs);
  tb.a_cnt = tb.a_e + x.A_max;
  tb.a_pst = tb.a_cnt + x.A_max;
  tb.a_row = tb.a_pst + x.A_max;
  tb.a_full = tb.a_row + x.A_max;
  tb.cnt = tb.a_full + x.A_max;
  tb.tl = reinterpret_cast<uint32_t*>(sm + L.tl);
  int* vo = reinterpret_cast<int*>(sm + L.vo);   // [2 max_tiles + 1] first float of each (h, tile) in zv
  GuItem* it = reinterpret_cast<GuItem*>(sm + L.item);
  int* tok = reinterpret_cast<int*>(sm + L.tok);
  float* corr = reinterpret_cast<float*>(sm + L.corr);   // [2][kMaxNT]
  ExpertDesc* xdc = reinterpret_cast<ExpertDesc*>(sm + L.xdc);   // the producer's item: gate, up descriptors
  uint64_t* full = reinterpret_cast<uint64_t*>(sm + L.bars);   // [kNI]
  uint64_t* cons = full + kNI;                                 // [kNI]
  uint64_t* ready = cons + kNI;                                // [2]
  uint64_t* mdone = ready + 2;                                 // [2]
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(sm + L.slot);
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;

  pdl_trigger();
  pdl_wait();   // routing, z, zT and zmax come from earlier kernels
  build_tiles(p, x, tb);
  const int ntiles = tb.cnt[1];
  if (ntiles > x.max_tiles || tb.cnt[3] > x.Rtot) {
    if (tid == 0) atomicCAS(p.status, 0, BITSMOE_ERR_WORKSPACE_STATE);
    return;
  }
  const int nitems = ntiles * p.NRB;
  if (snake_item(0, nitems) < 0) return;
  if (wid == 0) zv_offsets(p, x, tb, vo, vo + 2 * x.max_tiles + 1);
  if (tid == 0) {
    for (int i = 0; i < kNI; ++i) {
      mbar_init_n(full + i, 1);
      mbar_init_n(cons + i, kCW);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init_n(ready + b, kCW);
      mbar_init_n(mdone + b, 1);
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (wid == kCW + 1) tmem_alloc(tmem_slot, 256);
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = *tmem_slot;
  bool ok = true;

  if (wid == kCW) {
    // ---- producer: K-block records and their copies into the ring, up to kNI ahead.  A
    // pass takes up to 8 consecutive K-blocks of one (item, projection): lane j computes
    // record j, lane 0 places them in the ring, lane 4 j + q issues copy q of record j.
    GuCur cur;
    cur.r = 0;
    cur.e = -1;
    cur.item = -1;
    if (lane == 0) gu_load(p, tb, nitems, x.NT, cur, xdc);
    int issued = 0, oldest = 0;
    uint32_t head = 0;
    auto retire = [&]() {   // wait until the oldest live K-block's ring bytes are free
      ok &= mbar_wait(cons + oldest % kNI, (uint32_t)(oldest / kNI) & 1u);
      ++oldest;
    };
    for (;;) {
      int nb = 0;
      if (lane == 0 && cur.item >= 0) {
        nb = min(8, (cur.h ? cur.nkb1 : cur.nkb0) - cur.kb);
        while (issued + nb - oldest > kNI) retire();
      }
      nb = __shfl_sync(0xFFFFFFFFu, nb, 0);
      if (nb == 0) {   // the end
        if (lane == 0) {
          while (issued - oldest >= kNI) retire();
          rec[issued % kNI].flags = kFlagEnd;
          mbar_expect_tx(full + issued % kNI, 0);
        }
        break;
      }
      GuCur cj;   // every lane: the cursor of its record
      cj.r = __shfl_sync(0xFFFFFFFFu, cur.r, 0);
      cj.item = __shfl_sync(0xFFFFFFFFu, cur.item, 0);
      cj.e = __shfl_sync(0xFFFFFFFFu, cur.e, 0);
      cj.rb = __shfl_sync(0xFFFFFFFFu, cur.rb, 0);
      cj.h = __shfl_sync(0xFFFFFFFFu, cur.h, 0);
      cj.kb = __shfl_sync(0xFFFFFFFFu, cur.kb, 0);
      cj.nkb0 = __shfl_sync(0xFFFFFFFFu, cur.nkb0, 0);
      cj.nkb1 = __shfl_sync(0xFFFFFFFFu, cur.nkb1, 0);
      cj.tau = __shfl_sync(0xFFFFFFFFu, cur.tau, 0);
      cj.N = __shfl_sync(0xFFFFFFFFu, cur.N, 0);
      __syncwarp();   // xdc written by lane 0
      const int kb0 = cj.kb;
      uint32_t bytes = 0, sstart = 0;
      if (lane < nb) {
        cj.kb = kb0 + lane;
        GuRec& g = rec[(issued + lane) % kNI];
        bytes = gu_record(xdc, cj, g);
        sstart = g.pos;
      }
      __syncwarp();
      // lane 0 places the records (sizes from lanes 0 .. nb - 1)
      uint32_t bsz[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) bsz[j] = __shfl_sync(0xFFFFFFFFu, bytes, j);
      int placed = 0;
      if (lane == 0) {   // retire only earlier passes' K-blocks: the pass shrinks to what fits
        for (int j = 0; j < nb; ++j) {
          uint32_t pos;
          const int q = issued + j;
          bool fit;
          for (;;) {
            fit = ring_alloc(x.ring, head, q > oldest ? rec[oldest % kNI].pos : head, q - oldest, bsz[j], pos);
            if (fit || oldest >= issued) break;
            retire();
          }
          if (!fit) break;
          rec[q % kNI].pos = pos;
          mbar_expect_tx(full + q % kNI, bsz[j]);
          ++placed;
        }
      }
      nb = __shfl_sync(0xFFFFFFFFu, placed, 0);
      __syncwarp();
      {
        const int j = lane >> 2, qc = lane & 3;
        const uint32_t ss = __shfl_sync(0xFFFFFFFFu, sstart, j & 7);
        if (j < nb) {
          const GuRec& g = rec[(issued + j) % kNI];
          const ExpertDesc& xd = xdc[cj.h];
          uint64_t* bar = full + (issued + j) % kNI;
          if (g.nval > 0) {   // copy 0: codes, 1: gathered z, 2: alphas, 3: scale/zero row
            fence_proxy_async();   // the ring space was last read by the generic proxy
            const uint32_t mb = 4u * (uint32_t)g.nval, cpos = g.pos + g.vbytes;
            if (qc == 0) {
              const uint8_t* src = p.img + xd.code_base + (size_t)cj.rb * xd.rb_stride + ss;
              for (uint32_t o = 0; o < g.cbytes; o += 32768u)
                bulk_g2s(ring + cpos + o, src + o, min(32768u, g.cbytes - o), bar);
            } else if (qc == 1) {
              const int vq = vo[cj.h * ntiles + cj.tau] + (kb0 + j) * 128 * cj.N;
              bulk_g2s(ring + g.pos, x.zv + (uint32_t)vq, g.vbytes, bar);
            } else if (qc == 2) {
              bulk_g2s(ring + cpos + g.cbytes, p.img + xd.alpha_off + (size_t)g.s0 * 4, mb, bar);
            } else {
              const int gg = (cj.rb * kRows) / p.group;
              bulk_g2s(ring + cpos + g.cbytes + mb, p.img + xd.sz_off + ((size_t)gg * xd.nslots + g.s0) * 4, mb, bar);
            }
          }
        }
      }
      issued += nb;
      __syncwarp();   // the descriptors may change below
      if (lane == 0) {
        for (int j = 0; j < nb; ++j) gu_next(p, tb, nitems, x.NT, cur, xdc);
      }
    }
  } else if (wid == kCW + 1) {
    // ---- MMA issuer
    if (lane == 0) {
      for (int i = 0;; ++i) {
        const int ab = i & 1;
        ok &= mbar_wait(ready + ab, (uint32_t)(i >> 1) & 1u);
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        const MRec m = mrec[ab];
        if (m.flags & kFlagEnd) break;
        if (m.N != 16 && m.N != 32 && m.N != 64) {   // never: the record is corrupt
          ok = false;
          mma_commit(mdone + ab);
          continue;
        }
        // B = [hi rows | lo rows] of each 64-slot half: one MMA of width 2N a K-step, the
        // two halves of the accumulator added in the epilogue
        const uint32_t idesc = idesc_f16(2 * m.N);
        const uint32_t acc = tmem + (uint32_t)(m.h * 2 * kMaxNT);
        const uint32_t a0 = smem_u32(sm + L.a + (size_t)ab * kAStage), b0 = smem_u32(sm + L.b + (size_t)ab * L.b_stage);
        const int kh = m.nval > 64 ? 2 : 1;
        for (int hf = 0; hf < kh; ++hf) {
#pragma unroll
          for (int k16 = 0; k16 < 4; ++k16)
            mma_f16(acc, sw128_desc(a0 + hf * kAHalf + 32 * k16), sw128_desc(b0 + (uint32_t)hf * 2u * m.N * 128u + 32u * k16),
                     idesc, ((m.flags & 2) && hf == 0 && k16 == 0) ? 0u : 1u);
        }
        mma_commit(mdone + ab);
      }
    }
  } else {
    // ---- compute warps
    float cs = 0.f;   // this thread's zero-point correction of its token, current projection

    // epilogue of the item in `it` (its last K-block is i1): h = SiLU(gate) up of the tile's
    // rows, written as the down kernel's B tile with its per-(token, row block) sums and scale
    auto epilogue = [&](int i1) {
      if (cs != 0.f) atomicAdd(corr + it->cur_h * kMaxNT + (tid & (it->N - 1)), cs);
      cs = 0.f;
      ok &= mbar_wait(mdone + (i1 & 1), (uint32_t)(i1 >> 1) & 1u);
      cbar<kCT>();
      asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      const int N = it->N, nt = it->nt, rb = it->rb;
      float* hs = reinterpret_cast<float*>(sm + L.a);   // [N][128] h of the tile (the A buffers are free)
      {
        const int q = wid & 3, r = 32 * q + lane, ig = rb * kRows + r;
        const uint32_t tl = tmem + ((uint32_t)(32 * q) << 16);
        for (int c0 = 8 * (wid >> 2); c0 < N; c0 += 8 * (kCW / 4)) {
          uint32_t vg[8], vu[8], wg[8], wu[8];
#pragma unroll
          for (int u = 0; u < 8; ++u) vg[u] = vu[u] = wg[u] = wu[u] = 0u;
          if (it->has[0]) {
            tmem_ld8(tl + (uint32_t)c0, vg);
            tmem_ld8(tl + (uint32_t)(N + c0), wg);
          }
          if (it->has[1]) {
            tmem_ld8(tl + (uint32_t)(2 * kMaxNT + c0), vu);
            tmem_ld8(tl + (uint32_t)(2 * kMaxNT + N + c0), wu);
          }
#pragma unroll
          for (int u = 0; u < 8; ++u) {
            const int t = c0 + u;
            const float ag = __uint_as_float(vg[u]) + __uint_as_float(wg[u]);
            const float au = __uint_as_float(vu[u]) + __uint_as_float(wu[u]);
            const float g = ag * it->f24[0] - corr[t] * it->fS[0];
            const float uu = au * it->f24[1] - corr[kMaxNT + t] * it->fS[1];
            hs[t * 128 + r] = (t < nt && ig < p.I) ? g / (1.f + __expf(-g)) * uu : 0.f;
          }
        }
      }
      asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
      cbar<kCT>();
      for (int t = wid; t < N; t += kCW) {   // one warp per token row: 4 rows a lane
        const float4 v = *reinterpret_cast<const float4*>(hs + t * 128 + 4 * lane);
        float am = fmaxf(fmaxf(fabsf(v.x), fabsf(v.y)), fmaxf(fabsf(v.z), fabsf(v.w)));
        float sum = (v.x + v.y) + (v.z + v.w);
#pragma unroll
        for (int o = 16; o; o >>= 1) {
          am = fmaxf(am, __shfl_xor_sync(0xFFFFFFFFu, am, o));
          sum += __shfl_xor_sync(0xFFFFFFFFu, sum, o);
        }
        const int S = scale_exp(am);
        const float sc = ldexpf(1.f, S);
        uint32_t h0, l0, h1, l1;
        split_f16(v.x * sc, v.y * sc, h0, l0);
        split_f16(v.z * sc, v.w * sc, h1, l1);
        const int i0 = 4 * lane, half = i0 >> 6, c8 = (i0 & 63) >> 3;
        uint8_t* base = x.hb + ((size_t)rb * x.Rtot + it->R0) * 512 + (uint32_t)half * 2u * N * 128u +
                        (uint32_t)(t & 7) * 128u + ((uint32_t)(c8 ^ (t & 7)) << 4) + (uint32_t)(i0 & 4) * 2u;
        *reinterpret_cast<uint2*>(base + (uint32_t)(t >> 3) * 1024u) = make_uint2(h0, h1);
        *reinterpret_cast<uint2*>(base + (uint32_t)((N + t) >> 3) * 1024u) = make_uint2(l0, l1);
        if (lane == 0) x.hs[(size_t)rb * x.Rtot + it->R0 + t] = make_float2(sum, ldexpf(1.f, 24 - S));
      }
      cbar<kCT>();   // the A buffers and the item state are reused
    };

    for (int i = 0;; ++i) {
      if (tid == 0) X_MARK(0, i, 0);
      const int ab = i & 1;
      ok &= mbar_wait(full + i % kNI, (uint32_t)(i / kNI) & 1u);
      if (tid == 0) X_MARK(0, i, 1);
      const GuRec& g = rec[i % kNI];
      const int flags = g.flags;
      if (flags & kFlagEnd) {
        if (i > 0) epilogue(i - 1);
        if (i >= 2) ok &= mbar_wait(mdone + ab, (uint32_t)((i - 2) >> 1) & 1u);
        if (tid == 0) mrec[ab].flags = kFlagEnd;
        __syncwarp();
        if (lane == 0) mbar_arrive(ready + ab);
        break;
      }
      const int h = g.h, nval = g.nval;
      if (flags & 1) {
        if (i > 0) epilogue(i - 1);
        if (wid == 0) {   // item prologue: the tile's tokens and the B scales
          const int item = g.item, tau = item / p.NRB, rb = item - tau * p.NRB;
          const uint32_t tw = tb.tl[tau];
          const int a = (int)(tw & 0xFFFFu), tt = (int)(tw >> 16), e = tb.a_e[a];
          const int nt = min(x.NT, tb.a_cnt[a] - tt * x.NT);
          float zm0 = 0.f, zm1 = 0.f;
          for (int t = lane; t < kMaxNT; t += 32) {
            int tk = 0;
            if (t < nt) {
              tk = p.pair_list[tb.a_pst[a] + tt * x.NT + t] / p.k;
              zm0 = fmaxf(zm0, __uint_as_float(__ldcg(x.zmax + tk)));
              zm1 = fmaxf(zm1, __uint_as_float(__ldcg(x.zmax + p.T + tk)));
            }
            tok[t] = tk;
            corr[t] = 0.f;
            corr[kMaxNT + t] = 0.f;
          }
#pragma unroll
          for (int o = 16; o; o >>= 1) {
            zm0 = fmaxf(zm0, __shfl_xor_sync(0xFFFFFFFFu, zm0, o));
            zm1 = fmaxf(zm1, __shfl_xor_sync(0xFFFFFFFFu, zm1, o));
          }
          if (lane == 0) {
            it->item = item;
            it->tau = tau;
            it->rb = rb;
            it->a = a;
            it->e = e;
            it->nt = nt;
            it->N = tile_n(nt);
            it->R0 = tb.a_row[a] + tt * x.NT;
            it->cur_h = h;
            const float zm[2] = {zm0, zm1};
#pragma unroll
            for (int hh = 0; hh < 2; ++hh) {
              it->has[hh] = p.desc[hh * p.E + e].nslots > 0 || (hh == 0 && p.desc[p.E + e].nslots == 0);
              const int S = scale_exp(x.msa[hh * p.E + e] * zm[hh]);
              it->bs[hh] = ldexpf(1.f, S);
              it->f24[hh] = ldexpf(1.f, 24 - S);
              it->fS[hh] = ldexpf(1.f, -S);
            }
          }
        }
        cbar<kCT>();
      } else if (flags & 2) {   // first K-block of up: gate's corrections are complete
        if (cs != 0.f) atomicAdd(corr + it->cur_h * kMaxNT + (tid & (it->N - 1)), cs);
        cs = 0.f;
        cbar<kCT>();
        if (tid == 0) it->cur_h = h;
        cbar<kCT>();
      }
      if (tid == 0) X_MARK(0, i, 2);
      if (i >= 2) ok &= mbar_wait(mdone + ab, (uint32_t)((i - 2) >> 1) & 1u);   // A/B buffer ab is free
      if (tid == 0) X_MARK(0, i, 3);
      const float* sv = reinterpret_cast<const float*>(ring + g.pos);   // gathered z [128 slots][N]
      const uint8_t* st = ring + g.pos + g.vbytes;                      // codes
      const float* sal = reinterpret_cast<const float*>(st + g.cbytes);
      const uint32_t* ssz = reinterpret_cast<const uint32_t*>(sal + nval);
      // B items: thread = (token row t, 8-slot chunks c = c0, c0 + cstep, ..); a thread keeps its t
      const int N = it->N;
      const int lgN = 31 - __clz(N);
      const int bt = tid & (N - 1), cstep = kCT >> lgN, c0 = tid >> lgN;
      const int nch = nval > 64 ? 16 : 8;
      constexpr int kMaxC = (16 * kMaxNT + kCT - 1) / kCT;   // most items a thread takes (N = 64)
      if (tid == 0) X_MARK(0, i, 8);
      if (tid < 128) {   // per-slot factors of B
        float wv = 0.f, zr = 0.f;
        if (tid < nval) {
          const uint32_t szw = ssz[tid];
          wv = __half2float(__ushort_as_half((unsigned short)(szw & 0xFFFFu))) * sal[tid] * it->bs[h];
          zr = __half2float(__ushort_as_half((unsigned short)(szw >> 16)));
        }
        swf[ab * 128 + tid] = wv;
        szr[ab * 128 + tid] = zr;
      }
      if (tid == 0) X_MARK(0, i, 9);
      // A: one warp per row-lane tile; slots past the last tile are zero up to the MMA's K
      uint8_t* A = sm + L.a + (size_t)ab * kAStage;
      {
        const int kend = nval > 64 ? 128 : 64;
        for (int q = tid; q < 128 * ((kend - nval) >> 2); q += kCT) {
          const int r = q & 127, sl = nval + 4 * (q >> 7);
          sts64(A + (uint32_t)(sl >> 6) * kAHalf + (uint32_t)(r >> 3) * 1024u + (uint32_t)(r & 7) * 128u +
                    ((uint32_t)(((sl & 63) >> 3) ^ (r & 7)) << 4) + ((uint32_t)((sl >> 2) & 1) << 3),
                make_uint2(0u, 0u));
        }
        int ntl = 0;
        for (int s = 0; s < g.nseg; ++s) ntl += g.snt[s];
        for (int ti = wid; ti < 2 * ntl; ti += kCW) {   // items: (tile, rotations rho and rho + 2)
          int s = 0, tt = ti >> 1;
          while (tt >= g.snt[s]) tt -= g.snt[s++];
          const int b = g.sbits[s];
          const uint8_t* tile = st + g.soff[s] + tt * rl_chunks(b) * kChunkBytes;
          const int slot = g.sslot[s] + tt * rl_units(b), rho = ti & 1;
          switch (b) {
            case 1: dec_rl<1>(tile, slot, nval, A, lane, rho); break;
            case 2: dec_rl<2>(tile, slot, nval, A, lane, rho); break;
            case 3: dec_rl<3>(tile, slot, nval, A, lane, rho); break;
            case 4: dec_rl<4>(tile, slot, nval, A, lane, rho); break;
            case 6: dec_rl<6>(tile, slot, nval, A, lane, rho); break;
            default: dec_rl<8>(tile, slot, nval, A, lane, rho); break;
          }
        }
      }
      if (tid == 0) X_MARK(0, i, 4);
      cbar<kCT>();   // slot factors
      if (tid == 0) X_MARK(0, i, 5);
      // B from the requested z: scale * alpha * 2^S * z as an fp16 pair
      uint8_t* Bb = sm + L.b + (size_t)ab * L.b_stage;
      {
        const float* wf = swf + ab * 128;
        const float* zf = szr + ab * 128;
#pragma unroll
        for (int ci = 0; ci < kMaxC; ++ci) {
          const int c = c0 + ci * cstep, sl0 = 8 * c;
          if (c >= nch) continue;
          uint32_t hw[4] = {0u, 0u, 0u, 0u}, lw[4] = {0u, 0u, 0u, 0u};
          if (sl0 < nval) {
            const float4 wa = *reinterpret_cast<const float4*>(wf + sl0), wb = *reinterpret_cast<const float4*>(wf + sl0 + 4);
            const float4 za = *reinterpret_cast<const float4*>(zf + sl0), zb = *reinterpret_cast<const float4*>(zf + sl0 + 4);
            const float wv[8] = {wa.x, wa.y, wa.z, wa.w, wb.x, wb.y, wb.z, wb.w};
            const float zr[8] = {za.x, za.y, za.z, za.w, zb.x, zb.y, zb.z, zb.w};
#pragma unroll
            for (int m = 0; m < 4; ++m) {
              const float v0 = wv[2 * m] * sv[(sl0 + 2 * m) * N + bt], v1 = wv[2 * m + 1] * sv[(sl0 + 2 * m + 1) * N + bt];
              cs = fmaf(zr[2 * m], v0, cs);
              cs = fmaf(zr[2 * m + 1], v1, cs);
              split_f16(v0, v1, hw[m], lw[m]);
            }
          }
          const uint32_t off = (uint32_t)(c >> 3) * 2u * (uint32_t)N * 128u + (uint32_t)(bt >> 3) * 1024u +
                               (uint32_t)(bt & 7) * 128u + ((uint32_t)((c & 7) ^ (bt & 7)) << 4);
          *reinterpret_cast<uint4*>(Bb + off) = make_uint4(hw[0], hw[1], hw[2], hw[3]);
          *reinterpret_cast<uint4*>(Bb + (uint32_t)N * 128u + off) = make_uint4(lw[0], lw[1], lw[2], lw[3]);
        }
      }
      if (tid == 0) X_MARK(0, i, 6);
      if (tid == 0) {
        MRec m;
        m.h = h;
        m.nval = nval;
        m.flags = flags;
        m.N = N;
        mrec[ab] = m;
      }
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");   // generic writes -> tensor-core reads
      asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(ready + ab);
        mbar_arrive(cons + i % kNI);
      }
      if (tid == 0) X_MARK(0, i, 7);
    }
  }
  if (!ok) atomicCAS(p.status, 0, BITSMOE_ERR_TIMEOUT);
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  if (wid == kCW + 1) tmem_dealloc(tmem, 256);
}

// ---------------------------------------------------------------------------
// Down kernel
// ---------------------------------------------------------------------------
struct DnRec {                 // one staged row block of an item
  int item, rb, flags;         // flags: 1 first row block of the item, 4 last, 8 end
  uint32_t pos;                // ring offset: [h tile: half 2, piece 2, N rows, 128 B][codes cb][scale|zero 128 x 4][h sums N x 8]
  uint32_t cb, N;
  int bits[4], coff[4];        // the item's four unit-lane tiles (bits 0: no tile)
};

struct DnMRec {
  int N, flags;
  uint32_t pos;
  int pad_;
};

struct DnCur {
  int r, item, tau, mt, rb, e, N, R0;
};

struct DnItem {                // per item (two, by parity: one finishing while the next starts)
  int nt, N, nsl, pad_;
  int tok[kMaxNT];
  float pw[kMaxNT];
  int unit[128];
  float alpha[128];
};

struct DnPlan {
  uint32_t a, ring, rec, mrec, hsm, tabs, tl, dbase, item, xdc, bars, slot, total;
};
__host__ __device__ inline DnPlan dn_plan(const XArgs& x) {
  DnPlan s;
  uint32_t o = 0;
  s.a = o;
  o += 2 * kAStage;
  s.ring = o;
  o += x.ring;
  s.rec = o;
  o += kNI * (uint32_t)sizeof(DnRec);
  s.mrec = o;
  o += 2 * (uint32_t)sizeof(DnMRec);
  s.hsm = o;
  o += 2 * kMaxNT * 8;
  s.tabs = o;
  o += 5u * (uint32_t)x.A_max * 4 + 16;
  s.tl = o;
  o += ((uint32_t)x.max_tiles * 4 + 15) & ~15u;
  s.dbase = o;
  o += (((uint32_t)x.max_tiles + 1) * 4 + 15) & ~15u;
  s.item = o;
  o += 2 * (((uint32_t)sizeof(DnItem) + 15) & ~15u);
  s.xdc = o;
  o += ((uint32_t)sizeof(ExpertDesc) + 15) & ~15u;
  s.bars = o;
  o += (2 * kNI + 4) * 8;
  s.slot = o;
  o += 16;
  s.total = o;
  return s;
}

__device__ void dn_load(const Fwd& p, const XArgs& x, const Tiles& t, const int* dbase, int ntiles, int nitems,
                        DnCur& c, ExpertDesc* xdc) {
  c.item = snake_item(c.r, nitems);
  if (c.item < 0) return;
  int lo = 0, hi = ntiles;   // last tile whose first item is at or before c.item
  while (hi - lo > 1) {
    const int m = (lo + hi) >> 1;
    if (dbase[m] <= c.item) lo = m;
    else hi = m;
  }
  c.tau = lo;
  c.mt = c.item - dbase[lo];
  const uint32_t tw = t.tl[lo];
  const int a = (int)(tw & 0xFFFFu), tt = (int)(tw >> 16);
  const int e = t.a_e[a];
  if (e != c.e) {   // the expert's down descriptor into shared memory
    desc_copy(xdc, p.desc + 2 * p.E + e);
    c.e = e;
  }
  c.N = tile_n(min(x.NT, t.a_cnt[a] - tt * x.NT));
  c.R0 = t.a_row[a] + tt * x.NT;
  c.rb = 0;
}

// Eight codes of rows kk .. kk + 7 (kk a multiple of 8 inside the row block) -> A[slot m]
// in one 16-byte store; the lanes of a warp hold consecutive slots, so eight lanes cover
// the eight 16-byte positions of the swizzle.
__device__ __forceinline__ void store_a8(uint8_t* A, int m, int kk, uint2 lo, uint2 hi) {
  sts128(A + (uint32_t)(kk >> 6) * kAHalf + (uint32_t)(m >> 3) * 1024u + (uint32_t)(m & 7) * 128u +
             ((uint32_t)(((kk & 63) >> 3) ^ (m & 7)) << 4),
         lo, hi);
}
// Unit-lane rows 32 hq .. 32 hq + 31 of one slot (its 16-byte chunks at `ln`, chunk c
// at ln + 512 c) -> A row m (fp16 codes).
template <int B>
__device__ __forceinline__ void dec_ul(const uint8_t* ln, int hq, int m, uint8_t* A) {
  if (B == 3) {   // low 2-bit plane: chunk hq / 2, a word = 16 rows; high bit: chunk 2, a word = 32 rows
    const uint8_t* lo = ln + (hq >> 1) * kChunkBytes;
    const uint32_t wh = lds32(ln + 2 * kChunkBytes + 4 * hq);
#pragma unroll
    for (int w2 = 0; w2 < 2; ++w2) {
      const int w = 2 * (hq & 1) + w2;   // word of the low chunk: rows 64 (hq / 2) + 16 w ..
      const uint32_t wl = lds32(lo + 4 * w);
#pragma unroll
      for (int kp = 0; kp < 2; ++kp) {
        uint32_t q[2];
#pragma unroll
        for (int u = 0; u < 2; ++u) {
          const int k = 2 * kp + u;
          q[u] = ((wl >> (2 * k)) & 0x03030303u) | (((wh >> (4 * w2 + k)) & 0x01010101u) << 2);
        }
        store_a8(A, m, 32 * hq + 16 * w2 + 8 * kp, codes_f16(q[0]), codes_f16(q[1]));
      }
    }
  } else if (B == 6) {   // low 4-bit plane: chunk hq, a word = 8 rows; high 2 bits: chunk 4 + hq / 2, a word = 16 rows
    const uint8_t* lo = ln + hq * kChunkBytes;
    const uint8_t* hi = ln + (4 + (hq >> 1)) * kChunkBytes;
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      const int r0 = 32 * (hq & 1) + 8 * w;   // row inside the 64 rows of the high chunk
      const uint32_t wl = lds32(lo + 4 * w), wh = lds32(hi + 4 * (r0 >> 4));
      uint32_t q[2];
#pragma unroll
      for (int k = 0; k < 2; ++k) {
        const int rr = r0 + 4 * k;
        q[k] = ((wl >> (4 * k)) & 0x0F0F0F0Fu) | (((wh >> (2 * ((rr & 15) >> 2))) & 0x03030303u) << 4);
      }
      store_a8(A, m, 32 * hq + 8 * w, codes_f16(q[0]), codes_f16(q[1]));
    }
  } else if (B == 8) {   // a word = 4 rows: two words a store
#pragma unroll
    for (int wi = 0; wi < 8; wi += 2) {
      const int gw = 8 * hq + wi;
      const uint32_t a = lds32(ln + (gw >> 2) * kChunkBytes + 4 * (gw & 3));
      const uint32_t b = lds32(ln + ((gw + 1) >> 2) * kChunkBytes + 4 * ((gw + 1) & 3));
      store_a8(A, m, gw * 4, codes_f16(a), codes_f16(b));
    }
  } else {   // 1, 2, 4: chunk c covers rows 128c/B .., a word 32/B rows, group k at bit B k
    constexpr int RPW = 32 / B;
    constexpr uint32_t kMask = B == 1 ? 0x01010101u : B == 2 ? 0x03030303u : 0x0F0F0F0Fu;
#pragma unroll
    for (int wi = 0; wi < B; ++wi) {
      const int gw = B * hq + wi;
      const uint32_t wv = lds32(ln + (gw >> 2) * kChunkBytes + 4 * (gw & 3));
#pragma unroll
      for (int kp = 0; kp < RPW / 8; ++kp)
        store_a8(A, m, gw * RPW + 8 * kp, codes_f16((wv >> (B * 2 * kp)) & kMask),
                 codes_f16((wv >> (B * (2 * kp + 1))) & kMask));
    }
  }
}

__global__ void __launch_bounds__(kDnThreads, 1) k_dn16(Fwd p, XArgs x) {
  constexpr int kCW = kDnCW, kCT = kDnCW * 32;
  constexpr int kOut = kMaxNT / 8 / (kCT / 128);   // 8-column chunks of a thread's accumulator columns
  extern __shared__ uint8_t dsm_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(dsm_raw) + 1023) & ~(uintptr_t)1023);
  const DnPlan L = dn_plan(x);
  uint8_t* ring = sm + L.ring;
  DnRec* rec = reinterpret_cast<DnRec*>(sm + L.rec);
  DnMRec* mrec = reinterpret_cast<DnMRec*>(sm + L.mrec);
  float2* hsm = reinterpret_cast<float2*>(sm + L.hsm);   // [2][kMaxNT] (h sum, 2^(24 - S)) of a row block
  Tiles tb;
  tb.a_e = reinterpret_cast<int*>(sm + L.tabs);
  tb.a_cnt = tb.a_e + x.A_max;
  tb.a_pst = tb.a_cnt + x.A_max;
  tb.a_row = tb.a_pst + x.A_max;
  tb.a_full = tb.a_row + x.A_max;
  tb.cnt = tb.a_full + x.A_max;
  tb.tl = reinterpret_cast<uint32_t*>(sm + L.tl);
  int* dbase = reinterpret_cast<int*>(sm + L.dbase);   // [ntiles + 1] first item of each tile
  const uint32_t isz = ((uint32_t)sizeof(DnItem) + 15) & ~15u;
  ExpertDesc* xdc = reinterpret_cast<ExpertDesc*>(sm + L.xdc);   // the producer's item: down descriptor
  uint64_t* full = reinterpret_cast<uint64_t*>(sm + L.bars);
  uint64_t* cons = full + kNI;
  uint64_t* ready = cons + kNI;
  uint64_t* mdone = ready + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(sm + L.slot);
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  const int m = tid & 127, hq = (tid >> 7) & 3;   // A row / accumulator lane, and quarter of the rows or columns

  pdl_trigger();
  pdl_wait();   // routing and the h tiles come from earlier kernels
  build_tiles(p, x, tb);
  const int ntiles = tb.cnt[1];
  if (ntiles > x.max_tiles || tb.cnt[3] > x.Rtot) {
    if (tid == 0) atomicCAS(p.status, 0, BITSMOE_ERR_WORKSPACE_STATE);
    return;
  }
  if (wid == 0) {   // items per tile: the expert's 128-slot groups of down tiles
    int run = 0;
    for (int t0 = 0; t0 < ntiles; t0 += 32) {
      const int t = t0 + lane;
      const int c = t < ntiles ? (p.desc[2 * p.E + tb.a_e[tb.tl[t] & 0xFFFFu]].ntiles + 3) / 4 : 0;
      int ci = c;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int v = __shfl_up_sync(0xFFFFFFFFu, ci, o);
        if (lane >= o) ci += v;
      }
      if (t < ntiles) dbase[t] = run + ci - c;
      run += __shfl_sync(0xFFFFFFFFu, ci, 31);
    }
    if (lane == 0) dbase[ntiles] = run;
  }
  __syncthreads();
  const int nitems = dbase[ntiles];
  if (snake_item(0, nitems) < 0) return;
  if (tid == 0) {
    for (int i = 0; i < kNI; ++i) {
      mbar_init_n(full + i, 1);
      mbar_init_n(cons + i, 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init_n(ready + b, kCW);
      mbar_init_n(mdone + b, 1);
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (wid == kCW + 1) tmem_alloc(tmem_slot, 256);
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = *tmem_slot;
  const ExpertDesc* ddesc = p.desc + 2 * p.E;
  bool ok = true;

  if (wid == kCW) {
    // ---- producer: lane 0 keeps the records and the ring; lanes 0-6 each own one copy of
    // a row block (0: the h tile, 1-4: the four unit-lane tiles, 5: scale/zero, 6: h sums),
    // whose source is found once per item and steps by a fixed stride per row block
    DnCur cur;
    cur.r = 0;
    cur.e = -1;
    cur.item = -1;
    int issued = 0, oldest = 0;
    uint32_t head = 0;
    auto retire = [&]() {   // the oldest live row block's MMAs are done: its ring bytes are free
      ok &= mbar_wait(cons + oldest % kNI, (uint32_t)(oldest / kNI) & 1u);
      ++oldest;
    };
    const uint8_t* csrc = nullptr;   // this lane's source at row block 0, its step and bytes, its ring offset
    uint64_t cstep = 0;
    uint32_t cbytes = 0, cdst = 0;
    int ibits[4] = {0, 0, 0, 0}, icoff[4] = {0, 0, 0, 0};
    uint32_t icb = 0, ibytes = 0, itx = 0, iN = 0;
    auto item_setup = [&]() {   // every lane: this item's copies (after lane 0's dn_load)
      const int item = __shfl_sync(0xFFFFFFFFu, cur.item, 0);
      if (item < 0) return false;
      const int mt = __shfl_sync(0xFFFFFFFFu, cur.mt, 0), R0 = __shfl_sync(0xFFFFFFFFu, cur.R0, 0);
      const int N = __shfl_sync(0xFFFFFFFFu, cur.N, 0);
      __syncwarp();   // xdc written by lane 0
      const ExpertDesc& xd = *xdc;
      uint32_t cb = 0;
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int gt = 4 * mt + q;
        int k = 0;
        for (int kk = 1; kk < xd.nbk; ++kk)
          if (gt >= xd.bk[kk].tile0) k = kk;
        ibits[q] = gt < xd.ntiles ? xd.bk[k].bits : 0;
        icoff[q] = (int)cb;
        cb += (uint32_t)ibits[q] * kChunkBytes;
        if (lane == 1 + q) {
          csrc = ibits[q] ? p.img + xd.code_base + xd.bk[k].code_off +
                                (uint64_t)(gt - xd.bk[k].tile0) * p.NRB * ibits[q] * kChunkBytes
                          : nullptr;
          cstep = (uint64_t)ibits[q] * kChunkBytes;
          cbytes = (uint32_t)ibits[q] * kChunkBytes;
        }
      }
      icb = cb;
      iN = (uint32_t)N;
      const uint32_t hbytes = (uint32_t)N * 512u;
      const int m0 = 128 * mt, nsl = min(128, xd.nslots - m0);
      ibytes = (hbytes + cb + 512u + (uint32_t)N * 8u + 1023u) & ~1023u;
      itx = hbytes + cb + 4u * (uint32_t)nsl + (uint32_t)N * 8u;
      if (lane == 0) {
        csrc = x.hb + (size_t)R0 * 512;
        cstep = (uint64_t)x.Rtot * 512;
        cbytes = hbytes;
        cdst = 0;
      } else if (lane <= 4) {
        cdst = hbytes + (uint32_t)icoff[lane - 1];
      } else if (lane == 5) {   // row g of the scale/zero matrix, g = rb 128 / group
        csrc = p.img + xd.sz_off + (size_t)m0 * 4;
        cstep = (uint64_t)xd.nslots * 4;
        cbytes = 4u * (uint32_t)nsl;
        cdst = hbytes + cb;
      } else if (lane == 6) {
        csrc = reinterpret_cast<const uint8_t*>(x.hs + R0);
        cstep = (uint64_t)x.Rtot * 8;
        cbytes = (uint32_t)N * 8u;
        cdst = hbytes + cb + 512u;
      } else {
        csrc = nullptr;
        cbytes = 0;
      }
      return true;
    };
    if (lane == 0) dn_load(p, x, tb, dbase, ntiles, nitems, cur, xdc);
    bool more = item_setup();
    for (int rb = 0; more; ++issued) {
      uint32_t pos = 0;
      if (lane == 0) {
        X_MARK(1, issued, 8);
        while (issued - oldest >= kNI) retire();
        while (!ring_alloc(x.ring, head, issued > oldest ? rec[oldest % kNI].pos : head, issued - oldest, ibytes, pos))
          retire();
        DnRec& g = rec[issued % kNI];
        g.item = cur.item;
        g.rb = rb;
        g.flags = (rb == 0 ? 1 : 0) | (rb == p.NRB - 1 ? 4 : 0);
        g.N = iN;
        g.cb = icb;
        g.pos = pos;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          g.bits[q] = ibits[q];
          g.coff[q] = icoff[q];
        }
        X_MARK(1, issued, 9);
        mbar_expect_tx(full + issued % kNI, itx);
      }
      pos = __shfl_sync(0xFFFFFFFFu, pos, 0);
      if (cbytes) {
        const uint64_t step = lane == 5 ? (uint64_t)((rb * kRows) / p.group) * cstep : (uint64_t)rb * cstep;
        fence_proxy_async();   // the ring space was last read by the generic proxy
        bulk_g2s(ring + pos + cdst, csrc + step, cbytes, full + issued % kNI);
      }
      if (lane == 0) X_MARK(1, issued, 10);
      if (++rb == p.NRB) {
        rb = 0;
        if (lane == 0) {
          ++cur.r;
          dn_load(p, x, tb, dbase, ntiles, nitems, cur, xdc);
        }
        more = item_setup();
      }
    }
    if (lane == 0) {   // end record
      while (issued - oldest >= kNI) retire();
      rec[issued % kNI].flags = kFlagEnd;
      mbar_expect_tx(full + issued % kNI, 0);
    }
  } else if (wid == kCW + 1) {
    // ---- MMA issuer: A from the A buffer, B = the staged h tile; commits free the A buffer
    // (mdone) and the row block's ring bytes (cons)
    if (lane == 0) {
      for (int i = 0;; ++i) {
        const int ab = i & 1;
        ok &= mbar_wait(ready + ab, (uint32_t)(i >> 1) & 1u);
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        const DnMRec mr = mrec[ab];
        if (mr.flags & kFlagEnd) break;
        if (mr.N != 16 && mr.N != 32 && mr.N != 64) {   // never: the record is corrupt
          ok = false;
          mma_commit(mdone + ab);
          mma_commit(cons + i % kNI);
          continue;
        }
        const uint32_t idesc = idesc_f16(2 * mr.N);
        const uint32_t acc = tmem + (uint32_t)(ab * 2 * kMaxNT);
        const uint32_t a0 = smem_u32(sm + L.a + (size_t)ab * kAStage), b0 = smem_u32(ring + mr.pos);
#pragma unroll
        for (int kh = 0; kh < 2; ++kh) {
#pragma unroll
          for (int k16 = 0; k16 < 4; ++k16)
            mma_f16(acc, sw128_desc(a0 + kh * kAHalf + 32 * k16),
                     sw128_desc(b0 + (uint32_t)kh * 2u * mr.N * 128u + 32 * k16), idesc, (kh | k16) ? 1u : 0u);
        }
        mma_commit(mdone + ab);
        mma_commit(cons + i % kNI);
        X_MARK(1, i, 11);
      }
    }
  } else {
    // ---- compute warps
    float out[8 * kOut];   // this thread's columns: chunks 8 hq + 32 k, k < kOut
#pragma unroll
    for (int c = 0; c < 8 * kOut; ++c) out[c] = 0.f;
    int itc = -1;                 // items started (their state slot: itc & 1)
    float pend_sc = 0.f, pend_zp = 0.f;
    int pend_flags = 0, pend_slot = 0;

    // row block i1's partial sums out of TMEM into out; at an item's last row block, the
    // item's s += g alpha out
    auto epilogue = [&](int i1) {
      ok &= mbar_wait(mdone + (i1 & 1), (uint32_t)(i1 >> 1) & 1u);
      asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      const DnItem* di = reinterpret_cast<const DnItem*>(sm + L.item + pend_slot * isz);
      const int N = di->N, nt = di->nt;
      const float2* hv = hsm + (i1 & 1) * kMaxNT;
      const uint32_t ta = tmem + ((uint32_t)(32 * (wid & 3)) << 16) + (uint32_t)((i1 & 1) * 2 * kMaxNT);
#pragma unroll
      for (int k = 0; k < kOut; ++k) {
        const int c0 = 8 * hq + 32 * k;
        if (c0 < N) {
          uint32_t v[8], w[8];
          tmem_ld8(ta + (uint32_t)c0, v);
          tmem_ld8(ta + (uint32_t)(N + c0), w);
#pragma unroll
          for (int u = 0; u < 8; ++u) {
            const float2 hz = hv[c0 + u];
            const float pv = __uint_as_float(v[u]) + __uint_as_float(w[u]);
            out[8 * k + u] = fmaf(pend_sc, fmaf(pv, hz.y, -pend_zp * hz.x), out[8 * k + u]);
          }
        }
      }
      if (pend_flags & 4) {
        if (m < di->nsl) {
          const float al = di->alpha[m];
          float* sp = p.s + di->unit[m];
#pragma unroll
          for (int k = 0; k < kOut; ++k)
#pragma unroll
            for (int u = 0; u < 8; ++u) {
              const int t = 8 * hq + 32 * k + u;
              if (t < nt && al != 0.f) atomicAdd(sp + (size_t)di->tok[t] * p.n_pad, di->pw[t] * al * out[8 * k + u]);
            }
        }
#pragma unroll
        for (int c = 0; c < 8 * kOut; ++c) out[c] = 0.f;
      }
    };

    for (int i = 0;; ++i) {
      if (tid == 0) X_MARK(1, i, 0);
      const int ab = i & 1;
      ok &= mbar_wait(full + i % kNI, (uint32_t)(i / kNI) & 1u);
      if (tid == 0) X_MARK(1, i, 1);
      cbar<kCT>();   // every compute warp is done with row block i - 1 (its epilogue, hsm, item slot)
      if (tid == 0) X_MARK(1, i, 2);
      const DnRec& g = rec[i % kNI];
      const int flags = g.flags;
      if (flags & kFlagEnd) {
        if (i > 0) epilogue(i - 1);
        if (i >= 2) ok &= mbar_wait(mdone + ab, (uint32_t)((i - 2) >> 1) & 1u);
        if (tid == 0) mrec[ab].flags = kFlagEnd;
        __syncwarp();
        if (lane == 0) mbar_arrive(ready + ab);
        break;
      }
      const uint32_t gN = g.N, gcb = g.cb, gpos = g.pos;
      const uint8_t* st = ring + gpos;
      const uint32_t hbytes = gN * 512u;
      if (flags & 1) {   // item prologue: tokens, gate weights, slot units and alphas
        ++itc;
        DnItem* di = reinterpret_cast<DnItem*>(sm + L.item + (itc & 1) * isz);
        const int item = g.item;
        int lo = 0, hi = ntiles;
        while (hi - lo > 1) {
          const int md = (lo + hi) >> 1;
          if (dbase[md] <= item) lo = md;
          else hi = md;
        }
        const uint32_t tw = tb.tl[lo];
        const int a = (int)(tw & 0xFFFFu), tt = (int)(tw >> 16), e = tb.a_e[a];
        const int nt = min(x.NT, tb.a_cnt[a] - tt * x.NT);
        const int m0 = 128 * (item - dbase[lo]);
        const ExpertDesc& xd = ddesc[e];
        const int nsl = min(128, xd.nslots - m0);
        if (tid < kMaxNT) {
          const int q = tid < nt ? p.pair_list[tb.a_pst[a] + tt * x.NT + tid] : 0;
          di->tok[tid] = q / p.k;
          di->pw[tid] = tid < nt ? p.pair_weight[q] : 0.f;
        }
        if (tid < 128) {
          di->unit[tid] = tid < nsl ? reinterpret_cast<const int*>(p.img + xd.unit_off)[m0 + tid] : 0;
          di->alpha[tid] = tid < nsl ? reinterpret_cast<const float*>(p.img + xd.alpha_off)[m0 + tid] : 0.f;
        }
        if (tid == 0) {
          di->nt = nt;
          di->N = (int)gN;
          di->nsl = nsl;
        }
      }
      if (i >= 2) ok &= mbar_wait(mdone + ab, (uint32_t)((i - 2) >> 1) & 1u);   // A buffer ab is free
      if (tid == 0) X_MARK(1, i, 3);
      // this row block's scale / zero of the thread's slot, and the h sums of its tokens
      const int q = m >> 5;
      const int bq = g.bits[q];
      float nsc = 0.f, nzp = 0.f;
      if (bq) {
        const uint32_t szw = reinterpret_cast<const uint32_t*>(st + hbytes + gcb)[m];
        nsc = __half2float(__ushort_as_half((unsigned short)(szw & 0xFFFFu)));
        nzp = __half2float(__ushort_as_half((unsigned short)(szw >> 16)));
      }
      if (tid < (int)gN) hsm[ab * kMaxNT + tid] = reinterpret_cast<const float2*>(st + hbytes + gcb + 512u)[tid];
      // A: thread = (slot m, quarter hq of the row block's rows)
      uint8_t* A = sm + L.a + (size_t)ab * kAStage;
      {
        const uint8_t* ln = st + hbytes + g.coff[q] + (m & 31) * 16;
        switch (bq) {
          case 1: dec_ul<1>(ln, hq, m, A); break;
          case 2: dec_ul<2>(ln, hq, m, A); break;
          case 3: dec_ul<3>(ln, hq, m, A); break;
          case 4: dec_ul<4>(ln, hq, m, A); break;
          case 6: dec_ul<6>(ln, hq, m, A); break;
          case 8: dec_ul<8>(ln, hq, m, A); break;
          default: {
#pragma unroll
            for (int kk = 0; kk < 32; kk += 8) store_a8(A, m, 32 * hq + kk, make_uint2(0u, 0u), make_uint2(0u, 0u));
          }
        }
      }
      if (tid == 0) X_MARK(1, i, 4);
      if (tid == 0) {
        DnMRec mr;
        mr.N = (int)gN;
        mr.flags = flags;
        mr.pos = gpos;
        mr.pad_ = 0;
        mrec[ab] = mr;
      }
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
      __syncwarp();
      if (lane == 0) mbar_arrive(ready + ab);
      if (tid == 0) X_MARK(1, i, 5);
      if (i > 0) epilogue(i - 1);
      if (tid == 0) X_MARK(1, i, 6);
      pend_sc = nsc;
      pend_zp = nzp;
      pend_flags = flags;
      pend_slot = itc & 1;
    }
  }
  if (!ok) atomicCAS(p.status, 0, BITSMOE_ERR_TIMEOUT);
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  if (wid == kCW + 1) tmem_dealloc(tmem, 256);
}

}  // namespace

namespace bmoe {

// Sizes of the multi-token expert kernels' buffers for a call of T tokens.
XArgs x_args(const ImageHeader& hd, int T, int k) {
  XArgs x;
  std::memset(&x, 0, sizeof(x));
  x.NT = T <= 16 ? 16 : 32;   // 32-token tiles keep the copy ring several K-blocks deep
  const int P = T * k;
  x.A_max = std::min(hd.E, P);
  x.max_tiles = P / x.NT + x.A_max;
  x.Rtot = (int)align_up((uint64_t)2 * P + 16 * (uint64_t)x.A_max, 16);   // >= the sum of tile_rows
  // gathered z: 2 projections x (tiles' widths <= Rtot) x K-blocks of 128 slots; a
  // projection has at most n units plus the padding of its seven buckets (< 32 slots each)
  x.zv_floats = 2ull * (uint64_t)x.Rtot * align_up((uint64_t)hd.n + 7 * 32, 128);
  return x;
}

static size_t x_smem(const XArgs& x, bool gu) {
  return 1024 + (gu ? gu_plan(x).total : dn_plan(x).total);
}

// The ring takes what the other parts leave of the shared memory of one CTA.
static cudaError_t x_launch(bool gu, const Fwd& p, XArgs x, int sms, cudaStream_t st, bool pdl) {
  int dev = 0, optin = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  if (e != cudaSuccess) return e;
  x.ring = 0;
  const size_t base = x_smem(x, gu);
  const size_t avail = (size_t)optin > base + 4096 ? (size_t)optin - base - 2048 : 0;
  x.ring = (uint32_t)(avail & ~(size_t)1023);
  const uint32_t need = gu ? (128u * 128u + 3072u + 12u * 128u) : (64u * 512u + 8u * 4u * kChunkBytes + 512u + 1024u);
  if (x.ring < need) return cudaErrorInvalidValue;
  const size_t smem = x_smem(x, gu);
  static std::mutex mu;
  static size_t done[2] = {0, 0};
  {
    std::lock_guard<std::mutex> lock(mu);
    if (smem > done[gu ? 0 : 1]) {
      e = cudaFuncSetAttribute(gu ? k_gu16 : k_dn16, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
      if (e != cudaSuccess) return e;
      done[gu ? 0 : 1] = smem;
    }
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)std::max(1, sms));
  cfg.blockDim = dim3(gu ? kGuThreads : kDnThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, gu ? k_gu16 : k_dn16, p, x);
}

cudaError_t launch_zgather(const Fwd& p, const XArgs& x, int sms, cudaStream_t st, bool pdl) {
  const size_t smem = 16 + ((size_t)5 * x.A_max + 4 + x.max_tiles + 2 * (2 * (size_t)x.max_tiles + 1) + 128 + kMaxNT) * 4;
  static std::mutex mu;
  static size_t done = 0;
  {
    std::lock_guard<std::mutex> lock(mu);
    if (smem > done) {
      const cudaError_t e = cudaFuncSetAttribute(k_zgather, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
      if (e != cudaSuccess) return e;
      done = smem;
    }
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)std::max(1, 4 * sms));
  cfg.blockDim = dim3(kZgThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, k_zgather, p, x);
}

cudaError_t launch_gu16(const Fwd& p, const XArgs& x, int sms, cudaStream_t st, bool pdl) {
  return x_launch(true, p, x, sms, st, pdl);
}
cudaError_t launch_dn16(const Fwd& p, const XArgs& x, int sms, cudaStream_t st, bool pdl) {
  return x_launch(false, p, x, sms, st, pdl);
}

}  // namespace bmoe

#ifdef BITSMOE_X_TRACE
extern "C" int bitsmoe_x_trace_read(void* dst) {
  return (int)cudaMemcpyFromSymbol(dst, g_x_trace, sizeof(g_x_trace));
}
#endif
