// Clustered single-token decode forward: the whole quantized MoE layer in one
// persistent kernel, for a batch of one token, with two grid-wide barriers.
//
// Same arithmetic as fused.cu and the kernel chain in forward.cu (Fig. 1
// Stage 3; the association of Eq. app_normalized_decomposition), organised
// around the expert's row blocks.  A gate or up row i of expert e needs every
// unit of the factor (P_hat row i against alpha * z), and the down factor needs
// h = SiLU(gate) * up only row by row: s_j = sum_i P_hat_dn[i, j] h_i splits
// into partial sums over 128-row blocks.  So one thread-block cluster owns one
// (routing slot a, row block rb) pair; its CL blocks each take a contiguous
// part of the expert's gate, up and down tiles:
//
//   prologue   bulk copies of this block's rows of the input bases into shared
//              memory (weights only: overlaps the previous kernel under
//              programmatic dependent launch)
//   A          x into shared memory, s cleared, z = Phi^T x for this block's
//              rows; meanwhile the control warps route the token and issue
//              the copies of the cluster's gate/up part (row block rb)
//                                                           -> grid barrier 1
//              (the freed projection buffer receives this block's down part
//              and its rows of Phi_dn)
//   C          gate/up: dp2a over the staged codes into partial gate and up
//              rows of the block's units; the CL blocks add their partial rows
//              through distributed shared memory (one cluster barrier), so
//              every block holds gate, up and h for the 128 rows
//   D          down: for each unit of the block's down part, the dot of its
//              codes over the 128 rows with h (int16, one scale per row
//              block), s_j += w_e * alpha_j * partial, fp32 atomics
//                                                           -> grid barrier 2
//   E          y = Phi_dn s for this block's rows
//
// The grid barriers are counters at a fixed place in the workspace, zero when
// a call starts and reset by the last block to finish; every wait on them or
// on a bulk copy is bounded and a timeout is reported in the status word.  The
// cluster barrier is the hardware one: every block of a cluster reaches it on
// every path (no early exit before it), so it cannot wait forever.
#include <algorithm>
#include <cstring>
#include <mutex>

#include "fused_common.cuh"

namespace {

// Phase timestamps of each block (%globaltimer), compiled in only with -DBITSMOE_F2_TRACE
// for timing studies; without it F2_MARK is empty.
#ifdef BITSMOE_F2_TRACE
__device__ unsigned long long g_f2_trace[1024][16];
#define F2_MARK(i)                                                                    \
  do {                                                                                \
    unsigned long long t_;                                                            \
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t_));                            \
    g_f2_trace[blockIdx.x & 1023][(i)] = t_;                                          \
  } while (0)
#else
#define F2_MARK(i) \
  do {             \
  } while (0)
#endif

__device__ __forceinline__ uint32_t al128(uint32_t v) { return (v + 127u) & ~127u; }

__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t cluster_id() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%clusterid.x;" : "=r"(r));
  return r;
}
// A float into the same shared-memory location of cluster block `rank`.
__device__ __forceinline__ void st_cluster_f32(const void* local, uint32_t rank, float v) {
  uint32_t ra;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(ra) : "r"(smem_u32(local)), "r"(rank));
  asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(ra), "f"(v) : "memory");
}
// All threads of all blocks of the cluster; the release/acquire pair orders the
// distributed shared-memory stores before it with the loads after it.
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ bool mbar_wait_for(uint64_t* bar, uint32_t parity, long long spin) {
  const long long t0 = clock64();
  while (!mbar_try_wait(bar, parity))
    if (clock64() - t0 > spin) return false;
  return true;
}
// 16-byte words of a record from global memory into shared memory (one lane per word).
__device__ __forceinline__ void copy_rec_words(void* dst, const void* src, int words, int i) {
  if (i < words) reinterpret_cast<uint4*>(dst)[i] = reinterpret_cast<const uint4*>(src)[i];
}

// L2 prefetch of the whole 16-byte chunks inside [p, p + bytes) (never past the buffer).
__device__ __forceinline__ void prefetch_inner(const void* p, size_t bytes) {
  const uintptr_t a = (reinterpret_cast<uintptr_t>(p) + 15) & ~(uintptr_t)15;
  const uintptr_t b = (reinterpret_cast<uintptr_t>(p) + bytes) & ~(uintptr_t)15;
  if (b > a) prefetch_run(reinterpret_cast<const uint8_t*>(a), (uint64_t)(b - a));
}

// Routing of the token by all threads of the block, from the order keys of its logits
// (written by the caller before a __syncthreads): the k largest logits (ties to the lower
// index; -0 and +0 tie; NaN below every number) into sel_e, their softmax into sel_w.  A
// key's rank is counted by tpk threads over interleaved parts of the keys (tpk = the
// largest power of two with tpk * E <= blockDim, at most 32), summed by shuffles.
// Contains __syncthreads.
__device__ __noinline__ void route_rank(int E, int k, const uint32_t* keys, int* sel_e, float* sel_w) {
  const int tid = threadIdx.x, nt = blockDim.x;
  int tpk = 1;
  while (tpk * 2 * E <= nt && tpk < 32) tpk *= 2;
  const int per = nt / tpk;   // keys handled at once
  for (int base = 0; base < E; base += per) {
    const int i = base + tid / tpk, q = tid & (tpk - 1);
    const bool live = i < E;
    const uint32_t key = live ? keys[i] : 0u;
    int rank = 0;
    if (live)
      for (int f = q; f < E; f += tpk) {
        const uint32_t o = keys[f];
        rank += (o > key) | ((o == key) & (f < i));
      }
    for (int o = 1; o < tpk; o <<= 1) rank += __shfl_xor_sync(0xFFFFFFFFu, rank, o);
    if (live && q == 0 && rank < k) {
      sel_e[rank] = i;
      sel_w[rank] = key ? __uint_as_float((key & 0x80000000u) ? (key & 0x7FFFFFFFu) : ~key)
                        : __int_as_float(0x7FC00000);   // key 0: a NaN logit
    }
  }
  __syncthreads();
  if (tid < 32) {
    const float m = sel_w[0];
    const float ev = tid < k ? expf(sel_w[tid] - m) : 0.f;
    float sum = ev;
#pragma unroll
    for (int o = 16; o; o >>= 1) sum += __shfl_xor_sync(0xFFFFFFFFu, sum, o);
    __syncwarp();
    if (tid < k) sel_w[tid] = ev * (1.f / sum);
  }
  __syncthreads();
}

// Offsets (inside a staging area) of one projection's staged gate/up part:
// codes of the row block, unit indices, alphas, then G scale/zero rows.
struct GuLay {
  uint32_t code, unit, alpha, sz, end;
};
__device__ __forceinline__ GuLay gu_lay(const F2Gu& r, uint32_t base, int G) {
  GuLay l;
  l.code = base;
  l.unit = base + al128(r.bytes);
  l.alpha = l.unit + r.nslot * 4;
  l.sz = l.alpha + r.nslot * 4;
  l.end = al128(l.sz + (uint32_t)G * r.nslot * 4);
  return l;
}

// Copies of one projection's gate/up part for row block rb, one per lane of the calling
// warp (lane 0 arms the barrier first): codes, unit indices, alphas, G scale/zero rows.
template <int G>
__device__ void stage_gu(const Fwd& p, const F2Gu& r, int rb, uint8_t* area, uint32_t base, uint64_t* bar, int lane) {
  const GuLay l = gu_lay(r, base, G);
  const uint32_t ms = r.nslot * 4;
  if (lane == 0) mbar_expect_tx(bar, r.bytes + (2 + G) * ms);
  __syncwarp();
  if (lane < 0) return;   // lanes before this projection's (the caller offsets them)
  if (lane == 0) bulk_g2s(area + l.code, p.img + r.code0 + (uint64_t)rb * r.rb_stride, r.bytes, bar);
  else if (lane == 1) bulk_g2s(area + l.unit, p.img + r.unit0, ms, bar);
  else if (lane == 2) bulk_g2s(area + l.alpha, p.img + r.alpha0, ms, bar);
  else if (lane < 3 + G) {
    const int gl = lane - 3, g_base = (rb * kRows) / p.group;
    bulk_g2s(area + l.sz + gl * ms, p.img + r.sz0 + (uint64_t)(g_base + gl) * r.sz_row, ms, bar);
  }
}

__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async4(void* dst, const void* src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(smem_u32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_all;" ::: "memory"); }

__device__ __forceinline__ uint32_t dn_code_bytes(const F2Dn& r) {
  uint32_t b = 0;
  for (int k = 0; k < r.nr; ++k) b += (uint32_t)r.ntl[k] * ul_chunks(r.bits[k]) * kChunkBytes;
  return b;
}

// Staged down part of row block rb: per tile its b 16-byte chunks per lane, then the
// part's unit indices, alphas and G scale/zero rows.  Every lane copies (cp.async, no
// bulk-copy descriptors) exactly the bytes it reads later -- its 16 bytes of each chunk
// of the warp's tiles tt = w, w + kFWarps, ... and its slot's metadata -- so no other
// thread needs to see them.
template <int G>
__device__ void load_dn_warp(const Fwd& p, const F2Dn& r, int rb, uint8_t* dst, int w, int lane) {
  const uint32_t ms = r.nslot * 4, mo = al128(dn_code_bytes(r));
  const int ntile = (int)(r.nslot / 32), g_base = (rb * kRows) / p.group;
  for (int tt = w; tt < ntile; tt += kFWarps) {
    int k = 0, t = tt;
    uint32_t off = 0;
    while (k < r.nr - 1 && t >= r.ntl[k]) {
      off += (uint32_t)r.ntl[k] * ul_chunks(r.bits[k]) * kChunkBytes;
      t -= r.ntl[k];
      ++k;
    }
    const int C = ul_chunks(r.bits[k]);
    const uint32_t cb = (uint32_t)C * kChunkBytes;
    off += (uint32_t)t * cb;
    const uint8_t* src = p.img + r.code[k] + ((uint64_t)t * p.NRB + rb) * cb + lane * 16;
    for (int q = 0; q < C; ++q) cp_async16(dst + off + q * kChunkBytes + lane * 16, src + q * kChunkBytes);
    const uint32_t slot = 32u * tt + lane;
    cp_async4(dst + mo + slot * 4, p.img + r.unit0 + slot * 4);
    cp_async4(dst + mo + ms + slot * 4, p.img + r.alpha0 + slot * 4);
#pragma unroll
    for (int gl = 0; gl < G; ++gl)
      cp_async4(dst + mo + (2 + gl) * ms + slot * 4, p.img + r.sz0 + (uint64_t)(g_base + gl) * r.sz_row + slot * 4);
  }
}

// One warp's share (kF2GuWarps-way byte split) of a staged gate/up part for the
// single token: the part's partial rows 4 * lane .. 4 * lane + 3 of row block rb
// (the sum over the share's units of P_hat[i, j] alpha_j z_j) in o.
//   c_j = alpha_j z_j scale_{j,g} as int16 with one scale per (warp, part),
//   o   = scale * (sum_j q_ij c_j - sum_j zero_{j,g} c_j)      (b < 16)
//       + sum_j p16_ij alpha_j z_j                              (b = 16, fp32)
template <int G, typename AfterGather>
__device__ void gu_share(const Fwd& p, const F2Gu& r, int h, const uint8_t* area, const GuLay& l, const float* zs,
                         int16_t* cq, int s16, int w, int lane, float (&o)[4], AfterGather&& after_gather) {
  const int* su = reinterpret_cast<const int*>(area + l.unit);
  const float* sa = reinterpret_cast<const float*>(area + l.alpha);
  const uint32_t* ssz = reinterpret_cast<const uint32_t*>(area + l.sz);
  // the record's fields in registers (the shared-memory record would be reloaded after
  // every shared-memory store below)
  const int nr = r.nr, nslot = (int)r.nslot;
  uint8_t rbits[kNumBk];
  uint16_t rntl[kNumBk];
#pragma unroll
  for (int k = 0; k < kNumBk; ++k) {
    rbits[k] = k < nr ? r.bits[k] : 0;
    rntl[k] = k < nr ? r.ntl[k] : 0;
  }
  const int t0 = rl_split_at(rbits, rntl, nr, w, kF2GuWarps);
  const int t1 = rl_split_at(rbits, rntl, nr, w + 1, kF2GuWarps);
  int sl0 = 0, nq = 0;
  {
    int t = 0;
    for (int k = 0; k < nr; ++k) {
      const int b = rbits[k], nt = rntl[k];
      const int lo = min(max(t0 - t, 0), nt), hi = min(max(t1 - t, 0), nt);
      sl0 += lo * rl_units(b);
      if (b < 16) nq += (hi - lo) * rl_units(b);
      t += nt;
    }
  }
  const float* zrow = zs + (size_t)h * p.n_pad;     // one token: z[h][:] (shared-memory copy)
  // activation table: the gathered z values stay in registers when the share has at most
  // 32 * kFZ quantised slots (the usual case); larger shares gather them again
  float zr[kFZ];
  float mx = 0.f;
  const bool one_batch = nq <= 32 * kFZ;
  for (int i0 = 0; i0 < nq; i0 += 32 * kFZ) {
#pragma unroll
    for (int m = 0; m < kFZ; ++m) {
      const int i = i0 + lane + 32 * m;
      zr[m] = i < nq ? zrow[su[sl0 + i]] * sa[sl0 + i] : 0.f;
    }
#pragma unroll
    for (int m = 0; m < kFZ; ++m) {
      const int i = i0 + lane + 32 * m;
      if (i < nq) {
#pragma unroll
        for (int gl = 0; gl < G; ++gl) {
          const float sc = __half2float(__ushort_as_half((unsigned short)(ssz[gl * nslot + sl0 + i] & 0xFFFFu)));
          mx = fmaxf(mx, fabsf(zr[m] * sc));
        }
      }
    }
  }
  mx = warp_max(mx);
  if (threadIdx.x == 0) F2_MARK(13);
  after_gather();   // the warp's z loads are back: its other copies no longer queue ahead of them
  const float inv = mx > 0.f ? 32767.f / mx : 0.f;
  const float scl = mx * (1.f / 32767.f);
  float corr[G];
#pragma unroll
  for (int gl = 0; gl < G; ++gl) corr[gl] = 0.f;
  for (int i0 = 0; i0 < nq; i0 += 32 * kFZ) {
    if (!one_batch) {
#pragma unroll
      for (int m = 0; m < kFZ; ++m) {
        const int i = i0 + lane + 32 * m;
        zr[m] = i < nq ? zrow[su[sl0 + i]] * sa[sl0 + i] : 0.f;
      }
    }
#pragma unroll
    for (int m = 0; m < kFZ; ++m) {
      const int i = i0 + lane + 32 * m;
      if (i < nq) {
#pragma unroll
        for (int gl = 0; gl < G; ++gl) {
          const uint32_t wd = ssz[gl * nslot + sl0 + i];
          const float sc = __half2float(__ushort_as_half((unsigned short)(wd & 0xFFFFu)));
          const float zp = __half2float(__ushort_as_half((unsigned short)(wd >> 16)));
          const int ci = __float2int_rn(zr[m] * sc * inv);
          cq[(size_t)gl * s16 + i] = (int16_t)ci;
          corr[gl] = fmaf((float)ci, zp, corr[gl]);
        }
      }
    }
  }
#pragma unroll
  for (int gl = 0; gl < G; ++gl) corr[gl] = warp_sum(corr[gl]);
  __syncwarp();
  if (threadIdx.x == 0) F2_MARK(14);
  const int gl_lane = G == 1 ? 0 : (4 * lane) / p.group;
  const int* cq32 = reinterpret_cast<const int*>(cq + (size_t)gl_lane * s16);
  float accf[4] = {0.f, 0.f, 0.f, 0.f};
  float acc16[4][1];
#pragma unroll
  for (int q = 0; q < 4; ++q) acc16[q][0] = 0.f;
  const float* const zrows[1] = {zrow};
  int t = 0, sl = 0;
  uint32_t bo = 0;
  for (int k = 0; k < nr; ++k) {
    const int b = rbits[k], nt = rntl[k];
    const int lo = min(max(t0 - t, 0), nt), hi = min(max(t1 - t, 0), nt);
    const int C = rl_chunks(b), U = rl_units(b);
    if (hi > lo) {
      const uint8_t* code = area + l.code + bo + (uint32_t)lo * C * kChunkBytes + lane * 16;
      const int ls = sl + lo * U;
      if (b < 16) rl_range_rt(b, code, hi - lo, cq32 + (ls - sl0) / 2, accf);
      else rl_range16<1, true>(code, hi - lo, su + ls, sa + ls, zrows, acc16);
    }
    t += nt;
    sl += nt * U;
    bo += (uint32_t)nt * C * kChunkBytes;
  }
  float cl = corr[0];
#pragma unroll
  for (int gl = 1; gl < G; ++gl)
    if (gl == gl_lane) cl = corr[gl];
#pragma unroll
  for (int q = 0; q < 4; ++q) o[q] = fmaf(scl, accf[q] - cl, acc16[q][0]);
}

// One unit-lane tile of the staged down part over the cluster's row block:
// sum_g scale_g (sum_i q_i hq_i - zero_g sum_i hq_i) over the lane's unit (b < 16),
// or sum_i p16_i hq_i (b = 16); the caller multiplies by h's scale.
template <int G>
__device__ float dn_tile(int b, const uint8_t* cb, const int* hq32, int gshift, const int* hsum, const uint32_t* szl,
                         int nslot) {
  if (b == 16) {   // fp16 values: chunk c = rows 8c .. 8c + 7, two rows per word
    float tmp = 0.f;
#pragma unroll 1
    for (int c = 0; c < 16; ++c) {
      const uint4 v = lds128(cb + (size_t)c * kChunkBytes);
      const uint32_t wv[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int hp = hq32[4 * c + q];
        tmp = fmaf((float)(int16_t)(hp & 0xFFFF), f16lo(wv[q]), fmaf((float)(hp >> 16), f16hi(wv[q]), tmp));
      }
    }
    return tmp;
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
  float d = 0.f;
#pragma unroll
  for (int g = 0; g < G; ++g) {
    const uint32_t szw = szl[(size_t)g * nslot];
    const float sc = __half2float(__ushort_as_half((unsigned short)(szw & 0xFFFFu)));
    const float zp = __half2float(__ushort_as_half((unsigned short)(szw >> 16)));
    d = fmaf(sc, fmaf(-zp, (float)hsum[g], (float)(lo_g[g] + (hi_g[g] << hs))), d);
  }
  return d;
}

template <int G>
__global__ void __launch_bounds__(kFThreads, 1) k_f2(Fwd p, F2Args f) {
  extern __shared__ __align__(128) uint8_t fsm[];
  uint64_t* bar_b = reinterpret_cast<uint64_t*>(fsm);   // [kMaxBStages] input-basis stages
  uint64_t* bar_g = bar_b + kMaxBStages;                 // gate part
  uint64_t* bar_u = bar_g + 1;                           // up part
  uint64_t* bar_rec = bar_g + 2;                         // this rank's records
  uint64_t* bar_e = bar_g + 3;                           // output-basis rows
  uint64_t* bar_z = bar_g + 4;                           // z into shared memory
  volatile int* flags = reinterpret_cast<volatile int*>(bar_g + 5);   // [0..1] grid barriers passed, [2] bad ws
  F2Gu* rg = reinterpret_cast<F2Gu*>(fsm + f.off_rec);
  F2Gu* ru = rg + 1;
  F2Dn* rd = reinterpret_cast<F2Dn*>(ru + 1);
  uint32_t* keys = reinterpret_cast<uint32_t*>(fsm + f.off_route);   // [E]
  int* sel_e = reinterpret_cast<int*>(keys + p.E);                     // [k]
  float* sel_w = reinterpret_cast<float*>(sel_e + p.k);                // [k]
  uint16_t* xs = reinterpret_cast<uint16_t*>(fsm + f.off_xs);
  float* pw = reinterpret_cast<float*>(fsm + f.off_pw);                // [kFWarps][128] partial rows
  float* xch = reinterpret_cast<float*>(fsm + f.off_xch);              // [CL][2][128], written by the cluster
  int16_t* hq = reinterpret_cast<int16_t*>(fsm + f.off_h);             // [128] h as int16
  float* hred = reinterpret_cast<float*>(hq + kRows);                  // [4] warp maxima, then [4] the scale
  int* hws = reinterpret_cast<int*>(hred + 8);                         // [4] warp sums of hq
  uint8_t* r1 = fsm + f.off_r1;
  uint8_t* r2 = fsm + f.off_r2;
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  const int nb = gridDim.x, blk = blockIdx.x;
  const int CL = f.CL;
  const int crank = CL > 1 ? (int)cluster_rank() : 0;
  const int cid = CL > 1 ? (int)cluster_id() : blk;
  const bool pair = cid < f.npairs;                   // uniform over the cluster
  const int a = pair ? cid / p.NRB : 0, rb = pair ? cid - (cid / p.NRB) * p.NRB : 0;
  const uint32_t row_in = (uint32_t)p.D_pad * 2, row_out = (uint32_t)p.n_pad * 2;
  const int nrows_b = 2 * p.n;
  // blocks [0, npairs * CL) own pairs; the others take larger shares of the bases
  const int npb = f.npairs * CL;
  const int b0 = min(nrows_b, pair ? blk * f.b_per : npb * f.b_per + (blk - npb) * f.b_free);
  const int b1 = min(nrows_b, b0 + (pair ? f.b_per : f.b_free));
  const int e0 = min(p.D, pair ? blk * f.e_per : npb * f.e_per + (blk - npb) * f.e_free);
  const int e1 = min(p.D, e0 + (pair ? f.e_per : f.e_free));

  // ---- prologue (may overlap the previous kernel): L2 prefetches of the token's x and
  // logits (a prefetch returns no data, so it cannot see stale values; the loads after
  // the wait read what the previous kernel wrote), of this rank's records, then the bulk
  // copies of this block's input-basis rows
  if (tid == 0) {
    F2_MARK(0);
    for (int i = 0; i < kMaxBStages + 5; ++i) mbar_init(bar_b + i);
    if (pair && f.rec_smem) {   // this rank's records of every expert, into the (still free) staging area
      mbar_expect_tx(bar_rec, f.rank_bytes);
      bulk_run(r2, f.tab + (size_t)crank * f.rank_bytes, f.rank_bytes, bar_rec);
    }
    flags[0] = flags[1] = flags[2] = 0;
    if (f.prefetch_io) {
      prefetch_inner(p.x, (size_t)p.D * 2);
      if (pair) prefetch_inner(p.logits, (size_t)p.E * 4);
    }
    for (int st = 0; st < f.b_nst; ++st) {
      const int r0 = b0 + st * f.b_stage, r1e = min(b1, r0 + f.b_stage);
      if (r1e > r0) {
        mbar_expect_tx(bar_b + st, (uint32_t)(r1e - r0) * row_in);
        bulk_run(r1 + (size_t)st * f.b_stage * row_in, reinterpret_cast<const uint8_t*>(p.basis_in) + (size_t)r0 * row_in,
                 (uint32_t)(r1e - r0) * row_in, bar_b + st);
      }
    }
  } else if (tid == 32 && pair && !f.rec_smem) {
    prefetch_run(f.tab + (size_t)crank * f.rank_bytes, f.rank_bytes);
  }
  if (pair) {   // code warm-up on dummy keys
    for (int i = tid; i < p.E; i += kFThreads) keys[i] = 0u;
    __syncthreads();
    route_rank(p.E, p.k, keys, sel_e, sel_w);
  }
  __syncthreads();
  pdl_trigger();   // the next forward's blocks may take SMs as soon as ours leave
  pdl_wait();      // x, logits, y and the workspace belong to earlier kernels until here
  if (tid == 0) F2_MARK(1);

  const uint32_t epoch = __ldcg(f.sync);
  uint32_t* cnt = sync_set(f.sync, epoch);
  // counters 1 and 2 of this call's set must be zero (counter 0 is the only one of this
  // kernel's that can move before every block has passed this check)
  if (tid == 0) {
    const int v = (__ldcg(cnt + 1) | __ldcg(cnt + 2)) != 0u;
    flags[2] = v;
    if (v) {
      atomicExch(p.status, BITSMOE_ERR_WORKSPACE_STATE);
    } else if (blk == 0) {
      p.status[0] = 0;
      sync_clear_next(f.sync, epoch);
    }
  }
  // x into shared memory (a token row inside a batch starts at 2*D*t bytes: 16-byte loads
  // only when x is 16-byte aligned), s cleared
  {
    const bool x16 = (reinterpret_cast<uintptr_t>(p.x) & 15) == 0;
    for (int i = tid; i < p.D_pad / 8; i += kFThreads) {
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
    // the logits' order keys, in the same round trip
    if (pair)
      for (int i = tid; i < p.E; i += kFThreads) keys[i] = order_key(__ldcg(p.logits + i));
  }
  __syncthreads();
  if (flags[2]) {   // every block sees the same counters: the whole grid returns here
    if (tid == 0) {
      for (int st = 0; st < f.b_nst; ++st)
        if (b0 + st * f.b_stage < b1) mbar_wait_for(bar_b + st, 0, f.spin);
      if (pair && f.rec_smem) mbar_wait_for(bar_rec, 0, f.spin);
    }
    return;
  }
  for (int i = blk * kFThreads + tid; i < p.n_pad / 4; i += nb * kFThreads)
    reinterpret_cast<float4*>(p.s)[i] = make_float4(0.f, 0.f, 0.f, 0.f);
  if (pair) {
    // ---- routing by the whole block, the cluster part's records, the gate/up copies
    route_rank(p.E, p.k, keys, sel_e, sel_w);
    if (tid == 0) F2_MARK(3);
    if (wid == 0) {
      const int e = sel_e[a];
      // the three records, from the staging area (copied there before the wait) or from L2
      bool from_smem = f.rec_smem != 0;
      if (from_smem && !mbar_wait_for(bar_rec, 0, f.spin)) {
        if (lane == 0) atomicCAS(p.status, 0, BITSMOE_ERR_TIMEOUT);
        from_smem = false;
      }
      const uint8_t* tr = from_smem ? r2 : f.tab + (size_t)crank * f.rank_bytes;
      if (lane < 5) copy_rec_words(rg, tr + (size_t)e * sizeof(F2Gu), 5, lane);
      else if (lane < 10) copy_rec_words(ru, tr + ((size_t)p.E + e) * sizeof(F2Gu), 5, lane - 5);
      else if (lane < 17) copy_rec_words(rd, tr + (size_t)2 * p.E * sizeof(F2Gu) + (size_t)e * sizeof(F2Dn), 7, lane - 10);
      __syncwarp();
      if ((f.dbg & 2) && lane == 0) {   // debug bounds checks of the three records
        const int g_base = (rb * kRows) / p.group;
        for (int h = 0; h < 2; ++h) {
          F2Gu* r = h ? ru : rg;
          const uint64_t ms = (uint64_t)r->nslot * 4;
          if (r->bytes && !(in_image(p, r->code0 + (uint64_t)rb * r->rb_stride, r->bytes) &&
                            in_image(p, r->unit0, ms) && in_image(p, r->alpha0, ms) &&
                            in_image(p, r->sz0 + (uint64_t)(g_base + G - 1) * r->sz_row, ms))) {
            r->bytes = 0;
            report_bounds(p.status);
          }
        }
        if (rd->nslot) {
          const uint64_t ms = (uint64_t)rd->nslot * 4;
          bool ok = in_image(p, rd->unit0, ms) && in_image(p, rd->alpha0, ms) &&
                    in_image(p, rd->sz0 + (uint64_t)(g_base + G - 1) * rd->sz_row, ms);
          for (int k = 0; k < rd->nr; ++k)
            ok = ok && in_image(p, rd->code[k], (uint64_t)rd->ntl[k] * p.NRB * ul_chunks(rd->bits[k]) * kChunkBytes);
          if (!ok) {
            rd->nslot = 0;
            report_bounds(p.status);
          }
        }
      }
      __syncwarp();
      fence_proxy_async();   // the table's generic reads before the copies that overwrite it
      if (rg->bytes) stage_gu<G>(p, *rg, rb, r2, 0, bar_g, lane);
      if (ru->bytes) stage_gu<G>(p, *ru, rb, r2, gu_lay(*rg, 0, G).end, bar_u, lane - 8);
      if (lane == 0) F2_MARK(4);
    }
  }
  // ---- z = Phi^T x for rows [b0, b1): all warps, but warp 0 of a pair block (it stages)
  if (tid == 0) F2_MARK(2);
  const int bw0 = pair ? 1 : 0;
  for (int ri = wid - bw0; ri >= 0 && ri < b1 - b0; ri += kFWarps - bw0) {
    const int st = ri / f.b_stage;
    if (!mbar_wait_for(bar_b + st, 0, f.spin)) {
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
  __syncthreads();   // z rows and the cleared s are written; the projection rows are consumed
  if (tid == 0) {
    F2_MARK(5);
    if (!((f.dbg & 1) && blk == 0)) grid_arrive(cnt + 0);
    // the freed buffer: a pair block's down part now and its output-basis rows after the
    // z gathers of the next phase; a free block's output-basis rows now
    fence_proxy_async();
    if (!pair && e1 > e0) {
      mbar_expect_tx(bar_e, (uint32_t)(e1 - e0) * row_out);
      bulk_run(r1, reinterpret_cast<const uint8_t*>(p.basis_out) + (size_t)e0 * row_out, (uint32_t)(e1 - e0) * row_out,
               bar_e);
    }
  }
  grid_wait(cnt + 0, nb, p.status, flags + 0, f.spin);
  if (tid == 0) F2_MARK(6);

  // ---- C: gate (warps 0-7) and up (warps 8-15) of the cluster's row block over this
  // block's part; the partial rows meet in the cluster
  if (pair) {
    // z of both projections into the freed projection buffer: the gathers below read shared
    // memory instead of issuing one L2 request per unit
    const float* zs = reinterpret_cast<const float*>(r1);
    if (tid == 0) {
      const uint32_t zb = (uint32_t)p.n_pad * 8;
      mbar_expect_tx(bar_z, zb);
      bulk_run(r1, reinterpret_cast<const uint8_t*>(p.z), zb, bar_z);
    }
    const bool z_ok = mbar_wait_for(bar_z, 0, f.spin);
    if (!z_ok && tid == 0) atomicCAS(p.status, 0, BITSMOE_ERR_TIMEOUT);
    const int h = wid < kF2GuWarps ? 0 : 1;
    const F2Gu& r = h ? *ru : *rg;
    const GuLay l = gu_lay(r, h ? gu_lay(*rg, 0, G).end : 0u, G);
    // each warp copies its down tiles once its own z loads are back
    auto load_dn = [&]() {
      if (rd->nslot) load_dn_warp<G>(p, *rd, rb, r1 + f.off_d, wid, lane);
    };
    float o[4] = {0.f, 0.f, 0.f, 0.f};
    if (r.bytes) {
      if (z_ok && mbar_wait_for(h ? bar_u : bar_g, 0, f.spin)) {
        if (tid == 0) F2_MARK(7);
        int16_t* cq = reinterpret_cast<int16_t*>(fsm + f.off_cq) + (size_t)wid * G * f.s16;
        gu_share<G>(p, r, h, r2, l, zs, cq, f.s16, wid - h * kF2GuWarps, lane, o, load_dn);
      } else {
        if (lane == 0) atomicCAS(p.status, 0, BITSMOE_ERR_TIMEOUT);
        load_dn();
      }
    } else {
      load_dn();
    }
    *reinterpret_cast<float4*>(pw + wid * kRows + 4 * lane) = make_float4(o[0], o[1], o[2], o[3]);
    if (tid == 0) F2_MARK(8);
    __syncthreads();
    if (tid == 0 && e1 > e0) {   // every warp's z gathers are done: this block's output-basis rows
      mbar_expect_tx(bar_e, (uint32_t)(e1 - e0) * row_out);
      bulk_run(r1, reinterpret_cast<const uint8_t*>(p.basis_out) + (size_t)e0 * row_out, (uint32_t)(e1 - e0) * row_out,
               bar_e);
    }
    if (tid < 2 * kRows) {   // this block's partial row (gate or up) into slot crank of every block
      const int hh = tid >> 7, row = tid & (kRows - 1);
      float v = 0.f;
#pragma unroll
      for (int w = 0; w < kF2GuWarps; ++w) v += pw[(hh * kF2GuWarps + w) * kRows + row];
      float* dst = xch + crank * 2 * kRows + tid;
      if (CL == 1) *dst = v;
      else
        for (int q = 0; q < CL; ++q) st_cluster_f32(dst, (uint32_t)q, v);
    }
    if (CL > 1) cluster_sync_all();
    else __syncthreads();
    if (tid == 0) F2_MARK(9);
    // h = SiLU(gate) * up of the 128 rows, as int16 with one scale, and its sums per
    // quantisation group (rows past I have gate = up = 0, so h = 0 there); the staging
    // area's end (free now) collects this block's down contributions s_j
    float* sdn = reinterpret_cast<float*>(fsm + f.off_ss);
    for (int i = tid; i < p.n_pad / 4; i += kFThreads) reinterpret_cast<float4*>(sdn)[i] = make_float4(0.f, 0.f, 0.f, 0.f);
    float hv = 0.f;
    if (tid < kRows) {
      float g = 0.f, u = 0.f;
      for (int q = 0; q < CL; ++q) {
        g += xch[q * 2 * kRows + tid];
        u += xch[q * 2 * kRows + kRows + tid];
      }
      hv = __fdividef(g, 1.f + __expf(-g)) * u;
      const float m = warp_max(fabsf(hv));
      if (lane == 0) hred[wid] = m;
    }
    __syncthreads();
    const float mx = fmaxf(fmaxf(hred[0], hred[1]), fmaxf(hred[2], hred[3]));
    if (tid < kRows) {
      const int qv = __float2int_rn(hv * (mx > 0.f ? 32767.f / mx : 0.f));
      hq[tid] = (int16_t)qv;
      const int sq = __reduce_add_sync(0xFFFFFFFFu, qv);
      if (lane == 0) hws[wid] = sq;
    }
    __syncthreads();
    // ---- D: the down part's tiles, one warp per tile; each unit of the part is distinct,
    // so its contribution is stored, then the block adds the whole vector into s
    int hsum[G];
    if (G == 1) {
      hsum[0] = hws[0] + hws[1] + hws[2] + hws[3];
    } else {
#pragma unroll
      for (int g = 0; g < G; ++g) {   // G = 128 / group groups of 4 / G warps each
        int sacc = 0;
        for (int q = g * (4 / G); q < (g + 1) * (4 / G); ++q) sacc += hws[q];
        hsum[g] = sacc;
      }
    }
    const float hsc = mx * (1.f / 32767.f);
    const F2Dn& d = *rd;
    if (d.nslot) {
      cp_async_wait_all();   // this lane's own copies
      if (tid == 0) F2_MARK(15);
      const uint8_t* dst = r1 + f.off_d;
      const uint32_t mo = al128(dn_code_bytes(d)), ms = d.nslot * 4;
      const int* du = reinterpret_cast<const int*>(dst + mo);
      const float* da = reinterpret_cast<const float*>(dst + mo + ms);
      const uint32_t* dsz = reinterpret_cast<const uint32_t*>(dst + mo + 2 * ms);
      const int gshift = 31 - __clz(p.group);
      const int* hq32 = reinterpret_cast<const int*>(hq);
      const float wa = sel_w[a];
      const int ntile = (int)(d.nslot / 32);
      for (int tt = wid; tt < ntile; tt += kFWarps) {
        int k = 0, t = tt;
        uint32_t off = 0;
        while (k < d.nr - 1 && t >= d.ntl[k]) {
          off += (uint32_t)d.ntl[k] * ul_chunks(d.bits[k]) * kChunkBytes;
          t -= d.ntl[k];
          ++k;
        }
        const int b = d.bits[k];
        off += (uint32_t)t * ul_chunks(b) * kChunkBytes;
        const int slot = 32 * tt + lane;
        const float v = dn_tile<G>(b, dst + off + lane * 16, hq32, gshift, hsum, dsz + slot, (int)d.nslot);
        const float al = da[slot];
        if (al != 0.f) sdn[du[slot]] = wa * al * hsc * v;
      }
    }
    __syncthreads();
    for (int i = tid; i < p.n_pad / 4; i += kFThreads) {
      const float4 v = reinterpret_cast<const float4*>(sdn)[i];
      if (v.x != 0.f || v.y != 0.f || v.z != 0.f || v.w != 0.f) red_add_v4(p.s + 4 * i, v.x, v.y, v.z, v.w);
    }
  }
  // the gate/up copies have landed before the staging area takes s (they have, unless a
  // wait above ran out)
  if (tid == 0 && pair) {
    if (rg->bytes) mbar_wait_for(bar_g, 0, f.spin);
    if (ru->bytes) mbar_wait_for(bar_u, 0, f.spin);
  }
  if (tid == 0) F2_MARK(10);
  grid_barrier(cnt + 1, nb, p.status, flags + 1, f.spin);
  if (tid == 0) F2_MARK(11);
  if (tid == 0 && blk == 0) sync_finish(f.sync);   // every block has read the epoch

  // ---- E: y = Phi_dn s for rows [e0, e1)
  float* ss = reinterpret_cast<float*>(fsm + f.off_ss);
  for (int i = tid; i < p.n_pad / 4; i += kFThreads)
    reinterpret_cast<float4*>(ss)[i] = __ldcg(reinterpret_cast<const float4*>(p.s) + i);
  __syncthreads();
  if (e1 > e0) {
    bool ok = mbar_wait_for(bar_e, 0, f.spin);
    if (!ok && tid == 0) atomicCAS(p.status, 0, BITSMOE_ERR_TIMEOUT);
    for (int ri = wid; ok && ri < e1 - e0; ri += kFWarps) {
      const uint8_t* rp = r1 + (size_t)ri * row_out;
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
  if (tid == 0) F2_MARK(12);
  // every copy into shared memory has landed before the block leaves
  cp_async_wait_all();
}

}  // namespace

namespace bmoe {

// First tile of a run of tiles (tile bytes cb[k] for nt[k] tiles of bucket k) whose
// byte prefix reaches num/den of the run's bytes (the cut used for cluster parts).
static int cut_at(const std::vector<uint64_t>& cb, const std::vector<int>& nt, int num, int den) {
  uint64_t tot = 0;
  int n = 0;
  for (size_t k = 0; k < cb.size(); ++k) {
    tot += cb[k] * (uint64_t)nt[k];
    n += nt[k];
  }
  if (num <= 0) return 0;
  if (num >= den) return n;
  const uint64_t target = tot * (uint64_t)num / (uint64_t)den;
  uint64_t pre = 0;
  int t = 0;
  for (size_t k = 0; k < cb.size(); ++k) {
    const uint64_t end = pre + cb[k] * (uint64_t)nt[k];
    if (end >= target) return t + (int)(target > pre ? (target - pre + cb[k] - 1) / cb[k] : 0);
    pre = end;
    t += nt[k];
  }
  return n;
}
static uint32_t al128h(uint64_t v) { return (uint32_t)((v + 127) / 128 * 128); }

bool build_f2_tables(const uint8_t* img, int CL, std::vector<uint8_t>& out, F2Sizes* sz) {
  const ImageHeader& hd = *header_of(img);
  // every copy a record describes must lie inside the image (checked here, on the host,
  // so that a wrong record can never send the kernel outside the layer's allocation)
  bool inside = true;
  auto in_img = [&](uint64_t off, uint64_t bytes) {
    if (off > hd.total_bytes || bytes > hd.total_bytes - off || off % 16 || bytes % 16) inside = false;
  };
  const ExpertDesc* desc = desc_of(img);
  const int E = hd.E;
  const int G = std::max(1, kRows / hd.group);
  const size_t rank_bytes = (size_t)E * (2 * sizeof(F2Gu) + sizeof(F2Dn));
  out.assign(rank_bytes * CL, 0);
  *sz = F2Sizes{0, 0, 0};
  std::vector<uint32_t> gu_need((size_t)CL * E, 0);
  for (int h = 0; h < 3; ++h)
    for (int e = 0; e < E; ++e) {
      const ExpertDesc& x = desc[(size_t)h * E + e];
      std::vector<uint64_t> cb;
      std::vector<int> nt;
      for (int k = 0; k < x.nbk; ++k) {
        const int b = x.bk[k].bits;
        cb.push_back(h < 2 ? (uint64_t)rl_chunks(b) * kChunkBytes : (uint64_t)ul_chunks(b) * kChunkBytes);
        nt.push_back(x.bk[k].ntiles);
      }
      for (int r = 0; r < CL; ++r) {
        const int p0 = cut_at(cb, nt, r, CL), p1 = cut_at(cb, nt, r + 1, CL);
        uint8_t* rank = out.data() + (size_t)r * rank_bytes;
        if (h < 2) {
          F2Gu g;
          std::memset(&g, 0, sizeof(g));
          for (int k = 0; k < x.nbk; ++k) {
            const BucketDesc& bd = x.bk[k];
            const int lo = std::min(std::max(p0 - bd.tile0, 0), bd.ntiles);
            const int hi = std::min(std::max(p1 - bd.tile0, 0), bd.ntiles);
            if (hi <= lo) continue;
            const int C = rl_chunks(bd.bits), U = rl_units(bd.bits);
            if (g.nr == 0) {
              const uint64_t slot0 = (uint64_t)bd.slot0 + (uint64_t)lo * U;
              g.code0 = x.code_base + bd.code_off + (uint64_t)lo * C * kChunkBytes;
              g.unit0 = x.unit_off + slot0 * 4;
              g.alpha0 = x.alpha_off + slot0 * 4;
              g.sz0 = x.sz_off + slot0 * 4;
            }
            g.bits[g.nr] = (uint8_t)bd.bits;
            g.ntl[g.nr] = (uint16_t)(hi - lo);
            ++g.nr;
            g.bytes += (uint32_t)((hi - lo) * C * kChunkBytes);
            g.nslot += (uint32_t)((hi - lo) * U);
          }
          g.rb_stride = (uint32_t)x.rb_stride;
          g.sz_row = (uint32_t)x.nslots * 4;
          if (g.bytes) {
            in_img(g.code0, (uint64_t)(hd.NRB - 1) * g.rb_stride + g.bytes);
            in_img(g.unit0, (uint64_t)g.nslot * 4);
            in_img(g.alpha0, (uint64_t)g.nslot * 4);
            in_img(g.sz0, (uint64_t)(hd.NG - 1) * g.sz_row + (uint64_t)g.nslot * 4);
          }
          std::memcpy(rank + ((size_t)h * E + e) * sizeof(F2Gu), &g, sizeof(g));
          if (g.bytes) {
            gu_need[(size_t)r * E + e] += al128h(al128h(g.bytes) + (uint64_t)g.nslot * 4 * (2 + G));
            for (int w = 0; w < kF2GuWarps; ++w) {   // quantised slots of each warp's share
              const int t0 = rl_split_at(g.bits, g.ntl, g.nr, w, kF2GuWarps);
              const int t1 = rl_split_at(g.bits, g.ntl, g.nr, w + 1, kF2GuWarps);
              int t = 0, nq = 0;
              for (int k = 0; k < g.nr; ++k) {
                const int lo = std::min(std::max(t0 - t, 0), (int)g.ntl[k]);
                const int hi = std::min(std::max(t1 - t, 0), (int)g.ntl[k]);
                if (g.bits[k] < 16) nq += (hi - lo) * rl_units(g.bits[k]);
                t += g.ntl[k];
              }
              sz->s16 = std::max(sz->s16, nq);
            }
          }
        } else {
          F2Dn d;
          std::memset(&d, 0, sizeof(d));
          uint64_t cbytes = 0;
          for (int k = 0; k < x.nbk; ++k) {
            const BucketDesc& bd = x.bk[k];
            const int lo = std::min(std::max(p0 - bd.tile0, 0), bd.ntiles);
            const int hi = std::min(std::max(p1 - bd.tile0, 0), bd.ntiles);
            if (hi <= lo) continue;
            const uint64_t tb = (uint64_t)ul_chunks(bd.bits) * kChunkBytes;
            if (d.nr == 0) {
              const uint64_t slot0 = (uint64_t)bd.slot0 + (uint64_t)lo * 32;
              d.unit0 = x.unit_off + slot0 * 4;
              d.alpha0 = x.alpha_off + slot0 * 4;
              d.sz0 = x.sz_off + slot0 * 4;
            }
            d.code[d.nr] = x.code_base + bd.code_off + (uint64_t)lo * hd.NRB * tb;
            d.bits[d.nr] = (uint8_t)bd.bits;
            d.ntl[d.nr] = (uint16_t)(hi - lo);
            ++d.nr;
            d.nslot += (uint32_t)(hi - lo) * 32;
            cbytes += (uint64_t)(hi - lo) * tb;
          }
          d.sz_row = (uint32_t)x.nslots * 4;
          if (d.nslot) {
            for (int k = 0; k < d.nr; ++k) {
              const uint64_t tb = (uint64_t)ul_chunks(d.bits[k]) * kChunkBytes;
              in_img(d.code[k], (uint64_t)d.ntl[k] * hd.NRB * tb);
            }
            in_img(d.unit0, (uint64_t)d.nslot * 4);
            in_img(d.alpha0, (uint64_t)d.nslot * 4);
            in_img(d.sz0, (uint64_t)(hd.NG - 1) * d.sz_row + (uint64_t)d.nslot * 4);
          }
          std::memcpy(rank + (size_t)2 * E * sizeof(F2Gu) + (size_t)e * sizeof(F2Dn), &d, sizeof(d));
          if (d.nslot)
            sz->dn_stage = std::max(sz->dn_stage, (int)(al128h(cbytes) + (uint64_t)d.nslot * 4 * (2 + G)));
        }
      }
    }
  for (uint32_t v : gu_need) sz->gu_stage = std::max(sz->gu_stage, (int)v);
  return inside;
}

int f2_max_clusters(int G, int CL) {
  void (*kernel)(Fwd, F2Args) = G == 1 ? k_f2<1> : G == 2 ? k_f2<2> : k_f2<4>;
  const int smem = 227 * 1024;
  if (cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  cudaLaunchConfig_t c = {};
  c.gridDim = dim3(CL * 32);
  c.blockDim = dim3(kFThreads);
  c.dynamicSmemBytes = smem;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeClusterDimension;
  at[0].val.clusterDim.x = CL;
  at[0].val.clusterDim.y = 1;
  at[0].val.clusterDim.z = 1;
  c.attrs = at;
  c.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, kernel, &c) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return n;
}

bool f2_plan(const ImageHeader& hd, int top_k, int CL, int nclusters, const F2Sizes& sz, F2Args* f) {
  std::memset(f, 0, sizeof(*f));
  const int npairs = top_k * hd.NRB;
  if (CL < 1 || nclusters < npairs || npairs < 1 || top_k > 32) return false;
  const int grid = nclusters * CL, P = npairs * CL, Q = grid - P;
  const int G = std::max(1, kRows / hd.group);
  const size_t row_in = (size_t)hd.D_pad * 2, row_out = (size_t)hd.n_pad * 2;
  const size_t budget = 227 * 1024;
  f->CL = CL;
  f->npairs = npairs;
  f->rank_bytes = (uint32_t)((size_t)hd.E * (2 * sizeof(F2Gu) + sizeof(F2Dn)));
  f->s16 = (int)align_up((uint64_t)std::max(sz.s16, 8), 8) + 8;
  size_t off = 512;   // mbarriers and flags
  f->off_rec = (int)off;
  off += 384;
  f->off_route = (int)off;
  off = align_up(off + (size_t)(hd.E + 2 * top_k) * 4, 128);
  f->off_xs = (int)off;
  off = align_up(off + row_in, 128);
  f->off_cq = (int)off;
  off = align_up(off + (size_t)kFWarps * G * f->s16 * 2, 128);
  f->off_pw = (int)off;
  off += (size_t)kFWarps * kRows * 4;
  f->off_xch = (int)off;
  off = align_up(off + (size_t)CL * 2 * kRows * 4, 128);
  f->off_h = (int)off;
  off += 512;
  f->off_r1 = (int)off;
  // the end of shared memory: the gate/up staging of pair blocks, whose last bytes take
  // s in the last phase (every block); free blocks' input-basis rows reach up to s
  const size_t ss_b = align_up((size_t)hd.n_pad * 4, 128);
  const size_t r2 = std::max((size_t)sz.gu_stage, ss_b);
  if (off + r2 > budget) return false;
  f->smem = (int)budget;
  f->off_r2 = (int)(budget - align_up(r2, 128));
  f->off_ss = (int)(budget - ss_b);
  const size_t cap_p = (size_t)f->off_r2 - off;   // pair blocks: input rows, or output rows + down part
  const size_t cap_f = (size_t)f->off_ss - off;   // free blocks: input rows, or output rows
  const size_t dn = align_up((size_t)sz.dn_stage, 128);
  // Shares of the two bases: pair blocks also stream their expert part, so the free
  // blocks take more rows; choose the split with the fewest bytes on the busiest block.
  // before barrier 1 a pair block needs its input rows and gate/up part, a free block its
  // input rows; after it, the down part and output rows, resp. the output rows
  double best = -1.0;
  for (int ep = (hd.D + grid - 1) / grid; ep >= 0; --ep) {
    const int ef = Q > 0 ? std::max(0, (hd.D - P * ep + Q - 1) / Q) : 0;
    if (Q == 0 && P * ep < hd.D) break;
    const size_t zb = align_up((size_t)hd.n_pad * 8, 128);   // a pair block's z copy, below its down part
    if (std::max(align_up((size_t)ep * row_out, 128), zb) + dn > cap_p || (size_t)ef * row_out > cap_f) continue;
    for (int bp = (2 * hd.n + grid - 1) / grid; bp >= 0; --bp) {
      const int bf = Q > 0 ? std::max(0, (2 * hd.n - P * bp + Q - 1) / Q) : 0;
      if (Q == 0 && P * bp < 2 * hd.n) break;
      if ((size_t)bp * row_in > cap_p || (size_t)bf * row_in > cap_f) continue;
      const double pre = std::max((double)sz.gu_stage + (double)bp * row_in, Q > 0 ? (double)bf * row_in : 0.0);
      const double post = std::max((double)sz.dn_stage + (double)ep * row_out, Q > 0 ? (double)ef * row_out : 0.0);
      const double worst = pre + post;
      if (best < 0 || worst < best) {
        best = worst;
        f->b_per = bp;
        f->b_free = bf;
        f->e_per = ep;
        f->e_free = ef;
      }
    }
  }
  if (best < 0) return false;
  // a pair block's z copy sits at the buffer's start, below its down part
  f->off_d = (int)std::max(align_up((size_t)f->e_per * row_out, 128), align_up((size_t)hd.n_pad * 8, 128));
  if ((size_t)f->off_d + dn > cap_p) return false;
  f->rec_smem = f->rank_bytes <= (uint32_t)(budget - (size_t)f->off_r2) ? 1 : 0;
  const int bmax = std::max(f->b_per, f->b_free);
  f->b_stage = std::max(1, (bmax + kMaxBStages - 1) / kMaxBStages);
  f->b_nst = (bmax + f->b_stage - 1) / f->b_stage;
  f->spin = kSpin;
  f->prefetch_io = 1;
  return true;
}

cudaError_t launch_f2(const Fwd& p, const F2Args& f, int nclusters, cudaStream_t st, bool pdl) {
  static std::mutex mu;
  static int done_smem[3] = {0, 0, 0};
  const int G = std::max(1, kRows / p.group);
  void (*kernel)(Fwd, F2Args) = G == 1 ? k_f2<1> : G == 2 ? k_f2<2> : k_f2<4>;
  const int gi = G == 1 ? 0 : G == 2 ? 1 : 2;
  {
    std::lock_guard<std::mutex> lock(mu);
    if (f.smem > done_smem[gi]) {
      cudaError_t r = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, f.smem);
      if (r != cudaSuccess) return r;
      done_smem[gi] = f.smem;
    }
  }
  cudaLaunchAttribute attr[2];
  int na = 0;
  if (f.CL > 1) {
    attr[na].id = cudaLaunchAttributeClusterDimension;
    attr[na].val.clusterDim.x = f.CL;
    attr[na].val.clusterDim.y = 1;
    attr[na].val.clusterDim.z = 1;
    ++na;
  }
  if (pdl) {
    attr[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[na].val.programmaticStreamSerializationAllowed = 1;
    ++na;
  }
  cudaLaunchConfig_t c = {};
  c.gridDim = dim3(nclusters * f.CL);
  c.blockDim = dim3(kFThreads);
  c.dynamicSmemBytes = f.smem;
  c.stream = st;
  c.attrs = attr;
  c.numAttrs = na;
  return cudaLaunchKernelEx(&c, kernel, p, f);
}

}  // namespace bmoe

#ifdef BITSMOE_F2_TRACE
extern "C" int bitsmoe_f2_trace_read(void* dst) {
  return (int)cudaMemcpyFromSymbol(dst, g_f2_trace, sizeof(g_f2_trace));
}
#endif
