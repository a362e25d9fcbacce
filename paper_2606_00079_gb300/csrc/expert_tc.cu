// Tensor-core gate/up factors for calls with several tokens per expert (Eq. 3's
// expert factors applied to the shared-basis coordinates):
//
//   gate/up[pair][h][i] = sum_j p_hat_{h,e}[i, j] * alpha_{h,e,j} * z_h[t][j]
//   p_hat[i, j] = scale_{j,g(i)} * (q_ij - zero_{j,g(i)})          (group g along i)
//
// as an M = 128 rows (one row block, inside one quantisation group) x N = the
// expert's tokens x K = the expert's unit slots contraction on tcgen05:
//
//   A[i][slot] = q_ij as bf16 (exact below 256), decoded once per row block from the
//                packed row-lane streams into 128-byte-swizzled K-major tiles (a byte
//                permute and a packed subtraction per two codes; no scales on A);
//   B[t][slot] = scale_{j,g} * alpha_j * z_h[t][j] as a bf16 pair hi + lo (two MMAs
//                into the same fp32 accumulator keep about 16 bits of it);
//   result     = A B - corr[t],  corr[t] = sum_slot zero_{j,g} * B[t][slot].
//
// One block per (routed expert, h, row block); it walks the expert's slots in
// ranges of R slots (R / 64 K-blocks resident at a time).  Each range's code
// bytes, unit indices, alphas and scale/zero are bulk-copied into one of two
// shared-memory buffers two ranges ahead; the block decodes A from there, builds
// B, and one thread issues the range's MMAs, whose commit frees A and B.  Each
// (pair, h, row) is written by exactly one block: plain stores, no atomics.
// Requires: every unit below 16 bits and the group a multiple of 128 rows (the
// host checks the layer once at upload), and zT = z stored [2][n_pad][T] (token
// fastest, which the tensor-core projection writes for this kernel).
#include <cuda_bf16.h>

#include <algorithm>
#include <cstring>
#include <mutex>

#include "device.cuh"
#include "tc.cuh"

namespace {

constexpr int kXThreads = 256;
constexpr uint32_t kXATile = 128 * 64 * 2;   // one A K-block: 128 rows x 64 slots bf16

// One row-lane code tile of an (h, e): its byte offset in the row block's stream (in
// the staged buffer once the range's start is subtracted), its first slot (relative to
// the range when decoding), its bit-width and its slot count.
struct TileRec {
  int off, slot, bits, pad_;
};

struct XArgs {
  int R;           // slots per range (multiple of 64)
  int NTmax;       // largest token tile (16 .. 64, power of two)
  int max_tiles;   // most row-lane tiles of any gate/up (h, e)
  int max_ranges;  // most slot ranges of any gate/up (h, e)
};

// 4 codes (bytes) -> two bf16x2 words, exact.  Codes below 128: bf16 bits 0x4300 | q
// are 128 + q, and one packed bf16 subtraction per two codes removes the 128 (an
// offset left in A would cost accuracy in the fp32 accumulation).  8-bit codes go
// through fp32 (2^23 + q - 2^23).
__device__ __forceinline__ uint2 codes_bf16(uint32_t q4, int bits) {
  if (bits < 8) {
    uint32_t lo = __byte_perm(q4, 0x43434343u, 0x4140), hi = __byte_perm(q4, 0x43434343u, 0x4342);
    const __nv_bfloat162 off = __floats2bfloat162_rn(128.f, 128.f);
    const __nv_bfloat162 a = __hsub2(*reinterpret_cast<__nv_bfloat162*>(&lo), off);
    const __nv_bfloat162 b = __hsub2(*reinterpret_cast<__nv_bfloat162*>(&hi), off);
    return make_uint2(*reinterpret_cast<const uint32_t*>(&a), *reinterpret_cast<const uint32_t*>(&b));
  }
  float f[4];
#pragma unroll
  for (int m = 0; m < 4; ++m) f[m] = __uint_as_float(__byte_perm(q4, 0x4B000000u, 0x7440 + m)) - 8388608.f;
  __nv_bfloat162 a = __floats2bfloat162_rn(f[0], f[1]), b = __floats2bfloat162_rn(f[2], f[3]);
  return make_uint2(*reinterpret_cast<uint32_t*>(&a), *reinterpret_cast<uint32_t*>(&b));
}

__device__ __forceinline__ uint32_t sw_off(int r, int c16) {   // byte offset of chunk c16 of row r
  return (uint32_t)(r >> 3) * 1024u + (uint32_t)(r & 7) * 128u + (uint32_t)((c16 ^ (r & 7)) << 4);
}

__device__ __forceinline__ uint32_t lds32(const uint8_t* p) { return *reinterpret_cast<const uint32_t*>(p); }

// Row `row` of one staged row-lane tile of B-bit codes into the A tiles: the lane's
// word(s) of the row hold all U units of the tile; group k (units 4k .. 4k + 3) sits
// at bit 8m + b * k' of its plane (see the packed format), four codes per extraction.
template <int B>
__device__ __forceinline__ void decode_tile(const uint8_t* cb, const TileRec& tr, int row, uint8_t* sa, int R) {
  constexpr int U = rl_units(B), C = rl_chunks(B), NG = U / 4;
  constexpr uint32_t kMask = B == 1 ? 0x01010101u : B == 2 ? 0x03030303u : B == 4 ? 0x0F0F0F0Fu : 0xFFFFFFFFu;
  const uint8_t* src = cb + tr.off + (row >> 2) * 16 + (row & 3) * 4;
  const uint32_t w0 = lds32(src);
  const uint32_t w1 = C > 1 ? lds32(src + kChunkBytes) : 0u;
  const uint32_t w2 = C > 2 ? lds32(src + 2 * kChunkBytes) : 0u;
  const uint32_t rbase = (uint32_t)(row >> 3) * 1024u + (uint32_t)(row & 7) * 128u;
  const int rx = row & 7;
#pragma unroll
  for (int k = 0; k < NG; ++k) {
    const int sl = tr.slot + 4 * k;
    if (sl < 0 || sl >= R) continue;
    uint32_t q;
    if (B == 3) q = (((k < 4 ? w0 : w1) >> (2 * (k & 3))) & 0x03030303u) | (((w2 >> k) & 0x01010101u) << 2);
    else if (B == 6) q = (((k < 2 ? w0 : w1) >> (4 * (k & 1))) & 0x0F0F0F0Fu) | (((w2 >> (2 * k)) & 0x03030303u) << 4);
    else q = (w0 >> (B * k)) & kMask;
    const uint2 v = codes_bf16(q, B);
    const uint32_t off = (uint32_t)(sl >> 6) * kXATile + rbase + ((uint32_t)(((sl & 63) >> 3) ^ rx) << 4) +
                         ((uint32_t)((sl >> 2) & 1) << 3);
    *reinterpret_cast<uint2*>(sa + off) = v;
  }
}

// Bytes of the staged code buffer for R slots: 128 bytes per slot at 8 bits, plus a
// partial tile (at most 3 chunks of 512 bytes) at each end.
__host__ __device__ constexpr uint32_t code_buf_bytes(int R) { return (uint32_t)R * 128u + 3072u; }

__global__ void __launch_bounds__(kXThreads, 2) k_gu_tc(Fwd p, XArgs xa) {
  extern __shared__ uint8_t xsm_raw[];
  uint8_t* xsm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(xsm_raw) + 1023) & ~(uintptr_t)1023);
  const int R = xa.R, nkb = R / 64;
  const uint32_t cbb = code_buf_bytes(R);
  uint8_t* sa = xsm;                                                   // [nkb][128 x 128 B]
  uint8_t* sb = sa + (size_t)nkb * kXATile;                            // hi [nkb][NT x 128 B], then lo
  const uint32_t b_half = (uint32_t)nkb * xa.NTmax * 128;
  uint8_t* cbuf = sb + 2 * (size_t)b_half;                             // [2][cbb] staged codes
  uint8_t* mbuf = cbuf + 2 * (size_t)cbb;                              // [2][unit R | alpha R | scale-zero R]
  TileRec* tl = reinterpret_cast<TileRec*>(mbuf + 2 * (size_t)R * 12); // [max_tiles] every tile of (h, e)
  float* sw = reinterpret_cast<float*>(tl + xa.max_tiles);             // [R] scale * alpha per slot
  float* scz = sw + R;                                                 // [R] zero point per slot
  int* rtb = reinterpret_cast<int*>(scz + R);                          // [max_ranges + 1] first tile of each range
  int* rte = rtb + xa.max_ranges + 1;                                  // [max_ranges + 1] end of its tiles
  int* tok = rte + xa.max_ranges + 1;                                  // [NTmax] token of tile row t
  int* pair = tok + xa.NTmax;                                          // [NTmax]
  float* corr = reinterpret_cast<float*>(pair + xa.NTmax);             // [NTmax]
  int* cstart = reinterpret_cast<int*>(corr + xa.NTmax);               // [2] stream byte of each code buffer
  uint64_t* cbar = reinterpret_cast<uint64_t*>(((uintptr_t)(cstart + 2) + 7) & ~(uintptr_t)7);   // [2] copies
  uint64_t* bar = cbar + 2;                                            // MMA commits
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bar + 1);
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;

  pdl_trigger();
  int w = blockIdx.x;
  const int rb = w % p.NRB;
  w /= p.NRB;
  const int h = w & 1, a = w >> 1;
  pdl_wait();   // routing and z come from earlier kernels
  if (a >= p.active[0]) return;
  const int e = p.active[1 + a];
  const int ntok = p.expert_count[e], pst = p.expert_start[e];
  if (ntok <= 0 || ntok < p.tc_gu_min) return;   // fewer tokens: the dp2a kernel's expert
  const ExpertDesc& xd = p.desc[h * p.E + e];
  const int nslots = xd.nslots, nbk = xd.nbk;
  const int g = (rb * kRows) / p.group;
  const uint8_t* code = p.img + xd.code_base + (size_t)rb * xd.rb_stride;
  const uint8_t* unit_g = p.img + xd.unit_off;
  const uint8_t* alpha_g = p.img + xd.alpha_off;
  const uint8_t* sz_g = p.img + xd.sz_off + (size_t)g * nslots * 4;
  const int nr = (nslots + R - 1) / R;

  // accumulator columns: the largest token tile this block needs
  const int nt_need = min(xa.NTmax, max(16, (int)((ntok + 15) & ~15)));
  int NT = 16;
  while (NT < nt_need) NT <<= 1;
  const uint32_t ncols = NT < 32 ? 32u : (uint32_t)NT;
  const int lgNT = 31 - __clz(NT);

  // every tile of (h, e) in slot order (warp 0: lane k lists bucket k's tiles), then the
  // tiles each slot range touches: [rtb, rte) (a tile may straddle two ranges)
  if (wid == 0) {
    int cnt = 0;
    if (lane < nbk) cnt = xd.bk[lane].ntiles;
    int incl = cnt;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int v = __shfl_up_sync(0xFFFFFFFFu, incl, o);
      if (lane >= o) incl += v;
    }
    if (lane < nbk) {
      const BucketDesc& bd = xd.bk[lane];
      const int b = bd.bits, U = rl_units(b), C = rl_chunks(b);
      for (int t = 0; t < cnt; ++t) {
        TileRec tr;
        tr.off = (int)bd.code_off + t * C * kChunkBytes;
        tr.slot = bd.slot0 + t * U;
        tr.bits = b;
        tr.pad_ = U;
        tl[incl - cnt + t] = tr;
      }
    }
  }
  if (tid == 0) {
    mbar_init_n(bar, 1);
    mbar_init(cbar);
    mbar_init(cbar + 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (wid == 1) tmem_alloc(tmem_slot, ncols);
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = *tmem_slot;
  const uint32_t idesc = idesc_bf16(NT);
  for (int r = tid; r < nr; r += kXThreads) {   // binary searches over the tile list
    const int s0 = r * R, s1 = min(s0 + R, nslots);
    int lo = 0, hi = xd.ntiles;   // first tile ending after s0
    while (lo < hi) {
      const int m = (lo + hi) >> 1;
      if (tl[m].slot + tl[m].pad_ <= s0) lo = m + 1;
      else hi = m;
    }
    rtb[r] = lo;
    hi = xd.ntiles;   // first tile starting at or after s1
    while (lo < hi) {
      const int m = (lo + hi) >> 1;
      if (tl[m].slot < s1) lo = m + 1;
      else hi = m;
    }
    rte[r] = lo;
  }

  // range r of the slots into buffer r & 1: the code bytes of its tiles, its unit
  // indices, alphas and this group's scale/zero (one thread; the range's tile list is ready)
  auto issue = [&](int r) {
    if (r >= nr) return;
    const int s0 = r * R, s1 = min(s0 + R, nslots);
    const TileRec& t0 = tl[rtb[r]];
    const TileRec& t1 = tl[rte[r] - 1];
    const uint32_t start = (uint32_t)t0.off;
    const uint32_t end = (uint32_t)t1.off + (uint32_t)rl_chunks(t1.bits) * kChunkBytes;
    const int buf = r & 1;
    cstart[buf] = (int)start;
    const uint32_t mb = (uint32_t)(s1 - s0) * 4;
    fence_proxy_async();   // earlier generic reads of this buffer, then async writes
    mbar_expect_tx(cbar + buf, (end - start) + 3 * mb);
    for (uint32_t o = start; o < end; o += 32768u)
      bulk_g2s(cbuf + (size_t)buf * cbb + (o - start), code + o, min(32768u, end - o), cbar + buf);
    uint8_t* m = mbuf + (size_t)buf * R * 12;
    bulk_g2s(m, unit_g + (size_t)s0 * 4, mb, cbar + buf);
    bulk_g2s(m + (size_t)R * 4, alpha_g + (size_t)s0 * 4, mb, cbar + buf);
    bulk_g2s(m + (size_t)R * 8, sz_g + (size_t)s0 * 4, mb, cbar + buf);
  };

  uint32_t ncommit = 0;
  uint32_t cuse = 0;   // bit b: parity of buffer b's next completion
  bool ok = true;
  for (int tt0 = 0; tt0 < ntok; tt0 += NT) {   // token tiles (one unless the expert has many tokens)
    const int nt = min(NT, ntok - tt0);
    for (int t = tid; t < NT; t += kXThreads) {
      const int q = t < nt ? p.pair_list[pst + tt0 + t] : 0;
      pair[t] = q;
      tok[t] = q / p.k;
      corr[t] = 0.f;
    }
    __syncthreads();   // range table
    if (tid == 32) issue(0);
    for (int r = 0; r < nr; ++r) {
      const int s0 = r * R, s1 = min(s0 + R, nslots), buf = r & 1;
      // the previous range's MMAs must be done with A and B, and this range's copies must
      // have landed: thread 0 waits, the block meets it at a barrier
      if (tid == 0) {
        if (ncommit > 0) ok &= mbar_wait(bar, (ncommit - 1) & 1u);
        ok &= mbar_wait(cbar + buf, (cuse >> buf) & 1u);
      }
      cuse ^= 1u << buf;
      asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
      __syncthreads();
      asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      // the next range's copies go out now (its buffer was last read by range r - 1)
      if (tid == 32) issue(r + 1);
      const uint8_t* cb = cbuf + (size_t)buf * cbb;
      const int* su = reinterpret_cast<const int*>(mbuf + (size_t)buf * R * 12);
      const float* sal = reinterpret_cast<const float*>(su + R);
      const uint32_t* ssz = reinterpret_cast<const uint32_t*>(sal + R);
      const int nval = s1 - s0;
      // per-slot scale * alpha and zero point; zeros for A beyond the expert's last slot
      for (int ls = tid; ls < R; ls += kXThreads) {
        float wv = 0.f, cz = 0.f;
        if (ls < nval) {
          const uint32_t szw = ssz[ls];
          wv = __half2float(__ushort_as_half((unsigned short)(szw & 0xFFFFu))) * sal[ls];
          cz = __half2float(__ushort_as_half((unsigned short)(szw >> 16)));
        }
        sw[ls] = wv;
        scz[ls] = cz;
      }
      {
        const int kend = min(R, (nval + 63) & ~63);
        for (int item = tid; item < 128 * ((kend - nval) >> 2); item += kXThreads) {
          const int row = item & 127, sl = nval + 4 * (item >> 7);
          const uint32_t off = (uint32_t)(sl >> 6) * kXATile + (uint32_t)(row >> 3) * 1024u + (uint32_t)(row & 7) * 128u +
                               ((uint32_t)(((sl & 63) >> 3) ^ (row & 7)) << 4) + ((uint32_t)((sl >> 2) & 1) << 3);
          *reinterpret_cast<uint2*>(sa + off) = make_uint2(0u, 0u);
        }
      }
      // A: warp item = (tile, 32-row group), lane = row; bit-width uniform in the warp
      {
        const int tb = rtb[r], nitem = (rte[r] - tb) * 4, cs0 = cstart[buf];
        for (int item = wid; item < nitem; item += kXThreads / 32) {
          TileRec tr = tl[tb + (item >> 2)];
          tr.off -= cs0;
          tr.slot -= s0;
          const int row = 32 * (item & 3) + lane;
          switch (tr.bits) {
            case 1: decode_tile<1>(cb, tr, row, sa, R); break;
            case 2: decode_tile<2>(cb, tr, row, sa, R); break;
            case 3: decode_tile<3>(cb, tr, row, sa, R); break;
            case 4: decode_tile<4>(cb, tr, row, sa, R); break;
            case 6: decode_tile<6>(cb, tr, row, sa, R); break;
            default: decode_tile<8>(cb, tr, row, sa, R); break;
          }
        }
      }
      __syncthreads();   // per-slot factors ready
      // B: thread (token row t, 8-slot chunk c); a thread keeps one t over its items
      {
        const int t = tid & (NT - 1);
        const float* zrow = p.zT + (size_t)h * p.n_pad * p.T + (t < nt ? tok[t] : 0);
        const uint32_t T32 = (uint32_t)p.T;
        float cs = 0.f;
        for (int item = tid; item < NT * (R / 8); item += kXThreads) {
          const int c = item >> lgNT, sl0 = 8 * c;
          float v[8];
          const int4 ja = *reinterpret_cast<const int4*>(su + sl0), jb = *reinterpret_cast<const int4*>(su + sl0 + 4);
          const int jj[8] = {ja.x, ja.y, ja.z, ja.w, jb.x, jb.y, jb.z, jb.w};
#pragma unroll
          for (int u = 0; u < 8; ++u) v[u] = (t < nt && sl0 + u < nval) ? __ldcg(zrow + (uint32_t)jj[u] * T32) : 0.f;
          const float4 wa = *reinterpret_cast<const float4*>(sw + sl0), wb = *reinterpret_cast<const float4*>(sw + sl0 + 4);
          const float4 ca = *reinterpret_cast<const float4*>(scz + sl0), cb4 = *reinterpret_cast<const float4*>(scz + sl0 + 4);
          const float wv[8] = {wa.x, wa.y, wa.z, wa.w, wb.x, wb.y, wb.z, wb.w};
          const float cz[8] = {ca.x, ca.y, ca.z, ca.w, cb4.x, cb4.y, cb4.z, cb4.w};
          uint32_t hw[4], lw[4];
#pragma unroll
          for (int m = 0; m < 4; ++m) {
            const float v0 = wv[2 * m] * v[2 * m], v1 = wv[2 * m + 1] * v[2 * m + 1];
            cs = fmaf(cz[2 * m], v0, cs);
            cs = fmaf(cz[2 * m + 1], v1, cs);
            // hi = v truncated to bf16, lo = v - hi (exact) rounded to bf16: about 16 bits of v
            const uint32_t h0 = __float_as_uint(v0) & 0xFFFF0000u, h1 = __float_as_uint(v1) & 0xFFFF0000u;
            hw[m] = __byte_perm(h0, h1, 0x7632);
            const __nv_bfloat162 bl = __floats2bfloat162_rn(v0 - __uint_as_float(h0), v1 - __uint_as_float(h1));
            lw[m] = *reinterpret_cast<const uint32_t*>(&bl);
          }
          const uint32_t off = (uint32_t)(c >> 3) * (uint32_t)NT * 128u + sw_off(t, c & 7);
          *reinterpret_cast<uint4*>(sb + off) = make_uint4(hw[0], hw[1], hw[2], hw[3]);
          *reinterpret_cast<uint4*>(sb + b_half + off) = make_uint4(lw[0], lw[1], lw[2], lw[3]);
        }
        if (t < nt && cs != 0.f) atomicAdd(corr + t, cs);
      }
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");   // generic writes -> tensor-core reads
      asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
      __syncthreads();
      if (tid == 0) {
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        const int kbn = min(nkb, (nval + 63) / 64);
        for (int kb = 0; kb < kbn; ++kb) {
          const uint32_t a0 = smem_u32(sa + (size_t)kb * kXATile);
          const uint32_t b0 = smem_u32(sb + (size_t)kb * NT * 128);
#pragma unroll
          for (int k16 = 0; k16 < 4; ++k16) {
            const uint64_t ad = sw128_desc(a0 + k16 * 32);
            mma_bf16(tmem, ad, sw128_desc(b0 + k16 * 32), idesc, (s0 | kb | k16) != 0);
            mma_bf16(tmem, ad, sw128_desc(b0 + b_half + k16 * 32), idesc, 1u);
          }
        }
        mma_commit(bar);
      }
      ++ncommit;
    }
    // epilogue: warps 0-3 own accumulator lanes (rows) 32w .. 32w + 31
    if (tid == 0) ok &= mbar_wait(bar, (ncommit - 1) & 1u);
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    if (wid < 4) {
      const int i = rb * kRows + 32 * wid + lane;
      for (int c0 = 0; c0 < nt; c0 += 8) {
        uint32_t rr[8];
        tmem_ld8(tmem + ((uint32_t)(32 * wid) << 16) + (uint32_t)c0, rr);
#pragma unroll
        for (int q = 0; q < 8; ++q)
          if (c0 + q < nt)
            p.gu[((size_t)pair[c0 + q] * 2 + h) * p.I_pad + i] = __uint_as_float(rr[q]) - corr[c0 + q];
      }
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();   // the accumulator and the tile's token table are reused by the next tile
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  }
  if (!ok && tid == 0) atomicCAS(p.status, 0, BITSMOE_ERR_TIMEOUT);
  if (wid == 1) tmem_dealloc(tmem, ncols);
}

// ---------------------------------------------------------------------------
// Down factor on tensor cores (Eq. 3's down projection, summed over the routed
// experts before the output basis):
//
//   s[t][j] += g_{t,e} * alpha_{dn,e,j} * sum_i p_hat[i, j] * h_{t,e}[i]
//   p_hat[i, j] = scale_{j,g(i)} * (q_ij - zero_{j,g(i)}),   h = SiLU(gate) * up
//
// One block per (routed expert, 128 down slots = four unit-lane tiles); the K
// dimension is the expert's rows i, one row block (two K-blocks) per step:
//   A[slot][i] = q_ij (bf16, exact), decoded from the unit-lane streams (a lane owns a
//                unit and its codes run along i);
//   B[t][i]    = h_t[i] as a bf16 pair hi + lo;
//   per group: P = A B in TMEM; out[slot][t] += scale * (P - zero * H_g[t]) in
//              registers, H_g[t] = sum over the group's rows of h_t[i];
//   finally s[t][unit] += g_{t,e} * alpha * out with fp32 reductions (experts meet in s).
// ---------------------------------------------------------------------------
constexpr int kDNT = 64;   // largest token tile of the down kernel

struct DArgs {
  int NTmax;   // 16 .. 64, power of two
  int mt_max;  // 128-slot tiles of the largest down (e)
};

// 4 codes of rows 4k .. 4k + 3 -> A[slot = row][K = kk .. kk + 3] (kk: row inside the row block)
__device__ __forceinline__ void store_a4(uint8_t* sa, int row, int kk, uint2 v) {
  const uint32_t off = (uint32_t)(kk >> 6) * kXATile + (uint32_t)(row >> 3) * 1024u + (uint32_t)(row & 7) * 128u +
                       ((uint32_t)(((kk & 63) >> 3) ^ (row & 7)) << 4) + ((uint32_t)((kk >> 2) & 1) << 3);
  *reinterpret_cast<uint2*>(sa + off) = v;
}

// Rows 64 hp .. 64 hp + 63 of one unit's staged row block (its 16-byte chunks at
// `ln`, chunk c at ln + 512 c) into A row `row`.
template <int B>
__device__ __forceinline__ void decode_ul(const uint8_t* ln, int hp, int row, uint8_t* sa) {
  if (B == 3) {   // low 2-bit plane: chunk hp, word w = rows 64 hp + 16 w ..; high bit: chunk 2, word = row / 32
    const uint8_t* lo = ln + hp * kChunkBytes;
    const uint8_t* hi = ln + 2 * kChunkBytes;
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      const uint32_t wl = lds32(lo + 4 * w), wh = lds32(hi + 4 * (2 * hp + (w >> 1)));
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const uint32_t q = ((wl >> (2 * k)) & 0x03030303u) | (((wh >> (4 * (w & 1) + k)) & 0x01010101u) << 2);
        store_a4(sa, row, 64 * hp + 16 * w + 4 * k, codes_bf16(q, 3));
      }
    }
  } else if (B == 6) {   // low 4-bit plane: chunks 2hp, 2hp+1 (rows 32c + 8w ..); high 2 bits: chunk 4 + hp (16 rows a word)
#pragma unroll
    for (int cc = 0; cc < 2; ++cc) {
      const uint8_t* lo = ln + (2 * hp + cc) * kChunkBytes;
#pragma unroll
      for (int w = 0; w < 4; ++w) {
        const int r0 = 32 * cc + 8 * w;   // row inside this half
        const uint32_t wl = lds32(lo + 4 * w), wh = lds32(ln + (4 + hp) * kChunkBytes + 4 * (r0 >> 4));
#pragma unroll
        for (int k = 0; k < 2; ++k) {
          const int rr = r0 + 4 * k;
          const uint32_t q = ((wl >> (4 * k)) & 0x0F0F0F0Fu) | (((wh >> (2 * ((rr & 15) >> 2))) & 0x03030303u) << 4);
          store_a4(sa, row, 64 * hp + rr, codes_bf16(q, 6));
        }
      }
    }
  } else {   // 1, 2, 4, 8: chunk c covers rows 128c/B .., word 32/B rows, group k at bit B*k
    constexpr int RPW = 32 / B;   // rows per word
    constexpr uint32_t kMask = B == 1 ? 0x01010101u : B == 2 ? 0x03030303u : B == 4 ? 0x0F0F0F0Fu : 0xFFFFFFFFu;
#pragma unroll
    for (int wi = 0; wi < 2 * B; ++wi) {   // the 2B words of rows 64 hp ..
      const int gw = 2 * B * hp + wi;      // word index over the row block
      const uint32_t wv = lds32(ln + (gw >> 2) * kChunkBytes + 4 * (gw & 3));
#pragma unroll
      for (int k = 0; k < RPW / 4; ++k) store_a4(sa, row, gw * RPW + 4 * k, codes_bf16((wv >> (B * k)) & kMask, B));
    }
  }
}

__global__ void __launch_bounds__(kXThreads, 2) k_dn_tc(Fwd p, DArgs da) {
  extern __shared__ uint8_t dsm_raw[];
  uint8_t* dsm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(dsm_raw) + 1023) & ~(uintptr_t)1023);
  constexpr uint32_t kCodeBuf = 4 * 8 * kChunkBytes;              // four tiles of at most 8 chunks
  uint8_t* sa = dsm;                                                // [2 K-blocks][128 x 128 B]
  uint8_t* sb = sa + 2 * kXATile;                                   // hi [2][NT x 128 B], then lo
  const uint32_t b_half = 2u * da.NTmax * 128u;
  uint8_t* cbuf = sb + 2 * (size_t)b_half;                          // [2][kCodeBuf]
  uint32_t* szb = reinterpret_cast<uint32_t*>(cbuf + 2 * kCodeBuf); // [2][128] scale | zero of the group
  int* su = reinterpret_cast<int*>(szb + 256);                      // [128] unit of each slot
  float* sal = reinterpret_cast<float*>(su + 128);                  // [128] alpha
  float* hs = sal + 128;                                            // [2][kDNT] group sums of h per token
  int* tok = reinterpret_cast<int*>(hs + 2 * kDNT);                 // [kDNT]
  float* pw = reinterpret_cast<float*>(tok + kDNT);                 // [kDNT] gate weight of the pair
  int* pairs = reinterpret_cast<int*>(pw + kDNT);                   // [kDNT]
  int* tq = pairs + kDNT;                                           // [4] bits | [4] buffer offset | [4] stream offset
  uint64_t* cbar = reinterpret_cast<uint64_t*>(tq + 12);            // [2]
  uint64_t* bar = cbar + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bar + 1);
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;

  pdl_trigger();
  const int mt = blockIdx.x % da.mt_max, a = blockIdx.x / da.mt_max;
  pdl_wait();   // routing and gate/up come from earlier kernels
  if (a >= p.active[0]) return;
  const int e = p.active[1 + a];
  const int ntok = p.expert_count[e], pst = p.expert_start[e];
  const ExpertDesc& xd = p.desc[2 * p.E + e];
  const int m0 = mt * 128;
  if (ntok <= 0 || ntok < p.tc_dn_min || m0 >= xd.nslots) return;   // fewer tokens: the dp2a kernel's expert
  const int nslots = xd.nslots, nsl = min(128, nslots - m0), nq = nsl / 32;
  const int nt_need = min(da.NTmax, max(16, (ntok + 15) & ~15));
  int NT = 16;
  while (NT < nt_need) NT <<= 1;
  const uint32_t ncols = NT < 32 ? 32u : (uint32_t)NT;
  const int lgNT = 31 - __clz(NT);

  if (tid < 4) {   // the block's unit-lane tiles: bits, offset in the code buffer, stream offset of row block 0
    const int t = 4 * mt + tid;
    int bits = 0, src = 0;
    if (tid < nq) {
      int k = 0;
      for (int q = 1; q < xd.nbk; ++q)
        if (t >= xd.bk[q].tile0) k = q;
      bits = xd.bk[k].bits;
      src = (int)xd.bk[k].code_off + (t - xd.bk[k].tile0) * p.NRB * bits * kChunkBytes;
    }
    tq[tid] = bits;
    tq[8 + tid] = src;
  }
  if (tid < 128) {
    su[tid] = tid < nsl ? reinterpret_cast<const int*>(p.img + xd.unit_off)[m0 + tid] : 0;
    sal[tid] = tid < nsl ? reinterpret_cast<const float*>(p.img + xd.alpha_off)[m0 + tid] : 0.f;
  }
  if (tid < 2 * kDNT) hs[tid] = 0.f;
  if (tid == 0) {
    mbar_init_n(bar, 1);
    mbar_init(cbar);
    mbar_init(cbar + 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (wid == 1) tmem_alloc(tmem_slot, ncols);
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  if (tid == 0) {
    int o = 0;
    for (int q = 0; q < 4; ++q) {
      tq[4 + q] = o;
      o += tq[q] * kChunkBytes;
    }
  }
  const uint32_t tmem = *tmem_slot;
  const uint32_t idesc = idesc_bf16(NT);
  const uint8_t* code = p.img + xd.code_base;
  const uint32_t* szg = reinterpret_cast<const uint32_t*>(p.img + xd.sz_off);

  // row block r of the four tiles (each tile's B chunks are contiguous per row block) and
  // the scale/zero of its group, into buffer r & 1 (one thread)
  auto issue = [&](int r) {
    if (r >= p.NRB) return;
    const int buf = r & 1, g = (r * kRows) / p.group;
    uint32_t bytes = (uint32_t)nsl * 4;
    for (int q = 0; q < nq; ++q) bytes += (uint32_t)tq[q] * kChunkBytes;
    fence_proxy_async();
    mbar_expect_tx(cbar + buf, bytes);
    for (int q = 0; q < nq; ++q)
      bulk_g2s(cbuf + (size_t)buf * kCodeBuf + tq[4 + q], code + tq[8 + q] + (size_t)r * tq[q] * kChunkBytes,
               (uint32_t)tq[q] * kChunkBytes, cbar + buf);
    bulk_g2s(szb + buf * 128, szg + (size_t)g * nslots + m0, (uint32_t)nsl * 4, cbar + buf);
  };

  float out[kDNT];
  uint32_t ncommit = 0, cuse = 0;
  bool ok = true;
  for (int tt0 = 0; tt0 < ntok; tt0 += NT) {
    const int nt = min(NT, ntok - tt0);
#pragma unroll
    for (int q = 0; q < kDNT; ++q) out[q] = 0.f;
    __syncthreads();   // the previous tile's scatter has read tok / pw
    for (int t = tid; t < NT; t += kXThreads) {
      const int q = t < nt ? p.pair_list[pst + tt0 + t] : 0;
      pairs[t] = q;
      tok[t] = q / p.k;
      pw[t] = t < nt ? p.pair_weight[q] : 0.f;
    }
    if (tid < 2 * kDNT) hs[tid] = 0.f;
    __syncthreads();
    if (tid == 32) issue(0);
    for (int r = 0; r < p.NRB; ++r) {
      const int buf = r & 1, g = (r * kRows) / p.group;
      const bool gfirst = (r * kRows) % p.group == 0, glast = ((r + 1) * kRows) % p.group == 0 || r == p.NRB - 1;
      if (tid == 0) {
        if (ncommit > 0) ok &= mbar_wait(bar, (ncommit - 1) & 1u);
        ok &= mbar_wait(cbar + buf, (cuse >> buf) & 1u);
      }
      cuse ^= 1u << buf;
      asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
      __syncthreads();
      asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      if (tid == 32) issue(r + 1);
      // A: thread = (slot, half of the rows); a warp holds 32 slots of one tile
      {
        const int m = tid & 127, hp = tid >> 7, q = m >> 5;
        const int bits = tq[q];
        const uint8_t* ln = cbuf + (size_t)buf * kCodeBuf + tq[4 + q] + (m & 31) * 16;
        switch (bits) {
          case 1: decode_ul<1>(ln, hp, m, sa); break;
          case 2: decode_ul<2>(ln, hp, m, sa); break;
          case 3: decode_ul<3>(ln, hp, m, sa); break;
          case 4: decode_ul<4>(ln, hp, m, sa); break;
          case 6: decode_ul<6>(ln, hp, m, sa); break;
          case 8: decode_ul<8>(ln, hp, m, sa); break;
          default: {   // slots past the expert's last tile: zeros
#pragma unroll
            for (int kk = 0; kk < 64; kk += 4) store_a4(sa, m, 64 * hp + kk, make_uint2(0u, 0u));
          }
        }
      }
      // B: h = SiLU(gate) * up of the expert's pairs for this row block, as the bf16 pair
      // prepared once per pair (k_h_pack): thread (token row t, 8-row chunk c), t fixed per thread
      {
        const int t = tid & (NT - 1);
        const bool live = t < nt;
        const size_t hrow = (size_t)pairs[t] * p.I_pad + (size_t)r * kRows;
        for (int item = tid; item < NT * 16; item += kXThreads) {
          const int c = item >> lgNT;
          uint4 hw = make_uint4(0, 0, 0, 0), lw = make_uint4(0, 0, 0, 0);
          if (live) {
            hw = __ldcg(reinterpret_cast<const uint4*>(p.hh + hrow + 8 * c));
            lw = __ldcg(reinterpret_cast<const uint4*>(p.hl + hrow + 8 * c));
          }
          const uint32_t off = (uint32_t)(c >> 3) * (uint32_t)NT * 128u + sw_off(t, c & 7);
          *reinterpret_cast<uint4*>(sb + off) = hw;
          *reinterpret_cast<uint4*>(sb + b_half + off) = lw;
        }
        if (gfirst && tid < NT) hs[(g & 1) * kDNT + tid] = tid < nt ? __ldcg(p.hsum + (size_t)pairs[tid] * p.NG + g) : 0.f;
      }
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
      __syncthreads();
      if (tid == 0) {
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
#pragma unroll
        for (int kb = 0; kb < 2; ++kb) {
          const uint32_t a0 = smem_u32(sa + (size_t)kb * kXATile);
          const uint32_t b0 = smem_u32(sb + (size_t)kb * NT * 128);
#pragma unroll
          for (int k16 = 0; k16 < 4; ++k16) {
            const uint64_t ad = sw128_desc(a0 + k16 * 32);
            mma_bf16(tmem, ad, sw128_desc(b0 + k16 * 32), idesc, (!gfirst || kb || k16) ? 1u : 0u);
            mma_bf16(tmem, ad, sw128_desc(b0 + b_half + k16 * 32), idesc, 1u);
          }
        }
        mma_commit(bar);
      }
      ++ncommit;
      if (glast) {   // the group's partial sums: out += scale * (P - zero * H)
        if (tid == 0) ok &= mbar_wait(bar, (ncommit - 1) & 1u);
        asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
        __syncthreads();
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        if (wid < 4) {
          const int m = 32 * wid + lane;
          const uint32_t szw = szb[buf * 128 + m];
          const float sc = m < nsl ? __half2float(__ushort_as_half((unsigned short)(szw & 0xFFFFu))) : 0.f;
          const float zp = m < nsl ? __half2float(__ushort_as_half((unsigned short)(szw >> 16))) : 0.f;
          const float* hg = hs + (g & 1) * kDNT;
#pragma unroll
          for (int c0 = 0; c0 < kDNT; c0 += 8) {
            if (c0 < nt) {
              uint32_t rr[8];
              tmem_ld8(tmem + ((uint32_t)(32 * wid) << 16) + (uint32_t)c0, rr);
#pragma unroll
              for (int q = 0; q < 8; ++q) out[c0 + q] = fmaf(sc, __uint_as_float(rr[q]) - zp * hg[c0 + q], out[c0 + q]);
            }
          }
        }
      }
    }
    // s[t][unit] += g_{t,e} * alpha * out (experts meet in s: fp32 reductions)
    if (wid < 4) {
      const int m = 32 * wid + lane;
      const float al = sal[m];
      if (m < nsl && al != 0.f) {
        float* sp = p.s + su[m];
#pragma unroll
        for (int q = 0; q < kDNT; ++q)
          if (q < nt) atomicAdd(sp + (size_t)tok[q] * p.n_pad, pw[q] * al * out[q]);
      }
    }
  }
  if (!ok && tid == 0) atomicCAS(p.status, 0, BITSMOE_ERR_TIMEOUT);
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  if (wid == 1) tmem_dealloc(tmem, ncols);
}

// h = SiLU(gate) * up of every routed pair whose expert takes the tensor-core down
// kernel, once: as the bf16 pair hi (truncation) + lo (rounded remainder) that the
// down kernel's B operand needs, and its sums over each quantisation group.  Thread =
// 8 consecutive rows of one pair; the threads of a group meet by warp shuffles.
__global__ void __launch_bounds__(256) k_h_pack(Fwd p) {
  pdl_trigger();
  const int per_pair = p.I_pad / 8;
  const size_t idx = (size_t)blockIdx.x * 256 + threadIdx.x;
  pdl_wait();   // gate/up come from the previous kernels
  if (idx >= (size_t)p.P * per_pair) return;   // whole 16-thread groups: I_pad / 8 is a multiple of 16
  const int q = (int)(idx / per_pair), c = (int)(idx - (size_t)q * per_pair);
  const int e = p.pair_expert[q];
  if (p.expert_count[e] < p.tc_dn_min) return;   // the dp2a down kernel's expert (whole pair: 16-thread groups)
  const float* gp = p.gu + (size_t)q * 2 * p.I_pad + 8 * c;
  const float4 g0 = __ldcg(reinterpret_cast<const float4*>(gp)), g1 = __ldcg(reinterpret_cast<const float4*>(gp + 4));
  const float4 u0 = __ldcg(reinterpret_cast<const float4*>(gp + p.I_pad));
  const float4 u1 = __ldcg(reinterpret_cast<const float4*>(gp + p.I_pad + 4));
  const float gg[8] = {g0.x, g0.y, g0.z, g0.w, g1.x, g1.y, g1.z, g1.w};
  const float uu[8] = {u0.x, u0.y, u0.z, u0.w, u1.x, u1.y, u1.z, u1.w};
  uint32_t hw[4], lw[4];
  float sum = 0.f;
#pragma unroll
  for (int m = 0; m < 4; ++m) {
    const float v0 = gg[2 * m] / (1.f + __expf(-gg[2 * m])) * uu[2 * m];
    const float v1 = gg[2 * m + 1] / (1.f + __expf(-gg[2 * m + 1])) * uu[2 * m + 1];
    sum += v0 + v1;
    const uint32_t h0 = __float_as_uint(v0) & 0xFFFF0000u, h1 = __float_as_uint(v1) & 0xFFFF0000u;
    hw[m] = __byte_perm(h0, h1, 0x7632);
    const __nv_bfloat162 bl = __floats2bfloat162_rn(v0 - __uint_as_float(h0), v1 - __uint_as_float(h1));
    lw[m] = *reinterpret_cast<const uint32_t*>(&bl);
  }
  *reinterpret_cast<uint4*>(p.hh + (size_t)q * p.I_pad + 8 * c) = make_uint4(hw[0], hw[1], hw[2], hw[3]);
  *reinterpret_cast<uint4*>(p.hl + (size_t)q * p.I_pad + 8 * c) = make_uint4(lw[0], lw[1], lw[2], lw[3]);
  // 16 consecutive threads cover one 128-row block of one pair; a group is one or more blocks
  const unsigned gm = __activemask();
#pragma unroll
  for (int o = 8; o; o >>= 1) sum += __shfl_xor_sync(gm, sum, o);
  if ((threadIdx.x & 15) == 0) atomicAdd(p.hsum + (size_t)q * p.NG + (8 * c) / p.group, sum);
}

}  // namespace

namespace bmoe {

// Shared memory of k_gu_tc.
static size_t gu_tc_smem(const XArgs& xa) {
  const int R = xa.R;
  return 1024 + (size_t)(R / 64) * kXATile + 2 * (size_t)(R / 64) * xa.NTmax * 128 + 2 * (size_t)code_buf_bytes(R) +
         2 * (size_t)R * 12 + (size_t)xa.max_tiles * sizeof(TileRec) + 2 * (size_t)R * 4 +
         2 * ((size_t)xa.max_ranges + 1) * 4 + 3 * (size_t)xa.NTmax * 4 + 8 + 8 + 3 * 8 + 16;
}

cudaError_t launch_gu_tc(const Fwd& p, int max_tiles, int max_slots, cudaStream_t st, bool pdl) {
  XArgs xa;
  int nt = 16;
  while (nt < p.T && nt < 64) nt <<= 1;   // experts with more tokens take several token tiles
  xa.NTmax = nt;
  xa.R = nt <= 32 ? 128 : 64;
  xa.max_tiles = std::max(1, max_tiles);
  xa.max_ranges = (max_slots + xa.R - 1) / xa.R;
  const size_t smem = gu_tc_smem(xa);
  static std::mutex mu;
  static size_t done = 0;
  {
    std::lock_guard<std::mutex> lock(mu);
    if (smem > done) {
      const cudaError_t r = cudaFuncSetAttribute(k_gu_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
      if (r != cudaSuccess) return r;
      done = smem;
    }
  }
  const int A_max = std::min(p.E, p.P);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(A_max * 2 * p.NRB));
  cfg.blockDim = dim3(kXThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, k_gu_tc, p, xa);
}

cudaError_t launch_h_pack(const Fwd& p, cudaStream_t st, bool pdl) {
  const size_t nth = (size_t)p.P * (p.I_pad / 8);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)((nth + 255) / 256));
  cfg.blockDim = dim3(256);
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, k_h_pack, p);
}

cudaError_t launch_dn_tc(const Fwd& p, int ul_max_tiles, cudaStream_t st, bool pdl) {
  DArgs da;
  int nt = 16;
  while (nt < p.T && nt < kDNT) nt <<= 1;   // experts with more tokens take several token tiles
  da.NTmax = nt;
  da.mt_max = std::max(1, (ul_max_tiles + 3) / 4);
  const size_t smem = 1024 + 2 * (size_t)kXATile + 4 * (size_t)nt * 128 + 2 * 4 * 8 * kChunkBytes + 256 * 4 +
                      128 * 8 + 2 * kDNT * 4 + 3 * kDNT * 4 + 12 * 4 + 3 * 8 + 16;
  static std::mutex mu;
  static size_t done = 0;
  {
    std::lock_guard<std::mutex> lock(mu);
    if (smem > done) {
      const cudaError_t r = cudaFuncSetAttribute(k_dn_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
      if (r != cudaSuccess) return r;
      done = smem;
    }
  }
  const int A_max = std::min(p.E, p.P);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(A_max * da.mt_max));
  cfg.blockDim = dim3(kXThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, k_dn_tc, p, da);
}

}  // namespace bmoe
