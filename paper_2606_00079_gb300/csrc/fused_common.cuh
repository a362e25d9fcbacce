// Device pieces shared by the two single-token kernels (fused.cu, fused2.cu):
// bounded grid barriers on workspace counters, bulk-copy and L2-prefetch runs,
// the integer dot products of the two packed layouts with the bit-width as a
// runtime parameter, and the routing of one token by the control warps.
// Included by CUDA translation units only (each gets its own internal copy).
#pragma once
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

// Grid barrier on a counter that is zero at kernel start.  Arrival: thread 0
// of a block, after the block's (or a warp group's) bar.sync has ordered the
// writes to publish, adds 1 with release semantics.  Wait: lane 0 of warps
// 0..3 poll with acquire loads, starting about 100 ns apart so that the
// polls interleave, until one of them sees every block; then the whole block
// synchronises.  Data written before the barrier is read with L2-coherent
// loads after it.
__device__ __forceinline__ void grid_arrive(uint32_t* cnt) {
  asm volatile("red.release.gpu.global.add.u32 [%0], 1;" ::"l"(cnt) : "memory");
}
__device__ __forceinline__ void grid_wait(uint32_t* cnt, uint32_t nblocks, int* status, volatile int* seen,
                                          long long spin = kSpin) {
  const int wid = threadIdx.x >> 5;
  if ((threadIdx.x & 31) == 0 && wid < 4) {
    if (wid) __nanosleep(100 * wid);
    const long long t0 = clock64();
    while (!*seen) {
      if (ld_acquire_u32(cnt) >= nblocks) {
        *seen = 1;
        break;
      }
      if (clock64() - t0 > spin) {
        if (wid == 0) atomicCAS(status, 0, BITSMOE_ERR_TIMEOUT);
        break;
      }
    }
  }
  __syncthreads();
}
// The same wait for the control warps only (lane 0 of each polls; then they sync on barrier 2).
__device__ __forceinline__ void grid_wait_ctl(uint32_t* cnt, uint32_t nblocks, int* status, volatile int* seen,
                                              int cw, int nthreads, long long spin = kSpin) {
  if ((threadIdx.x & 31) == 0) {
    if (cw) __nanosleep(100 * cw);
    const long long t0 = clock64();
    while (!*seen) {
      if (ld_acquire_u32(cnt) >= nblocks) {
        *seen = 1;
        break;
      }
      if (clock64() - t0 > spin) {
        if (cw == 0) atomicCAS(status, 0, BITSMOE_ERR_TIMEOUT);
        break;
      }
    }
  }
  asm volatile("bar.sync 2, %0;" ::"r"(nthreads) : "memory");
}
__device__ __forceinline__ void grid_barrier(uint32_t* cnt, uint32_t nblocks, int* status, volatile int* seen,
                                             long long spin = kSpin) {
  __syncthreads();
  if (threadIdx.x == 0) grid_arrive(cnt);
  grid_wait(cnt, nblocks, status, seen, spin);
}

// Barrier counters of the single-token kernels: kSyncWords words at a fixed workspace
// offset.  Word 0 counts the calls that have completed (the epoch); two sets of four
// counters follow (words 4-7 and 8-11; in each: grid barriers 1-3, then the norm mode's
// logits).  Call E uses set E & 1 and clears set (E + 1) & 1 for call E + 1: that set's
// last user, call E - 1, completed before this call's PDL wait returned.  Block 0 adds 1
// to the epoch after the last grid barrier, when every block has read it.  So nothing is
// reset at the end of a call (no block waits for an atomic's return before it exits), and
// a call whose waits ran out still leaves a clean set to the next call.  A zero-filled
// workspace is a valid start (epoch 0, both sets clear).
constexpr int kSyncWords = 12;
__device__ __forceinline__ uint32_t* sync_set(uint32_t* sync, uint32_t epoch) { return sync + 4 + 4 * (epoch & 1u); }
__device__ __forceinline__ void sync_clear_next(uint32_t* sync, uint32_t epoch) {
  *reinterpret_cast<uint4*>(sync_set(sync, epoch + 1u)) = make_uint4(0u, 0u, 0u, 0u);
}
__device__ __forceinline__ void sync_finish(uint32_t* sync) {
  asm volatile("red.relaxed.gpu.global.add.u32 [%0], 1;" ::"l"(sync) : "memory");
}

__device__ __forceinline__ void prefetch_run(const uint8_t* p, uint64_t bytes) {
  while (bytes > 0) {
    const uint32_t c = bytes > 65536 ? 65536u : (uint32_t)bytes;
    prefetch_l2(p, c);
    p += c;
    bytes -= c;
  }
}

// Debug bounds checks (dbg bit 1): a staging record's copies must lie inside the packed
// image; a record that fails is reported as BITSMOE_ERR_DEVICE_BOUNDS and its item skipped.
__device__ __forceinline__ bool in_image(const Fwd& p, uint64_t off, uint64_t len) {
  return off <= p.img_bytes && len <= p.img_bytes - off;
}
__device__ __forceinline__ void report_bounds(int* status) { atomicCAS(status, 0, BITSMOE_ERR_DEVICE_BOUNDS); }

// Issue `bytes` (16-byte multiple, 16-byte aligned) into shared memory on an
// mbarrier whose transaction count the caller has set.
__device__ __forceinline__ void bulk_run(void* dst, const uint8_t* src, uint32_t bytes, uint64_t* bar) {
  uint32_t o = 0;
  while (o < bytes) {
    const uint32_t c = bytes - o < 32768u ? bytes - o : 32768u;
    bulk_g2s(static_cast<uint8_t*>(dst) + o, src + o, c, bar);
    o += c;
  }
}

// ---------------------------------------------------------------------------
// Integer dot products with the bit-width as a runtime parameter: one small
// loop per bit plane keeps the code that a phase runs small (the kernel runs
// each phase once per call, so instruction fetch is on its critical path).
// ---------------------------------------------------------------------------
// Row-lane layout, one bit plane over `ntl` tiles: chunks c0 .. c0 + nc - 1 of
// each tile of C chunks hold PB-bit fields of consecutive unit groups (chunk
// c0 + q at activation offset q * coff); word w of the lane's 16 bytes is row
// w; unit 4k + m of a chunk at bit 8m + PB*k.  cp: int16 activation pairs,
// cstep int32 per tile.  One out-of-line copy per field width, accumulators
// passed by value (registers).
template <int PB>
__device__ __noinline__ int4 rl_plane(const uint8_t* code, int ntl, int C, int c0, int nc, int coff, const int* cp,
                                      int cstep, int4 acc) {
  // Field k of every byte is selected by one mask without a shift: the dot products of
  // field k then carry a factor 2^(PB k), so each field keeps its own accumulators and
  // is scaled back exactly (an arithmetic shift of a multiple of 2^(PB k)) at the end.
  // Headroom: at most 32 tiles x 2 chunks x 4 units x 32767 x 255 < 2^31 per accumulator.
  constexpr int NK = 8 / PB;
  constexpr uint32_t MASK = ((1u << PB) - 1u) * 0x01010101u;
  int4 ak[NK];
#pragma unroll
  for (int kq = 0; kq < NK; ++kq) ak[kq] = make_int4(0, 0, 0, 0);
#pragma unroll 1
  for (int t = 0; t < ntl; ++t) {
#pragma unroll 1
    for (int q = 0; q < nc; ++q) {
      const uint4 v = lds128(code + (size_t)(t * C + c0 + q) * kChunkBytes);
      const int* ct = cp + t * cstep + q * coff;
      int2 cc[NK];
#pragma unroll
      for (int kq = 0; kq < NK; ++kq) cc[kq] = *reinterpret_cast<const int2*>(ct + 2 * kq);
#pragma unroll
      for (int kq = 0; kq < NK; ++kq) {
        constexpr uint32_t M0 = MASK;
        const uint32_t m = M0 << (PB * kq);
        uint32_t b = v.x & m;
        ak[kq].x = dp2a_hi(cc[kq].y, b, dp2a_lo(cc[kq].x, b, ak[kq].x));
        b = v.y & m;
        ak[kq].y = dp2a_hi(cc[kq].y, b, dp2a_lo(cc[kq].x, b, ak[kq].y));
        b = v.z & m;
        ak[kq].z = dp2a_hi(cc[kq].y, b, dp2a_lo(cc[kq].x, b, ak[kq].z));
        b = v.w & m;
        ak[kq].w = dp2a_hi(cc[kq].y, b, dp2a_lo(cc[kq].x, b, ak[kq].w));
      }
    }
  }
#pragma unroll
  for (int kq = 0; kq < NK; ++kq) {
    acc.x += ak[kq].x >> (PB * kq);
    acc.y += ak[kq].y >> (PB * kq);
    acc.z += ak[kq].z >> (PB * kq);
    acc.w += ak[kq].w >> (PB * kq);
  }
  return acc;
}

// A bucket range of a gate/up item (b < 16): accf[w] += sum_u code_{w,u} * c_u,
// flushed to fp32 every 32 tiles (int32 headroom for 8-bit codes).
__device__ void rl_range_rt(int b, const uint8_t* code, int ntl, const int* cp, float (&accf)[4]) {
  const int C = rl_chunks(b), cstep = rl_units(b) / 2;
  const int hs = b == 3 ? 2 : 4;
  for (int t0 = 0; t0 < ntl; t0 += 32) {
    const int n = min(32, ntl - t0);
    const uint8_t* cb = code + (size_t)t0 * C * kChunkBytes;
    const int* cpp = cp + t0 * cstep;
    int4 lo = make_int4(0, 0, 0, 0), hi = make_int4(0, 0, 0, 0);
    switch (b) {
      case 1: lo = rl_plane<1>(cb, n, 1, 0, 1, 0, cpp, cstep, lo); break;
      case 2: lo = rl_plane<2>(cb, n, 1, 0, 1, 0, cpp, cstep, lo); break;
      case 4: lo = rl_plane<4>(cb, n, 1, 0, 1, 0, cpp, cstep, lo); break;
      case 8: lo = rl_plane<8>(cb, n, 1, 0, 1, 0, cpp, cstep, lo); break;
      case 3:   // low 2-bit plane of units 0-15 and 16-31, then the high bit of units 0-31
        lo = rl_plane<2>(cb, n, 3, 0, 2, 8, cpp, cstep, lo);
        hi = rl_plane<1>(cb, n, 3, 2, 1, 0, cpp, cstep, hi);
        break;
      default:  // 6: low 4-bit plane of units 0-7 and 8-15, then the high 2 bits of units 0-15
        lo = rl_plane<4>(cb, n, 3, 0, 2, 4, cpp, cstep, lo);
        hi = rl_plane<2>(cb, n, 3, 2, 1, 0, cpp, cstep, hi);
        break;
    }
    accf[0] += (float)(lo.x + (hi.x << hs));
    accf[1] += (float)(lo.y + (hi.y << hs));
    accf[2] += (float)(lo.z + (hi.z << hs));
    accf[3] += (float)(lo.w + (hi.w << hs));
  }
}

// Unit-lane layout, `nc` consecutive 16-byte chunks of PB-bit fields of the
// lane's unit (chunk q covers rows rbase + q * 128 / PB ..): word w of a chunk
// covers 32 / PB rows, row r' = 4k + m at bit 8m + PB*k.  Returns the dot with
// the int16 activations per group g of the row block (G <= 4) in .x .. .w.
template <int PB, int G>
__device__ __noinline__ int4 ul_plane(const uint8_t* cb, int nc, int rbase, const int* hq32, int gshift, int4 acc) {
  constexpr int NK = 8 / PB, RPW = 32 / PB;
  constexpr uint32_t MASK = ((1u << PB) - 1u) * 0x01010101u;
#pragma unroll 1
  for (int q = 0; q < nc; ++q) {
    const uint4 v = lds128(cb + (size_t)q * kChunkBytes);
    const uint32_t wv[4] = {v.x, v.y, v.z, v.w};
    const int rq = rbase + q * (kRows / PB);
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      const int r0 = rq + w * RPW;
      const int* hp = hq32 + r0 / 2;
      int2 hh[NK];
#pragma unroll
      for (int kq = 0; kq < NK; ++kq) hh[kq] = *reinterpret_cast<const int2*>(hp + 2 * kq);
      int tmp = 0;
#pragma unroll
      for (int kq = 0; kq < NK; ++kq) {
        const uint32_t b = (wv[w] >> (PB * kq)) & MASK;
        tmp = dp2a_hi(hh[kq].y, b, dp2a_lo(hh[kq].x, b, tmp));
      }
      const int gl = G == 1 ? 0 : (r0 >> gshift);
      if (gl == 0) acc.x += tmp;
      else if (gl == 1) acc.y += tmp;
      else if (gl == 2) acc.z += tmp;
      else acc.w += tmp;
    }
  }
  return acc;
}

// Warps 0 .. kBW-1 project (phase B); warps kBW .. kFWarps-1 route and stage.
constexpr int kBW = 12;
constexpr int kCT = (kFWarps - kBW) * 32;   // control threads

// Routing of the token by the kCT control threads: the k largest logits (ties to the
// lower index) into sel_e, their softmax into sel_w.  Out of line so that one copy of
// the code exists: the kernel runs it once on dummy keys (logits == nullptr) while it
// waits for the previous kernel, which brings the code into the instruction cache.
__device__ __noinline__ void route_token(const float* logits, int E, int k, uint32_t* keys, int* sel_e,
                                         float* sel_w, int ct) {
  for (int i = ct; i < E; i += kCT) keys[i] = logits ? order_key(__ldcg(logits + i)) : 0u;
  asm volatile("bar.sync 2, %0;" ::"r"(kCT) : "memory");
  for (int i = ct; i < E; i += kCT) {
    const uint32_t key = keys[i];
    int rank = 0;
    int f2 = 0;
    for (; f2 + 4 <= E; f2 += 4) {
      const uint4 o = *reinterpret_cast<const uint4*>(keys + f2);
      rank += (o.x > key) | ((o.x == key) & (f2 < i));
      rank += (o.y > key) | ((o.y == key) & (f2 + 1 < i));
      rank += (o.z > key) | ((o.z == key) & (f2 + 2 < i));
      rank += (o.w > key) | ((o.w == key) & (f2 + 3 < i));
    }
    for (; f2 < E; ++f2) {
      const uint32_t o = keys[f2];
      rank += (o > key) | ((o == key) & (f2 < i));
    }
    if (rank < k) {
      sel_e[rank] = i;
      sel_w[rank] = key ? __uint_as_float((key & 0x80000000u) ? (key & 0x7FFFFFFFu) : ~key)
                        : __int_as_float(0x7FC00000);   // key 0: a NaN logit
    }
  }
  asm volatile("bar.sync 2, %0;" ::"r"(kCT) : "memory");
  if (ct < 32) {
    const float m = sel_w[0];
    const float ev = ct < k ? expf(sel_w[ct] - m) : 0.f;
    float sum = ev;
#pragma unroll
    for (int o = 16; o; o >>= 1) sum += __shfl_xor_sync(0xFFFFFFFFu, sum, o);
    __syncwarp();   // every lane has read sel_w[0]
    if (ct < k) sel_w[ct] = ev * (1.f / sum);
  }
}

}  // namespace
