// Per-projection bit allocation: which bit-width every spectral unit gets.
//
// BitsMoE chooses b_u in {0,1,2,3,4,6,8,16} for the units of one projection
// type by the ILP of Eq. ilp_piecewise_eps: minimise sum_u C_u(b_u) subject to
// sum_u b_u <= B_h, with C_u(b) = alpha_u^2 beta_u^gamma E_u(b) (Eq.
// app_component_loss_final) and the piecewise distortion of Eq.
// piecewise_expected_eps (eta 2^(-2b) for b >= 6 with eta = d rho^2 / 3,
// kappa_b for 2..4, sin^2 theta = 1 - ||p||_1^2 / d for 1 bit, 1 for 0 bits).
// The paper hands the ILP to a commercial solver; here it is solved by the
// Lagrangian relaxation of the multiple-choice knapsack plus a greedy fill:
//
//   k_alloc_cost   one warp per 32 units, eight rows streamed side by side:
//                  rho = max |p| and ||p||_1 (an exact fixed-point sum, so the
//                  order of the lanes does not matter)
//                  per unit, then each lane builds its unit's costs and the
//                  lower convex hull of (b, C(b)) from b = 0 (ties to the
//                  smaller b, efficiencies capped so they never increase); an
//                  increment's key is (bits of its efficiency) << 32 | ~u
//   radix select   four passes over the 16-bit digits of the keys: a histogram
//                  of the increments' bit counts by digit (k_alloc_hist), then
//                  one block finds the digit where the bits taken so far would
//                  pass B_h (k_alloc_scan); after the last pass the cut K* is
//                  the key of the first increment group that does not fit
//   k_alloc_final  every unit takes its increments with key > K* (the
//                  Lagrangian solution) and exposes its next one
//   fill rounds    while a next increment fits the bits left, the one with
//                  the largest key is taken (grid-wide max, then one thread)
//
// Everything is fp32 with each operation rounded once, in the same steps as
// the allocation oracle, so the bit-widths are a deterministic function of
// the inputs.  The cost kernel streams the units once (HBM-bound); the rest
// works on 64 bytes per unit of workspace.
#include <cuda_runtime.h>
#include <stdint.h>

#include <algorithm>

#include "device.cuh"
#include "internal.h"

namespace {

constexpr int kAW = 8;                 // warps per block of the cost kernel
constexpr int kNB = 8;                 // bit-width options
constexpr int kNS = 7;                 // at most 7 hull increments
constexpr int kFillRounds = 16;        // the fill takes at most 15 increments (bits left < 16)
constexpr int kDigits = 65536;
__constant__ int c_bits[kNB] = {0, 1, 2, 3, 4, 6, 8, 16};

struct AllocState {
  unsigned long long prefix;   // key bits decided by the radix passes
  unsigned long long above;    // bits of the increments above the current bucket (all taken)
  unsigned long long kstar;    // the cut: increments with key > kstar are taken (0: all)
  unsigned long long used;     // bits after the cut
  unsigned long long best;     // fill round: largest fitting next key
  long long left;              // fill: bits left
  int all_fit;                 // every increment fits: nothing to select
  int fill_done;
};

struct AllocWs {
  AllocState* st;
  unsigned long long* hist;    // [kDigits]
  unsigned long long* keys;    // [U][kNS], 0 = none
  uint8_t* reach;              // [U][kNS] option index reached by each increment
  uint8_t* taken;              // [U]
  unsigned long long* nkey;    // [U] next increment's key (0 = none)
  uint8_t* ndb;                // [U] its bits
};

size_t ws_layout(int64_t U, size_t* off) {
  size_t o = 0;
  auto put = [&](int i, size_t bytes) {
    off[i] = o;
    o = (o + bytes + 255) / 256 * 256;
  };
  put(0, sizeof(AllocState));
  put(1, (size_t)kDigits * 8);
  put(2, (size_t)U * kNS * 8);
  put(3, (size_t)U * kNS);
  put(4, (size_t)U);
  put(5, (size_t)U * 8);
  put(6, (size_t)U);
  return o;
}

__device__ __forceinline__ float weight(float a, float b, float gamma) {
  float bg;
  if (gamma == 0.f) bg = 1.f;
  else if (gamma == 0.5f) bg = __fsqrt_rn(b);
  else if (gamma == 1.f) bg = b;
  else bg = powf(b, gamma);
  return __fmul_rn(__fmul_rn(a, a), bg);
}

// Costs and hull of one unit (one lane), written to its rows of the workspace.
__device__ void unit_hull(float rho, long long l1fix, int d, float w, float k2, float k3, float k4, uint32_t u,
                          unsigned long long* keys, uint8_t* reach) {
  const float l1 = __fmul_rn(__ll2float_rn(l1fix), 9.094947017729282e-13f);   // 2^-40
  const float sin2 = __fsub_rn(1.f, __fdiv_rn(__fmul_rn(l1, l1), (float)d));
  const float eta = __fdiv_rn(__fmul_rn(__fmul_rn(rho, rho), (float)d), 3.f);
  float C[kNB];
  C[0] = w;                                  // w * 1
  C[1] = __fmul_rn(w, sin2);
  C[2] = __fmul_rn(w, k2);
  C[3] = __fmul_rn(w, k3);
  C[4] = __fmul_rn(w, k4);
  C[5] = __fmul_rn(w, __fmul_rn(eta, 2.44140625e-4f));       // 2^-12
  C[6] = __fmul_rn(w, __fmul_rn(eta, 1.52587890625e-5f));    // 2^-16
  C[7] = __fmul_rn(w, __fmul_rn(eta, 2.3283064365386963e-10f));   // 2^-32
  int cur = 0;
  float curc = C[0], prev = __int_as_float(0x7F800000);
  const unsigned long long low = 0xFFFFFFFFull - u;
#pragma unroll 1
  for (int s = 0; s < kNS; ++s) {
    float be = 0.f;
    int bj = -1;
#pragma unroll
    for (int j = 1; j < kNB; ++j) {
      if (j > cur) {
        const float e = __fdiv_rn(__fsub_rn(curc, C[j]), (float)(c_bits[j] - c_bits[cur]));
        if (e > 0.f && e > be) {
          be = e;
          bj = j;
        }
      }
    }
    if (bj < 0) {
      for (int r = s; r < kNS; ++r) {
        keys[r] = 0ull;
        reach[r] = 0xFF;
      }
      return;
    }
    const float e = fminf(be, prev);
    keys[s] = ((unsigned long long)__float_as_uint(e) << 32) | low;
    reach[s] = (uint8_t)bj;
    curc = C[bj];
    cur = bj;
    prev = e;
  }
}

struct CostArgs {
  const float* p;
  const float* alpha;
  const float* beta;
  float gamma, k2, k3, k4;
  int64_t U;
  int d;
  AllocWs w;
};

// floor(|x| 2^40) for |x| < 32 as A 2^22 + B with A = floor(y), B = floor(frac(y) 2^22),
// y = |x| 2^18 < 2^23: each is read off the bits of a round-toward-zero add of 2^23
// (2^23 + floor(v) for 0 <= v < 2^23).  The raw bit patterns are summed; the caller
// subtracts count * bits(2^23) (mod 2^32).  Also the running max |x|.
__device__ __forceinline__ void fix_add(float ax, float& mx, uint32_t& sa, uint32_t& sb) {
  mx = fmaxf(mx, ax);
  const float y = __fmul_rn(ax, 262144.f);                                          // 2^18
  const float ty = __fadd_rz(y, 8388608.f);                                         // 2^23 + floor(y)
  const float z = __fmul_rn(__fsub_rn(y, __fsub_rn(ty, 8388608.f)), 4194304.f);   // frac(y) 2^22
  sa += __float_as_uint(ty);
  sb += __float_as_uint(__fadd_rz(z, 8388608.f));
}

// One warp per 32 consecutive units; lane l keeps unit (base + l)'s rho and ||p||_1.
// The warp streams kUK units' rows side by side, so kUK 16-byte loads per lane are in
// flight at once.
constexpr int kUK = 8;
__global__ void __launch_bounds__(kAW * 32) k_alloc_cost(CostArgs a) {
  const int lane = threadIdx.x & 31;
  const int64_t nwarps = (int64_t)gridDim.x * kAW;
  const bool v4 = (a.d & 3) == 0;
  for (int64_t base = ((int64_t)blockIdx.x * kAW + (threadIdx.x >> 5)) * 32; base < a.U; base += nwarps * 32) {
    const int nu = a.U - base < 32 ? (int)(a.U - base) : 32;
    float my_rho = 0.f;
    long long my_l1 = 0;
    for (int k0 = 0; k0 < nu; k0 += kUK) {
      float mx[kUK];
      uint32_t sa[kUK], sb[kUK];
#pragma unroll
      for (int q = 0; q < kUK; ++q) {
        mx[q] = 0.f;
        sa[q] = sb[q] = 0u;
      }
      const float* rows[kUK];
#pragma unroll
      for (int q = 0; q < kUK; ++q) rows[q] = a.p + (size_t)(base + (k0 + q < nu ? k0 + q : 0)) * a.d;
      uint32_t cnt = 0;
      if (v4) {
        for (int i = lane; i < a.d / 4; i += 32) {
          float4 x[kUK];
#pragma unroll
          for (int q = 0; q < kUK; ++q) x[q] = __ldcs(reinterpret_cast<const float4*>(rows[q]) + i);
#pragma unroll
          for (int q = 0; q < kUK; ++q) {
            fix_add(fabsf(x[q].x), mx[q], sa[q], sb[q]);
            fix_add(fabsf(x[q].y), mx[q], sa[q], sb[q]);
            fix_add(fabsf(x[q].z), mx[q], sa[q], sb[q]);
            fix_add(fabsf(x[q].w), mx[q], sa[q], sb[q]);
          }
          cnt += 4;
        }
      } else {
        for (int i = lane; i < a.d; i += 32) {
          float x[kUK];
#pragma unroll
          for (int q = 0; q < kUK; ++q) x[q] = __ldcs(rows[q] + i);
#pragma unroll
          for (int q = 0; q < kUK; ++q) fix_add(fabsf(x[q]), mx[q], sa[q], sb[q]);
          cnt += 1;
        }
      }
#pragma unroll
      for (int q = 0; q < kUK; ++q) {
        const uint32_t A = sa[q] - cnt * 0x4B000000u, B = sb[q] - cnt * 0x4B000000u;
        long long sum = ((long long)A << 22) + (long long)B;
        const float m = warp_max(mx[q]);
#pragma unroll
        for (int o = 16; o; o >>= 1) sum += __shfl_xor_sync(0xFFFFFFFFu, sum, o);
        if (lane == k0 + q) {
          my_rho = m;
          my_l1 = sum;
        }
      }
    }
    if (lane < nu) {
      const int64_t u = base + lane;
      const float w = weight(__ldg(a.alpha + u), __ldg(a.beta + u), a.gamma);
      unit_hull(my_rho, my_l1, a.d, w, a.k2, a.k3, a.k4, (uint32_t)u, a.w.keys + (size_t)u * kNS,
                a.w.reach + (size_t)u * kNS);
    }
  }
}

__device__ __forceinline__ int step_bits(const uint8_t* r, int s) {
  return c_bits[r[s]] - (s ? c_bits[r[s - 1]] : 0);
}

// Radix pass: bits of the increments in the current bucket, by the digit at `shift`.
// Many increments share a digit (the leading digits hold the efficiency's exponent), so
// the lanes of a warp that hit the same digit add their bits first and one of them
// updates the histogram.
__global__ void k_alloc_hist(AllocWs w, int64_t U, int shift) {
  const AllocState& st = *w.st;
  if (st.all_fit) return;
  const int hs = shift + 16;
  const unsigned long long pre = st.prefix;
  const int lane = threadIdx.x & 31;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  // whole warps walk the units together, so that every lane reaches the shuffles
  for (int64_t u0 = (int64_t)blockIdx.x * blockDim.x + (threadIdx.x & ~31); u0 < U; u0 += stride) {
    const int64_t u = u0 + lane;
    const bool live = u < U;
    const unsigned long long* k = w.keys + (size_t)(live ? u : 0) * kNS;
    const uint8_t* r = w.reach + (size_t)(live ? u : 0) * kNS;
    bool more = live;
#pragma unroll 1
    for (int s = 0; s < kNS; ++s) {
      const unsigned long long key = more ? k[s] : 0ull;
      more = more && key != 0ull;
      const bool take = more && (hs >= 64 || (key >> hs) == (pre >> hs));
      const unsigned act = __ballot_sync(0xFFFFFFFFu, take);
      if (!__any_sync(0xFFFFFFFFu, more)) break;
      if (take) {
        const unsigned dgt = (unsigned)((key >> shift) & 0xFFFFull);
        const unsigned grp = __match_any_sync(act, dgt);
        const unsigned tot = __reduce_add_sync(grp, (unsigned)step_bits(r, s));
        if (lane == __ffs(grp) - 1) atomicAdd(w.hist + dgt, (unsigned long long)tot);
      }
    }
  }
}

// One block: find the largest digit d with above + sum_{d' >= d} hist[d'] > budget.  Two
// levels, every load coalesced: warp w sums its 2048 digits (lane-strided), warp 0 finds
// the warp whose range holds the cut from the suffix sums of the 32 warp totals, then the
// block scans that range's digits in pairs.
__global__ void __launch_bounds__(1024) k_alloc_scan(AllocWs w, long long budget, int shift, int last) {
  constexpr int kPerW = kDigits / 32;
  __shared__ unsigned long long wtot[32];
  __shared__ unsigned long long part[1024];
  __shared__ unsigned long long wabove;
  __shared__ int cutw, found;
  AllocState& st = *w.st;
  const int t = threadIdx.x, lane = t & 31, wid = t >> 5;
  const bool skip = st.all_fit != 0;
  const unsigned long long above = st.above;
  const unsigned long long bud = (unsigned long long)budget;
  {
    const unsigned long long* hw = w.hist + (size_t)wid * kPerW;
    unsigned long long sum = 0;
#pragma unroll 8
    for (int i = 0; i < kPerW / 32; ++i) sum += hw[i * 32 + lane];
#pragma unroll
    for (int o = 16; o; o >>= 1) sum += __shfl_xor_sync(0xFFFFFFFFu, sum, o);
    if (lane == 0) wtot[wid] = sum;
  }
  if (t == 0) {
    cutw = -1;
    found = 0;
  }
  __syncthreads();
  if (wid == 0 && !skip) {
    const unsigned long long mine = wtot[lane];
    unsigned long long sfx = mine;   // sum of the warps at or above this one
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const unsigned long long v = __shfl_down_sync(0xFFFFFFFFu, sfx, o);
      if (lane + o < 32) sfx += v;
    }
    if (above + sfx > bud && above + sfx - mine <= bud) {
      cutw = lane;
      wabove = sfx - mine;
    }
  }
  __syncthreads();
  const int cw = cutw;
  if (cw >= 0) {
    // the cut warp's digits, two per thread (d0 = 2t, d1 = 2t + 1 of its range)
    const unsigned long long* hc = w.hist + (size_t)cw * kPerW;
    const unsigned long long h0 = hc[2 * t], h1 = hc[2 * t + 1];
    part[t] = h0 + h1;
    __syncthreads();
    for (int o = 1; o < 1024; o <<= 1) {   // inclusive suffix scan over the pairs
      const unsigned long long v = t + o < 1024 ? part[t + o] : 0ull;
      __syncthreads();
      part[t] += v;
      __syncthreads();
    }
    const unsigned long long run = above + wabove + (t + 1 < 1024 ? part[t + 1] : 0ull);
    if (run + h0 + h1 > bud && run <= bud) {
      const int d1 = cw * kPerW + 2 * t + 1;
      if (run + h1 > bud) {
        st.prefix |= (unsigned long long)d1 << shift;
        st.above = run;
      } else {
        st.prefix |= (unsigned long long)(d1 - 1) << shift;
        st.above = run + h1;
      }
      found = 1;
    }
  }
  __syncthreads();
  if (t == 0 && !skip) {
    if (!found) {   // only possible in the first pass: every increment fits
      st.all_fit = 1;
      st.kstar = 0ull;
    } else if (last) {
      st.kstar = st.prefix;
    }
  }
  for (int i = t; i < kDigits; i += 1024) w.hist[i] = 0ull;   // ready for the next pass
}

// Step 3 for every unit, and its next increment for the fill.
__global__ void k_alloc_final(AllocWs w, int64_t U, uint8_t* bits) {
  const unsigned long long ks = w.st->kstar;
  unsigned long long used = 0;
  for (int64_t u = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; u < U; u += (int64_t)gridDim.x * blockDim.x) {
    const unsigned long long* k = w.keys + (size_t)u * kNS;
    const uint8_t* r = w.reach + (size_t)u * kNS;
    int t = 0;
    while (t < kNS && k[t] > ks) ++t;
    const int b = t ? c_bits[r[t - 1]] : 0;
    bits[u] = (uint8_t)b;
    used += (unsigned long long)b;
    w.taken[u] = (uint8_t)t;
    const bool more = t < kNS && k[t] != 0ull;
    w.nkey[u] = more ? k[t] : 0ull;
    w.ndb[u] = more ? (uint8_t)step_bits(r, t) : (uint8_t)0;
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) used += __shfl_xor_sync(0xFFFFFFFFu, used, o);
  if ((threadIdx.x & 31) == 0 && used) atomicAdd(&w.st->used, used);
}

__global__ void k_fill_init(AllocWs w, long long budget) {
  AllocState& st = *w.st;
  st.left = budget - (long long)st.used;
  st.best = 0ull;
  st.fill_done = 0;
}

__global__ void k_fill_max(AllocWs w, int64_t U) {
  const AllocState& st = *w.st;
  if (st.fill_done) return;
  const long long left = st.left;
  unsigned long long best = 0ull;
  for (int64_t u = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; u < U; u += (int64_t)gridDim.x * blockDim.x) {
    const unsigned long long k = w.nkey[u];
    if (k > best && (long long)w.ndb[u] <= left) best = k;
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) {
    const unsigned long long v = __shfl_xor_sync(0xFFFFFFFFu, best, o);
    best = v > best ? v : best;
  }
  if ((threadIdx.x & 31) == 0 && best) atomicMax(&w.st->best, best);
}

__global__ void k_fill_take(AllocWs w, int64_t U, uint8_t* bits) {
  AllocState& st = *w.st;
  if (st.fill_done) return;
  const unsigned long long k = st.best;
  if (!k) {
    st.fill_done = 1;
    return;
  }
  const int64_t u = (int64_t)(0xFFFFFFFFull - (k & 0xFFFFFFFFull));
  if (u < 0 || u >= U) {   // cannot happen: keys carry their unit
    st.fill_done = 1;
    return;
  }
  const uint8_t* r = w.reach + (size_t)u * kNS;
  const unsigned long long* ks = w.keys + (size_t)u * kNS;
  const int t = w.taken[u];
  st.left -= (long long)w.ndb[u];
  bits[u] = (uint8_t)c_bits[r[t]];
  w.taken[u] = (uint8_t)(t + 1);
  const bool more = t + 1 < kNS && ks[t + 1] != 0ull;
  w.nkey[u] = more ? ks[t + 1] : 0ull;
  w.ndb[u] = more ? (uint8_t)step_bits(r, t + 1) : (uint8_t)0;
  st.best = 0ull;
}

int sms_of_current(int* sms) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(sms, cudaDevAttrMultiProcessorCount, dev);
  return e == cudaSuccess ? BITSMOE_OK : bmoe::record_cuda_error((int)e);
}

int allocate_impl(const float* p, const float* alpha, const float* beta, float gamma, int64_t U, int d,
                  const float* kappa, int64_t budget, uint8_t* bits, void* ws, size_t ws_bytes, cudaStream_t st,
                  float* phase_ms) {
  if (U < 0 || d < 1 || budget < 0 || !(gamma >= 0.f && gamma <= 1.f)) return BITSMOE_ERR_INVALID_ARG;
  if (U > 0xFFFFFFFEll || d > 16384) return BITSMOE_ERR_SHAPE;
  if (U == 0) return BITSMOE_OK;
  if (!p || !alpha || !beta || !kappa || !bits || !ws) return BITSMOE_ERR_INVALID_ARG;
  if ((uintptr_t)p % 16 || (uintptr_t)alpha % 4 || (uintptr_t)beta % 4 || (uintptr_t)ws % 256)
    return BITSMOE_ERR_ALIGNMENT;
  size_t off[7];
  if (ws_bytes < ws_layout(U, off)) return BITSMOE_ERR_WORKSPACE_TOO_SMALL;
  int sms = 0;
  int rc = sms_of_current(&sms);
  if (rc) return rc;
  uint8_t* wb = static_cast<uint8_t*>(ws);
  AllocWs w{reinterpret_cast<AllocState*>(wb + off[0]), reinterpret_cast<unsigned long long*>(wb + off[1]),
            reinterpret_cast<unsigned long long*>(wb + off[2]), wb + off[3], wb + off[4],
            reinterpret_cast<unsigned long long*>(wb + off[5]), wb + off[6]};
  cudaEvent_t ev[4] = {};
  if (phase_ms) {
    for (auto& e : ev)
      if (cudaEventCreate(&e) != cudaSuccess) return bmoe::record_cuda_error((int)cudaGetLastError());
  }
  auto fail = [&](cudaError_t e) {
    if (phase_ms)
      for (auto& x : ev) cudaEventDestroy(x);
    return bmoe::record_cuda_error((int)e);
  };
  cudaError_t e = cudaMemsetAsync(wb + off[0], 0, off[2], st);   // state and histogram
  if (e != cudaSuccess) return fail(e);
  if (phase_ms) cudaEventRecord(ev[0], st);
  CostArgs ca{p, alpha, beta, gamma, kappa[0], kappa[1], kappa[2], U, d, w};
  int per_sm = 0;
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_alloc_cost, kAW * 32, 0);
  if (e != cudaSuccess) return fail(e);
  const int64_t groups = (U + 31) / 32;
  const int64_t cost_blocks = std::min<int64_t>((groups + kAW - 1) / kAW, (int64_t)sms * std::max(per_sm, 1));
  k_alloc_cost<<<(unsigned)cost_blocks, kAW * 32, 0, st>>>(ca);
  if (phase_ms) cudaEventRecord(ev[1], st);
  const unsigned ub = (unsigned)std::min<int64_t>((U + 255) / 256, (int64_t)sms * 8);
  for (int pass = 0; pass < 4; ++pass) {
    const int shift = 48 - 16 * pass;
    k_alloc_hist<<<ub, 256, 0, st>>>(w, U, shift);
    k_alloc_scan<<<1, 1024, 0, st>>>(w, (long long)budget, shift, pass == 3);
  }
  k_alloc_final<<<ub, 256, 0, st>>>(w, U, bits);
  if (phase_ms) cudaEventRecord(ev[2], st);
  k_fill_init<<<1, 1, 0, st>>>(w, (long long)budget);
  for (int r = 0; r < kFillRounds; ++r) {
    k_fill_max<<<ub, 256, 0, st>>>(w, U);
    k_fill_take<<<1, 1, 0, st>>>(w, U, bits);
  }
  e = cudaGetLastError();
  if (e != cudaSuccess) return fail(e);
  if (phase_ms) {
    cudaEventRecord(ev[3], st);
    e = cudaEventSynchronize(ev[3]);
    if (e != cudaSuccess) return fail(e);
    for (int i = 0; i < 3; ++i) cudaEventElapsedTime(&phase_ms[i], ev[i], ev[i + 1]);
    for (auto& x : ev) cudaEventDestroy(x);
  }
  return BITSMOE_OK;
}

}  // namespace

extern "C" int bitsmoe_projection_budget(int64_t E, int64_t n, int64_t m, int64_t beq_num, int64_t beq_den,
                                         int64_t* out) {
  // floor(E n b_eq - 16 n^2 / m), b_eq = num / den, in exact int64 arithmetic
  if (!out || E < 1 || n < 1 || m < 1 || beq_den < 1 || beq_num < 0) return BITSMOE_ERR_INVALID_ARG;
  if (E > (1 << 20) || n > (1 << 20) || m > (1 << 24) || beq_num > (1 << 16) || beq_den > (1 << 16))
    return BITSMOE_ERR_SHAPE;
  // a / den - b / m with a = E n num (< 2^56), b = 16 n^2 (< 2^45): whole parts q1 - q2, and
  // the fractional parts r1 / den - r2 / m in (-1, 1) take one more off when negative
  // (r1 m and r2 den stay below 2^40)
  const int64_t a = E * n * beq_num, b = 16 * n * n;
  const int64_t q1 = a / beq_den, r1 = a % beq_den, q2 = b / m, r2 = b % m;
  *out = q1 - q2 - (r1 * m < r2 * beq_den ? 1 : 0);
  return BITSMOE_OK;
}

extern "C" size_t bitsmoe_allocate_workspace_bytes(int64_t U) {
  if (U < 0 || U > 0xFFFFFFFEll) return 0;
  size_t off[7];
  return ws_layout(U, off);
}

extern "C" int bitsmoe_allocate_bits(const float* p, const float* alpha, const float* beta, float gamma, int64_t U,
                                     int d, const float* kappa, int64_t budget, uint8_t* bits, void* ws,
                                     size_t ws_bytes, void* stream) {
  return allocate_impl(p, alpha, beta, gamma, U, d, kappa, budget, bits, ws, ws_bytes,
                       static_cast<cudaStream_t>(stream), nullptr);
}

extern "C" int bitsmoe_profile_allocate_bits(const float* p, const float* alpha, const float* beta, float gamma,
                                             int64_t U, int d, const float* kappa, int64_t budget, uint8_t* bits,
                                             void* ws, size_t ws_bytes, void* stream, float phase_ms[3]) {
  if (!phase_ms) return BITSMOE_ERR_INVALID_ARG;
  return allocate_impl(p, alpha, beta, gamma, U, d, kappa, budget, bits, ws, ws_bytes,
                       static_cast<cudaStream_t>(stream), phase_ms);
}
