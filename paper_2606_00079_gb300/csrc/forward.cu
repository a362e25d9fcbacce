// BitsMoE quantized MoE-layer forward on sm_103a (GB300).
//
// Stage 3 of the method (Fig. 1; "Inference Efficiency", Sec. Experiments):
// the activation is projected once onto the shared bases, then each routed
// expert's packed spectral factors are unpacked and applied inside the kernels
// without rebuilding the expert weights.  Phases, one kernel each, chained on
// the caller's stream with programmatic dependent launch (PDL) so that a
// kernel's prologue overlaps the tail of the previous one:
//
//   K0 k_router     top-k over the logits, softmax over the selected k, and
//                   token -> expert grouping (counts, offsets, pair lists)
//   K1 k_gemv<P>    z_g = Phi_g^T x, z_u = Phi_u^T x (bf16 rows streamed with
//                   128-bit loads); zeroes the accumulators; then prefetches
//                   the routed experts' packed factors and Phi_dn into L2
//   K2 k_gateup     gate/up = P_hat (alpha * z): mixed-bit dequant-GEMV over
//                   bucketed uniform-bit streams; in-register unpacking and
//                   dp2a integer dot products (int16 activation operand),
//                   fp32 partials reduced with vector red.add
//   K3 k_down       h = SiLU(gate) * up (fused into the prologue), then
//                   s += w_e * alpha_dn * (P_hat_dn^T h) per unit
//   K4 k_gemv<O>    y = Phi_dn s (fp32 out)
//
// The identity behind the association is Eq. app_normalized_decomposition
// (W = P A Phi^T for gate/up, W = Phi A P^T for down); summing the experts'
// n-dim spectral vectors before Phi_dn is exact by linearity.
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <cstring>
#include <functional>
#include <mutex>
#include <vector>

#include "internal.h"

using namespace bmoe;

struct bitsmoe_layer {
  int device;
  int num_sms;
  uint8_t* d_img;
  uint64_t bytes;
  std::vector<uint8_t> meta;   // host copy of header + descriptors + segment table
  const ImageHeader& hd() const { return *reinterpret_cast<const ImageHeader*>(meta.data()); }
  const ExpertDesc* desc() const {
    return reinterpret_cast<const ExpertDesc*>(meta.data() + hd().off_desc);
  }
};

namespace {

thread_local int g_last_cuda = 0;
int cuda_fail(cudaError_t e) {
  g_last_cuda = (int)e;
  return BITSMOE_ERR_CUDA;
}
#define BM_CK(call)                               \
  do {                                            \
    cudaError_t e_ = (call);                      \
    if (e_ != cudaSuccess) return cuda_fail(e_);  \
  } while (0)

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kK3Tiles = kWarps;     // UL tiles per K3 block (one per warp)
constexpr int kK3MaxRB = 8;          // row blocks per K3 block
constexpr uint32_t kPrefetchPiece = 16384;
constexpr uint64_t kPrefetchCap = 96ull << 20;

struct Fwd {
  const uint8_t* img;
  const ExpertDesc* desc;
  const int32_t* seg;
  const uint16_t* basis_in;
  const uint16_t* basis_out;
  int D, E, I, n, group, D_pad, n_pad, I_pad, NRB, NG, nseg, ul_max_tiles;
  int T, k, P;
  int s16;          // K2 smem row stride (int16 elements)
  int rbc;          // K3 row blocks per block
  const uint16_t* x;
  const float* logits;
  float* y;
  int* status;
  int* pair_expert;
  float* pair_weight;
  int* expert_count;
  int* expert_start;
  int* pair_list;
  int* active;      // [0] = number of routed experts, [1 + a] = expert id
  float* z;         // [2][T][n_pad]
  float* gu;        // [P][2][I_pad]
  float* s;         // [T][n_pad]
};

// ---------------------------------------------------------------------------
// PTX helpers
// ---------------------------------------------------------------------------
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

__device__ __forceinline__ uint4 ldg_stream(const void* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}
__device__ __forceinline__ void prefetch_l2(const void* p, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}
// a: two signed 16-bit values, b: four unsigned bytes (low or high pair used)
__device__ __forceinline__ int dp2a_lo(int a, uint32_t b, int c) {
  int d;
  asm("dp2a.lo.s32.u32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
  return d;
}
__device__ __forceinline__ int dp2a_hi(int a, uint32_t b, int c) {
  int d;
  asm("dp2a.hi.s32.u32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
  return d;
}
__device__ __forceinline__ void red_add_v4(float* addr, float a, float b, float c, float d) {
  asm volatile("red.global.add.v4.f32 [%0], {%1,%2,%3,%4};" ::"l"(addr), "f"(a), "f"(b), "f"(c), "f"(d)
               : "memory");
}
__device__ __forceinline__ float bf16lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }
__device__ __forceinline__ float f16lo(uint32_t w) {
  return __half2float(__ushort_as_half((unsigned short)(w & 0xFFFFu)));
}
__device__ __forceinline__ float f16hi(uint32_t w) {
  return __half2float(__ushort_as_half((unsigned short)(w >> 16)));
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xFFFFFFFFu, v, o));
  return v;
}
// total order on floats for top-k: larger float -> larger key; NaN below everything
__device__ __forceinline__ uint32_t order_key(float f) {
  const uint32_t u = __float_as_uint(f);
  if ((u & 0x7FFFFFFFu) > 0x7F800000u) return 0u;
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// ---------------------------------------------------------------------------
// K0: routing.  k largest logits per token (ties to the lower expert index),
// gate weights = softmax over the selected k, then a stable grouping of the
// (token, slot) pairs p = t * k + slot by expert.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(1024) k_router(Fwd p) {
  pdl_trigger();
  extern __shared__ uint32_t keys[];
  const int E = p.E, k = p.k, T = p.T, P = p.P;
  const int tid = threadIdx.x;
  if (tid == 0) *p.status = 0;
  const int tpb = max(1, (int)blockDim.x / E);
  for (int t0 = 0; t0 < T; t0 += tpb) {
    const int tt = tid / E, e = tid - tt * E, t = t0 + tt;
    const bool valid = tt < tpb && t < T;
    if (valid) keys[tt * E + e] = order_key(p.logits[(size_t)t * E + e]);
    __syncthreads();
    if (valid) {
      const uint32_t key = keys[tt * E + e];
      const uint32_t* row = keys + tt * E;
      int rank = 0;
      for (int f = 0; f < E; ++f) {
        const uint32_t o = row[f];
        rank += (o > key) | ((o == key) & (f < e));
      }
      if (rank < k) {
        p.pair_expert[t * k + rank] = e;
        p.pair_weight[t * k + rank] = p.logits[(size_t)t * E + e];
      }
    }
    __syncthreads();
  }
  for (int t = tid; t < T; t += blockDim.x) {
    float* w = p.pair_weight + (size_t)t * k;
    const float m = w[0];
    float sum = 0.f;
    for (int r = 0; r < k; ++r) sum += expf(w[r] - m);
    const float inv = 1.f / sum;
    for (int r = 0; r < k; ++r) w[r] = expf(w[r] - m) * inv;
  }
  __syncthreads();
  const int warp = tid >> 5, lane = tid & 31, nw = blockDim.x >> 5;
  for (int e = warp; e < E; e += nw) {
    int c = 0;
    for (int q0 = 0; q0 < P; q0 += 32) {
      const int q = q0 + lane;
      c += __popc(__ballot_sync(0xFFFFFFFFu, q < P && p.pair_expert[q] == e));
    }
    if (lane == 0) p.expert_count[e] = c;
  }
  __syncthreads();
  if (warp == 0) {
    int run = 0, act = 0;
    for (int e0 = 0; e0 < E; e0 += 32) {
      const int e = e0 + lane;
      const int c = e < E ? p.expert_count[e] : 0;
      int incl = c;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int v = __shfl_up_sync(0xFFFFFFFFu, incl, o);
        if (lane >= o) incl += v;
      }
      if (e < E) p.expert_start[e] = run + incl - c;
      const unsigned nz = __ballot_sync(0xFFFFFFFFu, c > 0);
      if (c > 0) p.active[1 + act + __popc(nz & ((1u << lane) - 1u))] = e;
      act += __popc(nz);
      run += __shfl_sync(0xFFFFFFFFu, incl, 31);
    }
    if (lane == 0) {
      p.expert_start[E] = run;
      p.active[0] = act;
    }
  }
  __syncthreads();
  for (int e = warp; e < E; e += nw) {
    int base = p.expert_start[e];
    for (int q0 = 0; q0 < P; q0 += 32) {
      const int q = q0 + lane;
      const bool m = q < P && p.pair_expert[q] == e;
      const unsigned b = __ballot_sync(0xFFFFFFFFu, m);
      if (m) p.pair_list[base + __popc(b & ((1u << lane) - 1u))] = q;
      base += __popc(b);
    }
  }
}

// ---------------------------------------------------------------------------
// L2 prefetch of what the later phases read: gate/up then down factors of the
// routed experts, then Phi_dn (warp 0 of every block, 16 KB pieces).
// ---------------------------------------------------------------------------
__device__ void prefetch_for_experts(const Fwd& p) {
  if (threadIdx.x >= 32) return;
  const int lane = threadIdx.x;
  const int A = p.active[0];
  const uint64_t slots = (uint64_t)gridDim.x * 32, me = (uint64_t)blockIdx.x * 32 + lane;
  uint64_t gi = 0, budget = kPrefetchCap;
  auto range = [&](uint64_t beg, uint64_t end) {
    if (end > beg + budget) end = beg + budget;
    budget -= end - beg;
    for (uint64_t o = beg; o < end; o += kPrefetchPiece, ++gi)
      if (gi % slots == me)
        prefetch_l2(p.img + o, (uint32_t)(end - o < kPrefetchPiece ? end - o : kPrefetchPiece));
  };
  for (int h = 0; h < 3 && budget; ++h)
    for (int a = 0; a < A && budget; ++a) {
      const ExpertDesc& xd = p.desc[h * p.E + p.active[1 + a]];
      range(xd.begin, xd.end);
    }
  const uint64_t bo = (uint64_t)((const uint8_t*)p.basis_out - p.img);
  if (budget) range(bo, bo + (uint64_t)p.D * p.n_pad * 2);
}

// ---------------------------------------------------------------------------
// K1 / K4: bf16 matrix rows x fp32 vectors.  PROJ: rows = [Phi_g^T; Phi_u^T]
// (2n rows of D_pad), vectors = x -> z.  !PROJ: rows = Phi_dn (D rows of
// n_pad), vectors = s -> y.  One warp per row, 128-bit streaming loads, the
// vectors staged in shared memory as fp32.
// ---------------------------------------------------------------------------
template <int TB, bool PROJ>
__global__ void __launch_bounds__(kThreads) k_gemv(Fwd p) {
  pdl_trigger();
  extern __shared__ float4 smem4[];
  float* vs = reinterpret_cast<float*>(smem4);
  const int ld = PROJ ? p.D_pad : p.n_pad;
  const int nrows = PROJ ? 2 * p.n : p.D;
  const int nch = ld >> 3;
  const uint16_t* mat = PROJ ? p.basis_in : p.basis_out;
  const int lane = threadIdx.x & 31;
  const int gw = blockIdx.x * kWarps + (threadIdx.x >> 5);
  const int nwt = gridDim.x * kWarps;
  if (PROJ) {
    const size_t ng = (size_t)p.P * 2 * p.I_pad / 4, ns = (size_t)p.T * p.n_pad / 4;
    const float4 z4 = make_float4(0.f, 0.f, 0.f, 0.f);
    for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < ng + ns;
         i += (size_t)gridDim.x * blockDim.x) {
      if (i < ng) reinterpret_cast<float4*>(p.gu)[i] = z4;
      else reinterpret_cast<float4*>(p.s)[i - ng] = z4;
    }
  } else {
    pdl_wait();
  }
  for (int t0 = 0; t0 < p.T; t0 += TB) {
    const int tb = min(TB, p.T - t0);
    __syncthreads();
    for (int i = threadIdx.x; i < TB * ld; i += blockDim.x) {
      const int tt = i / ld, c = i - tt * ld;
      float v = 0.f;
      if (tt < tb) {
        if (PROJ) {
          if (c < p.D) v = __uint_as_float((uint32_t)p.x[(size_t)(t0 + tt) * p.D + c] << 16);
        } else {
          if (c < p.n) v = p.s[(size_t)(t0 + tt) * p.n_pad + c];
        }
      }
      vs[i] = v;
    }
    __syncthreads();
    for (int row = gw; row < nrows; row += nwt) {
      const uint4* rp = reinterpret_cast<const uint4*>(mat + (size_t)row * ld);
      float acc[TB];
#pragma unroll
      for (int tt = 0; tt < TB; ++tt) acc[tt] = 0.f;
      for (int c0 = 0; c0 < nch; c0 += 32 * 8) {
        uint4 v[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const int c = c0 + u * 32 + lane;
          v[u] = c < nch ? ldg_stream(rp + c) : make_uint4(0, 0, 0, 0);
        }
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const int c = c0 + u * 32 + lane;
          if (c < nch) {
            const float w0 = bf16lo(v[u].x), w1 = bf16hi(v[u].x), w2 = bf16lo(v[u].y), w3 = bf16hi(v[u].y);
            const float w4 = bf16lo(v[u].z), w5 = bf16hi(v[u].z), w6 = bf16lo(v[u].w), w7 = bf16hi(v[u].w);
#pragma unroll
            for (int tt = 0; tt < TB; ++tt) {
              const float4* xv = reinterpret_cast<const float4*>(vs + tt * ld + c * 8);
              const float4 a = xv[0], b = xv[1];
              float r = acc[tt];
              r = fmaf(w0, a.x, r); r = fmaf(w1, a.y, r); r = fmaf(w2, a.z, r); r = fmaf(w3, a.w, r);
              r = fmaf(w4, b.x, r); r = fmaf(w5, b.y, r); r = fmaf(w6, b.z, r); r = fmaf(w7, b.w, r);
              acc[tt] = r;
            }
          }
        }
      }
#pragma unroll
      for (int tt = 0; tt < TB; ++tt) acc[tt] = warp_sum(acc[tt]);
      if (lane == 0) {
#pragma unroll
        for (int tt = 0; tt < TB; ++tt) {
          if (tt < tb) {
            const int t = t0 + tt;
            if (PROJ) {
              const int h = row >= p.n, j = row - h * p.n;
              p.z[((size_t)h * p.T + t) * p.n_pad + j] = acc[tt];
            } else {
              p.y[(size_t)t * p.D + row] = acc[tt];
            }
          }
        }
      }
    }
  }
  if (PROJ) {
    pdl_wait();
    prefetch_for_experts(p);
  }
}

// ---------------------------------------------------------------------------
// K2: gate/up factors.  out[i] = sum_j alpha_j z_j p_hat_ij
//                             = sum_j c_jg (q_ij - zero_jg),  c_jg = alpha_j z_j s_jg
// A warp item is (routed expert, projection, 128-row block, segment of tiles).
// The lane owns 4 rows; c of the segment's units is quantised to int16 with
// one scale per (item, token), so the inner loop is dp2a over unpacked code
// bytes; the zero-point term sum_j c_jg zero_jg is applied once per item.
// ---------------------------------------------------------------------------
struct Range {
  int bi;     // bucket index in the expert descriptor
  int lo, hi; // bucket-local tile range
  int ls0;    // local slot base of this range in the item's c table
};

template <int PB, int TB>
__device__ __forceinline__ void rl_dp(const uint4& v, const int* cp, int tstride, int (&acc)[4][TB]) {
  constexpr int NK = 8 / PB;
  constexpr uint32_t MASK = ((1u << PB) - 1u) * 0x01010101u;
  int c[TB][2 * NK];
#pragma unroll
  for (int tt = 0; tt < TB; ++tt)
#pragma unroll
    for (int q = 0; q < 2 * NK; ++q) c[tt][q] = cp[tt * tstride + q];
  const uint32_t wv[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int w = 0; w < 4; ++w)
#pragma unroll
    for (int kq = 0; kq < NK; ++kq) {
      const uint32_t bytes = (wv[w] >> (PB * kq)) & MASK;
#pragma unroll
      for (int tt = 0; tt < TB; ++tt) {
        acc[w][tt] = dp2a_lo(c[tt][2 * kq], bytes, acc[w][tt]);
        acc[w][tt] = dp2a_hi(c[tt][2 * kq + 1], bytes, acc[w][tt]);
      }
    }
}

template <int B, int TB>
__device__ __forceinline__ void rl_range(const uint8_t* code, int ntl, const int* cq32, int tstride,
                                         float (&accf)[4][TB]) {
  constexpr int U = rl_units(B), C = rl_chunks(B);
  int acc[4][TB], acch[4][TB];
#pragma unroll
  for (int w = 0; w < 4; ++w)
#pragma unroll
    for (int tt = 0; tt < TB; ++tt) acc[w][tt] = acch[w][tt] = 0;
  int since = 0;
  for (int t = 0; t < ntl; ++t) {
    uint4 v[C];
#pragma unroll
    for (int c = 0; c < C; ++c) v[c] = ldg_stream(code + (size_t)(t * C + c) * kChunkBytes);
    const int* cp = cq32 + t * (U / 2);
    if (B == 3) {
      rl_dp<2, TB>(v[0], cp, tstride, acc);
      rl_dp<2, TB>(v[1], cp + 8, tstride, acc);
      rl_dp<1, TB>(v[2], cp, tstride, acch);
    } else if (B == 6) {
      rl_dp<4, TB>(v[0], cp, tstride, acc);
      rl_dp<4, TB>(v[1], cp + 4, tstride, acc);
      rl_dp<2, TB>(v[2], cp, tstride, acch);
    } else {
      rl_dp<B, TB>(v[0], cp, tstride, acc);
    }
    if (++since == 32 || t == ntl - 1) {
      since = 0;
#pragma unroll
      for (int w = 0; w < 4; ++w)
#pragma unroll
        for (int tt = 0; tt < TB; ++tt) {
          const int hi_shift = B == 3 ? 2 : 4;
          const int tot = (B == 3 || B == 6) ? acc[w][tt] + (acch[w][tt] << hi_shift) : acc[w][tt];
          accf[w][tt] += (float)tot;
          acc[w][tt] = acch[w][tt] = 0;
        }
    }
  }
}

template <int TB>
__device__ __forceinline__ void rl_range16(const uint8_t* code, int ntl, const int32_t* unit, const float* alpha,
                                           const float* const (&zrow)[TB], float (&acc16)[4][TB]) {
  for (int t = 0; t < ntl; ++t) {
    const uint4 v = ldg_stream(code + (size_t)t * kChunkBytes);
    const int j0 = unit[2 * t], j1 = unit[2 * t + 1];
    const float a0 = alpha[2 * t], a1 = alpha[2 * t + 1];
    const uint32_t wv[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int tt = 0; tt < TB; ++tt) {
      const float c0 = a0 * zrow[tt][j0], c1 = a1 * zrow[tt][j1];
#pragma unroll
      for (int w = 0; w < 4; ++w) acc16[w][tt] = fmaf(c0, f16lo(wv[w]), fmaf(c1, f16hi(wv[w]), acc16[w][tt]));
    }
  }
}

template <int G, int TB>
__global__ void __launch_bounds__(kThreads) k_gateup(Fwd p) {
  pdl_trigger();
  pdl_wait();
  extern __shared__ int4 smem_k2[];
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  int16_t* cq = reinterpret_cast<int16_t*>(smem_k2) + (size_t)wid * G * TB * p.s16;
  const int A = p.active[0];
  const int per_e = 2 * p.NRB * p.nseg;
  const int total = A * per_e;
  const int gl_lane = G == 1 ? 0 : (4 * lane) / p.group;   // lane's group inside the row block
  for (int item = blockIdx.x * kWarps + wid; item < total; item += gridDim.x * kWarps) {
    const int a = item / per_e;
    int r = item - a * per_e;
    const int h = r / (p.NRB * p.nseg);
    r -= h * p.NRB * p.nseg;
    const int rb = r / p.nseg, sg = r - rb * p.nseg;
    const int e = p.active[1 + a];
    const int32_t* segp = p.seg + ((size_t)h * p.E + e) * (p.nseg + 1);
    const int t0 = segp[sg], t1 = segp[sg + 1];
    if (t0 >= t1) continue;
    const ExpertDesc& xd = p.desc[h * p.E + e];
    const int32_t* unit = reinterpret_cast<const int32_t*>(p.img + xd.unit_off);
    const float* alpha = reinterpret_cast<const float*>(p.img + xd.alpha_off);
    // tile ranges of this item, per bucket
    Range rg[kNumBk];
    int nr = 0, nls = 0;
    for (int bi = 0; bi < xd.nbk; ++bi) {
      const BucketDesc& bd = xd.bk[bi];
      const int lo = max(t0, bd.tile0) - bd.tile0, hi = min(t1, bd.tile0 + bd.ntiles) - bd.tile0;
      if (lo < hi) {
        rg[nr] = Range{bi, lo, hi, nls};
        if (bd.bits < 16) nls += (hi - lo) * rl_units(bd.bits);
        ++nr;
      }
    }
    const int g_base = (rb * kRows) / p.group;
    const int ntok = p.expert_count[e], pst = p.expert_start[e];
    for (int tb0 = 0; tb0 < ntok; tb0 += TB) {
      const int tb = min(TB, ntok - tb0);
      int pair[TB];
      const float* zrow[TB];
#pragma unroll
      for (int tt = 0; tt < TB; ++tt) {
        pair[tt] = p.pair_list[pst + tb0 + min(tt, tb - 1)];
        zrow[tt] = p.z + ((size_t)h * p.T + pair[tt] / p.k) * p.n_pad;
      }
      // pass 1: max |c| per token over the item's quantised units
      float mx[TB];
#pragma unroll
      for (int tt = 0; tt < TB; ++tt) mx[tt] = 0.f;
      for (int ri = 0; ri < nr; ++ri) {
        const BucketDesc& bd = xd.bk[rg[ri].bi];
        if (bd.bits == 16) continue;
        const int U = rl_units(bd.bits), s0 = rg[ri].lo * U, ns = (rg[ri].hi - rg[ri].lo) * U;
        const uint32_t* sz = reinterpret_cast<const uint32_t*>(p.img + bd.sz_off);
        for (int i = lane; i < ns; i += 32) {
          const int bs = s0 + i, gs = bd.slot0 + bs;
          const int j = unit[gs];
          const float al = alpha[gs];
#pragma unroll
          for (int gl = 0; gl < G; ++gl) {
            const float sc = __half2float(__ushort_as_half((unsigned short)(sz[(size_t)(g_base + gl) * bd.nslots + bs] & 0xFFFFu)));
#pragma unroll
            for (int tt = 0; tt < TB; ++tt) mx[tt] = fmaxf(mx[tt], fabsf(al * sc * zrow[tt][j]));
          }
        }
      }
      float inv[TB], scl[TB];
#pragma unroll
      for (int tt = 0; tt < TB; ++tt) {
        mx[tt] = warp_max(mx[tt]);
        inv[tt] = mx[tt] > 0.f ? 32767.f / mx[tt] : 0.f;
        scl[tt] = mx[tt] * (1.f / 32767.f);
      }
      // pass 2: quantise into shared memory, zero-point correction per group
      float corr[G][TB];
#pragma unroll
      for (int gl = 0; gl < G; ++gl)
#pragma unroll
        for (int tt = 0; tt < TB; ++tt) corr[gl][tt] = 0.f;
      for (int ri = 0; ri < nr; ++ri) {
        const BucketDesc& bd = xd.bk[rg[ri].bi];
        if (bd.bits == 16) continue;
        const int U = rl_units(bd.bits), s0 = rg[ri].lo * U, ns = (rg[ri].hi - rg[ri].lo) * U;
        const uint32_t* sz = reinterpret_cast<const uint32_t*>(p.img + bd.sz_off);
        for (int i = lane; i < ns; i += 32) {
          const int bs = s0 + i, gs = bd.slot0 + bs;
          const int j = unit[gs];
          const float al = alpha[gs];
#pragma unroll
          for (int gl = 0; gl < G; ++gl) {
            const uint32_t szw = sz[(size_t)(g_base + gl) * bd.nslots + bs];
            const float sc = __half2float(__ushort_as_half((unsigned short)(szw & 0xFFFFu)));
            const float zp = __half2float(__ushort_as_half((unsigned short)(szw >> 16)));
#pragma unroll
            for (int tt = 0; tt < TB; ++tt) {
              const int ci = __float2int_rn(al * sc * zrow[tt][j] * inv[tt]);
              cq[(size_t)(gl * TB + tt) * p.s16 + rg[ri].ls0 + i] = (int16_t)ci;
              corr[gl][tt] = fmaf((float)ci, zp, corr[gl][tt]);
            }
          }
        }
      }
#pragma unroll
      for (int gl = 0; gl < G; ++gl)
#pragma unroll
        for (int tt = 0; tt < TB; ++tt) corr[gl][tt] = warp_sum(corr[gl][tt]);
      __syncwarp();
      // main loop over the item's tiles
      float accf[4][TB], acc16[4][TB];
#pragma unroll
      for (int w = 0; w < 4; ++w)
#pragma unroll
        for (int tt = 0; tt < TB; ++tt) accf[w][tt] = acc16[w][tt] = 0.f;
      const int* cq32 = reinterpret_cast<const int*>(cq + (size_t)gl_lane * TB * p.s16);
      const int tstride = p.s16 / 2;
      for (int ri = 0; ri < nr; ++ri) {
        const BucketDesc& bd = xd.bk[rg[ri].bi];
        const int ntl = rg[ri].hi - rg[ri].lo;
        const uint8_t* code = p.img + xd.code_base + (size_t)rb * xd.rb_stride + bd.code_off +
                              (size_t)rg[ri].lo * rl_chunks(bd.bits) * kChunkBytes + lane * 16;
        const int* cp = cq32 + rg[ri].ls0 / 2;
        switch (bd.bits) {
          case 1: rl_range<1, TB>(code, ntl, cp, tstride, accf); break;
          case 2: rl_range<2, TB>(code, ntl, cp, tstride, accf); break;
          case 3: rl_range<3, TB>(code, ntl, cp, tstride, accf); break;
          case 4: rl_range<4, TB>(code, ntl, cp, tstride, accf); break;
          case 6: rl_range<6, TB>(code, ntl, cp, tstride, accf); break;
          case 8: rl_range<8, TB>(code, ntl, cp, tstride, accf); break;
          default: {
            const int gs0 = bd.slot0 + rg[ri].lo * 2;
            rl_range16<TB>(code, ntl, unit + gs0, alpha + gs0, zrow, acc16);
          }
        }
      }
      // write partial sums of the lane's 4 rows
      const int row = rb * kRows + 4 * lane;
#pragma unroll
      for (int tt = 0; tt < TB; ++tt) {
        if (tt < tb) {
          float cl = corr[0][tt];
#pragma unroll
          for (int gl = 1; gl < G; ++gl)
            if (gl == gl_lane) cl = corr[gl][tt];
          float o[4];
#pragma unroll
          for (int w = 0; w < 4; ++w) o[w] = fmaf(scl[tt], accf[w][tt] - cl, acc16[w][tt]);
          red_add_v4(p.gu + ((size_t)pair[tt] * 2 + h) * p.I_pad + row, o[0], o[1], o[2], o[3]);
        }
      }
      __syncwarp();
    }
  }
}

// ---------------------------------------------------------------------------
// K3: down factor.  h = SiLU(gate) * up for the block's rows (quantised to
// int16 with one scale per token), then per unit j (one per lane):
//   d_j = sum_g s_jg (sum_{i in g} q_ij h_i - zero_jg * sum_{i in g} h_i)
//   s[t][j] += w_(t,e) * alpha_j * d_j
// A block item is (routed expert, 8 UL tiles, up to 8 row blocks).
// ---------------------------------------------------------------------------
template <int PB, int TB>
__device__ __forceinline__ void ul_dp(uint32_t word, const int* hp, int tstride, int (&acc)[TB]) {
  constexpr int NK = 8 / PB;
  constexpr uint32_t MASK = ((1u << PB) - 1u) * 0x01010101u;
#pragma unroll
  for (int kq = 0; kq < NK; ++kq) {
    const uint32_t bytes = (word >> (PB * kq)) & MASK;
#pragma unroll
    for (int tt = 0; tt < TB; ++tt) {
      acc[tt] = dp2a_lo(hp[tt * tstride + 2 * kq], bytes, acc[tt]);
      acc[tt] = dp2a_hi(hp[tt * tstride + 2 * kq + 1], bytes, acc[tt]);
    }
  }
}

// One plane chunk (16 bytes) of a UL lane: rows rbase + w * (32 / PB) + r'
template <int PB, int G, int TB>
__device__ __forceinline__ void ul_chunk(const uint4& v, int rbase, const int* hq32, int tstride, int gshift,
                                         int (&acc)[G][TB]) {
  constexpr int RPW = 32 / PB;
  const uint32_t wv[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int w = 0; w < 4; ++w) {
    const int r0 = rbase + w * RPW;
    int tmp[TB];
#pragma unroll
    for (int tt = 0; tt < TB; ++tt) tmp[tt] = 0;
    ul_dp<PB, TB>(wv[w], hq32 + r0 / 2, tstride, tmp);
    const int gl = G == 1 ? 0 : (r0 >> gshift);
#pragma unroll
    for (int g = 0; g < G; ++g)
      if (g == gl)
#pragma unroll
        for (int tt = 0; tt < TB; ++tt) acc[g][tt] += tmp[tt];
  }
}

template <int B, int G, int TB>
__device__ __forceinline__ void ul_tile(const Fwd& p, const uint8_t* code, int rb0, int rb1, const int16_t* hq,
                                        int hstride, const int* Hg, const uint32_t* sz, int nslots, int bs,
                                        float (&accf)[TB]) {
  constexpr int C = ul_chunks(B);
  const int gshift = 31 - __clz(p.group);
  const int tstride = hstride / 2;
  for (int rb = rb0; rb < rb1; ++rb) {
    const int* hq32 = reinterpret_cast<const int*>(hq + (rb - rb0) * kRows);
    const uint8_t* cb = code + (size_t)(rb - rb0) * C * kChunkBytes;
    if (B == 16) {
#pragma unroll 4
      for (int c = 0; c < 16; ++c) {
        const uint4 v = ldg_stream(cb + (size_t)c * kChunkBytes);
        const uint32_t wv[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int w = 0; w < 4; ++w) {
          const int r = 8 * c + 2 * w;
#pragma unroll
          for (int tt = 0; tt < TB; ++tt) {
            const int hp = hq32[tt * tstride + r / 2];
            const float h0 = (float)(int16_t)(hp & 0xFFFF), h1 = (float)(hp >> 16);
            accf[tt] = fmaf(h0, f16lo(wv[w]), fmaf(h1, f16hi(wv[w]), accf[tt]));
          }
        }
      }
      continue;
    }
    int acc[G][TB], acch[G][TB];
#pragma unroll
    for (int g = 0; g < G; ++g)
#pragma unroll
      for (int tt = 0; tt < TB; ++tt) acc[g][tt] = acch[g][tt] = 0;
    uint4 v[C];
#pragma unroll
    for (int c = 0; c < C; ++c) v[c] = ldg_stream(cb + (size_t)c * kChunkBytes);
    if (B == 3) {
      ul_chunk<2, G, TB>(v[0], 0, hq32, tstride, gshift, acc);
      ul_chunk<2, G, TB>(v[1], 64, hq32, tstride, gshift, acc);
      ul_chunk<1, G, TB>(v[2], 0, hq32, tstride, gshift, acch);
    } else if (B == 6) {
#pragma unroll
      for (int c = 0; c < 4; ++c) ul_chunk<4, G, TB>(v[c], 32 * c, hq32, tstride, gshift, acc);
      ul_chunk<2, G, TB>(v[4], 0, hq32, tstride, gshift, acch);
      ul_chunk<2, G, TB>(v[5], 64, hq32, tstride, gshift, acch);
    } else {
#pragma unroll
      for (int c = 0; c < C; ++c) ul_chunk<B, G, TB>(v[c], c * (kRows / B), hq32, tstride, gshift, acc);
    }
    // apply the group scales (groups of >= 128 rows span several row blocks)
    const int gfirst = (rb * kRows) >> gshift;
#pragma unroll
    for (int g = 0; g < G; ++g) {
      const uint32_t szw = sz[(size_t)(gfirst + g) * nslots + bs];
      const float sc = __half2float(__ushort_as_half((unsigned short)(szw & 0xFFFFu)));
      const float zp = __half2float(__ushort_as_half((unsigned short)(szw >> 16)));
      const bool starts = G > 1 || ((rb * kRows) & (p.group - 1)) == 0;
      const int hgi = (((rb * kRows) >> gshift) + g) - ((rb0 * kRows) >> gshift);
#pragma unroll
      for (int tt = 0; tt < TB; ++tt) {
        const int tot = (B == 3 || B == 6) ? acc[g][tt] + (acch[g][tt] << (B == 3 ? 2 : 4)) : acc[g][tt];
        float d = (float)tot;
        if (starts) d = fmaf(-zp, (float)Hg[tt * 64 + hgi], d);
        accf[tt] = fmaf(sc, d, accf[tt]);
      }
    }
  }
}

template <int G, int TB>
__global__ void __launch_bounds__(kThreads) k_down(Fwd p) {
  pdl_trigger();
  pdl_wait();
  extern __shared__ int4 smem_k3[];
  const int rbc = p.rbc;
  const int nrows_max = rbc * kRows;
  float* hf = reinterpret_cast<float*>(smem_k3);                       // [TB][nrows_max]
  int16_t* hq = reinterpret_cast<int16_t*>(hf + TB * nrows_max);       // [TB][nrows_max]
  int* Hg = reinterpret_cast<int*>(hq + TB * nrows_max);               // [TB][64]
  float* red = reinterpret_cast<float*>(Hg + TB * 64);                 // [kWarps][TB]
  float* shs = red + kWarps * TB;                                      // [TB] scales
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const int A = p.active[0];
  const int ntg = (p.ul_max_tiles + kK3Tiles - 1) / kK3Tiles;
  const int nrc = (p.NRB + rbc - 1) / rbc;
  const int total = A * ntg * nrc;
  const int gshift = 31 - __clz(p.group);
  for (int item = blockIdx.x; item < total; item += gridDim.x) {
    const int a = item / (ntg * nrc);
    const int r = item - a * ntg * nrc;
    const int tg = r / nrc, rc = r - tg * nrc;
    const int e = p.active[1 + a];
    const ExpertDesc& xd = p.desc[2 * p.E + e];
    if (tg * kK3Tiles >= xd.ntiles) continue;
    const int rb0 = rc * rbc, rb1 = min(p.NRB, rb0 + rbc);
    const int row0 = rb0 * kRows, nrows = (rb1 - rb0) * kRows;
    const int ntok = p.expert_count[e], pst = p.expert_start[e];
    // this warp's tile and bucket
    const int tile = tg * kK3Tiles + wid;
    int bi = -1;
    if (tile < xd.ntiles)
      for (int q = 0; q < xd.nbk; ++q)
        if (tile >= xd.bk[q].tile0 && tile < xd.bk[q].tile0 + xd.bk[q].ntiles) bi = q;
    for (int tb0 = 0; tb0 < ntok; tb0 += TB) {
      const int tb = min(TB, ntok - tb0);
      __syncthreads();
      // h = SiLU(gate) * up for the rows of this block
      float mx[TB];
#pragma unroll
      for (int tt = 0; tt < TB; ++tt) mx[tt] = 0.f;
      for (int i = threadIdx.x; i < nrows; i += blockDim.x) {
#pragma unroll
        for (int tt = 0; tt < TB; ++tt) {
          float hv = 0.f;
          if (tt < tb) {
            const int pr = p.pair_list[pst + tb0 + tt];
            const float g = p.gu[((size_t)pr * 2) * p.I_pad + row0 + i];
            const float u = p.gu[((size_t)pr * 2 + 1) * p.I_pad + row0 + i];
            hv = g / (1.f + __expf(-g)) * u;
          }
          hf[tt * nrows_max + i] = hv;
          mx[tt] = fmaxf(mx[tt], fabsf(hv));
        }
      }
#pragma unroll
      for (int tt = 0; tt < TB; ++tt) {
        const float m = warp_max(mx[tt]);
        if (lane == 0) red[wid * TB + tt] = m;
      }
      __syncthreads();
      if (threadIdx.x < TB) {
        float m = 0.f;
        for (int w = 0; w < kWarps; ++w) m = fmaxf(m, red[w * TB + threadIdx.x]);
        shs[threadIdx.x] = m;
      }
      __syncthreads();
      for (int i = threadIdx.x; i < nrows; i += blockDim.x) {
#pragma unroll
        for (int tt = 0; tt < TB; ++tt) {
          const float m = shs[tt];
          const float inv = m > 0.f ? 32767.f / m : 0.f;
          hq[tt * nrows_max + i] = (int16_t)__float2int_rn(hf[tt * nrows_max + i] * inv);
        }
      }
      __syncthreads();
      // group sums of the quantised h (groups lie inside the block's rows)
      const int ngr = nrows >> gshift;
      for (int q = wid; q < TB * ngr; q += kWarps) {
        const int tt = q / ngr, g = q - tt * ngr;
        int sacc = 0;
        for (int i = lane; i < p.group; i += 32) sacc += hq[tt * nrows_max + (g << gshift) + i];
#pragma unroll
        for (int o = 16; o; o >>= 1) sacc += __shfl_xor_sync(0xFFFFFFFFu, sacc, o);
        if (lane == 0) Hg[tt * 64 + g] = sacc;
      }
      __syncthreads();
      if (bi < 0) continue;
      const BucketDesc& bd = xd.bk[bi];
      const int bs = (tile - bd.tile0) * 32 + lane;     // bucket-local slot
      const int gs = bd.slot0 + bs;
      const int j = reinterpret_cast<const int32_t*>(p.img + xd.unit_off)[gs];
      const float al = reinterpret_cast<const float*>(p.img + xd.alpha_off)[gs];
      const uint8_t* code = p.img + xd.code_base + bd.code_off +
                            ((size_t)(tile - bd.tile0) * p.NRB + rb0) * ul_chunks(bd.bits) * kChunkBytes + lane * 16;
      const uint32_t* sz = reinterpret_cast<const uint32_t*>(p.img + bd.sz_off);
      float accf[TB];
#pragma unroll
      for (int tt = 0; tt < TB; ++tt) accf[tt] = 0.f;
      switch (bd.bits) {
        case 1: ul_tile<1, G, TB>(p, code, rb0, rb1, hq, nrows_max, Hg, sz, bd.nslots, bs, accf); break;
        case 2: ul_tile<2, G, TB>(p, code, rb0, rb1, hq, nrows_max, Hg, sz, bd.nslots, bs, accf); break;
        case 3: ul_tile<3, G, TB>(p, code, rb0, rb1, hq, nrows_max, Hg, sz, bd.nslots, bs, accf); break;
        case 4: ul_tile<4, G, TB>(p, code, rb0, rb1, hq, nrows_max, Hg, sz, bd.nslots, bs, accf); break;
        case 6: ul_tile<6, G, TB>(p, code, rb0, rb1, hq, nrows_max, Hg, sz, bd.nslots, bs, accf); break;
        case 8: ul_tile<8, G, TB>(p, code, rb0, rb1, hq, nrows_max, Hg, sz, bd.nslots, bs, accf); break;
        default: ul_tile<16, G, TB>(p, code, rb0, rb1, hq, nrows_max, Hg, sz, bd.nslots, bs, accf); break;
      }
      if (al != 0.f) {
#pragma unroll
        for (int tt = 0; tt < TB; ++tt) {
          if (tt < tb) {
            const int pr = p.pair_list[pst + tb0 + tt];
            const float scale = shs[tt] * (1.f / 32767.f);
            atomicAdd(p.s + (size_t)(pr / p.k) * p.n_pad + j, p.pair_weight[pr] * al * scale * accf[tt]);
          }
        }
      }
    }
  }
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
struct WsLayout {
  size_t status, pair_expert, pair_weight, expert_count, expert_start, pair_list, active, z, gu, s;
  size_t x_stage, logits_stage, y_stage, total;
};

WsLayout ws_layout(const ImageHeader& hd, int T, int k) {
  WsLayout w;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off = align_up(off + bytes, 256);
    return o;
  };
  const size_t P = (size_t)T * k;
  w.status = take(16);
  w.pair_expert = take(P * 4);
  w.pair_weight = take(P * 4);
  w.expert_count = take((size_t)hd.E * 4);
  w.expert_start = take(((size_t)hd.E + 1) * 4);
  w.pair_list = take(P * 4);
  w.active = take(((size_t)hd.E + 1) * 4);
  w.z = take(2 * (size_t)T * hd.n_pad * 4);
  w.gu = take(P * 2 * hd.I_pad * 4);
  w.s = take((size_t)T * hd.n_pad * 4);
  w.x_stage = take((size_t)T * hd.D * 2);
  w.logits_stage = take((size_t)T * hd.E * 4);
  w.y_stage = take((size_t)T * hd.D * 4);
  w.total = off;
  return w;
}

int k3_rbc(const ImageHeader& hd) {
  int rbc = std::min(hd.NRB, kK3MaxRB);
  const int need = std::max(1, hd.group / kRows);   // whole groups per block
  rbc = std::max(need, rbc / need * need);
  return rbc;
}

template <class K>
int launch(K kernel, dim3 grid, dim3 block, size_t smem, cudaStream_t st, bool pdl, const Fwd& p) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  BM_CK(cudaLaunchKernelEx(&cfg, kernel, p));
  return BITSMOE_OK;
}

template <class K>
int set_smem(K kernel, size_t smem) {
  if (smem > 48 * 1024) BM_CK(cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
  return BITSMOE_OK;
}

template <int TB>
int launch_gemv(bool proj, const Fwd& p, int sms, cudaStream_t st, bool pdl) {
  const int ld = proj ? p.D_pad : p.n_pad;
  const size_t smem = (size_t)TB * ld * 4;
  int rc;
  if (proj) {
    if ((rc = set_smem(k_gemv<TB, true>, smem))) return rc;
    return launch(k_gemv<TB, true>, dim3(sms * 4), dim3(kThreads), smem, st, pdl, p);
  }
  if ((rc = set_smem(k_gemv<TB, false>, smem))) return rc;
  return launch(k_gemv<TB, false>, dim3(sms * 4), dim3(kThreads), smem, st, pdl, p);
}

int launch_gemv_any(bool proj, const Fwd& p, int sms, cudaStream_t st, bool pdl) {
  if (p.T <= 1) return launch_gemv<1>(proj, p, sms, st, pdl);
  if (p.T <= 2) return launch_gemv<2>(proj, p, sms, st, pdl);
  if (p.T <= 4) return launch_gemv<4>(proj, p, sms, st, pdl);
  return launch_gemv<8>(proj, p, sms, st, pdl);
}

template <int G, int TB>
int launch_k2k3(const Fwd& p, int sms, cudaStream_t st, bool pdl, const std::function<int()>& between) {
  int rc;
  const size_t sm2 = (size_t)kWarps * G * TB * p.s16 * 2;
  if ((rc = set_smem(k_gateup<G, TB>, sm2))) return rc;
  if ((rc = launch(k_gateup<G, TB>, dim3(sms * 2), dim3(kThreads), sm2, st, pdl, p))) return rc;
  if (between && (rc = between())) return rc;
  const size_t nrm = (size_t)p.rbc * kRows;
  const size_t sm3 = TB * nrm * 4 + TB * nrm * 2 + TB * 64 * 4 + kWarps * TB * 4 + TB * 4;
  if ((rc = set_smem(k_down<G, TB>, sm3))) return rc;
  return launch(k_down<G, TB>, dim3(sms * 2), dim3(kThreads), sm3, st, pdl, p);
}

template <int G>
int launch_k2k3_tb(const Fwd& p, int sms, cudaStream_t st, bool pdl, const std::function<int()>& between) {
  return p.T == 1 ? launch_k2k3<G, 1>(p, sms, st, pdl, between) : launch_k2k3<G, 4>(p, sms, st, pdl, between);
}

bool aligned(const void* ptr, size_t a) { return ((uintptr_t)ptr % a) == 0; }

int forward_impl(const void* x, const float* logits, int T, int top_k, const bitsmoe_layer* L, float* y,
                 void* ws, size_t ws_bytes, cudaStream_t st, cudaEvent_t* ev = nullptr) {
  const ImageHeader& hd = L->hd();
  const bool pdl = ev == nullptr;   // profiling runs the phases back to back without overlap
  const WsLayout w = ws_layout(hd, T, top_k);
  uint8_t* wb = static_cast<uint8_t*>(ws);
  Fwd p;
  std::memset(&p, 0, sizeof(p));
  p.img = L->d_img;
  p.desc = reinterpret_cast<const ExpertDesc*>(L->d_img + hd.off_desc);
  p.seg = reinterpret_cast<const int32_t*>(L->d_img + hd.off_seg);
  p.basis_in = reinterpret_cast<const uint16_t*>(L->d_img + hd.off_basis_in);
  p.basis_out = reinterpret_cast<const uint16_t*>(L->d_img + hd.off_basis_out);
  p.D = hd.D; p.E = hd.E; p.I = hd.I; p.n = hd.n; p.group = hd.group;
  p.D_pad = hd.D_pad; p.n_pad = hd.n_pad; p.I_pad = hd.I_pad; p.NRB = hd.NRB; p.NG = hd.NG;
  p.nseg = hd.nseg; p.ul_max_tiles = hd.ul_max_tiles;
  p.T = T; p.k = top_k; p.P = T * top_k;
  p.s16 = (int)align_up(std::max(hd.seg_max_slots, 8), 64) + 8;
  p.rbc = k3_rbc(hd);
  p.x = static_cast<const uint16_t*>(x);
  p.logits = logits;
  p.y = y;
  p.status = reinterpret_cast<int*>(wb + w.status);
  p.pair_expert = reinterpret_cast<int*>(wb + w.pair_expert);
  p.pair_weight = reinterpret_cast<float*>(wb + w.pair_weight);
  p.expert_count = reinterpret_cast<int*>(wb + w.expert_count);
  p.expert_start = reinterpret_cast<int*>(wb + w.expert_start);
  p.pair_list = reinterpret_cast<int*>(wb + w.pair_list);
  p.active = reinterpret_cast<int*>(wb + w.active);
  p.z = reinterpret_cast<float*>(wb + w.z);
  p.gu = reinterpret_cast<float*>(wb + w.gu);
  p.s = reinterpret_cast<float*>(wb + w.s);
  const int sms = L->num_sms;
  int rc;
  auto mark = [&](int i) -> int {
    if (ev) BM_CK(cudaEventRecord(ev[i], st));
    return BITSMOE_OK;
  };
  const int tpb = std::max(1, 1024 / hd.E);
  if ((rc = mark(0))) return rc;
  if ((rc = launch(k_router, dim3(1), dim3(1024), (size_t)tpb * hd.E * 4, st, false, p))) return rc;
  if ((rc = mark(1))) return rc;
  if ((rc = launch_gemv_any(true, p, sms, st, pdl))) return rc;
  if ((rc = mark(2))) return rc;
  const int G = std::max(1, kRows / hd.group);
  if (G == 1) rc = launch_k2k3_tb<1>(p, sms, st, pdl, ev ? [&]() { return mark(3); } : std::function<int()>());
  else if (G == 2) rc = launch_k2k3_tb<2>(p, sms, st, pdl, ev ? [&]() { return mark(3); } : std::function<int()>());
  else rc = launch_k2k3_tb<4>(p, sms, st, pdl, ev ? [&]() { return mark(3); } : std::function<int()>());
  if (rc) return rc;
  if ((rc = mark(4))) return rc;
  if ((rc = launch_gemv_any(false, p, sms, st, pdl))) return rc;
  return mark(5);
}

int check_device(const bitsmoe_layer* L) {
  int dev = -1;
  BM_CK(cudaGetDevice(&dev));
  return dev == L->device ? BITSMOE_OK : BITSMOE_ERR_INVALID_ARG;
}

int upload(std::vector<uint8_t>&& img, int device, bitsmoe_layer** out) {
  int cnt = 0;
  BM_CK(cudaGetDeviceCount(&cnt));
  if (device < 0 || device >= cnt) return BITSMOE_ERR_INVALID_ARG;
  int prev = 0;
  BM_CK(cudaGetDevice(&prev));
  BM_CK(cudaSetDevice(device));
  int sms = 0;
  cudaError_t e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, device);
  uint8_t* d = nullptr;
  if (e == cudaSuccess) e = cudaMalloc(&d, img.size());
  if (e == cudaSuccess) e = cudaMemcpy(d, img.data(), img.size(), cudaMemcpyHostToDevice);
  cudaSetDevice(prev);
  if (e != cudaSuccess) {
    if (d) cudaFree(d);
    return e == cudaErrorMemoryAllocation ? BITSMOE_ERR_OOM : cuda_fail(e);
  }
  bitsmoe_layer* L = new (std::nothrow) bitsmoe_layer;
  if (!L) {
    cudaFree(d);
    return BITSMOE_ERR_OOM;
  }
  const ImageHeader* hd = header_of(img.data());
  const size_t meta_end = hd->off_basis_in;   // header + descriptors + segments
  L->device = device;
  L->num_sms = sms;
  L->d_img = d;
  L->bytes = img.size();
  L->meta.assign(img.begin(), img.begin() + meta_end);
  *out = L;
  return BITSMOE_OK;
}

// Scratch of bitsmoe_moe_forward_noalloc: one fixed array per device that
// loads the library.  Host code only ever sees a host-side stand-in for this
// symbol; the device address comes from cudaGetSymbolAddress, once per device.
constexpr size_t kNoAllocBytes = BITSMOE_NOALLOC_SCRATCH_BYTES;
constexpr int kNoAllocMaxDevices = 64;
static __device__ __align__(256) uint8_t g_noalloc_scratch[kNoAllocBytes];
std::mutex g_noalloc_mu;
void* g_noalloc_addr[kNoAllocMaxDevices] = {};

// Device address of the scratch on `device` (which must be current).
int noalloc_scratch(int device, void** out) {
  if (device < 0 || device >= kNoAllocMaxDevices) return BITSMOE_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> lock(g_noalloc_mu);
  if (!g_noalloc_addr[device]) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess || !p) return cuda_fail(e != cudaSuccess ? e : cudaErrorInvalidSymbol);
    g_noalloc_addr[device] = p;
  }
  *out = g_noalloc_addr[device];
  return BITSMOE_OK;
}

}  // namespace

extern "C" {

int bitsmoe_moe_forward_noalloc(const void* x, const float* logits, int T, int top_k, const bitsmoe_layer* L,
                                float* y, void* stream) {
  if (!L || T < 0) return BITSMOE_ERR_INVALID_ARG;
  const ImageHeader& hd = L->hd();
  if (top_k < 1 || top_k > std::min(hd.E, 32)) return BITSMOE_ERR_INVALID_ARG;
  if ((int64_t)T * top_k > (1 << 24) || (int64_t)T * hd.D > (1ll << 31)) return BITSMOE_ERR_SHAPE;
  if (T == 0) return BITSMOE_OK;
  if (!x || !logits || !y) return BITSMOE_ERR_INVALID_ARG;
  if (!aligned(x, 16) || !aligned(logits, 16) || !aligned(y, 16)) return BITSMOE_ERR_ALIGNMENT;
  if (ws_layout(hd, T, top_k).total > kNoAllocBytes) return BITSMOE_ERR_WORKSPACE_TOO_SMALL;
  int rc = check_device(L);
  if (rc) return rc;
  void* ws = nullptr;
  if ((rc = noalloc_scratch(L->device, &ws))) return rc;
  return forward_impl(x, logits, T, top_k, L, y, ws, kNoAllocBytes, static_cast<cudaStream_t>(stream));
}

int bitsmoe_pack(const bitsmoe_layer_host* src, int device, bitsmoe_layer** out) {
  if (!src || !out) return BITSMOE_ERR_INVALID_ARG;
  *out = nullptr;
  std::vector<uint8_t> img;
  int rc = build_image(src, img);
  if (rc) return rc;
  return upload(std::move(img), device, out);
}

int bitsmoe_load_blob(const void* blob, size_t bytes, int device, bitsmoe_layer** out) {
  if (!blob || !out) return BITSMOE_ERR_INVALID_ARG;
  *out = nullptr;
  const uint8_t* b = static_cast<const uint8_t*>(blob);
  int rc = validate_image(b, bytes);
  if (rc) return rc;
  std::vector<uint8_t> img(b, b + bytes);
  return upload(std::move(img), device, out);
}

int bitsmoe_unpack(const bitsmoe_layer* L, bitsmoe_layer_host_out* dst) {
  if (!L || !dst) return BITSMOE_ERR_INVALID_ARG;
  std::vector<uint8_t> img(L->bytes);
  int prev = 0;
  BM_CK(cudaGetDevice(&prev));
  BM_CK(cudaSetDevice(L->device));
  cudaError_t e = cudaMemcpy(img.data(), L->d_img, L->bytes, cudaMemcpyDeviceToHost);
  cudaSetDevice(prev);
  if (e != cudaSuccess) return cuda_fail(e);
  return unpack_image(img.data(), img.size(), dst);
}

int bitsmoe_layer_dims(const bitsmoe_layer* L, int32_t dims[5]) {
  if (!L || !dims) return BITSMOE_ERR_INVALID_ARG;
  const ImageHeader& hd = L->hd();
  dims[0] = hd.D; dims[1] = hd.E; dims[2] = hd.I; dims[3] = hd.n; dims[4] = hd.group;
  return BITSMOE_OK;
}

int bitsmoe_layer_bytes(const bitsmoe_layer* L, bitsmoe_bytes* out) {
  if (!L || !out) return BITSMOE_ERR_INVALID_ARG;
  const ImageHeader& hd = L->hd();
  out->total = hd.total_bytes;
  out->basis = 3ull * hd.D * hd.n * 2;
  out->codes_padded = hd.codes_bytes;
  out->meta = hd.meta_bytes;
  return BITSMOE_OK;
}

int bitsmoe_expert_moved_bytes(const bitsmoe_layer* L, int e, uint64_t out[3]) {
  if (!L || !out) return BITSMOE_ERR_INVALID_ARG;
  const ImageHeader& hd = L->hd();
  if (e < 0 || e >= hd.E) return BITSMOE_ERR_INVALID_ARG;
  const ExpertDesc* d = L->desc();
  for (int h = 0; h < 3; ++h) out[h] = d[h * hd.E + e].moved;
  return BITSMOE_OK;
}

size_t bitsmoe_workspace_bytes(const bitsmoe_layer* L, int T, int top_k) {
  if (!L || T < 0 || top_k < 1 || top_k > std::min(L->hd().E, 32)) return 0;
  return ws_layout(L->hd(), T, top_k).total;
}

int bitsmoe_moe_forward(const void* x, const float* logits, int T, int top_k, const bitsmoe_layer* L, float* y,
                        void* ws, size_t ws_bytes, void* stream) {
  if (!L || T < 0) return BITSMOE_ERR_INVALID_ARG;
  const ImageHeader& hd = L->hd();
  if (top_k < 1 || top_k > std::min(hd.E, 32)) return BITSMOE_ERR_INVALID_ARG;
  if ((int64_t)T * top_k > (1 << 24) || (int64_t)T * hd.D > (1ll << 31)) return BITSMOE_ERR_SHAPE;
  if (T == 0) return BITSMOE_OK;
  if (!x || !logits || !y || !ws) return BITSMOE_ERR_INVALID_ARG;
  if (!aligned(x, 16) || !aligned(logits, 16) || !aligned(y, 16) || !aligned(ws, 256)) return BITSMOE_ERR_ALIGNMENT;
  if (ws_bytes < ws_layout(hd, T, top_k).total) return BITSMOE_ERR_WORKSPACE_TOO_SMALL;
  int rc = check_device(L);
  if (rc) return rc;
  return forward_impl(x, logits, T, top_k, L, y, ws, ws_bytes, static_cast<cudaStream_t>(stream));
}

int bitsmoe_moe_forward_host(const void* x_host, const float* logits_host, int T, int top_k,
                             const bitsmoe_layer* L, float* y_host, void* ws, size_t ws_bytes, void* stream) {
  if (!L || T < 0) return BITSMOE_ERR_INVALID_ARG;
  const ImageHeader& hd = L->hd();
  if (top_k < 1 || top_k > std::min(hd.E, 32)) return BITSMOE_ERR_INVALID_ARG;
  if ((int64_t)T * top_k > (1 << 24) || (int64_t)T * hd.D > (1ll << 31)) return BITSMOE_ERR_SHAPE;
  if (T == 0) return BITSMOE_OK;
  if (!x_host || !logits_host || !y_host || !ws) return BITSMOE_ERR_INVALID_ARG;
  if (!aligned(ws, 256)) return BITSMOE_ERR_ALIGNMENT;
  const WsLayout w = ws_layout(hd, T, top_k);
  if (ws_bytes < w.total) return BITSMOE_ERR_WORKSPACE_TOO_SMALL;
  int rc = check_device(L);
  if (rc) return rc;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  uint8_t* wb = static_cast<uint8_t*>(ws);
  BM_CK(cudaMemcpyAsync(wb + w.x_stage, x_host, (size_t)T * hd.D * 2, cudaMemcpyHostToDevice, st));
  BM_CK(cudaMemcpyAsync(wb + w.logits_stage, logits_host, (size_t)T * hd.E * 4, cudaMemcpyHostToDevice, st));
  rc = forward_impl(wb + w.x_stage, reinterpret_cast<const float*>(wb + w.logits_stage), T, top_k, L,
                    reinterpret_cast<float*>(wb + w.y_stage), ws, ws_bytes, st);
  if (rc) return rc;
  BM_CK(cudaMemcpyAsync(y_host, wb + w.y_stage, (size_t)T * hd.D * 4, cudaMemcpyDeviceToHost, st));
  BM_CK(cudaStreamSynchronize(st));
  return BITSMOE_OK;
}

int bitsmoe_profile_forward(const void* x, const float* logits, int T, int top_k, const bitsmoe_layer* L,
                            float* y, void* ws, size_t ws_bytes, void* stream, float phase_ms[5]) {
  if (!phase_ms) return BITSMOE_ERR_INVALID_ARG;
  if (!L || T < 0) return BITSMOE_ERR_INVALID_ARG;
  const ImageHeader& hd = L->hd();
  if (top_k < 1 || top_k > std::min(hd.E, 32)) return BITSMOE_ERR_INVALID_ARG;
  if ((int64_t)T * top_k > (1 << 24) || (int64_t)T * hd.D > (1ll << 31)) return BITSMOE_ERR_SHAPE;
  for (int i = 0; i < 5; ++i) phase_ms[i] = 0.f;
  if (T == 0) return BITSMOE_OK;
  if (!x || !logits || !y || !ws) return BITSMOE_ERR_INVALID_ARG;
  if (!aligned(x, 16) || !aligned(logits, 16) || !aligned(y, 16) || !aligned(ws, 256)) return BITSMOE_ERR_ALIGNMENT;
  if (ws_bytes < ws_layout(hd, T, top_k).total) return BITSMOE_ERR_WORKSPACE_TOO_SMALL;
  int rc = check_device(L);
  if (rc) return rc;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  cudaEvent_t ev[6] = {};
  for (int i = 0; i < 6 && rc == BITSMOE_OK; ++i)
    if (cudaEventCreate(&ev[i]) != cudaSuccess) rc = BITSMOE_ERR_CUDA;
  if (rc == BITSMOE_OK) rc = forward_impl(x, logits, T, top_k, L, y, ws, ws_bytes, st, ev);
  if (rc == BITSMOE_OK) {
    cudaError_t e = cudaEventSynchronize(ev[5]);
    for (int i = 0; i < 5 && e == cudaSuccess; ++i) e = cudaEventElapsedTime(&phase_ms[i], ev[i], ev[i + 1]);
    if (e != cudaSuccess) rc = cuda_fail(e);
  }
  for (int i = 0; i < 6; ++i)
    if (ev[i]) cudaEventDestroy(ev[i]);
  return rc;
}

int bitsmoe_last_device_status(void* ws, void* stream) {
  if (!ws) return BITSMOE_ERR_INVALID_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  int v = 0;
  BM_CK(cudaMemcpyAsync(&v, ws, sizeof(int), cudaMemcpyDeviceToHost, st));
  BM_CK(cudaStreamSynchronize(st));
  if (v != 0) {
    const int zero = 0;
    BM_CK(cudaMemcpyAsync(ws, &zero, sizeof(int), cudaMemcpyHostToDevice, st));
    BM_CK(cudaStreamSynchronize(st));
  }
  return v;
}

void bitsmoe_free(bitsmoe_layer* L) {
  if (!L) return;
  int prev = 0;
  if (cudaGetDevice(&prev) == cudaSuccess) {
    cudaSetDevice(L->device);
    cudaFree(L->d_img);
    cudaSetDevice(prev);
  }
  delete L;
}

int bitsmoe_last_cuda_error(void) { return g_last_cuda; }

}  // extern "C"
