// BitsMoE quantized MoE-layer forward on sm_103a (GB300): the kernel chains
// and the C ABI.
//
// Stage 3 of the method (Fig. 1; "Inference Efficiency", Sec. Experiments):
// the activation is projected once onto the shared bases, then each routed
// expert's packed spectral factors are unpacked and applied inside the kernels
// without rebuilding the expert weights.  A call runs one of three plans
// (forward_impl), kernels chained on the caller's stream with programmatic
// dependent launch (PDL) so that a kernel's prologue overlaps the tail of the
// previous one:
//
//   one token      k_fused (fused.cu): the whole layer in one persistent kernel
//   2 .. 8 tokens  k_route_publish   routing by one block, published with a flag
//                  k_gemv_bulk<P>    z_g = Phi_g^T x, z_u = Phi_u^T x (rows through
//                                    a bulk-copy ring); zeroes the accumulators
//                  k_gateup_dec      gate/up = P_hat (alpha * z): dp2a over
//                                    bucketed uniform-bit streams staged per warp
//                                    item, int16 activation operand, vector red.add
//                  k_down_dec        h = SiLU(gate) * up, then
//                                    s += w_e * alpha_dn * (P_hat_dn^T h) per unit
//                  k_gemv_bulk<O>    y = Phi_dn s (fp32 out)
//   more tokens    k_router (multi-block), k_gemm_tc (gemm.cu: tensor cores) for
//                  both projections, the same gate/up and down kernels
//
// The identity behind the association is Eq. app_normalized_decomposition
// (W = P A Phi^T for gate/up, W = Phi A P^T for down); summing the experts'
// n-dim spectral vectors before Phi_dn is exact by linearity.
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstring>
#include <functional>
#include <limits>
#include <mutex>
#include <vector>

#include "device.cuh"
#include "internal.h"

using namespace bmoe;

struct bitsmoe_layer {
  int device;
  int num_sms;
  uint8_t* d_img;
  uint64_t bytes;
  uint8_t* d_stage = nullptr;  // staging records of the fused single-token kernel
  const CStage* d_cst = nullptr;
  const DStage* d_dst = nullptr;
  uint64_t stage_bytes = 0;
  const uint8_t* d_meta = nullptr;   // metadata mirror of the staging items (inside d_stage's allocation)
  uint64_t meta_bytes = 0;
  bool meta_ok = false;              // the mirror was built (the fused kernel needs it)
  alignas(64) uint8_t map_in[128];    // TMA maps of the two input bases and of the output basis
  alignas(64) uint8_t map_out[128];
  bool maps = false;
  bool tcx = false;            // expert factors on tensor cores: no 16-bit units, groups of whole row blocks
  const float* d_msa = nullptr;   // [2][E] max |scale * alpha| of each gate/up (h, e) (inside d_stage's allocation)
  std::vector<uint8_t> meta;   // host copy of header + descriptors + segment table
  int seg_bytes = 0;           // largest gate/up item: code bytes inside one row block
  int ul_max_chunks = 1;       // largest 16-byte chunks per row block of any down unit
  // clustered single-token kernel: records per cluster size (kF2Sizes), the most
  // clusters of that size that fit the device at once, the staged sizes
  uint8_t* d_f2 = nullptr;
  uint64_t f2_off[5] = {};
  int f2_nc[5] = {};
  F2Sizes f2_sz[5] = {};
  // the clustered kernel's plan per top_k (1..32), computed on first use
  mutable std::mutex f2_mu;
  mutable signed char f2_ci[33];
  mutable F2Args f2_args[33];
  bitsmoe_layer() { std::memset(f2_ci, 0x7F, sizeof(f2_ci)); }
  const ImageHeader& hd() const { return *reinterpret_cast<const ImageHeader*>(meta.data()); }
  const ExpertDesc* desc() const {
    return reinterpret_cast<const ExpertDesc*>(meta.data() + hd().off_desc);
  }
};

namespace {

// Cluster sizes of the clustered single-token kernel, largest first (index into
// bitsmoe_layer's f2_* arrays).
constexpr int kF2Sizes[5] = {8, 4, 3, 2, 1};

// Testing hook (bitsmoe_debug_wait_limit): bound of the single-token kernels' waits
// and whether block 0 skips its arrival at their first grid barrier.
std::atomic<long long> g_dbg_spin{0};
std::atomic<int> g_dbg_skip{0};
// Testing hook (bitsmoe_debug_single_token_kernel): 1 keeps single-token forwards on the
// kernel without clusters, 2 takes the clustered one wherever it fits.
std::atomic<int> g_dbg_kernel{0};
// testing hook: debug bounds checks in the single-token kernels; layers uploaded while it is
// on get a zero-filled slack of the image's own size after it (so that a record shifted past
// the image, as the tests do, still reads mapped memory)
std::atomic<int> g_dbg_bounds{0};

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

// ---------------------------------------------------------------------------
// Pre-norm of a stacked MoE block: r = h / sqrt(mean(h^2) + eps) (unit weight),
// x = bf16(r), router logits = W_r x (fp32 accumulate).  Each block computes a
// slice of the experts' logits; its warps load their router rows in the PDL
// prologue, before waiting for the kernel that produced h.  It lets the next
// kernel launch only once x and the logits are written.
// ---------------------------------------------------------------------------
struct NormArgs {
  const float* h;
  const uint16_t* w;
  float eps;
  int T, D, E, D_pad8;
  uint16_t* x;
  float* logits;
};

template <int TB>
__global__ void __launch_bounds__(kThreads) k_norm_router(NormArgs a) {
  extern __shared__ float4 smem_nr[];
  float* xs = reinterpret_cast<float*>(smem_nr);          // [TB][D_pad8] bf16-rounded r
  float* red = xs + (size_t)TB * a.D_pad8;                 // [kWarps][TB]
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const int nch = a.D >> 3;                                // 16-byte chunks of a row (D % 8 == 0)
  const int row0 = blockIdx.x * kWarps + wid;
  const int nrw = gridDim.x * kWarps;
  uint4 pre[8];
  if (row0 < a.E) {
    const uint4* rp = reinterpret_cast<const uint4*>(a.w + (size_t)row0 * a.D);
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const int c = u * 32 + lane;
      pre[u] = c < nch ? ldg_stream(rp + c) : make_uint4(0, 0, 0, 0);
    }
  }
  pdl_wait();
  for (int t0 = 0; t0 < a.T; t0 += TB) {
    const int tb = min(TB, a.T - t0);
    __syncthreads();
    float ss[TB];
#pragma unroll
    for (int tt = 0; tt < TB; ++tt) ss[tt] = 0.f;
    for (int d = threadIdx.x; d < a.D; d += blockDim.x)
#pragma unroll
      for (int tt = 0; tt < TB; ++tt)
        if (tt < tb) {
          const float v = a.h[(size_t)(t0 + tt) * a.D + d];
          ss[tt] = fmaf(v, v, ss[tt]);
        }
#pragma unroll
    for (int tt = 0; tt < TB; ++tt) {
      const float v = warp_sum(ss[tt]);
      if (lane == 0) red[wid * TB + tt] = v;
    }
    __syncthreads();
    float inv[TB];
#pragma unroll
    for (int tt = 0; tt < TB; ++tt) {
      float sum = 0.f;
      for (int w = 0; w < kWarps; ++w) sum += red[w * TB + tt];
      inv[tt] = rsqrtf(sum / (float)a.D + a.eps);
    }
    for (int i = threadIdx.x; i < TB * a.D; i += blockDim.x) {
      const int tt = i / a.D, d = i - tt * a.D;
      float r = 0.f;
      if (tt < tb) {
        float iv = inv[0];
#pragma unroll
        for (int u = 1; u < TB; ++u)
          if (u == tt) iv = inv[u];
        // round to bf16 (nearest even): both the MoE input and the router use it
        uint32_t u32 = __float_as_uint(a.h[(size_t)(t0 + tt) * a.D + d] * iv);
        u32 = (u32 + 0x7FFFu + ((u32 >> 16) & 1u)) & 0xFFFF0000u;
        r = __uint_as_float(u32);
        if (blockIdx.x == 0) a.x[(size_t)(t0 + tt) * a.D + d] = (uint16_t)(u32 >> 16);
      }
      xs[tt * a.D_pad8 + d] = r;
    }
    __syncthreads();
    for (int row = row0; row < a.E; row += nrw) {
      const uint4* rp = reinterpret_cast<const uint4*>(a.w + (size_t)row * a.D);
      float acc[TB];
#pragma unroll
      for (int tt = 0; tt < TB; ++tt) acc[tt] = 0.f;
      for (int c0 = 0; c0 < nch; c0 += 256) {
        uint4 v[8];
        if (row == row0 && c0 == 0 && t0 == 0) {
#pragma unroll
          for (int u = 0; u < 8; ++u) v[u] = pre[u];
        } else {
#pragma unroll
          for (int u = 0; u < 8; ++u) {
            const int c = c0 + u * 32 + lane;
            v[u] = c < nch ? ldg_stream(rp + c) : make_uint4(0, 0, 0, 0);
          }
        }
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const int c = c0 + u * 32 + lane;
          if (c < nch) {
            const float w0 = bf16lo(v[u].x), w1 = bf16hi(v[u].x), w2 = bf16lo(v[u].y), w3 = bf16hi(v[u].y);
            const float w4 = bf16lo(v[u].z), w5 = bf16hi(v[u].z), w6 = bf16lo(v[u].w), w7 = bf16hi(v[u].w);
#pragma unroll
            for (int tt = 0; tt < TB; ++tt) {
              const float4* xv = reinterpret_cast<const float4*>(xs + tt * a.D_pad8 + c * 8);
              const float4 xa = xv[0], xb = xv[1];
              float r = acc[tt];
              r = fmaf(w0, xa.x, r); r = fmaf(w1, xa.y, r); r = fmaf(w2, xa.z, r); r = fmaf(w3, xa.w, r);
              r = fmaf(w4, xb.x, r); r = fmaf(w5, xb.y, r); r = fmaf(w6, xb.z, r); r = fmaf(w7, xb.w, r);
              acc[tt] = r;
            }
          }
        }
      }
#pragma unroll
      for (int tt = 0; tt < TB; ++tt) acc[tt] = warp_sum(acc[tt]);
      if (lane == 0)
#pragma unroll
        for (int tt = 0; tt < TB; ++tt)
          if (tt < tb) a.logits[(size_t)(t0 + tt) * a.E + row] = acc[tt];
    }
  }
  __syncthreads();
  __threadfence();
  pdl_trigger();   // only now: the next kernels read x and the logits in their prologues
}

// ---------------------------------------------------------------------------
// Decode-mode router: first kernel of the chain.  It lets the projection
// kernel launch at once, then routes while the memory system is still idle
// (the logits load is not queued behind the basis streams) and publishes the
// routing with a release flag that the gate/up and down kernels wait on.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kThreads) k_route_publish(Fwd p) {
  if (threadIdx.x == 0) {   // before the trigger: no later kernel may see the previous call's flag
    p.status[0] = 0;
    p.route_flag[0] = 0;
    __threadfence();
  }
  __syncthreads();
  pdl_trigger();
  extern __shared__ uint32_t smem_rp[];
  const RouteView rv = route_block(p, smem_rp);
  for (int i = threadIdx.x; i < p.P; i += blockDim.x) {
    p.pair_expert[i] = rv.pe[i];
    p.pair_weight[i] = rv.pw[i];
    p.pair_list[i] = rv.plist[i];
  }
  for (int i = threadIdx.x; i <= p.E; i += blockDim.x) {
    if (i < p.E) p.expert_count[i] = rv.cnt[i];
    p.expert_start[i] = rv.start[i];
    p.active[i] = rv.act[i];
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    st_release(p.route_flag, 1);
  }
}

// ---------------------------------------------------------------------------
// K0: routing.  k largest logits per token (ties to the lower expert index),
// gate weights = softmax over the selected k, then a stable grouping of the
// (token, slot) pairs p = t * k + slot by expert.  Blocks select for tpb
// tokens each; the last block to finish (a counter in the workspace, which it
// resets) groups all pairs and publishes the routing with a release flag.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(1024) k_router(Fwd p) {
  if (blockIdx.x == 0 && threadIdx.x == 0) {   // before the trigger: no later kernel may see the previous flag
    p.status[0] = 0;
    p.route_flag[0] = 0;
    __threadfence();
  }
  __syncthreads();
  pdl_trigger();
  // shared: keys [tpb][E] | pair expert [P] | count [E] | start [E+1]
  extern __shared__ uint32_t keys[];
  __shared__ int last;
  const int E = p.E, k = p.k, T = p.T, P = p.P;
  const int tid = threadIdx.x;
  const int tpb = max(1, (int)blockDim.x / E);
  {   // this block's tokens
    const int tt = tid / E, e = tid - tt * E, t = blockIdx.x * tpb + tt;
    const bool valid = tt < tpb && t < T;
    float lg = 0.f;
    if (valid) {
      lg = p.logits[(size_t)t * E + e];
      keys[tt * E + e] = order_key(lg);
    }
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
        reinterpret_cast<float*>(keys)[tpb * E + tt * k + rank] = lg;   // logits of the selected, in rank order
      }
    }
    __syncthreads();
    for (int q = tid; q < tpb * k; q += blockDim.x) {   // softmax over the k selected of each token
      const int t2 = blockIdx.x * tpb + q / k, r = q - (q / k) * k;
      if (t2 >= T) continue;
      const float* w = reinterpret_cast<const float*>(keys) + tpb * E + (q / k) * k;
      const float m = w[0];
      float sum = 0.f;
      for (int r2 = 0; r2 < k; ++r2) sum += expf(w[r2] - m);
      p.pair_weight[t2 * k + r] = expf(w[r] - m) * (1.f / sum);
    }
  }
  __syncthreads();
  if (tid == 0) {
    __threadfence();
    const int old = atomicAdd(p.status + 2, 1);
    last = old == (int)gridDim.x - 1;
    if (last) p.status[2] = 0;   // reset for the next call
  }
  __syncthreads();
  if (!last) return;
  __threadfence();
  int* s_pe = reinterpret_cast<int*>(keys);   // reuse: all pairs' experts
  int* s_cnt = s_pe + P;
  int* s_start = s_cnt + E;
  for (int q = tid; q < P; q += blockDim.x) s_pe[q] = __ldcg(p.pair_expert + q);
  __syncthreads();
  const int warp = tid >> 5, lane = tid & 31, nw = blockDim.x >> 5;
  for (int e = warp; e < E; e += nw) {
    int c = 0;
    for (int q0 = 0; q0 < P; q0 += 32) {
      const int q = q0 + lane;
      c += __popc(__ballot_sync(0xFFFFFFFFu, q < P && s_pe[q] == e));
    }
    if (lane == 0) s_cnt[e] = c;
  }
  __syncthreads();
  if (warp == 0) {
    int run = 0, act = 0;
    for (int e0 = 0; e0 < E; e0 += 32) {
      const int e = e0 + lane;
      const int c = e < E ? s_cnt[e] : 0;
      int incl = c;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int v = __shfl_up_sync(0xFFFFFFFFu, incl, o);
        if (lane >= o) incl += v;
      }
      if (e < E) {
        s_start[e] = run + incl - c;
        p.expert_start[e] = run + incl - c;
        p.expert_count[e] = c;
      }
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
    int base = s_start[e];
    for (int q0 = 0; q0 < P; q0 += 32) {
      const int q = q0 + lane;
      const bool m = q < P && s_pe[q] == e;
      const unsigned b = __ballot_sync(0xFFFFFFFFu, m);
      if (m) p.pair_list[base + __popc(b & ((1u << lane) - 1u))] = q;
      base += __popc(b);
    }
  }
  __syncthreads();
  if (tid == 0) {   // the routing is published: kernels that stage by it may go on
    __threadfence();
    st_release(p.route_flag, 1);
  }
}

// ---------------------------------------------------------------------------
// L2 prefetch of what the later phases read: gate/up then down factors of the
// routed experts, then Phi_dn.  Range r goes to block r % gridDim (warp 0);
// its 32 lanes split it into 16-byte-aligned pieces.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void prefetch_range(const uint8_t* base, uint64_t beg, uint64_t end, int lane) {
  uint64_t piece = (((end - beg) + 31) / 32 + 15) & ~15ull;   // 16-byte multiple
  if (piece < 4096) piece = 4096;
  uint64_t o = beg + (uint64_t)lane * piece;
  const uint64_t stop = end < o + piece ? end : o + piece;
  while (o < stop) {
    const uint64_t c = stop - o < (1u << 19) ? stop - o : (1u << 19);
    prefetch_l2(base + o, (uint32_t)c);
    o += c;
  }
}

__device__ void prefetch_for_experts(const Fwd& p) {
  if (threadIdx.x >= 32) return;
  const int lane = threadIdx.x;
  const int A = p.active[0];
  const int nr = 3 * A + 1;
  const uint64_t bo = (uint64_t)((const uint8_t*)p.basis_out - p.img);
  uint64_t budget = kPrefetchCap;
  for (int r = 0; r < nr; ++r) {
    uint64_t beg, end;
    if (r < 3 * A) {
      const int h = r / A, a = r - h * A;
      const ExpertDesc& xd = p.desc[h * p.E + p.active[1 + a]];
      beg = xd.begin;
      end = xd.end;
    } else {
      beg = bo;
      end = bo + (uint64_t)p.D * p.n_pad * 2;
    }
    if (end - beg > budget) end = beg + budget;
    budget -= end - beg;
    if ((int)(r % gridDim.x) == (int)blockIdx.x && end > beg) prefetch_range(p.img, beg, end, lane);
    if (!budget) break;
  }
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
  uint4 pre[8];
  const bool have_pre = gw < nrows;
  if (have_pre) {   // the warp's first row batch: issued before anything it waits on
    const uint4* rp = reinterpret_cast<const uint4*>(mat + (size_t)gw * ld);
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const int c = u * 32 + lane;
      pre[u] = c < nch ? ldg_stream(rp + c) : make_uint4(0, 0, 0, 0);
    }
  }
  if (PROJ) {
    if (p.decode && blockIdx.x == 0 && threadIdx.x == 0) *p.status = 0;
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
        if (have_pre && t0 == 0 && row == gw && c0 == 0) {
#pragma unroll
          for (int u = 0; u < 8; ++u) v[u] = pre[u];
        } else {
#pragma unroll
          for (int u = 0; u < 8; ++u) {
            const int c = c0 + u * 32 + lane;
            v[u] = c < nch ? ldg_stream(rp + c) : make_uint4(0, 0, 0, 0);
          }
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
              p.y[(size_t)t * p.D + row] = p.accum ? p.y[(size_t)t * p.D + row] + acc[tt] : acc[tt];
            }
          }
        }
      }
    }
  }
  if (PROJ && !p.decode) {
    pdl_wait();
    prefetch_for_experts(p);
  }
}

// ---------------------------------------------------------------------------
// K1 / K4, bulk-copy form: one block per SM owns a contiguous range of rows and
// streams it through a two-stage shared-memory ring filled by cp.async.bulk
// (one copy per stage), so few registers are held and the row bytes are in
// flight from the block's first instructions (K4 issues its first stages before
// waiting for the down kernel).  Warps take rows of a stage round-robin.
// ---------------------------------------------------------------------------
template <int TB, bool PROJ>
__global__ void __launch_bounds__(kThreads) k_gemv_bulk(Fwd p, int stage_rows) {
  pdl_trigger();
  extern __shared__ int4 smem_gb[];
  const int ld = PROJ ? p.D_pad : p.n_pad;
  const int nrows = PROJ ? 2 * p.n : p.D;
  const uint32_t row_bytes = (uint32_t)ld * 2;
  const uint16_t* mat = PROJ ? p.basis_in : p.basis_out;
  uint8_t* ring = reinterpret_cast<uint8_t*>(smem_gb);                          // [2][stage_rows][ld] bf16
  float* vs = reinterpret_cast<float*>(ring + 2 * (size_t)stage_rows * row_bytes);   // [TB][ld]
  uint64_t* bars = reinterpret_cast<uint64_t*>(vs + (size_t)TB * ld);             // [2]
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const int per = (nrows + gridDim.x - 1) / gridDim.x;
  const int r0 = min(nrows, blockIdx.x * per), r1 = min(nrows, r0 + per);
  const int nst = (r1 - r0 + stage_rows - 1) / stage_rows;
  auto issue = [&](int st) {
    const int a = r0 + st * stage_rows, b = min(r1, a + stage_rows);
    uint64_t* bar = bars + (st & 1);
    mbar_expect_tx(bar, (uint32_t)(b - a) * row_bytes);
    bulk_g2s(ring + (size_t)(st & 1) * stage_rows * row_bytes, mat + (size_t)a * ld, (uint32_t)(b - a) * row_bytes, bar);
  };
  if (threadIdx.x == 0) {
    mbar_init(bars);
    mbar_init(bars + 1);
    for (int st = 0; st < min(2, nst); ++st) issue(st);
  }
  if (PROJ) {
    const size_t ng = (size_t)p.P * 2 * p.I_pad / 4, ns = (size_t)p.T * p.n_pad / 4;
    const float4 z4 = make_float4(0.f, 0.f, 0.f, 0.f);
    for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < ng + ns; i += (size_t)gridDim.x * blockDim.x) {
      if (i < ng) reinterpret_cast<float4*>(p.gu)[i] = z4;
      else reinterpret_cast<float4*>(p.s)[i - ng] = z4;
    }
  } else {
    pdl_wait();
  }
  bool ok = true;
  int uses[2] = {0, 0};   // completed phases of each ring buffer (uniform across the block)
  for (int t0 = 0; t0 < p.T; t0 += TB) {
    const int tb = min(TB, p.T - t0);
    __syncthreads();   // every stage of the previous token batch has been consumed
    if (t0 > 0 && threadIdx.x == 0)
      for (int st = 0; st < min(2, nst); ++st) issue(st);
    // stage the vectors: 8 independent loads per thread in flight at a time
    for (int i0 = threadIdx.x; i0 < TB * ld; i0 += 8 * blockDim.x) {
      float v[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int i = i0 + u * blockDim.x;
        const int tt = i / ld, c = i - tt * ld;
        v[u] = 0.f;
        if (i < TB * ld && tt < tb) {
          if (PROJ) {
            if (c < p.D) v[u] = __uint_as_float((uint32_t)p.x[(size_t)(t0 + tt) * p.D + c] << 16);
          } else {
            if (c < p.n) v[u] = p.s[(size_t)(t0 + tt) * p.n_pad + c];
          }
        }
      }
#pragma unroll
      for (int u = 0; u < 8; ++u)
        if (i0 + u * blockDim.x < TB * ld) vs[i0 + u * blockDim.x] = v[u];
    }
    __syncthreads();
    for (int st = 0; st < nst; ++st) {
      const uint32_t parity = (uint32_t)uses[st & 1] & 1u;
      ++uses[st & 1];
      if (!mbar_wait(bars + (st & 1), parity)) {
        if (threadIdx.x == 0) atomicCAS(p.status, 0, BITSMOE_ERR_TIMEOUT);
        ok = false;
        break;
      }
      const int a = r0 + st * stage_rows, b = min(r1, a + stage_rows);
      const uint8_t* buf = ring + (size_t)(st & 1) * stage_rows * row_bytes;
      for (int row = a + wid; row < b; row += kWarps) {
        const uint8_t* rp = buf + (size_t)(row - a) * row_bytes;
        float acc[TB];
#pragma unroll
        for (int tt = 0; tt < TB; ++tt) acc[tt] = 0.f;
        for (int c = lane; c < (ld >> 3); c += 32) {
          const uint4 v = lds128(rp + (size_t)c * 16);
          const float w0 = bf16lo(v.x), w1 = bf16hi(v.x), w2 = bf16lo(v.y), w3 = bf16hi(v.y);
          const float w4 = bf16lo(v.z), w5 = bf16hi(v.z), w6 = bf16lo(v.w), w7 = bf16hi(v.w);
#pragma unroll
          for (int tt = 0; tt < TB; ++tt) {
            const float4* xv = reinterpret_cast<const float4*>(vs + tt * ld + c * 8);
            const float4 xa = xv[0], xb = xv[1];
            float r = acc[tt];
            r = fmaf(w0, xa.x, r); r = fmaf(w1, xa.y, r); r = fmaf(w2, xa.z, r); r = fmaf(w3, xa.w, r);
            r = fmaf(w4, xb.x, r); r = fmaf(w5, xb.y, r); r = fmaf(w6, xb.z, r); r = fmaf(w7, xb.w, r);
            acc[tt] = r;
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
                p.y[(size_t)t * p.D + row] = p.accum ? p.y[(size_t)t * p.D + row] + acc[tt] : acc[tt];
              }
            }
          }
        }
      }
      __syncthreads();   // stage consumed: refill its buffer with stage st + 2
      if (threadIdx.x == 0 && st + 2 < nst) issue(st + 2);
    }
    if (!ok) break;
  }
  if (PROJ && !p.decode) {
    pdl_wait();
    prefetch_for_experts(p);
  }
  if (PROJ && p.decode) pdl_wait();   // (a preceding kernel, if any, completes before this grid)
}

// ---------------------------------------------------------------------------
// K2: gate/up factors.  out[i] = sum_j alpha_j z_j p_hat_ij
//                             = sum_j c_jg (q_ij - zero_jg),  c_jg = alpha_j z_j s_jg
// A warp item is (routed expert, projection, 128-row block, segment of tiles).
// The lane owns 4 rows; c of the segment's units is quantised to int16 with
// one scale per (item, token), so the inner loop is dp2a over unpacked code
// bytes; the zero-point term sum_j c_jg zero_jg is applied once per item.
//
// K3: down factor.  h = SiLU(gate) * up for the block's rows (quantised to
// int16 with one scale per token), then per unit j (one per lane):
//   d_j = sum_g s_jg (sum_{i in g} q_ij h_i - zero_jg * sum_{i in g} h_i)
//   s[t][j] += w_(t,e) * alpha_j * d_j
// A block item is (routed expert, one UL tile per warp, a chunk of row blocks).
// ---------------------------------------------------------------------------

// scale/zero of group g of the lane's unit: sz[(g - szg0) * szstride + szcol]
template <int B, int G, int TB, bool SH = false>
__device__ __forceinline__ void ul_tile(const Fwd& p, const uint8_t* code, int rb0, int rb1, const int16_t* hq,
                                        int hstride, const int* Hg, const uint32_t* sz, int szstride, int szg0,
                                        int szcol, float (&accf)[TB]) {
  constexpr int C = ul_chunks(B);
  const int gshift = 31 - __clz(p.group);
  const int tstride = hstride / 2;
  for (int rb = rb0; rb < rb1; ++rb) {
    const int* hq32 = reinterpret_cast<const int*>(hq + (rb - rb0) * kRows);
    const uint8_t* cb = code + (size_t)(rb - rb0) * C * kChunkBytes;
    if (B == 16) {
#pragma unroll 4
      for (int c = 0; c < 16; ++c) {
        const uint4 v = ld128<SH>(cb + (size_t)c * kChunkBytes);
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
    for (int c = 0; c < C; ++c) v[c] = ld128<SH>(cb + (size_t)c * kChunkBytes);
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
      const uint32_t szw = sz[(size_t)(gfirst + g - szg0) * szstride + szcol];
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

// ---------------------------------------------------------------------------
// Decode mode (small T): the gate/up and down kernels compute the routing
// themselves from the logits, then, in the PDL prologue that overlaps the
// previous kernel, stage their packed codes into shared memory with bulk
// copies and their per-unit metadata into registers.  After
// griddepcontrol.wait only the data dependency (z, gate/up) remains.
// ---------------------------------------------------------------------------
constexpr int kK2DecWarps = 4;
constexpr int kDecMaxT = 8;        // decode mode: at most this many tokens
constexpr int kZ = 12;             // item slots per lane whose z values are gathered at once
constexpr int kK3DecWarps = 4;

template <int G, int TB>
__global__ void __launch_bounds__(kK2DecWarps * 32) k_gateup_dec(Fwd p) {
  pdl_trigger();
  extern __shared__ int4 smem_k2d[];
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const int smax = p.s16 - 8;                      // slots of the largest item, multiple of 8
  const size_t per_warp = (size_t)p.seg_bytes + (size_t)smax * 4 * (2 + G) + (size_t)G * TB * p.s16 * 2 + 16;
  uint8_t* codes = reinterpret_cast<uint8_t*>(smem_k2d) + wid * per_warp;
  int* su = reinterpret_cast<int*>(codes + p.seg_bytes);           // unit index per local slot
  float* sa = reinterpret_cast<float*>(su + smax);                 // alpha
  uint32_t* ssz = reinterpret_cast<uint32_t*>(sa + smax);          // [G][smax] scale | zero << 16
  int16_t* cq = reinterpret_cast<int16_t*>(ssz + G * smax);        // [G][TB][s16]
  uint64_t* bar = reinterpret_cast<uint64_t*>(codes + per_warp - 16);
  const int per_e = 2 * p.NRB * p.nseg;
  const int item = blockIdx.x * kK2DecWarps + wid;
  const int a = item / per_e;
  // the routing, published by the projection kernel's first block
  if (!wait_flag(p.route_flag)) {
    if (lane == 0) atomicCAS(p.status, 0, BITSMOE_ERR_TIMEOUT);
    pdl_wait();
    return;
  }
  const int A = p.active[0];
  const int e_raw = p.active[1 + min(a, p.E - 1)];
  // every warp waits for the previous kernel before it exits, so that this
  // grid completes only after it (PDL completion is then transitive)
  if (item >= A * per_e) {
    pdl_wait();
    return;
  }
  int r = item - a * per_e;
  const int h = r / (p.NRB * p.nseg);
  r -= h * p.NRB * p.nseg;
  const int rb = r / p.nseg, sg = r - rb * p.nseg;
  const int e = e_raw;
  const ExpertDesc& xd = p.desc[h * p.E + e];
  const ItemRec it = p.items[((size_t)h * p.E + e) * p.nseg + sg];
  const int ntok = p.expert_count[e], pst = p.expert_start[e];
  if (it.nr == 0 || (p.tc_min > 0 && ntok >= p.tc_min)) {   // empty, or the tensor-core kernels' expert
    pdl_wait();
    return;
  }
  const int g_base = (rb * kRows) / p.group;
  if (lane == 0) {
    const uint32_t mb = (uint32_t)it.nslot * 4;
    mbar_init(bar);
    mbar_expect_tx(bar, it.bytes + (2 + G) * mb);
    bulk_g2s(codes, p.img + xd.code_base + (size_t)rb * xd.rb_stride + it.byte0, it.bytes, bar);
    bulk_g2s(su, p.img + xd.unit_off + (size_t)it.slot0 * 4, mb, bar);
    bulk_g2s(sa, p.img + xd.alpha_off + (size_t)it.slot0 * 4, mb, bar);
#pragma unroll
    for (int gl = 0; gl < G; ++gl)
      bulk_g2s(ssz + gl * smax, p.img + xd.sz_off + ((size_t)(g_base + gl) * xd.nslots + it.slot0) * 4, mb, bar);
  }
  int plist[kDecMaxT];   // the expert's (token, slot) pairs
#pragma unroll
  for (int q = 0; q < kDecMaxT; ++q) plist[q] = q < ntok ? p.pair_list[pst + q] : 0;
  pdl_wait();
  // ranges: consecutive buckets, quantised ones first, 16-bit last
  int nls = 0;
  for (int q = 0; q < it.nr; ++q)
    if (it.bits[q] < 16) nls += it.ntl[q] * rl_units(it.bits[q]);
  const int gl_lane = G == 1 ? 0 : (4 * lane) / p.group;
  const int tstride = p.s16 / 2;
  if (!mbar_wait(bar, 0)) {
    if (lane == 0) atomicCAS(p.status, 0, BITSMOE_ERR_TIMEOUT);
    mbar_wait(bar, 0);
    return;
  }
  for (int tb0 = 0; tb0 < ntok; tb0 += TB) {
    const int tb = min(TB, ntok - tb0);
    int pair[TB];
    const float* zrow[TB];
#pragma unroll
    for (int tt = 0; tt < TB; ++tt) {
      const int q = tb0 + min(tt, tb - 1);
      int pv = plist[0];
#pragma unroll
      for (int u = 1; u < kDecMaxT; ++u)
        if (u == q) pv = plist[u];
      if (q >= kDecMaxT) pv = p.pair_list[pst + q];   // more tokens than the prologue held
      pair[tt] = pv;
      zrow[tt] = p.z + ((size_t)h * p.T + pair[tt] / p.k) * p.n_pad;
    }
    // c = alpha * z * scale per (slot, group, token): int16 with one scale per token.
    // The z gathers are issued together (one L2 round trip): kZ slots per lane.
    const bool fast = nls <= 32 * kZ;
    float zr[kZ][TB];
    if (fast) {
#pragma unroll
      for (int m = 0; m < kZ; ++m) {
        const int i = lane + 32 * m;
        const int j = i < nls ? su[i] : 0;
#pragma unroll
        for (int tt = 0; tt < TB; ++tt) zr[m][tt] = i < nls ? zrow[tt][j] : 0.f;
      }
#pragma unroll
      for (int m = 0; m < kZ; ++m) {
        const int i = lane + 32 * m;
        const float al = i < nls ? sa[i] : 0.f;
#pragma unroll
        for (int tt = 0; tt < TB; ++tt) zr[m][tt] *= al;
      }
    }
    float mx[TB];
#pragma unroll
    for (int tt = 0; tt < TB; ++tt) mx[tt] = 0.f;
    if (fast) {
#pragma unroll
      for (int m = 0; m < kZ; ++m) {
        const int i = lane + 32 * m;
        if (i < nls) {
#pragma unroll
          for (int gl = 0; gl < G; ++gl) {
            const float sc = __half2float(__ushort_as_half((unsigned short)(ssz[gl * smax + i] & 0xFFFFu)));
#pragma unroll
            for (int tt = 0; tt < TB; ++tt) mx[tt] = fmaxf(mx[tt], fabsf(zr[m][tt] * sc));
          }
        }
      }
    } else {
      for (int i = lane; i < nls; i += 32) {
        const int j = su[i];
        const float al = sa[i];
#pragma unroll
        for (int tt = 0; tt < TB; ++tt) {
          const float zv = al * zrow[tt][j];
#pragma unroll
          for (int gl = 0; gl < G; ++gl)
            mx[tt] = fmaxf(mx[tt], fabsf(zv * __half2float(__ushort_as_half((unsigned short)(ssz[gl * smax + i] & 0xFFFFu)))));
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
    float corr[G][TB];
#pragma unroll
    for (int gl = 0; gl < G; ++gl)
#pragma unroll
      for (int tt = 0; tt < TB; ++tt) corr[gl][tt] = 0.f;
    if (fast) {
#pragma unroll
      for (int m = 0; m < kZ; ++m) {
        const int i = lane + 32 * m;
        if (i < nls) {
#pragma unroll
          for (int gl = 0; gl < G; ++gl) {
            const uint32_t w = ssz[gl * smax + i];
            const float sc = __half2float(__ushort_as_half((unsigned short)(w & 0xFFFFu)));
            const float zp = __half2float(__ushort_as_half((unsigned short)(w >> 16)));
#pragma unroll
            for (int tt = 0; tt < TB; ++tt) {
              const int ci = __float2int_rn(zr[m][tt] * sc * inv[tt]);
              cq[(size_t)(gl * TB + tt) * p.s16 + i] = (int16_t)ci;
              corr[gl][tt] = fmaf((float)ci, zp, corr[gl][tt]);
            }
          }
        }
      }
    } else {
      for (int i = lane; i < nls; i += 32) {
        const int j = su[i];
        const float al = sa[i];
#pragma unroll
        for (int tt = 0; tt < TB; ++tt) {
          const float zv = al * zrow[tt][j];
#pragma unroll
          for (int gl = 0; gl < G; ++gl) {
            const uint32_t w = ssz[gl * smax + i];
            const float sc = __half2float(__ushort_as_half((unsigned short)(w & 0xFFFFu)));
            const float zp = __half2float(__ushort_as_half((unsigned short)(w >> 16)));
            const int ci = __float2int_rn(zv * sc * inv[tt]);
            cq[(size_t)(gl * TB + tt) * p.s16 + i] = (int16_t)ci;
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
    float accf[4][TB], acc16[4][TB];
#pragma unroll
    for (int w = 0; w < 4; ++w)
#pragma unroll
      for (int tt = 0; tt < TB; ++tt) accf[w][tt] = acc16[w][tt] = 0.f;
    const int* cq32 = reinterpret_cast<const int*>(cq + (size_t)gl_lane * TB * p.s16);
    uint32_t boff = 0;
    int ls = 0;
    for (int q = 0; q < it.nr; ++q) {
      const int b = it.bits[q], ntl = it.ntl[q];
      const uint8_t* code = codes + boff + lane * 16;
      const int* cp = cq32 + ls / 2;
      switch (b) {
        case 1: rl_range<1, TB, true>(code, ntl, cp, tstride, accf); break;
        case 2: rl_range<2, TB, true>(code, ntl, cp, tstride, accf); break;
        case 3: rl_range<3, TB, true>(code, ntl, cp, tstride, accf); break;
        case 4: rl_range<4, TB, true>(code, ntl, cp, tstride, accf); break;
        case 6: rl_range<6, TB, true>(code, ntl, cp, tstride, accf); break;
        case 8: rl_range<8, TB, true>(code, ntl, cp, tstride, accf); break;
        default: rl_range16<TB, true>(code, ntl, su + ls, sa + ls, zrow, acc16); break;
      }
      boff += (uint32_t)ntl * rl_chunks(b) * kChunkBytes;
      ls += ntl * rl_units(b);
    }
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

template <int G, int TB>
__global__ void __launch_bounds__(kK3DecWarps * 32) k_down_dec(Fwd p) {
  pdl_trigger();
  extern __shared__ int4 smem_k3d[];
  const int rbc = p.rbc;
  const int nrows_max = rbc * kRows;
  const int gshift = 31 - __clz(p.group);
  const int ngc_max = max(1, nrows_max >> gshift);
  float* hf = reinterpret_cast<float*>(smem_k3d);                      // [TB][nrows_max]
  int16_t* hq = reinterpret_cast<int16_t*>(hf + TB * nrows_max);       // [TB][nrows_max]
  int* Hg = reinterpret_cast<int*>(hq + TB * nrows_max);               // [TB][64]
  float* red = reinterpret_cast<float*>(Hg + TB * 64);                 // [warps][TB]
  float* shs = red + kK3DecWarps * TB;                                 // [TB], padded to 4
  const size_t per_warp = (size_t)p.ul_bytes + (size_t)ngc_max * 32 * 4 + 16;
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  uint8_t* codes = reinterpret_cast<uint8_t*>(shs + ((TB + 3) & ~3)) + wid * per_warp;
  uint32_t* szs = reinterpret_cast<uint32_t*>(codes + p.ul_bytes);
  uint64_t* bar = reinterpret_cast<uint64_t*>(codes + per_warp - 16);
  const int ntg = (p.ul_max_tiles + kK3DecWarps - 1) / kK3DecWarps;
  const int nrc = (p.NRB + rbc - 1) / rbc;
  const int item = blockIdx.x;
  const int a = item / (ntg * nrc);
  if (!wait_flag(p.route_flag)) {   // the routing, published by the projection kernel
    if (threadIdx.x == 0) atomicCAS(p.status, 0, BITSMOE_ERR_TIMEOUT);
    pdl_wait();
    return;
  }
  const int A = p.active[0];
  const int e = p.active[1 + min(a, p.E - 1)];
  if (item >= A * ntg * nrc) {   // wait before exiting: keeps PDL completion transitive
    pdl_wait();
    return;
  }
  const int r = item - a * ntg * nrc;
  const int tg = r / nrc, rc = r - tg * nrc;
  const ExpertDesc& xd = p.desc[2 * p.E + e];
  if (tg * kK3DecWarps >= xd.ntiles || (p.tc_min > 0 && p.expert_count[e] >= p.tc_min)) {
    pdl_wait();
    return;
  }
  const int rb0 = rc * rbc, rb1 = min(p.NRB, rb0 + rbc);
  const int row0 = rb0 * kRows, nrows = (rb1 - rb0) * kRows;
  const int tile = tg * kK3DecWarps + wid;
  int bi = -1;
  if (tile < xd.ntiles)
    for (int q = 0; q < xd.nbk; ++q)
      if (tile >= xd.bk[q].tile0 && tile < xd.bk[q].tile0 + xd.bk[q].ntiles) bi = q;
  int j = 0, bs = 0, szg0 = 0;
  float al = 0.f;
  if (bi >= 0) {
    const BucketDesc& bd = xd.bk[bi];
    const uint32_t nb = (uint32_t)(rb1 - rb0) * ul_chunks(bd.bits) * kChunkBytes;
    if (lane == 0)
      stage_bytes(codes,
                  p.img + xd.code_base + bd.code_off +
                      ((size_t)(tile - bd.tile0) * p.NRB + rb0) * ul_chunks(bd.bits) * kChunkBytes,
                  nb, bar);
    bs = (tile - bd.tile0) * 32 + lane;
    const int gs = bd.slot0 + bs;
    j = reinterpret_cast<const int32_t*>(p.img + xd.unit_off)[gs];
    al = reinterpret_cast<const float*>(p.img + xd.alpha_off)[gs];
    szg0 = row0 >> gshift;
    if (bd.bits < 16) {
      const uint32_t* sz = reinterpret_cast<const uint32_t*>(p.img + bd.sz_off);
      const int g1 = min(p.NG, ((rb1 * kRows - 1) >> gshift) + 1);
      for (int g0 = szg0; g0 < g1; g0 += 8) {   // 8 loads in flight at a time
        uint32_t v[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) v[u] = g0 + u < g1 ? sz[(size_t)(g0 + u) * xd.nslots + bs] : 0u;
#pragma unroll
        for (int u = 0; u < 8; ++u)
          if (g0 + u < g1) szs[(g0 + u - szg0) * 32 + lane] = v[u];
      }
    }
  }
  const int ntok = p.expert_count[e], pst = p.expert_start[e];
  int plist[kDecMaxT];
  float pwt[kDecMaxT];
#pragma unroll
  for (int q = 0; q < kDecMaxT; ++q) plist[q] = q < ntok ? p.pair_list[pst + q] : 0;
#pragma unroll
  for (int q = 0; q < kDecMaxT; ++q) pwt[q] = q < ntok ? p.pair_weight[plist[q]] : 0.f;
  pdl_wait();
  bool staged = false;
  constexpr int kMaxRowsPerThread = kK3MaxRB * kRows / (kK3DecWarps * 32);
  for (int tb0 = 0; tb0 < ntok; tb0 += TB) {
    const int tb = min(TB, ntok - tb0);
    __syncthreads();   // previous batch finished with hq / Hg
    for (int i = threadIdx.x; i < TB * 64; i += blockDim.x) Hg[i] = 0;
    // h = SiLU(gate) * up for this block's rows, kept in registers
    float hv[kMaxRowsPerThread][TB];
    float mx[TB];
#pragma unroll
    for (int tt = 0; tt < TB; ++tt) mx[tt] = 0.f;
#pragma unroll
    for (int m = 0; m < kMaxRowsPerThread; ++m) {
      const int i = threadIdx.x + m * kK3DecWarps * 32;
#pragma unroll
      for (int tt = 0; tt < TB; ++tt) {
        float v = 0.f;
        if (i < nrows && tt < tb) {
          int pr = plist[0];
#pragma unroll
          for (int u = 1; u < kDecMaxT; ++u)
            if (u == tb0 + tt) pr = plist[u];
          if (tb0 + tt >= kDecMaxT) pr = p.pair_list[pst + tb0 + tt];
          const float g = p.gu[((size_t)pr * 2) * p.I_pad + row0 + i];
          const float u = p.gu[((size_t)pr * 2 + 1) * p.I_pad + row0 + i];
          v = g / (1.f + __expf(-g)) * u;
        }
        hv[m][tt] = v;
        mx[tt] = fmaxf(mx[tt], fabsf(v));
      }
    }
#pragma unroll
    for (int tt = 0; tt < TB; ++tt) {
      const float m = warp_max(mx[tt]);
      if (lane == 0) red[wid * TB + tt] = m;
    }
    __syncthreads();
    float scale[TB];
#pragma unroll
    for (int tt = 0; tt < TB; ++tt) {
      float m = 0.f;
#pragma unroll
      for (int w = 0; w < kK3DecWarps; ++w) m = fmaxf(m, red[w * TB + tt]);
      scale[tt] = m;
      const float inv = m > 0.f ? 32767.f / m : 0.f;
#pragma unroll
      for (int mm = 0; mm < kMaxRowsPerThread; ++mm) {
        const int i = threadIdx.x + mm * kK3DecWarps * 32;
        if (i < nrows) {
          const int q = __float2int_rn(hv[mm][tt] * inv);
          hq[tt * nrows_max + i] = (int16_t)q;
          // a warp's 32 consecutive rows lie in one group (group >= 32)
          int sq = q;
#pragma unroll
          for (int o = 16; o; o >>= 1) sq += __shfl_xor_sync(0xFFFFFFFFu, sq, o);
          if (lane == 0) atomicAdd(&Hg[tt * 64 + (i >> gshift)], sq);
        }
      }
    }
    if (threadIdx.x == 0)
#pragma unroll
      for (int tt = 0; tt < TB; ++tt) shs[tt] = scale[tt];
    __syncthreads();
    if (bi < 0) continue;
    if (!staged) {
      if (!mbar_wait(bar, 0)) {
        if (lane == 0) atomicCAS(p.status, 0, BITSMOE_ERR_TIMEOUT);
        mbar_wait(bar, 0);
        bi = -1;
        continue;
      }
      staged = true;
    }
    const BucketDesc& bd = xd.bk[bi];
    const uint8_t* code = codes + lane * 16;
    float accf[TB];
#pragma unroll
    for (int tt = 0; tt < TB; ++tt) accf[tt] = 0.f;
    switch (bd.bits) {
      case 1: ul_tile<1, G, TB, true>(p, code, rb0, rb1, hq, nrows_max, Hg, szs, 32, szg0, lane, accf); break;
      case 2: ul_tile<2, G, TB, true>(p, code, rb0, rb1, hq, nrows_max, Hg, szs, 32, szg0, lane, accf); break;
      case 3: ul_tile<3, G, TB, true>(p, code, rb0, rb1, hq, nrows_max, Hg, szs, 32, szg0, lane, accf); break;
      case 4: ul_tile<4, G, TB, true>(p, code, rb0, rb1, hq, nrows_max, Hg, szs, 32, szg0, lane, accf); break;
      case 6: ul_tile<6, G, TB, true>(p, code, rb0, rb1, hq, nrows_max, Hg, szs, 32, szg0, lane, accf); break;
      case 8: ul_tile<8, G, TB, true>(p, code, rb0, rb1, hq, nrows_max, Hg, szs, 32, szg0, lane, accf); break;
      default: ul_tile<16, G, TB, true>(p, code, rb0, rb1, hq, nrows_max, Hg, szs, 32, szg0, lane, accf); break;
    }
    if (al != 0.f) {
#pragma unroll
      for (int tt = 0; tt < TB; ++tt) {
        if (tt < tb) {
          int pr = plist[0];
          float wv = pwt[0];
#pragma unroll
          for (int u = 1; u < kDecMaxT; ++u)
            if (u == tb0 + tt) {
              pr = plist[u];
              wv = pwt[u];
            }
          if (tb0 + tt >= kDecMaxT) {
            pr = p.pair_list[pst + tb0 + tt];
            wv = p.pair_weight[pr];
          }
          const float scale = shs[tt] * (1.f / 32767.f);
          atomicAdd(p.s + (size_t)(pr / p.k) * p.n_pad + j, wv * al * scale * accf[tt]);
        }
      }
    }
  }
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
#ifndef BITSMOE_DECODE_MAX_TOKENS
#define BITSMOE_DECODE_MAX_TOKENS 8
#endif
// Tokens from which an expert's factors use the tensor-core kernels (their cost follows the
// codes, the dp2a kernels' the tokens): measured crossovers on GB300 are about 8 tokens for
// Qwen3-sized experts (768 x 2048 codes a matrix) and at most 4 for Mixtral-sized ones
// (14336 x 4096), whose per-item costs amortise over far more codes.
#ifndef BITSMOE_TC_MIN_TOKENS
inline int tc_min_tokens(const ImageHeader& hd) {
  return (uint64_t)hd.I_pad * (uint64_t)hd.n_pad >= (8ull << 20) ? 4 : 8;
}
#else
inline int tc_min_tokens(const ImageHeader&) { return BITSMOE_TC_MIN_TOKENS; }
#endif

// Small batches run the decode chain (every kernel routes all tokens itself; the
// single token also the fused kernel), larger ones the tensor-core chain.
inline bool decode_mode(const ImageHeader& hd, int T) {
  return T <= BITSMOE_DECODE_MAX_TOKENS && T * hd.E <= 4096;
}

struct WsLayout {
  size_t status, pair_expert, pair_weight, expert_count, expert_start, pair_list, active, z, gu, s, zmax, zt, hb, hs, zv;
  size_t x_stage, logits_stage, y_stage;
  size_t sync;   // fused single-token kernel: grid-barrier counters
  size_t total;
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
  w.status = take(64);   // [0] status, [1] routing flag, [2] router block count; bytes 16..63: single-token kernels' sync words
  w.pair_expert = take(P * 4);
  w.pair_weight = take(P * 4);
  w.expert_count = take((size_t)hd.E * 4);
  w.expert_start = take(((size_t)hd.E + 1) * 4);
  w.pair_list = take(P * 4);
  w.active = take(((size_t)hd.E + 1) * 4);
  w.z = take(2 * (size_t)T * hd.n_pad * 4);
  w.gu = take(P * 2 * hd.I_pad * 4);
  w.s = take((size_t)T * hd.n_pad * 4);
  // tensor-core expert factors (calls past the decode chain): max |z| per token (directly after
  // s: one clear for both), z token fastest, h tiles and their row-block sums and scales
  const bool tcx = !decode_mode(hd, T);
  const XArgs xa = tcx ? x_args(hd, T, k) : XArgs{};
  w.zmax = take(tcx ? 2 * (size_t)T * 4 : 0);
  w.zt = take(tcx ? 2 * (size_t)T * hd.n_pad * 4 : 0);
  w.hb = take(tcx ? (size_t)hd.NRB * xa.Rtot * 512 : 0);
  w.hs = take(tcx ? (size_t)hd.NRB * xa.Rtot * 8 : 0);
  w.zv = take(tcx ? (size_t)xa.zv_floats * 4 : 0);
  w.x_stage = take((size_t)T * hd.D * 2);
  w.logits_stage = take((size_t)T * hd.E * 4);
  w.y_stage = take((size_t)T * hd.D * 4);
  w.sync = w.status + 16;   // fixed offset: no other layout of the workspace writes there (12 words)
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

// Every kernel asks for the largest shared-memory carveout, so that blocks of
// consecutive kernels of the chain can be resident on one SM at the same time
// (an SM cannot hold blocks configured with different L1/shared splits).
template <class K>
int set_smem(K kernel, size_t smem) {
  static std::mutex mu;
  static std::vector<std::pair<const void*, size_t>> done;
  std::lock_guard<std::mutex> lock(mu);
  const void* key = reinterpret_cast<const void*>(kernel);
  for (auto& d : done)
    if (d.first == key && d.second >= smem) return BITSMOE_OK;
  BM_CK(cudaFuncSetAttribute(kernel, cudaFuncAttributePreferredSharedMemoryCarveout, cudaSharedmemCarveoutMaxShared));
  if (smem > 48 * 1024) BM_CK(cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
  done.emplace_back(key, std::max<size_t>(smem, 48 * 1024));
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

template <int TB>
int launch_gemv_bulk_tb(bool proj, const Fwd& p, int sms, cudaStream_t st, bool pdl) {
  const int ld = proj ? p.D_pad : p.n_pad;
  const int nrows = proj ? 2 * p.n : p.D;
  const size_t row_bytes = (size_t)ld * 2;
  const size_t vec = (size_t)TB * ld * 4;
#ifndef BITSMOE_GEMV_PROJ_KB
#define BITSMOE_GEMV_PROJ_KB 128   // shared memory of the projection GEMV's two-stage ring (bytes in flight per SM)
#endif
  const size_t budget = proj ? BITSMOE_GEMV_PROJ_KB * 1024 : (vec < 150 * 1024 ? 200 * 1024 - vec : 48 * 1024);
  const int grid = std::min(nrows, sms);
  const int per = (nrows + grid - 1) / grid;
  int stage_rows = (int)std::max<size_t>(1, std::min<size_t>((budget / 2) / row_bytes, (size_t)(per + 1) / 2));
  const size_t smem = 2 * (size_t)stage_rows * row_bytes + vec + 16;
  int rc;
  if (proj) {
    if ((rc = set_smem(k_gemv_bulk<TB, true>, smem))) return rc;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    BM_CK(cudaLaunchKernelEx(&cfg, k_gemv_bulk<TB, true>, p, stage_rows));
    return BITSMOE_OK;
  }
  if ((rc = set_smem(k_gemv_bulk<TB, false>, smem))) return rc;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  BM_CK(cudaLaunchKernelEx(&cfg, k_gemv_bulk<TB, false>, p, stage_rows));
  return BITSMOE_OK;
}

int launch_gemv_bulk(bool proj, const Fwd& p, int sms, cudaStream_t st, bool pdl) {
  if (p.T <= 1) return launch_gemv_bulk_tb<1>(proj, p, sms, st, pdl);
  if (p.T <= 2) return launch_gemv_bulk_tb<2>(proj, p, sms, st, pdl);
  if (p.T <= 4) return launch_gemv_bulk_tb<4>(proj, p, sms, st, pdl);
  return launch_gemv_bulk_tb<8>(proj, p, sms, st, pdl);
}

// parts: 1 the gate/up kernel, 2 the down kernel, 3 both
template <int G, int TB>
int launch_k2k3_dec(const Fwd& p, int A_max, int sms, cudaStream_t st, bool pdl,
                    const std::function<int()>& between, int parts = 3) {
  int rc;
  const size_t rbytes = 0;
  if (parts & 1) {
    const size_t smax = (size_t)p.s16 - 8;
    const size_t pw2 = (size_t)p.seg_bytes + smax * 4 * (2 + G) + (size_t)G * TB * p.s16 * 2 + 16;
    const size_t sm2 = rbytes + kK2DecWarps * pw2;
    const int items2 = A_max * 2 * p.NRB * p.nseg;
    if ((rc = set_smem(k_gateup_dec<G, TB>, sm2))) return rc;
    if ((rc = launch(k_gateup_dec<G, TB>, dim3((items2 + kK2DecWarps - 1) / kK2DecWarps), dim3(kK2DecWarps * 32),
                     sm2, st, pdl, p)))
      return rc;
  }
  if (between && (rc = between())) return rc;
  if (!(parts & 2)) return BITSMOE_OK;
  const size_t nrm = (size_t)p.rbc * kRows;
  const int ngc_max = std::max(1, (int)(nrm / p.group));
  const size_t pw3 = (size_t)p.ul_bytes + (size_t)ngc_max * 32 * 4 + 16;
  const size_t sm3 = rbytes + TB * nrm * 6 + TB * 64 * 4 + kK3DecWarps * TB * 4 + ((TB + 3) & ~3) * 4 +
                     kK3DecWarps * pw3;
  const int ntg = (p.ul_max_tiles + kK3DecWarps - 1) / kK3DecWarps;
  const int nrc = (p.NRB + p.rbc - 1) / p.rbc;
  if ((rc = set_smem(k_down_dec<G, TB>, sm3))) return rc;
  return launch(k_down_dec<G, TB>, dim3(std::max(1, A_max * ntg * nrc)), dim3(kK3DecWarps * 32), sm3, st, pdl, p);
}

bool aligned(const void* ptr, size_t a) { return ((uintptr_t)ptr % a) == 0; }

// The device address of `bytes` of pinned, device-mapped host memory at p (null for
// anything else, when not aligned to `a` bytes, or when the last byte is not mapped at
// the same offset, i.e. [p, p + bytes) does not lie inside one mapping).
const void* mapped_host(const void* p, size_t bytes, size_t a) {
  cudaPointerAttributes at, end;
  if (bytes == 0 || cudaPointerGetAttributes(&at, p) != cudaSuccess ||
      cudaPointerGetAttributes(&end, static_cast<const uint8_t*>(p) + bytes - 1) != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  if (at.type != cudaMemoryTypeHost || !at.devicePointer || !aligned(at.devicePointer, a)) return nullptr;
  if (end.type != cudaMemoryTypeHost || !end.devicePointer ||
      static_cast<const uint8_t*>(end.devicePointer) != static_cast<const uint8_t*>(at.devicePointer) + bytes - 1)
    return nullptr;
  return at.devicePointer;
}

template <int TB>
int launch_norm_router_tb(const NormArgs& a, int sms, cudaStream_t st) {
  const size_t smem = (size_t)TB * a.D_pad8 * 4 + kWarps * TB * 4;
  int rc;
  if ((rc = set_smem(k_norm_router<TB>, smem))) return rc;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(std::max(1, std::min((a.E + kWarps - 1) / kWarps, sms)));
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  BM_CK(cudaLaunchKernelEx(&cfg, k_norm_router<TB>, a));
  return BITSMOE_OK;
}

int launch_norm_router(const NormArgs& a, int sms, cudaStream_t st) {
  if (a.T <= 1) return launch_norm_router_tb<1>(a, sms, st);
  if (a.T <= 2) return launch_norm_router_tb<2>(a, sms, st);
  if (a.T <= 4) return launch_norm_router_tb<4>(a, sms, st);
  return launch_norm_router_tb<8>(a, sms, st);
}

int num_sms_current(int* sms) {
  int dev = 0;
  BM_CK(cudaGetDevice(&dev));
  BM_CK(cudaDeviceGetAttribute(sms, cudaDevAttrMultiProcessorCount, dev));
  return BITSMOE_OK;
}


// norm != nullptr: a pre-norm block (y = h accumulates); x and logits are the workspace buffers that
// the norm/router step fills, either as its own kernel or inside the one-token fused kernel.

// Up to this many tokens run as one fused single-token forward per token when the layer
// fits the fused kernel (T fused forwards beat the decode chain there).
constexpr int kFusedMaxTokens = 4;

bool fused_fits(const bitsmoe_layer* L, int top_k) {
  const ImageHeader& hd = L->hd();
  FusedArgs fa;
  const int s16 = (int)align_up(std::max(hd.seg_max_slots, 8), 64) + 8;
  return decode_mode(hd, 1) && L->meta_ok &&
         fused_plan(hd, 1, top_k, L->seg_bytes, L->ul_max_chunks, s16, L->num_sms, &fa);
}

// The clustered single-token plan for this layer and top_k: the index of its cluster
// size in kF2Sizes (the largest whose co-resident clusters hold one (routing slot, row
// block) pair each and whose shared-memory plan fits), or -1.
// Taken automatically only where its expert phase spans at least 90% of the SMs: with
// fewer, the blocks that hold pairs carry the whole factor work and the kernel without
// clusters (which deals that work over every block) is faster (Qwen3-shaped layer on 152
// SMs: 48 pairs fit clusters of 2 but not of 3, so 96 blocks: 24.8 against 23.1 us).
int f2_choose(const bitsmoe_layer* L, int top_k, F2Args* fa) {
  const int dbg = g_dbg_kernel.load();
  if (top_k < 1 || top_k > 32 || dbg == 1) return -1;
  std::lock_guard<std::mutex> lock(L->f2_mu);
  if (L->f2_ci[top_k] == 0x7F) {
    const ImageHeader& hd = L->hd();
    int ci = -1;
    for (int i = 0; i < 5 && ci < 0; ++i)
      if (L->f2_nc[i] > 0 && f2_plan(hd, top_k, kF2Sizes[i], L->f2_nc[i], L->f2_sz[i], &L->f2_args[top_k])) ci = i;
    L->f2_ci[top_k] = (signed char)ci;
  }
  const int ci = L->f2_ci[top_k];
  if (ci < 0) return -1;
  *fa = L->f2_args[top_k];
  if (dbg != 2 && 10 * fa->npairs * fa->CL < 9 * L->num_sms) return -1;
  return ci;
}

int forward_impl(const void* x, const float* logits, int T, int top_k, const bitsmoe_layer* L, float* y,
                 void* ws, size_t ws_bytes, cudaStream_t st, cudaEvent_t* ev = nullptr, bool accum = false,
                 const NormArgs* norm = nullptr, bool host_io = false) {
  const ImageHeader& hd = L->hd();
  if (T > 1 && T <= kFusedMaxTokens && fused_fits(L, top_k)) {
    // a few tokens: one fused forward each, on the same workspace (profiled as one phase)
    if (ev) BM_CK(cudaEventRecord(ev[0], st));
    for (int t = 0; t < T; ++t) {
      NormArgs nt;
      if (norm) {
        nt = *norm;
        nt.h = norm->h + (size_t)t * hd.D;
        nt.T = 1;
      }
      const int rc = forward_impl(static_cast<const uint16_t*>(x) + (size_t)t * hd.D, logits + (size_t)t * hd.E, 1,
                                  top_k, L, y + (size_t)t * hd.D, ws, ws_bytes, st, nullptr, accum,
                                  norm ? &nt : nullptr);
      if (rc) return rc;
    }
    if (ev)
      for (int i = 1; i <= 5; ++i) BM_CK(cudaEventRecord(ev[i], st));
    return BITSMOE_OK;
  }
  const bool pdl = ev == nullptr;   // profiling runs the phases back to back without overlap
  const WsLayout w = ws_layout(hd, T, top_k);
  uint8_t* wb = static_cast<uint8_t*>(ws);
  Fwd p;
  std::memset(&p, 0, sizeof(p));
  p.img = L->d_img;
  p.img_bytes = L->bytes;
  p.desc = reinterpret_cast<const ExpertDesc*>(L->d_img + hd.off_desc);
  p.seg = reinterpret_cast<const int32_t*>(L->d_img + hd.off_seg);
  p.items = reinterpret_cast<const ItemRec*>(L->d_img + hd.off_items);
  p.basis_in = reinterpret_cast<const uint16_t*>(L->d_img + hd.off_basis_in);
  p.basis_out = reinterpret_cast<const uint16_t*>(L->d_img + hd.off_basis_out);
  p.D = hd.D; p.E = hd.E; p.I = hd.I; p.n = hd.n; p.group = hd.group;
  p.D_pad = hd.D_pad; p.n_pad = hd.n_pad; p.I_pad = hd.I_pad; p.NRB = hd.NRB; p.NG = hd.NG;
  p.nseg = hd.nseg; p.ul_max_tiles = hd.ul_max_tiles;
  p.T = T; p.k = top_k; p.P = T * top_k;
  p.s16 = (int)align_up(std::max(hd.seg_max_slots, 8), 64) + 8;
  p.rbc = k3_rbc(hd);
  p.seg_bytes = L->seg_bytes;
  // decode mode: every kernel can afford the routing of all tokens
  p.decode = decode_mode(hd, T);
  {   // down staging: keep a warp's tile within ~48 KB of shared memory
    const int need = std::max(1, hd.group / kRows);
    int rbc = std::min(p.rbc, std::max(1, (48 * 1024) / (L->ul_max_chunks * kChunkBytes)));
    rbc = std::max(need, rbc / need * need);
    p.rbc = rbc;
    p.ul_bytes = rbc * L->ul_max_chunks * kChunkBytes;
  }
  p.x = static_cast<const uint16_t*>(x);
  p.logits = logits;
  p.y = y;
  p.accum = accum ? 1 : 0;
  p.status = reinterpret_cast<int*>(wb + w.status);
  p.route_flag = p.status + 1;
  p.pair_expert = reinterpret_cast<int*>(wb + w.pair_expert);
  p.pair_weight = reinterpret_cast<float*>(wb + w.pair_weight);
  p.expert_count = reinterpret_cast<int*>(wb + w.expert_count);
  p.expert_start = reinterpret_cast<int*>(wb + w.expert_start);
  p.pair_list = reinterpret_cast<int*>(wb + w.pair_list);
  p.active = reinterpret_cast<int*>(wb + w.active);
  p.z = reinterpret_cast<float*>(wb + w.z);
  p.gu = reinterpret_cast<float*>(wb + w.gu);
  p.s = reinterpret_cast<float*>(wb + w.s);
  p.zT = reinterpret_cast<float*>(wb + w.zt);
  const int sms = L->num_sms;
  int rc;
  auto mark = [&](int i) -> int {
    if (ev) BM_CK(cudaEventRecord(ev[i], st));
    return BITSMOE_OK;
  };
  const int G = std::max(1, kRows / hd.group);
  if (T == 1 && !norm) {   // one token: the clustered kernel when the layer fits it
    F2Args f2;
    const int ci = f2_choose(L, top_k, &f2);
    if (ci >= 0) {
      f2.sync = reinterpret_cast<uint32_t*>(wb + w.sync);
      f2.tab = L->d_f2 + L->f2_off[ci];
      f2.dbg = g_dbg_skip.load() | (g_dbg_bounds.load() ? 2 : 0);
      f2.prefetch_io = host_io ? 0 : 1;   // no L2 prefetch of host memory mapped into the address space
      const long long sp = g_dbg_spin.load();
      if (sp > 0) f2.spin = sp;
      if ((rc = mark(0))) return rc;
      const cudaError_t e = launch_f2(p, f2, L->f2_nc[ci], st, pdl);
      if (e != cudaSuccess) return cuda_fail(e);
      for (int i = 1; i <= 5; ++i)
        if ((rc = mark(i))) return rc;
      return BITSMOE_OK;
    }
  }
  FusedArgs fa;
  if (p.decode && L->meta_ok && fused_plan(hd, T, top_k, L->seg_bytes, L->ul_max_chunks, p.s16, sms, &fa)) {
    // one token: the whole layer in one persistent kernel
    fa.sync = reinterpret_cast<uint32_t*>(wb + w.sync);
    fa.dbg = g_dbg_skip.load() | (g_dbg_bounds.load() ? 2 : 0);
    if (g_dbg_spin.load() > 0) fa.spin = g_dbg_spin.load();
    fa.cst = L->d_cst;
    fa.dst = L->d_dst;
    fa.tab_bytes = L->stage_bytes;
    fa.meta = L->d_meta;
    fa.meta_bytes = L->meta_bytes;
    if (norm) {
      fa.norm = 1;
      fa.hn = norm->h;
      fa.wr = norm->w;
      fa.eps = norm->eps;
    }
    if ((rc = mark(0))) return rc;
    const cudaError_t e = launch_fused(p, fa, sms, st, pdl);
    if (e != cudaSuccess) return cuda_fail(e);
    for (int i = 1; i <= 5; ++i)
      if ((rc = mark(i))) return rc;
    return BITSMOE_OK;
  }
  if (norm && (rc = launch_norm_router(*norm, sms, st))) return rc;
  if (p.decode) {
    const int A_max = std::min(hd.E, p.P);
    const size_t rsm = (size_t)route_words(p.T, hd.E, p.P) * 4 + 16;
    if ((rc = mark(0))) return rc;
    if ((rc = set_smem(k_route_publish, rsm))) return rc;
    if ((rc = launch(k_route_publish, dim3(1), dim3(kThreads), rsm, st, false, p))) return rc;
    if ((rc = mark(1))) return rc;
    const bool tcp = L->maps && T >= 4;   // below 4 tokens the bulk-copy GEMV streams the bases faster
    if (tcp) {   // tensor-core projection; it also clears gate/up and s for the expert kernels
      const size_t zb = (size_t)(reinterpret_cast<uint8_t*>(p.s) - reinterpret_cast<uint8_t*>(p.gu)) +
                        (size_t)T * hd.n_pad * 4;
      BM_CK(launch_gemm_tc(0, L->map_in, p, sms, st, pdl, nullptr, p.gu, zb));
    } else if ((rc = launch_gemv_bulk(true, p, sms, st, pdl))) {
      return rc;
    }
    if ((rc = mark(2))) return rc;
    std::function<int()> between = ev ? std::function<int()>([&]() { return mark(3); }) : std::function<int()>();
    if (T == 1) {
      if (G == 1) rc = launch_k2k3_dec<1, 1>(p, A_max, sms, st, pdl, between);
      else if (G == 2) rc = launch_k2k3_dec<2, 1>(p, A_max, sms, st, pdl, between);
      else rc = launch_k2k3_dec<4, 1>(p, A_max, sms, st, pdl, between);
    } else {
      if (G == 1) rc = launch_k2k3_dec<1, 4>(p, A_max, sms, st, pdl, between);
      else if (G == 2) rc = launch_k2k3_dec<2, 4>(p, A_max, sms, st, pdl, between);
      else rc = launch_k2k3_dec<4, 4>(p, A_max, sms, st, pdl, between);
    }
    if (rc) return rc;
    if ((rc = mark(4))) return rc;
    if (tcp) BM_CK(launch_gemm_tc(1, L->map_out, p, sms, st, pdl));
    else if ((rc = launch_gemv_bulk(false, p, sms, st, pdl))) return rc;
    return mark(5);
  }
  const int tpb = std::max(1, 1024 / hd.E);
  const size_t router_smem =
      std::max((size_t)tpb * (hd.E + top_k), (size_t)p.P + 2 * (size_t)hd.E + 1) * 4;   // selection | grouping
  if (router_smem > 200 * 1024) return BITSMOE_ERR_SHAPE;
  if ((rc = mark(0))) return rc;
  if ((rc = set_smem(k_router, router_smem))) return rc;
  if ((rc = launch(k_router, dim3((T + tpb - 1) / tpb), dim3(1024), router_smem, st, false, p))) return rc;
  if ((rc = mark(1))) return rc;
  const bool tc = L->maps;          // tensor-core projections for multi-token calls
  const bool tcx = tc && L->tcx;    // and the expert factors on tensor cores
  const int A_max = std::min(hd.E, p.P);
  if (tcx) {
    // Experts with at least tc_min_tokens tokens take the tensor-core factor kernels (their codes
    // are decoded once for all their tokens), the others the dp2a kernels (whose cost follows
    // the tokens); each kind skips the other's experts, both add into s.  Cleared here: gu
    // (dp2a gate/up adds into it), s, and the max |z| per token that the projection takes;
    // z lies before them, zmax right after s.  The projection also stores z token-fastest.
    p.tc_min = tc_min_tokens(hd);
    XArgs xa = x_args(hd, T, top_k);
    xa.tc_min = p.tc_min;
    xa.msa = L->d_msa;
    xa.zmax = reinterpret_cast<const uint32_t*>(wb + w.zmax);
    xa.hb = wb + w.hb;
    xa.hs = reinterpret_cast<float2*>(wb + w.hs);
    xa.zv = reinterpret_cast<float*>(wb + w.zv);
    BM_CK(cudaMemsetAsync(p.z, 0, w.zmax + 2 * (size_t)T * 4 - w.z, st));
    BM_CK(launch_gemm_tc(0, L->map_in, p, sms, st, false, p.zT, nullptr, 0, reinterpret_cast<uint32_t*>(wb + w.zmax)));
    if ((rc = mark(2))) return rc;
    BM_CK(launch_zgather(p, xa, sms, st, pdl));
    BM_CK(launch_gu16(p, xa, sms, st, pdl));
    if (G == 1) rc = launch_k2k3_dec<1, 4>(p, A_max, sms, st, pdl, std::function<int()>(), 1);
    else if (G == 2) rc = launch_k2k3_dec<2, 4>(p, A_max, sms, st, pdl, std::function<int()>(), 1);
    else rc = launch_k2k3_dec<4, 4>(p, A_max, sms, st, pdl, std::function<int()>(), 1);
    if (rc) return rc;
    if ((rc = mark(3))) return rc;
    BM_CK(launch_dn16(p, xa, sms, st, pdl));
    if (G == 1) rc = launch_k2k3_dec<1, 4>(p, A_max, sms, st, pdl, std::function<int()>(), 2);
    else if (G == 2) rc = launch_k2k3_dec<2, 4>(p, A_max, sms, st, pdl, std::function<int()>(), 2);
    else rc = launch_k2k3_dec<4, 4>(p, A_max, sms, st, pdl, std::function<int()>(), 2);
    if (rc) return rc;
  } else {
    if (tc) {
      // the dp2a gate/up and down kernels add into gu and s (cleared here with z, which lies
      // before them); the projection stores z, the output basis stores y (or adds into it,
      // when it holds the residual)
      BM_CK(cudaMemsetAsync(p.z, 0, w.s + (size_t)T * hd.n_pad * 4 - w.z, st));
      BM_CK(launch_gemm_tc(0, L->map_in, p, sms, st, false));
    } else if ((rc = launch_gemv_any(true, p, sms, st, pdl))) {
      return rc;
    }
    if ((rc = mark(2))) return rc;
    // gate/up factors (the staged dp2a kernel over batches of 4 tokens), then down
    std::function<int()> between = ev ? std::function<int()>([&]() { return mark(3); }) : std::function<int()>();
    if (G == 1) rc = launch_k2k3_dec<1, 4>(p, A_max, sms, st, pdl, between);
    else if (G == 2) rc = launch_k2k3_dec<2, 4>(p, A_max, sms, st, pdl, between);
    else rc = launch_k2k3_dec<4, 4>(p, A_max, sms, st, pdl, between);
  }
  if (rc) return rc;
  if ((rc = mark(4))) return rc;
  if (tc) BM_CK(launch_gemm_tc(1, L->map_out, p, sms, st, pdl));
  else if ((rc = launch_gemv_any(false, p, sms, st, pdl))) return rc;
  return mark(5);
}

// Per gate/up (h, e): the largest |scale * alpha| over its groups and slots, in the fp32
// arithmetic of the tensor-core gate/up kernel (which bounds its operand by it).
std::vector<float> gate_up_scale_bounds(const uint8_t* img) {
  const ImageHeader& hd = *header_of(img);
  const ExpertDesc* xd = desc_of(img);
  std::vector<float> out(2 * (size_t)hd.E, 0.f);
  auto f16 = [](uint32_t b) {   // IEEE binary16 bits -> float
    const int s = (b >> 15) & 1, e = (b >> 10) & 31, m = b & 1023;
    const float v = e == 0 ? std::ldexp((float)m, -24)
                    : e == 31 ? (m ? std::numeric_limits<float>::quiet_NaN() : std::numeric_limits<float>::infinity())
                              : std::ldexp((float)(m | 1024), e - 25);
    return s ? -v : v;
  };
  for (int i = 0; i < 2 * hd.E; ++i) {
    const ExpertDesc& x = xd[i];
    const float* al = reinterpret_cast<const float*>(img + x.alpha_off);
    const uint32_t* sz = reinterpret_cast<const uint32_t*>(img + x.sz_off);
    float m = 0.f;
    for (int g = 0; g < hd.NG; ++g)
      for (int j = 0; j < x.nslots; ++j) m = std::max(m, std::fabs(f16(sz[(size_t)g * x.nslots + j] & 0xFFFFu) * al[j]));
    out[i] = m;
  }
  return out;
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
  // staging records of the fused single-token kernel, derived from the image
  std::vector<CStage> cst;
  std::vector<DStage> dst;
  std::vector<uint8_t> meta;
  const bool meta_ok = build_stage_tables(img.data(), cst, dst, meta);
  const size_t cst_bytes = cst.size() * sizeof(CStage), dst_bytes = dst.size() * sizeof(DStage);
  const size_t meta_at = align_up(cst_bytes + dst_bytes, 256);
  const std::vector<float> msa = gate_up_scale_bounds(img.data());
  const size_t msa_at = align_up(meta_at + meta.size(), 256);
  // records of the clustered single-token kernel for every cluster size, one buffer
  std::vector<uint8_t> f2all;
  uint64_t f2_off[5] = {};
  int f2_nc[5] = {};
  F2Sizes f2_sz[5] = {};
  {
    const int G = std::max(1, kRows / header_of(img.data())->group);
    for (int i = 0; i < 5; ++i) {
      std::vector<uint8_t> t;
      const bool ok = build_f2_tables(img.data(), kF2Sizes[i], t, &f2_sz[i]);
      f2_off[i] = f2all.size();
      f2all.insert(f2all.end(), t.begin(), t.end());
      f2all.resize(align_up(f2all.size(), 256), 0);
      if (e == cudaSuccess && ok) f2_nc[i] = f2_max_clusters(G, kF2Sizes[i]);
    }
  }
  uint8_t* d = nullptr;
  uint8_t* ds = nullptr;
  uint8_t* df2 = nullptr;
  const size_t slack = g_dbg_bounds.load() ? img.size() : 0;
  if (e == cudaSuccess) e = cudaMalloc(&d, img.size() + slack);
  if (e == cudaSuccess) e = cudaMemcpy(d, img.data(), img.size(), cudaMemcpyHostToDevice);
  if (e == cudaSuccess && slack) e = cudaMemset(d + img.size(), 0, slack);
  if (e == cudaSuccess) e = cudaMalloc(&ds, msa_at + msa.size() * 4 + 16);
  if (e == cudaSuccess) e = cudaMemcpy(ds + msa_at, msa.data(), msa.size() * 4, cudaMemcpyHostToDevice);
  if (e == cudaSuccess && cst_bytes) e = cudaMemcpy(ds, cst.data(), cst_bytes, cudaMemcpyHostToDevice);
  if (e == cudaSuccess && dst_bytes) e = cudaMemcpy(ds + cst_bytes, dst.data(), dst_bytes, cudaMemcpyHostToDevice);
  if (e == cudaSuccess && !meta.empty()) e = cudaMemcpy(ds + meta_at, meta.data(), meta.size(), cudaMemcpyHostToDevice);
  if (e == cudaSuccess) e = cudaMalloc(&df2, f2all.size() + 16);
  if (e == cudaSuccess && !f2all.empty()) e = cudaMemcpy(df2, f2all.data(), f2all.size(), cudaMemcpyHostToDevice);
  cudaSetDevice(prev);
  if (e != cudaSuccess) {
    if (d) cudaFree(d);
    if (ds) cudaFree(ds);
    if (df2) cudaFree(df2);
    return e == cudaErrorMemoryAllocation ? BITSMOE_ERR_OOM : cuda_fail(e);
  }
  bitsmoe_layer* L = new (std::nothrow) bitsmoe_layer;
  if (!L) {
    cudaFree(d);
    cudaFree(ds);
    cudaFree(df2);
    return BITSMOE_ERR_OOM;
  }
  L->d_f2 = df2;
  for (int i = 0; i < 5; ++i) {
    L->f2_off[i] = f2_off[i];
    L->f2_nc[i] = f2_nc[i];
    L->f2_sz[i] = f2_sz[i];
  }
  L->d_stage = ds;
  L->d_cst = reinterpret_cast<const CStage*>(ds);
  L->d_dst = reinterpret_cast<const DStage*>(ds + cst_bytes);
  L->stage_bytes = cst_bytes + dst_bytes;
  L->d_meta = ds + meta_at;
  L->meta_bytes = meta.size();
  L->meta_ok = meta_ok && !meta.empty();
  L->d_msa = reinterpret_cast<const float*>(ds + msa_at);
  {
    const ImageHeader* h = header_of(img.data());
    L->maps = make_basis_map(L->map_in, d + h->off_basis_in, 2 * h->n, h->D_pad) &&
              make_basis_map(L->map_out, d + h->off_basis_out, h->D, h->n_pad);
    bool ok16 = h->group % kRows == 0;
    const ExpertDesc* xd = desc_of(img.data());
    for (int i = 0; i < 2 * h->E; ++i) {
      for (int k = 0; k < xd[i].nbk; ++k)
        if (xd[i].bk[k].bits >= 16) ok16 = false;
    }
    for (int i = 2 * h->E; i < 3 * h->E; ++i)
      for (int k = 0; k < xd[i].nbk; ++k)
        if (xd[i].bk[k].bits >= 16) ok16 = false;
    L->tcx = ok16;
  }
  const ImageHeader* hd = header_of(img.data());
  const size_t meta_end = hd->off_basis_in;   // header + descriptors + segments
  L->device = device;
  L->num_sms = sms;
  L->d_img = d;
  L->bytes = img.size();
  L->meta.assign(img.begin(), img.begin() + meta_end);
  {
    const ExpertDesc* d = L->desc();
    const int32_t* sg = reinterpret_cast<const int32_t*>(L->meta.data() + hd->off_seg);
    for (int pi = 0; pi < 2 * hd->E; ++pi) {
      const ExpertDesc& x = d[pi];
      for (int q = 0; q < hd->nseg; ++q) {
        const int t0 = sg[(size_t)pi * (hd->nseg + 1) + q], t1 = sg[(size_t)pi * (hd->nseg + 1) + q + 1];
        int bytes = 0;
        for (int k = 0; k < x.nbk; ++k) {
          const int lo = std::max(t0, x.bk[k].tile0), hi = std::min(t1, x.bk[k].tile0 + x.bk[k].ntiles);
          if (hi > lo) bytes += (hi - lo) * rl_chunks(x.bk[k].bits) * kChunkBytes;
        }
        L->seg_bytes = std::max(L->seg_bytes, bytes);
      }
    }
    for (int pi = 2 * hd->E; pi < 3 * hd->E; ++pi)
      for (int k = 0; k < d[pi].nbk; ++k) L->ul_max_chunks = std::max(L->ul_max_chunks, ul_chunks(d[pi].bk[k].bits));
  }
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

// Device address of the scratch on `device` (which must be current).  The first
// lookup on a device is refused while `st` is capturing a graph: the symbol lookup
// is not a stream operation and may initialise the module, so it must happen
// before any capture.
int noalloc_scratch(int device, cudaStream_t st, void** out) {
  if (device < 0 || device >= kNoAllocMaxDevices) return BITSMOE_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> lock(g_noalloc_mu);
  if (!g_noalloc_addr[device]) {
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    const cudaError_t ce = cudaStreamIsCapturing(st, &cs);
    if (ce != cudaSuccess) return cuda_fail(ce);
    if (cs != cudaStreamCaptureStatusNone) return BITSMOE_ERR_INVALID_ARG;
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess || !p) return cuda_fail(e != cudaSuccess ? e : cudaErrorInvalidSymbol);
    g_noalloc_addr[device] = p;
  }
  *out = g_noalloc_addr[device];
  return BITSMOE_OK;
}

}  // namespace

namespace bmoe {
int record_cuda_error(int cuda_error) { return cuda_fail(static_cast<cudaError_t>(cuda_error)); }
}  // namespace bmoe

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
  if ((rc = noalloc_scratch(L->device, static_cast<cudaStream_t>(stream), &ws))) return rc;
  return forward_impl(x, logits, T, top_k, L, y, ws, kNoAllocBytes, static_cast<cudaStream_t>(stream));
}

int bitsmoe_noalloc_last_status(void* stream) {
  int dev = -1;
  BM_CK(cudaGetDevice(&dev));
  void* ws = nullptr;
  const int rc = noalloc_scratch(dev, static_cast<cudaStream_t>(stream), &ws);
  if (rc) return rc;
  return bitsmoe_last_device_status(ws, stream);
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

}  // extern "C"

namespace {
// Kernels one forward launches; allow_f2: the plain forward (the pre-norm block
// forward does not take the clustered kernel).
int forward_launches(const bitsmoe_layer* L, int T, int top_k, bool allow_f2) {
  if (!L || T < 0) return BITSMOE_ERR_INVALID_ARG;
  const ImageHeader& hd = L->hd();
  if (top_k < 1 || top_k > std::min(hd.E, 32)) return BITSMOE_ERR_INVALID_ARG;
  if (T == 0) return 0;
  F2Args f2;
  if (allow_f2 && T == 1 && f2_choose(L, top_k, &f2) >= 0) return 1;
  const bool decode = decode_mode(hd, T);
  FusedArgs fa;
  const int s16 = (int)align_up(std::max(hd.seg_max_slots, 8), 64) + 8;
  if (decode && L->meta_ok && fused_plan(hd, T, top_k, L->seg_bytes, L->ul_max_chunks, s16, L->num_sms, &fa)) return 1;
  if (T <= kFusedMaxTokens && fused_fits(L, top_k)) return T;   // one fused forward per token
  if (decode || !L->maps) return 5;
  return L->tcx ? 8 : 5;   // router, projection, [z gather, gate/up tc,] gate/up, [down tc,] down, output basis
}
}  // namespace

extern "C" {

int bitsmoe_forward_launches(const bitsmoe_layer* L, int T, int top_k) { return forward_launches(L, T, top_k, true); }

int bitsmoe_forward_plan(const bitsmoe_layer* L, int T, int top_k) {
  const int n = bitsmoe_forward_launches(L, T, top_k);
  if (n <= 0) return n;
  F2Args f2;
  if (T <= kFusedMaxTokens && (T == 1 || fused_fits(L, top_k)) && f2_choose(L, top_k, &f2) >= 0) return 1 | 32;
  if (T <= kFusedMaxTokens && fused_fits(L, top_k)) return 1;
  const ImageHeader& hd = L->hd();
  if (decode_mode(hd, T)) return 2 | (L->maps && T >= 4 ? 4 : 0);
  return L->maps ? 4 | (L->tcx ? 8 | 16 : 0) : 0;
}

int bitsmoe_block_forward_launches(const bitsmoe_layer* L, int T, int top_k) {
  const int n = forward_launches(L, T, top_k, false);
  if (n > 0 && T <= kFusedMaxTokens && fused_fits(L, top_k)) return n;   // the fused kernels norm in place
  return n > 1 ? n + 1 : n;
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

static int forward_host(const void* x_host, const float* logits_host, int T, int top_k, const bitsmoe_layer* L,
                        float* y_host, void* ws, size_t ws_bytes, void* stream, bool sync) {
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
  if (T == 1 && bitsmoe_forward_launches(L, T, top_k) == 1) {
    // One token on the fused kernel with pinned (device-mapped) host buffers: the kernel reads x
    // and the logits and writes y through the unified address space (the bytes cross the
    // host link inside the kernel), which saves the copy round trips of a few KB.
    const void* xd = mapped_host(x_host, (size_t)hd.D * 2, 16);
    const void* ld = mapped_host(logits_host, (size_t)hd.E * 4, 16);
    void* yd = const_cast<void*>(mapped_host(y_host, (size_t)hd.D * 4, 16));
    if (xd && ld && yd) {
      rc = forward_impl(xd, static_cast<const float*>(ld), T, top_k, L, static_cast<float*>(yd), ws, ws_bytes, st,
                        nullptr, false, nullptr, true);
      if (rc) return rc;
      if (sync) BM_CK(cudaStreamSynchronize(st));
      return BITSMOE_OK;
    }
  }
  BM_CK(cudaMemcpyAsync(wb + w.x_stage, x_host, (size_t)T * hd.D * 2, cudaMemcpyHostToDevice, st));
  BM_CK(cudaMemcpyAsync(wb + w.logits_stage, logits_host, (size_t)T * hd.E * 4, cudaMemcpyHostToDevice, st));
  rc = forward_impl(wb + w.x_stage, reinterpret_cast<const float*>(wb + w.logits_stage), T, top_k, L,
                    reinterpret_cast<float*>(wb + w.y_stage), ws, ws_bytes, st);
  if (rc) return rc;
  BM_CK(cudaMemcpyAsync(y_host, wb + w.y_stage, (size_t)T * hd.D * 4, cudaMemcpyDeviceToHost, st));
  if (sync) BM_CK(cudaStreamSynchronize(st));
  return BITSMOE_OK;
}

int bitsmoe_moe_forward_host(const void* x_host, const float* logits_host, int T, int top_k,
                             const bitsmoe_layer* L, float* y_host, void* ws, size_t ws_bytes, void* stream) {
  return forward_host(x_host, logits_host, T, top_k, L, y_host, ws, ws_bytes, stream, true);
}

int bitsmoe_moe_forward_host_async(const void* x_host, const float* logits_host, int T, int top_k,
                                   const bitsmoe_layer* L, float* y_host, void* ws, size_t ws_bytes, void* stream) {
  return forward_host(x_host, logits_host, T, top_k, L, y_host, ws, ws_bytes, stream, false);
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

int bitsmoe_rmsnorm_router(const float* h, const void* w_router, float eps, int T, int D, int E, void* x_out,
                           float* logits_out, void* stream) {
  if (T < 0 || D < 8 || D % 8 || E < 1 || E > 1024 || !(eps >= 0.f)) return BITSMOE_ERR_INVALID_ARG;
  if ((int64_t)T * D > (1ll << 31) || D > (1 << 16)) return BITSMOE_ERR_SHAPE;
  if (T == 0) return BITSMOE_OK;
  if (!h || !w_router || !x_out || !logits_out) return BITSMOE_ERR_INVALID_ARG;
  if (!aligned(h, 16) || !aligned(w_router, 16) || !aligned(x_out, 16) || !aligned(logits_out, 16))
    return BITSMOE_ERR_ALIGNMENT;
  int sms = 0, rc = num_sms_current(&sms);
  if (rc) return rc;
  NormArgs a{h, static_cast<const uint16_t*>(w_router), eps, T, D, E, (D + 7) / 8 * 8,
             static_cast<uint16_t*>(x_out), logits_out};
  return launch_norm_router(a, sms, static_cast<cudaStream_t>(stream));
}

int bitsmoe_moe_block_forward(float* h, const void* w_router, float eps, int T, int top_k, const bitsmoe_layer* L,
                              void* ws, size_t ws_bytes, void* stream) {
  if (!L || T < 0 || !(eps >= 0.f)) return BITSMOE_ERR_INVALID_ARG;
  const ImageHeader& hd = L->hd();
  if (top_k < 1 || top_k > std::min(hd.E, 32)) return BITSMOE_ERR_INVALID_ARG;
  if ((int64_t)T * top_k > 24576 || (int64_t)T * hd.D > (1ll << 31) || hd.D % 8 || hd.D > (1 << 16))
    return BITSMOE_ERR_SHAPE;
  if (T == 0) return BITSMOE_OK;
  if (!h || !w_router || !ws) return BITSMOE_ERR_INVALID_ARG;
  if (!aligned(h, 16) || !aligned(w_router, 16) || !aligned(ws, 256)) return BITSMOE_ERR_ALIGNMENT;
  const WsLayout w = ws_layout(hd, T, top_k);
  if (ws_bytes < w.total) return BITSMOE_ERR_WORKSPACE_TOO_SMALL;
  int rc = check_device(L);
  if (rc) return rc;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  uint8_t* wb = static_cast<uint8_t*>(ws);
  NormArgs a{h, static_cast<const uint16_t*>(w_router), eps, T, hd.D, hd.E, hd.D_pad,
             reinterpret_cast<uint16_t*>(wb + w.x_stage), reinterpret_cast<float*>(wb + w.logits_stage)};
  return forward_impl(wb + w.x_stage, reinterpret_cast<const float*>(wb + w.logits_stage), T, top_k, L, h, ws,
                      ws_bytes, st, nullptr, true, &a);
}

int bitsmoe_block_norm_outputs(const bitsmoe_layer* L, int T, int top_k, size_t* x_offset, size_t* logits_offset) {
  if (!L || T < 1 || top_k < 1 || top_k > std::min(L->hd().E, 32) || !x_offset || !logits_offset)
    return BITSMOE_ERR_INVALID_ARG;
  const WsLayout w = ws_layout(L->hd(), T, top_k);
  *x_offset = w.x_stage;
  *logits_offset = w.logits_stage;
  return BITSMOE_OK;
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
    cudaFree(L->d_stage);
    cudaFree(L->d_f2);
    cudaSetDevice(prev);
  }
  delete L;
}

int bitsmoe_last_cuda_error(void) { return g_last_cuda; }

int bitsmoe_debug_single_token_kernel(int which) {
  if (which < 0 || which > 2) return BITSMOE_ERR_INVALID_ARG;
  g_dbg_kernel.store(which);
  return BITSMOE_OK;
}

int bitsmoe_debug_wait_limit(int skip_arrival, long long spin_clocks) {
  g_dbg_skip.store(skip_arrival ? 1 : 0);
  g_dbg_spin.store(spin_clocks > 0 ? spin_clocks : 0);
  return BITSMOE_OK;
}

int bitsmoe_debug_bounds(int on) {
  g_dbg_bounds.store(on ? 1 : 0);
  return BITSMOE_OK;
}

int bitsmoe_debug_shift_expert_records(const bitsmoe_layer* L, int e, long long delta) {
  if (!L || e < 0) return BITSMOE_ERR_INVALID_ARG;
  const ImageHeader& hd = L->hd();
  if (e >= hd.E) return BITSMOE_ERR_INVALID_ARG;
  int prev = 0;
  BM_CK(cudaGetDevice(&prev));
  BM_CK(cudaSetDevice(L->device));
  auto shift = [&](uint8_t* rec) -> cudaError_t {   // the record's first field: its code offset
    uint64_t v = 0;
    cudaError_t r = cudaMemcpy(&v, rec, 8, cudaMemcpyDeviceToHost);
    if (r != cudaSuccess) return r;
    v += (uint64_t)delta;
    return cudaMemcpy(rec, &v, 8, cudaMemcpyHostToDevice);
  };
  cudaError_t r = cudaSuccess;
  // the kernel without clusters: CStage [2][E][nseg]
  for (int h = 0; h < 2 && r == cudaSuccess; ++h)
    for (int q = 0; q < hd.nseg && r == cudaSuccess; ++q)
      r = shift(L->d_stage + (((size_t)h * hd.E + e) * hd.nseg + q) * sizeof(CStage));
  // the clustered kernel: per cluster size, per rank [gate E][up E][down E]
  const size_t rank_bytes = (size_t)hd.E * (2 * sizeof(F2Gu) + sizeof(F2Dn));
  for (int i = 0; i < 5 && r == cudaSuccess; ++i) {
    if (!L->f2_nc[i]) continue;
    for (int rk = 0; rk < kF2Sizes[i] && r == cudaSuccess; ++rk)
      for (int h = 0; h < 2 && r == cudaSuccess; ++h)
        r = shift(L->d_f2 + L->f2_off[i] + rk * rank_bytes + ((size_t)h * hd.E + e) * sizeof(F2Gu));
  }
  cudaSetDevice(prev);
  return r == cudaSuccess ? BITSMOE_OK : cuda_fail(r);
}

}  // extern "C"
