// Importance beta of every spectral unit, from calibration tokens (the input of the bit
// allocation), on the GPU.
//
// The paper weighs the loss of quantising a unit by how strongly the calibration
// activations excite it (Sec. "Shared-basis Spectral Decomposition", the reconstruction
// loss; appendix Eqs. app_affinity_gram, app_beta_def, app_down_beta_approx,
// app_unified_beta_def):
//
//   H_e    = X Diag(g_e) X^T          activation metric of expert e (g_e: the tokens'
//                                     routing affinities to e, their gate weights)
//   beta   = phi_k^T H_e phi_k        gate, up   (phi_k: the shared input basis)
//          = sum_t g_{t,e} (phi_k^T x_t)^2 = sum_t g_{t,e} z_{k,t}^2
//   beta   = p_k^T H_e p_k            down       (p_k: the expert's spectral vector, H_e
//                                     over the expert's SwiGLU outputs h_t)
//          = sum_t g_{t,e} (p_k^T h_{t,e})^2
//
// all on the float factors of the decomposition, before anything is quantised.  Steps:
//
//   k_imp_route    one block per token: the k largest logits (ties to the lower index),
//                  softmax over them -> the dense affinity matrix G (T x E) and, per
//                  expert, the list of its tokens with their gate weights
//   k_gemm<Z>      Z_h = Phi_h^T X for h = gate, up            (n x T)
//   k_gemm<BGU>    beta_h[e, k] = sum_t Z_h[k, t]^2 G[t, e]    (a contraction over tokens)
//   k_gemm<AG>     a_g = P_g,e (alpha_g,e * Z_g[:, tokens of e])          per expert
//   k_gemm<AUH>    h   = SiLU(a_g) * (P_u,e (alpha_u,e * Z_u[:, tokens]))  per expert
//   k_gemm<DN>     beta_dn[e, k] = sum_j g_j (P_dn,e^T h)[k, j]^2          per expert
//
// Every contraction is fp32 on the CUDA cores (64 x 64 output tiles, four by four per
// thread): the factors are fp32 and the result is compared with an fp64 oracle at a tight
// tolerance, which bf16 tensor-core operands would not meet.
#include <cuda_runtime.h>
#include <stdint.h>

#include <algorithm>

#include "device.cuh"
#include "internal.h"

namespace {

constexpr int kTM = 64, kTN = 64, kTK = 16;   // output tile and K step
constexpr int kGT = 256;                      // threads of a GEMM block (16 x 16, 4 x 4 each)

enum GemmKind { kZ = 0, kBGU = 1, kAG = 2, kAUH = 3, kDN = 4 };

struct ImpArgs {
  const uint16_t* x;       // [T][D] bf16
  const float* logits;     // [T][E]
  const float* phi[2];     // gate, up: [D][n]
  const float* alpha[2];   // gate, up: [E][n]
  const float* P[3];       // gate, up, down: [E][I][n]
  float* beta;             // [3][E][n]
  int T, D, E, I, n, k;
  // workspace
  float* G;                // [T][E] affinities
  float* z;                // [2][n][T]
  int* cnt;                // [E] tokens per expert
  int* off;                // [E + 1] start of each expert's list (exclusive scan of cnt)
  int* tok;                // [T * k] token of each (expert, slot), grouped by expert
  float* tw;               // [T * k] its gate weight
  float* ag;               // [I][T * k] a_g, then h, by the expert's columns
  int* status;
};

__device__ __forceinline__ float bf16f(uint16_t v) { return __uint_as_float((uint32_t)v << 16); }

// ---------------------------------------------------------------------------
// Routing of every token (one block each), the same rule as the forward.
// ---------------------------------------------------------------------------
__global__ void k_imp_route(ImpArgs a) {
  extern __shared__ uint32_t keys[];   // [E], then sel_e [k], sel_w [k]
  int* sel_e = reinterpret_cast<int*>(keys + a.E);
  float* sel_w = reinterpret_cast<float*>(sel_e + a.k);
  const int t = blockIdx.x, tid = threadIdx.x;
  for (int i = tid; i < a.E; i += blockDim.x) {
    keys[i] = order_key(a.logits[(size_t)t * a.E + i]);
    a.G[(size_t)t * a.E + i] = 0.f;
  }
  __syncthreads();
  for (int i = tid; i < a.E; i += blockDim.x) {
    const uint32_t key = keys[i];
    int rank = 0;
    for (int f = 0; f < a.E; ++f) {
      const uint32_t o = keys[f];
      rank += (o > key) | ((o == key) & (f < i));
    }
    if (rank < a.k) {
      sel_e[rank] = i;
      sel_w[rank] = key ? __uint_as_float((key & 0x80000000u) ? (key & 0x7FFFFFFFu) : ~key)
                        : __int_as_float(0x7FC00000);
    }
  }
  __syncthreads();
  if (tid < 32) {
    const float m = sel_w[0];
    const float ev = tid < a.k ? expf(sel_w[tid] - m) : 0.f;
    float sum = ev;
#pragma unroll
    for (int o = 16; o; o >>= 1) sum += __shfl_xor_sync(0xFFFFFFFFu, sum, o);
    if (tid < a.k) {
      const float w = ev * (1.f / sum);
      a.G[(size_t)t * a.E + sel_e[tid]] = w;
      if (w != 0.f) atomicAdd(a.cnt + sel_e[tid], 1);   // the lists keep the tokens with g > 0
    }
  }
}

// Token lists per expert: one block; the experts' starts by an exclusive scan, then each
// token's (expert, weight) pairs in token order (one thread per expert keeps the order).
__global__ void k_imp_lists(ImpArgs a) {
  __shared__ int base[1025];
  if (threadIdx.x == 0) {
    int run = 0;
    for (int e = 0; e < a.E; ++e) {
      base[e] = run;
      a.off[e] = run;
      run += a.cnt[e];
    }
    a.off[a.E] = run;
  }
  __syncthreads();
  for (int e = threadIdx.x; e < a.E; e += blockDim.x) {
    int w = base[e];
    for (int t = 0; t < a.T; ++t) {
      const float g = a.G[(size_t)t * a.E + e];
      if (g != 0.f) {
        a.tok[w] = t;
        a.tw[w] = g;
        ++w;
      }
    }
  }
}

// ---------------------------------------------------------------------------
// fp32 contractions C = A B (M x N over K) with the operands of each step read in place
// (transposed, gathered, squared or scaled on load) and the step's epilogue.
// ---------------------------------------------------------------------------
template <int KIND>
struct Op {
  int M, N, K, e, col0;   // col0: first column of the expert's token list
};

template <int KIND>
__device__ __forceinline__ Op<KIND> op_of(const ImpArgs& a) {
  Op<KIND> o;
  o.e = blockIdx.z;
  o.col0 = 0;
  if (KIND == kZ) {
    o.M = a.n; o.N = a.T; o.K = a.D;
  } else if (KIND == kBGU) {
    o.M = a.n; o.N = a.E; o.K = a.T;
  } else if (KIND == kAG || KIND == kAUH) {
    o.col0 = a.off[o.e];
    o.M = a.I; o.N = a.off[o.e + 1] - o.col0; o.K = a.n;
  } else {
    o.col0 = a.off[o.e];
    o.M = a.n; o.N = a.off[o.e + 1] - o.col0; o.K = a.I;
  }
  return o;
}

// A(m, kk) and B(kk, j) of each kind (in bounds: the caller checks)
template <int KIND>
__device__ __forceinline__ float a_at(const ImpArgs& a, const Op<KIND>& o, int m, int kk) {
  if (KIND == kZ) return a.phi[o.e][(size_t)kk * a.n + m];                       // Phi_h^T
  if (KIND == kBGU) {
    const float v = a.z[((size_t)o.e * a.n + m) * a.T + kk];
    return v * v;                                                                  // z^2
  }
  if (KIND == kAG) return a.P[0][((size_t)o.e * a.I + m) * a.n + kk];
  if (KIND == kAUH) return a.P[1][((size_t)o.e * a.I + m) * a.n + kk];
  return a.P[2][((size_t)o.e * a.I + kk) * a.n + m];                               // P_dn^T
}
template <int KIND>
__device__ __forceinline__ float b_at(const ImpArgs& a, const Op<KIND>& o, int kk, int j) {
  const size_t TK = (size_t)a.T * a.k;
  if (KIND == kZ) return bf16f(a.x[(size_t)j * a.D + kk]);                        // X^T
  if (KIND == kBGU) return a.G[(size_t)kk * a.E + j];
  if (KIND == kAG || KIND == kAUH) {
    const int h = KIND == kAG ? 0 : 1;
    const int t = a.tok[o.col0 + j];
    return a.alpha[h][(size_t)o.e * a.n + kk] * a.z[((size_t)h * a.n + kk) * a.T + t];
  }
  return a.ag[(size_t)kk * TK + o.col0 + j];                                      // h
}
// whether consecutive kk are contiguous in memory (then a warp walks kk while loading)
template <int KIND>
__host__ __device__ constexpr bool a_k_contig() { return KIND == kBGU || KIND == kAG || KIND == kAUH; }
template <int KIND>
__host__ __device__ constexpr bool b_k_contig() { return KIND == kZ; }

template <int KIND>
__global__ void __launch_bounds__(kGT) k_gemm(ImpArgs a) {
  __shared__ float As[kTK][kTM + 4];
  __shared__ float Bs[kTK][kTN + 4];
  const Op<KIND> o = op_of<KIND>(a);
  const int m0 = blockIdx.y * kTM, j0 = blockIdx.x * kTN;
  if (m0 >= o.M || j0 >= o.N) return;
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  float acc[4][4];
#pragma unroll
  for (int r = 0; r < 4; ++r)
#pragma unroll
    for (int c = 0; c < 4; ++c) acc[r][c] = 0.f;
  for (int k0 = 0; k0 < o.K; k0 += kTK) {
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      const int idx = tid + kGT * r;
      int mm, kk, jj, kb;
      if (a_k_contig<KIND>()) {
        kk = idx % kTK;
        mm = idx / kTK;
      } else {
        mm = idx % kTM;
        kk = idx / kTM;
      }
      if (b_k_contig<KIND>()) {
        kb = idx % kTK;
        jj = idx / kTK;
      } else {
        jj = idx % kTN;
        kb = idx / kTN;
      }
      const int gm = m0 + mm, gk = k0 + kk, gj = j0 + jj, gkb = k0 + kb;
      As[kk][mm] = (gm < o.M && gk < o.K) ? a_at<KIND>(a, o, gm, gk) : 0.f;
      Bs[kb][jj] = (gkb < o.K && gj < o.N) ? b_at<KIND>(a, o, gkb, gj) : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < kTK; ++kk) {
      const float4 av = *reinterpret_cast<const float4*>(&As[kk][ty * 4]);
      const float4 bv = *reinterpret_cast<const float4*>(&Bs[kk][tx * 4]);
      const float ar[4] = {av.x, av.y, av.z, av.w}, br[4] = {bv.x, bv.y, bv.z, bv.w};
#pragma unroll
      for (int r = 0; r < 4; ++r)
#pragma unroll
        for (int c = 0; c < 4; ++c) acc[r][c] = fmaf(ar[r], br[c], acc[r][c]);
    }
    __syncthreads();
  }
  // epilogues
  const size_t TK = (size_t)a.T * a.k;
  if (KIND == kDN) {
    // beta_dn[e, m] += sum_j g_j acc(m, j)^2: the 16 threads of a row group add their columns
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      float v = 0.f;
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const int gj = j0 + tx * 4 + c;
        if (gj < o.N) v = fmaf(a.tw[o.col0 + gj], acc[r][c] * acc[r][c], v);
      }
#pragma unroll
      for (int sh = 8; sh; sh >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, sh);
      const int gm = m0 + ty * 4 + r;
      if (tx == 0 && gm < o.M && v != 0.f) atomicAdd(a.beta + ((size_t)2 * a.E + o.e) * a.n + gm, v);
    }
    return;
  }
#pragma unroll
  for (int r = 0; r < 4; ++r) {
    const int gm = m0 + ty * 4 + r;
    if (gm >= o.M) continue;
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const int gj = j0 + tx * 4 + c;
      if (gj >= o.N) continue;
      if (KIND == kZ) {
        a.z[((size_t)o.e * a.n + gm) * a.T + gj] = acc[r][c];
      } else if (KIND == kBGU) {
        a.beta[((size_t)o.e * a.E + gj) * a.n + gm] = acc[r][c];
      } else if (KIND == kAG) {
        a.ag[(size_t)gm * TK + o.col0 + gj] = acc[r][c];
      } else {   // h = SiLU(a_g) * a_u
        float* hp = a.ag + (size_t)gm * TK + o.col0 + gj;
        const float g = *hp;
        *hp = g / (1.f + expf(-g)) * acc[r][c];
      }
    }
  }
}

}  // namespace

namespace bmoe {

struct ImpLayout {
  size_t G, z, cnt, off, tok, tw, ag, total;
};
static ImpLayout imp_layout(int64_t T, int E, int I, int n, int k) {
  ImpLayout l;
  size_t o = 0;
  auto put = [&](size_t bytes) {
    const size_t r = o;
    o = (o + bytes + 255) / 256 * 256;
    return r;
  };
  l.G = put((size_t)T * E * 4);
  l.z = put((size_t)2 * n * T * 4);
  l.cnt = put((size_t)E * 4);
  l.off = put(((size_t)E + 1) * 4);
  l.tok = put((size_t)T * k * 4);
  l.tw = put((size_t)T * k * 4);
  l.ag = put((size_t)I * T * k * 4);
  l.total = o;
  return l;
}

}  // namespace bmoe

extern "C" {

size_t bitsmoe_importance_workspace_bytes(int64_t T, int E, int I, int n, int top_k) {
  if (T < 0 || E < 1 || I < 1 || n < 1 || top_k < 1 || top_k > std::min(E, 32)) return 0;
  return bmoe::imp_layout(T, E, I, n, top_k).total;
}

int bitsmoe_importance(const void* x, const float* logits, int64_t T, int D, int E, int I, int n, int top_k,
                       const float* const basis[2], const float* const alpha[2], const float* const factor[3],
                       float* beta, void* ws, size_t ws_bytes, void* stream) {
  if (T < 0 || D < 1 || E < 1 || E > 1024 || I < 1 || n < 1 || top_k < 1 || top_k > std::min(E, 32))
    return BITSMOE_ERR_INVALID_ARG;
  if (T > (1 << 24) || (int64_t)I * T * top_k > (1ll << 31)) return BITSMOE_ERR_SHAPE;
  if (!basis || !alpha || !factor || !beta || !ws) return BITSMOE_ERR_INVALID_ARG;
  if (!basis[0] || !basis[1] || !alpha[0] || !alpha[1] || !factor[0] || !factor[1] || !factor[2])
    return BITSMOE_ERR_INVALID_ARG;
  if (T > 0 && (!x || !logits)) return BITSMOE_ERR_INVALID_ARG;
  const bmoe::ImpLayout l = bmoe::imp_layout(T, E, I, n, top_k);
  if (ws_bytes < l.total) return BITSMOE_ERR_WORKSPACE_TOO_SMALL;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  auto fail = [](cudaError_t e) { return bmoe::record_cuda_error((int)e); };
  cudaError_t e = cudaMemsetAsync(beta, 0, (size_t)3 * E * n * 4, st);
  if (e != cudaSuccess) return fail(e);
  if (T == 0) return BITSMOE_OK;
  uint8_t* w = static_cast<uint8_t*>(ws);
  ImpArgs a;
  a.x = static_cast<const uint16_t*>(x);
  a.logits = logits;
  for (int h = 0; h < 2; ++h) {
    a.phi[h] = basis[h];
    a.alpha[h] = alpha[h];
  }
  for (int h = 0; h < 3; ++h) a.P[h] = factor[h];
  a.beta = beta;
  a.T = (int)T; a.D = D; a.E = E; a.I = I; a.n = n; a.k = top_k;
  a.G = reinterpret_cast<float*>(w + l.G);
  a.z = reinterpret_cast<float*>(w + l.z);
  a.cnt = reinterpret_cast<int*>(w + l.cnt);
  a.off = reinterpret_cast<int*>(w + l.off);
  a.tok = reinterpret_cast<int*>(w + l.tok);
  a.tw = reinterpret_cast<float*>(w + l.tw);
  a.ag = reinterpret_cast<float*>(w + l.ag);
  a.status = nullptr;
  if ((e = cudaMemsetAsync(a.cnt, 0, (size_t)E * 4, st)) != cudaSuccess) return fail(e);
  const size_t rsm = ((size_t)E + 2 * top_k) * 4;
  if (rsm > 48 * 1024) return BITSMOE_ERR_SHAPE;
  k_imp_route<<<(unsigned)T, 256, rsm, st>>>(a);
  k_imp_lists<<<1, 256, 0, st>>>(a);
  const unsigned tT = (unsigned)((T + kTN - 1) / kTN);
  k_gemm<kZ><<<dim3(tT, (n + kTM - 1) / kTM, 2), kGT, 0, st>>>(a);
  k_gemm<kBGU><<<dim3((E + kTN - 1) / kTN, (n + kTM - 1) / kTM, 2), kGT, 0, st>>>(a);
  // an expert has at most T tokens; blocks past its count return at once
  k_gemm<kAG><<<dim3(tT, (I + kTM - 1) / kTM, E), kGT, 0, st>>>(a);
  k_gemm<kAUH><<<dim3(tT, (I + kTM - 1) / kTM, E), kGT, 0, st>>>(a);
  k_gemm<kDN><<<dim3(tT, (n + kTM - 1) / kTM, E), kGT, 0, st>>>(a);
  e = cudaGetLastError();
  return e == cudaSuccess ? BITSMOE_OK : fail(e);
}

}  // extern "C"
