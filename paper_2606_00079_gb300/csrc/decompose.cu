// Shared-basis spectral decomposition of one projection type over the E experts
// (Sec. "Shared-basis Spectral Decomposition": Eq. shared_basis_input_proj for
// gate/up, the concatenation along input channels for down; Definitions
// spectral_energy_matrix / spectral_matrix), and the calibration Gram
// H = X Diag(g) X^T of the appendix (Eq. app_affinity_gram).
//
//   side "in"  (gate/up): W_e is d x D (rows: the expert's intermediate
//              channels), W_cat = [W_1; ...; W_E] = U S Phi^T, P~_cat = U S.
//   side "out" (down):    W_e is D x d, W_cat = [W_1 ... W_E] = Phi S V^T,
//              P~_cat = V S, split by the experts' input channels.
//
// Both sides are the same computation on A = the R x D matrix (R = E d) whose
// row r = (e, i) is row i of W_e ("in") or column i of W_e ("out"):
//   G   = A^T A (D x D, symmetric; its eigenvectors are Phi, its eigenvalues S^2)
//   P~  = A Phi (R x n), alpha_{e,k} = ||P~_e[:, k]||, P_e = P~_e / alpha_e.
// Kernels: a fp32 tile GEMM (CUDA cores) for G and P~ -- fp32 throughout,
// because the eigenvectors of G move with its rounding error divided by the
// eigenvalue gaps; a cyclic two-sided Jacobi eigensolver for G in one
// cooperative kernel (every block recomputes the round's rotations, rotates the
// rows of G and of V^T that it owns, one grid barrier per round); a sort of the
// eigenvalues with the sign of each eigenvector fixed (largest component
// positive); the column norms and the unit-major P.
#include <cuda.h>
#include <cuda_bf16.h>

#include <algorithm>
#include <cstring>

#include "device.cuh"
#include "internal.h"

#define BM_CK(call)                                             \
  do {                                                          \
    const cudaError_t e_ = (call);                              \
    if (e_ != cudaSuccess) return bmoe::record_cuda_error((int)e_); \
  } while (0)

namespace {

constexpr int kTM = 128, kTN = 128, kTK = 8, kGT = 256;   // GEMM tile and threads (8 x 8 outputs a thread)

__device__ __forceinline__ float to_f(float v) { return v; }
__device__ __forceinline__ float to_f(uint16_t v) { return __uint_as_float((uint32_t)v << 16); }   // bf16 bits

// Four consecutive elements of a row (a is a multiple of 4), zero past `lim`.
template <typename T>
__device__ __forceinline__ float4 load4(const T* row, int a, int lim) {
  float4 v;
  v.x = a < lim ? to_f(row[a]) : 0.f;
  v.y = a + 1 < lim ? to_f(row[a + 1]) : 0.f;
  v.z = a + 2 < lim ? to_f(row[a + 2]) : 0.f;
  v.w = a + 3 < lim ? to_f(row[a + 3]) : 0.f;
  return v;
}

// The 8 x 8 outputs of a thread over one K-step pair of tiles.
__device__ __forceinline__ void tile_fma(const float (*As)[kTM + 4], const float (*Bs)[kTN + 4], int ty, int tx,
                                         float (&acc)[8][8]) {
#pragma unroll
  for (int k = 0; k < kTK; ++k) {
    const float4 a0 = *reinterpret_cast<const float4*>(&As[k][ty * 8]);
    const float4 a1 = *reinterpret_cast<const float4*>(&As[k][ty * 8 + 4]);
    const float4 b0 = *reinterpret_cast<const float4*>(&Bs[k][tx * 8]);
    const float4 b1 = *reinterpret_cast<const float4*>(&Bs[k][tx * 8 + 4]);
    const float a[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
    const float b[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
      for (int j = 0; j < 8; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
  }
}

// G = sum_r w_r A[r, :]^T A[r, :]  (A: R x D, row stride lda; w = null: all 1).
// One block per upper-triangle tile pair (ta <= tb) of 128 x 128; the lower
// triangle is written by mirroring (so G is exactly symmetric).  The K loop runs over the rows r in steps
// of 8 with the next step's loads in flight during the current step's FMAs.
template <typename T>
__global__ void __launch_bounds__(kGT) k_gram(const T* __restrict__ A, const float* __restrict__ w, int64_t R, int D,
                                              int64_t lda, float* __restrict__ G, int64_t ldg, int ntile) {
  __shared__ __align__(16) float As[2][kTK][kTM + 4];
  __shared__ __align__(16) float Bs[2][kTK][kTN + 4];
  int t = blockIdx.x, ta = 0;
  while (t >= ntile - ta) {
    t -= ntile - ta;
    ++ta;
  }
  const int tb = ta + t;
  const int a0 = ta * kTM, b0 = tb * kTN;
  const int tid = threadIdx.x, ty = tid >> 4, tx = tid & 15;
  const int lk = tid >> 5, lc = (tid & 31) * 4;   // loader: row k of the step, 4 columns
  float acc[8][8];
#pragma unroll
  for (int i = 0; i < 8; ++i)
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[i][j] = 0.f;
  auto fetch = [&](int64_t r0, float4& va, float4& vb) {
    const int64_t r = r0 + lk;
    if (r < R) {
      const T* row = A + r * lda;
      const float wr = w ? w[r] : 1.f;
      va = load4(row, a0 + lc, D);
      vb = load4(row, b0 + lc, D);
      va.x *= wr;
      va.y *= wr;
      va.z *= wr;
      va.w *= wr;
    } else {
      va = vb = make_float4(0.f, 0.f, 0.f, 0.f);
    }
  };
  float4 va, vb;
  fetch(0, va, vb);
  int buf = 0;
  for (int64_t r0 = 0; r0 < R; r0 += kTK) {
    *reinterpret_cast<float4*>(&As[buf][lk][lc]) = va;
    *reinterpret_cast<float4*>(&Bs[buf][lk][lc]) = vb;
    __syncthreads();
    if (r0 + kTK < R) fetch(r0 + kTK, va, vb);
    tile_fma(As[buf], Bs[buf], ty, tx, acc);
    buf ^= 1;
  }
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int a = a0 + ty * 8 + i;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int b = b0 + tx * 8 + j;
      if (a < D && b < D && (ta != tb || a <= b)) {   // exactly symmetric: one value per pair
        G[(size_t)a * ldg + b] = acc[i][j];
        G[(size_t)b * ldg + a] = acc[i][j];
      }
    }
  }
}

// C = A Phi  (A: R x D fp32 row-major, Phi: D x n row-major, C: R x n).  Tiles of
// 128 rows of A (read 8 columns at a time and transposed into shared memory) by 128
// columns of Phi.
__global__ void __launch_bounds__(kGT) k_project(const float* __restrict__ A, const float* __restrict__ Phi, int64_t R,
                                                 int D, int n, float* __restrict__ C) {
  __shared__ __align__(16) float As[2][kTK][kTM + 4];
  __shared__ __align__(16) float Bs[2][kTK][kTN + 4];
  const int64_t m0 = (int64_t)blockIdx.y * kTM;
  const int n0 = blockIdx.x * kTN;
  const int tid = threadIdx.x, ty = tid >> 4, tx = tid & 15;
  const int am = tid >> 1, ak = (tid & 1) * 4;     // A loader: row am, columns ak .. ak + 3 of the step
  const int bk = tid >> 5, bc = (tid & 31) * 4;    // Phi loader: row bk, columns bc .. bc + 3
  float acc[8][8];
#pragma unroll
  for (int i = 0; i < 8; ++i)
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[i][j] = 0.f;
  auto fetch = [&](int k0, float4& va, float4& vb) {
    va = m0 + am < R ? load4(A + (m0 + am) * D, k0 + ak, D) : make_float4(0.f, 0.f, 0.f, 0.f);
    vb = k0 + bk < D ? load4(Phi + (size_t)(k0 + bk) * n, n0 + bc, n) : make_float4(0.f, 0.f, 0.f, 0.f);
  };
  float4 va, vb;
  fetch(0, va, vb);
  int buf = 0;
  for (int k0 = 0; k0 < D; k0 += kTK) {
    As[buf][ak][am] = va.x;
    As[buf][ak + 1][am] = va.y;
    As[buf][ak + 2][am] = va.z;
    As[buf][ak + 3][am] = va.w;
    *reinterpret_cast<float4*>(&Bs[buf][bk][bc]) = vb;
    __syncthreads();
    if (k0 + kTK < D) fetch(k0 + kTK, va, vb);
    tile_fma(As[buf], Bs[buf], ty, tx, acc);
    buf ^= 1;
  }
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int64_t m = m0 + ty * 8 + i;
    if (m >= R) continue;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int c = n0 + tx * 8 + j;
      if (c < n) C[m * n + c] = acc[i][j];
    }
  }
}

// A for side "out": row (e, i) = column i of W_e (W: E x D x d) -> A: (E d) x D.
__global__ void k_transpose_out(const float* __restrict__ W, int E, int D, int d, float* __restrict__ A) {
  __shared__ float tile[32][33];
  const int e = blockIdx.z;
  const int i0 = blockIdx.x * 32, a0 = blockIdx.y * 32;
  const float* We = W + (size_t)e * D * d;
  for (int y = threadIdx.y; y < 32; y += blockDim.y) {
    const int a = a0 + y, i = i0 + threadIdx.x;
    tile[y][threadIdx.x] = (a < D && i < d) ? We[(size_t)a * d + i] : 0.f;
  }
  __syncthreads();
  for (int y = threadIdx.y; y < 32; y += blockDim.y) {
    const int i = i0 + y, a = a0 + threadIdx.x;
    if (i < d && a < D) A[((size_t)e * d + i) * D + a] = tile[threadIdx.x][y];
  }
}

// ---------------------------------------------------------------------------
// Cyclic two-sided Jacobi (Golub & Van Loan, Alg. 8.5.3, parallel ordering).
// Players 0 .. m-1 (m = n rounded up to even; player n is a dummy when n is
// odd); in round r of a sweep the pairs are the positions (i, m-1-i) of the
// circle arrangement in which player 0 stays and the others advance by r.  For
// a pair (p, q) with a_pq != 0: tau = (a_qq - a_pp) / (2 a_pq), t = sign(tau) /
// (|tau| + sqrt(1 + tau^2)), c = 1 / sqrt(1 + t^2), s = t c; the rotation J
// (J_pp = J_qq = c, J_pq = s, J_qp = -s) makes (J^T G J)_pq = 0.  Stored per
// index j: its partner, c and the signed sine (-s for p, +s for q), so that
// both the row and the column rotations read new_j = c v_j + s_j v_partner.  A
// rotation is skipped (identity) while |a_pq| <= tol sqrt(|a_pp a_qq|) or |a_pq|
// <= 4e-7 max_j |a_jj| (rounding noise of fp32); the solver stops after the
// first sweep that skips every rotation.
//
// Every block computes all rotations of a round (each needs a_pp, a_qq, a_pq);
// it then rotates the rows of G and V^T of its own pairs.  The three numbers are
// read from a small table, not from G: the block that owns row p in round g
// writes (a_pp, a_p,partner) of the updated row for round g + 1 into the table
// of parity (g + 1) & 1, so no block reads G while another one rewrites it, and
// one grid barrier per round suffices.
// ---------------------------------------------------------------------------
struct JacobiArgs {
  float* G;          // n x ld (row stride ld), symmetric, overwritten (diagonal: the eigenvalues);
                     // columns n .. ld - 1 zero
  float* Vt;         // n x ld: row j = eigenvector j (set to the identity here)
  float2* tab;       // [2][m]: (a_jj, a_j,partner) of each index for a round
  int n, ld;
  int batch;         // pairs whose rows are in shared memory at once
  int max_sweeps;
  float tol;
  uint32_t* bar;     // grid-barrier counter (zero at launch)
  int* status;       // BITSMOE_ERR_TIMEOUT if a wait ran out
  int* sweeps;       // sweeps run (written by block 0)
  long long spin;    // bound of each barrier wait, in SM clocks
};

constexpr int kJBatch = 16;

// Clock totals of the solver's phases per block, compiled in only with -DBITSMOE_JACOBI_TRACE
// (timing studies): [0] rotations, [1] rows of G in, [2] rotations of G's rows, [3] rows of
// V^T, [4] barrier.
#ifdef BITSMOE_JACOBI_TRACE
__device__ unsigned long long g_jacobi_trace[1024][8];
#define JT_START() long long jt_ = clock64()
#define JT_MARK(i)                                                            \
  do {                                                                        \
    const long long jn_ = clock64();                                          \
    if (threadIdx.x == 0) g_jacobi_trace[blockIdx.x & 1023][(i)] += jn_ - jt_; \
    jt_ = jn_;                                                                \
  } while (0)
#else
#define JT_START() \
  do {             \
  } while (0)
#define JT_MARK(i) \
  do {             \
  } while (0)
#endif

__device__ __forceinline__ int jacobi_player(int pos, int r, int m) { return pos == 0 ? 0 : 1 + (pos - 1 + r) % (m - 1); }
__device__ __forceinline__ int jacobi_partner(int x, int r, int m) {
  const int pos = x == 0 ? 0 : 1 + ((x - 1 - r) % (m - 1) + (m - 1)) % (m - 1);
  return jacobi_player(m - 1 - pos, r, m);
}

__device__ __forceinline__ bool grid_sync_bounded(uint32_t* bar, uint32_t target, long long spin, int* status,
                                                  int* ok) {
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    asm volatile("red.release.gpu.global.add.u32 [%0], 1;" ::"l"(bar) : "memory");
    const long long t0 = clock64();
    int good = 1;
    for (;;) {
      uint32_t v;
      asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(bar) : "memory");
      if ((int)(v - target) >= 0) break;
      if (clock64() - t0 > spin) {
        atomicCAS(status, 0, BITSMOE_ERR_TIMEOUT);
        good = 0;
        break;
      }
    }
    __threadfence();
    *ok = good;
  }
  __syncthreads();
  return *ok != 0;
}

__device__ __forceinline__ void cp16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(dst)), "l"(src) : "memory");
}

// Rows (lo, hi) of the batch's pairs of M (row stride ld) into X[2j], X[2j + 1] by 16-byte
// copies of every thread, all in flight at once; only the rotated pairs when `only_rot`.
__device__ __forceinline__ void jacobi_rows_in(const float* M, int ld, int bn, const int* blo, const int* bhi,
                                              const float* sj, bool only_rot, int n, float* X) {
  const int q4 = ld / 4;
  for (int row = 0; row < 2 * bn; ++row) {
    const int jj = row >> 1, x = (row & 1) ? bhi[jj] : blo[jj];
    if (x >= n || (only_rot && sj[bhi[jj]] == 0.f)) continue;
    for (int c4 = threadIdx.x; c4 < q4; c4 += blockDim.x)
      cp16(X + (size_t)row * ld + 4 * c4, M + (size_t)x * ld + 4 * c4);
  }
  asm volatile("cp.async.wait_all;" ::: "memory");
  __syncthreads();
}
// ... and back (16-byte stores through L2).
__device__ __forceinline__ void jacobi_rows_out(float* M, int ld, int bn, const int* blo, const int* bhi,
                                               const float* sj, bool only_rot, int n, const float* X) {
  const int q4 = ld / 4;
  for (int row = 0; row < 2 * bn; ++row) {
    const int jj = row >> 1, x = (row & 1) ? bhi[jj] : blo[jj];
    if (x >= n || (only_rot && sj[bhi[jj]] == 0.f)) continue;
    for (int c4 = threadIdx.x; c4 < q4; c4 += blockDim.x)
      __stcg(reinterpret_cast<float4*>(M + (size_t)x * ld) + c4,
             *reinterpret_cast<const float4*>(X + (size_t)row * ld + 4 * c4));
  }
}
// Row rotation of the batch's row pairs in place (16 bytes a thread at a time).
__device__ __forceinline__ void jacobi_rotate_rows(int ld, int bn, const int* blo, const int* bhi, const float* cj,
                                                   const float* sj, bool only_rot, float* X) {
  const int q4 = ld / 4;
  for (int jj = 0; jj < bn; ++jj) {
    const int lo = blo[jj], hi = bhi[jj];
    const float c = cj[lo], s_lo = sj[lo], s_hi = sj[hi];
    if (only_rot && s_hi == 0.f) continue;
    float4* xl = reinterpret_cast<float4*>(X + (size_t)(2 * jj) * ld);
    float4* xh = reinterpret_cast<float4*>(X + (size_t)(2 * jj + 1) * ld);
    for (int c4 = threadIdx.x; c4 < q4; c4 += blockDim.x) {
      const float4 a = xl[c4], b = xh[c4];
      xl[c4] = make_float4(c * a.x + s_lo * b.x, c * a.y + s_lo * b.y, c * a.z + s_lo * b.z, c * a.w + s_lo * b.w);
      xh[c4] = make_float4(c * b.x + s_hi * a.x, c * b.y + s_hi * a.y, c * b.z + s_hi * a.z, c * b.w + s_hi * a.w);
    }
  }
}

__global__ void __launch_bounds__(512, 1) k_jacobi(JacobiArgs ja) {
  extern __shared__ __align__(16) uint8_t jsm[];
  const int n = ja.n, ld = ja.ld, m = n + (n & 1), half = m / 2;
  float* X = reinterpret_cast<float*>(jsm);                           // [2 batch][ld] a batch's rows
  int* partner = reinterpret_cast<int*>(X + (size_t)2 * ja.batch * ld);   // [m]
  float* cj = reinterpret_cast<float*>(partner + m);                  // [m]
  float* sj = cj + m;                                                 // [m]
  __shared__ int active, ok;
  // a batch's pairs: lower and upper index, first player, next partners, rotated diagonal
  __shared__ int blo[kJBatch], bhi[kJBatch], bp[kJBatch], bnl[kJBatch], bnh[kJBatch];
  __shared__ float bdl[kJBatch], bdh[kJBatch];
  const int tid = threadIdx.x, nt = blockDim.x, blk = blockIdx.x, nb = gridDim.x;
  // V^T = I (padding columns 0); the table of round 0
  for (size_t i = (size_t)blk * nt + tid; i < (size_t)n * ld; i += (size_t)nb * nt)
    ja.Vt[i] = (i / ld == i % ld) ? 1.f : 0.f;
  for (int x = blk * nt + tid; x < m; x += nb * nt) {
    const int y = jacobi_partner(x, 0, m);
    ja.tab[x] = x < n ? make_float2(ja.G[(size_t)x * ld + x], y < n ? ja.G[(size_t)x * ld + y] : 0.f)
                      : make_float2(0.f, 0.f);
  }
  uint32_t target = nb;
  if (!grid_sync_bounded(ja.bar, target, ja.spin, ja.status, &ok)) return;
  // absolute floor of the rotation test: a few units in the last place of the largest
  // diagonal element, below which an off-diagonal element is rounding noise
  __shared__ float dmax_s;
  {
    float dm = 0.f;
    for (int x = tid; x < n; x += nt) dm = fmaxf(dm, fabsf(__ldcg(ja.G + (size_t)x * ld + x)));
    for (int o = 16; o; o >>= 1) dm = fmaxf(dm, __shfl_xor_sync(0xFFFFFFFFu, dm, o));
    if (tid == 0) dmax_s = 0.f;
    __syncthreads();
    if ((tid & 31) == 0) atomicMax(reinterpret_cast<int*>(&dmax_s), __float_as_int(dm));   // non-negative floats
    __syncthreads();
  }
  const float atol = 4e-7f * dmax_s;
  int sweep = 0, g = 0;   // g: rounds run so far (table parity)
  for (; sweep < ja.max_sweeps; ++sweep) {
    int rotated = 0;
    for (int r = 0; r < m - 1; ++r, ++g) {
      JT_START();
      const float2* tin = ja.tab + (size_t)(g & 1) * m;
      float2* tout = ja.tab + (size_t)((g + 1) & 1) * m;
      const int rn = r + 1 < m - 1 ? r + 1 : 0;   // the next round (of this sweep or the next)
      if (tid == 0) active = 0;
      __syncthreads();
      // every rotation of the round, from the table
      int my_active = 0;
      for (int i = tid; i < half; i += nt) {
        const int p = jacobi_player(i, r, m), q = jacobi_player(m - 1 - i, r, m);
        float c = 1.f, s = 0.f;
        if (p < n && q < n) {
          const float2 tp = __ldcg(tin + p), tq = __ldcg(tin + q);
          const float app = tp.x, aqq = tq.x, apq = tp.y;
          if (fabsf(apq) > atol && fabsf(apq) > ja.tol * sqrtf(fabsf(app) * fabsf(aqq))) {
            const float tau = (aqq - app) / (2.f * apq);
            const float tt = (tau >= 0.f ? 1.f : -1.f) / (fabsf(tau) + sqrtf(1.f + tau * tau));
            c = 1.f / sqrtf(1.f + tt * tt);
            s = tt * c;
            ++my_active;
          }
        }
        partner[p] = q;
        partner[q] = p;
        cj[p] = c;
        cj[q] = c;
        sj[p] = -s;
        sj[q] = s;
      }
      if (my_active) atomicAdd(&active, my_active);
      __syncthreads();
      rotated += active;
      JT_MARK(0);
      // this block's pairs i = blk, blk + nb, ..., in batches of ja.batch
      const int npairs = blk < half ? (half - 1 - blk) / nb + 1 : 0;
      for (int b0 = 0; b0 < npairs; b0 += ja.batch) {
        const int bn = min(ja.batch, npairs - b0);
        if (tid < bn) {   // the batch's pairs and the next round's partners of their rows
          const int ii = blk + (b0 + tid) * nb;
          const int p = jacobi_player(ii, r, m), q = jacobi_player(m - 1 - ii, r, m);
          const int lo = p < q ? p : q, hi = p < q ? q : p;
          blo[tid] = lo;
          bhi[tid] = hi;
          bp[tid] = p;
          bnl[tid] = jacobi_partner(lo, rn, m);
          bnh[tid] = hi < n ? jacobi_partner(hi, rn, m) : n;
          if (sj[hi] != 0.f) {   // the rotated 2 x 2 block: off-diagonal 0, diagonal a_xx + (s_x / c) a_pq
            // (Golub & Van Loan's update, which keeps a_pp + a_qq to one rounding per element)
            const float apq = __ldcg(tin + p).y, cc = cj[lo];
            bdl[tid] = __ldcg(tin + lo).x + (sj[lo] / cc) * apq;
            bdh[tid] = hi < n ? __ldcg(tin + hi).x + (sj[hi] / cc) * apq : 0.f;
          }
        }
        __syncthreads();
        // the rows of G (a dummy row reads as zeros)
        for (int jj = 0; jj < bn; ++jj)
          if (bhi[jj] >= n)
            for (int k = tid; k < ld; k += nt) X[(size_t)(2 * jj + 1) * ld + k] = 0.f;
        jacobi_rows_in(ja.G, ld, bn, blo, bhi, sj, false, n, X);
        JT_MARK(1);
        // row rotation in place, then the column rotation in place (index k with its partner:
        // the lower of the two updates both), the rotated 2 x 2 blocks, the next table entries
        jacobi_rotate_rows(ld, bn, blo, bhi, cj, sj, false, X);
        __syncthreads();
        for (int k = tid; k < m; k += nt) {
          const int pk = partner[k];
          if (pk < k) continue;   // the pair (k, pk) is updated once, by its lower index
          const float ck = cj[k], sk = sj[k], cp = cj[pk], sp = sj[pk];
          for (int row = 0; row < 2 * bn; ++row) {
            float* xr = X + (size_t)row * ld;
            const float a = xr[k], b = xr[pk];
            xr[k] = ck * a + sk * b;
            xr[pk] = cp * b + sp * a;
          }
        }
        __syncthreads();
        if (tid < bn) {
          const int lo = blo[tid], hi = bhi[tid];
          float* xl = X + (size_t)(2 * tid) * ld;
          float* xh = xl + ld;
          if (sj[hi] != 0.f) {
            xl[hi] = 0.f;
            xl[lo] = bdl[tid];
            if (hi < n) {
              xh[lo] = 0.f;
              xh[hi] = bdh[tid];
            }
          }
          if (n & 1) {   // the dummy column stays 0
            xl[m - 1] = 0.f;
            xh[m - 1] = 0.f;
          }
          tout[lo] = make_float2(xl[lo], bnl[tid] < n ? xl[bnl[tid]] : 0.f);
          tout[hi] = hi < n ? make_float2(xh[hi], bnh[tid] < n ? xh[bnh[tid]] : 0.f) : make_float2(0.f, 0.f);
        }
        __syncthreads();
        jacobi_rows_out(ja.G, ld, bn, blo, bhi, sj, false, n, X);
        __syncthreads();
        JT_MARK(2);
        // the rows of V^T of the batch's rotated pairs: row rotation only
        jacobi_rows_in(ja.Vt, ld, bn, blo, bhi, sj, true, n, X);
        jacobi_rotate_rows(ld, bn, blo, bhi, cj, sj, true, X);
        __syncthreads();
        jacobi_rows_out(ja.Vt, ld, bn, blo, bhi, sj, true, n, X);
        __syncthreads();
        JT_MARK(3);
      }
      target += nb;
      if (!grid_sync_bounded(ja.bar, target, ja.spin, ja.status, &ok)) return;
      JT_MARK(4);
    }
    if (rotated == 0) break;
  }
  if (blk == 0 && tid == 0 && ja.sweeps) *ja.sweeps = sweep;
}

// Rank of each eigenvalue (descending, ties to the lower index), the sign of
// each eigenvector (its largest |component| made positive, the first one on
// ties), then Phi[:, rank] = sign * V^T[j, :] and sigma[rank] = sqrt(max(lambda, 0))
// for the n_out leading ones.
__global__ void k_order(const float* __restrict__ G, const float* __restrict__ Vt, int n, int ld, int n_out,
                        float* __restrict__ phi, float* __restrict__ sigma) {
  const int j = blockIdx.x;   // one block per eigenvector
  __shared__ float red_v[32];
  __shared__ int red_i[32], red_c[32];
  __shared__ float red_n[32];
  __shared__ int rank_s;
  __shared__ float scale_s;
  const float lj = __ldg(G + (size_t)j * ld + j);
  int cnt = 0;
  for (int i = threadIdx.x; i < n; i += blockDim.x) {
    const float li = __ldg(G + (size_t)i * ld + i);
    cnt += (li > lj) | ((li == lj) & (i < j));
  }
  // largest |component| of V^T[j, :] (first on ties) and its squared norm (the vector is
  // rescaled to unit length: the rotations' rounding moves it by a few units in the last place)
  float bv = -1.f, nn = 0.f;
  int bi = 0x7FFFFFFF;
  const float* vr = Vt + (size_t)j * ld;
  for (int i = threadIdx.x; i < n; i += blockDim.x) {
    const float v = vr[i], a = fabsf(v);
    nn = fmaf(v, v, nn);
    if (a > bv || (a == bv && i < bi)) {
      bv = a;
      bi = i;
    }
  }
  for (int o = 16; o; o >>= 1) {
    nn += __shfl_xor_sync(0xFFFFFFFFu, nn, o);
    cnt += __shfl_xor_sync(0xFFFFFFFFu, cnt, o);
    const float ov = __shfl_xor_sync(0xFFFFFFFFu, bv, o);
    const int oi = __shfl_xor_sync(0xFFFFFFFFu, bi, o);
    if (ov > bv || (ov == bv && oi < bi)) {
      bv = ov;
      bi = oi;
    }
  }
  const int w = threadIdx.x >> 5, nw = blockDim.x >> 5;
  if ((threadIdx.x & 31) == 0) {
    red_v[w] = bv;
    red_i[w] = bi;
    red_c[w] = cnt;
    red_n[w] = nn;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int rk = 0;
    float v = -1.f, tn = 0.f;
    int vi = 0x7FFFFFFF;
    for (int q = 0; q < nw; ++q) {
      rk += red_c[q];
      tn += red_n[q];
      if (red_v[q] > v || (red_v[q] == v && red_i[q] < vi)) {
        v = red_v[q];
        vi = red_i[q];
      }
    }
    rank_s = rk;
    red_i[0] = vi;
    scale_s = tn > 0.f ? 1.f / sqrtf(tn) : 1.f;
  }
  __syncthreads();
  const int rk = rank_s;
  if (rk >= n_out) return;
  const float sg = vr[red_i[0]] < 0.f ? -scale_s : scale_s;
  for (int i = threadIdx.x; i < n; i += blockDim.x) phi[(size_t)i * n_out + rk] = sg * vr[i];
  if (threadIdx.x == 0) sigma[rk] = sqrtf(fmaxf(lj, 0.f));
}

// alpha[e][k] = ||P~[e d .. e d + d - 1][k]||_2 and P[e][k][i] = P~[e d + i][k] / alpha
// (0 where alpha = 0).  One block per (expert, 32 columns): the column sums of
// squares, then the scaled transpose through a 32 x 33 tile.
__global__ void k_normalize(const float* __restrict__ Pt, int E, int d, int n, float* __restrict__ alpha,
                            float* __restrict__ P) {
  __shared__ float tile[32][33];
  __shared__ float part[8][32];
  __shared__ float inv[32];
  const int e = blockIdx.y, k0 = blockIdx.x * 32;
  const int tx = threadIdx.x, ty = threadIdx.y;   // 32 x 8
  const float* base = Pt + (size_t)e * d * n;
  float ss = 0.f;
  const int k = k0 + tx;
  if (k < n)
    for (int i = ty; i < d; i += 8) {
      const float v = base[(size_t)i * n + k];
      ss = fmaf(v, v, ss);
    }
  part[ty][tx] = ss;
  __syncthreads();
  if (ty == 0) {
    float t = 0.f;
    for (int q = 0; q < 8; ++q) t += part[q][tx];
    const float a = sqrtf(t);
    if (k < n) alpha[(size_t)e * n + k] = a;
    inv[tx] = a > 0.f ? 1.f / a : 1.f;
  }
  __syncthreads();
  for (int i0 = 0; i0 < d; i0 += 32) {
    for (int y = ty; y < 32; y += 8) {
      const int i = i0 + y;
      tile[y][tx] = (i < d && k < n) ? base[(size_t)i * n + k] : 0.f;
    }
    __syncthreads();
    for (int y = ty; y < 32; y += 8) {
      const int kk = k0 + y, i = i0 + tx;
      if (kk < n && i < d) P[((size_t)e * n + kk) * d + i] = tile[tx][y] * inv[y];
    }
    __syncthreads();
  }
}

struct DecLayout {
  size_t A, G, Vt, Pt, tab, sync, total;
};
DecLayout dec_layout(int side, int E, int d, int D) {
  const size_t R = (size_t)E * d, n = std::min<size_t>(D, R);
  DecLayout l;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off = (off + bytes + 255) / 256 * 256;
    return o;
  };
  l.A = take(side == 1 ? R * D * 4 : 0);
  const size_t ld = (size_t)(D + (D & 1) + 3) / 4 * 4;   // row stride of G and V^T: 16-byte rows with the dummy column
  l.G = take((size_t)D * ld * 4);
  l.Vt = take((size_t)D * ld * 4);
  l.Pt = take(R * n * 4);
  l.tab = take((size_t)2 * (D + 1) * 8);
  l.sync = take(256);
  l.total = off;
  return l;
}

}  // namespace

extern "C" size_t bitsmoe_decompose_workspace_bytes(int side, int E, int d, int D) {
  if ((side != 0 && side != 1) || E < 1 || d < 1 || D < 1) return 0;
  return dec_layout(side, E, d, D).total;
}

extern "C" int bitsmoe_shared_basis(int side, const float* W, int E, int d, int D, float* phi, float* sigma,
                                    float* alpha, float* P, void* ws, size_t ws_bytes, int max_sweeps, int* sweeps,
                                    int* status, void* stream) {
  using namespace bmoe;
  if ((side != 0 && side != 1) || E < 1 || d < 1 || D < 2 || D > BITSMOE_DECOMPOSE_MAX_D || max_sweeps < 1 || !W || !phi ||
      !sigma || !alpha || !P || !ws || !status)
    return BITSMOE_ERR_INVALID_ARG;
  const DecLayout l = dec_layout(side, E, d, D);
  if (ws_bytes < l.total) return BITSMOE_ERR_WORKSPACE_TOO_SMALL;
  if ((reinterpret_cast<uintptr_t>(ws) & 255) != 0) return BITSMOE_ERR_ALIGNMENT;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  uint8_t* wb = static_cast<uint8_t*>(ws);
  const int64_t R = (int64_t)E * d;
  const int n = (int)std::min<int64_t>(D, R);
  float* G = reinterpret_cast<float*>(wb + l.G);
  float* Vt = reinterpret_cast<float*>(wb + l.Vt);
  float* Pt = reinterpret_cast<float*>(wb + l.Pt);
  uint32_t* bar = reinterpret_cast<uint32_t*>(wb + l.sync);
  const float* A = W;
  const size_t ld = (size_t)(D + (D & 1) + 3) / 4 * 4;
  BM_CK(cudaMemsetAsync(bar, 0, 256, st));
  BM_CK(cudaMemsetAsync(G, 0, (size_t)D * ld * 4, st));   // the padding columns stay 0
  if (side == 1) {
    float* At = reinterpret_cast<float*>(wb + l.A);
    k_transpose_out<<<dim3((d + 31) / 32, (D + 31) / 32, E), dim3(32, 8), 0, st>>>(W, E, D, d, At);
    BM_CK(cudaGetLastError());
    A = At;
  }
  const int ntile = (D + kTM - 1) / kTM;
  k_gram<float><<<ntile * (ntile + 1) / 2, kGT, 0, st>>>(A, nullptr, R, D, D, G, ld, ntile);
  BM_CK(cudaGetLastError());
  // the eigensolver: one block per SM, all resident (cooperative launch)
  int dev = 0, sms = 0;
  BM_CK(cudaGetDevice(&dev));
  BM_CK(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
  const int m = D + (D & 1);
  const int nb = std::min(sms, m / 2);
  const int per_block = (m / 2 + nb - 1) / nb;
  const size_t room = 220 * 1024 - (size_t)m * 12;
  const int batch = std::max(1, std::min({per_block, kJBatch, (int)(room / ((size_t)ld * 8))}));
  const size_t smem = (size_t)m * 12 + (size_t)batch * ld * 8;
  BM_CK(cudaFuncSetAttribute(k_jacobi, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
  int per_sm = 0;
  BM_CK(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_jacobi, 512, smem));
  if (per_sm < 1) return BITSMOE_ERR_SHAPE;
  JacobiArgs ja;
  ja.G = G;
  ja.Vt = Vt;
  ja.tab = reinterpret_cast<float2*>(wb + l.tab);
  ja.n = D;
  ja.ld = (int)ld;
  ja.batch = batch;
  ja.max_sweeps = max_sweeps;
  ja.tol = 1e-7f;
  ja.bar = bar;
  ja.status = status;
  ja.sweeps = sweeps;
  ja.spin = 2ll << 30;
  void* args[] = {&ja};
  BM_CK(cudaLaunchCooperativeKernel(reinterpret_cast<void*>(k_jacobi), dim3(nb), dim3(512), args, smem, st));
  k_order<<<D, 256, 0, st>>>(G, Vt, D, ld, n, phi, sigma);
  BM_CK(cudaGetLastError());
  k_project<<<dim3((n + kTN - 1) / kTN, (unsigned)((R + kTM - 1) / kTM)), kGT, 0, st>>>(A, phi, R, D, n, Pt);
  BM_CK(cudaGetLastError());
  k_normalize<<<dim3((n + 31) / 32, E), dim3(32, 8), 0, st>>>(Pt, E, d, n, alpha, P);
  BM_CK(cudaGetLastError());
  return BITSMOE_OK;
}

extern "C" int bitsmoe_calibration_gram(const void* x, const float* g, int64_t T, int D, float* H, void* stream) {
  using namespace bmoe;
  if (T < 0 || D < 1 || !H || (T > 0 && !x)) return BITSMOE_ERR_INVALID_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const int ntile = (D + kTM - 1) / kTM;
  if (T == 0) {
    BM_CK(cudaMemsetAsync(H, 0, (size_t)D * D * 4, st));
    return BITSMOE_OK;
  }
  k_gram<uint16_t><<<ntile * (ntile + 1) / 2, kGT, 0, st>>>(static_cast<const uint16_t*>(x), g, T, D, D, H, D, ntile);
  BM_CK(cudaGetLastError());
  return BITSMOE_OK;
}

#ifdef BITSMOE_JACOBI_TRACE
extern "C" int bitsmoe_jacobi_trace_read(void* dst) {
  return (int)cudaMemcpyFromSymbol(dst, g_jacobi_trace, sizeof(g_jacobi_trace));
}
#endif
