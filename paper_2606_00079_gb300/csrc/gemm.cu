// Tensor-core (tcgen05) kernel for the two dense contractions of the forward
// when several tokens share a call:
//
//   projection   z_h[t][j] = sum_d Phi_h[d, j] x[t][d]      (h = gate, up)
//   output       y[t][d]   = sum_j Phi_dn[d, j] s[t][j]      (y written or accumulated)
//
// (the shared-basis factors of Eq. app_normalized_decomposition, applied once
// per call for all tokens).  A = the bf16 basis rows (K-major, M = rows, K =
// D or n), streamed by TMA through a ring of 128-byte-swizzled shared-memory
// stages; B = the tokens' activations (K-major, N = tokens) written into the
// same ring by eight staging warps: x as bf16 (exact), s as a bf16 pair hi + lo
// (s - hi), whose two products accumulate into the same fp32 accumulator, so
// the output keeps about 16 bits of s.  One thread issues tcgen05.mma
// (kind::f16, M = 128, N = tokens rounded up to 16, K = 16) into a TMEM
// accumulator.  The K range of a 128-row tile is split over the CTAs of a
// thread-block cluster; their partial tiles meet through distributed shared
// memory and each CTA stores its share of the rows.  Every wait is bounded.
#include <cuda.h>
#include <cuda_bf16.h>

#include <algorithm>
#include <cstring>
#include <mutex>

#include "device.cuh"
#include "tc.cuh"

namespace {

constexpr int kStagers = 256;                // warps 2-9 stage B; warps 2-5 then read the accumulator
constexpr int kGThreads = 64 + kStagers;     // warp 0 TMA, warp 1 MMA
constexpr int kKB = 64;                    // K elements per stage (one 128-byte swizzle row of bf16)
constexpr uint32_t kATile = 128 * kKB * 2; // bytes of an A stage (128 rows)

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int x, int y, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
      : "memory");
}

struct GemmArgs {
  int mode;          // 0: projection (B = x, writes z and optionally zT); 1: output basis (B = s hi/lo, y)
  int M;             // rows of A (2n or D)
  int K;             // reduction length (D or n); A rows hold K_pad >= K elements
  int T;             // tokens of the call
  int t0;            // first token of this launch
  int N;             // MMA N for this launch (tokens rounded up to 16, <= 256)
  int nkb;           // K-blocks of 64 in all
  int kbs;           // K-blocks per split (cluster rank)
  int splits;        // CTAs of a cluster: K splits of one 128-row tile
  int stages;        // ring depth
  uint32_t stage;    // bytes per stage (A, B, and B-lo for mode 1)
  int n;             // mode 0: rows per projection (z row j of h = row h * n + j)
  int n_pad;
  int D;             // mode 1: output row length
  int accum;         // mode 1: y += (y holds the residual) instead of y =
  const uint16_t* x; // mode 0: [T][D] bf16 bits
  const float* s;    // mode 1: [T][n_pad]
  float* z;          // mode 0: [2][T][n_pad]
  float* zT;         // mode 0: null, or [2][n_pad][T] (token fastest): also written
  uint32_t* zmax;    // mode 0: null, or [2][T] max_j |z_h[t][j]| as fp32 bits (zeroed before)
  float* y;          // mode 1: [T][D]
  float4* zero;      // null, or a buffer of later kernels to clear (after the PDL wait)
  size_t zero_n;     // its length in float4
  int* status;
};

// One cluster = the `splits` K ranges of one 128-row tile of A; one CTA per range.
// Warp 0 streams the basis tiles by TMA through a ring of stages, warps 2-9 stage
// the activations (B) into the same ring, warp 1 issues tcgen05.mma; then warps 2-5
// read the fp32 partial tile out of TMEM into shared memory, and the cluster's CTAs
// add the partials of their share of the rows through distributed shared memory
// and store the result (no atomics, nothing to clear beforehand).
__global__ void __launch_bounds__(kGThreads, 1) k_gemm_tc(const __grid_constant__ CUtensorMap amap, GemmArgs g) {
  extern __shared__ uint8_t gsm_raw[];
  uint8_t* gsm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(gsm_raw) + 1023) & ~(uintptr_t)1023);
  const int S = g.stages;
  const uint32_t ring = (uint32_t)S * g.stage;
  const uint32_t redb = 128u * (uint32_t)g.N * 4u;   // fp32 partial tile [N][128] (rows contiguous)
  float* red = reinterpret_cast<float*>(gsm);         // reuses the ring once the MMAs are done
  uint64_t* full_a = reinterpret_cast<uint64_t*>(gsm + (ring > redb ? ring : redb));   // [S]
  uint64_t* full_b = full_a + S;                                                        // [S]
  uint64_t* empty = full_b + S;                                                         // [S]
  uint64_t* done = empty + S;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 1);
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  uint32_t rank;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(rank));
  const int m0 = blockIdx.x * 128;
  const int kb0 = (int)rank * g.kbs, nk = max(0, min(g.kbs, g.nkb - kb0));
  const uint32_t ncols = g.N <= 32 ? 32u : g.N <= 64 ? 64u : g.N <= 128 ? 128u : 256u;
  const uint32_t b_bytes = (uint32_t)g.N * 128;   // one B stage (N rows x 128 bytes)

  pdl_trigger();
  if (tid == 0) {
    for (int i = 0; i < S; ++i) {
      mbar_init_n(full_a + i, 1);
      mbar_init_n(full_b + i, kStagers / 32);
      mbar_init_n(empty + i, 1);
    }
    mbar_init_n(done, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (wid == 1) tmem_alloc(tmem_slot, ncols);
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = *tmem_slot;
  bool ok = true;

  if (wid == 0) {
    if (lane == 0) {   // producer: the basis tiles (weights: before waiting for earlier kernels)
      for (int i = 0; i < nk; ++i) {
        const int st = i % S, u = i / S;
        if (u > 0) ok &= mbar_wait(empty + st, (uint32_t)(u - 1) & 1u);
        mbar_expect_tx(full_a + st, kATile);
        tma_load_2d(smem_u32(gsm + (size_t)st * g.stage), &amap, (kb0 + i) * kKB, m0, smem_u32(full_a + st));
      }
    }
  } else if (wid == 1) {
    if (lane == 0) {   // MMA issuer
      const uint32_t idesc = idesc_bf16(g.N);
      for (int i = 0; i < nk; ++i) {
        const int st = i % S, u = i / S;
        ok &= mbar_wait(full_a + st, (uint32_t)u & 1u);
        ok &= mbar_wait(full_b + st, (uint32_t)u & 1u);
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        const uint32_t a0 = smem_u32(gsm + (size_t)st * g.stage);
        const uint32_t b0 = a0 + kATile;
#pragma unroll
        for (int k16 = 0; k16 < kKB / 16; ++k16) {
          const uint64_t ad = sw128_desc(a0 + k16 * 32);
          mma_f16(tmem, ad, sw128_desc(b0 + k16 * 32), idesc, (i | k16) != 0);
          if (g.mode == 1) mma_f16(tmem, ad, sw128_desc(b0 + b_bytes + k16 * 32), idesc, 1u);
        }
        mma_commit(empty + st);
      }
      mma_commit(done);
    }
  } else {
    // B stagers: rows = tokens, 64 K elements a stage in 8 chunks of 16 bytes, 128-byte swizzle.
    // A thread's chunks go four at a time; the next four are requested before the current ones
    // are converted and stored (and before the wait for a ring slot).
    pdl_wait();   // activations come from earlier kernels
    const int bt = tid - 64;   // 0 .. kStagers - 1
    if (g.zero) {   // a buffer that the following kernels accumulate into
      const size_t nthr = (size_t)gridDim.x * gridDim.y * kStagers;
      for (size_t i = ((size_t)blockIdx.y * gridDim.x + blockIdx.x) * kStagers + bt; i < g.zero_n; i += nthr)
        g.zero[i] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
    const int nch = g.N * 8;
    auto load4 = [&](int i, int c0, float4 (&v)[4][2]) {
      const int kbase = (kb0 + i) * kKB;
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int c = c0 + q * kStagers;
        v[q][0] = v[q][1] = make_float4(0.f, 0.f, 0.f, 0.f);
        const int r = c >> 3, ch = c & 7;
        const int t = g.t0 + r, k = kbase + ch * 8;
        if (c >= nch || t >= g.T || k >= g.K) continue;
        if (g.mode == 0) {
          const uint16_t* xr = g.x + (size_t)t * g.K + k;
          if ((g.K & 7) == 0) {   // rows 16-byte aligned, chunk inside the row
            v[q][0] = *reinterpret_cast<const float4*>(xr);
          } else {
            uint32_t w[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              const uint32_t a = k + 2 * e < g.K ? xr[2 * e] : 0u, b = k + 2 * e + 1 < g.K ? xr[2 * e + 1] : 0u;
              w[e] = a | (b << 16);
            }
            v[q][0] = make_float4(__uint_as_float(w[0]), __uint_as_float(w[1]), __uint_as_float(w[2]),
                                  __uint_as_float(w[3]));
          }
        } else {   // s is zero beyond n (padding): whole chunks can be read
          v[q][0] = *reinterpret_cast<const float4*>(g.s + (size_t)t * g.n_pad + k);
          v[q][1] = *reinterpret_cast<const float4*>(g.s + (size_t)t * g.n_pad + k + 4);
        }
      }
    };
    float4 vc[4][2], vn[4][2];
    if (nk > 0) load4(0, bt, vc);
    for (int i = 0; i < nk; ++i) {
      const int st = i % S, u = i / S;
      uint8_t* bs = gsm + (size_t)st * g.stage + kATile;
      bool first = true;
      for (int c0 = bt; ; c0 += 4 * kStagers) {
        const bool last_batch = c0 + 4 * kStagers >= nch;
        if (!last_batch) load4(i, c0 + 4 * kStagers, vn);
        else if (i + 1 < nk) load4(i + 1, bt, vn);
        if (first && u > 0) {   // the ring slot: its previous MMAs must be done
          if (lane == 0) ok &= mbar_wait(empty + st, (uint32_t)(u - 1) & 1u);
          __syncwarp();
        }
        first = false;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int c = c0 + q * kStagers;
          if (c >= nch) continue;
          const int r = c >> 3, ch = c & 7;
          const uint32_t off = (uint32_t)(r >> 3) * 1024 + (uint32_t)(r & 7) * 128 + (uint32_t)((ch ^ (r & 7)) * 16);
          if (g.mode == 0) {
            *reinterpret_cast<float4*>(bs + off) = vc[q][0];
          } else {
            const float f[8] = {vc[q][0].x, vc[q][0].y, vc[q][0].z, vc[q][0].w,
                                vc[q][1].x, vc[q][1].y, vc[q][1].z, vc[q][1].w};
            uint32_t h2[4], l2[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              const __nv_bfloat16 ha = __float2bfloat16_rn(f[2 * e]), hb = __float2bfloat16_rn(f[2 * e + 1]);
              const __nv_bfloat16 la = __float2bfloat16_rn(f[2 * e] - __bfloat162float(ha));
              const __nv_bfloat16 lb = __float2bfloat16_rn(f[2 * e + 1] - __bfloat162float(hb));
              h2[e] = (uint32_t)__bfloat16_as_ushort(ha) | ((uint32_t)__bfloat16_as_ushort(hb) << 16);
              l2[e] = (uint32_t)__bfloat16_as_ushort(la) | ((uint32_t)__bfloat16_as_ushort(lb) << 16);
            }
            *reinterpret_cast<uint4*>(bs + off) = make_uint4(h2[0], h2[1], h2[2], h2[3]);
            *reinterpret_cast<uint4*>(bs + b_bytes + off) = make_uint4(l2[0], l2[1], l2[2], l2[3]);
          }
        }
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          vc[q][0] = vn[q][0];
          vc[q][1] = vn[q][1];
        }
        if (last_batch) break;
      }
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");   // generic writes -> tensor-core reads
      __syncwarp();
      if (lane == 0) mbar_arrive(full_b + st);
    }
    if (wid < 6) {
    // partial tile out of TMEM: warp w holds accumulator lanes (rows) 32 (w % 4) ..
    if (lane == 0) ok &= mbar_wait(done, 0);
    __syncwarp();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const int r = 32 * (wid & 3) + lane;
    for (int c0 = 0; c0 < g.N; c0 += 8) {
      uint32_t rr[8];
      if (nk > 0) {
        tmem_ld8(tmem + ((uint32_t)(32 * (wid & 3)) << 16) + (uint32_t)c0, rr);
      } else {
#pragma unroll
        for (int q = 0; q < 8; ++q) rr[q] = 0u;
      }
#pragma unroll
      for (int q = 0; q < 8; ++q) red[(size_t)(c0 + q) * 128 + r] = __uint_as_float(rr[q]);
    }
    }
  }
  // every CTA of the cluster has its partial in shared memory
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  asm volatile("barrier.cluster.arrive.release.aligned;\n" ::: "memory");
  asm volatile("barrier.cluster.wait.acquire.aligned;\n" ::: "memory");
  if (wid < 2) pdl_wait();   // the stores below target buffers of earlier kernels (y may hold the residual)
  {
    // this CTA's share of the rows: the sum over the cluster's partials, stored
    const int rs = 128 / g.splits, rbeg = (int)rank * rs;
    const uint32_t lred = smem_u32(red);
    const int ne = rs * g.N;
    for (int e0 = tid; e0 < ne; e0 += 4 * kGThreads) {   // four elements a thread at a time
      float v[4][4];   // [element][cluster rank]: every partial requested before the first is used
#pragma unroll
      for (int b = 0; b < 4; ++b) {
        const int e = e0 + b * kGThreads;
        const int c = e / rs, rr = rbeg + (e - c * rs);   // consecutive threads: consecutive rows
        const uint32_t la = lred + (uint32_t)(c * 128 + rr) * 4u;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          v[b][q] = 0.f;
          if (e < ne && q < g.splits) {
            uint32_t ra;
            asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(ra) : "r"(la), "r"(q));
            asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v[b][q]) : "r"(ra) : "memory");
          }
        }
      }
#pragma unroll
      for (int b = 0; b < 4; ++b) {
        const int e = e0 + b * kGThreads;
        if (e >= ne) continue;
        const int c = e / rs, rr = rbeg + (e - c * rs);
        const float sum = (v[b][0] + v[b][1]) + (v[b][2] + v[b][3]);
        const int m = m0 + rr, t = g.t0 + c;
        const bool in = m < g.M && t < g.T;
        if (in) {
          if (g.mode == 0) {
            const int h = m >= g.n, j = m - h * g.n;
            g.z[((size_t)h * g.T + t) * g.n_pad + j] = sum;
            if (g.zT) g.zT[((size_t)h * g.n_pad + j) * g.T + t] = sum;
          } else {
            float* yp = g.y + (size_t)t * g.D + m;
            *yp = g.accum ? *yp + sum : sum;
          }
        }
        if (g.mode == 0 && g.zmax) {   // max |z| per (h, token): one atomic per warp where its lanes agree
          const int key = in ? (m >= g.n ? g.T : 0) + t : -1;
          const uint32_t am = in ? __float_as_uint(fabsf(sum)) : 0u;
          const unsigned act = __activemask();
          const int k0 = __shfl_sync(act, key, __ffs(act) - 1);
          if (__all_sync(act, key == k0)) {
            const uint32_t wm = __reduce_max_sync(act, am);
            if (key >= 0 && lane == __ffs(act) - 1) atomicMax(g.zmax + key, wm);
          } else if (key >= 0) {
            atomicMax(g.zmax + key, am);
          }
        }
      }
    }
  }
  // no CTA leaves while others may still read its shared memory
  asm volatile("barrier.cluster.arrive.release.aligned;\n" ::: "memory");
  asm volatile("barrier.cluster.wait.acquire.aligned;\n" ::: "memory");
  if (!ok) atomicCAS(g.status, 0, BITSMOE_ERR_TIMEOUT);
  if (wid == 1) {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    tmem_dealloc(tmem, ncols);
  }
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static std::once_flag once;
  static EncodeTiledFn fn = nullptr;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

}  // namespace

namespace bmoe {

// Tensor map of a row-major bf16 matrix [rows][cols_pad] for 128-row x 64-column
// tiles with 128-byte swizzle.  cols_pad * 2 must be a multiple of 16.
bool make_basis_map(void* map_out, const void* base, int rows, int cols_pad) {
  EncodeTiledFn fn = encode_fn();
  if (!fn || rows < 1 || cols_pad < 8 || (cols_pad * 2) % 16 || (reinterpret_cast<uintptr_t>(base) & 15)) return false;
  CUtensorMap* m = static_cast<CUtensorMap*>(map_out);
  const cuuint64_t dims[2] = {(cuuint64_t)cols_pad, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)cols_pad * 2};
  const cuuint32_t box[2] = {(cuuint32_t)kKB, 128};
  const cuuint32_t estr[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// mode 0: z = Phi_{g,u}^T x (and zT, when given) for all T tokens; mode 1:
// y = Phi_dn s, or y += Phi_dn s when p.accum.  Plain stores: nothing to clear.
cudaError_t launch_gemm_tc(int mode, const void* map, const Fwd& p, int sms, cudaStream_t st, bool pdl, float* zT,
                           void* zero, size_t zero_bytes, uint32_t* zmax) {
  static_assert(sizeof(CUtensorMap) == 128, "tensor map size");
  GemmArgs g;
  std::memset(&g, 0, sizeof(g));
  g.mode = mode;
  g.M = mode == 0 ? 2 * p.n : p.D;
  g.K = mode == 0 ? p.D : p.n;
  const int K_pad = mode == 0 ? p.D_pad : p.n_pad;
  g.nkb = (K_pad + kKB - 1) / kKB;
  g.T = p.T;
  g.n = p.n;
  g.n_pad = p.n_pad;
  g.D = p.D;
  g.accum = p.accum;
  g.x = p.x;
  g.s = p.s;
  g.z = p.z;
  g.zT = zT;
  g.zmax = zmax;
  g.zero = static_cast<float4*>(zero);
  g.zero_n = zero_bytes / 16;
  g.y = p.y;
  g.status = p.status;
  CUtensorMap amap;
  std::memcpy(&amap, map, sizeof(amap));
  static std::mutex mu;
  static int done_smem = 0;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  const int mtiles = (g.M + 127) / 128;
  for (int t0 = 0; t0 < p.T; t0 += 256) {
    const int nt = std::min(256, p.T - t0);
    g.t0 = t0;
    g.N = (nt + 15) / 16 * 16;
    g.stage = kATile + (uint32_t)g.N * 128 * (mode == 1 ? 2 : 1);
    // K splits (a cluster per 128-row tile): at most one CTA per SM, at most 4 (larger clusters
    // do not all fit at once), four K-blocks each; as many ring stages as fit (all of a CTA's
    // K-blocks in flight when they fit)
    int splits = 1;
    while (splits < 4 && mtiles * splits * 2 <= sms && g.nkb >= 8 * splits) splits *= 2;
    g.splits = splits;
    g.kbs = (g.nkb + splits - 1) / splits;
    g.stages = (int)std::min<size_t>((size_t)g.kbs, (size_t)(200 * 1024) / g.stage);
    if (g.stages < 1) return cudaErrorInvalidValue;
    const size_t ring = (size_t)g.stages * g.stage, redb = (size_t)128 * g.N * 4;
    const size_t smem = 1024 + std::max(ring, redb) + ((size_t)3 * g.stages + 1) * 8 + 16;
    if (smem > 227 * 1024) return cudaErrorInvalidValue;
    {
      std::lock_guard<std::mutex> lock(mu);
      if ((int)smem > done_smem) {
        cudaError_t r = cudaFuncSetAttribute(k_gemm_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (r != cudaSuccess) return r;
        done_smem = (int)smem;
      }
    }
    attr[0].val.clusterDim.x = 1;
    attr[0].val.clusterDim.y = (unsigned)splits;
    attr[0].val.clusterDim.z = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(mtiles, splits);
    cfg.blockDim = dim3(kGThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 2 : 1;
    const cudaError_t e = cudaLaunchKernelEx(&cfg, k_gemm_tc, amap, g);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace bmoe
