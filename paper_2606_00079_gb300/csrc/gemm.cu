// Tensor-core (tcgen05) kernels for the two dense contractions of the
// forward when several tokens share a call:
//
//   projection   z_h[t][j] = sum_d Phi_h[d, j] x[t][d]      (h = gate, up)
//   output       y[t][d]   = sum_j Phi_dn[d, j] s[t][j]      (y written or accumulated)
//
// (the shared-basis factors of Eq. app_normalized_decomposition, applied once
// per call for all tokens).  A = the bf16 basis rows (K-major, M = rows, K =
// D or n), streamed by TMA into 128-byte-swizzled shared-memory tiles; B = the
// tokens' activations (K-major, N = tokens), written into the same swizzled
// layout by three staging warps: x as bf16 (exact), s as a bf16 pair
// hi + lo (s - hi), whose two products accumulate into the same fp32
// accumulator, so the output keeps about 16 bits of s.  One thread issues
// tcgen05.mma (kind::f16, M = 128, N = tokens rounded up to 16, K = 16) into
// a TMEM accumulator; the four warps read it back with tcgen05.ld.
// One block per 128-row tile of A and per group of at most 256 tokens; a ring
// of stages overlaps TMA, staging and MMA.  Every wait is bounded.
#include <cuda.h>
#include <cuda_bf16.h>

#include <algorithm>
#include <cstring>
#include <mutex>

#include "device.cuh"
#include "tc.cuh"

namespace {

constexpr int kGThreads = 128;
constexpr int kKB = 64;                    // K elements per stage (one 128-byte swizzle row of bf16)
constexpr uint32_t kATile = 128 * kKB * 2; // bytes of an A stage (128 rows)

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int x, int y, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
      : "memory");
}

struct GemmArgs {
  int mode;          // 0: projection (B = x, adds into z); 1: output basis (B = s hi/lo, adds into y)
  int M;             // rows of A (2n or D)
  int K;             // reduction length (D or n); A rows hold K_pad >= K elements
  int T;             // tokens of the call
  int t0;            // first token of this launch
  int N;             // MMA N for this launch (tokens rounded up to 16, <= 256)
  int nkb;           // K stages in all
  int kbs;           // K stages per split (blockIdx.y)
  uint32_t stage;    // bytes per stage (A, B, and B-lo for mode 1)
  int n;             // mode 0: rows per projection (z row j of h = row h * n + j)
  int n_pad;
  int D;             // mode 1: output row length
  const uint16_t* x; // mode 0: [T][D] bf16 bits
  const float* s;    // mode 1: [T][n_pad]
  float* z;          // mode 0: [2][T][n_pad], zeroed before
  float* zT;         // mode 0: null, or [2][n_pad][T] (token fastest), zeroed before: also written
  float* y;          // mode 1: [T][D], zeroed before unless accumulating
  int* status;
};

// One block: 128 rows of A (blockIdx.x) times a range of K stages (blockIdx.y),
// all resident in shared memory.  Partial sums of the K splits meet in global
// memory through fp32 reductions.
__global__ void __launch_bounds__(kGThreads, 1) k_gemm_tc(const __grid_constant__ CUtensorMap amap, GemmArgs g) {
  extern __shared__ uint8_t gsm_raw[];
  // 1024-byte aligned base for the swizzled tiles
  uint8_t* gsm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(gsm_raw) + 1023) & ~(uintptr_t)1023);
  const int kb0 = blockIdx.y * g.kbs, nk = min(g.kbs, g.nkb - kb0);
  uint64_t* full_a = reinterpret_cast<uint64_t*>(gsm + (size_t)g.kbs * g.stage + 8192);   // [kbs]
  uint64_t* done = full_a + g.kbs;                                                         // [1]
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 1);
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  const int m0 = blockIdx.x * 128;
  const uint32_t ncols = g.N <= 32 ? 32u : g.N <= 64 ? 64u : g.N <= 128 ? 128u : 256u;
  const uint32_t b_bytes = (uint32_t)g.N * 128;   // one B stage (N rows x 128 bytes)
  if (nk <= 0) return;

  if (tid == 0) {   // the basis tiles: weights, requested before waiting for earlier kernels
    for (int i = 0; i < nk; ++i) mbar_init_n(full_a + i, 1);
    mbar_init_n(done, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    for (int i = 0; i < nk; ++i) {
      mbar_expect_tx(full_a + i, kATile);
      tma_load_2d(smem_u32(gsm + (size_t)i * g.stage), &amap, (kb0 + i) * kKB, m0, smem_u32(full_a + i));
    }
  }
  if (wid == 0) {   // accumulator: 128 lanes x ncols fp32 columns of TMEM
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(ncols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  pdl_wait();   // activations come from earlier kernels

  // B: rows = tokens, 64 K elements per stage in 8 chunks of 16 bytes, 128-byte swizzle.
  // Chunks are loaded 4 at a time per thread so that their loads overlap.
  const int nchunk = nk * g.N * 8;
  for (int i0 = tid; i0 < nchunk; i0 += 4 * kGThreads) {
    uint4 hi[4], lo[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int i = i0 + u * kGThreads;
      hi[u] = lo[u] = make_uint4(0, 0, 0, 0);
      if (i >= nchunk) continue;
      const int st = i / (g.N * 8), rem = i - st * g.N * 8, r = rem >> 3, c = rem & 7;
      const int t = g.t0 + r, k = (kb0 + st) * kKB + c * 8;
      if (t >= g.T || k >= g.K) continue;
      if (g.mode == 0) {
        const uint16_t* xr = g.x + (size_t)t * g.K + k;
        if ((g.K & 7) == 0) {   // rows 16-byte aligned, chunk inside the row
          hi[u] = *reinterpret_cast<const uint4*>(xr);
        } else {
          uint32_t w[4];
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const uint32_t a = k + 2 * q < g.K ? xr[2 * q] : 0u, b = k + 2 * q + 1 < g.K ? xr[2 * q + 1] : 0u;
            w[q] = a | (b << 16);
          }
          hi[u] = make_uint4(w[0], w[1], w[2], w[3]);
        }
      } else {   // s is zero beyond n (padding): whole chunks can be read
        const float4 v0 = *reinterpret_cast<const float4*>(g.s + (size_t)t * g.n_pad + k);
        const float4 v1 = *reinterpret_cast<const float4*>(g.s + (size_t)t * g.n_pad + k + 4);
        const float v[8] = {v0.x, v0.y, v0.z, v0.w, v1.x, v1.y, v1.z, v1.w};
        uint32_t h2[4], l2[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const __nv_bfloat16 ha = __float2bfloat16_rn(v[2 * q]), hb = __float2bfloat16_rn(v[2 * q + 1]);
          const __nv_bfloat16 la = __float2bfloat16_rn(v[2 * q] - __bfloat162float(ha));
          const __nv_bfloat16 lb = __float2bfloat16_rn(v[2 * q + 1] - __bfloat162float(hb));
          h2[q] = (uint32_t)__bfloat16_as_ushort(ha) | ((uint32_t)__bfloat16_as_ushort(hb) << 16);
          l2[q] = (uint32_t)__bfloat16_as_ushort(la) | ((uint32_t)__bfloat16_as_ushort(lb) << 16);
        }
        hi[u] = make_uint4(h2[0], h2[1], h2[2], h2[3]);
        lo[u] = make_uint4(l2[0], l2[1], l2[2], l2[3]);
      }
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int i = i0 + u * kGThreads;
      if (i >= nchunk) continue;
      const int st = i / (g.N * 8), rem = i - st * g.N * 8, r = rem >> 3, c = rem & 7;
      uint8_t* bt = gsm + (size_t)st * g.stage + kATile;
      const uint32_t off = (uint32_t)(r >> 3) * 1024 + (uint32_t)(r & 7) * 128 + (uint32_t)((c ^ (r & 7)) * 16);
      *reinterpret_cast<uint4*>(bt + off) = hi[u];
      if (g.mode == 1) *reinterpret_cast<uint4*>(bt + b_bytes + off) = lo[u];
    }
  }
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");   // generic writes -> tensor-core reads
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = *tmem_slot;

  if (tid == 0) {   // MMA issuer: each stage as soon as its basis tile has landed
    const uint32_t idesc = idesc_bf16(g.N);
    bool ok = true;
    for (int i = 0; i < nk && ok; ++i) {
      ok = mbar_wait(full_a + i, 0);
      if (!ok) break;
      asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      const uint32_t a0 = smem_u32(gsm + (size_t)i * g.stage);
      const uint32_t b0 = a0 + kATile;
#pragma unroll
      for (int k16 = 0; k16 < kKB / 16; ++k16) {
        const uint64_t ad = sw128_desc(a0 + k16 * 32);
        mma_bf16(tmem, ad, sw128_desc(b0 + k16 * 32), idesc, (i | k16) != 0);
        if (g.mode == 1) mma_bf16(tmem, ad, sw128_desc(b0 + b_bytes + k16 * 32), idesc, 1u);
      }
    }
    mma_commit(done);
    if (!ok) atomicCAS(g.status, 0, BITSMOE_ERR_TIMEOUT);
  }
  __syncwarp();

  // epilogue: warp w reads accumulator lanes 32w .. 32w + 31 (rows m0 + 32w + lane) and adds them out
  if (!mbar_wait(done, 0) && lane == 0) atomicCAS(g.status, 0, BITSMOE_ERR_TIMEOUT);
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const int m = m0 + 32 * wid + lane;
  for (int c0 = 0; c0 < g.N; c0 += 8) {
    uint32_t r[8];
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7])
                 : "r"(tmem + ((uint32_t)(32 * wid) << 16) + (uint32_t)c0));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
    if (m < g.M) {
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        const int t = g.t0 + c0 + q;
        if (c0 + q < g.N && t < g.T) {
          const float v = __uint_as_float(r[q]);
          if (g.mode == 0) {
            const int h = m >= g.n, j = m - h * g.n;
            atomicAdd(g.z + ((size_t)h * g.T + t) * g.n_pad + j, v);
            if (g.zT) atomicAdd(g.zT + ((size_t)h * g.n_pad + j) * g.T + t, v);
          } else {
            atomicAdd(g.y + (size_t)t * g.D + m, v);
          }
        }
      }
    }
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  if (wid == 0) {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(ncols) : "memory");
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

// mode 0: z += Phi_{g,u}^T x for all T tokens; mode 1: y += Phi_dn s.  The
// target must hold zeros (or the residual, for y) before the launch.
cudaError_t launch_gemm_tc(int mode, const void* map, const Fwd& p, int sms, cudaStream_t st, bool pdl, float* zT) {
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
  g.x = p.x;
  g.s = p.s;
  g.z = p.z;
  g.y = p.y;
  g.status = p.status;
  g.zT = zT;
  CUtensorMap amap;
  std::memcpy(&amap, map, sizeof(amap));
  static std::mutex mu;
  static int done_smem = 0;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  const int mtiles = (g.M + 127) / 128;
  for (int t0 = 0; t0 < p.T; t0 += 256) {
    const int nt = std::min(256, p.T - t0);
    g.t0 = t0;
    g.N = (nt + 15) / 16 * 16;
    g.stage = kATile + (uint32_t)g.N * 128 * (mode == 1 ? 2 : 1);
    // K splits: the fewest that keep a block's stages within 200 KB and give about one block per SM
    int splits = 1;
    while (splits < g.nkb && ((size_t)((g.nkb + splits - 1) / splits) * g.stage > 200 * 1024 ||
                              mtiles * splits < sms * 3 / 4))
      splits *= 2;
    g.kbs = (g.nkb + splits - 1) / splits;
    if ((size_t)g.kbs * g.stage > 200 * 1024) return cudaErrorInvalidValue;
    splits = (g.nkb + g.kbs - 1) / g.kbs;
    const size_t smem = 1024 + (size_t)g.kbs * g.stage + 8192 + ((size_t)g.kbs + 1) * 8 + 16;
    {
      std::lock_guard<std::mutex> lock(mu);
      if ((int)smem > done_smem) {
        cudaError_t r = cudaFuncSetAttribute(k_gemm_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (r != cudaSuccess) return r;
        done_smem = (int)smem;
      }
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(mtiles, splits);
    cfg.blockDim = dim3(kGThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    const cudaError_t e = cudaLaunchKernelEx(&cfg, k_gemm_tc, amap, g);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace bmoe
