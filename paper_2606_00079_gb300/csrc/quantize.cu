// Per-unit quantiser: normalised spectral vectors (fp32) -> the stored unit
// format the forward reads (codes, fp16 scale and zero per group).
//
// BitsMoE quantises every spectral unit p (a column of P, length I) with its
// own bit-width b in {0,1,2,3,4,6,8,16} (appendix "Piecewise Reconstruction
// Error for Bit Allocation"), one scale per group of `group` elements along
// the unit (group 128 in the paper's experiments):
//   b = 2, 3, 4  symmetric uniform Q_b (Eq. app_scalar_quantization_uk) with
//                the MSE-optimal scale (Eq. app_low_bit_opt_scale), searched
//                over `grid` fp16 candidates s_c = fp16(rho 2^(2-b) c / grid)
//   b = 6, 8     Q_b with s = rho / q_max, rho = ||p||_inf (Eqs.
//                app_high_bit_rho_eta, app_uk_scale)
//   b = 1        sign quantiser s_1 sign(p), s_1 = mean |p|, sign(0) = +1
//                (Eq. app_one_bit_quantization)
//   b = 0        evicted (Eq. app_zero_bit_vector); b = 16: fp16 values
// Stored as code = q + 2^(b-1), zero = 2^(b-1) (sign: code [p >= 0], zero
// 1/2, scale 2 s_1), so that p_hat = scale (code - zero).
//
// Arithmetic: fp32 with every operation rounded once (no contraction in the
// error sums), the quotient p / s as p times the correctly rounded fp32
// reciprocal of s, error sums over the group's elements in order, the least
// error winning with ties to the smaller candidate index, so the result is a
// deterministic function of the inputs.
//
// Work decomposition: one warp per (unit, group).  The group's elements are
// staged in shared memory; for the scale search each lane owns grid / 32
// candidates in registers and scores them all on every element it reads (a
// broadcast read), so the inner loop is eight fp32 instructions per
// (element, candidate) — six for the upper quarter of the candidates, which
// provably never clip — and no shuffles; one lexicographic (error, index)
// warp reduction picks the scale.  The search is ALU-bound: the fp32 input is
// read once and the codes written once.
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "device.cuh"
#include "internal.h"

namespace {

constexpr int kQWarps = 8;
constexpr int kQThreads = kQWarps * 32;
constexpr int kQMaxGroup = 256;
constexpr float kRne = 12582912.f;   // 1.5 * 2^23: t + kRne - kRne rounds |t| <= 2^22 to nearest even

struct QArgs {
  const float* p;
  const uint8_t* bits;
  int64_t items;   // U * ng
  int I, group, ng, grid;
  uint16_t* codes;
  uint16_t* scale;
  uint16_t* zero;
  int* status;
};

__device__ __forceinline__ float f16_round(float x) { return __half2float(__float2half_rn(x)); }
__device__ __forceinline__ uint32_t f16_bits(float x) { return (uint32_t)__half_as_ushort(__float2half_rn(x)); }
__device__ __forceinline__ bool bits_supported(int b) {
  return b == 0 || b == 1 || b == 2 || b == 3 || b == 4 || b == 6 || b == 8 || b == 16;
}
// a scale that is positive and finite in fp16
__device__ __forceinline__ bool usable(float s) { return s > 0.f && s <= 65504.f; }
// clamp(round(v * r), qmin, qmax): clamping first gives the same level (the bounds are integers)
__device__ __forceinline__ float level(float v, float r, float qmin, float qmax) {
  const float t = fminf(fmaxf(__fmul_rn(v, r), qmin), qmax);
  return __fsub_rn(__fadd_rn(t, kRne), kRne);
}
// candidate c (1-based) of the scale search
__device__ __forceinline__ float candidate(float top, int c, int grid) {
  return f16_round(__fdiv_rn(__fmul_rn(top, (float)c), (float)grid));
}

// Scores of the NC candidates of a lane over the group.  With FREE, the candidates
// m >= kFree(NC) skip the clamp: their index c > 3 grid / 4, so with a normal fp16 scale
// |v| / s <= 2^(b-2) (grid / c) (1 + 2^-10) < 1.34 * 2^(b-2) < 2^(b-1) - 1/2 for b <= 4,
// and round(v / s) is already a level: the clamp would change nothing.
template <int NC>
__host__ __device__ constexpr int kFree() { return (3 * NC + 3) / 4; }
template <int NC, bool FREE>
__device__ __forceinline__ void score(const float* v, int g, const float (&sc)[NC], const float (&rc)[NC],
                                      float (&e)[NC], float qmin, float qmax) {
#pragma unroll 2
  for (int i = 0; i < g; i += 4) {
    const float4 x4 = *reinterpret_cast<const float4*>(v + i);
    const float xs[4] = {x4.x, x4.y, x4.z, x4.w};
#pragma unroll
    for (int k = 0; k < 4; ++k) {
#pragma unroll
      for (int m = 0; m < NC; ++m) {
        const float q = (FREE && m >= kFree<NC>())
                            ? __fsub_rn(__fadd_rn(__fmul_rn(xs[k], rc[m]), kRne), kRne)
                            : level(xs[k], rc[m], qmin, qmax);
        const float d = fmaf(-sc[m], q, xs[k]);   // sc * q is exact (11 x 4 significant bits)
        e[m] = __fadd_rn(e[m], __fmul_rn(d, d));
      }
    }
  }
}

// Scale search of one group for b in {2, 3, 4}: NC candidates per lane.
template <int NC>
__device__ float search_scale(const float* v, int g, float rho, int b, int grid, int lane) {
  const float qmax = (float)((1 << (b - 1)) - 1), qmin = -(float)(1 << (b - 1));
  const float top = __fmul_rn(rho, b == 2 ? 1.f : (b == 3 ? 0.5f : 0.25f));
  const float kInf = __int_as_float(0x7F800000);
  float sc[NC], rc[NC], e[NC];
#pragma unroll
  for (int m = 0; m < NC; ++m) {   // a skipped candidate starts (and stays) at +inf error
    const float s = candidate(top, lane + 1 + 32 * m, grid);
    const bool ok = usable(s);
    sc[m] = ok ? s : 1.f;
    rc[m] = __frcp_rn(sc[m]);
    e[m] = ok ? 0.f : kInf;
  }
  // the clamp-free path needs every lane's upper candidates to be normal fp16 scales (or skipped)
  bool normal = true;
#pragma unroll
  for (int m = kFree<NC>(); m < NC; ++m) normal &= (sc[m] >= 6.103515625e-05f) || e[m] == kInf;
  if (__all_sync(0xFFFFFFFFu, normal)) score<NC, true>(v, g, sc, rc, e, qmin, qmax);
  else score<NC, false>(v, g, sc, rc, e, qmin, qmax);
  float be = e[0];
  int bc = lane + 1;
#pragma unroll
  for (int m = 1; m < NC; ++m) {
    if (e[m] < be) {
      be = e[m];
      bc = lane + 1 + 32 * m;
    }
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) {
    const float oe = __shfl_xor_sync(0xFFFFFFFFu, be, o);
    const int oc = __shfl_xor_sync(0xFFFFFFFFu, bc, o);
    if (oe < be || (oe == be && oc < bc)) {
      be = oe;
      bc = oc;
    }
  }
  return be == kInf ? 0.f : candidate(top, bc, grid);
}

template <int NC>
__global__ void __launch_bounds__(kQThreads) k_quantize(QArgs a) {
  __shared__ __align__(16) float sv[kQWarps][kQMaxGroup];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  float* v = sv[w];
  const int g = a.group;
  for (int64_t it = (int64_t)blockIdx.x * kQWarps + w; it < a.items; it += (int64_t)gridDim.x * kQWarps) {
    const int64_t u = it / a.ng;
    const int gi = (int)(it - u * a.ng);
    const int b = __ldg(a.bits + u);
    const size_t base = (size_t)u * a.I + (size_t)gi * g;
    uint32_t* dst = reinterpret_cast<uint32_t*>(a.codes + base);   // two codes a word
    float mx = 0.f;
    __syncwarp();   // the previous item's reads of v are done
    for (int i = lane; i < g / 4; i += 32) {
      const float4 x = __ldcs(reinterpret_cast<const float4*>(a.p + base) + i);
      reinterpret_cast<float4*>(v)[i] = x;
      mx = fmaxf(mx, fmaxf(fmaxf(fabsf(x.x), fabsf(x.y)), fmaxf(fabsf(x.z), fabsf(x.w))));
    }
    const float rho = warp_max(mx);
    __syncwarp();
    float s = 0.f, zp = 0.f;
    if (b == 0 || !bits_supported(b)) {
      for (int i = lane; i < g / 2; i += 32) dst[i] = 0u;
      if (b != 0 && lane == 0 && a.status) atomicCAS(a.status, 0, BITSMOE_ERR_UNSUPPORTED_BITS);
    } else if (b == 16) {
      for (int i = lane; i < g / 2; i += 32) dst[i] = f16_bits(v[2 * i]) | (f16_bits(v[2 * i + 1]) << 16);
    } else if (b == 1) {
      // s_1 = mean |p| over the group, summed in element order
      float acc = 0.f;
      if (lane == 0) {
#pragma unroll 8
        for (int i = 0; i < g; ++i) acc = __fadd_rn(acc, fabsf(v[i]));
      }
      acc = __shfl_sync(0xFFFFFFFFu, acc, 0);
      s = f16_round(__fmul_rn(2.f, __fdiv_rn(acc, (float)g)));
      zp = 0.5f;
      for (int i = lane; i < g / 2; i += 32)
        dst[i] = (v[2 * i] >= 0.f ? 1u : 0u) | ((v[2 * i + 1] >= 0.f ? 1u : 0u) << 16);
    } else {
      const float half = (float)(1 << (b - 1));
      if (b <= 4) {
        s = search_scale<NC>(v, g, rho, b, a.grid, lane);
      } else {
        s = f16_round(__fdiv_rn(rho, half - 1.f));
        if (!usable(s)) s = 0.f;
      }
      zp = half;
      const float r = s > 0.f ? __frcp_rn(s) : 0.f;
      const float qmax = half - 1.f, qmin = -half;
      for (int i = lane; i < g / 2; i += 32) {
        const float q0 = s > 0.f ? level(v[2 * i], r, qmin, qmax) : 0.f;
        const float q1 = s > 0.f ? level(v[2 * i + 1], r, qmin, qmax) : 0.f;
        dst[i] = (uint32_t)(int)(q0 + half) | ((uint32_t)(int)(q1 + half) << 16);
      }
    }
    if (lane == 0) {
      const size_t o = (size_t)u * a.ng + gi;
      a.scale[o] = (uint16_t)f16_bits(s);
      a.zero[o] = (uint16_t)f16_bits(zp);
    }
  }
}

template <int NC>
cudaError_t launch_q(const QArgs& a, cudaStream_t st) {
  int dev = 0, sms = 0, per_sm = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e == cudaSuccess) e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_quantize<NC>, kQThreads, 0);
  if (e != cudaSuccess) return e;
  const int64_t need = (a.items + kQWarps - 1) / kQWarps;
  const int64_t full = (int64_t)sms * (per_sm > 0 ? per_sm : 1);
  const int blocks = (int)(need < full ? need : full);
  k_quantize<NC><<<blocks, kQThreads, 0, st>>>(a);
  return cudaGetLastError();
}

}  // namespace

extern "C" int bitsmoe_quantize_units(const float* p, const uint8_t* bits, int64_t U, int I, int group, int grid,
                                      uint16_t* codes, uint16_t* scale, uint16_t* zero, int* status,
                                      void* stream) {
  if (U < 0 || I < 1) return BITSMOE_ERR_INVALID_ARG;
  if (!bmoe::group_ok(group) || I % group) return BITSMOE_ERR_SHAPE;
  if (grid != 32 && grid != 64 && grid != 128 && grid != 256 && grid != 512 && grid != 1024)
    return BITSMOE_ERR_INVALID_ARG;
  if (U == 0) return BITSMOE_OK;
  if (!p || !bits || !codes || !scale || !zero) return BITSMOE_ERR_INVALID_ARG;
  if ((uintptr_t)p % 16 || (uintptr_t)codes % 16 || (uintptr_t)scale % 2 || (uintptr_t)zero % 2 ||
      (uintptr_t)status % 4)
    return BITSMOE_ERR_ALIGNMENT;
  QArgs a{p, bits, U * (int64_t)(I / group), I, group, I / group, grid, codes, scale, zero, status};
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  cudaError_t e;
  switch (grid) {
    case 32: e = launch_q<1>(a, st); break;
    case 64: e = launch_q<2>(a, st); break;
    case 128: e = launch_q<4>(a, st); break;
    case 256: e = launch_q<8>(a, st); break;
    case 512: e = launch_q<16>(a, st); break;
    default: e = launch_q<32>(a, st); break;
  }
  return e == cudaSuccess ? BITSMOE_OK : bmoe::record_cuda_error((int)e);
}
