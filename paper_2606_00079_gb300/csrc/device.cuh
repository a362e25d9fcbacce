// Device-side pieces shared by the kernels of the forward (forward.cu) and
// the fused decode kernel (fused.cu): the argument block, PTX wrappers, the
// block-level router and the integer dot-product helpers of the two packed
// layouts.  Included by CUDA translation units only.
#pragma once
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <vector>

#include "internal.h"

namespace bmoe {

struct Fwd {
  const uint8_t* img;
  uint64_t img_bytes;   // size of the packed image (the bounds of the debug checks)
  const ExpertDesc* desc;
  const int32_t* seg;
  const ItemRec* items;
  const uint16_t* basis_in;
  const uint16_t* basis_out;
  int D, E, I, n, group, D_pad, n_pad, I_pad, NRB, NG, nseg, ul_max_tiles;
  int T, k, P;
  int s16;          // K2 smem row stride (int16 elements)
  int rbc;          // K3 row blocks per block
  int decode;       // small-batch mode: routing published once, prologue staging
  int accum;        // output basis adds into y (residual) instead of writing it
  int seg_bytes;    // largest gate/up item (bytes of codes in one row block)
  int ul_bytes;     // largest down item (bytes of one tile over rbc row blocks)
  const uint16_t* x;
  const float* logits;
  float* y;
  int* status;
  int* route_flag;  // decode mode: set once the routing below is published
  int* pair_expert;
  float* pair_weight;
  int* expert_count;
  int* expert_start;
  int* pair_list;
  int* active;      // [0] = number of routed experts, [1 + a] = expert id
  float* z;         // [2][T][n_pad]
  float* gu;        // [P][2][I_pad]
  float* s;         // [T][n_pad]
  float* zT;        // [2][n_pad][T]: z again, token fastest (written for the tensor-core gate/up kernel)
  int tc_min;       // > 0: experts with at least this many tokens take the tensor-core factor kernels,
                    //      the dp2a kernels skip them (and the tensor-core kernels the others)
};

// Buffers and sizes of the multi-token tensor-core expert kernels (expert_tc.cu).
struct XArgs {
  int NT;                 // rows of a token tile (16, 32 or 64): an expert's tokens in tiles of NT
  int max_tiles;          // bound on the call's token tiles
  int A_max;              // bound on the call's routed experts
  int Rtot;               // rows of the h buffers (multiple of 16)
  uint32_t ring;          // bytes of a CTA's copy ring (set at launch)
  const float* msa;       // [2][E] max over groups and slots of |scale * alpha| of gate/up (h, e)
  const uint32_t* zmax;   // [2][T] max over j of |z_h[t][j]| (fp32 bits)
  uint8_t* hb;            // [NRB][Rtot rows x 512 B]: h as an fp16 pair, a token tile of N rows at its first
                          //   row R0 as the down kernel's B tile [half 2][piece 2][N rows][128 B] (swizzled)
  float2* hs;             // [NRB][Rtot]: (sum of h over the row block's rows, 2^(24 - S) of its scaling)
  int tc_min;             // experts with fewer tokens are left to the dp2a kernels
  float* zv;              // z gathered per (projection, token tile) in unit-slot order: [K-block][128 slots][N]
  uint64_t zv_floats;     // its length
};

// Staging records of the fused single-token kernel, derived from the image
// when a layer is uploaded (flat image offsets, so that a block finds every
// copy of a work item with one vector load).
struct CStage {            // one per gate/up item (h < 2, e, segment)
  uint64_t code0;          // image offset of the item's code bytes in row block 0
  uint64_t unit0, alpha0;  // image offsets of its slots' unit indices and alphas
  uint64_t sz0;            // image offset of its first slot's scale/zero in group row 0
  uint32_t rb_stride;      // bytes between row blocks of the code stream
  uint32_t sz_row;         // bytes between group rows of the scale/zero matrix
  uint32_t bytes;          // code bytes per row block (0: empty item)
  uint32_t mb;             // bytes of the slot arrays (4 per slot)
  uint16_t nls;            // quantised slots (the 16-bit ones come last)
  uint8_t nr;              // buckets the item touches
  uint8_t bits[kNumBk];    // their bit-widths
  uint16_t ntl[kNumBk];    // tiles per touched bucket
  uint32_t meta0;          // offset in the metadata mirror of row block 0's [unit | alpha | scale/zero G rows]
  uint8_t pad_[4];
};
static_assert(sizeof(CStage) == 80, "CStage layout");

struct DStage {            // one per down tile (e, tile < ul_max_tiles)
  uint64_t code;           // image offset of the tile's codes over all row blocks
  uint64_t unit, alpha;    // image offsets of its 32 unit indices and alphas
  uint64_t sz;             // image offset of its first slot's scale/zero in group row 0
  uint32_t sz_row;         // bytes between group rows
  uint32_t bits;           // 0: the expert has no tile of this index
  uint32_t meta;           // offset in the metadata mirror of [unit 32 | alpha 32 | scale/zero NG rows of 32]
  uint32_t pad_;
};
static_assert(sizeof(DStage) == 48, "DStage layout");

// Fused single-token decode kernel (fused.cu): workspace pointers and the
// shared-memory plan chosen on the host.
struct FusedArgs {
  uint32_t* sync;    // [kSyncWords] epoch and two sets of barrier counters (fused_common.cuh)
  const CStage* cst; // [2][E][nseg]
  const uint8_t* meta;   // metadata mirror: each staging item's unit indices, alphas and scale/zero rows
  uint64_t meta_bytes;   //   contiguous, so that one copy stages them
  const DStage* dst; // [E][ul_max_tiles] (directly after cst)
  uint64_t tab_bytes;  // bytes of both tables
  const float* hn;     // norm mode (pre-norm block): hidden state h [D] to normalise; y = h accumulates
  const uint16_t* wr;  // norm mode: router matrix [E][D] bf16
  float eps;           // norm mode: RMSNorm epsilon
  int norm;            // 1: compute x = bf16(RMSNorm(h)) and the router logits in the kernel
  int b_per, b_stage, b_nst, e_per;     // basis rows per block, rows per stage, stages; output rows per block
  int nslot_c, slot_c, nslot_d, slot_d; // gate/up and down staging slots (count, bytes)
  int off_route, off_xs, off_r1, off_d, off_rc, off_cq, off_rec, off_part, smem;
  int smax, s16, seg_al, ul_max_tiles, d_code_bytes, d_h_bytes;
  int dbg;             // bit 0: block 0 skips its arrival at grid barrier 1 (tests of the bounded waits);
                       // bit 1: every staging record is checked against the image before its copies
  long long spin;      // bound of the grid-barrier waits, in SM clocks
};

// Records of the clustered single-token kernel (fused2.cu), derived at upload for
// each cluster size CL: the tiles of every (projection, expert) are cut into CL
// contiguous parts of about equal code bytes, and cluster rank r works on part r.
struct F2Gu {              // gate/up part r of (h, e): a run of row-lane tiles
  uint64_t code0;          // image offset of the part's codes in row block 0
  uint64_t unit0, alpha0;  // image offsets of its first slot's unit index and alpha
  uint64_t sz0;            // image offset of its first slot's scale/zero in group row 0
  uint32_t rb_stride;      // bytes between row blocks of the code stream
  uint32_t sz_row;         // bytes between group rows of the scale/zero matrix
  uint32_t bytes;          // code bytes per row block (0: empty part)
  uint32_t nslot;          // slots (a multiple of 4)
  uint8_t nr;              // buckets the part touches
  uint8_t bits[kNumBk];    // their bit-widths (ascending; 16 last)
  uint16_t ntl[kNumBk];    // tiles per touched bucket
  uint8_t pad_[10];
};
static_assert(sizeof(F2Gu) == 80, "F2Gu layout");

struct F2Dn {              // down part r of e: a run of unit-lane tiles
  uint64_t code[kNumBk];   // per touched bucket: image offset of its first part tile in row block 0
  uint64_t unit0, alpha0;  // image offsets of the part's first slot's unit index and alpha
  uint64_t sz0;            // image offset of its first slot's scale/zero in group row 0
  uint32_t sz_row;         // bytes between group rows
  uint32_t nslot;          // slots (32 per tile; 0: empty part)
  uint8_t nr;
  uint8_t bits[kNumBk];
  uint16_t ntl[kNumBk];
  uint8_t pad_[2];
};
static_assert(sizeof(F2Dn) == 112, "F2Dn layout");

// Warps of the clustered kernel per gate/up projection in the factor phase.
constexpr int kF2GuWarps = 8;

// Tile index at which warp w of nw starts on a run of row-lane tiles (buckets
// bits[0..nr), ntl tiles each): the first tile whose code-byte prefix reaches
// w/nw of the run's bytes.  The host sizes the activation tables with it.
__host__ __device__ inline int rl_split_at(const uint8_t* bits, const uint16_t* ntl, int nr, int w, int nw) {
  // in 512-byte chunks (a part stays far below 2^32 bytes), 32-bit arithmetic only
  uint32_t tot = 0;
  int nt = 0;
  for (int k = 0; k < nr; ++k) {
    tot += (uint32_t)ntl[k] * (uint32_t)rl_chunks(bits[k]);
    nt += ntl[k];
  }
  if (w <= 0) return 0;
  if (w >= nw) return nt;
  const uint32_t target = (tot * (uint32_t)w + (uint32_t)nw - 1) / (uint32_t)nw;   // ceil: first chunk at or past w/nw
  uint32_t pre = 0;
  int t = 0;
  for (int k = 0; k < nr; ++k) {
    const uint32_t cb = (uint32_t)rl_chunks(bits[k]);
    const uint32_t end = pre + (uint32_t)ntl[k] * cb;
    if (end >= target) return t + (int)(target > pre ? (target - pre + cb - 1) / cb : 0);
    pre = end;
    t += ntl[k];
  }
  return nt;
}

// Launch plan of the clustered kernel (fused2.cu).
struct F2Args {
  uint32_t* sync;          // [kSyncWords] epoch and two sets of barrier counters (workspace)
  const uint8_t* tab;      // records of this cluster size: per rank [gate E][up E][down E]
  uint32_t rank_bytes;     // bytes of one rank's records
  int CL, npairs;          // cluster size; (routing slot, row block) pairs, one per cluster
  int b_per, e_per;         // input- and output-basis rows of a pair block
  int b_free, e_free;       // the same for the other blocks (they stream no expert part)
  int b_stage, b_nst;       // input-basis rows per stage, stages
  int s16;                 // int16 activation table row (elements) per warp and group
  int off_rec, off_route, off_xs, off_cq, off_pw, off_xch, off_h, off_r1, off_d, off_r2, off_ss, smem;
  int dbg;                 // bit 0: block 0 skips its arrival at grid barrier 1 (tests of the bounded waits);
                           // bit 1: every staging record is checked against the image before its copies
  int prefetch_io;         // x and the logits are device memory: prefetch them into L2 before the wait
  int rec_smem;            // this rank's record table fits the gate/up staging area (copied there first)
  long long spin;          // bound of every wait, in SM clocks
};

// Sizes of a layer's clustered-kernel parts for one cluster size (host side).
struct F2Sizes {
  int gu_stage;            // most shared-memory bytes of one block's staged gate + up part
  int dn_stage;            // most bytes of one block's staged down part
  int s16;                 // most quantised slots of one warp's share of a gate/up part
};

// Shared-memory plan of the fused kernel for this layer, or false when the
// layer does not fit it (then the kernel chain runs).
bool fused_plan(const ImageHeader& hd, int T, int top_k, int seg_bytes, int ul_max_chunks, int s16, int sms,
                FusedArgs* f);
// Prep kernel + fused kernel on `st` (grid = sms blocks).
cudaError_t launch_fused(const Fwd& p, const FusedArgs& f, int sms, cudaStream_t st, bool pdl);
// Tensor-core projections (gemm.cu): a TMA map of a bf16 basis [rows][cols_pad]
// (128 bytes, written to map_out), and the launch of z += Phi^T x (mode 0) or
// y += Phi_dn s (mode 1) for all T tokens of p (z, resp. y, zeroed before
// unless y carries a residual).
bool make_basis_map(void* map_out, const void* base, int rows, int cols_pad);
cudaError_t launch_gemm_tc(int mode, const void* map, const Fwd& p, int sms, cudaStream_t st, bool pdl,
                           float* zT = nullptr, void* zero = nullptr, size_t zero_bytes = 0,
                           uint32_t* zmax = nullptr);
// Multi-token expert factors on tensor cores (expert_tc.cu): buffer sizes for T tokens,
// z gathered per token tile in unit-slot order (reads zT), gate/up with h = SiLU(gate) up
// into x.hb / x.hs (reads zmax), then the down factor of every routed expert into s
// (zeroed before).  Persistent: `sms` CTAs.
XArgs x_args(const ImageHeader& hd, int T, int k);
cudaError_t launch_zgather(const Fwd& p, const XArgs& x, int sms, cudaStream_t st, bool pdl);
cudaError_t launch_gu16(const Fwd& p, const XArgs& x, int sms, cudaStream_t st, bool pdl);
cudaError_t launch_dn16(const Fwd& p, const XArgs& x, int sms, cudaStream_t st, bool pdl);
// Staging records of a packed image (host side, at upload).
bool build_stage_tables(const uint8_t* img, std::vector<CStage>& cst, std::vector<DStage>& dst,
                        std::vector<uint8_t>& meta);
// Records of the clustered kernel for cluster size CL (host side, at upload):
// per rank r, [F2Gu gate E][F2Gu up E][F2Dn E]; and the largest staged sizes.
// False when a record would reach outside the image (the kernel is then not used).
bool build_f2_tables(const uint8_t* img, int CL, std::vector<uint8_t>& out, F2Sizes* sizes);
// Most clusters of CL blocks of the clustered kernel that can be resident at once
// (1 block per SM), or 0.
int f2_max_clusters(int G, int CL);
// Shared-memory plan of the clustered kernel, or false when the layer does not fit it.
bool f2_plan(const ImageHeader& hd, int top_k, int CL, int nclusters, const F2Sizes& sz, F2Args* f);
// The clustered kernel on `st` (grid = nclusters x CL blocks).
cudaError_t launch_f2(const Fwd& p, const F2Args& f, int nclusters, cudaStream_t st, bool pdl);

}  // namespace bmoe

namespace {
using namespace bmoe;

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kK3Tiles = kWarps;     // UL tiles per K3 block (one per warp)
constexpr int kK3MaxRB = 8;          // row blocks per K3 block
constexpr uint32_t kPrefetchPiece = 16384;
constexpr uint64_t kPrefetchCap = 96ull << 20;

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
__device__ __forceinline__ uint32_t smem_u32(const void* ptr) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(ptr));
}
__device__ __forceinline__ uint4 lds128(const void* p) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(smem_u32(p)));
  return v;
}
template <bool SH>
__device__ __forceinline__ uint4 ld128(const uint8_t* p) {
  if (SH) return lds128(p);
  return ldg_stream(p);
}
// mbarrier + bulk copy (global -> shared, completion counted in bytes on the mbarrier)
__device__ __forceinline__ void mbar_init(uint64_t* bar) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_u32(bar)) : "memory");
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes) : "memory");
}
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
               ::"r"(smem_u32(dst)), "l"(src), "r"(bytes), "r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile("{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
               : "=r"(ok) : "r"(smem_u32(bar)), "r"(parity) : "memory");
  return ok != 0;
}
// Bounded wait on an mbarrier phase (about one second of SM clock at most).
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity) {
  const long long t0 = clock64();
  while (!mbar_try_wait(bar, parity))
    if (clock64() - t0 > (2ll << 30)) return false;
  return true;
}
// Copy `bytes` (16-byte multiple, 16-byte aligned ends) to shared memory on one
// mbarrier; called by one lane.
__device__ __forceinline__ void stage_bytes(void* dst, const uint8_t* src, uint32_t bytes, uint64_t* bar) {
  mbar_init(bar);
  mbar_expect_tx(bar, bytes);
  uint32_t o = 0;
  while (o < bytes) {
    const uint32_t c = bytes - o < 32768u ? bytes - o : 32768u;
    bulk_g2s(static_cast<uint8_t*>(dst) + o, src + o, c, bar);
    o += c;
  }
}
__device__ __forceinline__ void fence_proxy_async() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ int ld_acquire(const int* ptr) {
  int v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(ptr) : "memory");
  return v;
}
__device__ __forceinline__ void st_release(int* ptr, int v) {
  asm volatile("st.release.gpu.global.b32 [%0], %1;" ::"l"(ptr), "r"(v) : "memory");
}
// Bounded wait (about one second of SM clock) for a flag published by another block.
__device__ __forceinline__ bool wait_flag(const int* flag) {
  const long long t0 = clock64();
  while (ld_acquire(flag) == 0) {
    if (clock64() - t0 > (2ll << 30)) return false;
    __nanosleep(64);
  }
  return true;
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
  if (u == 0x80000000u) return 0x80000000u;   // -0 and +0 are equal logits: they tie
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// ---------------------------------------------------------------------------
// Routing of all T tokens by one block into shared memory (small batches):
// keys[T*E] | pe[P] | pw[P] | cnt[E] | start[E+1] | act[E+1] | plist[P].
// Same rule as k_router.  Contains __syncthreads (call from the whole block).
// ---------------------------------------------------------------------------
__host__ __device__ constexpr int route_words(int T, int E, int P) { return T * E + 3 * P + 3 * E + 3; }

struct RouteView {
  const int* pe;
  const float* pw;
  const int* cnt;
  const int* start;
  const int* act;
  const int* plist;
};

__device__ RouteView route_block(const Fwd& p, uint32_t* sm) {
  const int E = p.E, k = p.k, T = p.T, P = p.P, tid = threadIdx.x, nt = blockDim.x;
  uint32_t* keys = sm;
  int* pe = reinterpret_cast<int*>(keys + T * E);
  float* pw = reinterpret_cast<float*>(pe + P);
  int* cnt = reinterpret_cast<int*>(pw + P);
  int* start = cnt + E;
  int* act = start + E + 1;
  int* plist = act + E + 1;
  for (int i = tid; i < T * E; i += nt) keys[i] = order_key(p.logits[i]);
  for (int i = tid; i < E; i += nt) cnt[i] = 0;
  __syncthreads();
  // rank of each logit in its token's row (ties to the lower index)
  for (int i = tid; i < T * E; i += nt) {
    const int t = i / E, e = i - t * E;
    const uint32_t key = keys[i];
    // the logit back from its key (the key map is a bijection on non-NaN floats)
    const float logit = __uint_as_float((key & 0x80000000u) ? (key & 0x7FFFFFFFu) : ~key);
    const uint32_t* row = keys + t * E;
    int rank = 0;
    if ((E & 3) == 0 && ((t * E) & 3) == 0) {
      const uint4* r4 = reinterpret_cast<const uint4*>(row);
#pragma unroll 4
      for (int f4 = 0; f4 < (E >> 2); ++f4) {
        const uint4 o = r4[f4];
        const int f = f4 << 2;
        rank += (o.x > key) | ((o.x == key) & (f < e));
        rank += (o.y > key) | ((o.y == key) & (f + 1 < e));
        rank += (o.z > key) | ((o.z == key) & (f + 2 < e));
        rank += (o.w > key) | ((o.w == key) & (f + 3 < e));
      }
    } else {
      for (int f = 0; f < E; ++f) {
        const uint32_t o = row[f];
        rank += (o > key) | ((o == key) & (f < e));
      }
    }
    if (rank < k) {
      pe[t * k + rank] = e;
      pw[t * k + rank] = key ? logit : __int_as_float(0x7FC00000);   // key 0: NaN logit
    }
  }
  __syncthreads();
  for (int t = tid; t < T; t += nt) {
    float* w = pw + t * k;
    const float m = w[0];
    float sum = 0.f;
    for (int r = 0; r < k; ++r) sum += expf(w[r] - m);
    const float inv = 1.f / sum;
    for (int r = 0; r < k; ++r) w[r] = expf(w[r] - m) * inv;
  }
  for (int q = tid; q < P; q += nt) atomicAdd(&cnt[pe[q]], 1);
  __syncthreads();
  if (tid < 32) {   // exclusive scans of counts and of "routed" flags, one warp
    const int lane = tid, per = (E + 31) >> 5, e0 = min(E, lane * per), e1 = min(E, e0 + per);
    int c = 0, na = 0;
    for (int e = e0; e < e1; ++e) {
      c += cnt[e];
      na += cnt[e] > 0;
    }
    int ci = c, ai = na;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int vc = __shfl_up_sync(0xFFFFFFFFu, ci, o), va = __shfl_up_sync(0xFFFFFFFFu, ai, o);
      if (lane >= o) {
        ci += vc;
        ai += va;
      }
    }
    int run = ci - c, ra = ai - na;
    for (int e = e0; e < e1; ++e) {
      start[e] = run;
      run += cnt[e];
      if (cnt[e] > 0) act[1 + ra++] = e;
    }
    if (lane == 31) {
      start[E] = ci;
      act[0] = ai;
    }
  }
  __syncthreads();
  for (int q = tid; q < P; q += nt) {   // stable order: pairs of one expert by increasing q
    const int ex = pe[q];
    int r = 0;
    for (int q2 = 0; q2 < q; ++q2) r += pe[q2] == ex;
    plist[start[ex] + r] = q;
  }
  __syncthreads();
  return RouteView{pe, pw, cnt, start, act, plist};
}

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

template <int B, int TB, bool SH = false>
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
    for (int c = 0; c < C; ++c) v[c] = ld128<SH>(code + (size_t)(t * C + c) * kChunkBytes);
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

// 16-bit units: tile of 4 units in 2 chunks; chunk c, word w = fp16(unit 2c, row w) | fp16(unit 2c+1, row w)
template <int TB, bool SH = false>
__device__ __forceinline__ void rl_range16(const uint8_t* code, int ntl, const int32_t* unit, const float* alpha,
                                           const float* const (&zrow)[TB], float (&acc16)[4][TB]) {
  for (int t = 0; t < ntl; ++t) {
#pragma unroll
    for (int c = 0; c < 2; ++c) {
      const uint4 v = ld128<SH>(code + (size_t)(2 * t + c) * kChunkBytes);
      const int j0 = unit[4 * t + 2 * c], j1 = unit[4 * t + 2 * c + 1];
      const float a0 = alpha[4 * t + 2 * c], a1 = alpha[4 * t + 2 * c + 1];
      const uint32_t wv[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
      for (int tt = 0; tt < TB; ++tt) {
        const float c0 = a0 * zrow[tt][j0], c1 = a1 * zrow[tt][j1];
#pragma unroll
        for (int w = 0; w < 4; ++w) acc16[w][tt] = fmaf(c0, f16lo(wv[w]), fmaf(c1, f16hi(wv[w]), acc16[w][tt]));
      }
    }
  }
}

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

}  // namespace
