/*
 * bitsmoe.h - C ABI of libbitsmoe: the BitsMoE quantized MoE-layer forward
 * (Stage 3 of the method) on one GB300 (sm_103a).
 *
 * The method (BitsMoE paper, Sec. "Shared-basis Spectral Decomposition" and
 * Fig. 1 Stage 3; identity of Eq. app_normalized_decomposition) stores each
 * routed expert e and projection h in {gate, up, down} as
 *
 *     W_e^(h) = P_e^(h) A_e^(h) Phi_h^T     (gate, up;  P: I x n,  Phi: D x n)
 *     W_e^(h) = Phi_h A_e^(h) P_e^(h)^T     (down)
 *
 * with an unquantised shared basis Phi_h per projection type, spectral
 * energies A = diag(alpha) and a normalised spectral factor P whose columns
 * ("units", one rank-1 direction each, length I) are quantised with their own
 * bit-width b in {0,1,2,3,4,6,8,16} (Eqs. quantized_spectral_vector,
 * piecewise_error_surrogate).  At inference the activation is projected once
 * onto the shared bases and the quantised factors are applied inside the
 * kernels without rebuilding W ("Inference Efficiency", Sec. Experiments):
 *
 *     z_g = Phi_g^T x,  z_u = Phi_u^T x                          (once per layer)
 *     h_e = SiLU(P_g,e (alpha_g,e * z_g)) * (P_u,e (alpha_u,e * z_u))
 *     s   = sum_{e in topk} w_e * alpha_dn,e * (P_dn,e^T h_e)
 *     y   = Phi_dn s                                              (once per token)
 *
 * Conventions for every entry point:
 *   - return BITSMOE_OK (0) on success, a negative BITSMOE_ERR_* code otherwise;
 *     no exception, abort, assert or device trap crosses the ABI;
 *   - "device" pointers are CUDA device (or managed) memory of the device the
 *     layer was packed on; "host" pointers are ordinary host memory;
 *   - a stream is a cudaStream_t passed as void* (NULL = legacy default stream).
 */
#ifndef BITSMOE_H
#define BITSMOE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define BITSMOE_OK                      0
#define BITSMOE_ERR_INVALID_ARG        -1  /* null pointer, bad top_k, negative T ...            */
#define BITSMOE_ERR_SHAPE              -2  /* unsupported dims / group size                      */
#define BITSMOE_ERR_UNSUPPORTED_BITS   -3  /* a unit bit-width outside {0,1,2,3,4,6,8,16}         */
#define BITSMOE_ERR_WORKSPACE_TOO_SMALL -4
#define BITSMOE_ERR_ALIGNMENT          -5  /* device pointer not 16-byte aligned                 */
#define BITSMOE_ERR_CUDA               -6  /* a CUDA runtime call failed (see bitsmoe_last_cuda_error) */
#define BITSMOE_ERR_OOM                -7  /* host or device allocation failed                   */
#define BITSMOE_ERR_TIMEOUT            -8  /* a bounded device-side wait ran out                  */
#define BITSMOE_ERR_DEVICE_BOUNDS      -9  /* a device-side bounds check failed (access skipped) */
#define BITSMOE_ERR_BLOB              -10  /* packed blob is malformed / wrong version           */
#define BITSMOE_ERR_WORKSPACE_STATE   -11  /* workspace not zero-filled before its first use    */

/* Host description of one quantised MoE layer (all host pointers, read-only,
 * owned by the caller; row-major, C order).
 *
 *   D      hidden size (>= 1)
 *   E      routed experts (1 .. 1024)
 *   I      expert intermediate size = length of a spectral unit; I % group == 0
 *   n      shared-basis rank = units per (projection, expert), 1 .. 65535
 *   group  quantisation group along the unit vector: 32, 64, 128 or 256
 *   basis  [3] pointers, h = 0 gate, 1 up, 2 down; each D x n bf16 bit patterns,
 *          element (d, j) at d * n + j, so column j is phi_{h,j}
 *   bits   [3][E][n] unit bit-widths, each in {0,1,2,3,4,6,8,16}
 *   alpha  [3][E][n] fp32 spectral energies alpha_{e,h,j}
 *   codes  [3][E][n][I] uint16: for 0 < b < 16 the code q in [0, 2^b) of element i;
 *          for b == 16 the fp16 bit pattern of p_hat[i]; ignored for b == 0
 *   scale, zero  [3][E][n][I / group] fp16 bit patterns; a unit with
 *          0 < b < 16 dequantises as p_hat[i] = scale[g] * (q[i] - zero[g]),
 *          g = i / group; ignored for b in {0, 16}
 */
typedef struct bitsmoe_layer_host {
  int32_t D, E, I, n, group;
  const uint16_t* basis[3];
  const uint8_t* bits;
  const float* alpha;
  const uint16_t* codes;
  const uint16_t* scale;
  const uint16_t* zero;
} bitsmoe_layer_host;

/* Writable destination of an unpack (same layout as bitsmoe_layer_host;
 * every array allocated by the caller at its full size). */
typedef struct bitsmoe_layer_host_out {
  int32_t D, E, I, n, group;
  uint16_t* basis[3];
  uint8_t* bits;
  float* alpha;
  uint16_t* codes;
  uint16_t* scale;
  uint16_t* zero;
} bitsmoe_layer_host_out;

/* Sizes of the packed layer (bytes).  `moved_*` are the algorithmic bytes a
 * forward must read per routed expert: codes of units with b > 0 at b bits per
 * element, fp16 scale + zero per group of quantised units, fp32 alpha per unit
 * with b > 0 (layout padding and index metadata not counted). */
typedef struct bitsmoe_bytes {
  uint64_t total;            /* device image size                               */
  uint64_t basis;            /* 3 * D * n * 2                                   */
  uint64_t codes_padded;     /* code streams as stored (tiles padded)           */
  uint64_t meta;             /* unit indices, alpha, scale/zero, descriptors    */
} bitsmoe_bytes;

typedef struct bitsmoe_layer bitsmoe_layer;   /* opaque, library-owned, device-resident */

/* Pack a host layer into the bucketed device layout and upload it to `device`.
 * Allocates device memory (owned by the returned layer until bitsmoe_free),
 * copies synchronously.  Errors: INVALID_ARG (null pointer, or a code >= 2^b in
 * a unit of 0 < b < 16), SHAPE, UNSUPPORTED_BITS, OOM, CUDA. */
int bitsmoe_pack(const bitsmoe_layer_host* src, int device, bitsmoe_layer** out);

/* Same packing into a host blob (no GPU needed).  *blob is allocated by the
 * library (free with bitsmoe_blob_free); *bytes is its size. */
int bitsmoe_pack_to_host(const bitsmoe_layer_host* src, void** blob, size_t* bytes);
void bitsmoe_blob_free(void* blob);

/* Upload a blob made by bitsmoe_pack_to_host (validated on the host first). */
int bitsmoe_load_blob(const void* blob, size_t bytes, int device, bitsmoe_layer** out);

/* Inverse of packing: rebuild the host arrays bit-exactly from a blob or a
 * device layer (dims must match; arrays preallocated by the caller).  Values
 * not stored (codes/scale/zero of 0-bit units, scale/zero of 16-bit units) are
 * written as 0. */
int bitsmoe_unpack_blob(const void* blob, size_t bytes, bitsmoe_layer_host_out* dst);
int bitsmoe_unpack(const bitsmoe_layer* layer, bitsmoe_layer_host_out* dst);

/* Dims of a packed layer (D, E, I, n, group in that order). */
int bitsmoe_layer_dims(const bitsmoe_layer* layer, int32_t dims[5]);
int bitsmoe_layer_bytes(const bitsmoe_layer* layer, bitsmoe_bytes* out);
/* Algorithmic bytes of expert e, per projection (out[0] gate, out[1] up,
 * out[2] down): codes of units with b > 0 at b bits per element, fp16 scale and
 * zero per group of the quantised units, fp32 alpha per unit with b > 0
 * (layout padding and index metadata not counted). */
int bitsmoe_expert_moved_bytes(const bitsmoe_layer* layer, int e, uint64_t out[3]);

/* Workspace (device bytes) that bitsmoe_moe_forward needs for T tokens and
 * top_k; 0 if the arguments are invalid. */
size_t bitsmoe_workspace_bytes(const bitsmoe_layer* layer, int T, int top_k);

/* Kernels one bitsmoe_moe_forward call launches for (T, top_k) on this layer
 * (no counterpart in the paper: for callers that capture the forward into a
 * CUDA graph or count launches).  A single token runs as one fused persistent
 * kernel (1) when the layer's per-block shares of the bases and factors fit
 * in shared memory, and up to 4 tokens as one such kernel per token (T);
 * otherwise the forward is a chain of 5 kernels, 8 with the tensor-core expert
 * factors (z gather, gate/up and down on tensor cores beside the dp2a kernels;
 * see bitsmoe_forward_plan).
 * Returns a negative error code for invalid arguments. */
int bitsmoe_forward_launches(const bitsmoe_layer* layer, int T, int top_k);

/* How a forward of T tokens runs on this layer, as a bit set:
 *   1  the fused single-token kernel (once per token for up to 4 tokens)
 *   2  the small-batch decode chain (T <= 8 on a layer that does not fit the
 *      fused kernel, else 5 <= T <= 8)
 *   4  tensor-core (tcgen05) shared-basis projections (every T > 8; the decode
 *      chain from 4 tokens)
 *   8  tensor-core gate/up factors with SiLU(gate) * up fused (T > 8 on layers
 *      without 16-bit units whose group is a multiple of 128 rows; otherwise
 *      the dp2a kernel) for the experts with at least 8 tokens (4 when a
 *      factor matrix holds at least 8 M codes), the dp2a kernel for the
 *      others: the codes enter the MMA as fp16 bit patterns
 *  16  tensor-core down factor (the same condition; always set with 8)
 *  32  with 1: the fused kernel is the clustered one, in which a thread-block
 *      cluster owns one (routing slot, 128-row block) pair of the token and
 *      its blocks exchange partial gate/up rows through distributed shared
 *      memory (when the device holds a cluster per pair at once, the layer's
 *      parts fit in shared memory and the pairs' blocks span at least 90% of
 *      the SMs; see bitsmoe_debug_single_token_kernel)
 * Returns a negative error code for invalid arguments; 0 for T == 0. */
int bitsmoe_forward_plan(const bitsmoe_layer* layer, int T, int top_k);

/* Testing hook (no counterpart in the paper): bound every wait of the fused
 * single-token kernels to `spin_clocks` SM clocks (<= 0: the default, about one
 * second), and when skip_arrival is 1 let block 0 skip its arrival at the
 * first grid barrier, so that every other block's bounded wait runs out.  The
 * calls after it report BITSMOE_ERR_TIMEOUT through the device status word and
 * return; the workspace is left ready for the next call.  Applies to calls
 * issued after it on any host thread; skip_arrival = 0 with spin_clocks = 0
 * restores the normal behaviour.  Returns BITSMOE_OK. */
int bitsmoe_debug_wait_limit(int skip_arrival, long long spin_clocks);

/* Testing hook (no counterpart in the paper): which = 1 keeps single-token
 * forwards on the fused kernel without clusters, which = 2 takes the clustered
 * one wherever the device and the layer fit it (bitsmoe_forward_plan reports
 * which), so that tests cover both fused kernels on the same cases; which = 0
 * restores the automatic choice.  Applies to calls issued after it.  Returns
 * BITSMOE_OK, or BITSMOE_ERR_INVALID_ARG for another value. */
int bitsmoe_debug_single_token_kernel(int which);

/* Testing hook (no counterpart in the paper; the stand-in for a memory checker,
 * which this environment does not run): with on = 1 the single-token kernels
 * (both fused kernels) check every staging record before they copy from the
 * packed image -- each gate/up item's code, unit-index, alpha and scale/zero
 * ranges and each down tile's, against the image's size -- and a record that
 * fails is skipped (its item contributes nothing) and reported as
 * BITSMOE_ERR_DEVICE_BOUNDS in the workspace status word (the call's output is
 * then undefined).  Layers packed or loaded while it is on are given a
 * zero-filled slack of the image's own size after the image.  Applies to calls
 * issued after it; on = 0 turns the checks off.  Returns BITSMOE_OK. */
int bitsmoe_debug_bounds(int on);

/* Testing hook (no counterpart in the paper): add `delta` bytes to the code
 * offset of every gate/up staging record of expert e (both fused kernels'
 * tables), so that a test can make those records point outside the image
 * (into the slack of a layer loaded under bitsmoe_debug_bounds(1)) and shift
 * them back.  Synchronous.  Errors: INVALID_ARG, CUDA. */
int bitsmoe_debug_shift_expert_records(const bitsmoe_layer* layer, int e, long long delta);

/* Kernels one bitsmoe_moe_block_forward call launches: 1 a token when the
 * fused single-token kernel runs (it computes the pre-norm and router too),
 * otherwise the norm/router kernel plus bitsmoe_forward_launches. */
int bitsmoe_block_forward_launches(const bitsmoe_layer* layer, int T, int top_k);

/* The quantised MoE-layer forward, asynchronous on `stream`:
 *   x       device, T x D bf16 bit patterns (row-major), 16-byte aligned
 *   logits  device, T x E fp32 router logits (row-major), 16-byte aligned
 *   T       tokens (T == 0 is a successful no-op; T * top_k <= 24576)
 *   top_k   1 .. min(E, 32): experts per token; the k largest logits are
 *           selected (ties to the lower expert index) and weighted by a
 *           softmax over the selected k
 *   y       device, T x D fp32 output (row-major), 16-byte aligned, written
 *   ws      device workspace of >= bitsmoe_workspace_bytes(layer, T, top_k)
 *           bytes, 256-byte aligned, owned by the caller; must not be used by
 *           another call in flight.  Zero-fill it once before its first use
 *           (the single-token kernel keeps a call count and two sets of
 *           grid-barrier counters in its first 64 bytes; each call uses one set
 *           and clears the other for the next call); it may then be reused
 *           across calls, layers and token counts.  A workspace whose counters
 *           are not in that state is reported as BITSMOE_ERR_WORKSPACE_STATE
 *           by bitsmoe_last_device_status and the call computes nothing.
 * Host-side argument checks only: never allocates, never synchronises. */
int bitsmoe_moe_forward(const void* x, const float* logits, int T, int top_k,
                        const bitsmoe_layer* layer, float* y,
                        void* ws, size_t ws_bytes, void* stream);

/* Same forward from host buffers: copies x (T x D bf16) and logits (T x E fp32)
 * from host memory into the workspace, runs the forward, copies y (T x D fp32)
 * back to host memory and synchronises `stream`.  Pinned host memory gives
 * asynchronous copies; pageable memory works but is slower.  A single token
 * on the fused kernel with all three buffers pinned (device-mapped, 16-byte
 * aligned, each with its whole extent -- D x 2, E x 4 and D x 4 bytes -- inside
 * one mapped allocation) skips the copies: the kernel reads x and the logits
 * from, and writes y to, the host buffers directly.  Buffers that do not meet
 * this take the copies. */
int bitsmoe_moe_forward_host(const void* x_host, const float* logits_host, int T, int top_k,
                             const bitsmoe_layer* layer, float* y_host,
                             void* ws, size_t ws_bytes, void* stream);

/* The same without the final synchronisation (no counterpart in the paper: for
 * a serving loop that keeps several steps in flight): every copy and kernel is
 * enqueued on `stream` and the call returns.  The caller synchronises the
 * stream (or an event recorded after the call) before it reads y_host or
 * writes x_host / logits_host again; with pageable buffers the copies are
 * synchronous as in cudaMemcpyAsync.  Consecutive single-token calls on the
 * fused kernel overlap each other's prologue (programmatic dependent launch),
 * as bitsmoe_moe_forward does. */
int bitsmoe_moe_forward_host_async(const void* x_host, const float* logits_host, int T, int top_k,
                                   const bitsmoe_layer* layer, float* y_host,
                                   void* ws, size_t ws_bytes, void* stream);

/* Pre-norm of one MoE block of a decoder stack (the 48-layer MoE FFN stack
 * workload; attention is outside this library):
 *   r = h / sqrt(mean_d h^2 + eps)  (RMSNorm with unit weight), x = bf16(r),
 *   logits = W_r x  (fp32 accumulation of bf16 products).
 *   h          device, T x D fp32 (row-major), 16-byte aligned
 *   w_router   device, E x D bf16 bit patterns, row e = router row of expert e
 *   x_out      device, T x D bf16 bit patterns (written)
 *   logits_out device, T x E fp32 (written)
 * D must be a multiple of 8 (<= 65536), E <= 1024.  Asynchronous on `stream`.
 * The routing rule of the paper's MoE layers is the host model's; this is the
 * common pre-norm + linear router of the evaluated models. */
int bitsmoe_rmsnorm_router(const float* h, const void* w_router, float eps, int T, int D, int E,
                           void* x_out, float* logits_out, void* stream);

/* One pre-norm MoE block in place: h += MoE(x, logits) with x, logits from
 * bitsmoe_rmsnorm_router(h, w_router, eps) and MoE the quantised MoE-layer
 * forward of `layer`.  Workspace and errors as bitsmoe_moe_forward (the
 * normalised activations and logits live in the workspace).  Asynchronous.
 * When the forward runs as the fused single-token kernel, that kernel also
 * computes the norm and the router logits (in the same arithmetic order as
 * bitsmoe_rmsnorm_router, so x and logits are the same bits); otherwise the
 * norm/router kernel runs first. */
int bitsmoe_moe_block_forward(float* h, const void* w_router, float eps, int T, int top_k,
                              const bitsmoe_layer* layer, void* ws, size_t ws_bytes, void* stream);

/* Profiling variant of bitsmoe_moe_forward (same arguments and results): the
 * five phases run without overlap, each bracketed by CUDA events on `stream`,
 * and the call synchronises.  phase_ms[0..4] receive the durations of
 * routing, shared-basis projection (gate, up), gate/up factors + SwiGLU
 * inputs, down factor + weighted expert sum, output basis.  When the forward
 * runs as fused kernels (see bitsmoe_forward_plan), its phases cannot be
 * separated: phase_ms[0] receives the whole forward and the others 0. */
int bitsmoe_profile_forward(const void* x, const float* logits, int T, int top_k,
                            const bitsmoe_layer* layer, float* y,
                            void* ws, size_t ws_bytes, void* stream, float phase_ms[5]);

/* Largest workspace (bytes, as bitsmoe_workspace_bytes reports it) that
 * bitsmoe_moe_forward_noalloc can serve from its built-in scratch. */
#define BITSMOE_NOALLOC_SCRATCH_BYTES (8u << 20)

/* The forward of bitsmoe_moe_forward without a caller-provided workspace, for
 * callers that cannot allocate device memory themselves: a serving runtime
 * whose allocator has already reserved the device's memory, a plugin inside a
 * framework whose caching allocator owns all device memory, or a decode loop
 * that must not call cudaMalloc because cudaMalloc can synchronise the device.
 * (The BitsMoE paper has no counterpart; this is a deployment convenience.)
 *
 * The scratch is one fixed device array of BITSMOE_NOALLOC_SCRATCH_BYTES
 * (8 MiB) inside the library, present on every GPU that loads the library
 * until the process exits.  This call allocates nothing: no cudaMalloc, no
 * cudaFree, no allocating library routine.  The first call on a device looks
 * up that device's address of the array (once per device, with the device
 * current); make the first call before any stream capture (a first call on
 * a device while `stream` is capturing returns BITSMOE_ERR_INVALID_ARG).
 *   x, logits, y, T, top_k, layer, stream: as for bitsmoe_moe_forward.
 * Errors: as bitsmoe_moe_forward, and BITSMOE_ERR_WORKSPACE_TOO_SMALL when
 * bitsmoe_workspace_bytes(layer, T, top_k) > BITSMOE_NOALLOC_SCRATCH_BYTES.
 * Every call on a device shares the one array and it keeps the last call's
 * contents (each forward clears what it accumulates into before using it),
 * so calls that overlap on the GPU (different streams, or different host
 * threads) race and give wrong results: serialise them. */
int bitsmoe_moe_forward_noalloc(const void* x, const float* logits, int T, int top_k,
                                const bitsmoe_layer* layer, float* y, void* stream);

/* Device status word of the no-allocation scratch on the current device: what
 * bitsmoe_last_device_status reports for a caller's workspace, for the calls
 * of bitsmoe_moe_forward_noalloc (whose workspace the caller cannot name).
 * Synchronises `stream`, returns BITSMOE_OK or the first device-side error a
 * no-allocation call recorded (BITSMOE_ERR_TIMEOUT, BITSMOE_ERR_WORKSPACE_STATE,
 * BITSMOE_ERR_DEVICE_BOUNDS) and clears it.  Not during a stream capture. */
int bitsmoe_noalloc_last_status(void* stream);

/* Quantise spectral units into the stored unit format above (the offline
 * step that produces `codes`, `scale` and `zero` of bitsmoe_layer_host), on
 * the GPU, asynchronously on `stream`.  BitsMoE quantises every normalised
 * spectral vector p (a unit, length I) with its own bit-width b (appendix
 * "Piecewise Reconstruction Error for Bit Allocation"), one scale per group
 * of `group` consecutive elements (group 128 in the paper's experiments):
 *   b = 2, 3, 4  symmetric uniform quantiser Q_b(p; s) = s clamp(round(p / s),
 *                -2^(b-1), 2^(b-1) - 1) (Eq. app_scalar_quantization_uk) with
 *                the MSE-optimal scale (Eq. app_low_bit_opt_scale), searched
 *                over the fp16 candidates s_c = fp16(rho 2^(2-b) c / grid),
 *                c = 1 .. grid, rho = max |p| over the group
 *   b = 6, 8     Q_b with s = fp16(rho / (2^(b-1) - 1)) (Eq. app_uk_scale)
 *   b = 1        sign quantiser mean|p| sign(p), sign(0) = +1
 *                (Eq. app_one_bit_quantization)
 *   b = 0        evicted (Eq. app_zero_bit_vector); b = 16: fp16 values.
 * Stored: code = level + 2^(b-1), zero = 2^(b-1), scale = s (sign quantiser:
 * code = [p >= 0], zero = 1/2, scale = 2 mean|p|); 0-bit units store zeros,
 * 16-bit units the fp16 bit patterns and scale = zero = 0.  Arithmetic is
 * fp32 with every operation rounded once, the quotient p / s taken as p times
 * the rounded reciprocal of s, error sums in element order, ties to the
 * smaller c; the result is deterministic.  A group with no usable scale (all
 * zeros, or every candidate 0 or infinite in fp16) stores scale 0.
 *   p       device, U x I fp32 (row u = unit u), 16-byte aligned, finite values
 *   bits    device, U bit-widths
 *   U       units (U == 0 is a successful no-op); I % group == 0
 *   group   32, 64, 128 or 256
 *   grid    candidates of the scale search: 32, 64, 128, 256, 512 or 1024
 *   codes   device, U x I uint16 (written), 16-byte aligned
 *   scale, zero  device, U x (I / group) fp16 bit patterns (written)
 *   status  device int or NULL: a unit whose bit-width is not in
 *           {0,1,2,3,4,6,8,16} gets zero outputs and, if status is not NULL
 *           and holds 0, BITSMOE_ERR_UNSUPPORTED_BITS is written there
 * Host-side checks only (INVALID_ARG, SHAPE, ALIGNMENT); never allocates,
 * never synchronises.  One kernel launch. */
int bitsmoe_quantize_units(const float* p, const uint8_t* bits, int64_t U, int I, int group, int grid,
                           uint16_t* codes, uint16_t* scale, uint16_t* zero, int* status, void* stream);

/* Bit allocation for the units of one projection type (the offline step that
 * produces `bits` of bitsmoe_layer_host), on the GPU, asynchronously on
 * `stream`.  BitsMoE picks b_u in {0,1,2,3,4,6,8,16} for every unit u by the
 * ILP of Eq. ilp_piecewise_eps: minimise sum_u C_u(b_u) subject to
 * sum_u b_u <= budget, with C_u(b) = alpha_u^2 beta_u^gamma E_u(b) (Eq.
 * app_component_loss_final) and the piecewise distortion of Eq.
 * piecewise_expected_eps: E(0) = 1, E(1) = 1 - ||p_u||_1^2 / d,
 * E(2|3|4) = kappa_2|3|4 (Table kappa_values: 0.14949200, 0.04067890,
 * 0.01184786), E(6|8|16) = (d ||p_u||_inf^2 / 3) 2^(-2b).  The budget of the
 * paper is B_h = floor(E n b_eq - 16 n^2 / m) (Eq.
 * app_projection_normalized_budget) for E experts, rank n, unit length m.
 * The ILP is solved by its Lagrangian relaxation plus a greedy fill: per unit
 * the lower convex hull of (b, C(b)) from b = 0 (ties to the smaller b); hull
 * increments taken in descending efficiency (ties to the lower unit index)
 * while the bits fit, a group of equal efficiency within a unit whole or not
 * at all (this part is an exact optimum for the bits it uses); then, while
 * some unit's next increment fits the bits left, the most efficient one.
 * Arithmetic is fp32, each operation rounded once (||p||_1 as an exact
 * fixed-point sum of floor(|p_i| 2^40)); the result is deterministic.
 *   p       device, U x d fp32 (row u = unit u, the normalised spectral
 *           vector), 16-byte aligned, |p_i| < 32
 *   alpha   device, U fp32 spectral energies; beta device, U fp32 importances
 *           (beta_u = phi_u^T H phi_u, Eq. app_beta_vector_def), beta >= 0
 *   gamma   smoothing exponent in [0, 1]; 0, 1/2 and 1 are exact (1, sqrt,
 *           identity), other values use powf
 *   U       units, 0 .. 2^32 - 2 (U == 0 is a successful no-op); 1 <= d <= 16384
 *   kappa   host, 3 floats: the distortion of 2, 3 and 4 bits
 *   budget  >= 0, in bits per unit element (sum of b_u)
 *   bits    device, U bytes (written)
 *   ws      device workspace of >= bitsmoe_allocate_workspace_bytes(U)
 *           bytes, 256-byte aligned, caller-owned; no initialisation needed
 * Host-side checks only (INVALID_ARG, SHAPE, ALIGNMENT,
 * WORKSPACE_TOO_SMALL); never allocates, never synchronises.  43 kernel
 * launches and one memset on `stream`. */
size_t bitsmoe_allocate_workspace_bytes(int64_t U);
/* The budget of one projection type, B_h = floor(E n b_eq - 16 n^2 / m) (Eq.
 * app_projection_normalized_budget): E experts, shared rank n, unit length m,
 * target equivalent bits b_eq = beq_num / beq_den (the fp16 bases are
 * charged against it).  Exact integer arithmetic on the host; *out may be
 * negative for layers whose bases alone exceed the target (no allocation can
 * meet it).  Errors: INVALID_ARG (null out, non-positive sizes or
 * denominator, negative numerator), SHAPE (E, n > 2^20, m > 2^24, numerator
 * or denominator > 2^16). */
int bitsmoe_projection_budget(int64_t E, int64_t n, int64_t m, int64_t beq_num, int64_t beq_den, int64_t* out);
int bitsmoe_allocate_bits(const float* p, const float* alpha, const float* beta, float gamma, int64_t U, int d,
                          const float* kappa, int64_t budget, uint8_t* bits, void* ws, size_t ws_bytes,
                          void* stream);
/* Same, with the phases timed by CUDA events on `stream` and the call
 * synchronised: phase_ms[0] the cost and hull kernel, [1] the selection of the
 * cut and the per-unit result, [2] the fill. */
int bitsmoe_profile_allocate_bits(const float* p, const float* alpha, const float* beta, float gamma, int64_t U,
                                  int d, const float* kappa, int64_t budget, uint8_t* bits, void* ws,
                                  size_t ws_bytes, void* stream, float phase_ms[3]);

/* Importance beta of every spectral unit from calibration tokens, on the GPU:
 * the allocation's input (bitsmoe_allocate_bits' beta), computed on the float
 * factors of the shared-basis decomposition before anything is quantised.
 * BitsMoE weighs each unit's quantisation loss by the activation metric of its
 * expert, H_e = X Diag(g_e) X^T over the calibration activations X with the
 * tokens' routing affinities g_e (appendix Eq. app_affinity_gram):
 *   beta[h][e][k] = phi_{h,k}^T H_e phi_{h,k}
 *                 = sum_t g_{t,e} (phi_{h,k}^T x_t)^2                 h = gate, up
 *   beta[2][e][k] = p_{dn,e,k}^T H'_e p_{dn,e,k}
 *                 = sum_t g_{t,e} (p_{dn,e,k}^T h_{t,e})^2             down
 * with h_{t,e} = SiLU(P_g,e diag(alpha_g,e) Phi_g^T x_t) * (P_u,e diag(alpha_u,e)
 * Phi_u^T x_t) the expert's SwiGLU output (appendix Eqs. app_beta_def,
 * app_down_beta_approx, app_unified_beta_def).  A token's affinity to expert e
 * is its gate weight (softmax over its top_k logits, ties to the lower index)
 * when e is selected and 0 otherwise.
 *   x        device, T x D bf16 calibration activations (row-major)
 *   logits   device, T x E fp32 router logits of those tokens
 *   basis    host array of 2 device pointers: Phi_gate, Phi_up, each D x n fp32
 *            (row d, column k = phi_k)
 *   alpha    host array of 2 device pointers: alpha_gate, alpha_up, E x n fp32
 *   factor   host array of 3 device pointers: P_gate, P_up, P_down, each
 *            E x I x n fp32 (expert e's I x n factor, column k = p_{e,k})
 *   beta     device, 3 x E x n fp32 (written)
 *   ws       device workspace of >= bitsmoe_importance_workspace_bytes(T, E,
 *            I, n, top_k) bytes, 256-byte aligned, caller-owned
 * fp32 arithmetic throughout (the contractions on the CUDA cores).  T == 0
 * writes beta = 0.  Host-side checks only (INVALID_ARG, SHAPE,
 * WORKSPACE_TOO_SMALL); asynchronous on `stream`, never allocates. */
size_t bitsmoe_importance_workspace_bytes(int64_t T, int E, int I, int n, int top_k);
int bitsmoe_importance(const void* x, const float* logits, int64_t T, int D, int E, int I, int n, int top_k,
                       const float* const basis[2], const float* const alpha[2], const float* const factor[3],
                       float* beta, void* ws, size_t ws_bytes, void* stream);

/* Shared-basis spectral decomposition of one projection type over its E experts
 * (Sec. "Shared-basis Spectral Decomposition": Eq. shared_basis_input_proj and
 * Eq. app_cat_svd_absorbed for gate/up, the concatenation along input channels
 * of Eq. app_down_cat_svd_absorbed for down; alpha and P by Definitions
 * spectral_energy_matrix / spectral_matrix):
 *   side 0 ("in", gate/up): W is E x d x D (W_e = d x D), W_cat = [W_1; ...; W_E]
 *                           = U S Phi^T, P~_cat = U S split into E row blocks
 *   side 1 ("out", down):   W is E x D x d (W_e = D x d), W_cat = [W_1 ... W_E]
 *                           = Phi S V^T, P~_cat = V S split by input channels
 *   alpha[e][k] = ||P~_e[:, k]||_2, P_e = P~_e / alpha_e (P~_e where alpha = 0).
 * Computed as the eigendecomposition of G = W_cat^T W_cat (side 0) or W_cat W_cat^T
 * (side 1), D x D, in fp32 (cyclic two-sided Jacobi), then P~ = W_cat Phi (side 0)
 * or W_cat^T Phi (side 1).  n = min(D, E d) columns, by descending singular
 * value (ties: the lower eigenvector index); each basis column's largest
 * |component| is positive (the first one on ties).  Singular values and
 * vectors are those of W_cat up to fp32 rounding; a vector whose singular value
 * is repeated is any orthonormal basis of its space.
 *   W       device, fp32, 16-byte aligned, finite
 *   E, d, D experts, their intermediate size, the feature dimension
 *           (2 <= D <= BITSMOE_DECOMPOSE_MAX_D)
 *   phi     device, D x n fp32 (column k = phi_k) (written)
 *   sigma   device, n fp32 singular values, descending (written)
 *   alpha   device, E x n fp32 (written)
 *   P       device, E x n x d fp32, unit-major: P[e][k][:] = p_{e,k}, the row
 *           layout bitsmoe_quantize_units takes (written)
 *   ws      device workspace of >= bitsmoe_decompose_workspace_bytes(side, E, d, D)
 *           bytes, 256-byte aligned
 *   max_sweeps  Jacobi sweeps at most (>= 1; the solver stops earlier after a
 *           sweep in which no rotation was needed: every |g_pq| <= 1e-7
 *           sqrt(|g_pp g_qq|) or <= 4e-7 max_j |g_jj|)
 *   sweeps  device int or NULL: the sweeps run (written)
 *   status  device int: BITSMOE_ERR_TIMEOUT is written there if a bounded
 *           grid-barrier wait of the solver ran out (the call then leaves its
 *           outputs undefined); it is not cleared by the call
 * Host-side checks (INVALID_ARG, WORKSPACE_TOO_SMALL, ALIGNMENT, SHAPE when the
 * solver's block cannot be resident); never allocates, never synchronises.  Six
 * kernel launches (one cooperative). */
#define BITSMOE_DECOMPOSE_MAX_D 8192
size_t bitsmoe_decompose_workspace_bytes(int side, int E, int d, int D);
int bitsmoe_shared_basis(int side, const float* W, int E, int d, int D, float* phi, float* sigma, float* alpha,
                         float* P, void* ws, size_t ws_bytes, int max_sweeps, int* sweeps, int* status,
                         void* stream);

/* Calibration Gram H = X^T Diag(g) X = sum_t g_t x_t x_t^T (appendix,
 * Eq. app_affinity_gram: the activation metric of one expert with the routing
 * affinities g of its tokens), fp32.
 *   x   device, T x D bf16 (row t = x_t)
 *   g   device, T fp32 weights, or NULL (all 1)
 *   H   device, D x D fp32 (written; symmetric)
 * T == 0 writes zeros.  Never allocates, never synchronises; one launch. */
int bitsmoe_calibration_gram(const void* x, const float* g, int64_t T, int D, float* H, void* stream);

/* Where bitsmoe_moe_block_forward(T, top_k) leaves the block's normalised
 * activations x (T x D bf16) and router logits (T x E fp32) in its workspace:
 * byte offsets from the workspace start, valid after the call completes (the
 * fused single-token kernel, which normalises and routes inside, writes them
 * there too).  For inspection and tests; no counterpart in the paper.
 * Errors: INVALID_ARG. */
int bitsmoe_block_norm_outputs(const bitsmoe_layer* layer, int T, int top_k, size_t* x_offset,
                               size_t* logits_offset);

/* Synchronise `stream`, then read and clear the device status word kept in
 * `ws`: BITSMOE_OK, or the first device-side error recorded by the last
 * forward that used this workspace (each forward resets it when it starts). */
int bitsmoe_last_device_status(void* ws, void* stream);

/* Free a packed layer and its device memory (NULL is ignored). */
void bitsmoe_free(bitsmoe_layer* layer);

const char* bitsmoe_strerror(int code);
/* The cudaError_t of the last BITSMOE_ERR_CUDA on this thread. */
int bitsmoe_last_cuda_error(void);

#ifdef __cplusplus
}
#endif
#endif /* BITSMOE_H */
