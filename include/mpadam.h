/*
 * mpadam.h -- C ABI of the GB300 (sm_103a) fused M+Adam optimizer step.
 *
 * M+Adam (arxiv 2607.10611) updates every parameter w with two branches:
 *   additive (Algorithm 1, Sec. 4.1):   mu, nu Adam moments with bias
 *       correction, u_a = -eta_a mu-hat / (sqrt(nu-hat) + eps);
 *   multiplicative (Algorithm 1, Sec. 4.1): exponent gradient
 *       g_e = (ln 2) w g, second moment nu_e, proposal
 *       u~ = -eta_m g_e / (sqrt(nu_e-hat) + eps), rho = max(|w|, tau),
 *       u_m = clip(u~ / rho);
 * and combines them as w <- w + w u_m + u_a, then rounds w straight back into
 * its low-precision storage format (Appendix B's FP32-compute / BF16-storage
 * round trip; FP8 master weights of Sec. 5.2).  Algorithm 2 (Appendix A) adds
 * the optional clamp g_max of the normalised exponent gradient, the relative
 * bounds [-(0.75 - eps0), 0.75], the optional per-step cap |log2(1 + u_m)| <=
 * d_mult,max, the optional weight clip w_max and decoupled weight decay.
 *
 * One mpadam_step() is one fused pass over every element of a tensor list:
 * each element is read once (w, g, mu, nu, nu_e) and written once (w, mu, nu,
 * nu_e) by a single kernel launch.
 *
 * Arithmetic: IEEE binary32, round-to-nearest-even, with fused multiply-adds
 * exactly where the canonical sequence below has them; results are
 * bit-for-bit reproducible for a given (inputs, config, step).  Per element:
 *   mu'  = fma(b1, mu, (1-b1) g)          nu'  = fma(b2, nu, (1-b2) (g g))
 *   u_a  = (ka mu') / fma(sqrt(nu'), c2, eps)   [ - (eta_a lambda) w ]
 *   g_e  = ((ln 2) w) g                   nu_e'= fma(b2, nu_e, (1-b2) (g_e g_e))
 *   n    = g_e / fma(sqrt(nu_e'), c2, eps)      [ clamped to +-g_max ]
 *   u_m  = ((-eta_m) n) / max(|w|, tau),  clamped to [lo, hi]
 *   w'   = fma(w, u_m, w) + u_a                 [ clipped to +-w_max ]
 * with per-step binary32 scalars computed in binary64 and rounded once:
 *   ka = -eta_a / (1 - beta1^t), c2 = 1 / sqrt(1 - beta2^t) (both without
 *   the beta terms when bias_correction = 0), hi = min(rmax_pos, 2^d - 1) and
 *   lo = max(-rmax_neg, 2^-d - 1) rounded towards zero (d = dmult_max), which
 *   is the log2/exp2 cap of Algorithm 2 written as the equivalent clamp.
 * The updated moments are stored from the unrounded binary32 values.
 *
 * Storage rounding (the paper cites stochastic rounding but gives no
 * formula; these are this library's definitions):
 *   BF16 nearest: round-to-nearest-even; NaN stores 0x7FFF.
 *   BF16 stochastic: round away from zero iff R16 < (low 16 bits of the
 *     binary32), R16 the element's 16 random bits (exactly unbiased).
 *   E4M3 (OCP FP8 "fn": bias 7, largest finite 448, NaN 0x7F): the value is
 *     first multiplied by 2^-e (per-tensor power-of-two scale); nearest-even
 *     or stochastic (away iff R32 < floor(fraction * 2^32)); |x| >= 448 and
 *     infinities saturate to +-448; NaN stores 0x7F.
 *   Random bits: Philox4x32-10 (Salmon et al., SC'11) with key = seed and
 *     counter = (block lo, block hi, step lo, step hi).  Global element index
 *     i draws, for BF16 storage, 16-bit lane i mod 8 of block i div 8 (lane
 *     L is the low half of word L/2 when L is even, the high half when odd),
 *     and for E4M3 storage word i mod 4 of block i div 4.
 *   Global element index: tensor k's element j has index off[k] + j, where
 *     off[0] = 0 and off[k+1] = off[k] + numel[k] rounded up to a multiple of
 *     8.  Splitting a tensor at a multiple of 8 therefore changes nothing.
 *
 * E4M3 delayed scaling (the paper stores FP8 with scales but does not say
 * how they are chosen): tensor k's stored weights decode as code * 2^e_t.  A
 * step re-encodes with e_{t+1} = the smallest integer e with
 * A_t <= 448 * 2^e (kept at e_t when A_t = 0; clamped to [-100, 100]), where
 * A_t is the largest finite |w'| the previous step produced (or, before the
 * first step, the largest |decoded stored weight|), and records A_{t+1}.
 * The caller owns two device rings that hold this state:
 *   fp8_exp  : int32[2 n],  e_t of tensor k at fp8_exp[(t mod 2) n + k];
 *   fp8_amax : uint32[3 n], binary32 bits of A_t at fp8_amax[(t mod 3) n + k].
 * Step t reads slot t, writes slot t+1 and clears amax slot t+2.  Amax
 * slot t+1 must hold 0 when step t starts (mpadam_fp8_init and step t-1
 * leave it so): the step raises it with exact |w'| values only, and also
 * reads it while it runs as a lower bound of A_{t+1}.
 *
 * Conventions for every entry point:
 *   - returns MPADAM_OK (0) or a positive mpadam_status; never aborts or
 *     throws across the ABI; mpadam_last_error() then holds a message (per
 *     host thread);
 *   - `stream` is a cudaStream_t (NULL = legacy default stream);
 *   - device pointers are addresses in the current CUDA context's device;
 *     all tensor memory is owned by the caller; the library owns only the
 *     metadata it allocates in mpadam_create and frees in mpadam_destroy;
 *   - calls on one state are not thread-safe and must all be issued to the
 *     same stream (or ordered by the caller).
 */
#ifndef MPADAM_H
#define MPADAM_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

struct CUstream_st; /* cudaStream_t is `struct CUstream_st *` */

typedef enum {
  MPADAM_OK = 0,
  MPADAM_EINVAL = 1,       /* bad argument; nothing was launched */
  MPADAM_EALLOC = 2,       /* a device or pinned host allocation failed */
  MPADAM_ECUDA = 3,        /* a CUDA runtime call or launch failed */
  MPADAM_EUNSUPPORTED = 4  /* valid request this build does not implement */
} mpadam_status;

/* MPADAM_E4M3_B32: E4M3 codes with one FP16 power-of-two scale per 32
 * consecutive elements.  MPADAM_NVFP4: E2M1 codes (OCP FP4), two per byte,
 * with one E4M3 scale per 16 consecutive elements and one binary32 scale per
 * tensor.  Both are block-scaled weight formats (mpadam_create_ex). */
typedef enum {
  MPADAM_F32 = 0, MPADAM_BF16 = 1, MPADAM_E4M3 = 2, MPADAM_E4M3_B32 = 3, MPADAM_NVFP4 = 4
} mpadam_dtype;
typedef enum { MPADAM_ROUND_NEAREST = 0, MPADAM_ROUND_STOCHASTIC = 1 } mpadam_rounding;

/* One parameter tensor (Algorithm 1's state per parameter: w, mu, nu, nu_e),
 * a contiguous 1-D view of `numel` elements in caller-owned device memory.
 * w has the config's weight_dtype; m, v, ve its moment_dtype.  Pointers must
 * be aligned to their element size (may be NULL only when numel == 0).
 * Tensors whose pointers are all 32-byte aligned take the vectorised path;
 * others are correct but slower. */
typedef struct {
  void* w;
  void* m;
  void* v;
  void* ve;
  int64_t numel;
} mpadam_tensor;

/* Hyper-parameters (Algorithm 1 "Inputs", Algorithm 2 options).
 * Valid ranges (else MPADAM_EINVAL): lr_add, lr_mul >= 0 and finite;
 * 0 <= beta1, beta2 < 1; eps > 0, tau > 0 finite; rmax_pos > 0 finite;
 * 0 < rmax_neg < 1; g_max, dmult_max, w_max > 0 (+INFINITY switches the
 * option off); wd_add >= 0 finite (0 = off). */
typedef struct {
  float lr_add;            /* eta_a */
  float lr_mul;            /* eta_m */
  float beta1, beta2;
  float eps;               /* epsilon of both denominators */
  float tau;               /* rho = max(|w|, tau) */
  float rmax_pos;          /* u_m <= rmax_pos (Algorithm 2: 0.75) */
  float rmax_neg;          /* u_m >= -rmax_neg (Algorithm 2: 0.75 - eps0) */
  float g_max;             /* |n| <= g_max */
  float dmult_max;         /* |log2(1 + u_m)| <= dmult_max */
  float w_max;             /* |w'| <= w_max */
  float wd_add;            /* lambda: u_a -= eta_a lambda w (AdamW-style) */
  int32_t bias_correction; /* 1: Algorithm 1's mu-hat, nu-hat; 0: Algorithm 2 */
  int32_t rounding;        /* mpadam_rounding of the weight store */
  uint64_t seed;           /* Philox key of stochastic rounding */
  int32_t weight_dtype;    /* MPADAM_BF16 or MPADAM_E4M3 */
  int32_t grad_dtype;      /* MPADAM_F32 or MPADAM_BF16 */
  int32_t moment_dtype;    /* MPADAM_F32 or MPADAM_BF16 (stored nearest-even) */
  int32_t reserved;        /* must be 0 */
} mpadam_config;

typedef struct mpadam_state mpadam_state;

/* One parameter tensor of a list that may mix weight formats (the paper's
 * FP8 regime, Sec. 5.2 and the FP8-master figure: FP8 linear layers with
 * FP16 block scales, BF16 embeddings, norms and head).  w, m, v, ve, numel
 * as in mpadam_tensor (m, v, ve of the config's moment_dtype).
 *   weight_dtype: MPADAM_BF16, MPADAM_E4M3 (per-tensor scale, delayed, held
 *     in the fp8 rings as described above), MPADAM_E4M3_B32 or MPADAM_NVFP4;
 *   block_scale: E4M3_B32 and NVFP4 only (else NULL).  For E4M3_B32, a
 *     device array of ceil(numel/32) FP16 bit patterns, the scale of
 *     elements [32b, 32b + 32) at index b,
 *     2-byte aligned (16-byte aligned for the staged fast path).  Stored
 *     weights decode as code * scale.  A step rewrites every block's scale
 *     with 2^k, k the smallest integer with A <= 448 * 2^k (A = the block's
 *     largest finite |w'| of this step; current scaling), clamped to
 *     [-24, 15] (every such power is an FP16 number); a block whose A is 0
 *     keeps the exponent of its old scale.  The new codes encode w' * 2^-k
 *     (nearest-even or stochastic, saturating at +-448, as for E4M3).
 *     Scales should be powers of two; another FP16 value decodes as itself
 *     and counts as the power of two at or below it.  For NVFP4, a device
 *     array of ceil(numel/16) E4M3 codes, the scale s of elements
 *     [16b, 16b + 16) at index b (16-byte aligned for the staged fast path);
 *     w holds ceil(numel/2) bytes, element 2i in the low nibble of byte i
 *     (the spare high nibble of an odd-length tensor is written 0).  A
 *     weight decodes as q * d with d = s * G (G = global_scale; both
 *     products rounded to binary32).  A step rewrites every block's scale
 *     with the smallest E4M3 code c in [1, 126] such that 6 * (value(c) * G)
 *     (products rounded) >= A, the block's largest finite |w'| (126 when
 *     none; kept when A = 0), and the codes with E2M1(w' / d') (quotient
 *     rounded to binary32; nearest-even, or stochastic: away from zero iff
 *     R32 < floor(fraction * 2^32), with the E4M3 random lanes; |x| >= 6
 *     saturates, NaN stores +0);
 *   compute: optional (NULL = none; E4M3, E4M3_B32 and NVFP4 only): device
 *     array of numel BF16 values, 2-byte aligned (16-byte for the vector
 *     path), overwritten every step with the dequantised updated weights
 *     bf16(decoded weight) from the same kernel pass that writes the codes
 *     (Sec. 5.2's low-precision master weights feed a BF16 forward pass);
 *     for the E4M3 formats this is exact (code * scale is a BF16 number);
 *   global_scale: NVFP4 only, the tensor's binary32 scale G (finite, > 0),
 *     held fixed by the step; 0 for every other format. */
typedef struct {
  void* w;
  void* m;
  void* v;
  void* ve;
  int64_t numel;
  int32_t weight_dtype;
  float global_scale;
  void* block_scale;
  uint16_t* compute;
} mpadam_tensor_ex;

/* Build the fused step for a tensor list (Algorithm 1 "State").  Copies
 * `tensors` (the caller may free the array), validates, lays out the global
 * element index, allocates and uploads device metadata (synchronously, on the
 * current device).  fp8_exp / fp8_amax: the caller-owned device rings
 * described above, required for E4M3 weights, NULL otherwise.  n may be 0.
 * Errors: EINVAL (arguments), EALLOC, ECUDA.  On error *out is NULL. */
int32_t mpadam_create(const mpadam_tensor* tensors, int32_t n, const mpadam_config* cfg,
                      int32_t* fp8_exp, uint32_t* fp8_amax, mpadam_state** out);

/* The same for a list whose tensors each name their weight format (and
 * carry block scales and compute copies, see mpadam_tensor_ex); cfg's
 * weight_dtype is not used.  The tensors are stepped by one kernel launch
 * per format present, in the order BF16, E4M3, E4M3_B32, NVFP4, all on the stream
 * given to mpadam_step; global element indices (stochastic rounding) are
 * those of the whole list, and the fp8 rings (required when any tensor is
 * E4M3, else may be NULL) are indexed by list position k over all n
 * tensors; entries of other tensors are left alone by the step.
 * Errors: EINVAL (arguments), EALLOC, ECUDA.  On error *out is NULL. */
int32_t mpadam_create_ex(const mpadam_tensor_ex* tensors, int32_t n, const mpadam_config* cfg,
                         int32_t* fp8_exp, uint32_t* fp8_amax, mpadam_state** out);

/* E4M3 only: seed the scale state before `first_step` (t0 >= 1).  Writes
 * init_exp (host array of n exponents in [-100, 100], the exponents the
 * stored weights are currently encoded with) into both fp8_exp slots, clears
 * all fp8_amax slots and writes A_t0 = largest |decoded stored weight| of
 * each tensor into slot t0 mod 3, on `stream`.  In a mixed list only the
 * per-tensor-scaled E4M3 tensors' entries are checked and used (the others
 * are written as 0).  Errors: EINVAL, ECUDA. */
int32_t mpadam_fp8_init(mpadam_state* s, const int32_t* init_exp, int64_t first_step,
                        struct CUstream_st* stream);

/* One M+Adam step t (>= 1) over every tensor, asynchronously on `stream`.
 * grads: host array of n device pointers, grads[k] holding numel[k]
 * gradients of grad_dtype (read only).  The pointer table is re-uploaded
 * only when it differs from the previous call's.  On `stream` the call puts
 * one kernel launch per weight format and, while a tail pool is on (see
 * mpadam_set_tail_pool), one cudaMemsetAsync of the pool's counters before
 * them.  Steps of one state must not overlap on the GPU.  The same (inputs, t, seed) reproduce the
 * same bits, so a resumed run calls with the step it stopped at.
 * Errors: EINVAL (t < 1, NULL/misaligned grads), ECUDA (launch). */
int32_t mpadam_step(mpadam_state* s, const void* const* grads, int64_t step,
                    struct CUstream_st* stream);

/* The same step with gradients and weights in host memory: copies
 * host_grads[k] (numel[k] gradients each) to library-owned device staging,
 * runs the step, and copies every updated weight tensor back to
 * host_w_out[k] (numel[k] weights of its weight format each, NVFP4 packed
 * two per byte; block scales and compute copies stay in device memory).  The host buffers should be
 * pinned.  When the list has one weight format other than NVFP4 and
 * host_grads, host_w_out
 * and the device weights each follow the global-index layout of one flat
 * allocation (pointer k = base + off[k] * element size), the step is
 * pipelined in up to 8 chunks of whole
 * tiles: chunk c's gradients upload on an internal stream while chunk c-1 is
 * stepped on `stream` and chunk c-2's weights download on a second internal
 * stream (copies cover each chunk's whole global-index range, padding
 * included); otherwise the copies are one per tensor, before and after the
 * step.  Either way the work is ordered after earlier work on `stream`, and
 * `stream` completes only after the last download.  The first call allocates
 * the staging buffer and the pipeline's streams and events.
 * Errors: EINVAL, EALLOC, ECUDA. */
int32_t mpadam_step_host(mpadam_state* s, const void* const* host_grads, void* const* host_w_out,
                         int64_t step, struct CUstream_st* stream);

/* Page-locked host memory for mpadam_step_host's buffers (not from the
 * paper: a deployment aid).  Allocates `bytes` of anonymous memory advised
 * for transparent huge pages and preferring the host NUMA node nearest the
 * current device, touches it (so the pages are resident and large), and
 * registers it with the CUDA driver (cudaHostRegister).  Copies
 * from such a buffer keep the host link's full rate: on GB300 (Grace) hosts,
 * copies from ordinary pinned memory of 64 KB pages measured 4x slower at
 * times for buffers of several GB, huge-page buffers did not.  On the 7B list
 * (13.5 GB each way), mpadam_step_host on ordinary pinned buffers had steps of
 * up to 3.2x the usual 87.6 ms on some hosts, about one in four; on huge-page
 * buffers, none in 40 steps alternating with them.  Release with
 * mpadam_host_buffer_free (same size).  Errors: EINVAL, EALLOC, ECUDA. */
int32_t mpadam_host_buffer_alloc(int64_t bytes, void** out);
int32_t mpadam_host_buffer_free(void* ptr, int64_t bytes);

/* Fault injection for tests (the paper has no counterpart): the library's
 * device or pinned allocation after `after` more successful ones fails once,
 * as if the driver had refused it (every entry point then returns
 * MPADAM_EALLOC and releases what it had allocated); -1 disarms.  Process-
 * wide.  Errors: EINVAL. */
int32_t mpadam_debug_fail_allocation(int32_t after);

/* Host only, no GPU: the tile schedule mpadam_step's launches walk for a list
 * of n tensors (numel, in launch order) on `ctas` CTAs with the tail pool
 * (static_q, chunk_tiles) of mpadam_set_tail_pool.  Tiles are 3840 elements,
 * numbered tensor by tensor.  cta_runs[3b..3b+2] = (tb, ts, te): CTA b walks
 * [tb, ts) itself and its tiles [ts, te) go to the pool; cta_first[b] is the
 * tensor holding tile tb.  pool[3i..3i+2] = (first tile, tile count, tensor
 * of the first tile) of chunk i, in the order CTAs claim them;
 * *pool_count = number of chunks.  Outputs: cta_runs [3 * ctas],
 * cta_first [ctas], pool [3 * pool_cap].  Errors: EINVAL (arguments, or
 * pool_cap below the chunk count, which is still reported), EALLOC. */
int32_t mpadam_debug_tile_schedule(const int64_t* numel, int32_t n, int32_t ctas, int32_t static_q,
                                   int32_t chunk_tiles, int64_t* cta_runs, int32_t* cta_first,
                                   int64_t* pool, int32_t pool_cap, int32_t* pool_count);

/* Frees the library's metadata (synchronises the device first).  NULL is a
 * no-op.  Never touches caller-owned tensors. */
int32_t mpadam_destroy(mpadam_state* s);

/* Message of the last non-OK status returned on this host thread. */
const char* mpadam_last_error(void);

/* Layout queries: *offset = global index of tensor k's first element;
 * *length = total length of the padded global index space. */
int32_t mpadam_global_offset(const mpadam_state* s, int32_t k, int64_t* offset);
int32_t mpadam_global_length(const mpadam_state* s, int64_t* length);

/* Launch shape: ctas = number of CTAs of each step-kernel launch (0
 * restores the default, one full wave at the kernel's occupancy).  Results
 * do not depend on it.  Synchronises the device.  mpadam_launch_info
 * reports the current grid (of the first launch) and threads per CTA. */
int32_t mpadam_set_grid(mpadam_state* s, int32_t ctas);
int32_t mpadam_launch_info(const mpadam_state* s, int32_t* ctas, int32_t* threads);

/* Work balance of mpadam_step's launches.  Each CTA owns an equal run of
 * tiles (3840 elements each).  It keeps the first static_q / 1024 of that
 * run; the rest of every run goes to a pool of chunks of at most
 * chunk_tiles tiles, which the CTAs that finish first claim one at a time.
 * SMs do not all stream memory at the same rate, so without the pool a
 * launch waits on the slowest.  static_q = 1024 turns the pool off.
 * Default: static_q = 768, chunk_tiles = 4, for every weight format, except
 * that until this is called a format group with fewer than 8 tiles per CTA
 * keeps static runs (with a tile or two per CTA the pool's first claimants
 * would take several chunks each).  Results do not depend on any of this.
 * Synchronises the device.  The host-buffer and allocation-free entry
 * points always use static runs.
 * Errors: EINVAL (static_q outside [0, 1024], chunk_tiles outside
 * [1, 2^20]), EALLOC, ECUDA. */
int32_t mpadam_set_tail_pool(mpadam_state* s, int32_t static_q, int32_t chunk_tiles);

/* Device-side status of the steps issued so far: synchronises the device,
 * returns in *code the error bits the step kernel recorded (0 = none; a
 * non-zero value means a bounded wait inside the kernel gave up and that
 * launch's results are incomplete) and clears them.  Errors: EINVAL, ECUDA. */
int32_t mpadam_device_status(mpadam_state* s, int32_t* code);

/* Diagnostics: the random bits the step draws.  Writes into out (device,
 * uint32[n]) the lane of global element indices first, ..., first + n - 1 at
 * step `step` for weight storage `weight_dtype` (16-bit lanes for BF16,
 * 32-bit for the E4M3 formats and NVFP4), on `stream`.  Errors: EINVAL, ECUDA. */
int32_t mpadam_rng_lanes(uint64_t seed, int64_t step, int32_t weight_dtype, int64_t first,
                         int64_t n, uint32_t* out, struct CUstream_st* stream);

/* Allocation-free variant of mpadam_step (the paper has no counterpart: this
 * is a deployment aid).  It is for callers that must not call cudaMalloc --
 * for example a runtime whose device memory all belongs to its own caching
 * allocator or memory pool, or a service that fixes its device-memory budget
 * at start-up and may not allocate afterwards.  It takes the tensor list and
 * config of mpadam_create plus the arguments of mpadam_step, keeps no state
 * object, and calls no cudaMalloc, cudaFree or other allocating routine:
 * the metadata the step kernel reads (tensor descriptors, gradient pointers,
 * per-CTA start tensors) and the kernel's error word live in one file-scope
 * device array of 606,464 bytes that every GPU loading the library holds
 * until the process exits.  Limits: at most 8192 tensors (larger lists: MPADAM_EINVAL; use
 * mpadam_create).  The first call on a device looks up that array's device
 * address (set-up, once per device, with that device current); make that
 * first call before any stream capture.  Every call rewrites the array's
 * tables completely before the step kernel reads them, so calls issued to
 * one stream follow each other safely, but calls that overlap on the GPU
 * (different streams, or several host threads without ordering) race on
 * the shared array.  Results are bit-identical to mpadam_step on the same
 * inputs.  E4M3 weights use the caller's fp8_exp / fp8_amax rings exactly as
 * mpadam_step does (seed them with mpadam_fp8_init or equivalent values).
 * A bounded wait inside the step kernel that gives up (the launch's results
 * are then incomplete) sets a bit in the array's error word, which is not
 * reported by this call's return value: read it with mpadam_noalloc_status.
 * Errors: EINVAL, EUNSUPPORTED, ECUDA. */
int32_t mpadam_step_noalloc(const mpadam_tensor* tensors, int32_t n, const void* const* grads,
                            const mpadam_config* cfg, int32_t* fp8_exp, uint32_t* fp8_amax,
                            int64_t step, struct CUstream_st* stream);

/* Device-side status of the allocation-free steps on the current device
 * (companion of mpadam_step_noalloc; the paper has no counterpart).  Waits
 * for `stream`, returns in *code the error bits the step kernel recorded
 * since the last read (0 = none; non-zero: a bounded wait gave up and that
 * step's results are incomplete), and clears them.  The word is shared by
 * every allocation-free call on the device, like the tables: issue this on
 * the stream the steps went to.  It allocates nothing (the word lives in the
 * same file-scope array).  Errors: EINVAL (code NULL), EUNSUPPORTED, ECUDA. */
int32_t mpadam_noalloc_status(struct CUstream_st* stream, int32_t* code);

/* ------------------------------------------------------------------------
 * BF16-stored matrix-fitting diagnostic (the toy diagnostic of Sec. 5.1 and
 * its appendix): minimise c ||W - W*||_F^4 over W stored in BF16, with the
 * additive, multiplicative or combined step and no moments, to isolate how
 * each update survives BF16 storage.  One step samples `batch` entries
 * uniformly with replacement (sample s takes the 32-bit random lane s of
 * step t: word s mod 4 of Philox4x32-10 block s div 4 with counter (block,
 * t) and key `seed`, masked to the index range); the minibatch loss is
 * c (mean of the sampled squared residuals)^2, the mean a perfect binary
 * tree of binary64 sums over adjacent samples; the gradient of an entry hit
 * k times is its contribution 4 c M r / B added k times (binary32); the
 * entry then becomes bf16(w + w u_m + u_a) (nearest-even; u_a = -eta_a g,
 * u_m = clip(-eta_m ((ln 2) w) g / max(|w|, tau), +-rmax), the additive
 * step alone in mode 0, the multiplicative alone in mode 1).  With split,
 * entries [0, n/2) and [n/2, n) are separate problems (c_lo, c_hi; batch/2
 * samples each; the loss is the sum) -- the mixed-scales regime.
 * ------------------------------------------------------------------------ */
typedef enum { MPADAM_TOY_ADDITIVE = 0, MPADAM_TOY_MULTIPLICATIVE = 1, MPADAM_TOY_COMBINED = 2 } mpadam_toy_mode;

typedef struct {
  int32_t mode;      /* mpadam_toy_mode */
  int32_t split;     /* 0 or 1 */
  int32_t batch;     /* a power of two; 32 to 65536 samples per problem (per half when split) */
  int32_t reserved;  /* must be 0 */
  float lr_add;      /* eta_a (finite, >= 0) */
  float lr_mul;      /* eta_m (finite, >= 0) */
  float rmax;        /* clip of u_m (the paper: 0.75) */
  float tau;         /* floor of rho (the paper: 1e-8), > 0 */
  float c_lo, c_hi;  /* loss constants (c_lo alone when split = 0) */
  uint64_t seed;
} mpadam_toy_config;

typedef struct mpadam_toy_state mpadam_toy_state;

/* Set up the diagnostic for n entries (a power of two, 64 <= n <= 2^30):
 * validates cfg and allocates (and zeroes) two int32[n] scratch arrays and
 * the per-sample buffers, on the current device.  Errors: EINVAL, EALLOC,
 * ECUDA.  On error *out is NULL. */
int32_t mpadam_toy_create(int64_t n, const mpadam_toy_config* cfg, mpadam_toy_state** out);

/* One step t (>= 1) on w (device, n BF16 bit patterns, updated in place)
 * towards wstar (device, n binary32 targets), asynchronously on `stream`.
 * loss_out: device double receiving the minibatch loss of this step (before
 * the update), or NULL.  Three kernel launches.  Errors: EINVAL, ECUDA. */
int32_t mpadam_toy_step(mpadam_toy_state* s, uint16_t* w, const float* wstar, int64_t step, double* loss_out,
                        struct CUstream_st* stream);

/* `steps` consecutive steps first_step, first_step + 1, ... on `stream`, as
 * many mpadam_toy_step calls would give, with the loss of step first_step + i
 * written to losses[i] (device, double[steps]; or NULL).  The step number
 * lives in device memory, advanced by the last kernel of each step, so the
 * steps run as replays of a CUDA graph of 64 steps, captured on an internal
 * stream at the first call with these w, wstar and losses pointers (the
 * remainder runs as plain launches).  Errors: EINVAL, ECUDA. */
int32_t mpadam_toy_run(mpadam_toy_state* s, uint16_t* w, const float* wstar, int64_t first_step, int64_t steps,
                       double* losses, struct CUstream_st* stream);

/* Frees the scratch (synchronises the device first).  NULL is a no-op. */
int32_t mpadam_toy_destroy(mpadam_toy_state* s);

#ifdef __cplusplus
}
#endif
#endif /* MPADAM_H */
