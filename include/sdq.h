/*
 * sdq.h -- C ABI of the GB300 (sm_103a) Sigma-Delta-quantized linear layer.
 *
 * SDQ-LLM (arXiv 2510.03275) stores each linear layer's weights as
 * Sigma-Delta codes of the Hadamard-smoothed, OSR-times upsampled weight rows
 * (section 3, Algorithm 1).  This library implements, on one GPU:
 *
 *   sdq_encode_rows      Algorithm 1 (SDQuant + Resample) per output row:
 *                        randomised Hadamard smoothing (eq. 13), band-limited
 *                        upsampling, per-row scale, first-order Sigma-Delta
 *                        scan (eqs. 7-8) with the binary (eqs. 3-4) or ternary
 *                        (eqs. 5-6) quantizer, blocks independent.
 *   sdq_encode_rows_gptq the same with Algorithm 1's GPTQ block compensation
 *                        (inverse-Hessian update of the later columns).
 *   sdq_pack/sdq_unpack  plain <-> tiled code layouts (bit-exact).
 *   sdq_pack_base3 /     plain <-> base-3 storage of ternary codes (5 trits
 *   sdq_unpack_base3     per byte, 1.6 bits per code; eq. 14).
 *   sdq_prep_activations x_tilde = G x per block of B inputs, G = D^T Had^T:
 *                        the exact adjoint of the decimation and Hadamard
 *                        reconstruction, i.e. the activation upsampling of
 *                        section 3.5 (Fig. 5) that makes the inner product of
 *                        eq. (12) equal x . W_hat^T.
 *   sdq_contract         y[m,r] = alpha_r * sum_j c[r,j] x_tilde[m,j]
 *                        (decode path for M <= 64, tensor-core prefill path
 *                        above).
 *   sdq_linear_forward   sdq_prep_activations + sdq_contract.
 *
 * Conventions
 *  - Every entry point returns an int: SDQ_OK (0) or a negative sdq_status.
 *    Nothing throws across the ABI.
 *  - Device pointers are caller-owned device memory; host pointers are
 *    marked "host".  No entry point allocates device memory except
 *    sdq_plan_create (its tables) -- hot calls take a caller workspace.
 *  - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *    stream).  Launches are asynchronous; launch-configuration errors are
 *    reported as SDQ_ERR_CUDA.  A plan is immutable after creation and may be
 *    used from several host threads and streams at once, provided every
 *    concurrent call has its own workspace.
 *  - bf16 activations are passed as their 16-bit patterns (uint16_t).
 *
 * Code values.  Ternary codes are {-1, 0, +1}; binary codes are {-1, +1}.
 * The real weight block the codes stand for is
 *   W_hat[r, bB:(b+1)B] = alpha_r * Resample(c[r, b*n_b:(b+1)*n_b], B) . Had^T
 * with Had = diag(d) . H_B / sqrt(B) (H_B Sylvester, d the sign vector given
 * to sdq_plan_create) and Resample the FFT resampler of Algorithm 1.
 *
 * Plain layout (canonical; output of sdq_encode_rows): b bits per code
 * (b = 2 ternary, 1 binary).  Row r occupies words_per_row =
 * 4 * ceil(K_eff * b / 128) uint32 words starting at word r * words_per_row;
 * code j of the row sits at bit b * (j % (32/b)) of word j / (32/b).
 * Ternary fields: 00 = 0, 01 = +1, 11 = -1 (10 is invalid).  Binary: 1 = +1,
 * 0 = -1.  Padding bits are 0.
 *
 * Invalid codes.  The ternary pattern 10 has no value.  sdq_unpack reports
 * it (SDQ_ERR_BAD_CODE's condition) by adding the number of such fields to a
 * caller-owned device counter rather than through its return value, which
 * would need a device synchronization; the contraction kernels read the
 * pattern as 0.
 *
 * Tiled layout (input of sdq_contract; built by sdq_pack): the library's own
 * format (the paper prescribes no storage order).  K_eff is padded to
 * K_pad = 128 ceil(K_eff / 128) codes; rows are grouped by 128 (row tile T,
 * n_tiles = ceil(n_out / 128)) and codes by 64 (code group G,
 * n_groups = K_pad / 64).  Slab (T, G) holds rows [128T, 128T+128) x codes
 * [64G, 64G+64) in 128 wpg consecutive uint32 words starting at word
 * 128 wpg (T n_groups + G), wpg = 64 b / 32 (4 ternary, 2 binary): row
 * 128T + r owns the wpg words from 128 wpg (T n_groups + G) + wpg r, in
 * which its 64 codes sit in natural order with the plain layout's bit map
 * (code 64G + kk at bit b (kk % (32/b)) of word kk / (32/b)).  So every row
 * keeps a 16-byte (ternary) or 8-byte (binary) run of its plain words per
 * group, and the tile's slabs of consecutive groups are contiguous in
 * memory: one bulk copy streams a 128-row x (64 n)-code stage.  Codes past
 * n_out or K_eff are padding with field value 0.
 */
#ifndef SDQ_H_
#define SDQ_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  SDQ_OK = 0,
  SDQ_ERR_INVALID_ARG = -1,  /* bad descriptor, size, null or misaligned pointer */
  SDQ_ERR_UNSUPPORTED = -2,  /* valid but not implemented (e.g. device not sm_103) */
  SDQ_ERR_WORKSPACE = -3,    /* workspace smaller than sdq_workspace_bytes() */
  SDQ_ERR_CUDA = -4,         /* a CUDA runtime call or launch failed */
  SDQ_ERR_TIMEOUT = -5,      /* a bounded device-side wait gave up */
  SDQ_ERR_BAD_CODE = -6,     /* invalid ternary pattern 10 found */
  SDQ_ERR_ALLOC = -7         /* host or device allocation failed in plan creation */
} sdq_status;

typedef enum { SDQ_BINARY = 1, SDQ_TERNARY = 2 } sdq_quantizer; /* value = bits per code */
typedef enum { SDQ_ALPHA_MAXABS = 0, SDQ_ALPHA_MEANABS = 1 } sdq_alpha_mode;

/* One quantized linear layer.  OSR = osr_num / osr_den (section 3.2; a
 * fractional OSR such as 2.5 is allowed) with n_b = block * OSR an integer.
 *   n_out     N, output rows (d_row), 1 .. 2^24
 *   k_in      K, input columns (d_col), a positive multiple of block
 *   block     B, Hadamard / resampling block, a power of two in [2, 1024]
 *   osr_num, osr_den  OSR >= 1, block * osr_num divisible by osr_den,
 *             n_b = block * osr_num / osr_den <= 4096
 *   quantizer SDQ_BINARY or SDQ_TERNARY
 *   hadamard  1: Had = diag(d) H_B / sqrt(B); 0: Had = I
 *   alpha_mode SDQ_ALPHA_MAXABS (max |x_up| over the row, default) or
 *             SDQ_ALPHA_MEANABS (mean |x_up|, section 3.1's "mean(|W|)")
 */
typedef struct {
  int32_t n_out;
  int32_t k_in;
  int32_t block;
  int32_t osr_num;
  int32_t osr_den;
  int32_t quantizer;
  int32_t hadamard;
  int32_t alpha_mode;
} sdq_layer_desc;

typedef struct sdq_plan_s* sdq_plan;

/* Validate `desc`, build the fp64-derived tables (encode table
 * A_enc = fp32(U Had^T), activation table G = D^T Had^T) and upload them to
 * the current device.  `had_signs` (host, `block` entries, each +1 or -1) is
 * the sign vector d of the randomised Hadamard; NULL means all +1.  The plan
 * owns its device tables until sdq_plan_destroy.  Errors: INVALID_ARG,
 * UNSUPPORTED (current device is not compute capability 10.3), ALLOC, CUDA. */
int sdq_plan_create(const sdq_layer_desc* desc, const int8_t* had_signs, sdq_plan* out);
int sdq_plan_destroy(sdq_plan plan);

/* Geometry (host only, no device work).  Return 0 for an invalid descriptor. */
int64_t sdq_k_eff(const sdq_layer_desc* desc);         /* K * OSR */
size_t sdq_plain_bytes(const sdq_layer_desc* desc);    /* plain layout size */
size_t sdq_tiled_bytes(const sdq_layer_desc* desc);    /* tiled layout size */
/* Workspace needed by sdq_linear_forward / sdq_prep_activations /
 * sdq_contract at batch M (1 <= M <= 2^20).  0 on invalid input. */
size_t sdq_workspace_bytes(sdq_plan plan, int32_t M);

/* Host-only table builder used by sdq_plan_create, exposed for checking:
 * writes A_enc (n_b x block, row-major, fp32) and G (n_b x block, row-major,
 * fp32) to host buffers (either may be NULL).  Same error codes as
 * sdq_plan_create minus CUDA/UNSUPPORTED. */
int sdq_build_tables(const sdq_layer_desc* desc, const int8_t* had_signs,
                     float* a_enc_host, float* g_host);
/* Host-only: the fp32 G of sdq_encode_rows_gptq's block reconstruction (n_b x
 * block, row-major): the fp64 G rounded to the nearest multiple of 2^-30
 * (ties to even), then to fp32, so that its value does not depend on fp64
 * rounding in entries that result from cancellation.  INVALID_ARG for a NULL
 * g_host or an invalid descriptor. */
int sdq_build_gptq_table(const sdq_layer_desc* desc, const int8_t* had_signs, float* g_host);

/* Host-only (no GPU needed): the launch shape the decode contraction takes
 * at batch M (1..64) on a device with `sm_count` SMs, as sdq_plan_create
 * chooses it.  Writes 16 int64 values to `out_host`: T (e2m1 terms per
 * activation), NP (MMA N), S (k chunks), P (CTAs per chunk), CB (128-code
 * blocks per chunk), ring (stages in the shared-memory ring), sb (blocks per
 * stage), nbuf (accumulators per pipeline), dynamic shared memory bytes,
 * bytes per ring slot, bytes of the chunk-resident B operand image (0 when
 * it streams with the stages), TMEM columns between two blocks' B scales,
 * the kernel's shared-memory limit, MMA pipelines, TMEM A slots, and 1 when
 * each stage's B rows and scale words stream into its ring slot.
 * SDQ_ERR_UNSUPPORTED if no shape fits. */
int sdq_decode_launch_shape(const sdq_layer_desc* desc, int32_t M, int32_t sm_count, int64_t* out_host);

/* Algorithm 1 without compensation, on every row of W (device, fp32,
 * n_out x k_in row-major).  Writes codes in the plain layout
 * (sdq_plain_bytes) and alpha (device, fp32[n_out]).  Bit-exact contract:
 * x_up[j] = fl(...fl(fl(A[j,0] w_0) + fl(A[j,1] w_1))...) in ascending k,
 * i = fl(fl(i + x_up[j]) - y_prev), no FMA contraction; alpha exact max
 * (MAXABS) or fp32 sequential (block, index)-order sum / K_eff (MEANABS);
 * ternary: +1 if i > alpha/2, -1 if i < -alpha/2, else 0; binary: +1 if
 * i >= 0 else -1; y_prev = code * alpha.  Integrator reset every block.
 * Needs no workspace.  Pointers must be 16-byte aligned. */
int sdq_encode_rows(sdq_plan plan, const float* W, uint32_t* codes_plain, float* alpha,
                    void* stream);

/* Bytes of the workspace sdq_encode_rows_gptq needs: a working copy of W
 * (n_out x k_in fp32) and one block's normalised error per row (n_out x B
 * fp32).  0 for a NULL plan. */
size_t sdq_gptq_workspace_bytes(sdq_plan plan);
/* Algorithm 1 WITH its GPTQ block compensation (the outer loop's update of
 * the later columns with the inverse Hessian H^-1 = (2 X X^T + lambda I)^-1
 * of calibration activations X).  U (device, fp32, k_in x k_in row-major):
 * the upper-triangular factor with U^T U = H^-1 (Algorithm 1's
 * Cholesky(H^-1)^T), computed by the caller; only its upper triangle is read.
 * W (device, fp32, n_out x k_in) is not modified: the blocks are encoded in
 * order on a copy in `ws`.  Outputs as sdq_encode_rows.  alpha is taken from
 * the original W (pass 0 of sdq_encode_rows).  Then for every block b of B
 * columns F (later columns R), on the copy: the block's codes c by the same
 * canonical upsample and scan as sdq_encode_rows; s_k = sum_j fl(c_j G[j][k])
 * from +0 in ascending j (G = D^T Had^T in fp32, the reconstruction of the
 * block: Algorithm 1's SDQuant(W Had, OSR) Had^T = alpha c G); E_k =
 * fl(W_k - fl(alpha s_k)); the normalised error E~ = E U_FF^-1 by forward
 * substitution (l ascending: E~_l = fl(t_l / U_ll), then t_k = fl(t_k -
 * fl(E~_l U_lk)) for k > l, t = E at first); and W_R -= E~ U_FR with
 * acc = fl(...fl(fl(E~_0 U_0c) + fl(E~_1 U_1c))...) in ascending k and
 * W = fl(W - acc).  E~ U_FR is the exact block update E H_FR H_RR^-1 (the
 * printed update E H^-1_{F,R} read with GPTQ's normalisation by the factor's
 * diagonal block).  Requires B a multiple of 4; 2 nblk launches on `stream`.
 * Pointers 16-byte aligned; SDQ_ERR_WORKSPACE if ws_bytes is below
 * sdq_gptq_workspace_bytes; SDQ_ERR_UNSUPPORTED for B not a multiple of 4. */
int sdq_encode_rows_gptq(sdq_plan plan, const float* W, const float* U, uint32_t* codes_plain,
                         float* alpha, void* ws, size_t ws_bytes, void* stream);

/* Plain -> tiled (sdq_tiled_bytes).  Input and output must not overlap. */
int sdq_pack(sdq_plan plan, const uint32_t* codes_plain, uint32_t* codes_tiled, void* stream);
/* Tiled -> plain.  If `bad_count` (device, one uint32) is not NULL, the
 * number of invalid ternary fields (pattern 10) seen is ADDED to it; they
 * decode to 0.  The caller reads it after the stream completes and treats a
 * non-zero count as SDQ_ERR_BAD_CODE. */
int sdq_unpack(sdq_plan plan, const uint32_t* codes_tiled, uint32_t* codes_plain,
               uint32_t* bad_count, void* stream);

/* Base-3 storage of ternary codes (eq. 14 counts a ternary code as log2(3) =
 * 1.58 bits; 5 trits per byte store it in 1.6 bits, 80 % of the 2-bit plain
 * layout).  Row r starts at byte r * bpr, bpr = ceil(K_eff / 5) rounded up to
 * a multiple of 16; code j is trit t = code mod 3 (0 -> 0, +1 -> 1, -1 -> 2)
 * at digit j mod 5 of byte j / 5: byte = sum_d t_d 3^d (at most 242); trits
 * past K_eff and padding bytes are 0.  A storage and transfer format: the
 * contraction kernels read the tiled 2-bit layout (sdq_unpack_base3 then
 * sdq_pack rebuilds it).  Ternary plans only.
 * sdq_base3_bytes: n_out * bpr, host only; 0 for a binary or invalid
 * descriptor. */
size_t sdq_base3_bytes(const sdq_layer_desc* desc);
/* Plain (2-bit) -> base-3 (sdq_base3_bytes).  The invalid pattern 10 is
 * stored as 0.  Both pointers 16-byte aligned; SDQ_ERR_UNSUPPORTED for a
 * binary plan. */
int sdq_pack_base3(sdq_plan plan, const uint32_t* codes_plain, uint8_t* codes_base3, void* stream);
/* Base-3 -> plain (2-bit, padding 0).  A byte above 242 has no 5-trit
 * reading: it decodes as five 0 codes and, if `bad_count` (device, one
 * uint32) is not NULL, is ADDED to it (read it after the stream completes; a
 * non-zero count is SDQ_ERR_BAD_CODE's condition).  Both pointers 16-byte
 * aligned; SDQ_ERR_UNSUPPORTED for a binary plan. */
int sdq_unpack_base3(sdq_plan plan, const uint8_t* codes_base3, uint32_t* codes_plain, uint32_t* bad_count,
                     void* stream);

/* x_tilde = G x_b for every block b of every row of x (device, bf16 bits,
 * M x k_in row-major), written into the workspace `ws` for sdq_contract.
 * M <= 64: x_tilde is written in fp32 (M x K_pad, K_pad = 128
 * ceil(K_eff / 128), padding 0); the decode kernel forms its tensor-core B
 * operand from it.  M > 64: x_tilde is written in bf16 in the permuted K
 * order the prefill kernel reads.  Kernels are launched with programmatic
 * dependent launch.  Errors: INVALID_ARG (also when the current device is
 * not the plan's), WORKSPACE, CUDA. */
int sdq_prep_activations(sdq_plan plan, const uint16_t* x, int32_t M,
                         void* ws, size_t ws_bytes, void* stream);

/* Contraction against the tiled codes: y (device, fp32, M x n_out row-major)
 * = alpha_r * sum_j c[r,j] x_tilde[m,j], reading the x_tilde that
 * sdq_prep_activations left in `ws` for the same M.  M <= 64: decode kernel
 * (tcgen05 block-scaled 4-bit MMAs, kind::mxf4: the codes expanded into
 * tensor memory as e2m1 +-2 / 0, the activations as T e2m1 terms per batch
 * row with one power-of-two scale per 32 codes and term, x_tilde =
 * sum_t 2^(e_g - 3t) q_t, T = 6 for M <= 4, 4 up to 16, 3 above; the prepare
 * kernel writes these terms for all of K when n_b is a multiple of 64, else
 * each thread block forms those of its k chunk from x_tilde; split-K over
 * thread blocks with a deterministic last-block reduction: results are
 * bit-for-bit reproducible for a given plan, M and device; the launch shape
 * is chosen per batch size at plan creation and can be queried with
 * sdq_decode_launch_shape).  M > 64: tcgen05 bf16 prefill kernel.  Errors as
 * sdq_prep_activations, and UNSUPPORTED when no launch shape fits. */
int sdq_contract(sdq_plan plan, const uint32_t* codes_tiled, const float* alpha, int32_t M,
                 float* y, void* ws, size_t ws_bytes, void* stream);

/* y += the contraction above (M <= 64 only; UNSUPPORTED above): every
 * thread block adds its k chunk's share into y with float reductions, so y
 * must hold valid values (e.g. a residual stream the layer's output is added
 * to, or zeros).  The order of the additions is not fixed: results may
 * differ from run to run in the last bits.  Same inputs and errors as
 * sdq_contract otherwise. */
int sdq_contract_add(sdq_plan plan, const uint32_t* codes_tiled, const float* alpha, int32_t M,
                     float* y, void* ws, size_t ws_bytes, void* stream);

/* y = the layer applied to x: same inputs, outputs and errors as
 * sdq_prep_activations followed by sdq_contract, as two kernels.  For decode
 * batches (M <= 64) whose launch shape splits K over thread blocks, the
 * prepare kernel also clears y and the contraction adds its k chunks' shares
 * into it with float reductions (as sdq_contract_add): results agree with
 * sdq_contract to within the order of those additions, not bit for bit.
 * The contraction may start streaming the codes before the prepare kernel
 * completes (it reads nothing the prepare kernel writes until then).  Large
 * batches take the dense route where sdq_forward_route says 3: the weights
 * are rebuilt into the workspace (sdq_workspace_bytes includes n_out x k_in
 * bf16 for those batch sizes), then multiplied by x in one GEMM. */
int sdq_linear_forward(sdq_plan plan, const uint32_t* codes_tiled, const float* alpha,
                       const uint16_t* x, int32_t M, float* y, void* ws, size_t ws_bytes,
                       void* stream);

/* Kernels sdq_linear_forward launches for this plan, batch M and
 * activation pointer x: 2 (the prepare kernel, then the contraction; or, on
 * the dense route, the weight rebuild, then the dense GEMM).  0 on invalid
 * input.  Host only. */
int sdq_forward_kernels(sdq_plan plan, int32_t M, const uint16_t* x);

/* The route sdq_linear_forward takes for this plan and batch M: 1 decode
 * (M <= 64: prepare kernel, tcgen05 block-scaled 4-bit contraction); 2
 * prefill in the code domain (x_tilde = G x in bf16, tcgen05 bf16
 * contraction with the codes); 3 dense (M >= 768 where the plan allows it:
 * B = 128, n_b a multiple of 64 up to 384: the kernel rebuilds the weights
 * W' = 2 C G per block in bf16 into the workspace, then y = alpha / 2 x W'^T
 * as one bf16 GEMM with fp32 accumulation, the same result as route 2 up to
 * the bf16 rounding of W' in place of x_tilde's).  0 on invalid input.
 * Host only. */
int sdq_forward_route(sdq_plan plan, int32_t M);

/* Wait for `stream`, then report whether the last contraction that used
 * `ws` (same plan and M) completed its bounded device-side waits: SDQ_OK or
 * SDQ_ERR_TIMEOUT (a copy or an MMA did not complete within about 2 s; the
 * output of that call is invalid).  Covers the decode (M <= 64) and the
 * prefill (M > 64) kernels.  Workspace contents never need resetting: the
 * split-K tickets and this record carry a 48-bit tag per call (bit 47 set,
 * the other 47 bits a bijective scramble of a process-wide call counter),
 * so zeros, another call's tickets and structured leftovers of another plan
 * or batch size (counters, small floats) do not count (an arbitrary 64-bit
 * word matches a given call's tag with probability 2^-47), and the last
 * arrival at a ticket clears it.  One workspace may serve several plans in
 * turn (never two calls at once). */
int sdq_workspace_status(sdq_plan plan, int32_t M, const void* ws, void* stream);

/* Copy x_tilde for M <= 64 out of the workspace as fp32 (M x K_eff,
 * device), for checking sdq_prep_activations. */
int sdq_read_prep(sdq_plan plan, int32_t M, const void* ws, float* xt_out, void* stream);

/* Allocation-free decode forward, for callers that may not allocate device
 * memory or pass a workspace (for example a plugin whose host runtime owns
 * every device allocation, or a serving loop that forbids allocation after
 * start-up).  No counterpart in the paper: it is a packaging of
 * sdq_linear_forward.  Same inputs and outputs as sdq_linear_forward, but
 * the scratch is a library-owned device array of sdq_noalloc_scratch_bytes()
 * (16 MiB) per GPU, reserved when the library loads and held until the
 * process exits.  No cudaMalloc / cudaFree / allocating call is made.
 *   - M must be 1..64 (the decode path), and sdq_workspace_bytes(plan, M)
 *     must not exceed the array: otherwise SDQ_ERR_INVALID_ARG or
 *     SDQ_ERR_WORKSPACE is returned and nothing is launched.
 *   - The current device must be the plan's (else SDQ_ERR_INVALID_ARG): the
 *     array of the current device is used.
 *   - The first call on a device looks up the array's device address
 *     (cudaGetSymbolAddress, with that device current); make that first call
 *     before any stream capture.  The address is cached per device for the
 *     life of the process: after cudaDeviceReset the cached address is stale,
 *     so do not use this entry point after resetting a device.
 *   - All calls on a device share the array and it keeps the last call's
 *     contents, none of which needs resetting (see sdq_workspace_status).
 *     Calls that overlap on the GPU (other streams or host threads) race on
 *     the array: serialize them.
 *   - sdq_noalloc_status reports the bounded-wait outcome of the last call. */
int sdq_linear_forward_noalloc(sdq_plan plan, const uint32_t* codes_tiled, const float* alpha,
                               const uint16_t* x, int32_t M, float* y, void* stream);
size_t sdq_noalloc_scratch_bytes(void);
/* Wait for `stream`, then report whether the last sdq_linear_forward_noalloc
 * call on the current device with this plan and M completed its bounded
 * device-side waits: SDQ_OK or SDQ_ERR_TIMEOUT (that call's output is
 * invalid), as sdq_workspace_status does for a caller workspace.  Host only;
 * reads the call record inside the library's array.  Errors: INVALID_ARG
 * (also when the current device is not the plan's), WORKSPACE (no call of
 * this size can have run), CUDA. */
int sdq_noalloc_status(sdq_plan plan, int32_t M, void* stream);

/* Static string for a status code. */
const char* sdq_status_string(int status);

#ifdef __cplusplus
}
#endif
#endif /* SDQ_H_ */
