/*
 * lrqat.h -- C ABI of the GB300 (sm_103a) LR-QAT linear layer.
 *
 * LR-QAT (arXiv 2406.06385, Sec. 3) trains a quantized linear layer y = W x,
 * W in R^{m x k}, through the fake-quantized weight of Eq. 8:
 *
 *     W_hat = s * clip(round(phi^{-1}(Phi0) + (alpha/r) A B), n, p),
 *     Phi0  = phi(W0 / s0)                                        (Eq. 6)
 *
 * with [n, p] = [-2^{b-1}, 2^{b-1}-1], a frozen downcast base Phi0, trainable
 * rank-r adapters A [m, r], B [r, k] and a trainable scale s.  Tokens are
 * stacked as rows: Y[T, m] = X[T, k] W_hat^T.
 *
 * Conventions for every call:
 *   - Pointers are DEVICE pointers unless stated otherwise; arrays are dense
 *     row-major; the caller owns every buffer and every buffer must be 16-byte
 *     aligned (TMA).  bf16 tensors are passed as raw bfloat16 bits (uint16_t).
 *   - Calls are asynchronous on `stream` (NULL = legacy default stream) and
 *     allocate no device memory; scratch comes from the caller's workspace.
 *   - Return value: LRQAT_OK or a negative lrqat_status.  Host-side argument
 *     checks run before any CUDA work; the reason of the last failure on the
 *     calling thread is available from lrqat_last_error().  Device-side bounded
 *     waits that give up set a device status word, which
 *     lrqat_get_device_status() reports as LRQAT_ERR_TIMEOUT.
 *   - Rounding is round-half-to-even; the pre-round value
 *     u = phi^{-1}(Phi0) + (alpha/r) A B is formed in fp32.
 *   - Supported shapes: m and k multiples of 128, 1 <= r <= 256 (ranks above
 *     64 with bits <= 7), T >= 1 (any T; ragged token tails are handled),
 *     group_size 0 (per output channel) or a multiple of 128 that divides k.
 *   - W_hat is rebuilt on chip inside the GEMMs and never written.  Where the
 *     low-rank term comes from is a tuning choice (lrqat_set_lowrank_path): for
 *     ranks up to 64 and fewer than 3072 tokens each GEMM stage computes the
 *     low-rank tile (alpha/r) A B next to the main product; otherwise one
 *     tensor-core pass per call first writes one byte per weight into the
 *     workspace, the clipped code c = clip(round(u), n, p) biased by 64 (128 for
 *     8-bit weights) where only the forward and dX GEMMs read it, or the
 *     unclipped round(u) saturated to [-128, 127] (which keeps the clip mask)
 *     where the weight-gradient kernel needs the mask too (ranks above 64); the
 *     GEMMs then turn those bytes into W_hat on chip.  The results are the same
 *     codes, gradients and outputs.
 */
#ifndef LRQAT_H
#define LRQAT_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaStream_t / CUstream. */
typedef struct CUstream_st* lrqat_stream_t;

typedef enum {
  LRQAT_OK = 0,
  LRQAT_ERR_INVALID_ARG = -1, /* null pointer, bad shape, bad bit-width ...          */
  LRQAT_ERR_UNSUPPORTED = -2, /* valid for the method, not implemented (e.g. r > 256) */
  LRQAT_ERR_ALIGNMENT = -3,   /* a pointer is not 16-byte aligned                     */
  LRQAT_ERR_WORKSPACE = -4,   /* workspace missing or smaller than required           */
  LRQAT_ERR_CUDA = -5,        /* a CUDA runtime/driver call or launch failed          */
  LRQAT_ERR_TIMEOUT = -6      /* a kernel's bounded wait gave up (device status)      */
} lrqat_status;

/* Storage format of the frozen base Phi0 (Sec. 3, "Downcasting operator"). */
typedef enum {
  /* Eq. 7, phi = Qb.(8-b): int8 [m, k], value round(2^{8-b} clip(W0/s0, n, p)). */
  LRQAT_PHI_QFIXED = 0,
  /* phi = INT-b, double-packed (b <= 4): uint8 [m, k/2]; byte j of a row holds
   * column 2j in its low nibble and column 2j+1 in its high nibble, each a
   * 4-bit two's complement integer clip(round(W0/s0), n, p). */
  LRQAT_PHI_INT_PACKED = 1,
  /* Sec. 3's floating-point casts: Phi0 = cast(W0/s0) with W0/s0 one fp32 division,
   * round to nearest even, no clipping inside phi; phi^{-1} is the exact value.
   * Stored as bit patterns: uint16 [m, k] for BF16 and FP16, uint8 [m, k] for the
   * OCP FP8 formats (E4M3: bias 7, largest finite 448; E5M2: bias 15, largest
   * finite 57344); FP16 and FP8 casts saturate at the largest finite value.  Symmetric
   * grids only (zero == NULL), 2 <= bits <= 8. */
  LRQAT_PHI_BF16 = 2,
  LRQAT_PHI_FP16 = 3,
  LRQAT_PHI_FP8_E4M3 = 4,
  LRQAT_PHI_FP8_E5M2 = 5
} lrqat_phi_format;

/* Settings of one layer.  W is m x k (m = out features, k = in features). */
typedef struct {
  int64_t m;
  int64_t k;
  int32_t r;          /* adapter rank, 1..256 (above 64: bits <= 7)                 */
  float alpha;        /* adapter scaling: (alpha / r) A B enters Eq. 8              */
  int32_t bits;       /* b: 2..7 for QFIXED, 2..4 for INT_PACKED, 2..8 for the casts */
  int32_t group_size; /* 0: one scale per output row (pc); else scales per g-wide
                         group along k (g128 = 128), s has shape [m, k/g]           */
  int32_t phi_format; /* lrqat_phi_format                                           */
  int32_t act_bits;   /* 0: activations unquantized; 8: per-tensor symmetric int8
                         X_hat = s_x clip(round(X/s_x), -128, 127) (Sec. 4,
                         weight-activation quantization; Eq. 1 with z = 0)          */
  float* zero;        /* NULL: symmetric weight grid (Eq. 8 as written).  Otherwise
                         asymmetric weights with a frozen zero offset (Eq. 1 with z
                         outside the rounding, end of Sec. 3; the INT2 runs of Sec. 4):
                         a device array shaped like s, 16-byte aligned, holding the
                         integer offsets z as floats.  W_hat = s (W_Z - z) with
                         W_Z = clip(round(phi^{-1}(Phi0) + (alpha/r) A B), n, p), where
                         the stored base Phi0 = phi(W0 / s0 + z0) already carries the
                         offset (z integer: round(x) + z = round(x + z)).
                         lrqat_range_minmax writes z0; every other call reads z.     */
  int32_t act_per_token; /* with act_bits 8: 0 = one static scale s_x for the tensor
                         (passed by the caller); 1 = one dynamic absmax scale per
                         token, s_x[t] = max_j |X[t, j]| / 127 (the default of the
                         weight-activation runs, Sec. 4), computed inside the calls
                         (s_x may then be NULL).  It never clips, so dX
                         has no activation mask; the GEMMs take X_hat =
                         bf16(s_x[t] X_Z) as their token operand.                    */
  int32_t u_bf16;     /* 0: the pre-round value u = phi^{-1}(Phi0) + (alpha/r) A B of
                         Eq. 8 is formed in fp32.  1: in bf16, as Sec. 3 assumes for
                         "the rest of the computation": u = bf16(phi^{-1}(Phi0) +
                         bf16((alpha/r) bf16(A B))) (A B accumulated in fp32 first).
                         Needs alpha/r a power of two (then the product is exact), a
                         base exact in bf16 (not FP16) and zero == NULL
                         (LRQAT_ERR_UNSUPPORTED otherwise).                           */
} lrqat_layer;

/* Human-readable reason of the last non-OK status returned on this thread. */
const char* lrqat_last_error(void);

/* Min-max range setting (App. B, "PTQ initialization").  Symmetric (layer->zero
 * == NULL): s0[i] (or s0[i, g]) = max |W0[i, :]| (over the row or group) / p, fp32;
 * an all-zero row/group gets s0 = 1.  Asymmetric (layer->zero != NULL, written as
 * an output): s0 = (max - min) / (2^b - 1) in fp32 (1 if max == min) and
 * z0 = clip(round(n - min / s0), n, p), min / s0 one fp32 division.
 * W0: fp32 [m, k].  s0: fp32 [m] or [m, k/g] (output). */
int lrqat_range_minmax(const lrqat_layer* layer, const float* W0, float* s0, lrqat_stream_t stream);

/* L^p range setting (App. B, the alternative to min-max; symmetric grids only): per
 * row (or group) the scale minimising sum |w - s clip(round(w/s), n, p)|^p over the
 * candidates s_j = fl32(s_minmax * j / N), j = 1..N, with w/s one fp32 division; the
 * smaller j wins a tie (losses in fp32, so nearly equal candidates may be ordered
 * differently than in exact arithmetic).  p_norm > 0 (the paper uses 2, 2.4, 3,
 * 3.5, 4, 5); 1 <= n_candidates <= 256; the row or group must fit in 200 KB of shared
 * memory.  layer->zero must be NULL (LRQAT_ERR_UNSUPPORTED otherwise).
 * W0: fp32 [m, k].  s0: fp32 [m] or [m, k/g] (output). */
int lrqat_range_lp(const lrqat_layer* layer, const float* W0, float p_norm, int32_t n_candidates, float* s0,
                   lrqat_stream_t stream);

/* Downcasting operator of Eq. 6 / Eq. 7: Phi0 = phi(W0 / s0), with W0 / s0 one
 * fp32 IEEE division per element; with zero offsets phi(W0 / s0 + z0), the
 * integer offset added exactly.
 * W0: fp32 [m, k]; s0: fp32 [m] or [m, k/g];
 * Phi0 (output): int8 [m, k] (QFIXED), uint8 [m, k/2] (INT_PACKED), uint16 [m, k]
 * (BF16, FP16) or uint8 [m, k] (FP8) bit patterns. */
int lrqat_downcast(const lrqat_layer* layer, const float* W0, const float* s0, void* Phi0,
                   lrqat_stream_t stream);

/* Activation fake quantizer of the weight-activation runs (Sec. 4; Eq. 1 with z = 0,
 * b = 8), the step lrqat_linear_fwd / lrqat_linear_bwd run first when act_bits == 8,
 * on its own.  X: bf16 [T, k]; X_out: bf16 [T, k] (output); layer->act_bits must be 8.
 *   act_per_token == 0: X_out = X_Z = clip(round(X / s_x), -128, 127) as exact bf16
 *     codes, X / s_x one fp32 division, s_x a device scalar (required); mask
 *     (nullable): uint32 [k, ceil(T/32)], bit t % 32 of word [j, t / 32] is
 *     M_x = 1[-128 <= round(X[t, j] / s_x) <= 127];
 *   act_per_token == 1: s_x[t] = max_j |X[t, j]| / 127 in fp32 (1 for an all-zero
 *     token), X_out = bf16(s_x[t] X_Z); s_x and mask are not used (NULL allowed).
 * X and X_out 16-byte aligned; mask 4-byte aligned. */
int lrqat_act_quant(const lrqat_layer* layer, int64_t T, const uint16_t* X, const float* s_x, uint16_t* X_out,
                    uint32_t* mask, lrqat_stream_t stream);

/* Bytes of workspace lrqat_linear_fwd needs for T tokens (padded adapter
 * copies; int8 activation codes when act_bits == 8; the m x k int8 codes of the
 * weights for the codes path of lrqat_set_lowrank_path).  The size covers every
 * setting of lrqat_set_lowrank_path. */
size_t lrqat_fwd_workspace_bytes(const lrqat_layer* layer, int64_t T);

/* Forward of the LR-QAT layer (Eq. 8 inside y = W_hat x):
 *   Y = X_hat W_hat^T,  X_hat = X (act_bits 0) or s_x clip(round(X/s_x)) (act_bits 8).
 * W_hat is rebuilt tile by tile inside the GEMM and never written to memory.
 * X: bf16 [T, k]; Phi0 as produced by lrqat_downcast; s: fp32 [m] or [m, k/g];
 * A: bf16 [m, r]; B: bf16 [r, k]; s_x: device fp32 scalar (required iff
 * act_bits == 8, else may be NULL); Y (output): bf16 [T, m].
 * workspace: device buffer of at least lrqat_fwd_workspace_bytes() bytes. */
int lrqat_linear_fwd(const lrqat_layer* layer, int64_t T, const uint16_t* X, const void* Phi0,
                     const float* s, const uint16_t* A, const uint16_t* B, const float* s_x,
                     uint16_t* Y, void* workspace, size_t workspace_bytes, lrqat_stream_t stream);

/* Allocation-free forward (no counterpart in the paper: this is a deployment
 * convenience).  Same computation and arguments as lrqat_linear_fwd, but the
 * scratch comes from a fixed array inside the library instead of a caller
 * workspace, for callers that cannot allocate device memory: runtimes that own
 * all device memory and hand an operator only its inputs and outputs, or that
 * forbid allocation after start-up because cudaMalloc can synchronize the
 * device and stall other work.
 *   - The array holds LRQAT_FWD_NOALLOC_SCRATCH_BYTES bytes; every device that
 *     loads the library keeps it until the process exits.  A layer/T whose
 *     scratch exceeds it is rejected with LRQAT_ERR_WORKSPACE (in practice:
 *     act_bits = 8 with large T * k, or a rank above 64 with a large m * k).
 *     For ranks up to 64 this forward always computes the low-rank tile inside
 *     the GEMM (lrqat_set_lowrank_path 1), so its scratch holds no weight codes.
 *   - The first call on a device looks the array's device address up (with
 *     that device current); make that first call before any stream capture.
 *   - All calls share the one array: calls that overlap on the GPU (different
 *     streams, or host threads without ordering) race; serialize them.
 *   - Every call rewrites the parts of the scratch it reads, so nothing has to
 *     be cleared between calls.  No device memory is allocated or freed. */
#define LRQAT_FWD_NOALLOC_SCRATCH_BYTES ((size_t)4 << 20)
int lrqat_linear_fwd_noalloc(const lrqat_layer* layer, int64_t T, const uint16_t* X, const void* Phi0,
                             const float* s, const uint16_t* A, const uint16_t* B, const float* s_x,
                             uint16_t* Y, lrqat_stream_t stream);

/* Bytes of workspace lrqat_linear_bwd needs for T tokens (covers every setting of
 * lrqat_set_lowrank_path). */
size_t lrqat_bwd_workspace_bytes(const lrqat_layer* layer, int64_t T);

/* Backward of the LR-QAT layer for the upstream gradient dY, with W_hat
 * recomputed rather than stored (the checkpointing of Sec. 3) and the
 * straight-through estimator for round() (Eq. 3/4 text).  With G = dY^T X_hat,
 * u, c = clip(round(u), n, p) and M = 1[n <= round(u) <= p]:
 *   dX = (dY W_hat) * M_x          (M_x: activation clip mask, ones if act_bits 0)
 *   dA = (alpha/r) (G * s * M) B^T,  dB = (alpha/r) A^T (G * s * M)
 *   ds = sum over the row (or group) of G * c
 * dY: bf16 [T, m]; X, Phi0, s, A, B, s_x as in lrqat_linear_fwd;
 * dX (output): bf16 [T, k]; dA: fp32 [m, r]; dB: fp32 [r, k]; ds: fp32 like s.
 * accumulate = 0 overwrites dA, dB, ds; 1 adds to them (gradient accumulation
 * over micro-batches).  dX is always overwritten.
 * workspace: device buffer of at least lrqat_bwd_workspace_bytes() bytes.
 * The weight-gradient work is spread over the SMs either as equal token splits of
 * every tile or as whole tiles followed by the remaining tiles cut into token
 * parts, one per SM, chosen per call unless lrqat_set_dw_schedule forces one.  Both
 * give the same dX bit for bit and the same dA, dB, ds up to rounding order. */
int lrqat_linear_bwd(const lrqat_layer* layer, int64_t T, const uint16_t* dY, const uint16_t* X,
                     const void* Phi0, const float* s, const uint16_t* A, const uint16_t* B,
                     const float* s_x, uint16_t* dX, float* dA, float* dB, float* ds, int accumulate,
                     void* workspace, size_t workspace_bytes, lrqat_stream_t stream);

/* Forward and backward on activations the caller has already quantized with
 * lrqat_act_quant (act_bits == 8 only), so that each input is quantized once per
 * training step rather than once in the forward and again in the backward (a
 * deployment convenience; the paper's computation is unchanged):
 *   X_q: bf16 [T, k], the X_out of lrqat_act_quant for this X and layer (per tensor:
 *     the codes X_Z; per token: X_hat = bf16(s_x[t] X_Z));
 *   mask (backward): the clip mask lrqat_act_quant wrote for this X, uint32
 *     [k, ceil(T/32)], 4-byte aligned; required per tensor, not used per token (NULL
 *     allowed);
 *   every other argument as in lrqat_linear_fwd / lrqat_linear_bwd, s_x included (the
 *     per-tensor scale the codes were made with).
 * The results equal those of lrqat_linear_fwd / lrqat_linear_bwd on X bit for bit (the
 * same kernels read the same operands); no quantizer runs.  The workspace sizes of
 * lrqat_fwd_workspace_bytes / lrqat_bwd_workspace_bytes suffice.  Errors as there, and
 * LRQAT_ERR_INVALID_ARG when act_bits != 8 or a per-tensor mask is NULL. */
int lrqat_linear_fwd_quantized(const lrqat_layer* layer, int64_t T, const uint16_t* X_q, const void* Phi0,
                               const float* s, const uint16_t* A, const uint16_t* B, const float* s_x,
                               uint16_t* Y, void* workspace, size_t workspace_bytes, lrqat_stream_t stream);
int lrqat_linear_bwd_quantized(const lrqat_layer* layer, int64_t T, const uint16_t* dY, const uint16_t* X_q,
                               const uint32_t* mask, const void* Phi0, const float* s, const uint16_t* A,
                               const uint16_t* B, const float* s_x, uint16_t* dX, float* dA, float* dB,
                               float* ds, int accumulate, void* workspace, size_t workspace_bytes,
                               lrqat_stream_t stream);

/* Fold the adapters into the final integer weight (Sec. 3, after Eq. 8):
 *   W_Z = clip(round(phi^{-1}(Phi0) + (alpha/r) A B), n, p),  so W_hat = s W_Z.
 * W_Z (output): int8 [m, k] with values in [n, p]. */
int lrqat_merge(const lrqat_layer* layer, const void* Phi0, const uint16_t* A, const uint16_t* B,
                int8_t* W_Z, lrqat_stream_t stream);

/* ---- Optimizer step on A, B, s (App. B, Table B1) ------------------------------
 * AdamW with decoupled weight decay, bias-corrected moments, separate learning rates
 * for the adapters and the scales, after clipping the global L2 norm of all
 * trainable gradients (every layer's dA, dB, ds) with the coefficient
 * min(1, max_grad_norm / (norm + 1e-6)).  Zero offsets stay frozen (Sec. 4). */
typedef struct {
  float lr_ab;           /* learning rate of A and B for this step (schedules are the caller's) */
  float lr_s;            /* learning rate of s (0 freezes the scales, s = s0)                  */
  float beta1, beta2;    /* (0.9, 0.95)                                                      */
  float eps;             /* 1e-8                                                             */
  float weight_decay_ab; /* 0                                                                */
  float weight_decay_s;  /* 0                                                                */
  float max_grad_norm;   /* 1.0; <= 0 disables clipping                                      */
  int32_t step;          /* 1, 2, ...: bias correction 1 - beta^step                         */
} lrqat_adamw;

/* Optimizer state of one layer: device arrays owned by the caller, the moments zeroed
 * and the master copies initialised from A and B before the first step.
 * A32 [m, r] and B32 [r, k] fp32 master copies; first/second moments shaped like
 * A, B and s.  All 16-byte aligned. */
typedef struct {
  float* A32;
  float* B32;
  float* mA;
  float* vA;
  float* mB;
  float* vB;
  float* ms;
  float* vs;
} lrqat_adamw_state;

/* Adds the squared L2 norm of one layer's gradients dA [m, r], dB [r, k] and ds
 * (shaped like s) to *sqnorm, a device fp32 scalar the caller zeroes once per step.
 * Deterministic: a fixed summation order within the layer; layers add in stream
 * order. */
int lrqat_grad_sqnorm(const lrqat_layer* layer, const float* dA, const float* dB, const float* ds, float* sqnorm,
                      lrqat_stream_t stream);

/* One clipped AdamW step on a layer's A, B (fp32 masters in `state`; the bf16 copies
 * A [m, r], B [r, k] are rewritten for the next forward) and s, with the step's global
 * squared gradient norm *sqnorm (after every layer's lrqat_grad_sqnorm). */
int lrqat_adamw_step(const lrqat_layer* layer, const lrqat_adamw* opt, const float* sqnorm, const float* dA,
                     const float* dB, const float* ds, const lrqat_adamw_state* state, float* s, uint16_t* A,
                     uint16_t* B, lrqat_stream_t stream);

/* Tuning (no counterpart in the paper): the schedule of the weight-gradient work of
 * lrqat_linear_bwd.  0 = chosen per call by a cost model (the default), 1 = equal token
 * splits of every tile, 2 = whole tiles followed by the remaining tiles cut into token
 * parts (falls back to 1 when every SM gets the same number of whole tiles).  The
 * setting is process-wide and changes the size lrqat_bwd_workspace_bytes reports, so
 * set it before querying sizes and keep it while those workspaces are in use.  The
 * environment variable LRQAT_DW_SCHEDULE ("split" or "tail") gives the start value; it
 * is read once, when the library is loaded.  Returns LRQAT_ERR_INVALID_ARG for other
 * values. */
int lrqat_set_dw_schedule(int schedule);

/* Tuning (no counterpart in the paper): the kernels of the forward, dX and dW GEMMs.
 * CTA pairs run tcgen05 MMAs of 256 rows across the two SMs of a cluster, each SM holding
 * half of the token operand (256 weight rows x 448 tokens per pair); they need a multiple
 * of 256 produced rows (m for the forward, k for dX; dW: ranks up to 64 and m, k multiples
 * of 256, on 256 x 256 tiles).  The one-SM kernels take 128 rows per SM.  0 (the default) =
 * pairs wherever they were measured faster, which is wherever the shapes allow; 1 = the
 * one-SM kernels always; 2 = pairs wherever the shapes allow.  All give the same codes;
 * outputs agree up to fp32 summation order.  Process-wide; the environment variable LRQAT_GEMM_VARIANT ("auto",
 * "single" or "pair") gives the start value, read once when the library is loaded.
 * Returns LRQAT_ERR_INVALID_ARG for other values. */
int lrqat_set_gemm_variant(int variant);

/* Tuning (no counterpart in the paper): where the forward and dX GEMMs take the low-rank
 * term (alpha/r) A B of Eq. 8 from.  1 = "tile": each GEMM stage computes the 64-column
 * low-rank tile of its weight rows on the tensor cores next to the main product (ranks up
 * to 64); 2 = "codes": one tensor-core pass per call writes the code of every weight as one
 * byte (clip(round(u), n, p) + 64, or + 128 for 8-bit weights) into the workspace and the
 * GEMMs read those bytes as their base, with no low-rank work in the stage; 0 (the default)
 * = codes from 3072 tokens
 * on, the tile below (the pass costs two bytes of HBM traffic per weight, the tile a low-rank
 * MMA chain per stage).  Ranks above 64 always take the codes pass.  dW is unaffected: it
 * computes its own low-rank tile for ranks up to 64.  All settings give the same codes up to
 * fp32 summation order of A B.  Process-wide; the environment variable LRQAT_LOWRANK_PATH
 * ("auto", "tile" or "codes") gives the start value, read once when the library is loaded.
 * Returns LRQAT_ERR_INVALID_ARG for other values. */
int lrqat_set_lowrank_path(int path);

/* The current settings of lrqat_set_gemm_variant, lrqat_set_dw_schedule and
 * lrqat_set_lowrank_path. */
int lrqat_get_gemm_variant(void);
int lrqat_get_dw_schedule(void);
int lrqat_get_lowrank_path(void);

/* Synchronizes `stream`, then reads and clears the device status word of the
 * current device.  Returns LRQAT_OK, LRQAT_ERR_TIMEOUT (a kernel's bounded
 * wait gave up since the last call) or LRQAT_ERR_CUDA. */
int lrqat_get_device_status(lrqat_stream_t stream);

/* ---------------------------------------------------------------------------
 * Tracing (instrumentation; not part of the method).  While enabled, every
 * kernel the library enqueues is bracketed by a pair of CUDA events recorded on
 * the stream it runs on, and counted per kernel name.  Tracing is off by
 * default and costs nothing then.
 * ------------------------------------------------------------------------- */
/* enable = 1 starts (and clears) a trace, 0 stops recording. */
int lrqat_trace_enable(int enable);
/* Synchronizes the recorded events and reports up to `max_entries` kernels:
 * names[i] (static strings), launches[i] and total device milliseconds[i];
 * *count receives the number of distinct kernels seen.  Host arrays. */
int lrqat_trace_read(int max_entries, const char** names, int64_t* launches, double* total_ms, int* count);

#ifdef __cplusplus
}
#endif

#endif /* LRQAT_H */
