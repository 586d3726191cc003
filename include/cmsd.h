/*
 * cmsd.h -- C ABI of libcmsd.so, the GB300 (sm_103a) logits pass of
 * confidence-modulated speculative decoding (CM-ASD; Sen, Dasgupta, Waghela,
 * arXiv 2508.15371).
 *
 * One decoding iteration of CM-ASD looks at vocabulary-wide logits of the
 * drafted window: per drafted position it derives the drafter's confidence
 * (Sec. III.B(1)), from the window mean the next draft length (Sec. III.B(b)),
 * and per position a confidence-modulated acceptance test against the
 * verifier (Sec. III.B(c)); verification stops at the first failure
 * (Sec. III.A(2)) and the failing position receives a correction token.
 *
 * Conventions shared by every entry point
 *   - Logit tensors are row-major, contiguous [B][K][V] (sequence b, drafted
 *     position i, vocabulary entry v), in the dtype given (cmsd_dtype), on the
 *     current CUDA device, 16-byte aligned base address.  Other [B][K] and [B]
 *     arrays are contiguous device arrays.  The caller owns all memory.
 *   - k_row (nullable, int32 [B], device): number of drafted positions present
 *     in sequence b (0 <= k_row[b] <= K); NULL means K everywhere.  Positions
 *     i >= k_row[b] are not read and their per-position outputs are left
 *     untouched.
 *   - Every call is asynchronous on `stream` (a cudaStream_t; NULL = the legacy
 *     default stream), allocates nothing and synchronises nothing.  Scratch
 *     lives in the caller's workspace (cmsd_workspace_bytes); calls that share
 *     one workspace must be ordered on one stream.
 *   - Return value: CMSD_OK, or a negative cmsd_status.  Argument errors are
 *     detected on the host before anything is enqueued.  Errors that only the
 *     device can see (a drafted token outside [0, V), k_row outside [0, K]) are
 *     clamped before any load and recorded in the workspace;
 *     cmsd_workspace_errors reads them.
 *   - Calls that draw a residual token (CMSD_RULE_SAMPLED) or use the bonus row
 *     launch a second kernel after the streaming kernel, on the same stream,
 *     which makes a second pass over one row of each sequence that needs it.
 *   - Logits must be finite or -inf (masked vocabulary entries, probability 0);
 *     |logit| < 1e29; every row needs at least one finite logit.  +inf and NaN
 *     give unspecified results.
 *   - Limits: 2 <= V < 2^31, 1 <= K <= 1024, 0 <= B, B*K*V < 2^46; with k_row,
 *     B <= 12000.  B == 0 or K == 0 is a valid empty call.
 */
#ifndef CMSD_H
#define CMSD_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  CMSD_OK = 0,
  CMSD_EINVAL = -1,     /* bad size, pointer or parameter */
  CMSD_EDTYPE = -2,     /* unknown dtype or rule */
  CMSD_ECUDA = -3,      /* a CUDA runtime call failed (see cmsd_last_cuda_error) */
  CMSD_ENOWS = -4,      /* workspace NULL or smaller than cmsd_workspace_bytes */
  CMSD_EALIGN = -5,     /* logit base pointer not 16-byte aligned */
  CMSD_ESCRATCH = -6    /* problem needs more than CMSD_STATIC_SCRATCH_BYTES of scratch */
} cmsd_status;

typedef enum { CMSD_F32 = 0, CMSD_BF16 = 1 } cmsd_dtype;

typedef enum {
  /* Sec. III.B(c) "modified verification rule": accept iff the draft is in the
   * verifier's top-beta (fewer than beta_rank logits strictly above it) and
   * log P(y1) - log P(draft) <= tau_t; the correction is the verifier argmax. */
  CMSD_RULE_PAPER = 0,
  /* Speculative sampling (the works cited in Sec. II, [5] and [6]) with the
   * same confidence-modulated slack: accept iff u * q(draft) < e^tau_t *
   * p(draft), u a Philox uniform; the correction is drawn from the normalised
   * residual max(0, p - q).  With tau_t = 0 and no rank gate the emitted token
   * has exactly the verifier's distribution. */
  CMSD_RULE_SAMPLED = 1
} cmsd_rule;

/* Hyper-parameters, the inputs of Algorithm 1 (Sec. III.B). */
typedef struct {
  int32_t k_min, k_max;   /* draft-length bounds, 1 <= k_min <= k_max (Sec. III.B(b)) */
  float   lambda[3];      /* ensemble weights (entropy, logit margin, softmax margin),
                             each in [0,1], summing to 1 within 1e-5 (Sec. III.B(1)) */
  float   beta_sig;       /* sigmoid sharpness of the logit margin, > 0 */
  int32_t beta_rank;      /* top-beta inclusion; 0 disables the rank gate */
  float   alpha;          /* aggressiveness in (0, 1] (Sec. III.B(b)) */
  float   tau_base;       /* base tolerance, e.g. 0.1 (Sec. III.B(c)) */
  float   gamma;          /* confidence gain of the tolerance (Sec. III.B(c)) */
  int32_t tau_sign;       /* +1: tau_t = tau_base + gamma (1 - C_t), the printed
                             equation; -1: tau_base + gamma C_t, the prose reading */
  int32_t rule;           /* cmsd_rule */
  int32_t k_fixed;        /* 0: adaptive draft length; k_min <= k_fixed <= k_max: the
                             next draft length is this constant (the fixed-k variants
                             of the ablation, Sec. IV, Table III) */
  int32_t bonus;          /* 1: the verifier scores one more position than was drafted
                             (Sec. III.A(2): the verifier's own prediction follows the
                             accepted prefix).  target_logits is then [B][K+1][V] (row
                             k_row[b] of sequence b is that extra row) and out_tokens is
                             [B][K+1]; when all k_row[b] drafts are accepted, slot
                             k_row[b] receives the extra row's argmax (PAPER rule) or a
                             draw from its softmax (SAMPLED rule).  Requires V * dtype
                             size to be a multiple of 16 bytes.  0: no extra row. */
} cmsd_params;

/* Defaults: k_min 1, k_max K, lambda 1/3 each, beta_sig 1, beta_rank 3 (PAPER)
 * or 0 (SAMPLED), alpha 1, tau_base 0.1, gamma 1, tau_sign +1, k_fixed 0,
 * bonus 0. */
void cmsd_params_default(cmsd_params* p, int K, int rule);

/* The variants of the ablation (Sec. IV, Table III) as parameter sets:
 * the defaults above, then
 *   FIXED_K       k_fixed = k_max (fixed draft length, adaptive tau)
 *   FIXED_TAU     gamma = 0 (adaptive draft length, fixed tau = tau_base)
 *   FIXED_K_TAU   both (no confidence modulation)
 *   ENTROPY_ONLY, MARGIN_ONLY, SOFTMAX_ONLY   lambda one-hot.
 * Returns CMSD_EINVAL for an unknown preset. */
typedef enum {
  CMSD_PRESET_FULL = 0,
  CMSD_PRESET_FIXED_K = 1,
  CMSD_PRESET_FIXED_TAU = 2,
  CMSD_PRESET_FIXED_K_TAU = 3,
  CMSD_PRESET_ENTROPY_ONLY = 4,
  CMSD_PRESET_MARGIN_ONLY = 5,
  CMSD_PRESET_SOFTMAX_ONLY = 6
} cmsd_preset;
int cmsd_params_preset(cmsd_params* p, int K, int rule, int preset);

/* Bytes of workspace a call with these sizes needs on the current device.
 * The workspace must be zeroed once (cmsd_workspace_init) before first use;
 * every call leaves its counters at zero again. */
size_t cmsd_workspace_bytes(int B, int K, int V);
int cmsd_workspace_init(void* ws, size_t ws_bytes, void* stream);

/* Device-detected errors since the last init/read (bit 0: drafted token out
 * of range, bit 1: k_row out of range, bit 2: the residual draw gave up after
 * waiting one second for a sequence's record, whose correction token then
 * stays -1); clears them.  Synchronises `stream`. */
int cmsd_workspace_errors(void* ws, size_t ws_bytes, void* stream, uint32_t* flags_out);

/* Test support, no counterpart in the paper: launches the sampled rule's
 * residual draw by group bounds alone, after clearing the per-sequence record
 * words that the streaming pass would release.  No record ever appears, so
 * every sequence's bounded wait runs out (about one second) and sets bit 2
 * of the error word; nothing else is written (out_tokens, int32 [B][K],
 * stays as it was).  Arguments as for cmsd_confidence_verify.  Returns
 * CMSD_EDTYPE, launching nothing, where the bounded draw does not take rows
 * of V entries. */
int cmsd_test_record_wait_timeout(const void* draft_logits, const void* target_logits, int B, int K, int V,
                                  int dtype, int32_t* out_tokens, void* ws, size_t ws_bytes, void* stream);

/*
 * Confidence pass (Sec. III.B(1) and (b)) over drafter logits.
 * Per present position (b, i): entropy H = -sum p log p (nats), logit margin
 * z(1) - z(2) (z(2): largest logit at an index other than the argmax), drafter
 * argmax (lowest index among equal maxima), unified confidence
 *   C = clamp(l1 (1 - H/log V) + l2 sigmoid(beta_sig margin)
 *             + l3 (P(1) - P(2)) / (1 - 1/V), 0, 1),
 * and lse = log sum exp of the row.  Per sequence: k_next = min(k_max,
 * max(k_min, floor(alpha * Cbar * k_max))), Cbar the mean C over the present
 * positions (k_next = k_min when k_row[b] == 0).
 * Outputs H, margin, argmax, conf, lse ([B][K]) and k_next ([B]) may be NULL.
 */
int cmsd_confidence(const void* draft_logits, int B, int K, int V, int dtype,
                    const int32_t* k_row, const cmsd_params* p,
                    float* H, float* margin, int32_t* argmax, float* conf, float* lse,
                    int32_t* k_next, void* ws, size_t ws_bytes, void* stream);

/*
 * The drafter's LM head fused with the confidence signals (Sec. I: the
 * estimator is a light layer over the drafter's output logits; Sec.
 * III.B(1): its signals).  For each of R hidden states h (one per drafted
 * row): z = h W^T over the whole vocabulary, then the per-row outputs of
 * cmsd_confidence (H, margin, argmax = the greedy drafted token, conf, lse)
 * from z, without writing z to memory.
 *   hidden: bf16 [R][d] device, row-major; weight: bf16 [V][d] device,
 *     row-major (the [out][in] layout of a linear layer); both 16-byte
 *     aligned; d a multiple of 64, 64 <= d <= 2^20; 2 <= V; R*V < 2^46;
 *     R == 0 is a valid empty call.  Entries must be finite.  Up to 256
 *     hidden rows share one pass over the weight (more take one pass per
 *     256 rows).
 *   z is accumulated in fp32 from exact bf16 products (tensor cores), in an
 *   order that differs from a sequential sum: each logit differs from the
 *   exact dot product by rounding only.
 *   H, margin, argmax, conf, lse: [R] device outputs, each may be NULL.
 *   logits: NULL, or fp32 [R][V] device: z is also written there (for
 *     checking; it costs R*V*4 bytes of writes).
 *   ws: a workspace of at least cmsd_lmhead_workspace_bytes(R, d, V) bytes on
 *     the current device (no initialisation needed; calls that share one
 *     must be ordered on one stream).
 * Two kernels on `stream`: the GEMM with the per-row statistics in its
 * epilogue, then a per-row merge of the statistics of the vocabulary runs.
 */
size_t cmsd_lmhead_workspace_bytes(int R, int d, int V);
int cmsd_lmhead_confidence(const void* hidden, const void* weight, int R, int d, int V,
                           const cmsd_params* p, float* H, float* margin, int32_t* argmax,
                           float* conf, float* lse, float* logits, void* ws, size_t ws_bytes,
                           void* stream);

/*
 * Verification (Sec. III.B(c)) given the confidence of each present position.
 * draft_tokens: int32 [B][K] device, the drafted token of each position.
 * conf: float [B][K] device, C_t (e.g. from cmsd_confidence).
 * draft_lse: float [B][K] device, drafter log-sum-exp; required for
 *   CMSD_RULE_SAMPLED (q(draft) = exp(z_draft - lse)), ignored otherwise.
 * seed, iteration key the Philox4x32-10 uniforms (SAMPLED), key (seed lo,
 *   seed hi), u = (word >> 8) 2^-24: acceptance uniform counter
 *   (0, b, i, iteration<<2 | 0) word 0.  The residual token is drawn by a
 *   two-level exponential race: group g of the 32 entries 32g .. 32g+31 gets
 *   uniform counter (g>>2, b, n, iteration<<2 | 2) word g&3 and the group with
 *   the least -log(1-U_g) / R_g wins (R_g its residual mass); entry v of that
 *   group gets counter (v>>2, b, n, iteration<<2 | 1) word v&3 and the least
 *   -log(1-U_v) / r_v wins.  The token's law is r_v / sum(r).  The bonus token
 *   (SAMPLED rule) is the same race over p of the extra row, with n = k_row[b].
 * Outputs: n_accept [B] (first rejected position, k_row[b] if none);
 *   out_tokens [B][K] ([B][K+1] with the bonus row): accepted drafts, then the
 *   correction at n_accept (when n_accept < k_row[b]) or the bonus token (when
 *   n_accept == k_row[b] and p->bonus), then -1; accept [B][K] (uint8, 0
 *   beyond k_row) may be NULL.
 */
int cmsd_verify(const void* draft_logits, const void* target_logits,
                const int32_t* draft_tokens, const int32_t* k_row,
                int B, int K, int V, int dtype, const cmsd_params* p,
                const float* conf, const float* draft_lse,
                uint64_t seed, uint32_t iteration,
                int32_t* n_accept, int32_t* out_tokens, uint8_t* accept,
                void* ws, size_t ws_bytes, void* stream);

/*
 * The fused pass: cmsd_confidence and cmsd_verify in one streaming read of
 * both logit tensors (plus a second pass over the rejected position of each
 * sequence that needs one -- its target row and the drafter logits of the
 * groups the draw races -- or over the bonus row).  Same arguments
 * and outputs as the two calls above; n_accept and out_tokens are required,
 * the rest may be NULL.
 */
int cmsd_confidence_verify(const void* draft_logits, const void* target_logits,
                           const int32_t* draft_tokens, const int32_t* k_row,
                           int B, int K, int V, int dtype, const cmsd_params* p,
                           uint64_t seed, uint32_t iteration,
                           float* H, float* margin, int32_t* argmax, float* conf, float* lse,
                           int32_t* k_next, int32_t* n_accept, int32_t* out_tokens,
                           uint8_t* accept, void* ws, size_t ws_bytes, void* stream);

/*
 * cmsd_confidence_verify without a workspace argument: the scratch is a fixed
 * array of CMSD_STATIC_SCRATCH_BYTES in the library's device image, one per
 * device.  This entry point has no counterpart in the paper; it exists for
 * callers that may not allocate device memory at call time -- e.g. a serving
 * loop that divides all of HBM once at start-up and treats any later
 * allocation as an error, or a C caller with no device allocator of its own.
 * It allocates nothing.
 *   - Arguments and outputs: as cmsd_confidence_verify, minus ws / ws_bytes.
 *   - Limit: a problem whose cmsd_workspace_bytes(B, K, V) exceeds
 *     CMSD_STATIC_SCRATCH_BYTES (4 MiB; the size does not depend on V, and on
 *     a 152-SM GB300 it admits B*K up to about 40,000 positions, e.g. about
 *     4,900 sequences of K = 8) is rejected with CMSD_ESCRATCH, after the other
 *     argument checks and before anything is enqueued.
 *   - Each call first zero-fills, on `stream`, the part of the scratch that
 *     its layout uses, so device-side error flags (cmsd_workspace_errors) of
 *     an earlier call are not kept; use cmsd_confidence_verify with a caller
 *     workspace to read them.
 *   - One scratch per device: calls whose execution overlaps on one device
 *     (different streams, or host threads without ordering) race on it and
 *     give wrong results.  Order all such calls on one stream.
 *   - The first call on each device does a one-time set-up (it looks up the
 *     scratch's device address, which may load the module); make that first
 *     call before any stream capture begins.
 */
#define CMSD_STATIC_SCRATCH_BYTES (4u << 20)
int cmsd_confidence_verify_static(const void* draft_logits, const void* target_logits,
                                  const int32_t* draft_tokens, const int32_t* k_row,
                                  int B, int K, int V, int dtype, const cmsd_params* p,
                                  uint64_t seed, uint32_t iteration,
                                  float* H, float* margin, int32_t* argmax, float* conf,
                                  float* lse, int32_t* k_next, int32_t* n_accept,
                                  int32_t* out_tokens, uint8_t* accept, void* stream);

/* Host-side Philox4x32-10 (the generator the kernels use), for tests:
 * returns output word `word` (0..3) of counter (c0, c1, c2, c3) under key
 * (seed lo, seed hi).  Runs on the CPU; needs no GPU. */
uint32_t cmsd_philox_u32(uint64_t seed, uint32_t c0, uint32_t c1, uint32_t c2, uint32_t c3,
                         int word);

/* Device Philox: out[j] = word (j & 3) of counter (c0 + (j >> 2), c1, c2, c3),
 * j < n (uint32 device array).  For bit-exactness tests of the device path. */
int cmsd_philox_fill(uint64_t seed, uint32_t c0, uint32_t c1, uint32_t c2, uint32_t c3,
                     uint32_t* out, size_t n, void* stream);

/* Kernel timing: while enabled, each cmsd_confidence / cmsd_verify /
 * cmsd_confidence_verify call records CUDA events on its stream around its
 * streaming kernel and around its resample kernel (sampled rule or bonus
 * row), for up to max_calls calls.  cmsd_profile_stop synchronises those
 * events and writes, per call, the streaming-kernel time and the
 * resample-kernel time in milliseconds (0 when there was none); either array
 * may be NULL; *n_out receives the number of calls recorded.  An event
 * between the two kernels keeps the second from starting during the first's
 * tail, so timed calls run a little slower than untimed ones.
 * Not thread-safe. */
int cmsd_profile_start(int max_calls);
int cmsd_profile_stop(float* stream_ms, float* resample_ms, int max_out, int* n_out);

/* Launch geometry of the streaming kernels on the current device:
 * resident warps used (persistent grid) and SM count. */
int cmsd_launch_info(int dtype, int* warps_out, int* sms_out);

const char* cmsd_strerror(int code);
int cmsd_last_cuda_error(void);   /* cudaError_t of the last CMSD_ECUDA */

#ifdef __cplusplus
}
#endif
#endif /* CMSD_H */
