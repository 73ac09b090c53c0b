/*
 * solo_readout.h -- C ABI of the SOLO shared-readout local loss on one GB300.
 *
 * SOLO (Shared-Output LOcal learning) splits a network into K
 * gradient-isolated modules.  Every module k predicts the next token through
 * a read-only copy of the terminal readout (paper, Section 2.2, Eq. 2 with
 * temperature tau_k = 1 and no bias):
 *
 *     xhat_i  = RMSNorm_gamma(h_i)          final RMSNorm with element-wise gain
 *     z_i     = W xhat_i                     W: [V, d], the terminal readout
 *     loss_i  = logsumexp(z_i) - z_{i, y_i}  cross-entropy against next token
 *     L_k     = mean of loss_i over the kept tokens of module k
 *
 * and receives only its own gradient back through the same readout (Eq. 3):
 * dL_k/dh_k = J_norm^T W^T (softmax(z) - onehot(y)) / Nvalid_k.  No gradient
 * ever reaches the copy of W; only the final module's loss updates W and
 * gamma (Algorithm 1, the terminal cross-entropy and the Step that follows
 * it), so dW and dgamma are produced for module K-1 (0-based) alone.
 *
 * Conventions for every entry point:
 *  - Pointers are DEVICE pointers unless the comment says "host".  The caller
 *    owns all memory; the library allocates nothing and keeps no state
 *    between calls besides per-device kernel attributes set on first use
 *    and a process-wide count of the kernels it has launched.
 *  - Calls are asynchronous on `stream` (a cudaStream_t; NULL = legacy
 *    default stream).  Errors the host can detect are returned before any
 *    work is enqueued; conditions found on the device set bits of a flag
 *    word in the workspace, read back with solo_readout_get_flags.
 *  - bf16 tensors are passed as their 16-bit patterns (solo_bf16_t).
 *  - Row-major layouts; every tensor pointer must be 16-byte aligned.
 *  - Calls using distinct workspaces may run concurrently on different
 *    streams.  W and gamma must not be written while a call that reads them
 *    is in flight (they are the read-only copy of Algorithm 1).
 *  - Requires a compute capability 10.3 device (GB300, sm_103a).
 */
#ifndef SOLO_READOUT_H
#define SOLO_READOUT_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef uint16_t solo_bf16_t;          /* bf16 bit pattern */
typedef struct CUstream_st* solo_stream_t; /* same type as cudaStream_t */
typedef int32_t solo_status_t;

enum {
  SOLO_OK = 0,
  SOLO_ERR_INVALID_ARG = -1,         /* NULL required pointer, K/N/d/V out of range */
  SOLO_ERR_UNSUPPORTED_SHAPE = -2,   /* d not a multiple of 8, V above 2^23, or K*N
                                        beyond 32-bit tile coordinates */
  SOLO_ERR_WORKSPACE_TOO_SMALL = -3, /* workspace_bytes below the query result */
  SOLO_ERR_CUDA = -4,                /* a CUDA runtime call failed */
  SOLO_ERR_NOT_SM103 = -5,           /* current device is not compute capability 10.3 */
  SOLO_ERR_MISALIGNED = -6,          /* a tensor pointer is not 16-byte aligned */
  SOLO_ERR_EXCEEDS_STATIC_SCRATCH = -7 /* solo_readout_fwd_bwd_static: the problem needs
                                          more than SOLO_STATIC_SCRATCH_BYTES of scratch */
};

/* Device-detected conditions, OR-ed into the workspace flag word. */
enum {
  SOLO_FLAG_BAD_TARGET = 1u, /* a target outside [0, V) that is not ignore_index;
                                the token is treated as masked */
  SOLO_FLAG_TIMEOUT = 2u,    /* a pipeline wait exceeded its bound (about 2 s);
                                the kernel stopped early and outputs are invalid */
  SOLO_FLAG_BOUNDS = 4u      /* checked builds only (solo_readout_build_flags bit
                                SOLO_BUILD_CHECKED): a computed global index fell
                                outside its buffer; the access was skipped and
                                outputs are invalid */
};

/* Maximum number of modules per call. */
#define SOLO_MAX_MODULES 16

/* Stages of one call, for solo_readout_fwd_bwd_events. */
enum {
  SOLO_STAGE_RMSNORM = 0,   /* r_i and xhat = bf16(gamma * h * r)           */
  SOLO_STAGE_LOGITS = 1,    /* tensor-core X W^T, per-tile max/sum, exps    */
  SOLO_STAGE_LSE = 2,       /* logsumexp, token loss, module means          */
  SOLO_STAGE_GRAD = 3,      /* dL/dz = tau (softmax - onehot) / Nvalid: the
                               per-row factors of most rows applied in place
                               (final module: target entry, scaled xhat),
                               bf16 G written for the rest (with bias
                               gradients: every row summed into db)          */
  SOLO_STAGE_DXHAT = 4,     /* tensor-core dXhat = G W; its epilogue takes
                               dH through the RMSNorm Jacobian and forms the
                               dgamma partial sums                           */
  SOLO_STAGE_NORM_BWD = 5,  /* the same for the few tiles whose reduction
                               was cut into parts (after their fix-up)       */
  SOLO_STAGE_DW = 6,        /* tensor-core dW = G^T Xhat, final module      */
  SOLO_STAGE_DGAMMA = 7,    /* dgamma reduction, final module               */
  SOLO_NUM_STAGES = 8
};

typedef struct {
  int32_t K;            /* modules, 1 .. SOLO_MAX_MODULES                    */
  int64_t N;            /* tokens per module, >= 1                           */
  int32_t d;            /* width, >= 8 and a multiple of 8                   */
  int32_t V;            /* vocabulary size, 1 .. 2^23                        */
  float eps;            /* RMSNorm epsilon, inside the square root (>= 0)    */
  int32_t ignore_index; /* target value of a masked token (e.g. -100)        */
} solo_dims_t;

/*
 * Bytes of device workspace one call with these dims needs (host-only; no
 * CUDA call).  The workspace holds the normalised inputs, the bf16
 * exponentials/gradient of the logits ([K*N, V], one row per kept token),
 * per-token statistics and factors,
 * at most 32 MiB of fp32 partial tiles of the backward products and the flag
 * word.  Returns SOLO_ERR_INVALID_ARG for NULL pointers or dims out of range,
 * SOLO_ERR_UNSUPPORTED_SHAPE when d % 8 != 0 or V > 2^23.
 */
solo_status_t solo_readout_workspace_bytes(const solo_dims_t* dims, size_t* bytes);

/*
 * One forward + backward of the shared-readout local loss for all K modules
 * (Eq. 2-3; Algorithm 1, the local cross-entropy of every module and the
 * terminal cross-entropy of the last).  All K modules run as one row space
 * of K*N tokens against one resident W.
 *
 *  hidden     host array [K] of device pointers, each bf16 [N, d]: h_k, the
 *             head output of module k before its final RMSNorm.
 *  gamma      bf16 [d]: the final RMSNorm gain.
 *  W          bf16 [V, d]: the readout; W-bar == W for this call. Never written.
 *  targets    int32 [K, N]: next-token ids, already shifted; ignore_index
 *             marks masked tokens; anything else outside [0, V) is treated
 *             as masked and sets SOLO_FLAG_BAD_TARGET.
 *  mask       uint8 [K, N] or NULL: 0 masks the token (ANDed with the above).
 *             Masked tokens are skipped by every product: the kept ones are
 *             compacted (in token order) into the first rows of the workspace's
 *             per-token buffers, so the call's tensor work scales with the kept
 *             tokens.
 *  loss_tok   fp32 [K, N] or NULL: per-token cross-entropy, 0 when masked.
 *  loss_mean  fp32 [K]: L_k, mean over kept tokens (0 when none is kept).
 *  dhidden    host array [K] of device pointers, each bf16 [N, d]:
 *             dL_k/dh_k.  Rows of masked tokens are exactly 0.
 *  dW         fp32 [V, d] or NULL: dL_{K-1}/dW (final module), overwritten.
 *  dgamma     fp32 [d] or NULL: dL_{K-1}/dgamma (final module), overwritten.
 *  workspace  device buffer of at least solo_readout_workspace_bytes bytes,
 *             16-byte aligned; its contents on entry do not matter.
 *
 * Output buffers (and the workspace) may not overlap inputs or each other;
 * an overlap is refused with SOLO_ERR_INVALID_ARG before anything is
 * enqueued (inputs may share memory).  Returns SOLO_OK once
 * the work is enqueued.
 */
solo_status_t solo_readout_fwd_bwd(const solo_dims_t* dims,
                                   const solo_bf16_t* const* hidden,
                                   const solo_bf16_t* gamma,
                                   const solo_bf16_t* W,
                                   const int32_t* targets,
                                   const uint8_t* mask,
                                   float* loss_tok,
                                   float* loss_mean,
                                   solo_bf16_t* const* dhidden,
                                   float* dW,
                                   float* dgamma,
                                   void* workspace, size_t workspace_bytes,
                                   solo_stream_t stream);

/*
 * Same as solo_readout_fwd_bwd, and records events[s] on `stream` right
 * before stage s is enqueued and events[SOLO_NUM_STAGES] after the last, so
 * that consecutive events bracket one stage (skipped stages have zero
 * length).  `events` is a host array of n_events cudaEvent_t handles created
 * by the caller; n_events must be SOLO_NUM_STAGES + 1.
 */
solo_status_t solo_readout_fwd_bwd_events(const solo_dims_t* dims,
                                          const solo_bf16_t* const* hidden,
                                          const solo_bf16_t* gamma,
                                          const solo_bf16_t* W,
                                          const int32_t* targets,
                                          const uint8_t* mask,
                                          float* loss_tok,
                                          float* loss_mean,
                                          solo_bf16_t* const* dhidden,
                                          float* dW,
                                          float* dgamma,
                                          void* workspace, size_t workspace_bytes,
                                          solo_stream_t stream,
                                          void* const* events, int32_t n_events);

/*
 * Early-exit readout, forward only: every module's hidden states decoded
 * through the shared readout, as the exits of a trained SOLO model are (paper,
 * Section 3 "Every module decodes" and Appendix E: each depth's next-token
 * prediction, its log-probability and perplexity).  Per token: xhat =
 * RMSNorm_gamma(h), z = W xhat, lse = logsumexp(z).
 *
 *  targets       int32 [K, N] or NULL (decoding only); same masking rules as
 *                solo_readout_fwd_bwd.  Required when loss_tok or loss_mean is
 *                given.
 *  loss_tok      fp32 [K, N] or NULL: -log p(y) = lse - z_y, 0 when masked.
 *  loss_mean     fp32 [K] or NULL: mean over kept tokens (exp gives the
 *                module's perplexity).
 *  top1          int32 [K, N] or NULL: argmax_v z, the first (lowest) index
 *                among equal maxima.
 *  top1_logprob  fp32 [K, N] or NULL: log p(top1) = max_v z - lse.
 *  workspace     at least solo_readout_exit_workspace_bytes bytes.
 *
 * Runs the RMSNorm, one tensor-core pass over the vocabulary (K*2NVd FLOPs)
 * and a combine; no exponential or gradient buffer is written.  Flags as for
 * solo_readout_fwd_bwd (read with solo_readout_get_flags on this workspace).
 * Outputs and the workspace may not overlap inputs or each other
 * (SOLO_ERR_INVALID_ARG).
 */
solo_status_t solo_readout_exit_workspace_bytes(const solo_dims_t* dims, size_t* bytes);
solo_status_t solo_readout_exit_forward(const solo_dims_t* dims,
                                        const solo_bf16_t* const* hidden,
                                        const solo_bf16_t* gamma,
                                        const solo_bf16_t* W,
                                        const int32_t* targets,
                                        const uint8_t* mask,
                                        float* loss_tok,
                                        float* loss_mean,
                                        int32_t* top1,
                                        float* top1_logprob,
                                        void* workspace, size_t workspace_bytes,
                                        solo_stream_t stream);

/* Stages of the exit readout, for solo_readout_exit_forward_events. */
enum {
  SOLO_EXIT_STAGE_RMSNORM = 0,  /* r_i and xhat                                      */
  SOLO_EXIT_STAGE_LOGITS = 1,   /* tensor-core X W^T with per-tile max/sum/argmax     */
  SOLO_EXIT_STAGE_COMBINE = 2,  /* logsumexp, top-1, losses, module means             */
  SOLO_EXIT_NUM_STAGES = 3
};

/*
 * Same as solo_readout_exit_forward, recording events[s] before stage s and
 * events[SOLO_EXIT_NUM_STAGES] after the last (n_events must be
 * SOLO_EXIT_NUM_STAGES + 1 caller-created cudaEvent_t handles).
 */
solo_status_t solo_readout_exit_forward_events(const solo_dims_t* dims,
                                               const solo_bf16_t* const* hidden,
                                               const solo_bf16_t* gamma,
                                               const solo_bf16_t* W,
                                               const int32_t* targets,
                                               const uint8_t* mask,
                                               float* loss_tok,
                                               float* loss_mean,
                                               int32_t* top1,
                                               float* top1_logprob,
                                               void* workspace, size_t workspace_bytes,
                                               solo_stream_t stream,
                                               void* const* events, int32_t n_events);

/*
 * Each auxiliary head's own readout parameters (Algorithm 1): the local loss
 * of module k is CE(softmax(tau_k W-bar xhat + b_k), y) and the terminal loss
 * CE(softmax(W xhat + b), y).  All pointers are device pointers or NULL.
 */
typedef struct {
  const float* tau;   /* [K] temperatures tau_k, or NULL for all 1; the terminal
                         module's entry is normally 1 (the paper's terminal loss
                         has none); its dW is the gradient for the given value */
  const float* bias;  /* [K, V] biases: b_k for k < K-1 and the terminal b for
                         k = K-1, or NULL for all 0 */
  float* dtau;        /* [K] or NULL: dL_k/dtau_k = mean over kept tokens of
                         E_p[s] - s_y, s = W-bar xhat (before tau and bias) */
  float* dbias;       /* [K, V] or NULL: dL_k/db_k = sum over module k's tokens
                         of (softmax - onehot) / Nvalid_k */
} solo_heads_t;

/*
 * solo_readout_fwd_bwd with the heads' temperature and bias (Eq. 2 with tau_k;
 * Algorithm 1's b_k and b).  heads == NULL is exactly solo_readout_fwd_bwd.
 * dhidden, dW and dgamma include the factor tau_k of the chain rule.  events:
 * NULL, or SOLO_NUM_STAGES + 1 cudaEvent_t handles recorded as in
 * solo_readout_fwd_bwd_events (n_events must then be SOLO_NUM_STAGES + 1).
 * The workspace size is the same as for solo_readout_fwd_bwd.
 */
solo_status_t solo_readout_fwd_bwd_heads(const solo_dims_t* dims,
                                         const solo_bf16_t* const* hidden,
                                         const solo_bf16_t* gamma,
                                         const solo_bf16_t* W,
                                         const int32_t* targets,
                                         const uint8_t* mask,
                                         const solo_heads_t* heads,
                                         float* loss_tok,
                                         float* loss_mean,
                                         solo_bf16_t* const* dhidden,
                                         float* dW,
                                         float* dgamma,
                                         void* workspace, size_t workspace_bytes,
                                         solo_stream_t stream,
                                         void* const* events, int32_t n_events);

/*
 * Private readouts (the paper's PRIV arm, Table "Readout sources") with a
 * head-owned final norm: module k predicts through its own readout W_k and
 * final RMSNorm gain gamma_k, both trained by its own loss, so every module
 * gets dW_k and dgamma_k.  Each module is computed as a single-module
 * problem; the modules run one after another on `stream`, sharing the
 * workspace (solo_readout_private_workspace_bytes: the size for one module).
 *
 *  gamma, W   host arrays [K] of device pointers: gamma_k bf16 [d], W_k bf16 [V, d].
 *  dW, dgamma host arrays [K] of device pointers (fp32 [V, d] / [d]); the
 *             arrays or any entry may be NULL (not computed).
 *  heads      as for solo_readout_fwd_bwd_heads (tau [K], bias [K, V], ...),
 *             or NULL.
 * Other arguments as for solo_readout_fwd_bwd.  Device flags of all modules
 * accumulate in the workspace's flag word.
 */
solo_status_t solo_readout_private_workspace_bytes(const solo_dims_t* dims, size_t* bytes);
solo_status_t solo_readout_fwd_bwd_private(const solo_dims_t* dims,
                                           const solo_bf16_t* const* hidden,
                                           const solo_bf16_t* const* gamma,
                                           const solo_bf16_t* const* W,
                                           const int32_t* targets,
                                           const uint8_t* mask,
                                           const solo_heads_t* heads,
                                           float* loss_tok,
                                           float* loss_mean,
                                           solo_bf16_t* const* dhidden,
                                           float* const* dW,
                                           float* const* dgamma,
                                           void* workspace, size_t workspace_bytes,
                                           solo_stream_t stream);

/* Stages of the on-chip variant, for solo_readout_fwd_bwd_onchip's events. */
enum {
  SOLO_ONCHIP_STAGE_FINAL = 0,     /* the final module on the stored path (all its
                                      products, dW and dgamma)                     */
  SOLO_ONCHIP_STAGE_AUX_PREP = 1,  /* auxiliary modules: RMSNorm and kept counts   */
  SOLO_ONCHIP_STAGE_AUX = 2,       /* auxiliary modules: the single on-chip pass   */
  SOLO_ONCHIP_STAGE_AUX_MEANS = 3, /* auxiliary modules' mean losses               */
  SOLO_ONCHIP_NUM_STAGES = 4
};

/*
 * The same forward + backward as solo_readout_fwd_bwd, with the auxiliary
 * modules (0 .. K-2) computed in one pass whose logits never leave the chip
 * (paper, Section 2.2, Eq. 2-3: the local loss and its readout factor
 * W-bar^T delta_k).  Per token, with the reference m = a running row maximum,
 *     dxhat = ((sum over v != y of e^{z_v - m} W_v) / S - (S'/S) W_y) / Nvalid,
 *     S' = sum over v != y of e^{z_v - m},  S = S' + e^{z_y - m},
 * and loss = lse - z_y with lse = m + ln S, accumulated over 128-column
 * vocabulary tiles: each cluster of CTAs keeps a 128-row block's slice of
 * xhat, its partial logits, the exponentials P and sum_v P_v W_v in tensor
 * and shared memory.  Nothing of size tokens x vocabulary is written for
 * these modules, so their workspace is xhat and a few floats per token.  The
 * final module, whose dW needs the whole logit gradient, takes the stored path
 * of solo_readout_fwd_bwd over its own N tokens.
 *
 * Arguments and outputs are those of solo_readout_fwd_bwd; the workspace is
 * solo_readout_onchip_workspace_bytes (the final module's stored-path
 * workspace for N tokens plus K-1 modules' xhat, r and token losses).
 * events: NULL, or SOLO_ONCHIP_NUM_STAGES + 1 cudaEvent_t handles, recorded
 * before each stage and after the last (n_events must then be
 * SOLO_ONCHIP_NUM_STAGES + 1).  Widths above 2048 are refused with
 * SOLO_ERR_UNSUPPORTED_SHAPE (a 128-row block's accumulator would need more
 * than the 8 CTAs of a portable cluster).  Results agree with
 * solo_readout_fwd_bwd within the parity tolerances, not bit for bit (the
 * exponentials are formed against a different reference).
 */
solo_status_t solo_readout_onchip_workspace_bytes(const solo_dims_t* dims, size_t* bytes);
solo_status_t solo_readout_fwd_bwd_onchip(const solo_dims_t* dims,
                                          const solo_bf16_t* const* hidden,
                                          const solo_bf16_t* gamma,
                                          const solo_bf16_t* W,
                                          const int32_t* targets,
                                          const uint8_t* mask,
                                          float* loss_tok,
                                          float* loss_mean,
                                          solo_bf16_t* const* dhidden,
                                          float* dW,
                                          float* dgamma,
                                          void* workspace, size_t workspace_bytes,
                                          solo_stream_t stream,
                                          void* const* events, int32_t n_events);

/*
 * The final RMSNorm alone (the first step of every call): for each module k
 * and token i, r_i = (mean_j h_ij^2 + eps)^-1/2 and xhat_ij = bf16(gamma_j
 * h_ij r_i), rounded to nearest even on the exact value of gamma h r (paper,
 * Section 2.2: the head's final RMSNorm with element-wise gain), i.e. the
 * x-hat that the readout multiplies.  Of dims, K, N, d and eps are used (V
 * must still be valid).
 *
 *  hidden  host array [K] of device pointers, each bf16 [N, d].
 *  gamma   bf16 [d].
 *  xhat    bf16 [K*N, d], module-major rows: row k*N + i is token i of module k.
 *  r       fp32 [K*N] or NULL.
 *
 * Asynchronous on `stream`; allocates nothing.  xhat and r may not overlap
 * the inputs or each other (SOLO_ERR_INVALID_ARG).
 */
solo_status_t solo_readout_rmsnorm(const solo_dims_t* dims, const solo_bf16_t* const* hidden,
                                   const solo_bf16_t* gamma, solo_bf16_t* xhat, float* r,
                                   solo_stream_t stream);

/*
 * Waits for `stream`, then copies the flag word of the last call that used
 * `workspace` into *flags (host).  The word is cleared at the start of
 * every call.
 */
solo_status_t solo_readout_get_flags(const void* workspace, solo_stream_t stream,
                                     uint32_t* flags);

/* Static description of a status code (never NULL). */
const char* solo_readout_strerror(solo_status_t status);

/*
 * Self-test of the bounded waits that guard every pipeline wait in the
 * library's kernels (a wait that does not complete gives up, sets
 * SOLO_FLAG_TIMEOUT and lets the kernel return instead of hanging).  Launches
 * one small kernel that waits on a barrier nothing arrives on, with a limit of
 * limit_us microseconds (1 .. 1000000), through the same wait routine; the
 * kernel then ORs SOLO_FLAG_TIMEOUT into *device_flags (a device uint32 the
 * caller clears first) and returns.  Nothing faults or hangs; the context
 * stays usable.  Asynchronous on `stream`.
 */
solo_status_t solo_readout_selftest_wait_timeout(uint32_t* device_flags, uint32_t limit_us,
                                                 solo_stream_t stream);

/* Library version, major * 10000 + minor * 100 + patch. */
int32_t solo_readout_version(void);

/* How the library was built: SOLO_BUILD_CHECKED is set in the checked build,
 * whose kernels test every computed global index of the row kernels and the
 * GEMM epilogues against its buffer and report SOLO_FLAG_BOUNDS instead of
 * making the access.  Its results are bitwise those of the release build. */
#define SOLO_BUILD_CHECKED 1
int32_t solo_readout_build_flags(void);

/*
 * Number of kernels this library has enqueued in the calling process so far
 * (all threads, all devices; each successful launch counts once).  A
 * caller that reads it before and after a sequence of calls gets the exact
 * number of the library's kernels in that sequence.  Host-only and
 * lock-free; it does not synchronise with the device.
 */
uint64_t solo_readout_kernel_launches(void);

/*
 * Size of the library's built-in scratch area used by
 * solo_readout_fwd_bwd_static: 64 MiB of device memory, reserved on every GPU
 * that loads the library's device code and held until the process exits.
 */
#define SOLO_STATIC_SCRATCH_BYTES (64u << 20)

/*
 * The same forward + backward as solo_readout_fwd_bwd, for callers that
 * cannot allocate device memory and so cannot supply a workspace: code that
 * runs where allocation is forbidden or unavailable, such as an inference or
 * plugin host that lets a step enqueue work but never allocate, or a loop
 * that froze its memory use after start-up.  This paper has no counterpart
 * of it; it is an addition of this library.
 *
 * Instead of a caller workspace it uses a fixed scratch array compiled into
 * the library (SOLO_STATIC_SCRATCH_BYTES).  The call itself allocates
 * nothing.  Limits and rules:
 *  - Problems whose solo_readout_workspace_bytes exceeds
 *    SOLO_STATIC_SCRATCH_BYTES are rejected with
 *    SOLO_ERR_EXCEEDS_STATIC_SCRATCH before anything is enqueued (roughly
 *    K*N*(2.047*V + 2*d + 60) bytes plus up to 32 MiB of partial tiles of the
 *    backward products must fit; e.g. K=2, N=256, d=128, V=4096 uses about
 *    8.3 MiB).
 *  - The first call on a device looks up the device address of the scratch
 *    array for that device (the array's name in host code is not a device
 *    address) and keeps it for the rest of the process.  Make that first call
 *    before any stream capture.  A cudaDeviceReset destroys the device's
 *    context and the array with it, so the kept address (like the kernel
 *    attributes every entry point sets on its first call on a device) is no
 *    longer valid: after a reset, do not call this library on that device
 *    again in the same process.
 *  - Every call on a device shares the one array, and it keeps the previous
 *    call's contents; the call clears what must start at zero itself.  Calls
 *    whose execution overlaps on the GPU (other streams, other host
 *    threads) race on the scratch and give wrong results: serialise them.
 *  - device_flags: NULL, or a device uint32 that receives this call's flag
 *    word (SOLO_FLAG_*) at the end of the call, asynchronously on `stream`.
 * Every other argument means what it means for solo_readout_fwd_bwd.
 */
solo_status_t solo_readout_fwd_bwd_static(const solo_dims_t* dims,
                                          const solo_bf16_t* const* hidden,
                                          const solo_bf16_t* gamma,
                                          const solo_bf16_t* W,
                                          const int32_t* targets,
                                          const uint8_t* mask,
                                          float* loss_tok,
                                          float* loss_mean,
                                          solo_bf16_t* const* dhidden,
                                          float* dW,
                                          float* dgamma,
                                          uint32_t* device_flags,
                                          solo_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* SOLO_READOUT_H */
