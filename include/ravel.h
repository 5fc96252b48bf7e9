/*
 * ravel.h -- C ABI of the GB300 rolling action-expert step.
 *
 * The step is the inner loop of RAVEL (asynchronous rolling inference for
 * flow-based VLAs): one denoising pass of the flow-matching action expert over
 * an H-slot action buffer whose slots sit at staggered flow times, followed by
 * a per-slot Euler update, release of the first slot, a shift and the append
 * of a fresh Gaussian slot (paper Sec. 3.1, Eq. 1 and Eq. 3).  The expert
 * attends to the latest cached VLM prefix K/V (Eq. 2), reused across steps
 * until a new one arrives (Sec. 3.2), plus Fast-Observation-Pathway tokens
 * (Eq. 4), and is conditioned on each slot's flow time and on the context age
 * delta_p = p / K (Sec. 3.1; App. A.1).
 *
 * Conventions shared by every call:
 *  - B robots, H slots, A action dims, D width, L layers, Hq / Hkv query / KV
 *    heads, hd head dim, Fm MLP width, P prefix tokens, F FOP tokens.
 *  - Flow time t = 1 - tau (t = 1 is pure noise).  Slot j (0-based; j = 0 is
 *    released next) carries slot_times[j]; the Euler step of slot j is
 *    dt_j = t_j - t_{j-1} with t_{-1} = 0 (the staggered schedule t_j = (j+1)/H
 *    gives the paper's uniform 1/K).
 *  - Every pointer argument documented "device" must be device memory on the
 *    library's device; "host" must be host memory.  Pointers are borrowed for
 *    the duration of the call and, for device pointers passed to asynchronous
 *    calls, until the work enqueued on the given stream has completed.
 *  - Streams are cudaStream_t values passed as void*.  NULL means the legacy
 *    default stream.
 *  - Every call returns a status and never aborts.  Asynchronous CUDA errors
 *    and errors raised by kernels (the device error word) surface on a later
 *    call as RAVEL_ECUDA / RAVEL_EDEVICE / RAVEL_ETIMEOUT.
 *  - A handle is not thread-safe: calls on one handle must be serialised.
 */
#ifndef RAVEL_H_
#define RAVEL_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  RAVEL_OK = 0,
  RAVEL_EINVAL = 1,      /* a null pointer or an argument out of its domain */
  RAVEL_ESHAPE = 2,      /* a size outside the handle's configuration */
  RAVEL_ENOMEM = 3,      /* device or host allocation failed */
  RAVEL_ECUDA = 4,       /* a CUDA call failed; ravel_last_error() has the text */
  RAVEL_ENOCONTEXT = 5,  /* ravel_roll_step before any ravel_set_context */
  RAVEL_EBUSY = 6,       /* ravel_set_context while the previous swap is pending */
  RAVEL_EDEVICE = 7,     /* a kernel raised the device error word (e.g. bad prefix length) */
  RAVEL_ETIMEOUT = 8,    /* a bounded device-side wait ran out */
  RAVEL_ENOTREADY = 9    /* a call that needs ravel_reset first */
} ravel_status;

enum { RAVEL_FP32 = 0, RAVEL_BF16 = 1 };
enum { RAVEL_MASK_FULL = 0, RAVEL_MASK_SLOT_ISOLATED = 1 };

/* Shape of the expert and capacity of the handle. */
typedef struct {
  int layers;       /* L */
  int width;        /* D, a multiple of 8, at most 4096 */
  int n_q_heads;    /* Hq, a multiple of n_kv_heads */
  int n_kv_heads;   /* Hkv */
  int head_dim;     /* hd, a multiple of 8, at most 256 */
  int mlp_dim;      /* Fm, a multiple of 64 */
  int slots;        /* H (the paper's K with one action per slot) */
  int action_dim;   /* A */
  int max_prefix;   /* largest prefix length a context may carry */
  int fop_tokens;   /* F (0 allowed) */
  int max_batch;    /* largest B accepted by ravel_reset */
  int dtype;        /* RAVEL_FP32: all arithmetic fp32; RAVEL_BF16: weights, prefix,
                       FOP tokens and GEMM activations bf16, fp32 accumulation,
                       fp32 residual stream, norms, softmax and buffer; where a
                       projection or the attention splits its reduction over
                       SMs (few tokens), each split's share crosses between
                       the SMs as bf16 and the shares are summed in fp32 */
  int mask_mode;    /* RAVEL_MASK_FULL: every action query sees the valid prefix,
                       all FOP tokens and all H slots; RAVEL_MASK_SLOT_ISOLATED
                       (a test mode): action query j sees the prefix, the FOP
                       tokens and slot j only */
  int fop_adapter_every; /* 0: the FOP tokens are extra keys / values of every
                       layer's self-attention; k in [1, layers]: they are no
                       keys of the self-attention and enter layers k-1, 2k-1,
                       ... through gated cross-attention adapters (Sec. 3.2:
                       "injected into selected action-expert layers through
                       gated cross-attention adapters"), each after its
                       layer's self-attention block:
                       x += tanh(a_gate) MHA(q = RMSNorm(x)(1 + a_gamma) a_wq,
                       [k | v] = RMSNorm(z)(1 + a_zgamma) a_wkv) a_wo */
  int per_robot_times; /* 0: one slot-time schedule [H] shared by every robot;
                       1: every robot runs its own schedule, slot_times
                       [B, H] (the conditioning, the Euler step and the
                       relative shift use robot b's t_bj; the modulation is
                       then computed for B*H time rows every step, with no
                       conditioning cache) */
} ravel_config;

/*
 * Expert parameters, float32, math layout y = x @ W + b (W is [in, out],
 * row-major).  Per-layer tensors are stacked on a leading L axis.
 *   t_w1,t_w2 [D,D]  t_b1,t_b2 [D]   flow-time MLP  (Linear, SiLU, Linear)
 *   d_w1,d_w2 [D,D]  d_b1,d_b2 [D]   context-offset MLP (App. A.1)
 *   mod_w [D, 4LD+2D]  mod_b [4LD+2D] adaRMSNorm modulation; columns of layer l
 *                     are (scale1, shift1, scale2, shift2) at 4lD, then the
 *                     final norm's (scale, shift) at 4LD
 *   in_w [A,D] in_b [D]              action in-projection
 *   fop_gamma [L,D]                  per-layer FOP-token RMSNorm gain (1 + gamma)
 *   w_qkv [L,D,(Hq+2Hkv)hd]          columns [Q heads | K heads | V heads]
 *   w_o [L,Hq hd,D]  w_gate,w_up [L,D,Fm]  w_down [L,Fm,D]
 *   out_w [D,A] out_b [A]            velocity head
 * on_device = 0: host pointers; 1: device pointers.  ravel_create copies and
 * repacks everything; the caller keeps ownership.  In RAVEL_BF16 mode values
 * are rounded to bf16 (nearest, ties to even).
 */
typedef struct {
  const float *t_w1, *t_b1, *t_w2, *t_b2;
  const float *d_w1, *d_b1, *d_w2, *d_b2;
  const float *mod_w, *mod_b;
  const float *in_w, *in_b;
  const float *fop_gamma;
  const float *w_qkv, *w_o, *w_gate, *w_up, *w_down;
  const float *out_w, *out_b;
  int on_device;
  /* FOP adapters (cfg.fop_adapter_every > 0; NA = layers / fop_adapter_every
   * adapters, stacked): a_gamma, a_zgamma [NA, D]; a_wq [NA, D, Hq hd];
   * a_wkv [NA, D, 2 Hkv hd] (K heads, then V heads); a_wo [NA, Hq hd, D];
   * a_gate [NA].  NULL when there are no adapters. */
  const float *a_gamma, *a_zgamma, *a_wq, *a_wkv, *a_wo, *a_gate;
} ravel_weights;

typedef struct ravel_ctx ravel_t;

/* Validate cfg, allocate the handle on `device` (the CUDA ordinal), pack the
 * weights into HBM and allocate the double-buffered context, activations and
 * step state for cfg.max_batch robots.  Synchronous.  On success *out owns all
 * of it until ravel_destroy. */
ravel_status ravel_create(const ravel_config* cfg, const ravel_weights* w, int device, ravel_t** out);

/* Free everything the handle owns (after synchronising its device).  NULL is a no-op. */
void ravel_destroy(ravel_t* r);

/* Start a rollout of `batch` robots (warm start without extra initialisation,
 * App. A.1): robot b's noise seed is seeds[b] (host, [batch]); slot j of
 * buffer (device, float32 [batch, H, A], written) receives the Gaussian action
 * of index j, and the robot's next appended action gets index H.  Enqueued on
 * `stream`.  A new batch size invalidates the current context (set it again).
 * Also clears the handle's device error word (after synchronising the
 * device). */
ravel_status ravel_reset(ravel_t* r, int batch, const uint64_t* seeds, float* buffer, void* stream);

/* Install a new VLM context (Eq. 2): k and v are device arrays
 * [L, B, Hkv, prefix_len, hd] of the handle's dtype (float32 or bf16) for the
 * current batch B.  The copy goes into the inactive half of the double buffer
 * on `side_stream`, after the last enqueued step has finished reading it, so
 * steps on other streams continue meanwhile; the next ravel_roll_step makes
 * its stream wait for the copy and then switches to the new context.  The
 * caller may reuse k / v once the side stream has passed this call.
 * 1 <= prefix_len <= max_prefix, else RAVEL_ESHAPE.  A second call before a
 * step has consumed the first returns RAVEL_EBUSY.  Every robot has its own
 * half of the double buffer: this call is ravel_set_context_robots for all
 * robots of the batch. */
ravel_status ravel_set_context(ravel_t* r, const void* k, const void* v, int prefix_len, void* side_stream);

/* Install new VLM contexts for some robots only (Sec. 3.2: each robot's
 * context is refreshed whenever its own VLM pass completes, so robots run
 * with contexts of different ages and lengths):
 *   robots  host int [n], distinct robot indices < B
 *   k, v    device arrays [L, n, Hkv, prefix_len, hd] of the handle's dtype,
 *           entry i for robot robots[i]
 * Each listed robot's context goes into its own inactive half on
 * `side_stream` (after the last enqueued step and any earlier pending copy);
 * at the next step those robots switch to it with this prefix length while the
 * others keep theirs.  Robots still without a context make a step return
 * RAVEL_ENOCONTEXT.  RAVEL_EBUSY if a listed robot's previous context has not
 * yet been consumed by a step; RAVEL_EINVAL for a repeated or out-of-range
 * index; RAVEL_ESHAPE for n outside [1, B] or prefix_len outside
 * [1, max_prefix]. */
ravel_status ravel_set_context_robots(ravel_t* r, const int* robots, int n, const void* k, const void* v,
                                      int prefix_len, void* side_stream);

/* One rolling step (Eq. 3 plus release / shift / append) for the current
 * batch, enqueued on `stream` as one CUDA-graph launch:
 *   buffer      device float32 [B, H, A], read and updated in place
 *   slot_times  device float32 [H], increasing, slot_times[H-1] = 1 for the
 *               paper's schedule; [B, H] (one schedule per robot) for a
 *               handle created with per_robot_times
 *   obs_tokens  device [B, F, D] FOP tokens of the handle's dtype (NULL iff F = 0)
 *   delta       device float32 [B], context age p/K (+ bias) per robot
 *   released    device float32 [B, A], written: the action released by each robot
 *   velocity    device float32 [B, H, A] or NULL: the expert's velocity
 * The step graph is captured on first use and re-captured when any of these
 * pointers changes; graph capture needs no caller action. */
ravel_status ravel_roll_step(ravel_t* r, float* buffer, const float* slot_times, const void* obs_tokens,
                             const float* delta, float* released, float* velocity, void* stream);

/* The rolling step for an expert that predicts actions relative to the robot
 * state while the buffer keeps absolute targets (App. "LIBERO and RoboTwin
 * 2.0": absolute targets are stored, converted to actions relative to the
 * latest state before each expert update and back afterwards; the paired
 * noise stays in model coordinates).  Same arguments and effects as
 * ravel_roll_step, plus
 *   state   device float32 [B, A]: the latest robot state in the action
 *           coordinates (non-null)
 * A slot at flow time t holds a = t eps + (1 - t) a_hat, so on the relative
 * dimensions (ravel_set_relative_dims) the expert sees a - (1 - t_j) state,
 * the Euler step happens there, and each slot returns to absolute
 * coordinates at its new time t_{j-1}: a' = a + dt_j (v_j + mask * state).
 * The released slot (t = 0) is an absolute action; the appended slot is pure
 * noise (t = 1) and needs no shift.  With h > 1 actions per slot
 * (action_dim = h * the robot's action size) the mask repeats per action. */
ravel_status ravel_roll_step_rel(ravel_t* r, float* buffer, const float* slot_times, const void* obs_tokens,
                                 const float* delta, const float* state, float* released, float* velocity,
                                 void* stream);

/* Which action dimensions the expert predicts relative to the robot state:
 * mask host float32 [A], 1 = relative (for example joint or pose targets),
 * 0 = absolute (for example a gripper command).  A new handle has none.
 * Synchronous. */
ravel_status ravel_set_relative_dims(ravel_t* r, const float* mask);

/* The full-horizon (synchronous) denoising that the paper compares rolling
 * inference with (Experiments, synchronous simulation: ten full-horizon
 * denoising steps per policy query; Table 1): every robot draws a fresh chunk
 * of H Gaussian actions -- its next H action indices; its counter advances by
 * H -- and all H slots then take n_steps Euler steps together, each one pass
 * of the same action expert with every slot at one flow time t_n = 1 - n /
 * n_steps (float32), followed by a += (t_n - t_{n+1}) v with t_{n_steps} = 0.
 * Nothing is released, shifted or appended: the returned chunk (t = 0) is
 * executed as a whole.
 *   chunk        device float32 [B, H, A], written: the denoised chunk
 *   n_steps      1 .. 64 (the paper's baseline uses 10)
 *   obs_tokens, delta: as for ravel_roll_step
 *   velocity     device float32 [B, H, A] or NULL: the last pass's velocity
 * Enqueued on `stream` as one CUDA-graph launch (captured on first use, and
 * again when n_steps or a pointer changes); a pending context swap is applied
 * first, as for ravel_roll_step. */
ravel_status ravel_denoise_chunk(ravel_t* r, float* chunk, int n_steps, const void* obs_tokens, const float* delta,
                                 float* velocity, void* stream);

/* Per-robot action counters (the index of the next appended action), host
 * uint64 [B].  get synchronises the handle's device; set is synchronous and
 * lets a rollout resume bit-exactly. */
ravel_status ravel_get_state(ravel_t* r, uint64_t* counters);
ravel_status ravel_set_state(ravel_t* r, const uint64_t* counters);

/* Number of kernel launches one ravel_roll_step graph contains (0 before the
 * first step). */
int ravel_step_kernel_count(const ravel_t* r);

/* ravel_roll_step run eagerly (no graph) with a CUDA event after every kernel
 * launch, for per-kernel timing: same arguments and effects, plus host
 * outputs launch_ms [cap] (duration of each launch in ms) and launch_kind
 * [cap] (kind id, see ravel_kernel_kind_name); *n_launches receives the
 * number of launches (entries beyond cap are dropped).  The stream is first
 * held for ~5 ms so that all launches are queued before the first one starts.
 * The step's launches are followed by 16 launches of an empty kernel, timed
 * the same way (kind "launch_gap"): the overhead every interval holds.
 * Synchronous. */
ravel_status ravel_profile_step(ravel_t* r, float* buffer, const float* slot_times, const void* obs_tokens,
                                const float* delta, float* released, float* velocity, void* stream,
                                float* launch_ms, int* launch_kind, int cap, int* n_launches);

/* One projection GEMM of the kind the step runs, through the step's own
 * dispatcher (tcgen05 tensor cores for a RAVEL_BF16 handle whose operands
 * are 16-byte aligned with K, lda, ldw multiples of 8; the fp32 SIMT kernel
 * otherwise): a building block of ravel_roll_step exposed for kernel tests.
 *   X   device [M, lda] activations of the handle's dtype, first K columns used
 *   W   device [N, ldw] weights (K-major: row n holds output feature n)
 *   epi 0: out = X W^T + bias            1: out = SiLU(X W^T + bias)
 *       2: out += X W^T + bias (float32 out)
 *       3: GeGLU (bf16 handle, N % 128 == 0): W rows in 128-row blocks of 64
 *          gate rows then the 64 matching up rows; out[m][f] =
 *          gelu_tanh(gate + bias) * (up + bias) for f < N/2, each bias
 *          that of its W row
 *   out device [M, ldo], out_dtype RAVEL_FP32 or RAVEL_BF16; bias device [N] or NULL
 * Accumulation is fp32 throughout and split-K partials stay fp32 here (the
 * step's own projections send theirs between the SMs as bf16).
 * Enqueued on `stream`; uses the handle's split-K workspace, so it must not
 * overlap another call on the same handle.  Like ravel_roll_step it first
 * reports a device error raised by earlier work (RAVEL_EDEVICE /
 * RAVEL_ETIMEOUT) and mirrors the error word after its own launch. */
ravel_status ravel_gemm(ravel_t* r, const void* X, int M, int K, int lda, const void* W, int N, int ldw, int epi,
                        void* out, int ldo, int out_dtype, const float* bias, void* stream);

/* Allocation-free variant of ravel_gemm for callers that cannot allocate
 * device memory (and so cannot create a handle): for example code running in
 * another runtime's memory pool with raw allocation disabled, plugin hosts
 * that forbid cudaMalloc, or control loops that must not touch the allocator
 * after start-up.  The paper has no counterpart; this is a property of the
 * library, not of the method.
 * Same operation, arguments and epilogues as ravel_gemm, bf16 operands only
 * (X and W bf16, 16-byte aligned, K, lda, ldw multiples of 8), on the
 * current CUDA device.  It calls no cudaMalloc / cudaFree: its split-K
 * scratch is one fixed device array inside the library (8 MiB of partial
 * sums plus tile counters), held by every GPU that loads the library until
 * the process exits.  The split plan is chosen to fit that array.  M, N, K
 * above RAVEL_NOALLOC_MAX_M / _N / _K return RAVEL_ESHAPE; bad pointers or
 * modes RAVEL_EINVAL.  The first call on a device resolves the array's device
 * address (and the kernel set-up) for that device; make that first call
 * before any stream capture (a first call on a capturing stream returns
 * RAVEL_EINVAL and does nothing).  Each call clears the scratch's tile
 * counters on `stream` before the GEMM; every call shares the array, so calls
 * that overlap on the GPU race and must be serialised by the caller.  The
 * array also holds a device error word that calls never clear: a bounded wait
 * that runs out inside the GEMM (its output is then not valid) stays recorded
 * until ravel_gemm_noalloc_status reads it. */
#define RAVEL_NOALLOC_MAX_M 32768
#define RAVEL_NOALLOC_MAX_N 262144
#define RAVEL_NOALLOC_MAX_K 65536
ravel_status ravel_gemm_noalloc(const void* X, int M, int K, int lda, const void* W, int N, int ldw, int epi,
                                void* out, int ldo, int out_dtype, const float* bias, void* stream);

/* Error state of ravel_gemm_noalloc on the current device (allocates
 * nothing): waits for `stream`, then reads and clears the device error word of
 * the allocation-free entry point.  RAVEL_OK if no call has run into an error
 * since the last read (or none has run), RAVEL_ETIMEOUT if a bounded wait in
 * one of its GEMMs ran out (that call's output is not valid), RAVEL_EDEVICE for
 * any other kernel error, RAVEL_EINVAL on a capturing stream. */
ravel_status ravel_gemm_noalloc_status(void* stream);

/* Fault injection for tests of the failure-detection paths.  No GPU fault is
 * raised and every wait involved is bounded:
 *   RAVEL_FAULT_PREFIX_LEN: enqueue on `stream` a write of an out-of-range
 *     prefix length into the handle's device context state (r required; count
 *     unused).  The attention kernels of the next step refuse it, compute
 *     nothing and raise the device error word, and a later call on the handle
 *     returns RAVEL_EDEVICE.  The next ravel_set_context installs a valid
 *     state again and ravel_reset clears the error word.
 *   RAVEL_FAULT_WITHHOLD_ARRIVAL: the next `count` tensor-core GEMM launches
 *     that run without a thread-block cluster (for example ravel_gemm or
 *     ravel_gemm_noalloc with K <= 64) wait for an mbarrier arrival that
 *     nobody makes; each gives up after 2 ms, drains its copies, raises
 *     ERR_TIMEOUT and exits.  A later call on the handle returns
 *     RAVEL_ETIMEOUT (ravel_gemm_noalloc_status for the allocation-free
 *     entry point).  r may be NULL.
 * The paper has no counterpart; this serves the library's own tests. */
enum { RAVEL_FAULT_PREFIX_LEN = 1, RAVEL_FAULT_WITHHOLD_ARRIVAL = 2 };
ravel_status ravel_debug_inject(ravel_t* r, int fault, int count, void* stream);

/* Name of a kernel kind id of ravel_profile_step ("gemm_down", ...). */
const char* ravel_kernel_kind_name(int kind);

/* Static text of a status; per-handle text of the last error (never NULL). */
const char* ravel_status_string(ravel_status s);
const char* ravel_last_error(const ravel_t* r);

#ifdef __cplusplus
}
#endif
#endif /* RAVEL_H_ */
