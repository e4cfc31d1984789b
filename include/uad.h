/*
 * uad.h -- C ABI of the Urgency-Aware Denoising (UAD) library for GB300 (sm_103a).
 *
 * The library runs the denoising loop of a flow-matching action expert on one GPU:
 * per-action Euler steps with per-action flow times (Sec. 3, Eqs. 1-2; Sec. 4.2, Eqs. 4-5),
 * Urgency-Aware Early Release of actions whose budget ends before N* (Sec. 4.2),
 * Trajectory Reconciliation of released actions with zero extra evaluations (Sec. 4.3,
 * Eqs. 6-7), ghost actions, and Ghost Action Correction of the executable tail (Sec. 4.4,
 * Eqs. 8-9). Releases are handed to the host while the tail keeps refining on the GPU
 * (App. C.1, "Asynchronous Execution").
 *
 * Conventions
 *   - Every call returns an int: UAD_OK (0) or a negative code below. uad_last_error()
 *     gives a message for the last failure on a context.
 *   - Pointers marked "host or device" may point to either; the library inspects them.
 *   - The caller owns every buffer it passes and may reuse it as soon as the call returns
 *     (the library copies what it keeps). The library owns its weights, state, scratch and
 *     the pinned release buffer, all freed by uad_destroy.
 *   - All arguments are validated on the host before anything is launched.
 *   - No call waits on the GPU without a deadline; no call traps the GPU.
 *   - A context is used by one host thread at a time.
 */
#ifndef UAD_H
#define UAD_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define UAD_OK 0
#define UAD_EINVAL (-22)     /* invalid argument or configuration */
#define UAD_ESTATE (-1)      /* call out of order (e.g. finish without denoise) */
#define UAD_ENOMEM (-12)     /* device or pinned allocation failed */
#define UAD_ECUDA (-5)       /* a CUDA runtime call failed; see uad_last_error */
#define UAD_ETIMEDOUT (-110) /* the deadline passed before the GPU finished */
#define UAD_ENONFINITE (-33) /* a velocity was NaN or Inf; outputs are still written */

#define UAD_KIND_ADARMS 0    /* joint attention over prefix KV + chunk, adaptive RMSNorm */
#define UAD_KIND_DIT 1       /* chunk self-attention + cross-attention, adaLN-zero */
#define UAD_KIND_CONCAT 2    /* joint attention as ADARMS with plain RMSNorm; each token's time
                                embedding joins its action embedding in the input MLP (App. C.1,
                                the SmolVLA variant) */

#define UAD_DTYPE_F32 0
#define UAD_DTYPE_BF16 1

#define UAD_MAX_STEPS 64     /* largest step budget N_i */

/* Shape of the action expert F_theta (Sec. 3, Eq. 1). */
typedef struct uad_arch {
  int32_t kind;          /* UAD_KIND_ADARMS, UAD_KIND_DIT or UAD_KIND_CONCAT */
  int32_t dtype;         /* UAD_DTYPE_F32: fp32 everywhere; UAD_DTYPE_BF16: bf16 weights and
                            GEMM/attention operands, fp32 accumulation, state and velocities */
  int32_t n_layers;
  int32_t width;         /* W */
  int32_t n_heads;       /* query heads */
  int32_t n_kv_heads;    /* key/value heads (divides n_heads; DiT: == n_heads) */
  int32_t head_dim;
  int32_t mlp_dim;
  int32_t action_dim;    /* D */
  int32_t chunk_len;     /* H, actions per chunk (Sec. 3) */
  int32_t prefix_len;    /* P, observation prefix tokens */
  int32_t prefix_width;  /* DiT: width of the prefix tokens (cross-attention input) */
  int32_t rope;          /* ADARMS: RoPE on chunk queries/keys at positions P + i */
  int32_t max_batch;     /* robots per call, >= 1 */
} uad_arch;

/* The urgency schedule of one call (Sec. 4.2, Eq. 4, generalised to per-action budgets). */
typedef struct uad_schedule {
  const int32_t* budgets;  /* host, [batch][chunk_len], N_i >= 1; N* = max over a robot's row */
  int32_t batch;           /* robots in this call, 1..max_batch */
  int32_t n_exec;          /* S, actions executed before replanning; 0 means chunk_len */
  int32_t tr;              /* Trajectory Reconciliation on (1) or off (0, UAER-only ablation:
                              released actions are fed back frozen at flow time 1) */
  int32_t gac;             /* Ghost Action Correction on/off; needs tr unless chunk_relative */
  int32_t chunk_relative;  /* actions relative to the chunk start: GAC is skipped (Sec. 4.4) */
  const uint8_t* gac_mask; /* host [action_dim], 1 = additive dimension corrected by Eq. 9,
                              0 = left unchanged (rotation / gripper); NULL = all additive */
  int32_t rot_dim;         /* first of three dimensions holding a rotation vector (axis times
                              angle, radians) that GAC corrects by composition on SO(3)
                              (App. C.1): E_R = F_U ... F_2 F_1 with F_i = R(ghost_i)
                              R(released_i)^T over the early actions in token order (each applied
                              after the previous ones); every tail action
                              R <- exp(log(E_R)/|tail|) R.
                              These dimensions are never additive; -1 = no rotation dimensions.
                              Must be -1 or in 0..action_dim-3 (else UAD_EINVAL). */
} uad_schedule;

typedef struct uad_stats {
  int32_t evals;           /* velocity-network evaluations of the chunk (= N*; TR adds none) */
  int32_t n_star;          /* max step budget of the call */
  int32_t nonfinite;       /* count of non-finite velocity entries */
  int32_t tr_extra_evals;  /* evaluations spent on reconciliation: always 0 */
} uad_stats;

typedef struct uad_ctx uad_ctx;

/* Create a context on the current CUDA device.
 * weights: host or device fp32 blob of n_floats values, tensors in this order (linear
 *   weights [in][out], y = x W + b):
 *     t_w1[W][W] t_b1[W] t_w2[W][W] t_b2[W] in_w[D][W] in_b[W]
 *     per layer, ADARMS: mod1_w[W][3W] mod1_b[3W] wq[W][Hq*dh] wk[W][Hkv*dh] wv[W][Hkv*dh]
 *                        wo[Hq*dh][W] mod2_w[W][3W] mod2_b[3W] wg[W][F] wu[W][F] wd[F][W]
 *                DiT:    mod_w[W][6W] mod_b[6W] wq wk wv[W][Hq*dh] wo[Hq*dh][W]
 *                        wqc[W][Hq*dh] wkc wvc[Pw][Hq*dh] woc[Hq*dh][W]
 *                        w1[W][F] b1[F] w2[F][W] b2[W]
 *     modf_w[W][2W] modf_b[2W] out_w[W][D] out_b[D]
 *   CONCAT instead: in_w[D][W] in_b[W] ti_wa[W][W] ti_wt[W][W] ti_b[W] to_w[W][W] to_b[W],
 *     per layer wq wk wv wo wg wu wd (shapes as ADARMS), out_w[W][D] out_b[D]; the input is
 *     h = SiLU((u in_w + in_b) ti_wa + e(tau) ti_wt + ti_b) to_w + to_b with e the token's
 *     sinusoidal time embedding, every norm is RMSNorm without modulation and residuals are
 *     ungated.
 *   Modulation vectors are (scale, shift, gate) for ADARMS and (shift1, scale1, gate1,
 *   shift2, scale2, gate2) for DiT; the final one is (scale, shift) / (shift, scale).
 *   For bf16 architectures every weight is rounded to bf16 (nearest, ties to even).
 * The weights are copied into the library's own layout; the blob may be freed afterwards.
 * Errors: UAD_EINVAL (shape, n_floats), UAD_ENOMEM, UAD_ECUDA. */
int uad_init(const uad_arch* arch, const float* weights, size_t n_floats, uad_ctx** out);

/* Bind robot `robot`'s observation context (the cached vision-language prefix, Sec. 3).
 * ADARMS: k, v = per-layer prefix keys and values [L][P][Hkv][dh] (keys already carry
 *         their own position encoding).
 * DiT:    k = prefix tokens [P][prefix_width], v = NULL; the per-layer cross-attention K/V
 *         are projected here, once per observation.
 * dtype: UAD_DTYPE_F32 or UAD_DTYPE_BF16 element type of the given buffers (host or device);
 * they are copied (converted to the arch dtype). prefix_len must equal arch.prefix_len.
 * Errors: UAD_EINVAL, UAD_ESTATE (a chunk is in flight), UAD_ECUDA. Synchronous. */
int uad_set_prefix_kv(uad_ctx* ctx, int32_t robot, const void* k, const void* v,
                      int32_t prefix_len, int32_t dtype);

/* Precompute the per-action time conditioning for every flow time j/n, 1 <= n <= max_budget,
 * plus 1 (App. C.1). Optional: uad_denoise computes missing times itself. Synchronous. */
int uad_prepare_times(uad_ctx* ctx, int32_t max_budget);

/* Start denoising one chunk for sched->batch robots (robots 0..batch-1) on `stream`
 * (a cudaStream_t; NULL = legacy default stream). Asynchronous: returns once the work is
 * enqueued. noise: host or device fp32 [batch][H][D], the initial state x_0 (Sec. 3).
 * n_star: 0, or the largest budget of the call (checked). Every robot must have a prefix.
 * Early actions are released into pinned host memory after their last step (UAER); the
 * tail continues on the stream. Errors: UAD_EINVAL, UAD_ESTATE (previous chunk not
 * finished), UAD_ECUDA. */
int uad_denoise(uad_ctx* ctx, const float* noise, const uad_schedule* sched, int32_t n_star,
                void* stream);

/* Host-side hand-off of released actions (App. C.1: urgent actions go to the execution
 * queue while the tail refines). Waits until at least `min_ready` of robot `robot`'s
 * actions are available, or until timeout_us passes (0: do not wait).
 * out [H][D] (host): rows of ready actions are written (others untouched);
 * ready [H] (host, may be NULL): 1 if available; release_step [H] (may be NULL): the step
 * after which the action became available (N_i for early actions, N* for the tail, whose
 * rows already include GAC). Released actions never change afterwards (Sec. 4.4).
 * Returns the number of ready actions (>= min_ready), UAD_ETIMEDOUT, or an error (UAD_EINVAL
 * for min_ready > H). */
int uad_poll_released(uad_ctx* ctx, int32_t robot, int32_t min_ready, int64_t timeout_us,
                      float* out, int32_t* ready, int32_t* release_step);

/* Wait (at most timeout_us; < 0 = no limit) for the chunk to complete and read it back.
 * final [batch][H][D]: released actions for early actions, x_{N*} plus GAC (Eq. 9) for the
 *   executable tail, x_{N*} for the rest;
 * ghost [batch][H][D]: reconciled end states x'_{N*} (ghost actions, Sec. 4.3) for early
 *   actions, x_{N*} (before GAC) for the others;
 * gac_error [batch][D]: E of Eq. 8 (zeros where GAC did not run).
 * Any output may be NULL; each may be host or device memory.
 * Returns UAD_OK, UAD_ENONFINITE (outputs written), UAD_ETIMEDOUT (the chunk stays in
 * flight; call again), UAD_ESTATE, UAD_ECUDA. UAD_ECUDA after a bounded device-side wait ran
 * out: if the chunk ran on the persistent evaluation kernel (whose grid barriers need all of
 * its CTAs resident at once, which a shared or partitioned GPU may not grant), the context runs
 * every later chunk on the per-operation kernels (uad_set_wait_limit tries the persistent
 * kernel again). */
int uad_finish(uad_ctx* ctx, float* final_actions, float* ghost, float* gac_error,
               uad_stats* stats, int64_t timeout_us);

/* Device timestamps of the last finished chunk: ms[k-1] = time from the chunk's first
 * kernel to the end of step k (k = 1..n_star), from the GPU's global timer. Returns the
 * number of entries written. */
int uad_step_times(const uad_ctx* ctx, double* ms, int32_t max_entries);

/* Kernel launches the library enqueues per uad_denoise of the given batch and N*
 * (excluding one-time time-conditioning fills). */
int uad_launches_per_chunk(const uad_ctx* ctx, int32_t batch, int32_t n_star);

/* Per-kernel profile of one chunk (measurement support, not part of the method). */
typedef struct uad_kernel_stat {
  char name[32];          /* kernel class, e.g. "gate_up_proj", "attention", "euler_tr_gac" */
  int32_t launches;       /* launches of this class in the chunk */
  int32_t pad;
  double total_ms;        /* sum of CUDA-event durations of those launches */
  double bytes;           /* algorithmic HBM bytes of those launches (operands read once) */
  double flops;           /* algorithmic flops of those launches */
} uad_kernel_stat;

/* Run one chunk like uad_denoise + uad_finish, but launched eagerly (no graph) on the
 * library's worker stream with a CUDA event pair around every kernel, and return per-class
 * totals in out[0..n). Returns n, or an error. Synchronous; results are discarded. */
int uad_profile_chunk(uad_ctx* ctx, const float* noise, const uad_schedule* sched,
                      uad_kernel_stat* out, int32_t max_stats, int64_t timeout_us);

/* Testing aid for the bounded waits (not part of the method). Every wait inside the persistent
 * evaluation kernel gives up after wait_ns nanoseconds (> 0; the default is 2 s), records an
 * error code on the device and lets the launch wind down; the next uad_finish then returns
 * UAD_ECUDA, and the context stays usable. unreachable > 0 makes the first completion count of
 * every evaluation wait for that many arrivals more than the kernel ever makes, so that the
 * wait is sure to run out (0 restores normal operation). Applies to chunks started afterwards
 * (cached graphs are rebuilt), and re-enables the persistent kernel after a fall-back (see
 * uad_finish). Returns UAD_OK, UAD_EINVAL or UAD_ESTATE (chunk in flight). */
int uad_set_wait_limit(uad_ctx* ctx, int64_t wait_ns, int32_t unreachable);

/* Testing aid (not part of the method): the fp32 rotations that Ghost Action Correction applies
 * on SO(3) (App. C.1; Sec. 4.4, Eqs. 8-9), run on the GPU for n rotation vectors w[n][3] (host
 * memory, axis times angle in radians): log_exp[i] = log(exp(w_i)) and
 * log_comp[i] = log(exp(w_i) exp(w_{(i+1) mod n})^T), log giving the principal vector (angle in
 * [0, pi]). Synchronous; allocates its own device memory. Returns UAD_OK, UAD_EINVAL (null
 * pointer, n < 1 or n > 2^20) or UAD_ECUDA. */
int uad_so3_check(const float* w, int32_t n, float* log_exp, float* log_comp);

void uad_destroy(uad_ctx* ctx);
const char* uad_last_error(const uad_ctx* ctx);

/* ---- Host-only helpers (no GPU needed) ------------------------------------------------ */

/* Plan of step k (1-based) for one robot with budgets[H] (Sec. 4.2, Eqs. 4-5; Sec. 4.3, Eq. 7):
 * flags[i] bit 0 = active (k <= N_i: own Euler step 1/N_i), bit 1 = ghost input (early action
 * past its release, fed its reconciled state), bit 2 = released after this step, bit 3 =
 * early (N_i < N*: a TR running sum is kept), bit 4 = frozen input (TR off);
 * tau = tau_num[i] / tau_den[i] (reduced fraction), the flow time fed to the network.
 * Returns N* or UAD_EINVAL. */
int uad_plan_step(const int32_t* budgets, int32_t H, int32_t k, int32_t tr, int32_t* flags,
                  int32_t* tau_num, int32_t* tau_den);

/* Library version string. */
const char* uad_version(void);

/* ---- Kernel-level op: the step loop's tensor-core projection on caller buffers ------------ */

/* Re-lay out one linear weight for the tensor-core projection kernel (host only, no GPU).
 * w: host fp32 [K][N] (y = x w); out: host bf16 bit patterns, N * K values, as 128 x 64 blocks:
 * block (n / 128, k / 64) starts at element ((n / 128) * (K / 64) + k / 64) * 8192; inside it,
 * row n % 128 holds 64 values (128 bytes) whose eight 16-byte groups are permuted by
 * group ^ (n % 8) -- the 128-byte-swizzled K-major shared-memory layout the tensor cores read.
 * Values are rounded to bf16 (nearest, ties to even). Needs N % 128 == 0 and K % 64 == 0.
 * Returns UAD_OK or UAD_EINVAL. */
int uad_tile_weight(const float* w, int32_t K, int32_t N, uint16_t* out);

/* out[M][N] = x[M][K] w + bias on the tensor cores (tcgen05, bf16 operands, fp32 accumulation):
 * the projection kernel of every velocity-network layer (Sec. 3, Eq. 1).
 * x: device bf16 [M][K]; w_tiled: device, the layout of uad_tile_weight; bias: device fp32 [N]
 * or NULL; out: device fp32 [M][N]. Needs N % 128 == 0, K % 64 == 0, M >= 1.
 * Split-K scratch (an fp32 [M][N] accumulator and per-tile counters) is allocated by the library
 * with cudaMalloc on the first call on each device and grown on demand; it is kept until exit.
 * Asynchronous on `stream` (a cudaStream_t, NULL = legacy stream). Calls on one device must not
 * overlap on the GPU, since they share that scratch. Returns UAD_OK, UAD_EINVAL, UAD_ENOMEM or
 * UAD_ECUDA. */
int uad_linear(const void* x, const void* w_tiled, const float* bias, float* out, int32_t M,
               int32_t N, int32_t K, void* stream);

/* ---- The same projection op for callers that cannot allocate device memory ---------------
 * The paper has no counterpart: this serves deployments rather than the method. A real-time
 * controller that has finished start-up must not block on cudaMalloc (it can take unbounded
 * time and synchronize the device, stalling the control loop), and a host framework whose
 * caching allocator already holds the GPU's memory cannot take a stray allocation. This entry
 * point computes exactly what uad_linear computes but allocates nothing: no cudaMalloc,
 * cudaFree or allocating library call. Its split-K scratch is a fixed array inside the
 * library's device image (about 4 MiB), held by every GPU that loads the library until exit.
 *   - Limits: M * N <= UAD_LINEAR_STATIC_MAX_ELEMS and (N / 128) * ceil(M / 64) <=
 *     UAD_LINEAR_STATIC_MAX_TILES; larger calls return UAD_ETOOBIG and launch nothing.
 *   - The first call on a device looks up the array's device address (cudaGetSymbolAddress,
 *     which may load the library's device code: with lazy module loading, the CUDA default,
 *     the driver reserves the array only then). Make one warm-up call per device during
 *     start-up, before any stream capture begins and before the control loop runs, so that
 *     the device code and its array are resident when "allocates nothing" matters.
 *   - Every call on a device shares the one array and it keeps the previous call's contents:
 *     each call clears the part it uses (asynchronously, on `stream`) before its kernel.
 *     Calls whose work overlaps on the GPU (different streams, or threads racing) corrupt
 *     each other's results; order them on one stream.
 * Arguments, layout and other errors are those of uad_linear. */
#define UAD_ETOOBIG (-7)
#define UAD_LINEAR_STATIC_MAX_ELEMS (1 << 20)
#define UAD_LINEAR_STATIC_MAX_TILES 4096
int uad_linear_static_scratch(const void* x, const void* w_tiled, const float* bias, float* out,
                              int32_t M, int32_t N, int32_t K, void* stream);

#ifdef __cplusplus
}
#endif
#endif /* UAD_H */
