/*
 * curvadion.h -- C ABI of the GB300 CurvaDion optimizer-step library.
 *
 * One call, dion_step(), runs one optimizer step of CurvaDion (arXiv 2512.13728) over a
 * stack of matrix layers that live in GPU memory:
 *
 *   for every layer l (Algorithm 2):
 *     B      = M + G                                   buffer ("update buffer" line)
 *     RMMC_l = | ||B|| - prev_norm_l | / (prev_norm_l + eps_rmmc),  prev_norm_l = ||B||
 *   g = max_l RMMC_l  (the AllReduce_max over one worker)
 *   per layer, if it synchronizes (Algorithm 1's body):
 *     P = B Q;  P = Orthogonalize(P);  R = B^T P
 *     M = B - (1 - mu) P R^T;  Q = ColumnNormalize(R);  X = X - eta sqrt(m/n) P Q^T
 *   otherwise (Algorithm 2's local branch):
 *     M = B;  X = X - eta_local G
 *
 * On one GPU the data-parallel AllReduce lines of Algorithms 1 and 2 are the identity and
 * no collective is issued.  Norms are Frobenius norms.  Orthogonalize returns the Q factor
 * of the thin QR of P with a positive-diagonal triangular factor (computed by Cholesky QR,
 * which gives that factor for full-rank P).  ColumnNormalize divides column j of R by
 * (||R[:, j]||_2 + eps_col).
 *
 * Conventions for every entry point:
 *   - All matrices are row-major.  "ld" arguments are leading dimensions in ELEMENTS.
 *   - Tensor pointers are DEVICE pointers owned by the caller; the library never frees them.
 *   - A host-detectable error returns a status != DION_OK and enqueues no work.
 *   - A device-detected error (see dion_get_device_status) leaves the affected layer's
 *     outputs unspecified; the other layers are still updated.
 *   - dion_step only enqueues work on the given stream: it never blocks the host and
 *     never allocates.  One plan must not be used on two streams at the same time.
 */
#ifndef CURVADION_H
#define CURVADION_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define DION_ABI_VERSION 3

typedef enum {
  DION_OK = 0,
  DION_ERR_INVALID_ARG = 1,  /* NULL pointer, bad size, r > min(m, n), unknown enum */
  DION_ERR_UNSUPPORTED = 2,  /* valid request outside the library's limits (e.g. r > 512) */
  DION_ERR_ALIGNMENT = 3,    /* pointer or leading dimension breaks the 16-byte rule */
  DION_ERR_CUDA = 4,         /* a CUDA runtime call failed (no device, launch error, OOM) */
  DION_ERR_BREAKDOWN = 5,    /* device: Cholesky pivot <= 0 or non-finite (rank-deficient P) */
  DION_ERR_NONFINITE = 6,    /* device: ||B|| is not finite for some layer */
  DION_ERR_TIMEOUT = 7,      /* device: a bounded wait gave up */
  DION_ERR_CORRUPT = 8       /* device: a workspace guard was overwritten, or (debug build) a
                              * kernel was given a tile outside its layer */
} dion_status;

/* Which layers run the synchronized Dion branch (Algorithm 1 body) in a step. */
enum {
  DION_GATE_ALWAYS = 0,     /* Algorithm 1: every layer, every step; RMMC/flags only reported */
  DION_GATE_GLOBAL = 1,     /* Algorithm 2: all layers iff max_l RMMC_l > tau_global */
  DION_GATE_PER_LAYER = 2,  /* layer l iff RMMC_l > tau_l */
  DION_GATE_SCHEDULED = 3   /* Scheduled Sync Dion (Section 4.3): all layers iff step % period == 0 */
};

/* Element type of a gradient buffer G. */
enum { DION_DTYPE_FP32 = 0, DION_DTYPE_BF16 = 1 };

/* Arithmetic of the contractions (B Q, Gram, triangular solve, B^T P, P R^T, P Q^T).
 * Every mode accumulates in fp32 and keeps M, X, Q in fp32.
 *   DION_PREC_FP32   : fp32 operands on CUDA cores (FFMA).
 *   DION_PREC_BF16   : bf16 operands on tcgen05 tensor cores, fp32 accumulators in TMEM; the
 *                      Gram and triangular solve of Orthogonalize as tf32 on tensor cores.
 *   DION_PREC_BF16X3 : B Q, B^T P, P R^T and P Q^T on tcgen05 with each operand split as a high
 *                      and a low bf16 half (x ~ hi + lo, |x - hi - lo| <= 2^-18 |x|) and three
 *                      products per step (hi*hi + hi*lo + lo*hi); Orthogonalize's Gram and
 *                      triangular solves on tcgen05 kind::tf32 with fp32 operands split the same
 *                      way into tf32 halves (3xTF32), the first Cholesky's trailing update
 *                      likewise, the rest of the Cholesky in fp32 on CUDA cores:
 *                      fp32-class accuracy for ill-conditioned P.  Ranks up to 256
 *                      (dion_plan_create returns DION_ERR_UNSUPPORTED above). */
enum { DION_PREC_FP32 = 0, DION_PREC_BF16 = 1, DION_PREC_BF16X3 = 2 };

/* Largest supported rank r (one 128 x r fp32 accumulator fills the 512 TMEM columns). */
#define DION_MAX_RANK 512

/* One matrix layer.  X, M: m x n fp32; Q: n x r fp32; G: m x n of g_dtype.
 * Pointers must be 16-byte aligned and ld * sizeof(element) a multiple of 16 bytes;
 * ld >= number of columns.  1 <= r <= min(m, n).  The pointers are captured by
 * dion_plan_create and must stay valid (and unchanged) for the plan's lifetime:
 * the caller writes each step's gradient into the same G buffer. */
typedef struct {
  int64_t m, n, r;
  float *X;        int64_t ldx;  /* parameters, in/out */
  float *M;        int64_t ldm;  /* momentum, in/out; M_0 = 0 (Algorithm 2 initialization) */
  float *Q;        int64_t ldq;  /* right factor Q_{t-1} in, Q_t out (unchanged on local steps) */
  const void *G;   int64_t ldg;  /* gradient, read only */
  int32_t g_dtype;               /* DION_DTYPE_* */
  float tau;                     /* per-layer threshold for DION_GATE_PER_LAYER */
} dion_layer;

/* Per-step scalars.  Passed by value into the kernels: changing eta every step (a learning
 * rate schedule) costs nothing. */
typedef struct {
  float mu;          /* momentum (paper: 0.95) */
  float eta;         /* learning rate of the Dion update */
  float eta_local;   /* learning rate of the local branch */
  float eps_rmmc;    /* epsilon of Algorithm 2's RMMC denominator (and Equation 1's) */
  float eps_col;     /* epsilon of ColumnNormalize */
  float tau_global;  /* threshold on max_l RMMC_l */
  int32_t gate_mode; /* DION_GATE_* */
  int32_t period;    /* H of DION_GATE_SCHEDULED (>= 1) */
  int64_t step;      /* 1-based step index t */
  float weight_decay; /* decoupled weight decay (Section 4 trains with 0.01; 0 = Algorithms 1/2 as
                       * printed): X is multiplied by (1 - lr * weight_decay) before the branch's
                       * update, lr = eta in the Dion branch and eta_local in the local branch.
                       * Must be finite and >= 0. */
} dion_hparams;

typedef struct dion_plan dion_plan;

/* Validates the layers, allocates the plan's device workspace (P, R, Gram and factor
 * buffers, norm partials, tile lists, status word) on the current CUDA device and stores
 * the layer pointers.  precision: DION_PREC_*.  On success *out owns the workspace until
 * dion_plan_destroy.  Errors: INVALID_ARG, ALIGNMENT, UNSUPPORTED, CUDA (allocation). */
dion_status dion_plan_create(const dion_layer *layers, int32_t num_layers, int32_t precision,
                             dion_plan **out);

/* Enqueues one step on `stream` (a cudaStream_t; NULL = legacy default stream).
 *   prev_norm       device double[L], in/out: Algorithm 2's prev_norm_l (start at 0)
 *   rmmc_out        device double[L], out: Algorithm 2's RMMC_l of this step
 *   rmmc_eq1_out    device double[L] or NULL, out: Equation 1's RMMC from ||M_t||, ||M_{t-1}||
 *                   (with eps_rmmc added to the denominator)
 *   sync_flags_out  device uint8[L], out: 1 iff RMMC_l > tau_l (non-finite counts as above)
 *   global_flag_out device uint8[1], out: 1 iff max_l RMMC_l > tau_global
 * Which layers take the Dion branch follows hp->gate_mode; the decision is made on the
 * device, so the host never waits.  Errors: INVALID_ARG, CUDA (launch failure). */
dion_status dion_step(dion_plan *plan, const dion_hparams *hp, double *prev_norm,
                      double *rmmc_out, double *rmmc_eq1_out, uint8_t *sync_flags_out,
                      uint8_t *global_flag_out, void *stream);

/* Data-parallel steps (Algorithm 2 with W workers, one plan per worker; no collective is
 * issued by the library).  Algorithm 2 reduces across workers at three points: the maximum of
 * RMMC before the branch (the AllReduce_max), P after PowerIter and R after it is formed from
 * the orthonormal P (the AllReduce_DP lines, read as the mean over the workers).
 * dion_step_phase runs one step as four phases, in order, on `stream`; between them the caller
 * performs the reductions on device buffers (with NCCL, or any other means), on the same stream
 * or ordered after it:
 *   DION_PHASE_NORMS   B = M + G (written into M), ||B|| and this worker's RMMC_l into rmmc_out,
 *                      prev_norm_l = ||B|| (each worker keeps its own prev_norm).
 *                      Then: rmmc_out <- elementwise max over the workers.
 *   DION_PHASE_POWER   sync flags, global flag and branch from the reduced rmmc_out (final
 *                      values of those outputs), then P = B Q on the layers that synchronize.
 *                      Then: the P range of dion_plan_exchange <- mean over the workers.
 *   DION_PHASE_ORTHO   P = Orthogonalize(mean P), R = B^T P on the synchronizing layers.
 *                      Then: the R range <- mean over the workers.
 *   DION_PHASE_UPDATE  Q_t = ColumnNormalize(mean R), M = B - (1 - mu) P R^T (this worker's B),
 *                      X = X - eta sqrt(m/n) P Q_t^T; local layers: X = X - eta_local G.
 * Every phase takes the same hp and output pointers as dion_step.  A layer that stays local
 * leaves stale values in its part of the exchange ranges; averaging them is harmless, and a
 * caller that wants to skip the exchanges of a step with no synchronizing layer reads
 * global_flag_out / sync_flags_out after DION_PHASE_POWER.  Workers' plans must have the same
 * layer shapes and precision and the same Q at the start (as Algorithm 2's identical Q_t);
 * their exchange ranges then line up element for element.  With one worker the reductions are
 * the identity and the four phases compute what dion_step computes.  Errors: as dion_step, and
 * INVALID_ARG for a phase out of order (dion_step and dion_step_host are refused while a phased
 * step is unfinished). */
enum { DION_PHASE_NORMS = 1, DION_PHASE_POWER = 2, DION_PHASE_ORTHO = 3, DION_PHASE_UPDATE = 4 };
dion_status dion_step_phase(dion_plan *plan, int32_t phase, const dion_hparams *hp, double *prev_norm,
                            double *rmmc_out, double *rmmc_eq1_out, uint8_t *sync_flags_out,
                            uint8_t *global_flag_out, void *stream);
/* The device range a worker reduces after `phase`: DION_PHASE_POWER gives P (every layer's m x r
 * fp32 P, rows padded to a multiple of 8 floats, layers one after another with small zeroed
 * gaps), DION_PHASE_ORTHO gives R (n x r per layer, the same layout).  *buf_out (device, owned
 * by the plan) and *count_out (fp32 elements) are fixed for the plan's lifetime.  Errors:
 * INVALID_ARG (NULL argument, other phase). */
dion_status dion_plan_exchange(dion_plan *plan, int32_t phase, float **buf_out, int64_t *count_out);

/* Gradients from host memory (no counterpart in the paper: it moves Algorithm 1's input G_t
 * onto the device).  dion_plan_enable_host_gradients allocates, once, two device gradient
 * buffers per layer (the layer's g_dtype, rows padded to 16 bytes: 2 x sum m n x 2 or 4
 * bytes), a copy stream and four events; the G pointers given to dion_plan_create are no
 * longer read by dion_step_host (dion_step still reads them).  Calling it again is a no-op.
 * Errors: INVALID_ARG (NULL plan), CUDA (allocation).
 *
 * dion_step_host is dion_step with layer l's G_t read from host memory: host_G[l] points to
 * m x n elements of the layer's g_dtype, row-major with leading dimension host_ldg[l] >= n
 * (elements).  Consecutive calls alternate between the two device buffers.  The copies of
 * this call go on the plan's copy stream, which waits only for the step two calls back (the
 * last reader of the same buffer), so they overlap the previous step's kernels; the step is
 * then enqueued on `stream` behind the copies.  Outputs and errors as dion_step.  The host
 * memory should be page-locked (cudaHostAlloc / cudaHostRegister) for the copies to run
 * asynchronously, and must not change until they have executed, i.e. until `stream` has
 * passed this step's first kernel (synchronizing `stream` after the call is enough).
 * Errors also: INVALID_ARG when host gradients were not enabled or a pointer or leading
 * dimension is invalid. */
dion_status dion_plan_enable_host_gradients(dion_plan *plan);
dion_status dion_step_host(dion_plan *plan, const dion_hparams *hp, const void *const *host_G,
                           const int64_t *host_ldg, double *prev_norm, double *rmmc_out,
                           double *rmmc_eq1_out, uint8_t *sync_flags_out, uint8_t *global_flag_out,
                           void *stream);

/* Host helpers for the training loop of Section 4 (no device work, callable without a GPU).
 * dion_lr_schedule: learning rate at 1-based `step` of a `total_steps` run with linear warmup
 * and warmdown (Section 4: 1% warmup, 10% or 20% warmdown): with W = warmup_frac T and
 * D = warmdown_frac T rounded half up, base_lr * step / W for step <= W, base_lr * (T - step) / D for
 * step > T - D (0 at the last step), base_lr otherwise; step is clamped to [1, T].  Returns
 * NaN for total_steps < 1, fractions outside [0, 1] or warmup + warmdown steps > T.
 * dion_rank_for: Dion rank for a rank fraction (Section 4: 0.125): ceil(fraction min(m, n)),
 * clamped to [1, min(m, n)]; returns 0 for m < 1, n < 1 or fraction outside (0, 1]. */
float dion_lr_schedule(int64_t step, int64_t total_steps, float base_lr, float warmup_frac, float warmdown_frac);
int64_t dion_rank_for(int64_t m, int64_t n, double fraction);

/* Reads the plan's device status word (synchronously; call after the step's stream has
 * been synchronized) into *code_out as a dion_status, and clears it if `clear` != 0.
 * The first device error of any step since the last clear is kept. */
dion_status dion_get_device_status(dion_plan *plan, int32_t clear, int32_t *code_out);

/* The tensor-core modes keep a bf16 copy of every layer's Q (made by dion_plan_create and
 * updated by each step that writes Q).  A caller that writes Q itself between steps (for
 * example when restoring a checkpoint) calls dion_plan_refresh before the next dion_step;
 * it enqueues the re-copy on `stream` and allocates nothing.  No-op in DION_PREC_FP32.
 * Errors: INVALID_ARG (NULL plan), CUDA. */
dion_status dion_plan_refresh(dion_plan *plan, void *stream);

/* Number of kernel launches one dion_step enqueues for this plan. */
int32_t dion_step_launch_count(const dion_plan *plan);

/* Per-launch timing with CUDA events (measurement support; not part of the paper's method).
 * dion_timing_enable(plan, max_steps): while max_steps > 0, every dion_step records one CUDA
 * event before its first launch and one after each launch, on the step's stream, for up to
 * max_steps steps (events are created here, so this call may allocate; dion_step does not).
 * max_steps = 0 disables timing and frees the events.
 * dion_timing_read(plan, cap, ms_out, names_out, count_out): synchronizes on the recorded
 * events, writes the average duration in milliseconds of each launch position over the
 * recorded steps (ms_out[i], names_out[i] = static kernel name) for i < min(cap, launches),
 * sets *count_out to the number of launches per step and to 0 steps recorded afterwards.
 * Errors: INVALID_ARG (NULL plan/outputs), CUDA. */
dion_status dion_timing_enable(dion_plan *plan, int32_t max_steps);
dion_status dion_timing_read(dion_plan *plan, int32_t cap, float *ms_out, const char **names_out,
                             int32_t *count_out, int32_t *steps_out);

/* Limits of dion_buffer_norms_noalloc.  Its fixed device scratch holds two doubles per tile,
 * 1 MB per GPU; a tile is whole rows of about 64K elements of one layer. */
#define DION_NOALLOC_MAX_LAYERS 256
#define DION_NOALLOC_MAX_TILES 65536

/* The buffer step without any allocation.  The paper has no counterpart: this entry point is
 * for callers that cannot call cudaMalloc -- a framework whose caching allocator has reserved
 * the device memory up front and owns every byte of it, or a latency-critical loop in which a
 * cudaMalloc or cudaFree would synchronize the device -- and so cannot hold a plan, whose
 * workspace dion_plan_create allocates.
 * For each layer it adds G into M in place (M = M + G, the buffer that dion_step forms) and
 * writes two Frobenius norms: norm_b_out[l] = ||M + G|| (the new M) and norm_m_out[l] = ||M||
 * (M as it was before the call).  Only m, n, M, ldm, G, ldg and g_dtype of each layer are used,
 * with the same rules as in dion_layer.  norm_b_out, norm_m_out: device double[num_layers],
 * written.  The work is enqueued on `stream` (a cudaStream_t; NULL = legacy default stream).
 * Scratch: one fixed array of per-tile partial sums inside this library, in device memory,
 * held by every GPU that loads the library until the process exits.  Every call shares it and
 * it keeps the last call's contents; each call writes every slot it reads before reading it,
 * so nothing needs clearing, but calls whose work overlaps on the GPU (two streams, or two host
 * threads) race on it: serialize them.  The first call on a device (and the first after a
 * cudaDeviceReset) looks up the array's device address with cudaGetSymbolAddress; make that
 * first call before any stream capture.  The layer table is passed to the kernels as a kernel
 * parameter, so no host-to-device copy is made.  No device or host memory is allocated.
 * Errors: INVALID_ARG, ALIGNMENT, UNSUPPORTED (num_layers > DION_NOALLOC_MAX_LAYERS, or the
 * layers need more than DION_NOALLOC_MAX_TILES tiles; nothing is enqueued then), CUDA (the
 * address lookup or a launch failed). */
dion_status dion_buffer_norms_noalloc(const dion_layer *layers, int32_t num_layers, double *norm_b_out,
                                      double *norm_m_out, void *stream);

/* Bounded device waits (failure detection; no counterpart in the paper).  Every wait of a
 * tensor-core kernel on another role of the same CTA (a TMA load landing, an MMA finishing, an
 * accumulator being drained) gives up after a limit, sets DION_ERR_TIMEOUT in the plan's status
 * word and lets the kernel drain what it already issued and return; the step's later kernels
 * still run, and the layers the kernel did not finish have unspecified outputs.
 * dion_plan_set_wait_limit sets that limit, in nanoseconds, for the hand-off waits of the
 * update kernel (error feedback and parameter update) of this plan; limit_ns <= 0 restores the
 * default of 2 s.  The waits that drain copies and MMAs already in flight keep the default, so
 * the kernel never exits with work in flight.  Meant for testing the timeout path: with a limit
 * of a few nanoseconds the first wait that does not succeed at once gives up.  Host only;
 * takes effect from the next dion_step.  Errors: INVALID_ARG (NULL plan). */
dion_status dion_plan_set_wait_limit(dion_plan *plan, int64_t limit_ns);

/* Workspace guards (memory-safety check; no counterpart in the paper).  Every region the plan
 * carves from its workspace is followed by 64 guard words of a fixed pattern, written at
 * creation.  dion_plan_check_guards synchronizes the device, counts the guard words that no
 * longer hold their pattern into *damaged_out (0 when no kernel wrote past a region) and
 * changes nothing.  Errors: INVALID_ARG (NULL argument), CUDA.
 * A library built with DION_DEBUG_CHECKS (dion_debug_checks() returns 1; built as
 * libcurvadion_debug.so) also checks the guards at the end of every step and checks every tile
 * a kernel decodes against its layer's shape; either failure sets DION_ERR_CORRUPT in the
 * status word, and a bad tile is skipped.  Such a step launches one more kernel. */
dion_status dion_plan_check_guards(dion_plan *plan, int32_t *damaged_out);
int32_t dion_debug_checks(void);

/* Frees the plan's workspace (synchronizes the device first).  NULL is a no-op. */
void dion_plan_destroy(dion_plan *plan);

/* Static description of a status code. */
const char *dion_status_string(dion_status status);

/* DION_ABI_VERSION of the loaded library. */
int32_t dion_abi_version(void);

#ifdef __cplusplus
}
#endif

#endif /* CURVADION_H */
