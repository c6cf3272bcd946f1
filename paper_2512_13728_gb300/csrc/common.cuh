// Internal declarations shared by the kernels and the host runtime of the CurvaDion library.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>
#include <cuda_bf16.h>

struct dion_plan;

namespace cd {

// Step-sequence timing hooks (plan.cu): no-ops unless dion_timing_enable was called.
void tick_begin(dion_plan *p, cudaStream_t s);
void tick(dion_plan *p, cudaStream_t s, const char *name);
void tick_end(dion_plan *p);

// Status codes mirror dion_status in include/curvadion.h.
enum : int32_t {
  ST_OK = 0,
  ST_BREAKDOWN = 5,
  ST_NONFINITE = 6,
  ST_TIMEOUT = 7,
  ST_CORRUPT = 8,
};

// Workspace guards: every region carved from a plan's workspace is followed by kGuardWords
// 32-bit words of a fixed pattern (guard_fill), checked by guard_check.
constexpr int kGuardWords = 64;
void launch_guard_fill(char *base, const uint64_t *offsets, int32_t n, cudaStream_t s);
// Counts damaged guard words into *bad (device) and, when status is not null, sets ST_CORRUPT there.
void launch_guard_check(const char *base, const uint64_t *offsets, int32_t n, int32_t *bad, int32_t *status,
                        cudaStream_t s);

// DION_DEBUG_CHECKS builds check every tile a kernel decodes against its layer's shape; a bad
// tile sets ST_CORRUPT and the block returns.  Other builds compile the checks away.
#ifdef DION_DEBUG_CHECKS
#define DION_TILE_CHECK(cond, status)        \
  do {                                       \
    if (!(cond)) {                           \
      atomicCAS((status), 0, (int32_t)ST_CORRUPT); \
      return;                                \
    }                                        \
  } while (0)
#else
#define DION_TILE_CHECK(cond, status) \
  do {                                \
  } while (0)
#endif

enum : int32_t { GATE_ALWAYS = 0, GATE_GLOBAL = 1, GATE_PER_LAYER = 2, GATE_SCHEDULED = 3 };
enum : int32_t { DT_FP32 = 0, DT_BF16 = 1 };
enum : int32_t { PREC_FP32 = 0, PREC_BF16 = 1, PREC_BF16X3 = 2 };

// One layer as the kernels see it: the caller's tensors plus this layer's workspace.
struct DevLayer {
  int64_t m, n, r;
  float *X;
  int64_t ldx;
  float *M;  // holds B = M + G between the buffer kernel and the update kernel (unless b_deferred)
  int64_t ldm;
  float *Q;
  int64_t ldq;
  const void *G;
  int64_t ldg;
  int32_t g_dtype;
  float tau;
  float sqrt_m_over_n;
  int32_t ldp;  // leading dimension of P_raw, P, R (r rounded up to a multiple of 8)
  // workspace (row-major)
  float *P_raw;  // m x r (ld ldp)  P = B Q before orthogonalization
  float *P;      // m x r (ld ldp)  orthonormal P
  float *R;      // n x r (ld ldp)  R = B^T P
  float *S;      // r x r (ld ldp)  Gram X^T X; lower triangle becomes the Cholesky factor L
  float *Linv;   // r x r (ld ldp)  L^{-1} (lower triangular, zeros above the diagonal)
  // tensor-core operand copies (bf16, rows of pitch ldp unless stated); null in FP32 mode
  __nv_bfloat16 *P_hi;   // m x r : P
  __nv_bfloat16 *R_hi;   // n x r : R
  __nv_bfloat16 *Qn_hi;  // n x r : Q (Q_{t-1} when a step starts, Q_t after a sync step)
  __nv_bfloat16 *Bh;     // m x n, pitch ldbh : B rounded to bf16
  int64_t ldbh;
  // BF16X3 low halves (x - bf16(x), rounded to bf16), same layouts as the copies above; null
  // in the other modes
  __nv_bfloat16 *Bl, *P_lo, *R_lo, *Qn_lo;
  float *PT_raw, *PT;    // r x m, pitch ldmt : transposed copies of P_raw and P (tensor-core Gram)
  int64_t ldmt;
  double *colsq;         // [row tiles of R][ldp]: per-tile column sums of squares of R
  float *colinv;         // [ldp]: 1 / (||R[:, j]|| + eps_col)
  int32_t rtile_cnt;
  // 1: the buffer pass leaves M_{t-1} in place (it writes only the norms and the bf16 copy of B),
  // and the update or the local branch forms B = M + G itself (tensor-core mode, bf16 G)
  int32_t b_deferred;
  int32_t bpart_off, bpart_cnt;  // slots of the ||B||^2 / ||M_{t-1}||^2 partials
  int32_t upart_off, upart_cnt;  // slots of the ||M_t||^2 partials
};

// Per-step scalars and output pointers, passed by value to the kernels.
struct StepArgs {
  float mu, eta, eta_local, eps_rmmc, eps_col, tau_global;
  float keep_sync, keep_local;  // decoupled weight decay: X scaled by 1 - lr * weight_decay
  int32_t gate_mode, period;
  int64_t step;
  double *prev_norm;
  double *rmmc;
  double *eq1;  // may be null
  uint8_t *flags;
  uint8_t *gflag;
};

// Workspace shared by all kernels of a plan.
constexpr int kScratchActive = 3;   // gate_scratch slot holding the count of Dion-branch layers
constexpr int kScratchShifted = 4;  // gate_scratch slot: layers whose Cholesky took the shifted retry
constexpr int kScratchSlots = 8;
struct Shared {
  DevLayer *layers;
  int32_t num_layers;
  uint8_t *active;       // [L] 1 = layer takes the Dion branch this step
  double *bpart;         // [2 * row tiles] per tile: sum B^2, sum M_{t-1}^2
  double *upart;         // [update tiles]  per tile: sum M_t^2
  double *norm_m_before; // [L]
  double *norm_b;        // [L]
  int32_t *status;       // [1] first device error
  uint8_t *orth_shifted; // [L] 1 = a Cholesky pass of this step needed the shift (third pass runs)
  // [kScratchSlots]: the gate's running max of RMMC (ordered key), its finished-block count, the
  // norms pass's finished-block count, (written by the gate) the number of layers that take the
  // Dion branch this step, which lets the later persistent kernels return at once when it is 0,
  // and (reset by the gate, counted by the Cholesky kernels) the layers that took the shifted
  // retry, which lets the third CholeskyQR pass return at once when it is 0
  unsigned long long *gate_scratch;
  // 1 when this step's norms pass has already written B = M + G into M (gated modes with bf16
  // gradients): the fused kernel and the update then read B from M without G, and the local
  // branch leaves M alone
  int32_t b_in_m;
  // limit of the update kernel's hand-off waits between its roles (dion_plan_set_wait_limit)
  uint64_t handoff_limit_ns;
};

// A contraction C = op(A) op(B) for the CUDA-core path.
// op(A)[i][k] = transA ? A[k*lda + i] : A[i*lda + k]   (i < Mrows, k < K)
// op(B)[k][j] = transB ? B[j*ldb + k] : B[k*ldb + j]   (k < K, j < Ncols)
// mode: GEMM_ACTIVE runs on active layers; GEMM_SHIFTED only where orth_shifted is set;
// GEMM_SHIFTED_OR_COPY multiplies where orth_shifted is set and copies A to C elsewhere.
enum : int32_t { GEMM_ACTIVE = 0, GEMM_SHIFTED = 1, GEMM_SHIFTED_OR_COPY = 2 };
constexpr int kGemmTile = 128;  // output tile edge of the CUDA-core grouped GEMM
constexpr int kUpdTileM = 128, kUpdTileN = 64;  // output tile of the CUDA-core update (FP32 mode)
struct GemmProblem {
  const float *A;
  const float *B;
  float *C;
  int64_t Mrows, Ncols, K, lda, ldb, ldc;
  int32_t transA, transB, layer, mode;
};

__device__ __forceinline__ void set_status(int32_t *st, int32_t code) { atomicCAS(st, 0, code); }

__device__ __forceinline__ float bf16_bits_to_float(uint32_t bits16) {
  return __uint_as_float(bits16 << 16);
}

// Deterministic block sum of one double per thread (fixed shuffle tree + fixed warp order).
template <int THREADS>
__device__ __forceinline__ double block_sum(double v, double *red /* >= THREADS/32 */) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) red[warp] = v;
  __syncthreads();
  double s = 0.0;
  if (threadIdx.x == 0) {
    for (int w = 0; w < THREADS / 32; ++w) s += red[w];
  }
  __syncthreads();
  return s;  // valid in thread 0
}

// ---------------------------------------------------------------- launch wrappers ---
// CUDA-core (fp32) kernels, kernels_simt.cu
void launch_form_b(const Shared &sh, const int4 *tiles, int32_t ntiles, cudaStream_t s, bool halves = true);
void launch_split_b(const Shared &sh, const int4 *tiles, int32_t ntiles, bool needed, cudaStream_t s);
void launch_gate(const Shared &sh, const StepArgs &a, cudaStream_t s);
// the branch from RMMC values already in a.rmmc (reduced over data-parallel workers)
void launch_gate_reduced(const Shared &sh, const StepArgs &a, cudaStream_t s);
void launch_gemm(const Shared &sh, const GemmProblem *probs, const int4 *tiles, int32_t ntiles,
                 cudaStream_t s);
cudaError_t prepare_chol_inv(int32_t max_r, size_t *smem_out);
// near_identity: Frobenius bound on S - I below which passes 1 and 2 use the first-order factor
void launch_chol_inv(const Shared &sh, size_t smem, int32_t pass, float near_identity, cudaStream_t s);
// the first CholeskyQR pass with the trailing update on tensor cores (chol_tc.cu, BF16 mode)
cudaError_t prepare_chol_inv_tc(int32_t max_r, size_t *smem_out);
namespace tc { struct LayerMaps; }
void launch_chol_inv_tc(const Shared &sh, const tc::LayerMaps *maps, size_t smem, cudaStream_t s);
void launch_colnorm(const Shared &sh, const int4 *tiles, int32_t ntiles, float eps_col,
                    cudaStream_t s);
void launch_update(const Shared &sh, const int4 *tiles, int32_t ntiles, float mu, float eta, float keep,
                   cudaStream_t s);
void launch_norms_gate(const Shared &sh, const StepArgs &a, const int4 *tiles, int32_t ntiles, cudaStream_t s);
void launch_local(const Shared &sh, const int4 *tiles, int32_t ntiles, float eta_local, float keep,
                  cudaStream_t s);
void launch_finalize(const Shared &sh, const StepArgs &a, cudaStream_t s);

}  // namespace cd
