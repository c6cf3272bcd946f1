// Host runtime and C ABI of the CurvaDion library: plan creation (validation, workspace,
// tile lists), the per-step launch sequence, device status and teardown.
#include "../../include/curvadion.h"
#include "common.cuh"
#include "tc.cuh"

#include <algorithm>
#include <cmath>
#include <cstring>
#include <new>
#include <vector>

using namespace cd;

struct dion_plan {
  int device = 0;
  int32_t L = 0;
  int32_t precision = PREC_FP32;
  int32_t max_r = 0;
  int num_sms = 0;
  void *ws = nullptr;  // one device allocation holding everything below
  Shared sh{};
  // tile lists (device)
  int4 *btiles = nullptr;
  int32_t n_btiles = 0;  // buffer / local row tiles
  int4 *utiles = nullptr;
  int32_t n_utiles = 0;  // update tiles
  int4 *ctiles = nullptr;
  int32_t n_ctiles = 0;  // column-normalization tiles
  static constexpr int kSets = 8;
  GemmProblem *probs[kSets] = {};
  int4 *gtiles[kSets] = {};
  int32_t n_gtiles[kSets] = {};
  size_t chol_smem = 0;
  tc::TcPlan tcp{};  // tensor-core path (BF16 / BF16X3)
  int32_t launches_per_step = 0;
  // data-parallel phases (dion_step_phase): the exchange ranges (offsets into ws, fp32 counts)
  // and the phase the next call must run
  size_t xp_off = 0, xr_off = 0;
  int64_t xp_count = 0, xr_count = 0;
  int32_t next_phase = DION_PHASE_NORMS;
  // workspace guards (device list of offsets, damaged-word counter)
  uint64_t *guard_off = nullptr;
  int32_t *guard_bad = nullptr;
  int32_t n_guards = 0;
  // per-launch timing (dion_timing_enable)
  std::vector<cudaEvent_t> ev;  // [max_steps][launches + 1]
  std::vector<const char *> names;
  int32_t timing_steps = 0, recorded = 0, cursor = 0;
  // host gradients (dion_step_host): two device gradient buffers per layer, filled in turn
  std::vector<DevLayer> dl_host;  // the layer records as uploaded at creation
  struct HostGrad {
    bool on = false;
    void *mem = nullptr;  // both buffers' gradients, both layer tables, both map tables
    DevLayer *layers[2] = {};
    tc::LayerMaps *maps[2] = {};
    std::vector<char *> g[2];     // per layer device gradient of each buffer
    std::vector<int64_t> ldg;     // their leading dimension (elements)
    cudaStream_t copy = nullptr;
    cudaEvent_t up[2] = {}, used[2] = {};
    int parity = 0;
  } hg;
};

namespace cd {
// Called by the step sequences: records the event that closes launch `cursor` when timing is on.
void tick(dion_plan *p, cudaStream_t s, const char *name) {
  if (p->timing_steps <= 0 || p->recorded >= p->timing_steps) return;
  const int32_t per = p->launches_per_step + 1;
  if (p->cursor < p->launches_per_step) {
    if ((int32_t)p->names.size() < p->launches_per_step) p->names.resize(p->launches_per_step, "");
    p->names[p->cursor] = name;
    cudaEventRecord(p->ev[(size_t)p->recorded * per + p->cursor + 1], s);
  }
  ++p->cursor;
}
void tick_begin(dion_plan *p, cudaStream_t s) {
  p->cursor = 0;
  if (p->timing_steps <= 0 || p->recorded >= p->timing_steps) return;
  cudaEventRecord(p->ev[(size_t)p->recorded * (p->launches_per_step + 1)], s);
}
void tick_end(dion_plan *p) {
  if (p->timing_steps <= 0 || p->recorded >= p->timing_steps) return;
  ++p->recorded;
}
}  // namespace cd

namespace {

constexpr size_t kAlign = 256;
constexpr uint64_t kDefaultWaitLimitNs = 2000000000ull;  // the bounded waits' default: 2 s

// Carves the workspace: 256-byte aligned regions, each followed (unless guard = false) by
// kGuardWords guard words whose offsets are recorded.
struct Carver {
  size_t off = 0;
  std::vector<uint64_t> guards;
  template <class T>
  size_t take(size_t count, bool guard = true) {
    off = (off + kAlign - 1) / kAlign * kAlign;
    const size_t at = off;
    off += count * sizeof(T);
    if (guard) add_guard();
    return at;
  }
  void add_guard() {
    off = (off + 3) / 4 * 4;
    guards.push_back(off);
    off += kGuardWords * sizeof(uint32_t);
  }
};

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

dion_status validate_layer(const dion_layer &ly) {
  if (ly.m < 1 || ly.n < 1 || ly.r < 1) return DION_ERR_INVALID_ARG;
  if (ly.r > std::min(ly.m, ly.n)) return DION_ERR_INVALID_ARG;
  if (ly.r > DION_MAX_RANK) return DION_ERR_UNSUPPORTED;
  if (ly.m > (int64_t(1) << 31) - 1 || ly.n > (int64_t(1) << 31) - 1) return DION_ERR_UNSUPPORTED;
  if (!ly.X || !ly.M || !ly.Q || !ly.G) return DION_ERR_INVALID_ARG;
  if (ly.g_dtype != DION_DTYPE_FP32 && ly.g_dtype != DION_DTYPE_BF16) return DION_ERR_INVALID_ARG;
  if (ly.ldx < ly.n || ly.ldm < ly.n || ly.ldg < ly.n || ly.ldq < ly.r) return DION_ERR_INVALID_ARG;
  if (!std::isfinite(ly.tau)) {
    if (!(ly.tau > 0)) return DION_ERR_INVALID_ARG;  // +inf allowed (never above), NaN/-inf not
  }
  const int64_t gsz = ly.g_dtype == DION_DTYPE_BF16 ? 2 : 4;
  if (!aligned16(ly.X) || !aligned16(ly.M) || !aligned16(ly.Q) || !aligned16(ly.G))
    return DION_ERR_ALIGNMENT;
  if ((ly.ldx * 4) % 16 || (ly.ldm * 4) % 16 || (ly.ldq * 4) % 16 || (ly.ldg * gsz) % 16)
    return DION_ERR_ALIGNMENT;
  return DION_OK;
}

template <class T>
cudaError_t upload(T *dst, const std::vector<T> &src) {
  if (src.empty()) return cudaSuccess;
  return cudaMemcpy(dst, src.data(), src.size() * sizeof(T), cudaMemcpyHostToDevice);
}

}  // namespace

extern "C" {

int32_t dion_abi_version(void) { return DION_ABI_VERSION; }

const char *dion_status_string(dion_status s) {
  switch (s) {
    case DION_OK: return "DION_OK";
    case DION_ERR_INVALID_ARG: return "DION_ERR_INVALID_ARG: invalid argument";
    case DION_ERR_UNSUPPORTED: return "DION_ERR_UNSUPPORTED: outside the library's limits";
    case DION_ERR_ALIGNMENT: return "DION_ERR_ALIGNMENT: pointer or leading dimension not 16-byte aligned";
    case DION_ERR_CUDA: return "DION_ERR_CUDA: CUDA runtime error";
    case DION_ERR_BREAKDOWN: return "DION_ERR_BREAKDOWN: Cholesky breakdown (rank-deficient P)";
    case DION_ERR_NONFINITE: return "DION_ERR_NONFINITE: non-finite buffer norm";
    case DION_ERR_TIMEOUT: return "DION_ERR_TIMEOUT: bounded device wait gave up";
    case DION_ERR_CORRUPT: return "DION_ERR_CORRUPT: workspace guard overwritten or tile out of range";
  }
  return "unknown dion_status";
}

dion_status dion_plan_create(const dion_layer *layers, int32_t num_layers, int32_t precision,
                             dion_plan **out) {
  if (out == nullptr) return DION_ERR_INVALID_ARG;
  *out = nullptr;
  if (num_layers < 0 || (num_layers > 0 && layers == nullptr)) return DION_ERR_INVALID_ARG;
  if (precision != DION_PREC_FP32 && precision != DION_PREC_BF16 && precision != DION_PREC_BF16X3)
    return DION_ERR_INVALID_ARG;
  for (int32_t l = 0; l < num_layers; ++l) {
    const dion_status st = validate_layer(layers[l]);
    if (st != DION_OK) return st;
  }
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return DION_ERR_CUDA;
  int sms = 0;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return DION_ERR_CUDA;

  dion_plan *p = new (std::nothrow) dion_plan();
  if (!p) return DION_ERR_CUDA;
  p->device = dev;
  p->L = num_layers;
  p->precision = precision;
  p->num_sms = sms;

  // ---- host-side layout of the workspace ----
  Carver cv;
  std::vector<DevLayer> dl(num_layers);
  std::vector<size_t> o_Praw(num_layers), o_P(num_layers), o_R(num_layers), o_S(num_layers), o_Li(num_layers);
  std::vector<int4> bt, ut, ct;
  // P_raw and R of all layers each in one contiguous range (256-byte gaps between layers): the
  // buffers a data-parallel caller averages between the phases of dion_step_phase
  // (no guards inside them: a caller's average of equal words is exact, but not every reduction is)
  for (int32_t l = 0; l < num_layers; ++l)
    o_Praw[l] = cv.take<float>(layers[l].m * ((layers[l].r + 7) / 8 * 8), false);
  if (num_layers > 0) cv.add_guard();
  for (int32_t l = 0; l < num_layers; ++l)
    o_R[l] = cv.take<float>(layers[l].n * ((layers[l].r + 7) / 8 * 8), false);
  if (num_layers > 0) cv.add_guard();
  if (num_layers > 0) {
    const dion_layer &a = layers[num_layers - 1];
    const int64_t lp = (a.r + 7) / 8 * 8;
    p->xp_off = o_Praw[0];
    p->xp_count = (int64_t)((o_Praw[num_layers - 1] - o_Praw[0]) / sizeof(float)) + a.m * lp;
    p->xr_off = o_R[0];
    p->xr_count = (int64_t)((o_R[num_layers - 1] - o_R[0]) / sizeof(float)) + a.n * lp;
  }
  for (int32_t l = 0; l < num_layers; ++l) {
    const dion_layer &ly = layers[l];
    DevLayer &d = dl[l];
    std::memset(&d, 0, sizeof(d));
    d.m = ly.m; d.n = ly.n; d.r = ly.r;
    d.X = ly.X; d.ldx = ly.ldx;
    d.M = ly.M; d.ldm = ly.ldm;
    d.Q = ly.Q; d.ldq = ly.ldq;
    d.G = ly.G; d.ldg = ly.ldg; d.g_dtype = ly.g_dtype;
    d.tau = ly.tau;
    d.sqrt_m_over_n = (float)std::sqrt((double)ly.m / (double)ly.n);
    d.ldp = (int32_t)((ly.r + 7) / 8 * 8);
    p->max_r = std::max<int32_t>(p->max_r, (int32_t)ly.r);
    o_P[l] = cv.take<float>(ly.m * d.ldp);
    o_S[l] = cv.take<float>(ly.r * d.ldp);
    o_Li[l] = cv.take<float>(ly.r * d.ldp);
    // row tiles of about 64K elements for the buffer and local kernels
    const int64_t rows = std::max<int64_t>(1, std::min<int64_t>(ly.m, 65536 / ly.n));
    d.bpart_off = (int32_t)bt.size();
    for (int64_t r0 = 0; r0 < ly.m; r0 += rows)
      bt.push_back(make_int4(l, (int)r0, (int)std::min(rows, ly.m - r0), (int)bt.size()));
    d.bpart_cnt = (int32_t)bt.size() - d.bpart_off;
    // update tiles of the CUDA-core update kernel (FP32 mode)
    d.upart_off = (int32_t)ut.size();
    for (int64_t ti = 0; ti < (ly.m + kUpdTileM - 1) / kUpdTileM; ++ti)
      for (int64_t tj = 0; tj < (ly.n + kUpdTileN - 1) / kUpdTileN; ++tj)
        ut.push_back(make_int4(l, (int)ti, (int)tj, (int)ut.size()));
    d.upart_cnt = (int32_t)ut.size() - d.upart_off;
    for (int64_t cg = 0; cg < (ly.r + 31) / 32; ++cg) ct.push_back(make_int4(l, (int)cg, 0, 0));
  }
  // GEMM problem sets of the CUDA-core path:
  //   0     P_raw = B Q
  //   1..3  Gram of pass j:  S = X_j^T X_j        (X_0 = P_raw, X_1 = P, X_2 = P_raw)
  //   4..6  TRSM of pass j:  X_{j+1} = X_j L^{-T}  (X_3 = P); pass 2 only where a shift was needed
  //   7     R = B^T P
  constexpr int kSets = dion_plan::kSets;
  std::vector<GemmProblem> gp[kSets];
  std::vector<int4> gt[kSets];
  const size_t o_layers = cv.take<DevLayer>(std::max(num_layers, 1));
  const size_t o_active = cv.take<uint8_t>(std::max(num_layers, 1));
  // norm-partial slots: one per buffer row tile, or one per 128-row tile when the tensor-core
  // path fuses the buffer pass into B Q
  size_t tile128 = 0;
  for (int32_t l = 0; l < num_layers; ++l) tile128 += (size_t)((layers[l].m + 127) / 128);
  const size_t o_bpart = cv.take<double>(2 * std::max<size_t>(std::max(bt.size(), tile128), 1));
  const size_t o_upart = cv.take<double>(std::max<size_t>(ut.size(), 1));
  const size_t o_nmb = cv.take<double>(std::max(num_layers, 1));
  const size_t o_nb = cv.take<double>(std::max(num_layers, 1));
  const size_t o_status = cv.take<int32_t>(1);
  const size_t o_gate = cv.take<unsigned long long>(kScratchSlots);
  const size_t o_bt = cv.take<int4>(std::max<size_t>(bt.size(), 1));
  const size_t o_ut = cv.take<int4>(std::max<size_t>(ut.size(), 1));
  const size_t o_ct = cv.take<int4>(std::max<size_t>(ct.size(), 1));
  // tensor-core workspace (operand copies, tile lists); sized by the tc module
  tc::TcLayout tcl{};
  if (precision != DION_PREC_FP32) {
    const dion_status st = tc::layout(layers, num_layers, precision, sms, cv.off, &tcl);
    if (st != DION_OK) {
      delete p;
      return st;
    }
    cv.off = tcl.end;
    cv.guards.insert(cv.guards.end(), tcl.guards.begin(), tcl.guards.end());
  }
  const size_t o_shift = cv.take<uint8_t>(std::max(num_layers, 1));
  size_t o_gp[kSets], o_gt[kSets];
  for (int k = 0; k < kSets; ++k) {
    for (int32_t l = 0; l < num_layers; ++l) {
      const dion_layer &ly = layers[l];
      const int64_t ldp = dl[l].ldp;
      GemmProblem q{};
      q.layer = l;
      if (k == 0) {
        q.Mrows = ly.m; q.Ncols = ly.r; q.K = ly.n; q.lda = ly.ldm; q.ldb = ly.ldq; q.ldc = ldp;
      } else if (k <= 3) {
        q.Mrows = ly.r; q.Ncols = ly.r; q.K = ly.m; q.lda = ldp; q.ldb = ldp; q.ldc = ldp; q.transA = 1;
        q.mode = (k == 3) ? GEMM_SHIFTED : GEMM_ACTIVE;
      } else if (k <= 6) {
        q.Mrows = ly.m; q.Ncols = ly.r; q.K = ly.r; q.lda = ldp; q.ldb = ldp; q.ldc = ldp; q.transB = 1;
        // the third solve runs on shifted layers only; it also copies the second pass's result
        // into P for the others
        q.mode = (k == 6) ? GEMM_SHIFTED_OR_COPY : GEMM_ACTIVE;
      } else {
        q.Mrows = ly.n; q.Ncols = ly.r; q.K = ly.m; q.lda = ly.ldm; q.ldb = ldp; q.ldc = ldp; q.transA = 1;
      }
      const int32_t pi = (int32_t)gp[k].size();
      gp[k].push_back(q);
      for (int64_t ti = 0; ti < (q.Mrows + kGemmTile - 1) / kGemmTile; ++ti)
        for (int64_t tj = 0; tj < (q.Ncols + kGemmTile - 1) / kGemmTile; ++tj)
          gt[k].push_back(make_int4(pi, (int)ti, (int)tj, 0));
    }
    o_gp[k] = cv.take<GemmProblem>(std::max<size_t>(gp[k].size(), 1));
    o_gt[k] = cv.take<int4>(std::max<size_t>(gt[k].size(), 1));
  }

  // the guard list itself and the check's counter come last, unguarded
  const size_t o_guards = cv.take<uint64_t>(std::max<size_t>(cv.guards.size(), 1), false);
  const size_t o_gbad = cv.take<int32_t>(1, false);
  p->n_guards = (int32_t)cv.guards.size();
  if (cudaMalloc(&p->ws, cv.off) != cudaSuccess) {
    delete p;
    return DION_ERR_CUDA;
  }
  char *base = static_cast<char *>(p->ws);
  for (int32_t l = 0; l < num_layers; ++l) {
    dl[l].P_raw = reinterpret_cast<float *>(base + o_Praw[l]);
    dl[l].P = reinterpret_cast<float *>(base + o_P[l]);
    dl[l].R = reinterpret_cast<float *>(base + o_R[l]);
    dl[l].S = reinterpret_cast<float *>(base + o_S[l]);
    dl[l].Linv = reinterpret_cast<float *>(base + o_Li[l]);
  }
  if (precision != DION_PREC_FP32) tc::bind(tcl, base, dl.data(), num_layers, &p->tcp);
  for (int k = 0; k < kSets; ++k) {
    for (auto &q : gp[k]) {
      const DevLayer &d = dl[q.layer];
      float *Xs[4] = {d.P_raw, d.P, d.P_raw, d.P};
      if (k == 0) { q.A = d.M; q.B = d.Q; q.C = d.P_raw; }
      else if (k <= 3) { q.A = Xs[k - 1]; q.B = Xs[k - 1]; q.C = d.S; }
      else if (k <= 6) { q.A = Xs[k - 4]; q.B = d.Linv; q.C = Xs[k - 3]; }
      else { q.A = d.M; q.B = d.P; q.C = d.R; }
    }
    p->probs[k] = reinterpret_cast<GemmProblem *>(base + o_gp[k]);
    p->gtiles[k] = reinterpret_cast<int4 *>(base + o_gt[k]);
    p->n_gtiles[k] = (int32_t)gt[k].size();
  }
  p->sh.layers = reinterpret_cast<DevLayer *>(base + o_layers);
  p->sh.num_layers = num_layers;
  p->sh.active = reinterpret_cast<uint8_t *>(base + o_active);
  p->sh.bpart = reinterpret_cast<double *>(base + o_bpart);
  p->sh.upart = reinterpret_cast<double *>(base + o_upart);
  p->sh.norm_m_before = reinterpret_cast<double *>(base + o_nmb);
  p->sh.norm_b = reinterpret_cast<double *>(base + o_nb);
  p->sh.status = reinterpret_cast<int32_t *>(base + o_status);
  p->sh.gate_scratch = reinterpret_cast<unsigned long long *>(base + o_gate);
  p->sh.orth_shifted = reinterpret_cast<uint8_t *>(base + o_shift);
  p->sh.handoff_limit_ns = kDefaultWaitLimitNs;
  p->btiles = reinterpret_cast<int4 *>(base + o_bt);
  p->n_btiles = (int32_t)bt.size();
  p->utiles = reinterpret_cast<int4 *>(base + o_ut);
  p->n_utiles = (int32_t)ut.size();
  p->ctiles = reinterpret_cast<int4 *>(base + o_ct);
  p->n_ctiles = (int32_t)ct.size();

  // zeroed once, so the gaps and row padding inside the exchange ranges hold zeros
  cudaError_t e = cudaMemset(p->ws, 0, cv.off);
  p->guard_off = reinterpret_cast<uint64_t *>(base + o_guards);
  p->guard_bad = reinterpret_cast<int32_t *>(base + o_gbad);
  if (e == cudaSuccess) e = upload(p->guard_off, cv.guards);
  if (e == cudaSuccess) launch_guard_fill(base, p->guard_off, p->n_guards, nullptr);
  if (e == cudaSuccess) e = upload(p->sh.layers, dl);
  p->dl_host = dl;
  if (e == cudaSuccess) e = upload(p->btiles, bt);
  if (e == cudaSuccess) e = upload(p->utiles, ut);
  if (e == cudaSuccess) e = upload(p->ctiles, ct);
  for (int k = 0; k < kSets && e == cudaSuccess; ++k) {
    e = upload(p->probs[k], gp[k]);
    if (e == cudaSuccess) e = upload(p->gtiles[k], gt[k]);
  }
  if (e == cudaSuccess) e = cudaMemset(p->sh.status, 0, sizeof(int32_t));
  if (e == cudaSuccess)
    e = cudaMemset(p->sh.gate_scratch, 0, kScratchSlots * sizeof(unsigned long long));  // key 0 < every RMMC
  if (e == cudaSuccess && num_layers > 0) e = prepare_chol_inv(p->max_r, &p->chol_smem);
  if (e == cudaSuccess && precision != DION_PREC_FP32) {
    p->tcp.probs = p->probs;
    p->tcp.gtiles = p->gtiles;
    p->tcp.n_gtiles = p->n_gtiles;
    e = tc::init(tcl, base, dl.data(), num_layers, &p->tcp);
    if (e == cudaSuccess) {  // the tensor-core path works from a bf16 copy of Q
      tc::refresh(p->tcp, p->sh, nullptr);
      e = cudaGetLastError();
    }
  }
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  if (e != cudaSuccess) {
    cudaFree(p->ws);
    delete p;
    return DION_ERR_CUDA;
  }
  p->launches_per_step = (precision == DION_PREC_FP32) ? 17 : tc::launches_per_step(p->tcp);
#ifdef DION_DEBUG_CHECKS
  p->launches_per_step += 1;  // the guard check at the end of every step
#endif
  *out = p;
  return DION_OK;
}

}  // extern "C"

namespace {

dion_status check_step_args(const dion_plan *p, const dion_hparams *hp, const double *prev_norm,
                            const double *rmmc_out, const uint8_t *sync_flags_out, const uint8_t *global_flag_out) {
  if (!p || !hp || !prev_norm || !rmmc_out || !sync_flags_out || !global_flag_out) return DION_ERR_INVALID_ARG;
  if (hp->gate_mode < DION_GATE_ALWAYS || hp->gate_mode > DION_GATE_SCHEDULED) return DION_ERR_INVALID_ARG;
  if (hp->gate_mode == DION_GATE_SCHEDULED && hp->period < 1) return DION_ERR_INVALID_ARG;
  if (hp->step < 1) return DION_ERR_INVALID_ARG;
  if (!std::isfinite(hp->mu) || !std::isfinite(hp->eta) || !std::isfinite(hp->eta_local) ||
      !std::isfinite(hp->eps_rmmc) || !std::isfinite(hp->eps_col) || std::isnan(hp->tau_global))
    return DION_ERR_INVALID_ARG;
  if (hp->eps_rmmc < 0.f || hp->eps_col < 0.f) return DION_ERR_INVALID_ARG;
  if (!std::isfinite(hp->weight_decay) || hp->weight_decay < 0.f) return DION_ERR_INVALID_ARG;
  return DION_OK;
}

// Enqueues the step's launch sequence on s with the given layer table and tensor maps (the
// plan's own, or those of a host-gradient buffer).  The caller has checked the arguments and
// made the plan's device current.
StepArgs make_args(const dion_hparams *hp, double *prev_norm, double *rmmc_out, double *rmmc_eq1_out,
                   uint8_t *sync_flags_out, uint8_t *global_flag_out) {
  StepArgs a{};
  a.mu = hp->mu; a.eta = hp->eta; a.eta_local = hp->eta_local;
  a.eps_rmmc = hp->eps_rmmc; a.eps_col = hp->eps_col; a.tau_global = hp->tau_global;
  a.keep_sync = (float)(1.0 - (double)hp->eta * (double)hp->weight_decay);
  a.keep_local = (float)(1.0 - (double)hp->eta_local * (double)hp->weight_decay);
  a.gate_mode = hp->gate_mode; a.period = hp->period < 1 ? 1 : hp->period; a.step = hp->step;
  a.prev_norm = prev_norm; a.rmmc = rmmc_out; a.eq1 = rmmc_eq1_out;
  a.flags = sync_flags_out; a.gflag = global_flag_out;
  return a;
}

void enqueue_step(dion_plan *p, const Shared &sh, const tc::TcPlan &tcp, const dion_hparams *hp, double *prev_norm,
                  double *rmmc_out, double *rmmc_eq1_out, uint8_t *sync_flags_out, uint8_t *global_flag_out,
                  cudaStream_t s) {
  const StepArgs a = make_args(hp, prev_norm, rmmc_out, rmmc_eq1_out, sync_flags_out, global_flag_out);
  tick_begin(p, s);
  if (p->precision == DION_PREC_FP32) {
    launch_form_b(sh, p->btiles, p->n_btiles, s);
    tick(p, s, "form_b");
    launch_gate(sh, a, s);
    tick(p, s, "gate");
    launch_gemm(sh, p->probs[0], p->gtiles[0], p->n_gtiles[0], s);  // P = B Q
    tick(p, s, "gemm_bq");
    static const char *kGram[3] = {"gemm_gram0", "gemm_gram1", "gemm_gram2"};
    static const char *kChol[3] = {"chol_inv0", "chol_inv1", "chol_inv2"};
    static const char *kTrsm[3] = {"gemm_trsm0", "gemm_trsm1", "gemm_trsm2"};
    for (int pass = 0; pass < 3; ++pass) {  // CholeskyQR2, third pass only after a shifted retry
      launch_gemm(sh, p->probs[1 + pass], p->gtiles[1 + pass], p->n_gtiles[1 + pass], s);  // S = X^T X
      tick(p, s, kGram[pass]);
      launch_chol_inv(sh, p->chol_smem, pass, 1e-3f, s);  // L, L^{-1}
      tick(p, s, kChol[pass]);
      launch_gemm(sh, p->probs[4 + pass], p->gtiles[4 + pass], p->n_gtiles[4 + pass], s);  // X L^{-T}
      tick(p, s, kTrsm[pass]);
    }
    launch_gemm(sh, p->probs[7], p->gtiles[7], p->n_gtiles[7], s);  // R = B^T P
    tick(p, s, "gemm_btp");
    launch_colnorm(sh, p->ctiles, p->n_ctiles, a.eps_col, s);       // Q = ColumnNormalize(R)
    tick(p, s, "colnorm");
    launch_update(sh, p->utiles, p->n_utiles, a.mu, a.eta, a.keep_sync, s);  // M, X
    tick(p, s, "update");
    launch_local(sh, p->btiles, p->n_btiles, a.eta_local, a.keep_local, s);  // local branch
    tick(p, s, "local");
    launch_finalize(sh, a, s);                                      // Equation 1
    tick(p, s, "finalize");
  } else {
    tc::step(p, tcp, sh, a, p->btiles, p->n_btiles, p->ctiles, p->n_ctiles, p->chol_smem, s);
  }
#ifdef DION_DEBUG_CHECKS
  launch_guard_check(static_cast<const char *>(p->ws), p->guard_off, p->n_guards, p->guard_bad, sh.status, s);
  tick(p, s, "guard_check");
#endif
  tick_end(p);
}

// One phase of a data-parallel step (dion_step_phase).  The caller reduces rmmc (max) between
// NORMS and POWER, the P range (mean) between POWER and ORTHO and the R range (mean) between
// ORTHO and UPDATE.
void enqueue_phase(dion_plan *p, const StepArgs &a, int32_t phase, cudaStream_t s) {
  const Shared &sh = p->sh;
  if (p->precision != DION_PREC_FP32) {
    tc::step_phase(p->tcp, sh, a, phase, p->btiles, p->n_btiles, p->ctiles, p->n_ctiles, p->chol_smem, s);
    return;
  }
  switch (phase) {
    case DION_PHASE_NORMS:  // B = M + G, ||B||, this worker's RMMC, prev_norm <- ||B||
      launch_form_b(sh, p->btiles, p->n_btiles, s);
      launch_gate(sh, a, s);
      break;
    case DION_PHASE_POWER:  // the branch from the reduced RMMC, then P = B Q on the Dion layers
      launch_gate_reduced(sh, a, s);
      launch_gemm(sh, p->probs[0], p->gtiles[0], p->n_gtiles[0], s);
      break;
    case DION_PHASE_ORTHO:  // Orthogonalize the averaged P, then R = B^T P
      for (int pass = 0; pass < 3; ++pass) {
        launch_gemm(sh, p->probs[1 + pass], p->gtiles[1 + pass], p->n_gtiles[1 + pass], s);
        launch_chol_inv(sh, p->chol_smem, pass, 1e-3f, s);
        launch_gemm(sh, p->probs[4 + pass], p->gtiles[4 + pass], p->n_gtiles[4 + pass], s);
      }
      launch_gemm(sh, p->probs[7], p->gtiles[7], p->n_gtiles[7], s);
      break;
    default:  // UPDATE: Q_t from the averaged R, error feedback and parameter update, local branch
      launch_colnorm(sh, p->ctiles, p->n_ctiles, a.eps_col, s);
      launch_update(sh, p->utiles, p->n_utiles, a.mu, a.eta, a.keep_sync, s);
      launch_local(sh, p->btiles, p->n_btiles, a.eta_local, a.keep_local, s);
      launch_finalize(sh, a, s);
      break;
  }
}

// Makes the plan's device current for the duration of a call.
struct DeviceGuard {
  int prev = -1;
  bool ok = true;
  explicit DeviceGuard(int dev) {
    if (cudaGetDevice(&prev) != cudaSuccess || prev != dev) ok = cudaSetDevice(dev) == cudaSuccess;
  }
  ~DeviceGuard() {
    if (prev >= 0 && ok) cudaSetDevice(prev);
  }
};

}  // namespace

extern "C" {

dion_status dion_step(dion_plan *p, const dion_hparams *hp, double *prev_norm, double *rmmc_out,
                      double *rmmc_eq1_out, uint8_t *sync_flags_out, uint8_t *global_flag_out,
                      void *stream) {
  const dion_status st = check_step_args(p, hp, prev_norm, rmmc_out, sync_flags_out, global_flag_out);
  if (st != DION_OK) return st;
  if (p->next_phase != DION_PHASE_NORMS) return DION_ERR_INVALID_ARG;  // a phased step is unfinished
  DeviceGuard g(p->device);
  if (!g.ok) return DION_ERR_CUDA;
  enqueue_step(p, p->sh, p->tcp, hp, prev_norm, rmmc_out, rmmc_eq1_out, sync_flags_out, global_flag_out,
               static_cast<cudaStream_t>(stream));
  return cudaGetLastError() == cudaSuccess ? DION_OK : DION_ERR_CUDA;
}

dion_status dion_step_phase(dion_plan *p, int32_t phase, const dion_hparams *hp, double *prev_norm, double *rmmc_out,
                            double *rmmc_eq1_out, uint8_t *sync_flags_out, uint8_t *global_flag_out, void *stream) {
  const dion_status st = check_step_args(p, hp, prev_norm, rmmc_out, sync_flags_out, global_flag_out);
  if (st != DION_OK) return st;
  if (phase < DION_PHASE_NORMS || phase > DION_PHASE_UPDATE || phase != p->next_phase) return DION_ERR_INVALID_ARG;
  DeviceGuard g(p->device);
  if (!g.ok) return DION_ERR_CUDA;
  const StepArgs a = make_args(hp, prev_norm, rmmc_out, rmmc_eq1_out, sync_flags_out, global_flag_out);
  enqueue_phase(p, a, phase, static_cast<cudaStream_t>(stream));
#ifdef DION_DEBUG_CHECKS
  if (phase == DION_PHASE_UPDATE)
    launch_guard_check(static_cast<const char *>(p->ws), p->guard_off, p->n_guards, p->guard_bad, p->sh.status,
                       static_cast<cudaStream_t>(stream));
#endif
  if (cudaGetLastError() != cudaSuccess) return DION_ERR_CUDA;
  p->next_phase = (phase == DION_PHASE_UPDATE) ? DION_PHASE_NORMS : phase + 1;
  return DION_OK;
}

dion_status dion_plan_exchange(dion_plan *p, int32_t phase, float **buf_out, int64_t *count_out) {
  if (!p || !buf_out || !count_out) return DION_ERR_INVALID_ARG;
  if (phase == DION_PHASE_POWER) {
    *buf_out = p->L > 0 ? reinterpret_cast<float *>(static_cast<char *>(p->ws) + p->xp_off) : nullptr;
    *count_out = p->xp_count;
  } else if (phase == DION_PHASE_ORTHO) {
    *buf_out = p->L > 0 ? reinterpret_cast<float *>(static_cast<char *>(p->ws) + p->xr_off) : nullptr;
    *count_out = p->xr_count;
  } else {
    return DION_ERR_INVALID_ARG;
  }
  return DION_OK;
}

dion_status dion_plan_enable_host_gradients(dion_plan *p) {
  if (!p) return DION_ERR_INVALID_ARG;
  if (p->hg.on) return DION_OK;
  DeviceGuard g(p->device);
  if (!g.ok) return DION_ERR_CUDA;
  auto &hg = p->hg;
  const int32_t L = p->L;
  Carver cv;
  std::vector<size_t> off[2];
  hg.ldg.resize(L);
  for (int b = 0; b < 2; ++b) {
    off[b].resize(L);
    for (int32_t l = 0; l < L; ++l) {
      const DevLayer &d = p->dl_host[l];
      const int64_t esz = d.g_dtype == DT_BF16 ? 2 : 4, ld = (d.n * esz + 15) / 16 * 16 / esz;
      hg.ldg[l] = ld;
      off[b][l] = cv.take<char>((size_t)(d.m * ld * esz));
    }
  }
  const size_t o_layers[2] = {cv.take<DevLayer>(std::max(L, 1)), cv.take<DevLayer>(std::max(L, 1))};
  const bool tcm = p->precision != DION_PREC_FP32;
  size_t o_maps[2] = {0, 0};
  if (tcm) {
    cv.off = (cv.off + 127) / 128 * 128;
    o_maps[0] = cv.take<tc::LayerMaps>(std::max(L, 1));
    o_maps[1] = cv.take<tc::LayerMaps>(std::max(L, 1));
  }
  if (cudaMalloc(&hg.mem, cv.off) != cudaSuccess) {
    hg.mem = nullptr;
    return DION_ERR_CUDA;
  }
  char *base = static_cast<char *>(hg.mem);
  cudaError_t e = cudaSuccess;
  for (int b = 0; b < 2 && e == cudaSuccess; ++b) {
    std::vector<DevLayer> dl = p->dl_host;
    hg.g[b].resize(L);
    for (int32_t l = 0; l < L; ++l) {
      hg.g[b][l] = base + off[b][l];
      dl[l].G = hg.g[b][l];
      dl[l].ldg = hg.ldg[l];
    }
    hg.layers[b] = reinterpret_cast<DevLayer *>(base + o_layers[b]);
    e = upload(hg.layers[b], dl);
    if (e == cudaSuccess && tcm) {
      hg.maps[b] = reinterpret_cast<tc::LayerMaps *>(base + o_maps[b]);
      e = tc::encode_maps(dl.data(), L, hg.maps[b]);
    }
  }
  if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&hg.copy, cudaStreamNonBlocking);
  for (int b = 0; b < 2 && e == cudaSuccess; ++b) {
    e = cudaEventCreateWithFlags(&hg.up[b], cudaEventDisableTiming);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&hg.used[b], cudaEventDisableTiming);
  }
  if (e != cudaSuccess) {
    for (int b = 0; b < 2; ++b) {
      if (hg.up[b]) cudaEventDestroy(hg.up[b]);
      if (hg.used[b]) cudaEventDestroy(hg.used[b]);
      hg.up[b] = hg.used[b] = nullptr;
    }
    if (hg.copy) cudaStreamDestroy(hg.copy);
    hg.copy = nullptr;
    cudaFree(hg.mem);
    hg.mem = nullptr;
    return DION_ERR_CUDA;
  }
  hg.parity = 0;
  hg.on = true;
  return DION_OK;
}

dion_status dion_step_host(dion_plan *p, const dion_hparams *hp, const void *const *host_G, const int64_t *host_ldg,
                           double *prev_norm, double *rmmc_out, double *rmmc_eq1_out, uint8_t *sync_flags_out,
                           uint8_t *global_flag_out, void *stream) {
  const dion_status st = check_step_args(p, hp, prev_norm, rmmc_out, sync_flags_out, global_flag_out);
  if (st != DION_OK) return st;
  if (!p->hg.on || (p->L > 0 && (!host_G || !host_ldg))) return DION_ERR_INVALID_ARG;
  if (p->next_phase != DION_PHASE_NORMS) return DION_ERR_INVALID_ARG;  // a phased step is unfinished
  for (int32_t l = 0; l < p->L; ++l)
    if (!host_G[l] || host_ldg[l] < p->dl_host[l].n) return DION_ERR_INVALID_ARG;
  DeviceGuard g(p->device);
  if (!g.ok) return DION_ERR_CUDA;
  auto &hg = p->hg;
  const int b = hg.parity;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // buffer b was last read by the step two calls back
  if (cudaStreamWaitEvent(hg.copy, hg.used[b], 0) != cudaSuccess) return DION_ERR_CUDA;
  for (int32_t l = 0; l < p->L; ++l) {
    const DevLayer &d = p->dl_host[l];
    const size_t esz = d.g_dtype == DT_BF16 ? 2 : 4;
    cudaError_t e;
    if (host_ldg[l] == hg.ldg[l])
      e = cudaMemcpyAsync(hg.g[b][l], host_G[l], (size_t)(d.m * hg.ldg[l]) * esz, cudaMemcpyHostToDevice, hg.copy);
    else
      e = cudaMemcpy2DAsync(hg.g[b][l], (size_t)hg.ldg[l] * esz, host_G[l], (size_t)host_ldg[l] * esz,
                            (size_t)d.n * esz, (size_t)d.m, cudaMemcpyHostToDevice, hg.copy);
    if (e != cudaSuccess) return DION_ERR_CUDA;
  }
  if (cudaEventRecord(hg.up[b], hg.copy) != cudaSuccess || cudaStreamWaitEvent(s, hg.up[b], 0) != cudaSuccess)
    return DION_ERR_CUDA;
  Shared sh = p->sh;
  sh.layers = hg.layers[b];
  tc::TcPlan tcp = p->tcp;
  if (p->precision != DION_PREC_FP32) tcp.maps = hg.maps[b];
  enqueue_step(p, sh, tcp, hp, prev_norm, rmmc_out, rmmc_eq1_out, sync_flags_out, global_flag_out, s);
  if (cudaEventRecord(hg.used[b], s) != cudaSuccess) return DION_ERR_CUDA;
  hg.parity ^= 1;
  return cudaGetLastError() == cudaSuccess ? DION_OK : DION_ERR_CUDA;
}

float dion_lr_schedule(int64_t step, int64_t total_steps, float base_lr, float warmup_frac, float warmdown_frac) {
  if (total_steps < 1 || !(warmup_frac >= 0.f && warmup_frac <= 1.f) || !(warmdown_frac >= 0.f && warmdown_frac <= 1.f))
    return NAN;
  const int64_t T = total_steps;
  const int64_t W = (int64_t)std::floor((double)warmup_frac * (double)T + 0.5);  // rounded half up
  const int64_t D = (int64_t)std::floor((double)warmdown_frac * (double)T + 0.5);
  if (W + D > T) return NAN;
  const int64_t t = std::min(std::max<int64_t>(step, 1), T);
  if (W > 0 && t <= W) return (float)((double)base_lr * (double)t / (double)W);
  if (D > 0 && t > T - D) return (float)((double)base_lr * (double)(T - t) / (double)D);
  return base_lr;
}

int64_t dion_rank_for(int64_t m, int64_t n, double fraction) {
  if (m < 1 || n < 1 || !(fraction > 0.0 && fraction <= 1.0)) return 0;
  const int64_t k = std::min(m, n);
  const int64_t r = (int64_t)std::ceil(fraction * (double)k - 1e-12);
  return std::min(k, std::max<int64_t>(1, r));
}

dion_status dion_get_device_status(dion_plan *p, int32_t clear, int32_t *code_out) {
  if (!p || !code_out) return DION_ERR_INVALID_ARG;
  int32_t v = 0;
  if (cudaMemcpy(&v, p->sh.status, sizeof(v), cudaMemcpyDeviceToHost) != cudaSuccess) return DION_ERR_CUDA;
  if (clear && cudaMemset(p->sh.status, 0, sizeof(int32_t)) != cudaSuccess) return DION_ERR_CUDA;
  *code_out = v;
  return DION_OK;
}

int32_t dion_step_launch_count(const dion_plan *p) { return p ? p->launches_per_step : 0; }

dion_status dion_plan_check_guards(dion_plan *p, int32_t *damaged_out) {
  if (!p || !damaged_out) return DION_ERR_INVALID_ARG;
  DeviceGuard g(p->device);
  if (!g.ok) return DION_ERR_CUDA;
  if (cudaDeviceSynchronize() != cudaSuccess || cudaMemset(p->guard_bad, 0, sizeof(int32_t)) != cudaSuccess)
    return DION_ERR_CUDA;
  launch_guard_check(static_cast<const char *>(p->ws), p->guard_off, p->n_guards, p->guard_bad, nullptr, nullptr);
  int32_t v = 0;
  if (cudaGetLastError() != cudaSuccess || cudaMemcpy(&v, p->guard_bad, sizeof(v), cudaMemcpyDeviceToHost) != cudaSuccess)
    return DION_ERR_CUDA;
  *damaged_out = v;
  return DION_OK;
}

int32_t dion_debug_checks(void) {
#ifdef DION_DEBUG_CHECKS
  return 1;
#else
  return 0;
#endif
}

dion_status dion_plan_set_wait_limit(dion_plan *p, int64_t limit_ns) {
  if (!p) return DION_ERR_INVALID_ARG;
  p->sh.handoff_limit_ns = limit_ns > 0 ? (uint64_t)limit_ns : kDefaultWaitLimitNs;
  return DION_OK;
}

dion_status dion_plan_refresh(dion_plan *p, void *stream) {
  if (!p) return DION_ERR_INVALID_ARG;
  if (p->precision == DION_PREC_FP32) return DION_OK;
  tc::refresh(p->tcp, p->sh, static_cast<cudaStream_t>(stream));
  return cudaGetLastError() == cudaSuccess ? DION_OK : DION_ERR_CUDA;
}

static void free_events(dion_plan *p) {
  for (cudaEvent_t e : p->ev) cudaEventDestroy(e);
  p->ev.clear();
  p->timing_steps = p->recorded = 0;
}

dion_status dion_timing_enable(dion_plan *p, int32_t max_steps) {
  if (!p || max_steps < 0) return DION_ERR_INVALID_ARG;
  if (cudaDeviceSynchronize() != cudaSuccess) return DION_ERR_CUDA;
  free_events(p);
  if (max_steps == 0) return DION_OK;
  const size_t count = (size_t)max_steps * (p->launches_per_step + 1);
  p->ev.resize(count);
  for (size_t i = 0; i < count; ++i) {
    if (cudaEventCreate(&p->ev[i]) != cudaSuccess) {
      p->ev.resize(i);
      free_events(p);
      return DION_ERR_CUDA;
    }
  }
  p->timing_steps = max_steps;
  p->recorded = 0;
  return DION_OK;
}

dion_status dion_timing_read(dion_plan *p, int32_t cap, float *ms_out, const char **names_out, int32_t *count_out,
                             int32_t *steps_out) {
  if (!p || !count_out || !steps_out || (cap > 0 && (!ms_out || !names_out))) return DION_ERR_INVALID_ARG;
  const int32_t per = p->launches_per_step + 1;
  const int32_t n = std::min(cap, p->launches_per_step);
  for (int32_t i = 0; i < n; ++i) {
    double tot = 0.0;
    for (int32_t st = 0; st < p->recorded; ++st) {
      float ms = 0.f;
      if (cudaEventSynchronize(p->ev[(size_t)st * per + i + 1]) != cudaSuccess) return DION_ERR_CUDA;
      if (cudaEventElapsedTime(&ms, p->ev[(size_t)st * per + i], p->ev[(size_t)st * per + i + 1]) != cudaSuccess)
        return DION_ERR_CUDA;
      tot += ms;
    }
    ms_out[i] = p->recorded ? (float)(tot / p->recorded) : 0.f;
    names_out[i] = i < (int32_t)p->names.size() ? p->names[i] : "";
  }
  *count_out = p->launches_per_step;
  *steps_out = p->recorded;
  p->recorded = 0;
  return DION_OK;
}

void dion_plan_destroy(dion_plan *p) {
  if (!p) return;
  cudaDeviceSynchronize();
  free_events(p);
  for (int b = 0; b < 2; ++b) {
    if (p->hg.up[b]) cudaEventDestroy(p->hg.up[b]);
    if (p->hg.used[b]) cudaEventDestroy(p->hg.used[b]);
  }
  if (p->hg.copy) cudaStreamDestroy(p->hg.copy);
  cudaFree(p->hg.mem);
  tc::destroy(&p->tcp);
  cudaFree(p->ws);
  delete p;
}

}  // extern "C"
