// Tensor-core (tcgen05) path of the CurvaDion step: DION_PREC_BF16 and DION_PREC_BF16X3.
#pragma once

#include <cuda.h>

#include <vector>

#include "../../include/curvadion.h"
#include "common.cuh"

namespace cd {
namespace tc {

// Per-layer TMA descriptors (device memory, 64-byte aligned).  bf16 maps use a 128-byte
// swizzle with 64-element inner boxes; fp32 maps use 32-element (128-byte) inner boxes.
struct LayerMaps {
  CUtensorMap P_hi;   // m x r bf16:  box {64, 128}  update: A operand (K = r)
  CUtensorMap R_hi;   // n x r bf16:  box {64, 128}  update: B operand of P R^T
  CUtensorMap Qn_hi;  // n x r bf16:  box {64, 128}  update: B operand of P Q_t^T
  CUtensorMap Mf;     // m x n fp32 (caller M): box {32, 128}  update: B in / M_t out
  CUtensorMap Xf;     // m x n fp32 (caller X): box {32, 128}  update: X in / out
  CUtensorMap Mf16, Xf16;  // m x n fp32: box {16, 128}, 64-byte swizzle (update epilogue)
  CUtensorMap Gh16;        // m x n bf16 G: box {16, 128}, 32-byte swizzle (update epilogue)
  CUtensorMap Gh64;        // m x n bf16 G: box {64, 128}  fused buffer pass + B Q
  CUtensorMap Qn_mn;  // n x r bf16:  box {64, 64}   B Q: MN-major B operand (K = n)
  CUtensorMap P_mn;   // m x r bf16:  box {64, 64}   B^T P: MN-major B operand (K = m)
  CUtensorMap Bh_mn;  // m x n bf16:  box {64, 64}   B^T P: MN-major A operand (K = m)
  CUtensorMap Bh_k;   // m x n bf16:  box {64, 128}  B Q: K-major A operand (K = n)
  CUtensorMap Praw;   // m x r fp32:  box {32, 128}  B Q output; TRSM A operand / output
  CUtensorMap Rst;    // n x r fp32:  box {32, 128}  B^T P: output store
  CUtensorMap Pf;     // m x r fp32 (P):      box {32, 128}  TRSM A operand / output
  CUtensorMap PTraw;  // r x m fp32 (P_raw^T): box {32, 128}  Gram operands
  CUtensorMap PT;     // r x m fp32 (P^T):    box {32, 128}  Gram operands
  CUtensorMap PTraw_t;  // r x m fp32: box {32, 32}  transposed output store
  CUtensorMap PT_t;     // r x m fp32: box {32, 32}  transposed output store
  CUtensorMap Sst;    // r x r fp32:  box {32, 128}  Gram output
  CUtensorMap Linv;   // r x r fp32:  box {32, 128}  TRSM B operand (rows of L^{-1})
  CUtensorMap Linv32; // r x r fp32:  box {32, 32}   Cholesky trailing update (reduce-add)
  // BF16X3: the low halves, boxes as their high counterparts (zeroed maps in the other modes)
  CUtensorMap P_lo, R_lo, Qn_lo;  // K-major {64, 128}: update operands
  CUtensorMap Qn_lo_mn, P_lo_mn, Bl_mn;  // MN-major {64, 64}: B Q / B^T P operands
  CUtensorMap Bl_k;   // K-major {64, 128}: B Q A operand
  // BF16X3 update operands in 32-wide K chunks: K-major {32, 128}, 64-byte swizzle
  CUtensorMap P_hi32, P_lo32, R_hi32, R_lo32, Qn_hi32, Qn_lo32;
};

// Tiles of one persistent kernel, reordered so that CTA b processes tiles [off[b], off[b+1]).
struct Schedule {
  std::vector<int4> tiles;
  std::vector<int> off;
  int grid = 0;
  size_t o_tiles = 0, o_off = 0;  // workspace offsets
};

struct TcLayout {
  Schedule s_update, s_bq, s_btp, s_gram, s_trsm;
  size_t end = 0;
  size_t o_maps = 0;
  size_t o_utiles = 0, o_ftiles = 0, o_rtiles = 0, o_qtiles = 0, o_gtiles = 0, o_ttiles = 0;
  std::vector<size_t> o_phi, o_rhi, o_qnhi, o_bh, o_ptraw, o_pt, o_colsq, o_colinv;
  std::vector<size_t> o_bl, o_plo, o_rlo, o_qnlo;  // BF16X3 low halves
  std::vector<uint64_t> guards;  // offsets of the guard words after each region
  std::vector<int4> gram_tiles, trsm_tiles;
  // update tiles {layer, m-block, n-block, slot}; P-convert tiles {layer, row0, rows, 0};
  // B Q tiles {layer, m-block, 0, slot}; B^T P tiles {layer, n-block, 0, 0}; Q-copy tiles
  std::vector<int4> utiles, ftiles, rtiles, qtiles;
  int32_t precision = 0;
  int32_t max_r = 0;
  // every layer has bf16 G: the buffer pass is fused into B Q (norm slots = 128-row tiles)
  bool fuse_buffer = false;
};

struct DevSchedule {
  const int4 *tiles = nullptr;
  const int *off = nullptr;
  int grid = 0;
};

struct TcPlan {
  DevSchedule d_update, d_bq, d_btp, d_gram, d_trsm;
  LayerMaps *maps = nullptr;
  int4 *utiles = nullptr;
  int32_t n_utiles = 0;
  int4 *ftiles = nullptr;
  int32_t n_ftiles = 0;
  int4 *rtiles = nullptr;
  int32_t n_rtiles = 0;
  int4 *qtiles = nullptr;
  int32_t n_qtiles = 0;
  int4 *gram_tiles = nullptr;
  int32_t n_gram_tiles = 0;
  int4 *trsm_tiles = nullptr;
  int32_t n_trsm_tiles = 0;
  int32_t max_r = 0;
  int32_t f_stages = 0, r_stages = 0, o_stages = 0, t_stages = 0;  // t: the TRSM's (A + one B box per stage)
  uint32_t f_smem = 0, r_smem = 0, o_smem = 0, nb64 = 0, nb128 = 0, bq_boxes = 0, o_parts = 0, tmem_cols = 0;
  int32_t num_sms = 0;
  int32_t precision = 0;
  int32_t launches = 0;
  bool fuse_buffer = false;
  uint32_t fb_smem = 0;
  size_t chol_tc_smem = 0;  // the first pass's Cholesky on tensor cores (BF16 mode)
  // CUDA-core pieces reused by this path (set by the plan)
  const GemmProblem *const *probs = nullptr;
  const int4 *const *gtiles = nullptr;
  const int32_t *n_gtiles = nullptr;
  const int4 *utiles_simt = nullptr;
  int32_t n_utiles_simt = 0;
};

// Workspace needs of the tensor-core path, appended after `start`.
dion_status layout(const dion_layer *layers, int32_t L, int32_t precision, int num_sms, size_t start,
                   TcLayout *out);
// Stores the workspace pointers of this path into the layer records.
void bind(const TcLayout &lay, char *base, DevLayer *dl, int32_t L, TcPlan *tp);
// Encodes the per-layer tensor maps of these layer records into dst (device, L entries).
cudaError_t encode_maps(const DevLayer *dl, int32_t L, LayerMaps *dst);
// Encodes the tensor maps, uploads tile lists, sets kernel attributes.
cudaError_t init(const TcLayout &lay, char *base, const DevLayer *dl, int32_t L, TcPlan *tp);
int32_t launches_per_step(const TcPlan &tp);
// Enqueues one step.
void step(dion_plan *p, const TcPlan &tp, const Shared &sh, const StepArgs &a, const int4 *btiles,
          int32_t n_btiles, const int4 *ctiles, int32_t n_ctiles, size_t chol_smem, cudaStream_t s);
// Enqueues one phase of a data-parallel step (DION_PHASE_*).
void step_phase(const TcPlan &tp, const Shared &sh, const StepArgs &a, int32_t phase, const int4 *btiles,
                int32_t n_btiles, const int4 *ctiles, int32_t n_ctiles, size_t chol_smem, cudaStream_t s);
void destroy(TcPlan *tp);
// Re-derives the bf16 copy of every layer's Q from the caller's fp32 Q (plan creation and
// dion_plan_refresh).
void refresh(const TcPlan &tp, const Shared &sh, cudaStream_t s);
// Number of B Q tiles (one norm-partial slot each) the layout needs for these layers.

}  // namespace tc
}  // namespace cd
