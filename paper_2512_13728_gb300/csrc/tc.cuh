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
  CUtensorMap P_hi;   // m x r bf16 (pitch rp):   box {64, 128}  A operand of the update
  CUtensorMap R_hi;   // n x r bf16 (pitch rp):   box {64, 128}  B operand (P R^T)
  CUtensorMap Qn_hi;  // n x r bf16 (pitch rp):   box {64, 128}  B operand (P Q_t^T)
  CUtensorMap Mf;     // m x n fp32 (caller M):  box {32, 128}  B in / M_t out
  CUtensorMap Xf;     // m x n fp32 (caller X):  box {32, 128}  X in / out
};

struct TcLayout {
  size_t end = 0;
  size_t o_maps = 0;
  size_t o_utiles = 0, o_ptiles = 0;
  std::vector<size_t> o_phi, o_rhi, o_qnhi;
  std::vector<int4> utiles, ptiles;  // update tiles {layer, m-block, n-block, slot}; P-convert tiles
  int32_t precision = 0;
};

struct TcPlan {
  LayerMaps *maps = nullptr;
  int4 *utiles = nullptr;
  int32_t n_utiles = 0;
  int4 *ptiles = nullptr;
  int32_t n_ptiles = 0;
  int32_t num_sms = 0;
  int32_t precision = 0;
  int32_t launches = 0;
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
// Encodes the tensor maps, uploads tile lists, sets kernel attributes.
cudaError_t init(const TcLayout &lay, char *base, const DevLayer *dl, int32_t L, TcPlan *tp);
int32_t launches_per_step(const TcPlan &tp);
// Enqueues one step.
void step(dion_plan *p, const TcPlan &tp, const Shared &sh, const StepArgs &a, const int4 *btiles,
          int32_t n_btiles, const int4 *ctiles, int32_t n_ctiles, size_t chol_smem, cudaStream_t s);
void destroy(TcPlan *tp);

}  // namespace tc
}  // namespace cd
