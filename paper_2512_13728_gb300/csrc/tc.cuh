// Tensor-core (tcgen05) path of the CurvaDion step: DION_PREC_BF16 and DION_PREC_BF16X3.
#pragma once

#include "../../include/curvadion.h"
#include "common.cuh"

namespace cd {
namespace tc {

struct TcLayout {
  size_t end = 0;
  bool supported = false;
};

struct TcPlan {
  int32_t launches = 0;
};

inline dion_status layout(const dion_layer *, int32_t, int32_t, int, size_t start, TcLayout *out) {
  out->end = start;
  out->supported = false;
  return DION_ERR_UNSUPPORTED;
}
inline void bind(const TcLayout &, char *, DevLayer *, int32_t, TcPlan *) {}
inline cudaError_t init(const TcLayout &, const DevLayer *, int32_t, TcPlan *) { return cudaSuccess; }
inline int32_t launches_per_step(const TcPlan &p) { return p.launches; }
inline void step(dion_plan *, const TcPlan &, const Shared &, const StepArgs &, const int4 *, int32_t,
                 const int4 *, int32_t, size_t, cudaStream_t) {}
inline void destroy(TcPlan *) {}

}  // namespace tc
}  // namespace cd
