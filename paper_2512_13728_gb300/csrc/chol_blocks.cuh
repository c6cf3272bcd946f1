// 32 x 32 diagonal-block building blocks of the Cholesky + L^{-1} kernels (kernels_simt.cu:
// FFMA sweep; chol_tc.cu: sweep with the trailing update on tensor cores).
#pragma once

#include <cuda_runtime.h>

namespace cd {

constexpr int CB = 32, CBP = CB + 1;

// Row-tile index of tile p in a lower trapezoid whose row tile b holds c1 + b tiles: the
// largest b with b c1 + b (b - 1) / 2 <= p.
// fp32 estimate (p < 2^21 here), corrected exactly in integers.
__device__ __forceinline__ int trap_row(int p, int c1) {
  const float bq = 2.f * (float)c1 - 1.f;
  int b = (int)((sqrtf(bq * bq + 8.f * (float)p) - bq) * 0.5f);
  if (b < 0) b = 0;
  while ((b + 1) * c1 + (b + 1) * b / 2 <= p) ++b;
  while (b > 0 && b * c1 + b * (b - 1) / 2 > p) --b;
  return b;
}

__device__ __forceinline__ void load8(const float *p, float w[8]) {
  const float4 a = *reinterpret_cast<const float4 *>(p), b = *reinterpret_cast<const float4 *>(p + 4);
  w[0] = a.x; w[1] = a.y; w[2] = a.z; w[3] = a.w; w[4] = b.x; w[5] = b.y; w[6] = b.z; w[7] = b.w;
}
__device__ __forceinline__ void store8(float *p, const float w[8]) {
  *reinterpret_cast<float4 *>(p) = make_float4(w[0], w[1], w[2], w[3]);
  *reinterpret_cast<float4 *>(p + 4) = make_float4(w[4], w[5], w[6], w[7]);
}

// The 32 x 32 diagonal-block kernels below are unrolled through template recursion so that
// every register array is indexed by constants (no local-memory copies).
// Column J of the Cholesky factor of a 32 x 32 block held one row per lane.
template <int J>
__device__ __forceinline__ void chol32_col(float (&v)[CB], float *rd, int lane, bool &ok) {
  if constexpr (J < CB) {
    const float piv = __shfl_sync(0xffffffffu, v[J], J);
    ok = ok && (piv > 0.f) && (piv < INFINITY);  // uniform: every lane sees the same pivot
    const float rs = rsqrtf(piv), sq = piv * rs;
    v[J] = (lane == J) ? sq : (lane > J ? v[J] * rs : 0.f);
    if (lane == 0) rd[J] = rs;
#pragma unroll
    for (int k = J + 1; k < CB; ++k) {
      const float lkj = __shfl_sync(0xffffffffu, v[J], k);
      if (lane >= k) v[k] = fmaf(-v[J], lkj, v[k]);
    }
    chol32_col<J + 1>(v, rd, lane, ok);
  }
}

// Row I of the forward substitution L x = e_lane (lane c computes column c of L^{-1}).
template <int I>
__device__ __forceinline__ void trinv32_row(float (&x)[CB], const float *D, const float *rd, int lane) {
  if constexpr (I < CB) {
    float a = (I == lane) ? 1.f : 0.f;
#pragma unroll
    for (int k = 0; k < I; ++k) a = fmaf(-D[I * CBP + k], x[k], a);
    x[I] = a * rd[I];
    trinv32_row<I + 1>(x, D, rd, lane);
  }
}

// v <- T v for a lower-triangular 32 x 32 T (row-major, stride CB), in place from the bottom.
template <int C>
__device__ __forceinline__ void trmv32(float (&v)[CB], const float *T) {
  if constexpr (C >= 0) {
    float a0 = 0.f, a1 = 0.f;
#pragma unroll
    for (int c2 = 0; c2 <= C; c2 += 2) {
      a0 = fmaf(T[C * CB + c2], v[c2], a0);
      if (c2 + 1 <= C) a1 = fmaf(T[C * CB + c2 + 1], v[c2 + 1], a1);
    }
    v[C] = a0 + a1;
    trmv32<C - 1>(v, T);
  }
}

}  // namespace cd
