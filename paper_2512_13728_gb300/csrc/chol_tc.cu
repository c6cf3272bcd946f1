// Cholesky factor and inverse of the first CholeskyQR pass (DION_PREC_BF16) with the rank-32
// trailing update on tcgen05 tensor cores and TMA reduce-adds.
//
// Same right-looking sweep as chol_inv_kernel (kernels_simt.cu): one CTA of 16 warps per layer
// builds L^{-1} in place in the L^{-1} buffer W, over 32-wide block columns k (k0 = 32 k).  W
// starts as the lower triangle of S (+ the shift on the diagonal).  Before step k, for rows
// i >= k0, W[i][j] holds the Schur complement for j >= k0 and U[i][j] = -sum_{K < k} L[i, K]
// L^{-1}[K, j] for j < k0.  Step k:
//   warp 0     factors and inverts the 32 x 32 diagonal block in registers (D_k = L_kk^{-1});
//   warps 1..  finish block row k of L^{-1} (D_k U[k, :k0]) and form the panel
//              L[i, k] = A[i, k] D_k^T below the block; block k's columns of those rows are
//              then zeroed (their U values start from zero);
//   update     W[i][j] -= sum_c Yt[i][c] Yt[j][c] for rows i below the block and columns j <= i,
//              where Yt (r x 32) holds L^{-1}[k, :k0 + 32]^T in its rows j < k0 + 32 and the
//              panel in its rows below.
// The update is a GEMM with K = 32: D = Yt[rows] Yt[0 : N]^T, issued by one thread as
// kind::tf32 MMAs (M = 128 rows, N <= 256 columns per unit) into one of two 256-column TMEM
// slots, so the MMAs of the next unit run while the warps drain this one.  The drain writes -D
// of each 32 x 32 block into a swizzled shared-memory box and adds it into W with a TMA
// reduce-add (fp32 add in L2): W is never loaded for the update, and every global access of it
// is the TMA unit's, whole lines at a time.  Each element receives one add per step, so the
// result does not depend on timing.  Yt lives in shared memory as K-major rows of 32 fp32
// (128 bytes, 128-byte swizzle).
// Accuracy: each Yt value x is split into hi (x with the 13 low mantissa bits cleared, exact
// in tf32) and lo = x - hi, and every k-step issues hi hi + hi lo + lo hi (the lo lo term and
// tf32's rounding of lo leave ~2^-20 relative per product, against 2^-24 for FFMA; the Gram S
// of this mode already carries tf32's 2^-11).  A retry on S + s I after a failed pivot is as
// in chol_inv_kernel.
#include "chol_blocks.cuh"
#include "common.cuh"
#include "tc.cuh"
#include "tc_common.cuh"

#include <algorithm>

namespace cd {
namespace {

using namespace tc;

constexpr int kThreads = 512;
constexpr uint32_t kBox = 32u * 32u * 4u;  // one 32 x 32 fp32 staging box (4 KB) per warp

// Rows of the Yt buffers: r rounded up to 32, at least 128 (one A operand).  A row block that
// would run past them starts its MMA rows earlier; the rows outside the unit add zeros.
__host__ __device__ constexpr int yt_rows(int r) { return std::max((r + 31) / 32 * 32, 128); }

// Row `row` of Yt (32 values) as its hi and lo tf32 halves, in the 128-byte-swizzled layout.
__device__ __forceinline__ void write_yt(uint8_t *yth, uint8_t *ytl, int row, const float (&v)[CB]) {
#pragma unroll
  for (int c4 = 0; c4 < 8; ++c4) {
    float h[4], lo[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const float x = v[4 * c4 + e];
      h[e] = __uint_as_float(__float_as_uint(x) & 0xFFFFE000u);
      lo[e] = x - h[e];
    }
    const uint32_t off = sw128_f32((uint32_t)row, (uint32_t)c4);
    *reinterpret_cast<float4 *>(yth + off) = make_float4(h[0], h[1], h[2], h[3]);
    *reinterpret_cast<float4 *>(ytl + off) = make_float4(lo[0], lo[1], lo[2], lo[3]);
  }
}

struct TcState {
  uint8_t *yth, *ytl, *box;  // box: 16 staging boxes, one per warp
  uint64_t *bars;            // [0], [1]: slot s's MMAs complete; [2]: drain
  uint32_t tmem;
  uint32_t unit;             // units issued so far in this kernel (slot = unit & 1, use = unit >> 1)
  int ya;                    // rows of Yt
  const CUtensorMap *wmap;   // W (r x r fp32), 32 x 32 boxes
};

// Update unit u of a step: row blocks of 128 rows from R0 (i0: first row of the unit; a0: first
// row of the MMA's A operand, <= i0), each split into column parts of at most 256 (the block's
// columns j <= i end below its last row).  Returns false past the last unit.
__device__ __forceinline__ bool unit_of(int u, int R0, int r, int ya, int &i0, int &a0, int &n0, int &nn) {
  for (int b = 0, k = 0; R0 + 128 * b < r; ++b) {
    const int ib = R0 + 128 * b;
    const int N = (std::min(ib + 128, r) + 15) / 16 * 16;
    for (int h = 0; 256 * h < N; ++h, ++k) {
      if (k == u) {
        i0 = ib;
        a0 = std::min(ib, ya - 128);
        n0 = 256 * h;
        nn = std::min(N, 256 * (h + 1)) - n0;
        return true;
      }
    }
  }
  return false;
}

__device__ __forceinline__ void issue_unit(const TcState &ts, uint32_t g, int a0, int n0, int nn) {
  const uint32_t slot = g & 1u;
  const uint32_t ah = smem_u32(ts.yth) + (uint32_t)a0 * 128u, al = smem_u32(ts.ytl) + (uint32_t)a0 * 128u;
  const uint32_t bh = smem_u32(ts.yth) + (uint32_t)n0 * 128u, bl = smem_u32(ts.ytl) + (uint32_t)n0 * 128u;
  const uint32_t idesc = idesc_tf32(128, (uint32_t)nn, false, false), d = ts.tmem + slot * 256u;
#pragma unroll
  for (int k8 = 0; k8 < 4; ++k8) {
    const uint64_t dah = smem_desc_sw128(ah + k8 * 32, 0, 1024), dal = smem_desc_sw128(al + k8 * 32, 0, 1024);
    const uint64_t dbh = smem_desc_sw128(bh + k8 * 32, 0, 1024), dbl = smem_desc_sw128(bl + k8 * 32, 0, 1024);
    umma_tf32(d, dah, dbh, idesc, k8 > 0 ? 1u : 0u);
    umma_tf32(d, dah, dbl, idesc, 1u);
    umma_tf32(d, dal, dbh, idesc, 1u);
  }
  umma_commit(&ts.bars[slot]);
}

// 0: factored; 1: a pivot was not positive and finite (uniform over the block); 2: a wait for
// the tensor cores gave up.
__device__ int chol_inverse_tc(const float *__restrict__ S, float *__restrict__ W, int r, int64_t ls, float shift,
                               float *D, float *DI, float *rd, int *bad, TcState &ts, int32_t *status) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, q = tid - 32;
  // W <- lower triangle of S + shift I (coalesced; the upper triangle is never read before each
  // row's own step overwrites it)
  for (int i = warp; i < r; i += kThreads / 32)
    for (int j = lane; j <= i; j += 32) W[(int64_t)i * ls + j] = S[(int64_t)i * ls + j] + (j == i ? shift : 0.f);
  fence_async_global();  // these stores precede the TMA reduce-adds into the same rows
  __syncthreads();
  uint8_t *mybox = ts.box + (uint32_t)warp * kBox;
  for (int k0 = 0; k0 < r; k0 += CB) {
    const int nb = min(CB, r - k0), R0 = k0 + nb, t = r - R0;
    float v[CB];
    if (warp == 0) {
      // ---- diagonal block: lane i holds row k0 + i (identity padding below a short block)
      const int64_t row = k0 + lane;
      if (nb == CB) {
        load8(W + row * ls + k0, v);
        load8(W + row * ls + k0 + 8, v + 8);
        load8(W + row * ls + k0 + 16, v + 16);
        load8(W + row * ls + k0 + 24, v + 24);
      } else {
#pragma unroll
        for (int j = 0; j < CB; ++j) v[j] = (lane < nb && j < nb) ? W[row * ls + k0 + j] : 0.f;
      }
#pragma unroll
      for (int j = 0; j < CB; ++j) {
        if (j > lane) v[j] = 0.f;
        if (j == lane && lane >= nb) v[j] = 1.f;
      }
      bool ok = true;
      chol32_col<0>(v, rd, lane, ok);
#pragma unroll
      for (int j = 0; j < CB; ++j) D[lane * CBP + j] = v[j];
      __syncwarp();
      trinv32_row<0>(v, D, rd, lane);  // lane c: column c of D_k = L_kk^{-1}
#pragma unroll
      for (int i = 0; i < CB; ++i) DI[i * CB + lane] = v[i];
      if (lane == 0) *bad = ok ? 0 : 1;
    } else if (q < k0) {
      // ---- column q of U[k, :k0]
#pragma unroll
      for (int c = 0; c < CB; ++c) v[c] = (c < nb) ? W[(int64_t)(k0 + c) * ls + q] : 0.f;
    } else if (q < k0 + t) {
      // ---- panel row R0 + q - k0 (a full block: nb = 32 whenever rows remain below it)
      float *p = W + (int64_t)(R0 + q - k0) * ls + k0;
      load8(p, v);
      load8(p + 8, v + 8);
      load8(p + 16, v + 16);
      load8(p + 24, v + 24);
    }
    __syncthreads();
    if (*bad) return 1;
    if (warp > 0 && q < k0 + t) {
      trmv32<CB - 1>(v, DI);  // the finished L^{-1}[k, q], or the panel L[row, k0 ..] = A D_k^T
      if (q < k0) {
#pragma unroll
        for (int c = 0; c < CB; ++c)
          if (c < nb) W[(int64_t)(k0 + c) * ls + q] = v[c];
        if (t > 0) write_yt(ts.yth, ts.ytl, q, v);
      } else {
        write_yt(ts.yth, ts.ytl, R0 + q - k0, v);
      }
    }
    // block k's U columns of the rows below start from zero (their panel values were read
    // above): one 128-byte row segment per warp instruction
    for (int row = R0 + warp; row < r; row += kThreads / 32) W[(int64_t)row * ls + k0 + lane] = 0.f;
    // block row k right of k0: D_k on the diagonal block, zeros beyond
    for (int i = warp; i < nb; i += kThreads / 32)
      for (int c = lane; c < r - k0; c += 32) W[(int64_t)(k0 + i) * ls + k0 + c] = (c <= i) ? DI[i * CB + c] : 0.f;
    if (t > 0 && tid < CB) {  // rows k0 .. k0 + 31 of Yt: the columns of D_k
      float w[CB];
#pragma unroll
      for (int c = 0; c < CB; ++c) w[c] = DI[c * CB + tid];
      write_yt(ts.yth, ts.ytl, k0 + tid, w);
    }
    fence_async_smem();    // the Yt writes are read by the tensor cores
    fence_async_global();  // the zeroed columns precede the reduce-adds into them
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (t == 0) continue;
    // ---- update: units in two TMEM slots, the MMAs of unit u + 1 under the drain of unit u
    int i0, a0, n0, nn;
    const uint32_t g0 = ts.unit;
    if (tid == 0 && unit_of(0, R0, r, ts.ya, i0, a0, n0, nn)) issue_unit(ts, g0, a0, n0, nn);
    for (int u = 0; unit_of(u, R0, r, ts.ya, i0, a0, n0, nn); ++u) {
      const uint32_t g = g0 + (uint32_t)u, slot = g & 1u;
      int i1, a1, n1, nn1;
      if (tid == 0 && unit_of(u + 1, R0, r, ts.ya, i1, a1, n1, nn1)) issue_unit(ts, g + 1, a1, n1, nn1);
      const bool got = mbar_wait(&ts.bars[slot], (g >> 1) & 1u, status);
      if (!__syncthreads_and(got)) {
        ts.unit = g + 2;  // units g and (maybe) g + 1 were issued; the caller drains them
        return 2;
      }
      tc_fence_after();
      // warp w: TMEM lane quarter w % 4 (MMA rows a0 + 32 (w % 4) ..) and column chunks w / 4,
      // w / 4 + 4 of the unit (nn <= 256: at most 8 chunks of 32)
      const int q4 = warp & 3, rb = a0 + 32 * q4, i = rb + lane;
      const int iend = std::min(i0 + 128, r);
      const bool row_in = i >= i0 && i < iend;  // this lane's row belongs to the unit
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int jc = (warp >> 2) + 4 * h, j0 = n0 + jc * 32;
        // warp-uniform: the chunk starts inside the unit, not above every row of the warp, and
        // the warp has a row in the unit
        if (jc * 32 >= nn || j0 > rb + 31 || rb + 31 < i0 || rb >= iend) continue;
        uint32_t d[32];
        tmem_ld32(ts.tmem + ((uint32_t)(32 * q4) << 16) + slot * 256u + (uint32_t)(jc * 32), d);
        tmem_ld_wait();
        if (lane == 0) bulk_wait_read<0>();  // the box's previous reduce-add has read it
        __syncwarp();
#pragma unroll
        for (int c4 = 0; c4 < 8; ++c4) {
          float o[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const int j = j0 + 4 * c4 + e;
            o[e] = (row_in && j <= i) ? -__uint_as_float(d[4 * c4 + e]) : 0.f;
          }
          *reinterpret_cast<float4 *>(mybox + sw128_f32((uint32_t)lane, (uint32_t)c4)) = make_float4(o[0], o[1], o[2], o[3]);
        }
        fence_async_smem();
        __syncwarp();
        if (lane == 0) {
          tma_reduce_add_2d(ts.wmap, mybox, j0, rb);  // rows / columns past r are skipped
          bulk_commit();
        }
      }
      tc_fence_before();
      __syncthreads();  // the slot is read out before the MMAs of unit u + 2 reuse it
      tc_fence_after();
      ts.unit = g + 1;
    }
    // the step's reduce-adds are complete before the next step reads W
    if (lane == 0) {
      bulk_wait<0>();
      fence_async_global();
    }
    __syncthreads();
  }
  return 0;
}

__global__ void __launch_bounds__(kThreads, 1) chol_inv_tc_kernel(Shared sh, const LayerMaps *__restrict__ maps) {
  const int l = blockIdx.x;
  if (!sh.active[l]) return;
  const DevLayer &Ly = sh.layers[l];
  const int r = (int)Ly.r;
  const int64_t ls = Ly.ldp;
  const float *S = Ly.S;
  float *Li = Ly.Linv;
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = align1024(smem_raw);
  TcState ts;
  ts.ya = yt_rows(r);
  ts.yth = smem;
  ts.ytl = smem + (size_t)ts.ya * 128;
  ts.box = ts.ytl + (size_t)ts.ya * 128;
  float *D = reinterpret_cast<float *>(ts.box + (kThreads / 32) * kBox);  // CB x CBP
  float *rd = D + CB * CBP;                                                 // CB
  float *DI = rd + 32;                                                      // CB x CB
  ts.bars = reinterpret_cast<uint64_t *>(DI + CB * CB);
  ts.unit = 0;
  ts.wmap = &maps[l].Linv32;
  __shared__ uint32_t tmem_base_s;
  __shared__ int bad;
  __shared__ double red[kThreads / 32];
  __shared__ double trace_s;
  const int tid = threadIdx.x;
  if (tid == 0) {
    for (int i = 0; i < 3; ++i) mbar_init(&ts.bars[i], 1);
    fence_mbar_init();
  }
  if ((tid >> 5) == 0) {
    tmem_alloc(&tmem_base_s, 512);
    tmem_relinquish();
  }
  // rows of Yt that no step writes (past r) stay zero
  for (int e = tid; e < ts.ya * 32; e += kThreads) {
    reinterpret_cast<float *>(ts.yth)[e] = 0.f;
    reinterpret_cast<float *>(ts.ytl)[e] = 0.f;
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  ts.tmem = tmem_base_s;

  int res = chol_inverse_tc(S, Li, r, ls, 0.f, D, DI, rd, &bad, ts, sh.status);
  bool shifted = false;
  if (res == 1) {  // shifted retry from S + s I (shifted CholeskyQR, as in chol_inv_kernel)
    double tr = 0.0;
    for (int i = tid; i < r; i += kThreads) tr += (double)S[(int64_t)i * ls + i];
    tr = block_sum<kThreads>(tr, red);
    if (tid == 0) trace_s = tr;
    __syncthreads();
    const double u = 5.9604644775390625e-8;  // 2^-24
    const double sft = 11.0 * ((double)Ly.m * r + (double)r * (r + 1)) * u * trace_s;
    shifted = true;
    res = (trace_s > 0.0 && isfinite(trace_s)) ? chol_inverse_tc(S, Li, r, ls, (float)sft, D, DI, rd, &bad, ts, sh.status)
                                               : 1;
  }
  if (tid == 0) {
    sh.orth_shifted[l] = shifted ? 1 : 0;
    if (shifted) atomicAdd(&sh.gate_scratch[kScratchShifted], 1ull);
  }
  if (res != 0) {
    if ((tid & 31) == 0) bulk_wait<0>();  // reduce-adds issued before the failure
    if (tid == 0) {
      if (res == 1) set_status(sh.status, ST_BREAKDOWN);
      umma_commit(&ts.bars[2]);  // every MMA issued so far has completed before TMEM is freed
      mbar_wait(&ts.bars[2], 0, sh.status);
    }
    __syncthreads();
    for (int64_t e = tid; e < (int64_t)r * r; e += kThreads) Li[(e / r) * ls + e % r] = 0.f;
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if ((tid >> 5) == 0) tmem_dealloc(ts.tmem, 512);
}

}  // namespace

size_t chol_tc_smem(int32_t max_r) {
  return 1024 + 2 * (size_t)yt_rows(max_r) * 128 + (kThreads / 32) * (size_t)kBox +
         sizeof(float) * (CB * CBP + 32 + CB * CB) + 64;
}

cudaError_t prepare_chol_inv_tc(int32_t max_r, size_t *smem_out) {
  *smem_out = chol_tc_smem(max_r);
  if (*smem_out > 227u * 1024u) return cudaErrorInvalidValue;
  return cudaFuncSetAttribute(chol_inv_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)*smem_out);
}

void launch_chol_inv_tc(const Shared &sh, const tc::LayerMaps *maps, size_t smem, cudaStream_t s) {
  if (sh.num_layers > 0) chol_inv_tc_kernel<<<sh.num_layers, kThreads, smem, s>>>(sh, maps);
}

}  // namespace cd
