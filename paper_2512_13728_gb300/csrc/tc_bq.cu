// tcgen05 kernels of the power iteration and of R (DION_PREC_BF16).  The buffer B = M + G,
// its bf16 copy Bh and the RMMC norm partials come from the streaming buffer kernel; then
//
//   P = B Q_{t-1} (PowerIter)  and  R = B^T P (after Orthogonalize)
//
// run as one persistent TMA-fed GEMM kernel template: warp 0 issues TMA loads of both bf16
// operands into a shared-memory ring, warp 1 issues 128 x N x 16 tcgen05.mma (N <= 256 per
// instruction) into a 128 x r fp32 TMEM accumulator, warps 2..5 drain TMEM through swizzled
// shared boxes into TMA stores.  Bh serves both GEMMs (K-major rows for B Q, MN-major boxes for
// B^T P), the bf16 copy of Q is read MN-major and the bf16 copy of P MN-major, so no transposed
// copy of a large matrix is made.
//   qn_refresh   the bf16 copy of the caller's Q (plan creation, dion_plan_refresh).
#include "tc.cuh"
#include "tc_common.cuh"
#include "tc_kernels.cuh"

#include <type_traits>

namespace cd {
namespace tc {

constexpr uint32_t OPB_A = 128u * 64u * 2u;   // 128 x 64 bf16 A-operand tile (16 KB)
constexpr uint32_t BOX64 = 64u * 64u * 2u;    // 64 x 64 bf16 MN-major box (8 KB)
constexpr uint32_t EPI_BOX = 128u * 32u * 4u; // 128 x 32 fp32 output box (16 KB)

__device__ __forceinline__ uint32_t rpad16(int64_t r) { return (uint32_t)((r + 15) / 16 * 16); }

// ---------------------------------------------------------------------------------------
// Epilogue shared by tc_form_bq and tc_btp: the 128 x r fp32 accumulator in TMEM is written
// to global memory through two 16 KB swizzled staging boxes and TMA stores (rows/columns
// outside the matrix are clipped by the store).  Called by 128 threads (4 warps covering the
// 4 TMEM lane groups); `leader` issues the stores.
__device__ __forceinline__ void store_accumulator(uint32_t tmem, int warp, int lane, bool leader, uint8_t *stg,
                                                  const CUtensorMap *map, const CUtensorMap *map_t, int64_t r,
                                                  int64_t rows, int32_t row0, uint32_t &ecount, uint32_t bar_id,
                                                  int group, int ngroups) {
  // ngroups 128-thread groups (4 warps each, covering the 4 TMEM lane quarters) split the
  // 32-column chunks; each staging buffer is [row-major 128 x 32 box | 4 transposed 32 x 32
  // boxes].  With one group the two buffers alternate; with two, group g owns buffer g.
  const uint32_t lg = (uint32_t)(warp & 3), row = 32u * lg + lane;
  const int nch = (int)((r + 31) / 32);
  for (int j = group; j < nch; j += ngroups) {
    const uint32_t eb = (ngroups == 1) ? (ecount & 1u) : (uint32_t)group;
    uint8_t *box = stg + eb * 2 * EPI_BOX, *tbox = box + EPI_BOX + lg * (EPI_BOX / 4);
    if (leader) {  // the stores that last used this buffer have read it
      if (ngroups == 1) bulk_wait_read<1>();
      else bulk_wait_read<0>();
    }
    named_sync(bar_id, 128);
    uint32_t v[32];
    tmem_ld32(tmem + (lg * 32u << 16) + j * 32, v);
    tmem_ld_wait();
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      float4 f = make_float4(__uint_as_float(v[4 * q]), __uint_as_float(v[4 * q + 1]), __uint_as_float(v[4 * q + 2]),
                             __uint_as_float(v[4 * q + 3]));
      *reinterpret_cast<float4 *>(box + sw128_f32(row, q)) = f;
    }
    if (map_t != nullptr) {
#pragma unroll
      for (int c = 0; c < 32; ++c)
        *reinterpret_cast<float *>(tbox + c * 128 + ((((uint32_t)lane >> 2) ^ (c & 7)) << 4) + (lane & 3) * 4) =
            __uint_as_float(v[c]);
    }
    fence_async_smem();
    named_sync(bar_id, 128);
    if (leader) {
      tma_store_2d(map, box, j * 32, row0);
      if (map_t != nullptr)
        for (int w4 = 0; w4 < 4; ++w4)
          if ((int64_t)row0 + w4 * 32 < rows)
            tma_store_2d(map_t, box + EPI_BOX + w4 * (EPI_BOX / 4), row0 + w4 * 32, j * 32);
      bulk_commit();
    }
    ++ecount;
  }
}

// Epilogue of R = B^T P for one 128-row tile of R: the fp32 rows of R and their bf16 copy
// (TMA stores) and, per column, the tile's fp64 sum of squares for ColumnNormalize.
// Two 32-column chunks are handled together so the bf16 box is one 64-column SW128 box.
__device__ __forceinline__ void store_r_tile(uint32_t tmem, int warp, int lane, bool leader, uint8_t *stg,
                                             const LayerMaps &mp, const DevLayer &L, int tile, uint32_t &ecount) {
  const uint32_t lg = (uint32_t)(warp & 3), row = 32u * lg + lane;
  const int et = (warp - 2) * 32 + lane;  // 0..127 within the epilogue warps (warps 2..5)
  const int nch = (int)((L.r + 31) / 32), row0 = tile * 128;
  // staging: [fp32 box 16 KB][fp32 box 16 KB][bf16 box 16 KB] + column-partial scratch 4 x 64 floats
  uint8_t *f0 = stg, *f1 = stg + EPI_BOX, *hb = stg + 2 * EPI_BOX;
  float *red = reinterpret_cast<float *>(stg + 3 * EPI_BOX);
  for (int j = 0; j < nch; j += 2) {
    const bool two = (j + 1 < nch);
    if (leader) bulk_wait_read<0>();
    named_sync(1, 128);
    uint32_t v[32];
#pragma unroll 1
    for (int h = 0; h < (two ? 2 : 1); ++h) {
      tmem_ld32(tmem + (lg * 32u << 16) + (j + h) * 32, v);
      tmem_ld_wait();
      uint8_t *fb = h ? f1 : f0;
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        *reinterpret_cast<float4 *>(fb + sw128_f32(row, q)) =
            make_float4(__uint_as_float(v[4 * q]), __uint_as_float(v[4 * q + 1]), __uint_as_float(v[4 * q + 2]),
                        __uint_as_float(v[4 * q + 3]));
        const __nv_bfloat162 a = __floats2bfloat162_rn(__uint_as_float(v[4 * q]), __uint_as_float(v[4 * q + 1]));
        const __nv_bfloat162 b = __floats2bfloat162_rn(__uint_as_float(v[4 * q + 2]), __uint_as_float(v[4 * q + 3]));
        uint2 hv;
        hv.x = *reinterpret_cast<const uint32_t *>(&a);
        hv.y = *reinterpret_cast<const uint32_t *>(&b);
        // bf16 64-column box: columns h*32 + 4q .. live in 16-byte chunk (h*4 + q/2)
        *reinterpret_cast<uint2 *>(hb + sw128_offset(row, (uint32_t)(h * 4 + (q >> 1))) + (q & 1) * 8) = hv;
      }
    }
    if (!two) {  // a lone last chunk: zero the unused half of the bf16 box (clipped by the store anyway)
#pragma unroll
      for (int q = 4; q < 8; ++q) *reinterpret_cast<uint4 *>(hb + sw128_offset(row, q)) = make_uint4(0, 0, 0, 0);
    }
    fence_async_smem();
    named_sync(1, 128);
    if (leader) {
      tma_store_2d(&mp.Rst, f0, j * 32, row0);
      if (two) tma_store_2d(&mp.Rst, f1, (j + 1) * 32, row0);
      tma_store_2d(&mp.R_hi, hb, j * 32, row0);
      bulk_commit();
    }
    // column sums of squares: thread et sums column (et % 32) of chunk j + h over rows (et / 32) * 32 ..
    const int c = et & 31, quarter = et >> 5;
#pragma unroll 1
    for (int h = 0; h < (two ? 2 : 1); ++h) {
      const uint8_t *fb = h ? f1 : f0;
      float ssq = 0.f;
      for (int rr = 0; rr < 32; ++rr) {
        const uint32_t rw = (uint32_t)(quarter * 32 + rr);
        const float x = *reinterpret_cast<const float *>(fb + rw * 128u + ((((uint32_t)c >> 2) ^ (rw & 7u)) << 4) +
                                                         (c & 3) * 4);
        ssq = fmaf(x, x, ssq);
      }
      red[h * 128 + quarter * 32 + c] = ssq;
    }
    named_sync(1, 128);
    if (et < 64) {
      const int h = et >> 5, cc = et & 31, col = (j + h) * 32 + cc;
      if (h == 0 || two) {
        const double tot = ((double)red[h * 128 + cc] + red[h * 128 + 32 + cc]) +
                           ((double)red[h * 128 + 64 + cc] + red[h * 128 + 96 + cc]);
        if (col < L.r) L.colsq[(int64_t)tile * L.ldp + col] = tot;  // rows outside R held zeros
      }
    }
    ecount += two ? 2 : 1;
  }
}

// ========================================================= P = B Q and R = B^T P ===
constexpr int R_THREADS = 6 * 32;
enum : int { GEMM_BQ = 0, GEMM_BTP = 1 };

// KIND = GEMM_BQ : P = B Q_{t-1}. Tile = 128 rows of B; K loop over n.  A = Bh rows (K-major,
//                  one 128 x 64 box), B = the bf16 copy of Q as an MN-major operand (K = n).
//                  Epilogue: P and P^T (fp32) for the Gram of the first CholeskyQR pass.
// KIND = GEMM_BTP: R = B^T P.  Tile = 128 columns of B; K loop over m.  A = Bh^T and B = P_hi,
//                  both MN-major boxes of the row-major copies.  Epilogue: R, bf16 R, column
//                  sums of squares.
// Both run on layers that take the Dion branch only.
// Run in clusters of two CTAs that compute 256-row blocks with pair MMAs (cta_group::2): CTA c
// of the pair owns 128-row tile 2 p + c, holds that tile's A chunk and, of every N part of up
// to 256 columns, the half c of its B columns, and receives its 128 rows of the accumulator
// in its own TMEM.  Per SM and k-chunk that is 16 KB of A and 32 KB of B (r = 512) instead of
// 16 + 64 KB.  Tile = {layer, pair p}.
template <int KIND>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(R_THREADS, 1)
    tc_tma_gemm_kernel(Shared sh, const int4 *__restrict__ tiles, const int *__restrict__ off,
                       const LayerMaps *__restrict__ maps, int nstages, uint32_t stage_bytes, uint32_t tmem_cols) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = align1024(smem_raw);
  uint8_t *stg = smem + nstages * stage_bytes;
  uint64_t *bars = reinterpret_cast<uint64_t *>(stg + 4 * EPI_BOX);
  uint64_t *full = bars, *empty = bars + nstages;
  uint64_t *acc_full = bars + 2 * nstages, *acc_empty = acc_full + 1, *drain = acc_full + 2;
  __shared__ uint32_t tmem_base_s;
  __shared__ int abort_s;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const Abort ab{&abort_s};
  const uint32_t rank = cluster_ctarank();
  const int seg = blockIdx.x >> 1;
  if (threadIdx.x == 0) {
    for (int i = 0; i < nstages; ++i) {
      mbar_init(&full[i], 1);   // used in CTA 0: its arm, both CTAs' bytes
      mbar_init(&empty[i], 1);  // pair commit after the stage's MMAs
    }
    mbar_init(acc_full, 1);   // pair commit after the tile's MMAs
    mbar_init(acc_empty, 2);  // used in CTA 0: one arrival per CTA's epilogue
    mbar_init(drain, 1);
    abort_s = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc_pair(&tmem_base_s, tmem_cols);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  cluster_sync();  // both CTAs' barriers and TMEM exist before anything crosses the pair
  const uint32_t tmem = tmem_base_s;
  // N parts of up to 256 columns; each CTA holds half of a part's columns (64-column boxes)
  auto half_cols = [](uint32_t np, uint32_t part) { return min(256u, np - part * 256u) / 2u; };

  if (warp == 0) {
    if (lane == 0) {
      uint32_t it = 0;
      bool ok = true;
      for (int ti = off[seg]; ti < off[seg + 1] && ok; ++ti) {
        const int4 t = tiles[ti];
        if (!sh.active[t.x]) continue;
        const DevLayer &L = sh.layers[t.x];
        const LayerMaps *mp = maps + t.x;
        const int kch = (int)(((KIND == GEMM_BQ ? L.n : L.m) + 63) / 64);
        const int tr = 2 * t.y + (int)rank;  // past the last tile: zero-filled, not stored
        const uint32_t np = rpad16(L.r), nparts = (np + 255) / 256;
        uint32_t nbox = 0;  // 64-column B boxes per CTA and k-chunk
        for (uint32_t part = 0; part < nparts; ++part) nbox += (half_cols(np, part) + 63) / 64;
        for (int kc = 0; kc < kch; ++kc, ++it) {
          const uint32_t s = it % nstages, ph = (it / nstages) & 1u;
          if (!ab.wait(&empty[s], ph ^ 1u, sh.status)) { ok = false; break; }
          uint8_t *sA = smem + s * stage_bytes, *sB = sA + OPB_A;
          const uint32_t fb = cluster_addr(&full[s], 0);
          if (rank == 0) mbar_expect_tx(&full[s], 2u * (OPB_A + nbox * BOX64));
          if (KIND == GEMM_BQ) {
            tma_load_2d_pair(sA, &mp->Bh_k, fb, kc * 64, tr * 128);
          } else {
            tma_load_2d_pair(sA, &mp->Bh_mn, fb, tr * 128, kc * 64);
            tma_load_2d_pair(sA + BOX64, &mp->Bh_mn, fb, tr * 128 + 64, kc * 64);
          }
          const CUtensorMap *bmap = (KIND == GEMM_BQ) ? &mp->Qn_mn : &mp->P_mn;
          for (uint32_t part = 0; part < nparts; ++part) {
            const uint32_t hc = half_cols(np, part);
            const int x0 = (int)(part * 256u + rank * hc);
            for (uint32_t j = 0; j < (hc + 63) / 64; ++j)
              tma_load_2d_pair(sB + (part * 2u + j) * BOX64, bmap, fb, x0 + (int)j * 64, kc * 64);
          }
        }
      }
      // drain: the last stages' loads have landed and been consumed (their stage was freed)
      for (uint32_t k = (it > (uint32_t)nstages ? it - nstages : 0); k < it; ++k)
        mbar_wait(&empty[k % nstages], (k / nstages) & 1u, sh.status);
    }
  } else if (warp == 1) {
    if (lane == 0 && rank == 0) {
      uint32_t it = 0, tcount = 0;
      bool ok = true;
      for (int ti = off[seg]; ti < off[seg + 1] && ok; ++ti) {
        const int4 t = tiles[ti];
        if (!sh.active[t.x]) continue;
        const DevLayer &L = sh.layers[t.x];
        const int kch = (int)(((KIND == GEMM_BQ ? L.n : L.m) + 63) / 64);
        const uint32_t np = rpad16(L.r), nparts = (np + 255) / 256;
        if (!ab.wait(acc_empty, (tcount & 1u) ^ 1u, sh.status)) break;
        tc_fence_after();
        for (int kc = 0; kc < kch; ++kc, ++it) {
          const uint32_t s = it % nstages, ph = (it / nstages) & 1u;
          if (!ab.wait(&full[s], ph, sh.status)) { ok = false; break; }
          tc_fence_after();
          const uint32_t aB = smem_u32(smem + s * stage_bytes), bB = aB + OPB_A;
#pragma unroll
          for (int k16 = 0; k16 < 4; ++k16) {
            // A: K-major (B Q) advances 32 bytes per 16 k; MN-major (B^T P) two 8-row groups
            const uint64_t ad = (KIND == GEMM_BQ) ? smem_desc_sw128(aB + k16 * 32, 0, 1024)
                                                  : smem_desc_sw128(aB + k16 * 2048, BOX64, 1024);
            for (uint32_t part = 0; part < nparts; ++part) {
              const uint32_t n_here = 2u * half_cols(np, part);
              const uint64_t bd = smem_desc_sw128(bB + part * 2u * BOX64 + k16 * 2048, BOX64, 1024);
              umma_pair_bf16(tmem + part * 256u, ad, bd, idesc_bf16(256, n_here, KIND == GEMM_BTP, true),
                             (kc | k16) ? 1u : 0u);
            }
          }
          umma_pair_commit_mc(&empty[s], 0x3);  // the stage is free in both CTAs
        }
        if (!ok) break;
        umma_pair_commit_mc(acc_full, 0x3);
        ++tcount;
      }
      umma_pair_commit(drain);  // every MMA of the pair has completed before TMEM is freed
      mbar_wait(drain, 0, sh.status);
    }
  } else {
    const bool leader = (warp == 2 && lane == 0);
    uint32_t tcount = 0, ecount = 0;
    for (int ti = off[seg]; ti < off[seg + 1]; ++ti) {
      const int4 t = tiles[ti];
      if (!sh.active[t.x]) continue;
      const DevLayer &L = sh.layers[t.x];
      const int tr = 2 * t.y + (int)rank;
      if (!named_and(1, 128, ab.wait(acc_full, tcount & 1u, sh.status))) break;
      tc_fence_after();
      if ((int64_t)tr * 128 < (KIND == GEMM_BQ ? L.m : L.n)) {  // not the pair's empty second tile
        if (KIND == GEMM_BQ)
          store_accumulator(tmem, warp, lane, leader, stg, &maps[t.x].Praw, &maps[t.x].PTraw_t, L.r, L.m, tr * 128,
                            ecount, 1, 0, 1);
        else
          store_r_tile(tmem, warp, lane, leader, stg, maps[t.x], L, tr, ecount);
      }
      tc_fence_before();
      named_sync(1, 128);  // every thread's TMEM reads of this accumulator are done
      if (leader) mbar_arrive_cluster(cluster_addr(acc_empty, 0));
      ++tcount;
    }
    if (leader) bulk_wait<0>();
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();  // both CTAs are done with the pair's TMEM and barriers
  tc_fence_after();
  if (warp == 1) tmem_dealloc_pair(tmem, tmem_cols);
}

// ================================================================== Q -> bf16 copy ===
__global__ void __launch_bounds__(256) qn_refresh_kernel(Shared sh, const int4 *tiles) {
  const int4 t = tiles[blockIdx.x];  // {layer, first row, rows, 0}
  const DevLayer &L = sh.layers[t.x];
  const int64_t r = L.r, total = (int64_t)t.z * r;
  for (int64_t e = threadIdx.x; e < total; e += 256) {
    const int64_t i = t.y + e / r, j = e % r;
    L.Qn_hi[i * L.ldp + j] = __float2bfloat16_rn(L.Q[i * L.ldq + j]);
  }
}

// ======================================================================= launchers ===
uint32_t form_bq_smem(int nstages, uint32_t stage_bytes) {
  return 1024u + nstages * stage_bytes + 4 * EPI_BOX + 512u;  // + barriers
}
uint32_t btp_smem(int nstages, uint32_t stage_bytes) { return form_bq_smem(nstages, stage_bytes); }

cudaError_t setup_bq_kernels(uint32_t f_smem, uint32_t r_smem) {
  cudaError_t e =
      cudaFuncSetAttribute(tc_tma_gemm_kernel<GEMM_BQ>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)f_smem);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(tc_tma_gemm_kernel<GEMM_BTP>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)r_smem);
  return e;
}

void launch_form_bq(const Shared &sh, const TcPlan &tp, cudaStream_t s) {
  if (tp.d_bq.grid <= 0) return;
  const uint32_t stage = OPB_A + tp.bq_boxes * BOX64;
  tc_tma_gemm_kernel<GEMM_BQ><<<2 * tp.d_bq.grid, R_THREADS, tp.f_smem, s>>>(sh, tp.d_bq.tiles, tp.d_bq.off,
                                                                             tp.maps, tp.f_stages, stage, tp.tmem_cols);
}

void launch_btp(const Shared &sh, const TcPlan &tp, cudaStream_t s) {
  if (tp.d_btp.grid <= 0) return;
  const uint32_t stage = OPB_A + tp.bq_boxes * BOX64;
  tc_tma_gemm_kernel<GEMM_BTP><<<2 * tp.d_btp.grid, R_THREADS, tp.r_smem, s>>>(sh, tp.d_btp.tiles, tp.d_btp.off,
                                                                               tp.maps, tp.r_stages, stage, tp.tmem_cols);
}

void launch_qn_refresh(const Shared &sh, const TcPlan &tp, cudaStream_t s) {
  if (tp.n_qtiles > 0) qn_refresh_kernel<<<tp.n_qtiles, 256, 0, s>>>(sh, tp.qtiles);
}

// ColumnNormalize from the per-tile column sums of squares: colinv[j] = 1 / (||R_j|| + eps),
// fixed-order fp64 sum over the R tiles of the layer.  Grid: one block per (layer, 32 columns).
__global__ void __launch_bounds__(256) colnorm_reduce_kernel(Shared sh, const int4 *ctiles, float eps_col) {
  const int4 t = ctiles[blockIdx.x];  // {layer, 32-column group, 0, 0}
  if (!sh.active[t.x]) return;
  const DevLayer &L = sh.layers[t.x];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t j = (int64_t)t.y * 32 + lane;
  __shared__ double part[8][32];
  double acc = 0.0;
  if (j < L.r)
    for (int k = warp; k < L.rtile_cnt; k += 8) acc += L.colsq[(int64_t)k * L.ldp + j];
  part[warp][lane] = acc;
  __syncthreads();
  if (warp == 0 && j < L.r) {
    double s2 = 0.0;
    for (int w = 0; w < 8; ++w) s2 += part[w][lane];
    L.colinv[j] = (float)(1.0 / (sqrt(s2) + (double)eps_col));
  }
}

// Q_t = R diag(colinv) (fp32, caller's buffer) and its bf16 copy; tiles of rows of R.  One
// warp per row, 16-byte loads of R (rows padded to a multiple of 8 floats), the scale factors
// of the lane's columns kept in registers; the caller's Q is written only inside its r columns.
constexpr int kScaleThreads = 256;
__global__ void __launch_bounds__(kScaleThreads) colnorm_scale_kernel(Shared sh, const int4 *tiles) {
  const int4 t = tiles[blockIdx.x];  // {layer, first row, rows, 0}
  if (!sh.active[t.x]) return;
  const DevLayer &L = sh.layers[t.x];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int r = (int)L.r, r4 = (r + 3) / 4;  // r <= 512: at most 4 chunks per lane
  float4 cs[4];
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const int c = 4 * (lane + 32 * k);
    cs[k] = make_float4(c < r ? L.colinv[c] : 0.f, c + 1 < r ? L.colinv[c + 1] : 0.f,
                        c + 2 < r ? L.colinv[c + 2] : 0.f, c + 3 < r ? L.colinv[c + 3] : 0.f);
  }
  for (int64_t i = t.y + warp; i < (int64_t)t.y + t.z; i += kScaleThreads / 32) {
    const float *Rrow = L.R + i * L.ldp;
    float4 rv[4];
#pragma unroll
    for (int k = 0; k < 4; ++k)
      if (lane + 32 * k < r4) rv[k] = *reinterpret_cast<const float4 *>(Rrow + 4 * (lane + 32 * k));
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int c4 = lane + 32 * k;
      if (c4 >= r4) continue;
      const float4 q = make_float4(rv[k].x * cs[k].x, rv[k].y * cs[k].y, rv[k].z * cs[k].z, rv[k].w * cs[k].w);
      const __nv_bfloat162 h01 = __floats2bfloat162_rn(q.x, q.y), h23 = __floats2bfloat162_rn(q.z, q.w);
      uint2 hv;
      hv.x = *reinterpret_cast<const uint32_t *>(&h01);
      hv.y = *reinterpret_cast<const uint32_t *>(&h23);
      *reinterpret_cast<uint2 *>(L.Qn_hi + i * L.ldp + 4 * c4) = hv;  // workspace rows: padded
      float *Qrow = L.Q + i * L.ldq + 4 * c4;
      if (4 * c4 + 4 <= r) {
        *reinterpret_cast<float4 *>(Qrow) = q;
      } else {
        const float qq[4] = {q.x, q.y, q.z, q.w};
        for (int e = 0; e < r - 4 * c4; ++e) Qrow[e] = qq[e];
      }
    }
  }
}

void launch_colnorm_reduce(const Shared &sh, const int4 *ctiles, int32_t n_ctiles, float eps_col, cudaStream_t s) {
  if (n_ctiles > 0) colnorm_reduce_kernel<<<n_ctiles, 256, 0, s>>>(sh, ctiles, eps_col);
}
void launch_colnorm_scale(const Shared &sh, const TcPlan &tp, cudaStream_t s) {
  if (tp.n_qtiles > 0) colnorm_scale_kernel<<<tp.n_qtiles, kScaleThreads, 0, s>>>(sh, tp.qtiles);
}

}  // namespace tc
}  // namespace cd
