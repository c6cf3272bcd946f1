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

#include <algorithm>
#include <type_traits>

namespace cd {
namespace tc {

constexpr uint32_t OPB_A = 128u * 64u * 2u;   // 128 x 64 bf16 A-operand tile (16 KB)
constexpr uint32_t BOX64 = 64u * 64u * 2u;    // 64 x 64 bf16 MN-major box (8 KB)
constexpr uint32_t EPI_BOX = 128u * 32u * 4u; // 128 x 32 fp32 output box (16 KB)
// epilogue staging of the GEMM kernels: 4 boxes + 1 KB of column partials (R = B^T P)
constexpr uint32_t STG_BYTES = 4u * EPI_BOX + 1024u;

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
template <bool X3>
__device__ __forceinline__ void store_r_tile(uint32_t tmem, int warp, int lane, bool leader, uint8_t *stg,
                                             const LayerMaps &mp, const DevLayer &L, int tile, uint32_t &ecount) {
  const uint32_t lg = (uint32_t)(warp & 3), row = 32u * lg + lane;
  const int et = (warp - 2) * 32 + lane;  // 0..127 within the epilogue warps (warps 2..5)
  const int nch = (int)((L.r + 31) / 32), row0 = tile * 128;
  // staging: [fp32 box 16 KB][fp32 box 16 KB][bf16 box 16 KB][bf16 low-half box 16 KB (BF16X3)]
  // + column-partial scratch 2 x 128 floats
  uint8_t *f0 = stg, *f1 = stg + EPI_BOX, *hb = stg + 2 * EPI_BOX, *lb = stg + 3 * EPI_BOX;
  float *red = reinterpret_cast<float *>(stg + 4 * EPI_BOX);
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
        const uint32_t bo = sw128_offset(row, (uint32_t)(h * 4 + (q >> 1))) + (q & 1) * 8;
        *reinterpret_cast<uint2 *>(hb + bo) = hv;
        if (X3) {  // low halves: x - bf16(x), rounded to bf16
          const float2 af = __bfloat1622float2(a), bf = __bfloat1622float2(b);
          const __nv_bfloat162 al = __floats2bfloat162_rn(__uint_as_float(v[4 * q]) - af.x,
                                                          __uint_as_float(v[4 * q + 1]) - af.y);
          const __nv_bfloat162 bl = __floats2bfloat162_rn(__uint_as_float(v[4 * q + 2]) - bf.x,
                                                          __uint_as_float(v[4 * q + 3]) - bf.y);
          uint2 lv;
          lv.x = *reinterpret_cast<const uint32_t *>(&al);
          lv.y = *reinterpret_cast<const uint32_t *>(&bl);
          *reinterpret_cast<uint2 *>(lb + bo) = lv;
        }
      }
    }
    if (!two) {  // a lone last chunk: zero the unused half of the bf16 box (clipped by the store anyway)
#pragma unroll
      for (int q = 4; q < 8; ++q) {
        *reinterpret_cast<uint4 *>(hb + sw128_offset(row, q)) = make_uint4(0, 0, 0, 0);
        if (X3) *reinterpret_cast<uint4 *>(lb + sw128_offset(row, q)) = make_uint4(0, 0, 0, 0);
      }
    }
    fence_async_smem();
    named_sync(1, 128);
    if (leader) {
      tma_store_2d(&mp.Rst, f0, j * 32, row0);
      if (two) tma_store_2d(&mp.Rst, f1, (j + 1) * 32, row0);
      tma_store_2d(&mp.R_hi, hb, j * 32, row0);
      if (X3) tma_store_2d(&mp.R_lo, lb, j * 32, row0);
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
// X3 (DION_PREC_BF16X3): each operand comes as a high and a low bf16 half, a stage holds
// [A hi][A lo][B hi boxes][B lo boxes], and every k-step issues A_hi B_hi + A_hi B_lo + A_lo B_hi
// into the same accumulator (the A_lo B_lo term, 2^-18 relative, is left out).
template <int KIND, bool X3>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(R_THREADS, 1)
    tc_tma_gemm_kernel(Shared sh, const int4 *__restrict__ tiles, const int *__restrict__ off,
                       const LayerMaps *__restrict__ maps, int nstages, uint32_t stage_bytes, uint32_t tmem_cols) {
  if (sh.gate_scratch[kScratchActive] == 0ull) return;  // no layer takes the Dion branch
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = align1024(smem_raw);
  uint8_t *stg = smem + nstages * stage_bytes;
  uint64_t *bars = reinterpret_cast<uint64_t *>(stg + STG_BYTES);
  constexpr uint32_t A_BYTES = (X3 ? 2u : 1u) * OPB_A;  // the A halves of a stage
  const uint32_t b_half = X3 ? (stage_bytes - A_BYTES) / 2u : 0u;  // offset of the B low boxes
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
          uint8_t *sA = smem + s * stage_bytes, *sB = sA + A_BYTES;
          const uint32_t fb = cluster_addr(&full[s], 0);
          if (rank == 0) mbar_expect_tx(&full[s], 2u * (X3 ? 2u : 1u) * (OPB_A + nbox * BOX64));
          for (int hl = 0; hl < (X3 ? 2 : 1); ++hl) {  // high half, then (BF16X3) low half
            uint8_t *a = sA + hl * OPB_A;
            if (KIND == GEMM_BQ) {
              tma_load_2d_pair(a, hl ? &mp->Bl_k : &mp->Bh_k, fb, kc * 64, tr * 128);
            } else {
              const CUtensorMap *am = hl ? &mp->Bl_mn : &mp->Bh_mn;
              tma_load_2d_pair(a, am, fb, tr * 128, kc * 64);
              tma_load_2d_pair(a + BOX64, am, fb, tr * 128 + 64, kc * 64);
            }
            const CUtensorMap *bmap = (KIND == GEMM_BQ) ? (hl ? &mp->Qn_lo_mn : &mp->Qn_mn)
                                                        : (hl ? &mp->P_lo_mn : &mp->P_mn);
            uint8_t *b = sB + hl * b_half;
            for (uint32_t part = 0; part < nparts; ++part) {
              const uint32_t hc = half_cols(np, part);
              const int x0 = (int)(part * 256u + rank * hc);
              for (uint32_t j = 0; j < (hc + 63) / 64; ++j)
                tma_load_2d_pair(b + (part * 2u + j) * BOX64, bmap, fb, x0 + (int)j * 64, kc * 64);
            }
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
          const uint32_t aB = smem_u32(smem + s * stage_bytes), bB = aB + A_BYTES;
#pragma unroll
          for (int k16 = 0; k16 < 4; ++k16) {
            // A: K-major (B Q) advances 32 bytes per 16 k; MN-major (B^T P) two 8-row groups
            const uint32_t ak = (KIND == GEMM_BQ) ? (uint32_t)k16 * 32u : (uint32_t)k16 * 2048u;
            const uint32_t albo = (KIND == GEMM_BQ) ? 0u : BOX64;
            const uint64_t ad = smem_desc_sw128(aB + ak, albo, 1024);
            for (uint32_t part = 0; part < nparts; ++part) {
              const uint32_t n_here = 2u * half_cols(np, part);
              const uint32_t idesc = idesc_bf16(256, n_here, KIND == GEMM_BTP, true);
              const uint32_t bo = part * 2u * BOX64 + k16 * 2048;
              const uint64_t bd = smem_desc_sw128(bB + bo, BOX64, 1024);
              umma_pair_bf16(tmem + part * 256u, ad, bd, idesc, (kc | k16) ? 1u : 0u);
              if (X3) {
                umma_pair_bf16(tmem + part * 256u, ad, smem_desc_sw128(bB + b_half + bo, BOX64, 1024), idesc, 1u);
                umma_pair_bf16(tmem + part * 256u, smem_desc_sw128(aB + OPB_A + ak, albo, 1024), bd, idesc, 1u);
              }
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
          store_r_tile<X3>(tmem, warp, lane, leader, stg, maps[t.x], L, tr, ecount);
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

// ============================================== buffer pass fused with P = B Q_{t-1} ===
// Algorithm 1/2 with bf16 gradients: B = M_{t-1} + G is formed on the fly from TMA tiles of M
// (fp32) and G (bf16) and fed to the pair MMA of P = B Q_{t-1}, so B is read from HBM once.
// Per {layer, pair p} (CTA c owns 128-row tile 2 p + c) and 64-column k-chunk:
//   warps 12..15 M through the load/store path: 16-byte cp.async copies written in the same
//               swizzled layout as two 128 x 32 fp32 SW128 boxes, into the M ring (zero-filled
//               past the matrix); their landing completes the slot's barrier.  (Each SM's TMA
//               unit already carries G, Q, Bh and P: M, the largest stream, goes around it);
//   warp 0      TMA: G as one 128 x 64 bf16 SW128 box into the A ring;
//   warps 6..9  B = M + G in fp32, rounded to bf16 and written in place over the G box, which
//               has the layout of the K-major A operand; the per-tile sums of B^2 and M_{t-1}^2
//               (Algorithm 2's ||B|| and Equation 1's ||M_{t-1}||).  The M stage is free again
//               as soon as it is converted;
//   warp 11     TMA store of each converted box to Bh (the operand of B^T P); the A slot is
//               refilled once that store has read it and the chunk's MMAs have completed;
//   warp 10     TMA: this CTA's half of the Q_{t-1} chunk (MN-major boxes, bytes counted on
//               CTA 0's barrier) into the Q ring;
//   warp 1      (CTA 0) the pair MMAs of the chunk once both CTAs' A boxes and Q halves are in;
//   warps 2..5  drain the 128 x r accumulator into P_raw and its transpose (as in B Q), staged
//               through the Q ring: the next tile's MMAs wait for TMEM anyway, so its Q loads
//               wait until the staged stores have been read.
// Separate rings keep each slot's turnaround short: an M slot waits for one load and one
// conversion, an A slot for the load, conversion, MMA and store.
// With `gated` (the gated modes) the norms pass has already written B into M, computed the
// norms and run the gate: every role skips the layers that stay local, warp 0 loads no G (it
// only marks the A slot full) and the converters round M itself and form no norms.
constexpr int FB_MSTAGES = 3;  // M ring (2 x 16 KB per slot)
constexpr int FB_ASTAGES = 4;  // G / A ring (16 KB per slot)
constexpr int FB_QSTAGES = 2;  // Q ring (also the epilogue's staging)
constexpr int FB_THREADS = 16 * 32;
constexpr int FB_LOADERS = 128;  // threads of warps 12..15
constexpr uint32_t FB_MBOX = 128u * 32u * 4u;  // 128 x 32 fp32 box of M (16 KB)
constexpr uint32_t FB_GBOX = 128u * 64u * 2u;  // 128 x 64 bf16 box of G, then of B (16 KB)
constexpr uint32_t FB_MSLOT = 2u * FB_MBOX;
constexpr uint32_t FB_A_OFF = FB_MSTAGES * FB_MSLOT;
constexpr uint32_t FB_Q_OFF = FB_A_OFF + FB_ASTAGES * FB_GBOX;

__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(FB_THREADS, 1)
    tc_form_bq_kernel(Shared sh, const int4 *__restrict__ tiles, const int *__restrict__ off,
                      const LayerMaps *__restrict__ maps, uint32_t qstage_bytes, uint32_t qring_bytes,
                      uint32_t tmem_cols, int gated) {
  // gated: the norms pass and the gate ran first; only Dion-branch layers are processed and the
  // norm partials are not written again
  if (gated && sh.gate_scratch[kScratchActive] == 0ull) return;
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = align1024(smem_raw);
  uint8_t *aring = smem + FB_A_OFF;
  uint8_t *qring = smem + FB_Q_OFF;  // Q stages; the epilogue's staging between tiles
  uint64_t *bars = reinterpret_cast<uint64_t *>(qring + qring_bytes);
  uint64_t *mfull = bars, *mempty = mfull + FB_MSTAGES;
  uint64_t *gfull = mempty + FB_MSTAGES, *gempty = gfull + FB_ASTAGES, *afull = gempty + FB_ASTAGES,
           *cvt = afull + FB_ASTAGES;
  uint64_t *qfull = cvt + FB_ASTAGES, *qempty = qfull + FB_QSTAGES;
  uint64_t *acc_full = qempty + FB_QSTAGES, *acc_empty = acc_full + 1, *epi_free = acc_full + 2,
           *drain = acc_full + 3;
  __shared__ uint32_t tmem_base_s;
  __shared__ int abort_s;
  __shared__ double red_s[2][4];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const Abort ab{&abort_s};
  const uint32_t rank = cluster_ctarank();
  const int seg = blockIdx.x >> 1;
  if (threadIdx.x == 0) {
    for (int i = 0; i < FB_MSTAGES; ++i) {
      mbar_init(&mfull[i], FB_LOADERS);  // every loader thread's copies of this CTA's M chunk
      mbar_init(&mempty[i], 1);  // converted
    }
    for (int i = 0; i < FB_ASTAGES; ++i) {
      mbar_init(&gfull[i], 1);   // this CTA's G box
      mbar_init(&gempty[i], 2);  // pair commit after the chunk's MMAs + this CTA's Bh store read
      mbar_init(&afull[i], 2);   // used in CTA 0: one arrival per CTA's converted A box
      mbar_init(&cvt[i], 1);     // this CTA's box is converted (for the Bh store)
    }
    for (int i = 0; i < FB_QSTAGES; ++i) {
      mbar_init(&qfull[i], 1);   // used in CTA 0: its arm, both CTAs' Q bytes
      mbar_init(&qempty[i], 1);  // pair commit after the chunk's MMAs
    }
    mbar_init(acc_full, 1);
    mbar_init(acc_empty, 2);  // used in CTA 0: one arrival per CTA's epilogue
    mbar_init(epi_free, 1);   // this CTA's staged epilogue stores have been read
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
  cluster_sync();
  const uint32_t tmem = tmem_base_s;
  auto half_cols = [](uint32_t np, uint32_t part) { return min(256u, np - part * 256u) / 2u; };

  if (warp == 0) {  // G loads
    if (lane == 0) {
      uint32_t it = 0;
      bool ok = true;
      for (int ti = off[seg]; ti < off[seg + 1] && ok; ++ti) {
        const int4 t = tiles[ti];
        if (gated && !sh.active[t.x]) continue;
        const DevLayer &L = sh.layers[t.x];
        const LayerMaps *mp = maps + t.x;
        const int kch = (int)((L.n + 63) / 64);
        const int tr = 2 * t.y + (int)rank;  // past the last tile: zero-filled, not stored
        for (int kc = 0; kc < kch; ++kc, ++it) {
          const uint32_t sg = it % FB_ASTAGES, pg = (it / FB_ASTAGES) & 1u;
          if (!ab.wait(&gempty[sg], pg ^ 1u, sh.status)) { ok = false; break; }
          if (gated) {  // B is already in M: the slot only receives the converted A box
            mbar_arrive(&gfull[sg]);
            continue;
          }
          mbar_expect_tx(&gfull[sg], FB_GBOX);
          tma_load_2d(aring + sg * FB_GBOX, &mp->Gh64, &gfull[sg], kc * 64, tr * 128);
        }
      }
      for (uint32_t k = (it > (uint32_t)FB_ASTAGES ? it - FB_ASTAGES : 0); k < it; ++k)
        mbar_wait(&gempty[k % FB_ASTAGES], (k / FB_ASTAGES) & 1u, sh.status);
    }
  } else if (warp >= 12) {  // M loads (cp.async)
    const int lt = threadIdx.x - 12 * 32;  // 0..127
    uint32_t it = 0;
    for (int ti = off[seg]; ti < off[seg + 1]; ++ti) {
      const int4 t = tiles[ti];
      if (gated && !sh.active[t.x]) continue;
      const DevLayer &L = sh.layers[t.x];
      const int kch = (int)((L.n + 63) / 64);
      const int64_t row0 = (int64_t)(2 * t.y + (int)rank) * 128;
      bool ok = true;
      for (int kc = 0; kc < kch; ++kc, ++it) {
        const uint32_t sm = it % FB_MSTAGES, pm = (it / FB_MSTAGES) & 1u;
        if (!named_and(3, FB_LOADERS, ab.wait(&mempty[sm], pm ^ 1u, sh.status))) { ok = false; break; }
        uint8_t *sM = smem + sm * FB_MSLOT;
#pragma unroll 4
        for (int i = 0; i < 16; ++i) {
          // copy e: row e >> 4, 16-byte chunk e & 15 of the row's 64 columns (a warp covers two
          // whole 256-byte row segments); box = chunk >> 3, swizzled chunk within the box
          const uint32_t e = (uint32_t)(i * FB_LOADERS + lt), row = e >> 4, c16 = e & 15u;
          const uint32_t box = c16 >> 3, ch = c16 & 7u;
          uint8_t *dst = sM + box * FB_MBOX + row * 128u + ((ch ^ (row & 7u)) << 4);
          const int64_t gr = row0 + row, gc = (int64_t)kc * 64 + 4 * c16;
          const bool in = gr < L.m && gc < L.n;
          const uint32_t bytes = in ? (uint32_t)((L.n - gc < 4 ? L.n - gc : 4) * 4) : 0u;
          cp_async16(dst, in ? (const void *)(L.M + gr * L.ldm + gc) : (const void *)L.M, bytes);
        }
        cp_async_arrive(&mfull[sm]);
      }
      if (!ok) break;
    }
    cp_async_wait_all();
  } else if (warp == 10) {  // Q loads
    if (lane == 0) {
      uint32_t it = 0, tcount = 0;
      bool ok = true;
      for (int ti = off[seg]; ti < off[seg + 1] && ok; ++ti) {
        const int4 t = tiles[ti];
        if (gated && !sh.active[t.x]) continue;
        const DevLayer &L = sh.layers[t.x];
        const LayerMaps *mp = maps + t.x;
        const int kch = (int)((L.n + 63) / 64);
        const uint32_t np = rpad16(L.r), nparts = (np + 255) / 256;
        uint32_t nbox = 0;
        for (uint32_t part = 0; part < nparts; ++part) nbox += (half_cols(np, part) + 63) / 64;
        // the ring holds the previous tile's staged accumulator until its stores have read it
        if (tcount > 0 && !ab.wait(epi_free, (tcount - 1) & 1u, sh.status)) break;
        ++tcount;
        for (int kc = 0; kc < kch; ++kc, ++it) {
          const uint32_t s = it % FB_QSTAGES, ph = (it / FB_QSTAGES) & 1u;
          if (!ab.wait(&qempty[s], ph ^ 1u, sh.status)) { ok = false; break; }
          uint8_t *sQ = qring + s * qstage_bytes;
          const uint32_t qb = cluster_addr(&qfull[s], 0);
          if (rank == 0) mbar_expect_tx(&qfull[s], 2u * nbox * BOX64);
          for (uint32_t part = 0; part < nparts; ++part) {
            const uint32_t hc = half_cols(np, part);
            const int x0 = (int)(part * 256u + rank * hc);
            for (uint32_t j = 0; j < (hc + 63) / 64; ++j)
              tma_load_2d_pair(sQ + (part * 2u + j) * BOX64, &mp->Qn_mn, qb, x0 + (int)j * 64, kc * 64);
          }
        }
      }
      for (uint32_t k = (it > (uint32_t)FB_QSTAGES ? it - FB_QSTAGES : 0); k < it; ++k)
        mbar_wait(&qempty[k % FB_QSTAGES], (k / FB_QSTAGES) & 1u, sh.status);
    }
  } else if (warp == 11) {  // Bh stores
    if (lane == 0) {
      uint32_t it = 0;
      bool ok = true;
      for (int ti = off[seg]; ti < off[seg + 1] && ok; ++ti) {
        const int4 t = tiles[ti];
        if (gated && !sh.active[t.x]) continue;
        const DevLayer &L = sh.layers[t.x];
        const int kch = (int)((L.n + 63) / 64);
        const int tr = 2 * t.y + (int)rank;
        const bool real = (int64_t)tr * 128 < L.m;
        for (int kc = 0; kc < kch; ++kc, ++it) {
          const uint32_t sg = it % FB_ASTAGES, pg = (it / FB_ASTAGES) & 1u;
          if (!ab.wait(&cvt[sg], pg, sh.status)) { ok = false; break; }
          if (real) {
            tma_store_2d(&maps[t.x].Bh_k, aring + sg * FB_GBOX, kc * 64, tr * 128);
            bulk_commit();
            bulk_wait_read<0>();
          }
          mbar_arrive(&gempty[sg]);
        }
      }
      bulk_wait<0>();
    }
  } else if (warp == 1) {  // MMA issue (CTA 0)
    if (lane == 0 && rank == 0) {
      uint32_t it = 0, tcount = 0;
      bool ok = true;
      for (int ti = off[seg]; ti < off[seg + 1] && ok; ++ti) {
        const int4 t = tiles[ti];
        if (gated && !sh.active[t.x]) continue;
        const DevLayer &L = sh.layers[t.x];
        const int kch = (int)((L.n + 63) / 64);
        const uint32_t np = rpad16(L.r), nparts = (np + 255) / 256;
        if (!ab.wait(acc_empty, (tcount & 1u) ^ 1u, sh.status)) break;
        tc_fence_after();
        for (int kc = 0; kc < kch; ++kc, ++it) {
          const uint32_t sg = it % FB_ASTAGES, pg = (it / FB_ASTAGES) & 1u;
          const uint32_t q = it % FB_QSTAGES, qph = (it / FB_QSTAGES) & 1u;
          if (!ab.wait(&qfull[q], qph, sh.status) || !ab.wait(&afull[sg], pg, sh.status)) { ok = false; break; }
          tc_fence_after();
          const uint32_t aB = smem_u32(aring + sg * FB_GBOX), bB = smem_u32(qring + q * qstage_bytes);
#pragma unroll
          for (int k16 = 0; k16 < 4; ++k16) {
            const uint64_t ad = smem_desc_sw128(aB + k16 * 32, 0, 1024);
            for (uint32_t part = 0; part < nparts; ++part) {
              const uint32_t n_here = 2u * half_cols(np, part);
              const uint64_t bd = smem_desc_sw128(bB + part * 2u * BOX64 + k16 * 2048, BOX64, 1024);
              umma_pair_bf16(tmem + part * 256u, ad, bd, idesc_bf16(256, n_here, false, true), (kc | k16) ? 1u : 0u);
            }
          }
          umma_pair_commit_mc(&gempty[sg], 0x3);
          umma_pair_commit_mc(&qempty[q], 0x3);
        }
        if (!ok) break;
        umma_pair_commit_mc(acc_full, 0x3);
        ++tcount;
      }
      umma_pair_commit(drain);
      mbar_wait(drain, 0, sh.status);
    }
  } else if (warp <= 5) {  // epilogue
    const bool leader = (warp == 2 && lane == 0);
    uint32_t tcount = 0, ecount = 0;
    for (int ti = off[seg]; ti < off[seg + 1]; ++ti) {
      const int4 t = tiles[ti];
      if (gated && !sh.active[t.x]) continue;
      const DevLayer &L = sh.layers[t.x];
      const int tr = 2 * t.y + (int)rank;
      if (!named_and(1, 128, ab.wait(acc_full, tcount & 1u, sh.status))) break;
      tc_fence_after();
      if ((int64_t)tr * 128 < L.m)
        store_accumulator(tmem, warp, lane, leader, qring, &maps[t.x].Praw, &maps[t.x].PTraw_t, L.r, L.m, tr * 128,
                          ecount, 1, 0, 1);
      tc_fence_before();
      named_sync(1, 128);
      if (leader) {
        mbar_arrive_cluster(cluster_addr(acc_empty, 0));
        bulk_wait_read<0>();
        mbar_arrive(epi_free);
      }
      ++tcount;
    }
    if (leader) bulk_wait<0>();
  } else {  // warps 6..9: B = M + G
    const int ct = threadIdx.x - 6 * 32, cw = warp - 6;  // 0..127, 0..3
    uint32_t it = 0;
    for (int ti = off[seg]; ti < off[seg + 1]; ++ti) {
      const int4 t = tiles[ti];
      if (gated && !sh.active[t.x]) continue;
      const DevLayer &L = sh.layers[t.x];
      const int tr = 2 * t.y + (int)rank;
      const int kch = (int)((L.n + 63) / 64);
      double accb = 0.0, accm = 0.0;
      bool ok = true;
      for (int kc = 0; kc < kch; ++kc, ++it) {
        const uint32_t sm = it % FB_MSTAGES, pm = (it / FB_MSTAGES) & 1u;
        const uint32_t sg = it % FB_ASTAGES, pg = (it / FB_ASTAGES) & 1u;
        const bool in = ab.wait(&mfull[sm], pm, sh.status) && ab.wait(&gfull[sg], pg, sh.status);
        if (in) {
          const uint8_t *sM = smem + sm * FB_MSLOT;
          uint8_t *sG = aring + sg * FB_GBOX;
          float fb = 0.f, fm = 0.f;
#pragma unroll 4
          for (int i = 0; i < 8; ++i) {
            // element group e: rows 8 (e >> 6) + (e & 7), 16-byte chunk (e >> 3) & 7 (8 columns);
            // the 8 threads of a shared-memory phase take 8 rows of one chunk (distinct banks)
            const uint32_t e = (uint32_t)(i * 128 + ct);
            const uint32_t row = (e & 7u) + 8u * (e >> 6), c = (e >> 3) & 7u, sw = row & 7u;
            uint4 *ga = reinterpret_cast<uint4 *>(sG + row * 128u + ((c ^ sw) << 4));
            const uint4 g = gated ? make_uint4(0u, 0u, 0u, 0u) : *ga;  // gated: B is in M, no G
            const uint8_t *mrow = sM + (c >> 2) * FB_MBOX + row * 128u;
            const uint32_t mc = 2u * (c & 3u);
            const float4 m0 = *reinterpret_cast<const float4 *>(mrow + ((mc ^ sw) << 4));
            const float4 m1 = *reinterpret_cast<const float4 *>(mrow + (((mc + 1u) ^ sw) << 4));
            const float mv[8] = {m0.x, m0.y, m0.z, m0.w, m1.x, m1.y, m1.z, m1.w};
            const uint32_t gw[4] = {g.x, g.y, g.z, g.w};
            uint32_t hw[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              const float b0 = mv[2 * q] + __uint_as_float(gw[q] << 16);
              const float b1 = mv[2 * q + 1] + __uint_as_float(gw[q] & 0xffff0000u);
              fm = fmaf(mv[2 * q], mv[2 * q], fm);
              fm = fmaf(mv[2 * q + 1], mv[2 * q + 1], fm);
              fb = fmaf(b0, b0, fb);
              fb = fmaf(b1, b1, fb);
              const __nv_bfloat162 h = __floats2bfloat162_rn(b0, b1);
              hw[q] = *reinterpret_cast<const uint32_t *>(&h);
            }
            *ga = make_uint4(hw[0], hw[1], hw[2], hw[3]);
          }
          accb += (double)fb;
          accm += (double)fm;
          fence_async_smem();  // the A box is read by the MMA and the Bh store (async proxy)
        }
        if (!named_and(2, 128, in)) { ok = false; break; }
        if (ct == 0) {
          mbar_arrive(&mempty[sm]);
          mbar_arrive_cluster(cluster_addr(&afull[sg], 0));
          mbar_arrive(&cvt[sg]);
        }
      }
      if (!ok) break;
      // the row tile's sums of B^2 and M_{t-1}^2: fixed-order fp64 reduction
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        accb += __shfl_xor_sync(0xffffffffu, accb, o);
        accm += __shfl_xor_sync(0xffffffffu, accm, o);
      }
      if (lane == 0) {
        red_s[0][cw] = accb;
        red_s[1][cw] = accm;
      }
      named_sync(2, 128);
      if (ct == 0 && !gated && (int64_t)tr * 128 < L.m) {
        const int slot = L.bpart_off + tr;
        sh.bpart[2 * slot] = (red_s[0][0] + red_s[0][1]) + (red_s[0][2] + red_s[0][3]);
        sh.bpart[2 * slot + 1] = (red_s[1][0] + red_s[1][1]) + (red_s[1][2] + red_s[1][3]);
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();
  tc_fence_after();
  if (warp == 1) tmem_dealloc_pair(tmem, tmem_cols);
}

// ================================================================== Q -> bf16 copy ===
__global__ void __launch_bounds__(256) qn_refresh_kernel(Shared sh, const int4 *tiles) {
  const int4 t = tiles[blockIdx.x];  // {layer, first row, rows, 0}
  DION_TILE_CHECK(t.x >= 0 && t.x < sh.num_layers && t.y >= 0 && t.z >= 1 &&
                      (int64_t)t.y + t.z <= sh.layers[t.x].n, sh.status);
  const DevLayer &L = sh.layers[t.x];
  const int64_t r = L.r, total = (int64_t)t.z * r;
  for (int64_t e = threadIdx.x; e < total; e += 256) {
    const int64_t i = t.y + e / r, j = e % r;
    const float q = L.Q[i * L.ldq + j];
    const __nv_bfloat16 h = __float2bfloat16_rn(q);
    L.Qn_hi[i * L.ldp + j] = h;
    if (L.Qn_lo != nullptr) L.Qn_lo[i * L.ldp + j] = __float2bfloat16_rn(q - __bfloat162float(h));
  }
}

// ======================================================================= launchers ===
uint32_t form_bq_smem(int nstages, uint32_t stage_bytes) {
  return 1024u + nstages * stage_bytes + STG_BYTES + 512u;  // + barriers
}
uint32_t btp_smem(int nstages, uint32_t stage_bytes) { return form_bq_smem(nstages, stage_bytes); }
// Q ring of the fused kernel: FB_QSTAGES Q chunks, at least the epilogue's 4 staging boxes
uint32_t fused_bq_qring(uint32_t bq_boxes) { return std::max(FB_QSTAGES * bq_boxes * BOX64, 4u * EPI_BOX); }
uint32_t fused_bq_smem(uint32_t bq_boxes) { return 1024u + FB_Q_OFF + fused_bq_qring(bq_boxes) + 512u; }

cudaError_t setup_bq_kernels(uint32_t f_smem, uint32_t r_smem, bool x3) {
  cudaError_t e = x3 ? cudaFuncSetAttribute(tc_tma_gemm_kernel<GEMM_BQ, true>,
                                            cudaFuncAttributeMaxDynamicSharedMemorySize, (int)f_smem)
                     : cudaFuncSetAttribute(tc_tma_gemm_kernel<GEMM_BQ, false>,
                                            cudaFuncAttributeMaxDynamicSharedMemorySize, (int)f_smem);
  if (e == cudaSuccess)
    e = x3 ? cudaFuncSetAttribute(tc_tma_gemm_kernel<GEMM_BTP, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  (int)r_smem)
           : cudaFuncSetAttribute(tc_tma_gemm_kernel<GEMM_BTP, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  (int)r_smem);
  return e;
}

cudaError_t setup_fused_bq_kernel(uint32_t smem) {
  return cudaFuncSetAttribute(tc_form_bq_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
}

void launch_fused_bq(const Shared &sh, const TcPlan &tp, bool gated, cudaStream_t s) {
  if (tp.d_bq.grid <= 0) return;
  tc_form_bq_kernel<<<2 * tp.d_bq.grid, FB_THREADS, tp.fb_smem, s>>>(
      sh, tp.d_bq.tiles, tp.d_bq.off, tp.maps, tp.bq_boxes * BOX64, fused_bq_qring(tp.bq_boxes), tp.tmem_cols,
      gated ? 1 : 0);
}

void launch_form_bq(const Shared &sh, const TcPlan &tp, cudaStream_t s) {
  if (tp.d_bq.grid <= 0) return;
  const bool x3 = tp.precision == DION_PREC_BF16X3;
  const uint32_t stage = (x3 ? 2u : 1u) * (OPB_A + tp.bq_boxes * BOX64);
  if (x3)
    tc_tma_gemm_kernel<GEMM_BQ, true><<<2 * tp.d_bq.grid, R_THREADS, tp.f_smem, s>>>(
        sh, tp.d_bq.tiles, tp.d_bq.off, tp.maps, tp.f_stages, stage, tp.tmem_cols);
  else
    tc_tma_gemm_kernel<GEMM_BQ, false><<<2 * tp.d_bq.grid, R_THREADS, tp.f_smem, s>>>(
        sh, tp.d_bq.tiles, tp.d_bq.off, tp.maps, tp.f_stages, stage, tp.tmem_cols);
}

void launch_btp(const Shared &sh, const TcPlan &tp, cudaStream_t s) {
  if (tp.d_btp.grid <= 0) return;
  const bool x3 = tp.precision == DION_PREC_BF16X3;
  const uint32_t stage = (x3 ? 2u : 1u) * (OPB_A + tp.bq_boxes * BOX64);
  if (x3)
    tc_tma_gemm_kernel<GEMM_BTP, true><<<2 * tp.d_btp.grid, R_THREADS, tp.r_smem, s>>>(
        sh, tp.d_btp.tiles, tp.d_btp.off, tp.maps, tp.r_stages, stage, tp.tmem_cols);
  else
    tc_tma_gemm_kernel<GEMM_BTP, false><<<2 * tp.d_btp.grid, R_THREADS, tp.r_smem, s>>>(
        sh, tp.d_btp.tiles, tp.d_btp.off, tp.maps, tp.r_stages, stage, tp.tmem_cols);
}

// Data-parallel phases.  P_raw^T (r x m, the first Gram's operand) from the averaged P_raw:
// tile = {layer, 128-row block of P_raw}, 32 x 32 sub-tiles through shared memory.
__global__ void __launch_bounds__(256) transpose_praw_kernel(Shared sh, const int4 *tiles) {
  const int4 t = tiles[blockIdx.x];
  DION_TILE_CHECK(t.x >= 0 && t.x < sh.num_layers && t.y >= 0 && (int64_t)t.y * 128 < sh.layers[t.x].m, sh.status);
  if (!sh.active[t.x]) return;
  const DevLayer &L = sh.layers[t.x];
  __shared__ float tile[32][33];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t row_end = min((int64_t)t.y * 128 + 128, L.m);
  for (int64_t r0 = (int64_t)t.y * 128; r0 < row_end; r0 += 32) {
    for (int64_t c0 = 0; c0 < L.r; c0 += 32) {
      for (int i = warp; i < 32; i += 8) {  // rows r0 + i, columns c0 + lane of P_raw
        const int64_t row = r0 + i, col = c0 + lane;
        tile[i][lane] = (row < row_end && col < L.r) ? L.P_raw[row * L.ldp + col] : 0.f;
      }
      __syncthreads();
      for (int i = warp; i < 32; i += 8) {  // row c0 + i of P_raw^T, columns r0 + lane
        const int64_t col = c0 + i, row = r0 + lane;
        if (col < L.r && row < row_end) L.PT_raw[col * L.ldmt + row] = tile[lane][i];
      }
      __syncthreads();
    }
  }
}

// R's bf16 copy (and low half in BF16X3) and the per-tile column sums of squares that
// ColumnNormalize reads, from the averaged R: tile = {layer, 128-row block of R}; thread j
// takes columns j and j + 256, rows in order (fp32 over 32 rows, then fp64).
__global__ void __launch_bounds__(256) r_refresh_kernel(Shared sh, const int4 *tiles) {
  const int4 t = tiles[blockIdx.x];
  DION_TILE_CHECK(t.x >= 0 && t.x < sh.num_layers && t.y >= 0 && (int64_t)t.y * 128 < sh.layers[t.x].n, sh.status);
  if (!sh.active[t.x]) return;
  const DevLayer &L = sh.layers[t.x];
  const int64_t r0 = (int64_t)t.y * 128, r1 = min(r0 + 128, L.n);
  for (int64_t c = threadIdx.x; c < L.r; c += 256) {
    double acc = 0.0;
    float f = 0.f;
    for (int64_t i = r0; i < r1; ++i) {
      const float v = L.R[i * L.ldp + c];
      f = fmaf(v, v, f);
      if (((i - r0) & 31) == 31) { acc += (double)f; f = 0.f; }
      const __nv_bfloat16 h = __float2bfloat16_rn(v);
      L.R_hi[i * L.ldp + c] = h;
      if (L.R_lo != nullptr) L.R_lo[i * L.ldp + c] = __float2bfloat16_rn(v - __bfloat162float(h));
    }
    L.colsq[(int64_t)t.y * L.ldp + c] = acc + (double)f;
  }
}

void launch_transpose_praw(const Shared &sh, const TcPlan &tp, cudaStream_t s) {
  if (tp.n_trsm_tiles > 0) transpose_praw_kernel<<<tp.n_trsm_tiles, 256, 0, s>>>(sh, tp.trsm_tiles);
}
void launch_r_refresh(const Shared &sh, const TcPlan &tp, cudaStream_t s) {
  if (tp.n_rtiles > 0) r_refresh_kernel<<<tp.n_rtiles, 256, 0, s>>>(sh, tp.rtiles);
}

void launch_qn_refresh(const Shared &sh, const TcPlan &tp, cudaStream_t s) {
  if (tp.n_qtiles > 0) qn_refresh_kernel<<<tp.n_qtiles, 256, 0, s>>>(sh, tp.qtiles);
}

// ColumnNormalize from the per-tile column sums of squares: colinv[j] = 1 / (||R_j|| + eps),
// fixed-order fp64 sum over the R tiles of the layer.  Grid: one block per (layer, 32 columns).
__global__ void __launch_bounds__(256) colnorm_reduce_kernel(Shared sh, const int4 *ctiles, float eps_col) {
  const int4 t = ctiles[blockIdx.x];  // {layer, 32-column group, 0, 0}
  DION_TILE_CHECK(t.x >= 0 && t.x < sh.num_layers && t.y >= 0 && (int64_t)t.y * 32 < sh.layers[t.x].r, sh.status);
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
  DION_TILE_CHECK(t.x >= 0 && t.x < sh.num_layers && t.y >= 0 && t.z >= 1 &&
                      (int64_t)t.y + t.z <= sh.layers[t.x].n, sh.status);
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
      if (L.Qn_lo != nullptr) {  // BF16X3: q - bf16(q), rounded to bf16
        const float2 f01 = __bfloat1622float2(h01), f23 = __bfloat1622float2(h23);
        const __nv_bfloat162 l01 = __floats2bfloat162_rn(q.x - f01.x, q.y - f01.y);
        const __nv_bfloat162 l23 = __floats2bfloat162_rn(q.z - f23.x, q.w - f23.y);
        uint2 lv;
        lv.x = *reinterpret_cast<const uint32_t *>(&l01);
        lv.y = *reinterpret_cast<const uint32_t *>(&l23);
        *reinterpret_cast<uint2 *>(L.Qn_lo + i * L.ldp + 4 * c4) = lv;
      }
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

// ====================================================================== workspace guards ===
__device__ __forceinline__ uint32_t guard_word(int64_t g, int w) {
  return 0xA5A5A5A5u ^ (uint32_t)(g * kGuardWords + w);
}
__global__ void guard_fill_kernel(char *base, const uint64_t *offsets, int32_t n) {
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < (int64_t)n * kGuardWords;
       e += (int64_t)gridDim.x * blockDim.x) {
    const int64_t g = e / kGuardWords;
    const int w = (int)(e % kGuardWords);
    reinterpret_cast<uint32_t *>(base + offsets[g])[w] = guard_word(g, w);
  }
}
__global__ void guard_check_kernel(const char *base, const uint64_t *offsets, int32_t n, int32_t *bad,
                                   int32_t *status) {
  int mine = 0;
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < (int64_t)n * kGuardWords;
       e += (int64_t)gridDim.x * blockDim.x) {
    const int64_t g = e / kGuardWords;
    const int w = (int)(e % kGuardWords);
    mine += reinterpret_cast<const uint32_t *>(base + offsets[g])[w] != guard_word(g, w);
  }
  if (mine) {
    atomicAdd(bad, mine);
    if (status != nullptr) set_status(status, ST_CORRUPT);
  }
}
void launch_guard_fill(char *base, const uint64_t *offsets, int32_t n, cudaStream_t s) {
  if (n > 0) guard_fill_kernel<<<std::min(1024, (n * kGuardWords + 255) / 256), 256, 0, s>>>(base, offsets, n);
}
void launch_guard_check(const char *base, const uint64_t *offsets, int32_t n, int32_t *bad, int32_t *status,
                        cudaStream_t s) {
  if (n > 0)
    guard_check_kernel<<<std::min(1024, (n * kGuardWords + 255) / 256), 256, 0, s>>>(base, offsets, n, bad, status);
}
}  // namespace cd
