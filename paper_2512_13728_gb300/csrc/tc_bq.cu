// tcgen05 kernels of the power iteration and of R (DION_PREC_BF16):
//
//   tc_form_bq   B = M + G written back into M (Algorithm 1/2 buffer line), its bf16 copy
//                Bh, the fp64 per-tile partials of ||B||^2 and ||M_{t-1}||^2 (Algorithm 2's
//                RMMC and Equation 1), and P = B Q_{t-1} (PowerIter) -- one pass over M and G.
//                Tile = 128 rows of one layer; K loop over n in 64-column chunks.
//                  warps 0..7   producers: coalesced loads of M and G, B in registers, stores of
//                               B and Bh, bf16 B into the K-major 128-byte-swizzled A operand;
//                  warp 8       TMA: the bf16 copy of Q (n x r) as an MN-major B operand;
//                  warp 9       MMA: 128 x N x 16 tcgen05.mma (N <= 256 per instruction) into a
//                               128 x r fp32 TMEM accumulator;
//                  warps 10..13 epilogue: TMEM -> swizzled shared boxes -> TMA store of P (fp32).
//   tc_btp       R = B^T P (after Orthogonalize).  Tile = 128 columns of B (rows of R); K loop
//                over m.  A = Bh^T and B = P are both read as MN-major operands straight from
//                the row-major bf16 copies Bh (m x n) and P_hi (m x r), so no transpose is made.
//                  warp 0 TMA, warp 1 MMA, warps 2..5 epilogue (TMA store of R, fp32).
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

// =============================================================== B = M + G, P = B Q ===
constexpr int F_THREADS = 10 * 32;  // 8 producer/epilogue warps, TMA warp, MMA warp

// A chunk (128 rows x 64 columns of B) is produced in two halves of 64 rows.  Each producer
// thread owns 4 groups of 4 columns per half (row = h * 64 + u * 16 + warp * 2 + lane / 16,
// columns 4 * (lane % 16) ..).  All loads of a half are issued before any is used, and the next
// half's loads are in flight while the current half is processed.
template <int GT>
struct RawHalf {
  float4 m[4];
  typename std::conditional<GT == DT_BF16, uint2, float4>::type g[4];
};

template <int GT>
__device__ __forceinline__ void load_half(const DevLayer &L, int64_t r0, int64_t c0, int warp, int lane,
                                          RawHalf<GT> &raw) {
  const int prow = warp * 2 + (lane >> 4), pcol = (lane & 15) * 4;
  const int64_t gc = c0 + pcol;
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    const int64_t gi = r0 + u * 16 + prow;
    if (gi < L.m && gc + 4 <= L.n) {
      raw.m[u] = __ldg(reinterpret_cast<const float4 *>(L.M + gi * L.ldm + gc));
      if constexpr (GT == DT_BF16)
        raw.g[u] = __ldg(reinterpret_cast<const uint2 *>(static_cast<const __nv_bfloat16 *>(L.G) + gi * L.ldg + gc));
      else
        raw.g[u] = __ldg(reinterpret_cast<const float4 *>(static_cast<const float *>(L.G) + gi * L.ldg + gc));
    } else {  // ragged edge: element-wise, zeros outside the matrix
      float mm[4];
      uint32_t gb[4];
      float gf[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const bool in = gi < L.m && gc + e < L.n;
        mm[e] = in ? L.M[gi * L.ldm + gc + e] : 0.f;
        if constexpr (GT == DT_BF16)
          gb[e] = in ? (uint32_t)reinterpret_cast<const uint16_t *>(L.G)[gi * L.ldg + gc + e] : 0u;
        else
          gf[e] = in ? static_cast<const float *>(L.G)[gi * L.ldg + gc + e] : 0.f;
      }
      raw.m[u] = make_float4(mm[0], mm[1], mm[2], mm[3]);
      if constexpr (GT == DT_BF16)
        raw.g[u] = make_uint2(gb[0] | (gb[1] << 16), gb[2] | (gb[3] << 16));
      else
        raw.g[u] = make_float4(gf[0], gf[1], gf[2], gf[3]);
    }
  }
}

// B = M + G for one half: stores of B and Bh, bf16 B into the K-major 128-byte-swizzled A
// operand (zeros outside the matrix), squared-norm sums.  r0 is the half's first row and
// trow its first row inside the 128-row tile.
template <int GT>
__device__ __forceinline__ void process_half(const DevLayer &L, int64_t r0, int trow, int64_t c0, uint8_t *sA,
                                             int warp, int lane, const RawHalf<GT> &raw, float &sb, float &sm) {
  const int prow = warp * 2 + (lane >> 4), pcol = (lane & 15) * 4;
  const int64_t gc = c0 + pcol;
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    const int row = trow + u * 16 + prow;
    const int64_t gi = r0 + u * 16 + prow;
    const float mv[4] = {raw.m[u].x, raw.m[u].y, raw.m[u].z, raw.m[u].w};
    float gv[4];
    if constexpr (GT == DT_BF16) {
      gv[0] = bf16_bits_to_float(raw.g[u].x & 0xffffu); gv[1] = bf16_bits_to_float(raw.g[u].x >> 16);
      gv[2] = bf16_bits_to_float(raw.g[u].y & 0xffffu); gv[3] = bf16_bits_to_float(raw.g[u].y >> 16);
    } else {
      gv[0] = raw.g[u].x; gv[1] = raw.g[u].y; gv[2] = raw.g[u].z; gv[3] = raw.g[u].w;
    }
    float b[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      sm = fmaf(mv[e], mv[e], sm);
      b[e] = mv[e] + gv[e];
      sb = fmaf(b[e], b[e], sb);
    }
    const __nv_bfloat162 h01 = __floats2bfloat162_rn(b[0], b[1]), h23 = __floats2bfloat162_rn(b[2], b[3]);
    uint2 hv;
    hv.x = *reinterpret_cast<const uint32_t *>(&h01);
    hv.y = *reinterpret_cast<const uint32_t *>(&h23);
    if (gi < L.m && gc + 4 <= L.n) {
      *reinterpret_cast<float4 *>(L.M + gi * L.ldm + gc) = make_float4(b[0], b[1], b[2], b[3]);
      *reinterpret_cast<uint2 *>(L.Bh + gi * L.ldbh + gc) = hv;
    } else if (gi < L.m) {
#pragma unroll
      for (int e = 0; e < 4; ++e)
        if (gc + e < L.n) {
          L.M[gi * L.ldm + gc + e] = b[e];
          L.Bh[gi * L.ldbh + gc + e] = __float2bfloat16_rn(b[e]);
        }
    }
    *reinterpret_cast<uint2 *>(sA + sw128_offset((uint32_t)row, (uint32_t)(pcol >> 3)) + (pcol & 7) * 2) = hv;
  }
}

// The producer loop of one tile, in half-chunk steps h = 2 kc + half.
template <int GT>
__device__ __forceinline__ bool produce_tile(const DevLayer &L, int64_t r0, uint8_t *smem, uint32_t stage_bytes,
                                             int nstages, uint64_t *a_full, uint64_t *empty, uint32_t &it, int warp,
                                             int lane, const Abort &ab, int32_t *status, double &vb, double &vm) {
  const int kch = (int)((L.n + 63) / 64), nh = 2 * kch;
  RawHalf<GT> cur, nxt;
  load_half<GT>(L, r0, 0, warp, lane, cur);
  float sb = 0.f, sm = 0.f;
  for (int h = 0; h < nh; ++h) {
    const int kc = h >> 1, half = h & 1;
    if (h + 1 < nh)
      load_half<GT>(L, r0 + ((h + 1) & 1) * 64, (int64_t)((h + 1) >> 1) * 64, warp, lane, nxt);
    const uint32_t s = it % nstages, ph = (it / nstages) & 1u;
    if (half == 0) {
      if (!__all_sync(0xffffffffu, ab.wait(&empty[s], ph ^ 1u, status))) return false;  // warp-uniform
      sb = 0.f;
      sm = 0.f;
    }
    process_half<GT>(L, r0 + half * 64, half * 64, (int64_t)kc * 64, smem + s * stage_bytes, warp, lane, cur, sb, sm);
    if (half == 1) {  // fp32 sums of 32 squares per chunk, folded into fp64
      vb += (double)sb;
      vm += (double)sm;
      fence_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(&a_full[s]);
      ++it;
    }
    if (h + 1 < nh) cur = nxt;
  }
  return true;
}

// 10 warps: at most 3 per SM sub-partition, so up to 168 registers per thread fit the
// 16K-register file of each sub-partition (room for the producers' prefetch).
__global__ void __maxnreg__(168)
    tc_form_bq_kernel(Shared sh, const int4 *__restrict__ tiles, const int *__restrict__ off, const LayerMaps *__restrict__ maps,
                      int nstages, uint32_t stage_bytes, uint32_t tmem_cols) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = align1024(smem_raw);
  uint8_t *stg = smem + nstages * stage_bytes;  // 2 staging buffers of 2 output boxes
  uint64_t *bars = reinterpret_cast<uint64_t *>(stg + 4 * EPI_BOX);
  uint64_t *a_full = bars, *q_full = bars + nstages, *empty = bars + 2 * nstages;
  uint64_t *acc_full = bars + 3 * nstages, *acc_empty = acc_full + 1, *drain = acc_full + 2;
  __shared__ uint32_t tmem_base_s;
  __shared__ int abort_s;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const Abort ab{&abort_s};
  if (threadIdx.x == 0) {
    for (int i = 0; i < nstages; ++i) {
      mbar_init(&a_full[i], 8);  // one arrive per producer warp
      mbar_init(&q_full[i], 1);
      mbar_init(&empty[i], 1);
    }
    mbar_init(acc_full, 1);
    mbar_init(acc_empty, 256);  // all 8 producer/epilogue warps
    mbar_init(drain, 1);
    abort_s = 0;
    fence_mbar_init();
  }
  if (warp == 9) {
    tmem_alloc(&tmem_base_s, tmem_cols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base_s;

  if (warp < 8) {
    // ------------------------------------------------------- producers, then the tile's epilogue
    const int grp = warp >> 2;  // warps 0..3 and 4..7 each cover the 4 TMEM lane quarters
    const bool leader = (lane == 0 && (warp & 3) == 0);
    uint32_t it = 0, tcount = 0, ecount = 0;
    bool ok = true;
    for (int ti = off[blockIdx.x]; ti < off[blockIdx.x + 1] && ok; ++ti) {
      const int4 t = tiles[ti];
      const DevLayer &L = sh.layers[t.x];
      const int64_t r0 = (int64_t)t.y * 128;
      double vb = 0.0, vm = 0.0;
      ok = (L.g_dtype == DT_BF16)
               ? produce_tile<DT_BF16>(L, r0, smem, stage_bytes, nstages, a_full, empty, it, warp, lane, ab, sh.status, vb, vm)
               : produce_tile<DT_FP32>(L, r0, smem, stage_bytes, nstages, a_full, empty, it, warp, lane, ab, sh.status, vb, vm);
      if (!ok) break;
      // each producer warp owns norm-partial slot 8 * tile + warp (fixed-order sum in the gate)
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        vb += __shfl_xor_sync(0xffffffffu, vb, o);
        vm += __shfl_xor_sync(0xffffffffu, vm, o);
      }
      if (lane == 0) {
        sh.bpart[2 * (8 * t.w + warp)] = vb;
        sh.bpart[2 * (8 * t.w + warp) + 1] = vm;
      }
      // epilogue: P (row-major) and P^T of this tile from TMEM
      if (!named_and(3 + grp, 128, ab.wait(acc_full, tcount & 1u, sh.status))) { ok = false; break; }
      tc_fence_after();
      store_accumulator(tmem, warp, lane, leader, stg, &maps[t.x].Praw, &maps[t.x].PTraw_t, L.r, L.m, t.y * 128,
                        ecount, 3 + grp, grp, 2);
      tc_fence_before();
      mbar_arrive(acc_empty);
      ++tcount;
    }
    if (leader) bulk_wait<0>();
  } else if (warp == 8) {
    // ------------------------------------------------------------------ TMA (Q operand)
    if (lane == 0) {
      uint32_t it = 0;
      bool ok = true;
      for (int ti = off[blockIdx.x]; ti < off[blockIdx.x + 1] && ok; ++ti) {
        const int4 t = tiles[ti];
        const DevLayer &L = sh.layers[t.x];
        const LayerMaps *mp = maps + t.x;
        const int kch = (int)((L.n + 63) / 64);
        const int nb = (int)((L.r + 63) / 64);
        for (int kc = 0; kc < kch; ++kc, ++it) {
          const uint32_t s = it % nstages, ph = (it / nstages) & 1u;
          if (!ab.wait(&empty[s], ph ^ 1u, sh.status)) { ok = false; break; }
          uint8_t *sQ = smem + s * stage_bytes + OPB_A;
          mbar_expect_tx(&q_full[s], (uint32_t)nb * BOX64);
          for (int j = 0; j < nb; ++j) tma_load_2d(sQ + j * BOX64, &mp->Qn_mn, &q_full[s], j * 64, kc * 64);
        }
      }
      for (uint32_t k = (it > (uint32_t)nstages ? it - nstages : 0); k < it; ++k)
        mbar_wait(&q_full[k % nstages], (k / nstages) & 1u, sh.status);
    }
  } else if (warp == 9) {
    // ------------------------------------------------------------------ MMA
    if (lane == 0) {
      uint32_t it = 0, tcount = 0;
      bool ok = true;
      for (int ti = off[blockIdx.x]; ti < off[blockIdx.x + 1] && ok; ++ti, ++tcount) {
        const int4 t = tiles[ti];
        const DevLayer &L = sh.layers[t.x];
        const int kch = (int)((L.n + 63) / 64);
        const uint32_t np = rpad16(L.r), nparts = (np + 255) / 256;
        if (!ab.wait(acc_empty, (tcount & 1u) ^ 1u, sh.status)) break;
        tc_fence_after();
        for (int kc = 0; kc < kch; ++kc, ++it) {
          const uint32_t s = it % nstages, ph = (it / nstages) & 1u;
          if (!ab.wait(&a_full[s], ph, sh.status) || !ab.wait(&q_full[s], ph, sh.status)) { ok = false; break; }
          tc_fence_after();
          const uint32_t aB = smem_u32(smem + s * stage_bytes), qB = aB + OPB_A;
#pragma unroll
          for (int k16 = 0; k16 < 4; ++k16) {
            const uint64_t ad = smem_desc_sw128(aB + k16 * 32, 0, 1024);
            for (uint32_t part = 0; part < nparts; ++part) {
              const uint32_t n_here = min(256u, np - part * 256u);
              const uint64_t bd = smem_desc_sw128(qB + part * 4u * BOX64 + k16 * 2048, BOX64, 1024);
              umma_bf16(tmem + part * 256u, ad, bd, idesc_bf16(128, n_here, false, true), (kc | k16) ? 1u : 0u);
            }
          }
          umma_commit(&empty[s]);
        }
        if (!ok) break;
        umma_commit(acc_full);
      }
      umma_commit(drain);
      mbar_wait(drain, 0, sh.status);
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 9) tmem_dealloc(tmem, tmem_cols);
}

// ========================================================================= R = B^T P ===
constexpr int R_THREADS = 6 * 32;

__global__ void __launch_bounds__(R_THREADS, 1)
    tc_btp_kernel(Shared sh, const int4 *__restrict__ tiles, const int *__restrict__ off, const LayerMaps *__restrict__ maps,
                  int nstages, uint32_t stage_bytes, uint32_t tmem_cols) {
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
  if (threadIdx.x == 0) {
    for (int i = 0; i < nstages; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], 1);
    }
    mbar_init(acc_full, 1);
    mbar_init(acc_empty, 128);
    mbar_init(drain, 1);
    abort_s = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(&tmem_base_s, tmem_cols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base_s;

  if (warp == 0) {
    if (lane == 0) {
      uint32_t it = 0;
      bool ok = true;
      for (int ti = off[blockIdx.x]; ti < off[blockIdx.x + 1] && ok; ++ti) {
        const int4 t = tiles[ti];
        if (!sh.active[t.x]) continue;
        const DevLayer &L = sh.layers[t.x];
        const LayerMaps *mp = maps + t.x;
        const int kch = (int)((L.m + 63) / 64);
        const int nb = (int)((L.r + 63) / 64);
        for (int kc = 0; kc < kch; ++kc, ++it) {
          const uint32_t s = it % nstages, ph = (it / nstages) & 1u;
          if (!ab.wait(&empty[s], ph ^ 1u, sh.status)) { ok = false; break; }
          uint8_t *sA = smem + s * stage_bytes, *sB = sA + OPB_A;
          mbar_expect_tx(&full[s], OPB_A + (uint32_t)nb * BOX64);
          tma_load_2d(sA, &mp->Bh_mn, &full[s], t.y * 128, kc * 64);
          tma_load_2d(sA + BOX64, &mp->Bh_mn, &full[s], t.y * 128 + 64, kc * 64);
          for (int j = 0; j < nb; ++j) tma_load_2d(sB + j * BOX64, &mp->P_mn, &full[s], j * 64, kc * 64);
        }
      }
      for (uint32_t k = (it > (uint32_t)nstages ? it - nstages : 0); k < it; ++k)
        mbar_wait(&full[k % nstages], (k / nstages) & 1u, sh.status);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      uint32_t it = 0, tcount = 0;
      bool ok = true;
      for (int ti = off[blockIdx.x]; ti < off[blockIdx.x + 1] && ok; ++ti) {
        const int4 t = tiles[ti];
        if (!sh.active[t.x]) continue;
        const DevLayer &L = sh.layers[t.x];
        const int kch = (int)((L.m + 63) / 64);
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
            const uint64_t ad = smem_desc_sw128(aB + k16 * 2048, BOX64, 1024);
            for (uint32_t part = 0; part < nparts; ++part) {
              const uint32_t n_here = min(256u, np - part * 256u);
              const uint64_t bd = smem_desc_sw128(bB + part * 4u * BOX64 + k16 * 2048, BOX64, 1024);
              umma_bf16(tmem + part * 256u, ad, bd, idesc_bf16(128, n_here, true, true), (kc | k16) ? 1u : 0u);
            }
          }
          umma_commit(&empty[s]);
        }
        if (!ok) break;
        umma_commit(acc_full);
        ++tcount;
      }
      umma_commit(drain);
      mbar_wait(drain, 0, sh.status);
    }
  } else {
    const bool leader = (warp == 2 && lane == 0);
    uint32_t tcount = 0, ecount = 0;
    for (int ti = off[blockIdx.x]; ti < off[blockIdx.x + 1]; ++ti) {
      const int4 t = tiles[ti];
      if (!sh.active[t.x]) continue;
      const DevLayer &L = sh.layers[t.x];
      if (!named_and(1, 128, ab.wait(acc_full, tcount & 1u, sh.status))) break;
      tc_fence_after();
      store_r_tile(tmem, warp, lane, leader, stg, maps[t.x], L, t.y, ecount);
      tc_fence_before();
      mbar_arrive(acc_empty);
      ++tcount;
    }
    if (leader) bulk_wait<0>();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, tmem_cols);
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
  cudaError_t e = cudaFuncSetAttribute(tc_form_bq_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)f_smem);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(tc_btp_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)r_smem);
  return e;
}

void launch_form_bq(const Shared &sh, const TcPlan &tp, cudaStream_t s) {
  if (tp.d_bq.grid <= 0) return;
  const uint32_t stage = OPB_A + tp.nb64 * BOX64;
  tc_form_bq_kernel<<<tp.d_bq.grid, F_THREADS, tp.f_smem, s>>>(sh, tp.d_bq.tiles, tp.d_bq.off, tp.maps,
                                                               tp.f_stages, stage, tp.tmem_cols);
}

void launch_btp(const Shared &sh, const TcPlan &tp, cudaStream_t s) {
  if (tp.d_btp.grid <= 0) return;
  const uint32_t stage = OPB_A + tp.nb64 * BOX64;
  tc_btp_kernel<<<tp.d_btp.grid, R_THREADS, tp.r_smem, s>>>(sh, tp.d_btp.tiles, tp.d_btp.off, tp.maps,
                                                            tp.r_stages, stage, tp.tmem_cols);
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

// Q_t = R diag(colinv) (fp32, caller's buffer) and its bf16 copy; tiles of rows of R.
__global__ void __launch_bounds__(256) colnorm_scale_kernel(Shared sh, const int4 *tiles) {
  const int4 t = tiles[blockIdx.x];  // {layer, first row, rows, 0}
  if (!sh.active[t.x]) return;
  const DevLayer &L = sh.layers[t.x];
  const int64_t r = L.r, total = (int64_t)t.z * r;
  for (int64_t e = threadIdx.x; e < total; e += 256) {
    const int64_t i = t.y + e / r, j = e % r;
    const float q = L.R[i * L.ldp + j] * L.colinv[j];
    L.Q[i * L.ldq + j] = q;
    L.Qn_hi[i * L.ldp + j] = __float2bfloat16_rn(q);
  }
}

void launch_colnorm_reduce(const Shared &sh, const int4 *ctiles, int32_t n_ctiles, float eps_col, cudaStream_t s) {
  if (n_ctiles > 0) colnorm_reduce_kernel<<<n_ctiles, 256, 0, s>>>(sh, ctiles, eps_col);
}
void launch_colnorm_scale(const Shared &sh, const TcPlan &tp, cudaStream_t s) {
  if (tp.n_qtiles > 0) colnorm_scale_kernel<<<tp.n_qtiles, 256, 0, s>>>(sh, tp.qtiles);
}

}  // namespace tc
}  // namespace cd
