// Orthogonalize on tensor cores: the Gram matrix and the triangular solve of each
// CholeskyQR pass as kind::tf32 tcgen05 GEMMs on fp32 operands loaded by TMA (DION_PREC_BF16),
// or as three such products per k-step on split operands (DION_PREC_BF16X3, below).
//
//   Gram   S = X^T X (r x r), lower block triangle; K loop over m.  Operands are rows of the
//          transposed copy X^T (r x m, K-major), which the producing kernel (the B Q epilogue or
//          the previous TRSM) writes next to X.  r <= 256: one pair tile.  r > 256: one tile for
//          the two diagonal 256 x 256 blocks, whose A operands are read in place from their B
//          boxes, and one for the block below the first; each loads two boxes per chunk, so a
//          layer's tiles cost the same, run side by side and read X^T from DRAM about once.
//   TRSM   Y = X L^{-T} (m x r).  Tile = 128 rows of X; K loop over r.  A = rows of X
//          (K-major), B = rows of L^{-1} (K-major, lower triangular: K chunks above a column
//          part are skipped).  Epilogue stores Y (row-major) and Y^T (transposed boxes) for
//          the next pass, or, in the pass that ends Orthogonalize, only the bf16 copy of Y.
//          A tile runs as one sub-tile per 256-column part of N, each accumulated in one of two
//          alternating 256-column TMEM slots, so the epilogue of one sub-tile (the stores that
//          bound the solve) runs under the MMAs of the next; part 1 reads A chunks 0..7 a
//          second time, from L2.
//
// Accuracy: tf32 products (10-bit mantissa) with fp32 accumulation give ~5e-4 relative
// error in S and Y; the second CholeskyQR pass (on an already nearly orthonormal X) brings
// P back to orthonormal to that level, below the bf16 rounding the following kernels apply.
// Both run as pair MMAs over 256-row blocks (two CTAs on two SMs, cta_group::2), so each SM
// receives half of the B operand.  Roles: warp 0 TMA, warp 1 MMA (even CTA), warps 2..5 epilogue.
//
// BF16X3 (fp32-class): every fp32 operand x is split as hi = x with the low 13 mantissa bits
// cleared (exactly a tf32 value) and lo = x - hi (exact in fp32; its own tf32 rounding costs
// ~2^-21 |x|), and each k-step issues hi.hi + hi.lo + lo.hi into the same accumulator (lo.lo,
// ~2^-22 relative, is left out): the 3xTF32 scheme.  The split happens in shared memory, so the
// bytes each SM receives do not change: four converter warps (6..9) wait for a stage's TMA
// loads (counted on each CTA's own barrier), clear the low bits of every box in place, write
// the lo boxes into the second half of the stage, and report the stage to the even CTA, whose
// MMA warp waits for both CTAs' reports.  The solve that ends Orthogonalize writes the bf16
// high and low halves of P that R = B^T P and the update read.
#include "tc.cuh"
#include "tc_common.cuh"
#include "tc_kernels.cuh"

namespace cd {
namespace tc {

constexpr uint32_t O_BOX = 128u * 32u * 4u;  // one fp32 box: 128 rows x 32 (K) = 16 KB
constexpr uint32_t O_TBOX = 32u * 32u * 4u;  // one transposed output box: 32 x 32 fp32 = 4 KB
constexpr int O_THREADS = 6 * 32;
constexpr int O_THREADS_X3 = 10 * 32;  // + four converter warps

enum : int32_t { ORTH_GRAM = 0, ORTH_TRSM = 1 };

__device__ __forceinline__ uint32_t pad16(int64_t v) { return (uint32_t)((v + 15) / 16 * 16); }

struct OrthMaps {
  const CUtensorMap *A, *B, *out, *out_t;
};

template <int KIND>
__device__ __forceinline__ OrthMaps orth_maps(const LayerMaps &mp, int pass) {
  // X_0 = P_raw, X_1 = P, X_2 = P_raw, X_3 = P (ping-pong between the two buffers)
  const bool raw_in = (pass != 1);
  OrthMaps o;
  if (KIND == ORTH_GRAM) {
    o.A = raw_in ? &mp.PTraw : &mp.PT;
    o.B = o.A;
    o.out = &mp.Sst;
    o.out_t = nullptr;
  } else {
    o.A = raw_in ? &mp.Praw : &mp.Pf;
    o.B = &mp.Linv;
    o.out = raw_in ? &mp.Pf : &mp.Praw;
    o.out_t = raw_in ? &mp.PT_t : &mp.PTraw_t;
  }
  return o;
}

// Per tile: N columns and the K extent (the Gram's parts are those of gram_tile below), and
// whether K chunk kc feeds N part p (TRSM: L^{-1} is lower triangular, so column part p needs
// k < 256 (p + 1)).
template <int KIND>
__device__ __forceinline__ void orth_dims(const DevLayer &L, int blk, uint32_t &N, int64_t &K) {
  (void)blk;
  N = pad16(L.r);
  K = (KIND == ORTH_GRAM) ? L.m : L.r;
}

// A Gram pair tile.  Part q is an accumulator of N[q] <= 256 columns at TMEM column 256 q and
// S column 256 q (the first part of tile 1 at r > 256: column 0), fed by the B rows b_row[q] ..
// of X^T (CTA c holds N[q] / 2 of them from b_row[q] + c N[q] / 2) and by the A rows of its 128
// output rows: in place in B's box a_box[q], or the separate A box (rows a_row + 128 c).  Its
// rows of S are the 128-row tile o_row[q] + c.  Output chunk j (32 columns) belongs to part j / 8.
struct GramTile {
  uint32_t nparts, N[2], b_row[2];
  int a_box[2], o_row[2], a_row, nch;
  bool sep_a;
};

__device__ __forceinline__ GramTile gram_tile(int64_t r, int p) {
  GramTile g{};
  const uint32_t np = pad16(r);
  g.nch = (int)((r + 31) / 32);
  if (np <= 256u) {  // rows and columns 0 .. r
    g.nparts = 1;
    g.N[0] = np;
    g.sep_a = np != 256u;
    g.a_box[0] = g.sep_a ? -1 : 0;
  } else if (p == 0) {  // the diagonal blocks: rows and columns 0..255, then 256 .. r
    g.nparts = 2;
    g.N[0] = 256u;
    g.N[1] = np - 256u;
    g.b_row[1] = 256u;
    g.o_row[1] = 2;
    g.a_box[0] = 0;
    g.sep_a = g.N[1] != 256u;
    g.a_box[1] = g.sep_a ? -1 : 1;
    g.a_row = 256;
  } else {  // the block below the first: rows 256 .. r, columns 0..255
    g.nparts = 1;
    g.N[0] = 256u;
    g.o_row[0] = 2;
    g.sep_a = true;
    g.a_box[0] = -1;
    g.a_row = 256;
    g.nch = 8;
  }
  return g;
}

template <int KIND>
__device__ __forceinline__ bool part_needs(int kc, uint32_t part) {
  return (uint32_t)kc * 32u < 256u * (part + 1u);
}

// Run in clusters of two CTAs with pair MMAs (cta_group::2, M = 256): CTA c of the pair owns
// 128 rows of each accumulator part (the TRSM: 128-row tile 2 p + c of X; the Gram: as
// gram_tile says), its A chunk, and of every N part of up to 256 columns the half c of the B
// rows; the even CTA issues the MMAs and each CTA receives its 128 rows of the accumulator in
// its own TMEM.  For a diagonal block of S with a full 256-column part, the CTA's own rows of
// X^T are exactly its B half, so A is read in place.  Tile = {layer, pair p}.
template <int KIND, bool X3>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(X3 ? O_THREADS_X3 : O_THREADS, 1)
    tc_orth_kernel(Shared sh, const int4 *__restrict__ tiles, const int *__restrict__ off, const LayerMaps *__restrict__ maps,
                   int pass, int nstages, uint32_t stage_bytes, uint32_t tmem_cols) {
  if (sh.gate_scratch[kScratchActive] == 0ull) return;  // no layer takes the Dion branch
  if (pass == 2 && sh.gate_scratch[kScratchShifted] == 0ull) return;  // no layer took the shifted retry
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = align1024(smem_raw);
  uint8_t *stg = smem + nstages * stage_bytes;  // 2 x (row box 16 KB + 4 transposed boxes 16 KB)
  uint64_t *bars = reinterpret_cast<uint64_t *>(stg + 4 * O_BOX);
  uint64_t *full = bars, *empty = bars + nstages;
  // two accumulator slots (the TRSM alternates them; the Gram uses slot 0)
  uint64_t *acc_full = bars + 2 * nstages, *acc_empty = acc_full + 2, *drain = acc_full + 4;
  uint64_t *conv = drain + 1;  // BF16X3: a stage's boxes are split in both CTAs (used in CTA 0)
  const uint32_t lo_off = X3 ? stage_bytes / 2u : 0u;  // BF16X3: lo boxes, same layout as the hi half
  __shared__ uint32_t tmem_base_s;
  __shared__ int abort_s;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const Abort ab{&abort_s};
  const uint32_t rank = cluster_ctarank();
  const int seg = blockIdx.x >> 1;
  if (threadIdx.x == 0) {
    for (int i = 0; i < nstages; ++i) {
      mbar_init(&full[i], 1);   // BF16: used in CTA 0, its arm, both CTAs' bytes; BF16X3: this CTA's bytes
      mbar_init(&empty[i], 1);  // pair commit after the stage's MMAs
      if (X3) mbar_init(&conv[i], 2);  // one arrival per CTA's converters
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&acc_full[i], 1);   // pair commit after the (sub-)tile's MMAs
      mbar_init(&acc_empty[i], 2);  // used in CTA 0: one arrival per CTA's epilogue
    }
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
  auto skip = [&](int layer) { return !sh.active[layer] || (pass == 2 && !sh.orth_shifted[layer]); };
  // half of N part q held by each CTA (rows of the B operand)
  auto half_rows = [](uint32_t N, uint32_t q) { return min(256u, N - q * 256u) / 2u; };
  // TMA load of one box of a stage: BF16 counts both CTAs' bytes on CTA 0's barrier, BF16X3
  // each CTA's on its own (its converters wait for them)
  auto load = [&](void *dst, const CUtensorMap *map, uint32_t s, int32_t c0, int32_t c1) {
    if (X3) tma_load_2d(dst, map, &full[s], c0, c1);
    else tma_load_2d_pair(dst, map, cluster_addr(&full[s], 0), c0, c1);
  };
  auto expect = [&](uint32_t s, uint32_t boxes) {
    if (X3) mbar_expect_tx(&full[s], O_BOX * boxes);
    else if (rank == 0) mbar_expect_tx(&full[s], 2u * O_BOX * boxes);
  };

  if (warp == 0) {
    if (lane == 0) {
      uint32_t it = 0;
      bool ok = true;
      for (int ti = off[seg]; ti < off[seg + 1] && ok; ++ti) {
        const int4 t = tiles[ti];
        if (skip(t.x)) continue;
        const DevLayer &L = sh.layers[t.x];
        const OrthMaps om = orth_maps<KIND>(maps[t.x], pass);
        uint32_t N;
        int64_t K;
        orth_dims<KIND>(L, t.y, N, K);
        const int kch = (int)((K + 31) / 32);
        const uint32_t nparts = (N + 255) / 256;
        const int tr = 2 * t.y + (int)rank;  // past the last tile: zero-filled, not stored
        if constexpr (KIND == ORTH_TRSM) {
          // sub-tile q: K chunks below 256 (q + 1); A chunk and part q's B box in each stage
          for (uint32_t q = 0; q < nparts && ok; ++q) {
            const int kq = min(kch, (int)(8u * (q + 1u)));
            for (int kc = 0; kc < kq; ++kc, ++it) {
              const uint32_t s = it % nstages, ph = (it / nstages) & 1u;
              if (!ab.wait(&empty[s], ph ^ 1u, sh.status)) { ok = false; break; }
              uint8_t *sA = smem + s * stage_bytes, *sB = sA + O_BOX;
              expect(s, 2u);
              load(sA, om.A, s, kc * 32, tr * 128);
              load(sB, om.B, s, kc * 32, (int)(q * 256u + rank * half_rows(N, q)));
            }
          }
          continue;
        }
        const GramTile g = gram_tile(L.r, t.y);
        for (int kc = 0; kc < kch; ++kc, ++it) {
          const uint32_t s = it % nstages, ph = (it / nstages) & 1u;
          if (!ab.wait(&empty[s], ph ^ 1u, sh.status)) { ok = false; break; }
          uint8_t *sA = smem + s * stage_bytes, *sB = sA + O_BOX;
          expect(s, (g.sep_a ? 1u : 0u) + g.nparts);
          if (g.sep_a) load(sA, om.A, s, kc * 32, g.a_row + (int)rank * 128);
#pragma unroll
          for (uint32_t q = 0; q < 2u; ++q)
            if (q < g.nparts) load(sB + q * O_BOX, om.B, s, kc * 32, (int)(g.b_row[q] + rank * (g.N[q] / 2u)));
        }
      }
      // drain: the last stages' loads have landed and been consumed (their stage was freed)
      for (uint32_t k = (it > (uint32_t)nstages ? it - nstages : 0); k < it; ++k)
        mbar_wait(&empty[k % nstages], (k / nstages) & 1u, sh.status);
    }
  } else if (X3 && warp >= 6) {
    // converters (BF16X3): split every box of a landed stage, in the order the producer loads
    const int ct = threadIdx.x - 6 * 32;
    auto split_box = [&](uint8_t *box) {
#pragma unroll 4
      for (int i = ct; i < (int)(O_BOX / 16u); i += 128) {
        float4 *hp = reinterpret_cast<float4 *>(box + i * 16);
        const float4 x = *hp;
        float4 h, l;
        h.x = __uint_as_float(__float_as_uint(x.x) & 0xFFFFE000u);
        h.y = __uint_as_float(__float_as_uint(x.y) & 0xFFFFE000u);
        h.z = __uint_as_float(__float_as_uint(x.z) & 0xFFFFE000u);
        h.w = __uint_as_float(__float_as_uint(x.w) & 0xFFFFE000u);
        l.x = x.x - h.x;
        l.y = x.y - h.y;
        l.z = x.z - h.z;
        l.w = x.w - h.w;
        *hp = h;
        *reinterpret_cast<float4 *>(box + lo_off + i * 16) = l;
      }
    };
    auto report = [&](uint32_t s) {
      fence_async_smem();  // the converted boxes are visible to the tensor cores' reads
      named_sync(2, 128);
      if (ct == 0) mbar_arrive_cluster(cluster_addr(&conv[s], 0));
    };
    uint32_t it = 0;
    bool ok = true;
    for (int ti = off[seg]; ti < off[seg + 1] && ok; ++ti) {
      const int4 t = tiles[ti];
      if (skip(t.x)) continue;
      const DevLayer &L = sh.layers[t.x];
      uint32_t N;
      int64_t K;
      orth_dims<KIND>(L, t.y, N, K);
      const int kch = (int)((K + 31) / 32);
      const uint32_t nparts = (N + 255) / 256;
      if constexpr (KIND == ORTH_TRSM) {
        for (uint32_t q = 0; q < nparts && ok; ++q) {
          const int kq = min(kch, (int)(8u * (q + 1u)));
          for (int kc = 0; kc < kq; ++kc, ++it) {
            const uint32_t s = it % nstages, ph = (it / nstages) & 1u;
            if (!named_and(2, 128, ab.wait(&full[s], ph, sh.status))) { ok = false; break; }
            uint8_t *sA = smem + s * stage_bytes;
            split_box(sA);
            split_box(sA + O_BOX);
            report(s);
          }
        }
        continue;
      }
      const GramTile g = gram_tile(L.r, t.y);
      for (int kc = 0; kc < kch; ++kc, ++it) {
        const uint32_t s = it % nstages, ph = (it / nstages) & 1u;
        if (!named_and(2, 128, ab.wait(&full[s], ph, sh.status))) { ok = false; break; }
        uint8_t *sA = smem + s * stage_bytes, *sB = sA + O_BOX;
        if (g.sep_a) split_box(sA);
#pragma unroll
        for (uint32_t q = 0; q < 2u; ++q)
          if (q < g.nparts) split_box(sB + q * O_BOX);
        report(s);
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && rank == 0) {
      uint32_t it = 0, tcount = 0;
      bool ok = true;
      for (int ti = off[seg]; ti < off[seg + 1] && ok; ++ti) {
        const int4 t = tiles[ti];
        if (skip(t.x)) continue;
        const DevLayer &L = sh.layers[t.x];
        uint32_t N;
        int64_t K;
        orth_dims<KIND>(L, t.y, N, K);
        const int kch = (int)((K + 31) / 32);
        const uint32_t nparts = (N + 255) / 256;
        if constexpr (KIND == ORTH_TRSM) {
          for (uint32_t q = 0; q < nparts && ok; ++q) {
            const uint32_t slot = tcount & 1u;  // tcount counts sub-tiles here
            if (!ab.wait(&acc_empty[slot], ((tcount >> 1) & 1u) ^ 1u, sh.status)) { ok = false; break; }
            tc_fence_after();
            const int kq = min(kch, (int)(8u * (q + 1u)));
            const uint32_t idesc = idesc_tf32(256, 2u * half_rows(N, q), false, false);
            for (int kc = 0; kc < kq; ++kc, ++it) {
              const uint32_t s = it % nstages, ph = (it / nstages) & 1u;
              if (!ab.wait(X3 ? &conv[s] : &full[s], ph, sh.status)) { ok = false; break; }
              tc_fence_after();
              const uint32_t aB = smem_u32(smem + s * stage_bytes), bB = aB + O_BOX;
#pragma unroll
              for (int k8 = 0; k8 < 4; ++k8) {
                const uint64_t ad = smem_desc_sw128(aB + k8 * 32, 0, 1024), bd = smem_desc_sw128(bB + k8 * 32, 0, 1024);
                umma_pair_tf32(tmem + slot * 256u, ad, bd, idesc, (kc | k8) ? 1u : 0u);
                if (X3) {  // hi.lo + lo.hi
                  umma_pair_tf32(tmem + slot * 256u, ad, smem_desc_sw128(bB + lo_off + k8 * 32, 0, 1024), idesc, 1u);
                  umma_pair_tf32(tmem + slot * 256u, smem_desc_sw128(aB + lo_off + k8 * 32, 0, 1024), bd, idesc, 1u);
                }
              }
              umma_pair_commit_mc(&empty[s], 0x3);  // the stage is free in both CTAs
            }
            if (!ok) break;
            umma_pair_commit_mc(&acc_full[slot], 0x3);
            ++tcount;
          }
          continue;
        }
        const GramTile g = gram_tile(L.r, t.y);
        if (!ab.wait(acc_empty, (tcount & 1u) ^ 1u, sh.status)) break;
        tc_fence_after();
        for (int kc = 0; kc < kch; ++kc, ++it) {
          const uint32_t s = it % nstages, ph = (it / nstages) & 1u;
          if (!ab.wait(X3 ? &conv[s] : &full[s], ph, sh.status)) { ok = false; break; }
          tc_fence_after();
          const uint32_t aB = smem_u32(smem + s * stage_bytes), bB = aB + O_BOX;
#pragma unroll
          for (int k8 = 0; k8 < 4; ++k8) {
#pragma unroll
            for (uint32_t q = 0; q < 2u; ++q) {
              if (q >= g.nparts) break;
              const uint32_t aSrc = g.a_box[q] >= 0 ? bB + (uint32_t)g.a_box[q] * O_BOX : aB;
              const uint64_t ad = smem_desc_sw128(aSrc + k8 * 32, 0, 1024);
              const uint32_t idesc = idesc_tf32(256, g.N[q], false, false);
              const uint64_t bd = smem_desc_sw128(bB + q * O_BOX + k8 * 32, 0, 1024);
              // the first chunk that feeds a part starts its accumulation
              umma_pair_tf32(tmem + q * 256u, ad, bd, idesc, (kc | k8) ? 1u : 0u);
              if (X3) {  // hi.lo + lo.hi
                umma_pair_tf32(tmem + q * 256u, ad, smem_desc_sw128(bB + lo_off + q * O_BOX + k8 * 32, 0, 1024), idesc, 1u);
                umma_pair_tf32(tmem + q * 256u, smem_desc_sw128(aSrc + lo_off + k8 * 32, 0, 1024), bd, idesc, 1u);
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
    // epilogue: 128 threads, thread = output row (TMEM lane)
    const bool leader = (warp == 2 && lane == 0);
    const uint32_t lg = (uint32_t)(warp & 3), row = 32u * lg + lane;
    uint32_t tcount = 0, ecount = 0;
    for (int ti = off[seg]; ti < off[seg + 1]; ++ti) {
      const int4 t = tiles[ti];
      if (skip(t.x)) continue;
      const DevLayer &L = sh.layers[t.x];
      const OrthMaps om = orth_maps<KIND>(maps[t.x], pass);
      uint32_t N;
      int64_t K;
      orth_dims<KIND>(L, t.y, N, K);
      const int tr = 2 * t.y + (int)rank;
      const bool real = (int64_t)tr * 128 < L.m;  // TRSM: not the pair's empty second tile
      const GramTile g = gram_tile(L.r, KIND == ORTH_GRAM ? t.y : 0);
      const int nch = (KIND == ORTH_GRAM) ? g.nch : real ? (int)((min((int64_t)N, L.r) + 31) / 32) : 0;
      // The solve that ends Orthogonalize writes only the bf16 copy of P that R = B^T P and the
      // update read: pass 1 unless a shifted retry asked for pass 2, and pass 2 itself.
      const bool final_pass = (KIND == ORTH_TRSM) && (pass == 2 || (pass == 1 && !sh.orth_shifted[t.x]));
      // the Gram drains its accumulator in one go; the TRSM one sub-tile (256-column part) at a
      // time, from alternating slots (tcount counts sub-tiles there)
      const uint32_t nsub = (KIND == ORTH_TRSM) ? (N + 255) / 256 : 1u;
      bool stop = false;
      for (uint32_t q = 0; q < nsub; ++q) {
        const uint32_t slot = (KIND == ORTH_TRSM) ? (tcount & 1u) : 0u;
        const uint32_t aph = (KIND == ORTH_TRSM) ? ((tcount >> 1) & 1u) : (tcount & 1u);
        if (!named_and(1, 128, ab.wait(&acc_full[slot], aph, sh.status))) { stop = true; break; }
        tc_fence_after();
        // output chunks jb .. je - 1 (32 columns each); chunk j sits at TMEM column
        // slot * 256 + 32 (j - jb)
        const int jb = (KIND == ORTH_TRSM) ? (int)(8u * q) : 0;
        const int je = (KIND == ORTH_TRSM) ? min(nch, jb + 8) : nch;
        const uint32_t tcol = tmem + slot * 256u + (lg * 32u << 16);
        if (final_pass) {
          for (int j = jb; j < je; j += 2) {  // two 32-column chunks per 64-column bf16 box
            const uint32_t eb = ecount & 1u;
            uint8_t *hb = stg + eb * 2 * O_BOX, *lb = hb + O_BOX;  // lb: BF16X3's low halves
            if (leader) bulk_wait_read<1>();
            named_sync(1, 128);
#pragma unroll 1
            for (int h = 0; h < 2; ++h) {
              if (j + h < je) {
                uint32_t v[32];
                tmem_ld32(tcol + (uint32_t)(j + h - jb) * 32u, v);
                tmem_ld_wait();
#pragma unroll
                for (int c4 = 0; c4 < 8; ++c4) {
                  const __nv_bfloat162 a =
                      __floats2bfloat162_rn(__uint_as_float(v[4 * c4]), __uint_as_float(v[4 * c4 + 1]));
                  const __nv_bfloat162 b =
                      __floats2bfloat162_rn(__uint_as_float(v[4 * c4 + 2]), __uint_as_float(v[4 * c4 + 3]));
                  uint2 hv;
                  hv.x = *reinterpret_cast<const uint32_t *>(&a);
                  hv.y = *reinterpret_cast<const uint32_t *>(&b);
                  const uint32_t bo = sw128_offset(row, (uint32_t)(h * 4 + (c4 >> 1))) + (c4 & 1) * 8;
                  *reinterpret_cast<uint2 *>(hb + bo) = hv;
                  if (X3) {  // low halves: x - bf16(x), rounded to bf16
                    const float2 af = __bfloat1622float2(a), bf = __bfloat1622float2(b);
                    const __nv_bfloat162 al = __floats2bfloat162_rn(__uint_as_float(v[4 * c4]) - af.x,
                                                                    __uint_as_float(v[4 * c4 + 1]) - af.y);
                    const __nv_bfloat162 bl = __floats2bfloat162_rn(__uint_as_float(v[4 * c4 + 2]) - bf.x,
                                                                    __uint_as_float(v[4 * c4 + 3]) - bf.y);
                    uint2 lv;
                    lv.x = *reinterpret_cast<const uint32_t *>(&al);
                    lv.y = *reinterpret_cast<const uint32_t *>(&bl);
                    *reinterpret_cast<uint2 *>(lb + bo) = lv;
                  }
                }
              } else {  // a lone last chunk: the other half of the box (clipped by the store)
#pragma unroll
                for (int c4 = 4; c4 < 8; ++c4) {
                  *reinterpret_cast<uint4 *>(hb + sw128_offset(row, c4)) = make_uint4(0, 0, 0, 0);
                  if (X3) *reinterpret_cast<uint4 *>(lb + sw128_offset(row, c4)) = make_uint4(0, 0, 0, 0);
                }
              }
            }
            fence_async_smem();
            named_sync(1, 128);
            if (leader) {
              tma_store_2d(&maps[t.x].P_hi, hb, j * 32, tr * 128);
              if (X3) tma_store_2d(&maps[t.x].P_lo, lb, j * 32, tr * 128);
              bulk_commit();
            }
            ++ecount;
          }
        } else {
          for (int j = jb; j < je; ++j) {
            // the Gram's chunk j belongs to part j / 8, rows of S from tile o_row + rank; the
            // rows of a CTA past r are not stored (the same for every epilogue thread)
            const int otr = (KIND == ORTH_GRAM) ? (j >= 8 ? g.o_row[1] : g.o_row[0]) + (int)rank : tr;
            if (KIND == ORTH_GRAM && (int64_t)otr * 128 >= L.r) continue;
            const bool store_t = (KIND == ORTH_TRSM);  // transposed copy: the next Gram's operand
            const uint32_t eb = ecount & 1u;
            uint8_t *box = stg + eb * 2 * O_BOX, *tbox = box + O_BOX + lg * O_TBOX;
            if (leader) bulk_wait_read<1>();
            named_sync(1, 128);
            uint32_t v[32];
            tmem_ld32(tcol + (uint32_t)(j - jb) * 32u, v);
            tmem_ld_wait();
#pragma unroll
            for (int c4 = 0; c4 < 8; ++c4)
              *reinterpret_cast<float4 *>(box + sw128_f32(row, c4)) =
                  make_float4(__uint_as_float(v[4 * c4]), __uint_as_float(v[4 * c4 + 1]),
                              __uint_as_float(v[4 * c4 + 2]), __uint_as_float(v[4 * c4 + 3]));
            if (store_t) {
              // transposed 32 x 32 box of this warp's rows: box row c = output column j*32 + c
#pragma unroll
              for (int c = 0; c < 32; ++c)
                *reinterpret_cast<float *>(tbox + c * 128 + ((((uint32_t)lane >> 2) ^ (c & 7)) << 4) + (lane & 3) * 4) =
                    __uint_as_float(v[c]);
            }
            fence_async_smem();
            named_sync(1, 128);
            if (leader) {
              tma_store_2d(om.out, box, j * 32, otr * 128);
              if (store_t)
                for (int w4 = 0; w4 < 4; ++w4)
                  if ((int64_t)tr * 128 + w4 * 32 < L.m)
                    tma_store_2d(om.out_t, stg + eb * 2 * O_BOX + O_BOX + w4 * O_TBOX, tr * 128 + w4 * 32, j * 32);
              bulk_commit();
            }
            ++ecount;
          }
        }
        tc_fence_before();
        named_sync(1, 128);  // every thread's TMEM reads of this accumulator slot are done
        if (leader) mbar_arrive_cluster(cluster_addr(&acc_empty[slot], 0));
        ++tcount;
      }
      if (stop) break;
    }
    if (leader) bulk_wait<0>();
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();  // both CTAs are done with the pair's TMEM and barriers
  tc_fence_after();
  if (warp == 1) tmem_dealloc_pair(tmem, tmem_cols);
}

// alignment slack + operand stages + 2 staging buffers + barriers (2 x stages + 5 words)
uint32_t orth_smem(int nstages, uint32_t stage_bytes) { return 1024u + nstages * stage_bytes + 4u * O_BOX + 512u; }

cudaError_t setup_orth_kernels(uint32_t smem, bool x3) {
  const int sm = (int)smem;
  const cudaFuncAttribute at = cudaFuncAttributeMaxDynamicSharedMemorySize;
  cudaError_t e = x3 ? cudaFuncSetAttribute(tc_orth_kernel<ORTH_GRAM, true>, at, sm)
                     : cudaFuncSetAttribute(tc_orth_kernel<ORTH_GRAM, false>, at, sm);
  if (e == cudaSuccess)
    e = x3 ? cudaFuncSetAttribute(tc_orth_kernel<ORTH_TRSM, true>, at, sm)
           : cudaFuncSetAttribute(tc_orth_kernel<ORTH_TRSM, false>, at, sm);
  return e;
}

void launch_orth(const Shared &sh, const TcPlan &tp, bool gram, int pass, cudaStream_t s) {
  const DevSchedule &d = gram ? tp.d_gram : tp.d_trsm;
  if (d.grid <= 0) return;
  const bool x3 = tp.precision == DION_PREC_BF16X3;
  const uint32_t f = x3 ? 2u : 1u;  // BF16X3 stages hold the lo boxes too
  const uint32_t stage = f * O_BOX * (1 + tp.o_parts), tstage = f * 2u * O_BOX;  // TRSM: A box + one B box
  const int g = 2 * d.grid;
  if (gram && x3)
    tc_orth_kernel<ORTH_GRAM, true><<<g, O_THREADS_X3, tp.o_smem, s>>>(sh, d.tiles, d.off, tp.maps, pass,
                                                                        tp.o_stages, stage, tp.tmem_cols);
  else if (gram)
    tc_orth_kernel<ORTH_GRAM, false><<<g, O_THREADS, tp.o_smem, s>>>(sh, d.tiles, d.off, tp.maps, pass,
                                                                      tp.o_stages, stage, tp.tmem_cols);
  else if (x3)  // two 256-column accumulator slots
    tc_orth_kernel<ORTH_TRSM, true><<<g, O_THREADS_X3, tp.o_smem, s>>>(sh, d.tiles, d.off, tp.maps, pass,
                                                                        tp.t_stages, tstage, 512u);
  else
    tc_orth_kernel<ORTH_TRSM, false><<<g, O_THREADS, tp.o_smem, s>>>(sh, d.tiles, d.off, tp.maps, pass,
                                                                      tp.t_stages, tstage, 512u);
}

}  // namespace tc
}  // namespace cd
