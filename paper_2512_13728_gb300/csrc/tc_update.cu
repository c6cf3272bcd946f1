// Error feedback + parameter update (Algorithm 1/2, sync branch):
//   M = B - (1 - mu) P R^T,   X = X - eta sqrt(m/n) P Q_t^T
// run as one persistent, warp-specialized kernel over 128 x 128 output tiles:
//   warp 0      TMA producer: bf16 K-major chunks of P (A), R and Q_t (two B operands) into a
//               3-stage shared-memory ring (BF16X3: also their low halves);
//   warp 1      MMA issuer: two 128x128x16 tcgen05.mma per k-step into a double-buffered
//               pair of TMEM accumulators (U1 = P R^T, U2 = P Q_t^T; 4 x 128 = 512 columns);
//   warps 2..5  epilogue (both CTAs): TMA-load 128 x 16 fp32 boxes of B (in the M buffer) and X,
//               read U1/U2 from TMEM (thread = tile row), compute M_t and X_t in shared
//               memory, TMA-store both; per-tile fp64 partial of ||M_t||^2 for Equation 1.
#include "tc.cuh"
#include "tc_common.cuh"
#include "tc_kernels.cuh"

#include <algorithm>

namespace cd {
namespace tc {

// ============================================================ update (tcgen05) kernel ===
// CTAs 2 s and 2 s + 1 take row tiles 2 p and 2 p + 1 of the same column blocks in the same
// order (schedule segment s), so the R and Q_t chunks one of them loads are usually still in L2
// when the other asks for them.  Each CTA loads all three operand boxes of a stage itself.
constexpr uint32_t U_OPB = 128u * 64u * 2u;           // 128 x 64 bf16 operand box (BF16: one per operand)
constexpr uint32_t U_OPB32 = 128u * 32u * 2u;         // 128 x 32 bf16 operand box (BF16X3)
constexpr uint32_t U_EBOX = 128u * 16u * 4u;          // one 128 x 16 fp32 box (64-byte swizzle)
constexpr uint32_t U_GBOX = 128u * 16u * 2u;          // one 128 x 16 bf16 box of G (32-byte swizzle)
constexpr uint32_t U_EBUF2 = 2u * U_EBOX + U_GBOX;     // M, X and G of one 16-column sub-chunk (20 KB)
static_assert(U_EBUF2 % 1024u == 0, "every box of a sub-chunk buffer stays 1024-byte aligned");
constexpr int U_THREADS = 192;
constexpr uint32_t U_IDESC = idesc_bf16(128, 128, false, false);
// Ring depths.  BF16: 3 stages of {P, R, Q_t} in 64-wide K chunks (128-byte swizzle) and 4
// epilogue sub-chunk buffers of M, X and G.  BF16X3: each stage also holds the low halves of P,
// R and Q_t (P R^T = Ph Rh^T + Ph Rl^T + Pl Rh^T, the same for P Q_t^T), and B is already in M
// (no G box); its stages take 32-wide K chunks (64-byte swizzle), so 3 stages of 6 boxes leave
// room for 5 epilogue buffers of M and X (loads 4 sub-chunks ahead: with 2 buffers, one load in
// flight, the epilogue waited on every sub-chunk).
template <bool X3>
struct UpdCfg {
  static constexpr uint32_t KW = X3 ? 32u : 64u;  // K chunk width (bf16 elements per operand row)
  static constexpr uint32_t OPB = X3 ? U_OPB32 : U_OPB;
  static constexpr int STAGES = 3;
  static constexpr uint32_t STAGE = (X3 ? 6u : 3u) * OPB;  // P, R, Q_t [, P_lo, R_lo, Q_lo]
  static constexpr int EBUF = X3 ? 5 : 4;
  static constexpr uint32_t EBUF2 = X3 ? 2u * U_EBOX : U_EBUF2;  // bytes of one sub-chunk buffer
  static constexpr uint32_t SMEM = 1024u + STAGES * STAGE + EBUF * EBUF2 + 256u;
};
static_assert(UpdCfg<true>::SMEM <= 227u * 1024u && UpdCfg<false>::SMEM <= 227u * 1024u, "update smem");

// Tile = {layer, row-tile pair p, column tile, ||M_t|| slot of row tile 2 p}.
template <bool X3>
__global__ void __launch_bounds__(U_THREADS, 1)
    tc_update_kernel(Shared sh, const int4 *__restrict__ tiles, const int *__restrict__ off, const LayerMaps *__restrict__ maps,
                     float mu, float eta, float keep) {
  constexpr int U_STAGES = UpdCfg<X3>::STAGES;
  constexpr uint32_t U_STAGE = UpdCfg<X3>::STAGE;
  constexpr uint32_t KW = UpdCfg<X3>::KW, OPB = UpdCfg<X3>::OPB;
  constexpr int U_EBUF = UpdCfg<X3>::EBUF;
  constexpr uint32_t U_EBUFB = UpdCfg<X3>::EBUF2;
  if (sh.gate_scratch[kScratchActive] == 0ull) return;  // no layer takes the Dion branch
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = align1024(smem_raw);
  uint8_t *stage = smem;
  uint8_t *epi = smem + U_STAGES * U_STAGE;
  uint64_t *bars = reinterpret_cast<uint64_t *>(epi + U_EBUF * U_EBUFB);
  uint64_t *full = bars, *empty = bars + U_STAGES;
  uint64_t *acc_full = bars + 2 * U_STAGES, *acc_empty = acc_full + 2, *epi_full = acc_empty + 2;
  uint64_t *drain = epi_full + U_EBUF;
  __shared__ uint32_t tmem_base_s;
  __shared__ int abort_s;
  __shared__ double red_s[4];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // hand-off waits between the roles use the plan's limit; the drains below keep the default
  const Abort ab{&abort_s, sh.handoff_limit_ns};
  const uint32_t rank = blockIdx.x & 1u;  // row tile 2 p + rank of the segment's tiles
  const int seg = blockIdx.x >> 1;

  if (threadIdx.x == 0) {
    for (int i = 0; i < U_STAGES; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], 1);  // this CTA's MMA commit
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], 1);  // the epilogue leader, after its warps have read TMEM
    }
    for (int b = 0; b < U_EBUF; ++b) mbar_init(&epi_full[b], 1);
    mbar_init(drain, 1);
    abort_s = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(&tmem_base_s, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base_s;

  if (warp == 0) {
    // ---------------------------------------------------------------- TMA producer
    if (lane == 0) {
      uint32_t it = 0;
      bool ok = true;
      for (int ti = off[seg]; ti < off[seg + 1] && ok; ++ti) {
        const int4 t = tiles[ti];
        if (!sh.active[t.x]) continue;
        const LayerMaps *mp = maps + t.x;
        const int kch = (int)((sh.layers[t.x].r + KW - 1) / KW);
        const int mb = 2 * t.y + (int)rank;  // past the last row tile: zero-filled, not stored
        for (int kc = 0; kc < kch; ++kc, ++it) {
          const uint32_t s = it % U_STAGES, ph = (it / U_STAGES) & 1u;
          if (!ab.wait(&empty[s], ph ^ 1u, sh.status)) { ok = false; break; }
          uint8_t *sp = stage + s * U_STAGE;
          mbar_expect_tx(&full[s], U_STAGE);
          const int k0 = kc * (int)KW;
          if (X3) {
            tma_load_2d(sp, &mp->P_hi32, &full[s], k0, mb * 128);
            tma_load_2d(sp + OPB, &mp->R_hi32, &full[s], k0, t.z * 128);
            tma_load_2d(sp + 2 * OPB, &mp->Qn_hi32, &full[s], k0, t.z * 128);
            tma_load_2d(sp + 3 * OPB, &mp->P_lo32, &full[s], k0, mb * 128);
            tma_load_2d(sp + 4 * OPB, &mp->R_lo32, &full[s], k0, t.z * 128);
            tma_load_2d(sp + 5 * OPB, &mp->Qn_lo32, &full[s], k0, t.z * 128);
          } else {
            tma_load_2d(sp, &mp->P_hi, &full[s], k0, mb * 128);
            tma_load_2d(sp + OPB, &mp->R_hi, &full[s], k0, t.z * 128);
            tma_load_2d(sp + 2 * OPB, &mp->Qn_hi, &full[s], k0, t.z * 128);
          }
        }
      }
      // drain: every load this CTA issued has landed
      for (uint32_t k = (it > U_STAGES ? it - U_STAGES : 0); k < it; ++k)
        mbar_wait(&full[k % U_STAGES], (k / U_STAGES) & 1u, sh.status);
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      uint32_t it = 0, tcount = 0;
      bool ok = true;
      for (int ti = off[seg]; ti < off[seg + 1] && ok; ++ti) {
        const int4 t = tiles[ti];
        if (!sh.active[t.x]) continue;
        const int kch = (int)((sh.layers[t.x].r + KW - 1) / KW);
        const uint32_t b = tcount & 1u, aph = (tcount >> 1) & 1u;
        if (!ab.wait(&acc_empty[b], aph ^ 1u, sh.status)) break;
        tc_fence_after();
        const uint32_t d1 = tmem + b * 256u, d2 = d1 + 128u;
        for (int kc = 0; kc < kch; ++kc, ++it) {
          const uint32_t s = it % U_STAGES, ph = (it / U_STAGES) & 1u;
          if (!ab.wait(&full[s], ph, sh.status)) { ok = false; break; }
          tc_fence_after();
          const uint32_t base = smem_u32(stage + s * U_STAGE);
          // K-major operand box o of the stage, advanced by k16 steps of 16 elements (32 bytes)
          auto desc = [&](uint32_t o, int k16) {
            const uint32_t a = base + o * OPB + (uint32_t)k16 * 32u;
            return X3 ? smem_desc_sw64(a, 512) : smem_desc_sw128(a, 0, 1024);
          };
#pragma unroll
          for (int k16 = 0; k16 < (int)(KW / 16u); ++k16) {
            const uint64_t ad = desc(0, k16), rd = desc(1, k16), qd = desc(2, k16);
            const uint32_t acc = (kc | k16) ? 1u : 0u;
            umma_bf16(d1, ad, rd, U_IDESC, acc);
            umma_bf16(d2, ad, qd, U_IDESC, acc);
            if (X3) {  // P R^T = Ph Rh^T + Ph Rl^T + Pl Rh^T, P Q_t^T likewise
              const uint64_t adl = desc(3, k16);
              umma_bf16(d1, ad, desc(4, k16), U_IDESC, 1u);
              umma_bf16(d1, adl, rd, U_IDESC, 1u);
              umma_bf16(d2, ad, desc(5, k16), U_IDESC, 1u);
              umma_bf16(d2, adl, qd, U_IDESC, 1u);
            }
          }
          umma_commit(&empty[s]);  // the stage is free once its MMAs have read it
        }
        if (!ok) break;
        umma_commit(&acc_full[b]);
        ++tcount;
      }
      umma_commit(drain);  // every MMA of this CTA has completed before TMEM is freed
      mbar_wait(drain, 0, sh.status);
    }
  } else {
    // ---------------------------------------------------------------- epilogue (128 threads)
    // B and X stream in 16-column sub-chunks through U_EBUF buffers.  The leader keeps the
    // loads U_EBUF - 1 sub-chunks ahead of the one being written back, across tile boundaries
    // (they do not depend on the MMAs), so HBM latency is covered without taking shared memory
    // from the operand ring.
    const int et = threadIdx.x - 64;
    const uint32_t row = 32u * (warp & 3) + lane;  // TMEM lane = tile row
    const bool leader = (et == 0);
    const int tend = off[seg + 1];
    // 16-column sub-chunks of a tile that start inside the matrix; 0 for the pair's second tile
    // when it lies past the last row tile
    auto subs_of = [&](const int4 &t) -> int {
      const DevLayer &L = sh.layers[t.x];
      if ((int64_t)(2 * t.y + (int)rank) * 128 >= L.m) return 0;
      return (int)std::min<int64_t>(8, (L.n - (int64_t)t.z * 128 + 15) / 16);
    };
    int lt = off[seg], lj = 0;  // load cursor: tile, sub-chunk
    auto skip_empty = [&]() {
      while (lt < tend && (!sh.active[tiles[lt].x] || subs_of(tiles[lt]) == 0)) ++lt;
    };
    skip_empty();
    uint32_t ecount = 0, issued = 0;
    auto issue_upto = [&](uint32_t target) {  // leader: loads of sub-chunks [issued, target)
      while (issued < target && lt < tend) {
        const int4 t = tiles[lt];
        const LayerMaps *mp = maps + t.x;
        const uint32_t eb = issued % U_EBUF;
        // the buffer's previous sub-chunk (issued - U_EBUF) was stored at least one sub-chunk
        // ago: at most the latest store group may still be reading shared memory
        if (issued >= U_EBUF) bulk_wait_read<1>();
        uint8_t *bs = epi + eb * U_EBUFB;
        const int r0 = (2 * t.y + (int)rank) * 128, x0 = t.z * 128 + lj * 16;
        const bool defer = sh.layers[t.x].b_deferred != 0 && !sh.b_in_m;  // B = M + G is formed here
        mbar_expect_tx(&epi_full[eb], 2u * U_EBOX + (defer ? U_GBOX : 0u));
        tma_load_2d(bs, &mp->Mf16, &epi_full[eb], x0, r0);
        tma_load_2d(bs + U_EBOX, &mp->Xf16, &epi_full[eb], x0, r0);
        if (defer) tma_load_2d(bs + 2 * U_EBOX, &mp->Gh16, &epi_full[eb], x0, r0);
        ++issued;
        if (++lj == subs_of(t)) {
          lj = 0;
          ++lt;
          skip_empty();
        }
      }
    };
    if (leader) issue_upto(U_EBUF - 1);
    uint32_t tcount = 0;
    uint32_t waited = 0;  // sub-chunks whose load this role has waited for, in order
    bool ok = true;
    for (int ti = off[seg]; ti < tend && ok; ++ti) {
      const int4 t = tiles[ti];
      if (!sh.active[t.x]) continue;
      const DevLayer &L = sh.layers[t.x];
      const LayerMaps *mp = maps + t.x;
      const float dec = 1.f - mu, c = eta * L.sqrt_m_over_n;
      const int mb = 2 * t.y + (int)rank, r0 = mb * 128, c0 = t.z * 128;
      const int ntc = (int)((L.n + 127) / 128);
      const int ns = subs_of(t);
      const bool defer = L.b_deferred != 0 && !sh.b_in_m;
      const uint32_t b = tcount & 1u, aph = (tcount >> 1) & 1u;
      if (!named_and(1, 128, ab.wait(&acc_full[b], aph, sh.status))) break;
      tc_fence_after();
      float ss = 0.f;
      for (int j = 0; j < (ns + 1) / 2 && ok; ++j) {  // 32-column TMEM chunk j = sub-chunks 2j, 2j + 1
        uint32_t u1[32], u2[32];
        tmem_ld32(tmem + ((32u * (warp & 3)) << 16) + b * 256u + j * 32, u1);
        tmem_ld32(tmem + ((32u * (warp & 3)) << 16) + b * 256u + 128u + j * 32, u2);
        tmem_ld_wait();
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const int sub = 2 * j + h;
          if (sub >= ns) break;
          const uint32_t k = ecount + sub, eb = k % U_EBUF, eph = (k / U_EBUF) & 1u;
          if (!named_and(1, 128, ab.wait(&epi_full[eb], eph, sh.status))) {
            ok = false;
            break;
          }
          waited = k + 1;
          uint8_t *bs = epi + eb * U_EBUFB;
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const uint32_t o = sw64_f32(row, q);
            const int cc = h * 16 + q * 4;
            float4 bv = *reinterpret_cast<float4 *>(bs + o);
            float4 xv = *reinterpret_cast<float4 *>(bs + U_EBOX + o);
            if (defer) {  // B = M_{t-1} + G, the same fp32 additions as the buffer pass
              const uint2 gv = *reinterpret_cast<const uint2 *>(bs + 2 * U_EBOX + sw32_offset(row, (uint32_t)q >> 1) +
                                                                (q & 1) * 8);
              bv.x += __uint_as_float(gv.x << 16);
              bv.y += __uint_as_float(gv.x & 0xffff0000u);
              bv.z += __uint_as_float(gv.y << 16);
              bv.w += __uint_as_float(gv.y & 0xffff0000u);
            }
            bv.x = fmaf(-dec, __uint_as_float(u1[cc + 0]), bv.x);
            bv.y = fmaf(-dec, __uint_as_float(u1[cc + 1]), bv.y);
            bv.z = fmaf(-dec, __uint_as_float(u1[cc + 2]), bv.z);
            bv.w = fmaf(-dec, __uint_as_float(u1[cc + 3]), bv.w);
            xv.x = fmaf(-c, __uint_as_float(u2[cc + 0]), xv.x * keep);  // keep: decoupled weight decay
            xv.y = fmaf(-c, __uint_as_float(u2[cc + 1]), xv.y * keep);
            xv.z = fmaf(-c, __uint_as_float(u2[cc + 2]), xv.z * keep);
            xv.w = fmaf(-c, __uint_as_float(u2[cc + 3]), xv.w * keep);
            ss = fmaf(bv.x, bv.x, ss); ss = fmaf(bv.y, bv.y, ss);
            ss = fmaf(bv.z, bv.z, ss); ss = fmaf(bv.w, bv.w, ss);
            *reinterpret_cast<float4 *>(bs + o) = bv;
            *reinterpret_cast<float4 *>(bs + U_EBOX + o) = xv;
          }
          fence_async_smem();
          named_sync(1, 128);
          if (leader) {  // out-of-range rows/columns of a ragged tile are clipped by the store
            tma_store_2d(&mp->Mf16, bs, c0 + sub * 16, r0);
            tma_store_2d(&mp->Xf16, bs + U_EBOX, c0 + sub * 16, r0);
            bulk_commit();
            issue_upto(k + U_EBUF);  // sub-chunk k + U_EBUF - 1 reuses the buffer of k - 1
          }
        }
      }
      if (!ok) break;
      ecount += ns;
      // per-tile ||M_t||^2 (rows/columns outside the matrix hold 0), fixed reduction order;
      // the barrier also ends every thread's TMEM reads of this accumulator
      double v = (double)ss;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
      if (lane == 0) red_s[warp - 2] = v;
      tc_fence_before();
      named_sync(1, 128);
      if (leader) {
        mbar_arrive(&acc_empty[b]);  // every thread has read accumulator buffer b
        if (ns > 0) sh.upart[t.w + (int)rank * ntc] = (red_s[0] + red_s[1]) + (red_s[2] + red_s[3]);
      }
      ++tcount;
    }
    if (leader) {
      bulk_wait<0>();
      // loads issued but not waited for (only after an abort): at most U_EBUF - 1 of them, in
      // distinct buffers, so each wait is for the latest phase of its buffer
      for (uint32_t k = waited; k < issued; ++k) mbar_wait(&epi_full[k % U_EBUF], (k / U_EBUF) & 1u, sh.status);
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, 512);
}

// ========================================================================= launch ===
cudaError_t setup_update_kernel(bool x3) {
  return x3 ? cudaFuncSetAttribute(tc_update_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                   (int)UpdCfg<true>::SMEM)
            : cudaFuncSetAttribute(tc_update_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                   (int)UpdCfg<false>::SMEM);
}

void launch_update(const Shared &sh, const TcPlan &tp, float mu, float eta, float keep, cudaStream_t s) {
  if (tp.d_update.grid <= 0) return;
  if (tp.precision == DION_PREC_BF16X3)
    tc_update_kernel<true><<<2 * tp.d_update.grid, U_THREADS, UpdCfg<true>::SMEM, s>>>(
        sh, tp.d_update.tiles, tp.d_update.off, tp.maps, mu, eta, keep);
  else
    tc_update_kernel<false><<<2 * tp.d_update.grid, U_THREADS, UpdCfg<false>::SMEM, s>>>(
        sh, tp.d_update.tiles, tp.d_update.off, tp.maps, mu, eta, keep);
}

}  // namespace tc
}  // namespace cd
