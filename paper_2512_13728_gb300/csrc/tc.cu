// Tensor-core path of the CurvaDion step (DION_PREC_BF16, DION_PREC_BF16X3): plan layout, tensor
// maps and the step's launch sequence.  The kernels are in tc_update.cu (error feedback +
// parameter update), tc_bq.cu, tc_orth.cu and chol_tc.cu.
#include "tc.cuh"
#include "tc_common.cuh"
#include "tc_kernels.cuh"

#include <algorithm>
#include <cstring>

namespace cd {

void tick_begin(dion_plan *p, cudaStream_t s);
void tick(dion_plan *p, cudaStream_t s, const char *name);

namespace tc {

// ========================================================================= host side ===
namespace {

// Longest-processing-time-first assignment of tiles to at most `max_grid` persistent CTAs.
Schedule lpt(const std::vector<int4> &tiles, const std::vector<double> &cost, int max_grid) {
  Schedule sc;
  const int n = (int)tiles.size();
  sc.grid = std::max(0, std::min(n, max_grid));
  if (n == 0) {
    sc.off.assign(1, 0);
    return sc;
  }
  std::vector<int> order(n);
  for (int i = 0; i < n; ++i) order[i] = i;
  std::stable_sort(order.begin(), order.end(), [&](int a, int b) { return cost[a] > cost[b]; });
  std::vector<double> load(sc.grid, 0.0);
  std::vector<std::vector<int>> per(sc.grid);
  for (int i : order) {
    int best = 0;
    for (int c = 1; c < sc.grid; ++c)
      if (load[c] < load[best]) best = c;
    load[best] += cost[i];
    per[best].push_back(i);
  }
  sc.off.push_back(0);
  for (int c = 0; c < sc.grid; ++c) {
    for (int i : per[c]) sc.tiles.push_back(tiles[i]);
    sc.off.push_back((int)sc.tiles.size());
  }
  return sc;
}
}  // namespace

dion_status layout(const dion_layer *layers, int32_t L, int32_t precision, int num_sms, size_t start,
                   TcLayout *out) {
  if (precision != DION_PREC_BF16 && precision != DION_PREC_BF16X3) return DION_ERR_UNSUPPORTED;
  const bool x3 = precision == DION_PREC_BF16X3;
  // BF16X3 stages hold the low halves too: its operand rings fit shared memory up to r = 256
  for (int32_t l = 0; x3 && l < L; ++l)
    if (layers[l].r > 256) return DION_ERR_UNSUPPORTED;
  TcLayout &lo = *out;
  lo.precision = precision;
  size_t off = start;
  auto take = [&](size_t bytes, size_t align = 256) {  // a region and its guard words
    off = (off + align - 1) / align * align;
    const size_t at = off;
    off += bytes;
    off = (off + 3) / 4 * 4;
    lo.guards.push_back(off);
    off += kGuardWords * sizeof(uint32_t);
    return at;
  };
  lo.o_phi.resize(L);
  lo.o_rhi.resize(L);
  lo.o_qnhi.resize(L);
  lo.o_bh.resize(L);
  lo.o_ptraw.resize(L);
  lo.o_pt.resize(L);
  lo.o_colsq.resize(L);
  lo.o_colinv.resize(L);
  lo.o_bl.assign(L, 0);
  lo.o_plo.assign(L, 0);
  lo.o_rlo.assign(L, 0);
  lo.o_qnlo.assign(L, 0);
  for (int32_t l = 0; l < L; ++l) {
    const dion_layer &ly = layers[l];
    const int64_t ldp = (ly.r + 7) / 8 * 8, ldbh = (ly.n + 7) / 8 * 8;
    lo.max_r = std::max<int32_t>(lo.max_r, (int32_t)ly.r);
    lo.o_phi[l] = take(ly.m * ldp * 2);
    lo.o_rhi[l] = take(ly.n * ldp * 2);
    lo.o_qnhi[l] = take(ly.n * ldp * 2);
    lo.o_bh[l] = take(ly.m * ldbh * 2);
    if (x3) {
      lo.o_bl[l] = take(ly.m * ldbh * 2);
      lo.o_plo[l] = take(ly.m * ldp * 2);
      lo.o_rlo[l] = take(ly.n * ldp * 2);
      lo.o_qnlo[l] = take(ly.n * ldp * 2);
    }
    const int64_t ldmt = (ly.m + 7) / 8 * 8;
    lo.o_ptraw[l] = take(ly.r * ldmt * 4);
    lo.o_pt[l] = take(ly.r * ldmt * 4);
    lo.o_colsq[l] = take((size_t)((ly.n + 127) / 128) * ldp * 8);
    lo.o_colinv[l] = take(ldp * 4);
    for (int64_t rb = 0; rb < (ly.r + 127) / 128; ++rb) lo.gram_tiles.push_back(make_int4(l, (int)rb, 0, 0));
    for (int64_t mb = 0; mb < (ly.m + 127) / 128; ++mb) lo.trsm_tiles.push_back(make_int4(l, (int)mb, 0, 0));
    for (int64_t mb = 0; mb < (ly.m + 127) / 128; ++mb)
      for (int64_t nb = 0; nb < (ly.n + 127) / 128; ++nb)
        lo.utiles.push_back(make_int4(l, (int)mb, (int)nb, (int)lo.utiles.size()));
    const int64_t qrow = std::max<int64_t>(1, std::min<int64_t>(ly.n, 16384 / ly.r));
    for (int64_t r0 = 0; r0 < ly.n; r0 += qrow)
      lo.qtiles.push_back(make_int4(l, (int)r0, (int)std::min(qrow, ly.n - r0), 0));
    for (int64_t mb = 0; mb < (ly.m + 127) / 128; ++mb) lo.ftiles.push_back(make_int4(l, (int)mb, 0, 0));
    for (int64_t nb = 0; nb < (ly.n + 127) / 128; ++nb) lo.rtiles.push_back(make_int4(l, (int)nb, 0, 0));
  }
  // per-tile cost ~ K-loop length (+ a constant for the epilogue), LPT over the SMs

  // update: row-tile pairs (one per two consecutive CTAs); w = ||M_t|| slot of the pair's first tile
  std::vector<int4> upairs;
  for (size_t i = 0; i < lo.utiles.size(); ++i) {
    const int4 &u = lo.utiles[i];
    if (u.y % 2 == 0) upairs.push_back(make_int4(u.x, u.y / 2, u.z, u.w));
  }
  lo.s_update = lpt(upairs, std::vector<double>(upairs.size(), 1.0), std::max(num_sms / 2, 1));
  // B Q and B^T P run in CTA pairs over two consecutive 128-row tiles: tile {layer, pair}
  auto pairs_of = [](const std::vector<int4> &tl) {
    std::vector<int4> pr;
    for (const int4 &t : tl)
      if (t.y % 2 == 0) pr.push_back(make_int4(t.x, t.y / 2, 0, 0));
    return pr;
  };
  auto pair_sched = [&](const std::vector<int4> &tl, auto costf) {
    std::vector<double> c(tl.size());
    for (size_t i = 0; i < tl.size(); ++i) c[i] = costf(tl[i]);
    return lpt(tl, c, std::max(num_sms / 2, 1));
  };
  lo.s_bq = pair_sched(pairs_of(lo.ftiles), [&](const int4 &t) { return (double)layers[t.x].n + 2.0 * layers[t.x].r; });
  lo.s_btp = pair_sched(pairs_of(lo.rtiles), [&](const int4 &t) { return (double)layers[t.x].m + 2.0 * layers[t.x].r; });
  // equal cost for every tile of a layer (at r > 256 both load two boxes per chunk), so that
  // they run side by side and stream the layer's X^T from DRAM about once
  lo.s_gram = pair_sched(pairs_of(lo.gram_tiles), [&](const int4 &t) { return (double)layers[t.x].m * layers[t.x].r; });
  lo.s_trsm = pair_sched(pairs_of(lo.trsm_tiles), [&](const int4 &t) { return 3.0 * layers[t.x].r + 64.0; });
  for (Schedule *sc : {&lo.s_update, &lo.s_bq, &lo.s_btp, &lo.s_gram, &lo.s_trsm}) {
    sc->o_tiles = take(sizeof(int4) * std::max<size_t>(sc->tiles.size(), 1));
    sc->o_off = take(sizeof(int) * sc->off.size());
  }
  lo.o_maps = take(sizeof(LayerMaps) * std::max(L, 1), 128);
  lo.o_utiles = take(sizeof(int4) * std::max<size_t>(lo.utiles.size(), 1));
  lo.o_ftiles = take(sizeof(int4) * std::max<size_t>(lo.ftiles.size(), 1));
  lo.o_rtiles = take(sizeof(int4) * std::max<size_t>(lo.rtiles.size(), 1));
  lo.o_qtiles = take(sizeof(int4) * std::max<size_t>(lo.qtiles.size(), 1));
  lo.o_gtiles = take(sizeof(int4) * std::max<size_t>(lo.gram_tiles.size(), 1));
  lo.o_ttiles = take(sizeof(int4) * std::max<size_t>(lo.trsm_tiles.size(), 1));
  lo.fuse_buffer = L > 0 && !x3;  // BF16X3 forms B and its two bf16 halves in the buffer pass
  for (int32_t l = 0; l < L; ++l) lo.fuse_buffer = lo.fuse_buffer && layers[l].g_dtype == DION_DTYPE_BF16;
  lo.end = off;
  (void)num_sms;
  return DION_OK;
}

void bind(const TcLayout &lo, char *base, DevLayer *dl, int32_t L, TcPlan *tp) {
  for (int32_t l = 0; l < L; ++l) {
    dl[l].P_hi = reinterpret_cast<__nv_bfloat16 *>(base + lo.o_phi[l]);
    dl[l].R_hi = reinterpret_cast<__nv_bfloat16 *>(base + lo.o_rhi[l]);
    dl[l].Qn_hi = reinterpret_cast<__nv_bfloat16 *>(base + lo.o_qnhi[l]);
    dl[l].Bh = reinterpret_cast<__nv_bfloat16 *>(base + lo.o_bh[l]);
    dl[l].ldbh = (dl[l].n + 7) / 8 * 8;
    dl[l].PT_raw = reinterpret_cast<float *>(base + lo.o_ptraw[l]);
    dl[l].PT = reinterpret_cast<float *>(base + lo.o_pt[l]);
    dl[l].ldmt = (dl[l].m + 7) / 8 * 8;
    dl[l].colsq = reinterpret_cast<double *>(base + lo.o_colsq[l]);
    dl[l].colinv = reinterpret_cast<float *>(base + lo.o_colinv[l]);
    dl[l].rtile_cnt = (int32_t)((dl[l].n + 127) / 128);
    // the update forms B = M + G itself (BF16 mode with bf16 G); BF16X3 writes B into M
    dl[l].b_deferred = (dl[l].g_dtype == DT_BF16 && lo.precision == DION_PREC_BF16) ? 1 : 0;
    if (lo.precision == DION_PREC_BF16X3) {
      dl[l].Bl = reinterpret_cast<__nv_bfloat16 *>(base + lo.o_bl[l]);
      dl[l].P_lo = reinterpret_cast<__nv_bfloat16 *>(base + lo.o_plo[l]);
      dl[l].R_lo = reinterpret_cast<__nv_bfloat16 *>(base + lo.o_rlo[l]);
      dl[l].Qn_lo = reinterpret_cast<__nv_bfloat16 *>(base + lo.o_qnlo[l]);
    }
    dl[l].upart_off = -1;
  }
  if (lo.fuse_buffer) {  // the fused kernel writes one ||B||^2 / ||M_{t-1}||^2 slot per 128-row tile
    int32_t slot = 0;
    for (int32_t l = 0; l < L; ++l) {
      dl[l].bpart_off = slot;
      dl[l].bpart_cnt = (int32_t)((dl[l].m + 127) / 128);
      slot += dl[l].bpart_cnt;
    }
  }
  tp->fuse_buffer = lo.fuse_buffer;
  int32_t cur = -1;
  for (size_t i = 0; i < lo.utiles.size(); ++i) {
    const int l = lo.utiles[i].x;
    if (l != cur) {
      dl[l].upart_off = (int32_t)i;
      dl[l].upart_cnt = 0;
      cur = l;
    }
    ++dl[l].upart_cnt;
  }
  tp->maps = reinterpret_cast<LayerMaps *>(base + lo.o_maps);
  tp->utiles = reinterpret_cast<int4 *>(base + lo.o_utiles);
  tp->n_utiles = (int32_t)lo.utiles.size();
  tp->ftiles = reinterpret_cast<int4 *>(base + lo.o_ftiles);
  tp->n_ftiles = (int32_t)lo.ftiles.size();
  tp->rtiles = reinterpret_cast<int4 *>(base + lo.o_rtiles);
  tp->n_rtiles = (int32_t)lo.rtiles.size();
  tp->qtiles = reinterpret_cast<int4 *>(base + lo.o_qtiles);
  tp->n_qtiles = (int32_t)lo.qtiles.size();
  tp->gram_tiles = reinterpret_cast<int4 *>(base + lo.o_gtiles);
  tp->n_gram_tiles = (int32_t)lo.gram_tiles.size();
  tp->trsm_tiles = reinterpret_cast<int4 *>(base + lo.o_ttiles);
  tp->n_trsm_tiles = (int32_t)lo.trsm_tiles.size();
  tp->precision = lo.precision;
  tp->max_r = lo.max_r;
  auto bind_sched = [&](const Schedule &sc, DevSchedule &d) {
    d.tiles = reinterpret_cast<const int4 *>(base + sc.o_tiles);
    d.off = reinterpret_cast<const int *>(base + sc.o_off);
    d.grid = sc.grid;
  };
  bind_sched(lo.s_update, tp->d_update);
  bind_sched(lo.s_bq, tp->d_bq);
  bind_sched(lo.s_btp, tp->d_btp);
  bind_sched(lo.s_gram, tp->d_gram);
  bind_sched(lo.s_trsm, tp->d_trsm);
}

cudaError_t encode_maps(const DevLayer *dl, int32_t L, LayerMaps *dst) {
  std::vector<LayerMaps> maps(std::max(L, 1));
  std::memset(maps.data(), 0, sizeof(LayerMaps) * maps.size());
  for (int32_t l = 0; l < L; ++l) {
    const DevLayer &d = dl[l];
    LayerMaps &m = maps[l];
    const uint64_t p16 = (uint64_t)d.ldp * 2, p32 = (uint64_t)d.ldp * 4;
    const bool ok = encode_bf16_2d(&m.P_hi, d.P_hi, d.r, d.m, p16, 64, 128) &&
                    encode_bf16_2d(&m.R_hi, d.R_hi, d.r, d.n, p16, 64, 128) &&
                    encode_bf16_2d(&m.Qn_hi, d.Qn_hi, d.r, d.n, p16, 64, 128) &&
                    encode_f32_2d(&m.Mf, d.M, d.n, d.m, (uint64_t)d.ldm * 4, 32, 128) &&
                    encode_f32_2d(&m.Xf, d.X, d.n, d.m, (uint64_t)d.ldx * 4, 32, 128) &&
                    encode_f32_2d(&m.Mf16, d.M, d.n, d.m, (uint64_t)d.ldm * 4, 16, 128) &&
                    encode_f32_2d(&m.Xf16, d.X, d.n, d.m, (uint64_t)d.ldx * 4, 16, 128) &&
                    (d.g_dtype != DT_BF16 || encode_bf16_2d(&m.Gh16, d.G, d.n, d.m, (uint64_t)d.ldg * 2, 16, 128)) &&
                    (d.g_dtype != DT_BF16 || encode_bf16_2d(&m.Gh64, d.G, d.n, d.m, (uint64_t)d.ldg * 2, 64, 128)) &&
                    encode_bf16_2d(&m.Qn_mn, d.Qn_hi, d.r, d.n, p16, 64, 64) &&
                    encode_bf16_2d(&m.P_mn, d.P_hi, d.r, d.m, p16, 64, 64) &&
                    encode_bf16_2d(&m.Bh_mn, d.Bh, d.n, d.m, (uint64_t)d.ldbh * 2, 64, 64) &&
                    encode_bf16_2d(&m.Bh_k, d.Bh, d.n, d.m, (uint64_t)d.ldbh * 2, 64, 128) &&
                    encode_f32_2d(&m.Praw, d.P_raw, d.r, d.m, p32, 32, 128) &&
                    encode_f32_2d(&m.Rst, d.R, d.r, d.n, p32, 32, 128) &&
                    encode_f32_2d(&m.Pf, d.P, d.r, d.m, p32, 32, 128) &&
                    encode_f32_2d(&m.PTraw, d.PT_raw, d.m, d.r, (uint64_t)d.ldmt * 4, 32, 128) &&
                    encode_f32_2d(&m.PT, d.PT, d.m, d.r, (uint64_t)d.ldmt * 4, 32, 128) &&
                    encode_f32_2d(&m.PTraw_t, d.PT_raw, d.m, d.r, (uint64_t)d.ldmt * 4, 32, 32) &&
                    encode_f32_2d(&m.PT_t, d.PT, d.m, d.r, (uint64_t)d.ldmt * 4, 32, 32) &&
                    encode_f32_2d(&m.Sst, d.S, d.r, d.r, p32, 32, 128) &&
                    encode_f32_2d(&m.Linv, d.Linv, d.r, d.r, p32, 32, 128) &&
                    encode_f32_2d(&m.Linv32, d.Linv, d.r, d.r, p32, 32, 32) &&
                    (d.P_lo == nullptr ||
                     (encode_bf16_2d(&m.P_lo, d.P_lo, d.r, d.m, p16, 64, 128) &&
                      encode_bf16_2d(&m.R_lo, d.R_lo, d.r, d.n, p16, 64, 128) &&
                      encode_bf16_2d(&m.Qn_lo, d.Qn_lo, d.r, d.n, p16, 64, 128) &&
                      encode_bf16_2d(&m.Qn_lo_mn, d.Qn_lo, d.r, d.n, p16, 64, 64) &&
                      encode_bf16_2d(&m.P_lo_mn, d.P_lo, d.r, d.m, p16, 64, 64) &&
                      encode_bf16_2d(&m.Bl_mn, d.Bl, d.n, d.m, (uint64_t)d.ldbh * 2, 64, 64) &&
                      encode_bf16_2d(&m.Bl_k, d.Bl, d.n, d.m, (uint64_t)d.ldbh * 2, 64, 128) &&
                      encode_bf16_2d(&m.P_hi32, d.P_hi, d.r, d.m, p16, 32, 128) &&
                      encode_bf16_2d(&m.P_lo32, d.P_lo, d.r, d.m, p16, 32, 128) &&
                      encode_bf16_2d(&m.R_hi32, d.R_hi, d.r, d.n, p16, 32, 128) &&
                      encode_bf16_2d(&m.R_lo32, d.R_lo, d.r, d.n, p16, 32, 128) &&
                      encode_bf16_2d(&m.Qn_hi32, d.Qn_hi, d.r, d.n, p16, 32, 128) &&
                      encode_bf16_2d(&m.Qn_lo32, d.Qn_lo, d.r, d.n, p16, 32, 128)));
    if (!ok) return cudaErrorInvalidValue;
  }
  return cudaMemcpy(dst, maps.data(), sizeof(LayerMaps) * maps.size(), cudaMemcpyHostToDevice);
}

cudaError_t init(const TcLayout &lo, char *base, const DevLayer *dl, int32_t L, TcPlan *tp) {
  cudaError_t e = encode_maps(dl, L, tp->maps);
  auto up = [&](int4 *dst, const std::vector<int4> &v) {
    return v.empty() ? cudaSuccess : cudaMemcpy(dst, v.data(), sizeof(int4) * v.size(), cudaMemcpyHostToDevice);
  };
  if (e == cudaSuccess) e = up(tp->utiles, lo.utiles);
  if (e == cudaSuccess) e = up(tp->ftiles, lo.ftiles);
  if (e == cudaSuccess) e = up(tp->rtiles, lo.rtiles);
  if (e == cudaSuccess) e = up(tp->qtiles, lo.qtiles);
  if (e == cudaSuccess) e = up(tp->gram_tiles, lo.gram_tiles);
  if (e == cudaSuccess) e = up(tp->trsm_tiles, lo.trsm_tiles);
  for (const Schedule *sc : {&lo.s_update, &lo.s_bq, &lo.s_btp, &lo.s_gram, &lo.s_trsm}) {
    if (e == cudaSuccess && !sc->tiles.empty())
      e = cudaMemcpy(base + sc->o_tiles, sc->tiles.data(), sizeof(int4) * sc->tiles.size(), cudaMemcpyHostToDevice);
    if (e == cudaSuccess)
      e = cudaMemcpy(base + sc->o_off, sc->off.data(), sizeof(int) * sc->off.size(), cudaMemcpyHostToDevice);
  }
  // shared-memory budget: operand stages + 2 staging buffers of (128 x 32 + 4 x 32 x 32) fp32
  // and 1 KB of column partials
  const uint32_t budget = 227u * 1024u - 1024u - 4u * 128u * 32u * 4u - 1024u - 512u - 256u;
  const bool x3 = lo.precision == DION_PREC_BF16X3;
  const uint32_t nb64 = (uint32_t)std::max(1, (lo.max_r + 63) / 64);
  // B Q / B^T P (CTA pairs): A tile + per 256-column part of N, this CTA's half (two 64-column boxes)
  const uint32_t bq_boxes = 2u * (uint32_t)std::max(1, ((lo.max_r + 15) / 16 * 16 + 255) / 256);
  // BF16X3: the high and low halves of both operands
  const uint32_t stage = (x3 ? 2u : 1u) * (128u * 64u * 2u + bq_boxes * 64u * 64u * 2u);
  const int stages = (int)std::min<uint32_t>(4u, budget / stage);
  const uint32_t nb128 = (uint32_t)std::max(1, (lo.max_r + 127) / 128);
  // Gram / TRSM (CTA pairs): A box + per 256-column part of N, this CTA's half (one 128-row box)
  const uint32_t o_parts = (uint32_t)std::max(1, ((lo.max_r + 15) / 16 * 16 + 255) / 256);
  // BF16X3: every stage also holds the lo boxes its converters write
  const uint32_t ostage = (x3 ? 2u : 1u) * 128u * 32u * 4u * (1u + o_parts);
  const int ostages = (int)std::min<uint32_t>(4u, budget / ostage);
  // TRSM: one 256-column part per sub-tile, so a stage holds the A box and one B box; up to 5
  // stages (the solve gains from the bytes in flight: the final pass 0.294 -> 0.279 ms on the
  // 1.3B stack with 5 against 4)
  const uint32_t tstage = (x3 ? 2u : 1u) * 128u * 32u * 4u * 2u;
  const int tstages = (int)std::min<uint32_t>(5u, budget / tstage);
  if (stages < 2 || ostages < 2 || tstages < 2) return cudaErrorInvalidValue;
  tp->nb64 = nb64;
  tp->bq_boxes = bq_boxes;
  tp->nb128 = nb128;
  tp->o_parts = o_parts;
  tp->f_stages = tp->r_stages = stages;
  tp->o_stages = ostages;
  tp->t_stages = tstages;
  tp->f_smem = form_bq_smem(stages, stage);
  tp->r_smem = btp_smem(stages, stage);
  tp->o_smem = std::max(orth_smem(ostages, ostage), orth_smem(tstages, tstage));
  uint32_t cols = 32;
  while (cols < (uint32_t)((lo.max_r + 15) / 16 * 16)) cols <<= 1;
  tp->tmem_cols = cols;
  if (e == cudaSuccess) e = setup_update_kernel(x3);
  if (e == cudaSuccess) e = setup_bq_kernels(tp->f_smem, tp->r_smem, x3);
  tp->fb_smem = fused_bq_smem(bq_boxes);
  if (tp->fuse_buffer && tp->fb_smem > 227u * 1024u) return cudaErrorInvalidValue;
  if (e == cudaSuccess && tp->fuse_buffer) e = setup_fused_bq_kernel(tp->fb_smem);
  if (e == cudaSuccess) e = setup_orth_kernels(tp->o_smem, x3);
  if (e == cudaSuccess) e = prepare_chol_inv_tc(lo.max_r, &tp->chol_tc_smem);
  int dev = 0, sms = 0;
  if (e == cudaSuccess) e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  tp->num_sms = sms;
  tp->launches = tp->fuse_buffer ? 17 : x3 ? 19 : 18;  // BF16X3: the split of B after the gate
  return e;
}

int32_t launches_per_step(const TcPlan &tp) { return tp.launches; }

void refresh(const TcPlan &tp, const Shared &sh, cudaStream_t s) { launch_qn_refresh(sh, tp, s); }

void step(dion_plan *p, const TcPlan &tp, const Shared &sh_in, const StepArgs &a, const int4 *btiles,
          int32_t n_btiles, const int4 *ctiles, int32_t n_ctiles, size_t chol_smem, cudaStream_t s) {
  Shared sh = sh_in;
  sh.b_in_m = (tp.fuse_buffer && a.gate_mode != GATE_ALWAYS) ? 1 : 0;  // the norms pass writes B into M
  if (tp.fuse_buffer && a.gate_mode == GATE_ALWAYS) {
    launch_fused_bq(sh, tp, false, s);  // B = M + G, Bh, ||B||, ||M_{t-1}||, P = B Q_{t-1} (every layer)
    tick(p, s, "tc_form_bq");
    launch_gate(sh, a, s);
    tick(p, s, "gate");
  } else if (tp.fuse_buffer) {
    // gated modes: the norms and the gate first, then the fused kernel on the Dion-branch layers
    launch_norms_gate(sh, a, tp.ftiles, tp.n_ftiles, s);
    tick(p, s, "norms_gate");
    launch_fused_bq(sh, tp, true, s);
    tick(p, s, "tc_form_bq");
  } else {
    // BF16X3 in a gated mode writes the halves of B only for the Dion-branch layers, after the
    // gate (a local layer needs B alone): 10 B/element on every layer, 8 more on syncing ones
    const bool x3_split = tp.precision == DION_PREC_BF16X3 && a.gate_mode != GATE_ALWAYS;
    launch_form_b(sh, btiles, n_btiles, s, !x3_split);  // B = M + G (its bf16 copy or halves), the norms
    tick(p, s, "form_b");
    launch_gate(sh, a, s);
    tick(p, s, "gate");
    if (tp.precision == DION_PREC_BF16X3) {
      launch_split_b(sh, btiles, n_btiles, x3_split, s);
      tick(p, s, "split_b");
    }
    launch_form_bq(sh, tp, s);  // P = B Q_{t-1} on the layers that take the Dion branch
    tick(p, s, "tc_bq");
  }
  static const char *kChol[3] = {"chol_inv0", "chol_inv1", "chol_inv2"};
  static const char *kGram[3] = {"tc_gram0", "tc_gram1", "tc_gram2"};
  static const char *kTrsm[3] = {"tc_trsm0", "tc_trsm1", "tc_trsm2"};
  const bool x3 = tp.precision == DION_PREC_BF16X3;
  for (int pass = 0; pass < 3; ++pass) {  // CholeskyQR2; the third pass only after a shifted retry
    launch_orth(sh, tp, true, pass, s);  // S = X^T X
    tick(p, s, kGram[pass]);
    if (pass == 0) launch_chol_inv_tc(sh, tp.maps, tp.chol_tc_smem, s);  // trailing update on tensor cores (3xTF32)
    else launch_chol_inv(sh, chol_smem, pass, x3 ? 1e-3f : 6e-2f, s);  // passes 1-2: usually the first-order factor
    tick(p, s, kChol[pass]);
    launch_orth(sh, tp, false, pass, s);  // X L^{-T} and its transpose, or its bf16 copy (halves) at the end
    tick(p, s, kTrsm[pass]);
  }
  launch_btp(sh, tp, s);  // R = B^T P
  tick(p, s, "tc_btp");
  launch_colnorm_reduce(sh, ctiles, n_ctiles, a.eps_col, s);  // 1 / (||R_j|| + eps) from tile partials
  tick(p, s, "colnorm_reduce");
  launch_colnorm_scale(sh, tp, s);  // Q_t = R diag(...), its bf16 copy
  tick(p, s, "colnorm_scale");
  launch_update(sh, tp, a.mu, a.eta, a.keep_sync, s);  // M_t, X_t (error feedback, update)
  tick(p, s, "tc_update");
  launch_local(sh, btiles, n_btiles, a.eta_local, a.keep_local, s);
  tick(p, s, "local");
  launch_finalize(sh, a, s);
  tick(p, s, "finalize");
}

void step_phase(const TcPlan &tp, const Shared &sh_in, const StepArgs &a, int32_t phase, const int4 *btiles,
                int32_t n_btiles, const int4 *ctiles, int32_t n_ctiles, size_t chol_smem, cudaStream_t s) {
  Shared sh = sh_in;
  // with bf16 gradients the norms pass writes B into M before the branch is known (the flow
  // of the gated modes), whatever the gate mode; the later phases read B from M
  sh.b_in_m = tp.fuse_buffer ? 1 : 0;
  const bool x3 = tp.precision == DION_PREC_BF16X3;
  switch (phase) {
    case DION_PHASE_NORMS:  // B = M + G, ||B||, this worker's RMMC, prev_norm <- ||B||
      if (tp.fuse_buffer) {
        launch_norms_gate(sh, a, tp.ftiles, tp.n_ftiles, s);
      } else {
        launch_form_b(sh, btiles, n_btiles, s, !x3);  // BF16X3: the halves after the branch is known
        launch_gate(sh, a, s);
      }
      break;
    case DION_PHASE_POWER:  // the branch from the reduced RMMC, then P = B Q on the Dion layers
      launch_gate_reduced(sh, a, s);
      if (x3) launch_split_b(sh, btiles, n_btiles, true, s);
      if (tp.fuse_buffer) launch_fused_bq(sh, tp, true, s);
      else launch_form_bq(sh, tp, s);
      break;
    case DION_PHASE_ORTHO:  // Orthogonalize the averaged P, then R = B^T P
      launch_transpose_praw(sh, tp, s);  // the first Gram reads P_raw^T
      for (int pass = 0; pass < 3; ++pass) {
        launch_orth(sh, tp, true, pass, s);
        if (pass == 0) launch_chol_inv_tc(sh, tp.maps, tp.chol_tc_smem, s);
        else launch_chol_inv(sh, chol_smem, pass, x3 ? 1e-3f : 6e-2f, s);
        launch_orth(sh, tp, false, pass, s);
      }
      launch_btp(sh, tp, s);
      break;
    default:  // UPDATE: Q_t from the averaged R, error feedback and parameter update, local branch
      launch_r_refresh(sh, tp, s);
      launch_colnorm_reduce(sh, ctiles, n_ctiles, a.eps_col, s);
      launch_colnorm_scale(sh, tp, s);
      launch_update(sh, tp, a.mu, a.eta, a.keep_sync, s);
      launch_local(sh, btiles, n_btiles, a.eta_local, a.keep_local, s);
      launch_finalize(sh, a, s);
      break;
  }
}

void destroy(TcPlan *tp) { (void)tp; }

}  // namespace tc
}  // namespace cd
