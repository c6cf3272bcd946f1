// CUDA-core kernels of the CurvaDion step (fp32 operands, fp32 FMA, fp64 partial sums).
//
// These kernels serve the DION_PREC_FP32 mode end to end, and the buffer, gate, Cholesky,
// column-normalization, local-branch and finalize steps of every mode.  Every kernel reads
// its work list (tiles) from device memory and skips layers whose `active` flag says they
// do not take the Dion branch this step, so one fixed launch sequence serves every gate
// decision without a host round trip.
#include "common.cuh"

#include <cmath>

namespace cd {

// ===================================================================== buffer + norms ===
// B = M + G written into M (Algorithm 1/2 buffer line); per tile, sum of B^2 (Algorithm 2's
// ||B_t||) and sum of M_{t-1}^2 (Equation 1's ||M(t-1)||) as fp64 partials in a fixed slot.
// Tile = {layer, first row, rows, slot}.
constexpr int kRowThreads = 256;

template <int GT>
__device__ __forceinline__ void load_g4(const void *G, int64_t off, float g[4]) {
  if (GT == DT_BF16) {
    const uint2 v = *reinterpret_cast<const uint2 *>(static_cast<const __nv_bfloat16 *>(G) + off);
    g[0] = bf16_bits_to_float(v.x & 0xffffu);
    g[1] = bf16_bits_to_float(v.x >> 16);
    g[2] = bf16_bits_to_float(v.y & 0xffffu);
    g[3] = bf16_bits_to_float(v.y >> 16);
  } else {
    const float4 v = *reinterpret_cast<const float4 *>(static_cast<const float *>(G) + off);
    g[0] = v.x; g[1] = v.y; g[2] = v.z; g[3] = v.w;
  }
}

template <int GT>
__device__ __forceinline__ float load_g1(const void *G, int64_t off) {
  if (GT == DT_BF16) return __bfloat162float(static_cast<const __nv_bfloat16 *>(G)[off]);
  return static_cast<const float *>(G)[off];
}

template <int GT, bool HAS_BH>
__device__ void form_b_tile(const DevLayer &L, int64_t row0, int64_t nrows, float sb[4], float sm[4]) {
  const int64_t n = L.n, n4 = n >> 2;
  for (int64_t rr = 0; rr < nrows; ++rr) {
    const int64_t i = row0 + rr;
    float *Mrow = L.M + i * L.ldm;
    const int64_t goff = i * L.ldg;
    for (int64_t c4 = threadIdx.x; c4 < n4; c4 += kRowThreads) {
      float4 m = *reinterpret_cast<float4 *>(Mrow + 4 * c4);
      float g[4];
      load_g4<GT>(L.G, goff + 4 * c4, g);
      sm[0] = fmaf(m.x, m.x, sm[0]); sm[1] = fmaf(m.y, m.y, sm[1]);
      sm[2] = fmaf(m.z, m.z, sm[2]); sm[3] = fmaf(m.w, m.w, sm[3]);
      m.x += g[0]; m.y += g[1]; m.z += g[2]; m.w += g[3];
      sb[0] = fmaf(m.x, m.x, sb[0]); sb[1] = fmaf(m.y, m.y, sb[1]);
      sb[2] = fmaf(m.z, m.z, sb[2]); sb[3] = fmaf(m.w, m.w, sb[3]);
      *reinterpret_cast<float4 *>(Mrow + 4 * c4) = m;
      if (HAS_BH) {  // bf16 copy of B (operand of the tensor-core contractions)
        const __nv_bfloat162 h01 = __floats2bfloat162_rn(m.x, m.y), h23 = __floats2bfloat162_rn(m.z, m.w);
        uint2 hv;
        hv.x = *reinterpret_cast<const uint32_t *>(&h01);
        hv.y = *reinterpret_cast<const uint32_t *>(&h23);
        *reinterpret_cast<uint2 *>(L.Bh + i * L.ldbh + 4 * c4) = hv;
      }
    }
    for (int64_t c = 4 * n4 + threadIdx.x; c < n; c += kRowThreads) {
      const float mo = Mrow[c];
      const float b = mo + load_g1<GT>(L.G, goff + c);
      sm[0] = fmaf(mo, mo, sm[0]);
      sb[0] = fmaf(b, b, sb[0]);
      Mrow[c] = b;
      if (HAS_BH) L.Bh[i * L.ldbh + c] = __float2bfloat16_rn(b);
    }
  }
}

__global__ void __launch_bounds__(kRowThreads) form_b_kernel(Shared sh, const int4 *tiles) {
  __shared__ double red[kRowThreads / 32];
  const int4 t = tiles[blockIdx.x];
  const DevLayer &L = sh.layers[t.x];
  float sb[4] = {0.f, 0.f, 0.f, 0.f}, sm[4] = {0.f, 0.f, 0.f, 0.f};
  if (L.Bh != nullptr) {
    if (L.g_dtype == DT_BF16) form_b_tile<DT_BF16, true>(L, t.y, t.z, sb, sm);
    else form_b_tile<DT_FP32, true>(L, t.y, t.z, sb, sm);
  } else {
    if (L.g_dtype == DT_BF16) form_b_tile<DT_BF16, false>(L, t.y, t.z, sb, sm);
    else form_b_tile<DT_FP32, false>(L, t.y, t.z, sb, sm);
  }
  const double b = block_sum<kRowThreads>(((double)sb[0] + sb[1]) + ((double)sb[2] + sb[3]), red);
  const double mo = block_sum<kRowThreads>(((double)sm[0] + sm[1]) + ((double)sm[2] + sm[3]), red);
  if (threadIdx.x == 0) {
    sh.bpart[2 * t.w] = b;
    sh.bpart[2 * t.w + 1] = mo;
  }
}

void launch_form_b(const Shared &sh, const int4 *tiles, int32_t ntiles, cudaStream_t s) {
  if (ntiles > 0) form_b_kernel<<<ntiles, kRowThreads, 0, s>>>(sh, tiles);
}

// =============================================================================== gate ===
// Algorithm 2: RMMC_l = | ||B|| - prev_l | / (prev_l + eps); prev_l = ||B||; global max over
// layers; strict compare with tau (a non-finite RMMC counts as above every threshold); the
// gate mode then decides which layers take the Dion branch.
constexpr int kGateThreads = 1024;

__device__ __forceinline__ bool above(double v, float tau) {
  return !isfinite(v) || v > (double)tau;
}

__global__ void __launch_bounds__(kGateThreads) gate_kernel(Shared sh, StepArgs a) {
  __shared__ double wmax[kGateThreads / 32];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int L = sh.num_layers;
  double my_max = -INFINITY;
  for (int l = warp; l < L; l += kGateThreads / 32) {
    const DevLayer &Ly = sh.layers[l];
    double sb = 0.0, sm = 0.0;
    for (int k = lane; k < Ly.bpart_cnt; k += 32) {  // fixed lane/slot assignment
      sb += sh.bpart[2 * (Ly.bpart_off + k)];
      sm += sh.bpart[2 * (Ly.bpart_off + k) + 1];
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      sb += __shfl_xor_sync(0xffffffffu, sb, o);
      sm += __shfl_xor_sync(0xffffffffu, sm, o);
    }
    if (lane == 0) {
      const double nb = sqrt(sb);
      const double prev = a.prev_norm[l];
      const double rm = fabs(nb - prev) / (prev + (double)a.eps_rmmc);
      if (!isfinite(nb)) set_status(sh.status, ST_NONFINITE);
      a.rmmc[l] = rm;
      a.prev_norm[l] = nb;
      a.flags[l] = above(rm, Ly.tau) ? 1 : 0;
      sh.norm_b[l] = nb;
      sh.norm_m_before[l] = sqrt(sm);
      my_max = isfinite(rm) ? fmax(my_max, rm) : INFINITY;
    }
  }
  if (lane == 0) wmax[warp] = my_max;
  __syncthreads();  // makes the per-layer global writes above visible to the whole block
  __shared__ int gflag_s;
  if (threadIdx.x == 0) {
    double g = -INFINITY;
    for (int w = 0; w < kGateThreads / 32; ++w) g = fmax(g, wmax[w]);
    const int gf = (L > 0 && above(g, a.tau_global)) ? 1 : 0;
    a.gflag[0] = (uint8_t)gf;
    gflag_s = gf;
  }
  __syncthreads();
  for (int l = threadIdx.x; l < L; l += kGateThreads) {
    int act;
    switch (a.gate_mode) {
      case GATE_ALWAYS: act = 1; break;
      case GATE_GLOBAL: act = gflag_s; break;
      case GATE_PER_LAYER: act = a.flags[l]; break;
      default: act = (a.step % a.period) == 0; break;
    }
    sh.active[l] = (uint8_t)act;
  }
}

void launch_gate(const Shared &sh, const StepArgs &a, cudaStream_t s) {
  gate_kernel<<<1, kGateThreads, 0, s>>>(sh, a);
}

// ==================================================================== grouped GEMM ===
// C = op(A) op(B) over a list of problems; 64 x 64 output tiles, 16-deep k slices staged in
// shared memory, 4 x 4 register tile per thread.  Tile = {problem, tile row, tile col}.
constexpr int GBM = 64, GBN = 64, GBK = 16, kGemmThreads = 256;

__global__ void __launch_bounds__(kGemmThreads) gemm_kernel(Shared sh, const GemmProblem *probs,
                                                            const int4 *tiles) {
  const int4 t = tiles[blockIdx.x];
  const GemmProblem p = probs[t.x];
  if (!sh.active[p.layer]) return;
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  const int64_t i0 = (int64_t)t.y * GBM, j0 = (int64_t)t.z * GBN;
  if (p.mode != GEMM_ACTIVE && !sh.orth_shifted[p.layer]) {
    if (p.mode == GEMM_SHIFTED_OR_COPY) {  // C = A (same shape, A not transposed)
      for (int e = tid; e < GBM * GBN; e += kGemmThreads) {
        const int64_t gi = i0 + e / GBN, gj = j0 + e % GBN;
        if (gi < p.Mrows && gj < p.Ncols) p.C[gi * p.ldc + gj] = p.A[gi * p.lda + gj];
      }
    }
    return;
  }
  __shared__ float As[GBK][GBM + 4];
  __shared__ float Bs[GBK][GBN + 4];
  float acc[4][4] = {};
  for (int64_t k0 = 0; k0 < p.K; k0 += GBK) {
#pragma unroll
    for (int s = 0; s < (GBM * GBK) / kGemmThreads; ++s) {
      const int idx = tid + s * kGemmThreads;
      int ii, kk;
      if (p.transA) { ii = idx % GBM; kk = idx / GBM; } else { kk = idx % GBK; ii = idx / GBK; }
      const int64_t gi = i0 + ii, gk = k0 + kk;
      float v = 0.f;
      if (gi < p.Mrows && gk < p.K) v = p.transA ? p.A[gk * p.lda + gi] : p.A[gi * p.lda + gk];
      As[kk][ii] = v;
    }
#pragma unroll
    for (int s = 0; s < (GBN * GBK) / kGemmThreads; ++s) {
      const int idx = tid + s * kGemmThreads;
      int jj, kk;
      if (p.transB) { kk = idx % GBK; jj = idx / GBK; } else { jj = idx % GBN; kk = idx / GBN; }
      const int64_t gj = j0 + jj, gk = k0 + kk;
      float v = 0.f;
      if (gj < p.Ncols && gk < p.K) v = p.transB ? p.B[gj * p.ldb + gk] : p.B[gk * p.ldb + gj];
      Bs[kk][jj] = v;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < GBK; ++kk) {
      float av[4], bv[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) av[i] = As[kk][ty * 4 + i];
#pragma unroll
      for (int j = 0; j < 4; ++j) bv[j] = Bs[kk][tx * 4 + j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(av[i], bv[j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int64_t gi = i0 + ty * 4 + i;
    if (gi >= p.Mrows) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int64_t gj = j0 + tx * 4 + j;
      if (gj < p.Ncols) p.C[gi * p.ldc + gj] = acc[i][j];
    }
  }
}

void launch_gemm(const Shared &sh, const GemmProblem *probs, const int4 *tiles, int32_t ntiles,
                 cudaStream_t s) {
  if (ntiles > 0) gemm_kernel<<<ntiles, kGemmThreads, 0, s>>>(sh, probs, tiles);
}

// =========================================================== Cholesky + L^{-1} ===
// Orthogonalize by Cholesky QR: S = P^T P = L L^T, P <- P L^{-T}.  The step runs it twice
// (CholeskyQR2) so that P is orthonormal to fp32 roundoff.  When a pivot is <= 0 or not
// finite, the pass is retried on S + s I with the shift of shifted CholeskyQR (Fukaya,
// Kannan, Nakatsukasa, Yamamoto, Yanagisawa 2020): s = 11 (m r + r (r + 1)) u trace(S),
// u = 2^-24; the layer is then marked and a third pass runs.  Every pass multiplies P by an
// upper-triangular matrix with positive diagonal, so the final P is the Q factor of the
// thin QR of the original P with a positive-diagonal triangular factor.
// One CTA per layer (r <= 512): right-looking blocked Cholesky with 32-wide block columns,
// then L^{-1} block row by block row.  S and L^{-1} live in global memory (L2-resident);
// diagonal blocks, panels and partial products are staged in shared memory.  Only the lower
// triangle of S is overwritten, so a retry rebuilds S from its upper triangle and the saved
// diagonal.  If the shifted retry also fails, DION_ERR_BREAKDOWN is set and L^{-1} = 0 for
// the layer, so its P, R and Q become 0, M becomes B and X is unchanged (no NaN written).
constexpr int CB = 32, CBP = CB + 1, kCholThreads = 512;
constexpr int DION_MAX_RANK_PAD = 512;  // diag0 slot: r <= 512

__device__ __forceinline__ int64_t tri_row(int64_t p) {
  // largest b with b (b + 1) / 2 <= p
  int64_t b = (int64_t)((sqrt(8.0 * (double)p + 1.0) - 1.0) * 0.5);
  while ((b + 1) * (b + 2) / 2 <= p) ++b;
  while (b * (b + 1) / 2 > p) --b;
  return b;
}

// Factors the lower triangle of S (r x r, row-major) in place.  Returns false (uniformly over
// the block) on a pivot <= 0 or non-finite.  Smem: D (CB x CBP), Pn (r x CBP).
__device__ bool cholesky_blocked(float *S, int r, int64_t ls, float *D, float *Pn, int *bad) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  if (tid == 0) *bad = 0;
  __syncthreads();
  for (int k0 = 0; k0 < r; k0 += CB) {
    const int nb = min(CB, r - k0);
    for (int e = tid; e < CB * CB; e += kCholThreads) {
      const int i = e / CB, j = e % CB;
      float v;
      if (i < nb && j < nb) v = (j <= i) ? S[(int64_t)(k0 + i) * ls + k0 + j] : 0.f;
      else v = (i == j) ? 1.f : 0.f;  // identity padding of a short last block
      D[i * CBP + j] = v;
    }
    __syncthreads();
    if (warp == 0) {
      for (int j = 0; j < CB; ++j) {
        const float djj = D[j * CBP + j];
        if (!(djj > 0.f) || !isfinite(djj)) {
          if (lane == 0) *bad = 1;
          break;  // uniform across the warp: every lane read the same djj
        }
        const float sq = sqrtf(djj);
        __syncwarp();
        if (lane == j) D[j * CBP + j] = sq;
        if (lane > j) D[lane * CBP + j] /= sq;
        __syncwarp();
        if (lane > j) {
          const float lij = D[lane * CBP + j];
          for (int k = j + 1; k <= lane; ++k) D[lane * CBP + k] -= lij * D[k * CBP + j];
        }
        __syncwarp();
      }
    }
    __syncthreads();
    if (*bad) return false;
    for (int e = tid; e < nb * nb; e += kCholThreads) {
      const int i = e / nb, j = e % nb;
      if (j <= i) S[(int64_t)(k0 + i) * ls + k0 + j] = D[i * CBP + j];
    }
    // panel: rows below the block solve x L11^T = s
    const int t = r - k0 - nb;
    for (int ii = tid; ii < t; ii += kCholThreads) {
      const int64_t row = (int64_t)(k0 + nb + ii) * ls + k0;
      float x[CB];
#pragma unroll
      for (int j = 0; j < CB; ++j) x[j] = (j < nb) ? S[row + j] : 0.f;
#pragma unroll
      for (int j = 0; j < CB; ++j) {
        float v = x[j];
#pragma unroll
        for (int k = 0; k < j; ++k) v -= x[k] * D[j * CBP + k];
        x[j] = v / D[j * CBP + j];
      }
#pragma unroll
      for (int j = 0; j < CB; ++j) {
        Pn[ii * CBP + j] = x[j];
        if (j < nb) S[row + j] = x[j];
      }
    }
    __syncthreads();
    // trailing update of the lower triangle: S22 -= L21 L21^T, in 4 x 4 micro tiles
    const int64_t nbt = (t + 3) / 4, pairs = nbt * (nbt + 1) / 2;
    for (int64_t pidx = tid; pidx < pairs; pidx += kCholThreads) {
      const int64_t bi = tri_row(pidx), bj = pidx - bi * (bi + 1) / 2;
      float acc[4][4] = {};
#pragma unroll 8
      for (int k = 0; k < CB; ++k) {
        float a[4], b[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int64_t ri = bi * 4 + u, rj = bj * 4 + u;
          a[u] = (ri < t) ? Pn[ri * CBP + k] : 0.f;
          b[u] = (rj < t) ? Pn[rj * CBP + k] : 0.f;
        }
#pragma unroll
        for (int u = 0; u < 4; ++u)
#pragma unroll
          for (int v = 0; v < 4; ++v) acc[u][v] = fmaf(a[u], b[v], acc[u][v]);
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int64_t ri = bi * 4 + u;
        if (ri >= t) continue;
#pragma unroll
        for (int v = 0; v < 4; ++v) {
          const int64_t rj = bj * 4 + v;
          if (rj < t && rj <= ri) S[(k0 + nb + ri) * ls + k0 + nb + rj] -= acc[u][v];
        }
      }
    }
    __syncthreads();
  }
  return true;
}

// pass 0 and 1: every active layer; pass 2: only layers marked by a shifted retry.
// Passes 1 and 2 factor the Gram matrix of an already nearly orthonormal X: when 1.5 times a
// power-iteration estimate of ||S - I||_2 is below near_identity, the factor of S = I + E is
// taken to first order, L = I + F with F = strictly-lower(E) + diag(E) / 2 and
// L^{-1} = I - F; the resulting X L^{-T} is then orthonormal up to O(||E||_2^2).
__global__ void __launch_bounds__(kCholThreads) chol_inv_kernel(Shared sh, int pass, float near_identity) {
  const int l = blockIdx.x;
  if (!sh.active[l]) return;
  if (pass == 2 && !sh.orth_shifted[l]) return;
  const DevLayer &Ly = sh.layers[l];
  const int r = (int)Ly.r;
  const int64_t ls = Ly.ldp;  // leading dimension of S and L^{-1}
  float *S = Ly.S;
  float *Li = Ly.Linv;
  extern __shared__ float smem[];
  float *D = smem;            // CB x CBP: diagonal block
  float *DI = D + CB * CBP;   // CB x CBP: its inverse
  float *diag0 = DI + CB * CBP;  // r: the diagonal of S before factorization
  float *Pn = diag0 + DION_MAX_RANK_PAD;  // panel (r x CBP) or partial products (CB x r)
  __shared__ int bad;
  __shared__ double trace_s;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  // The Gram producers may write only the lower triangle: mirror it into the upper one, which
  // the factorization never touches and the shifted retry restores the lower triangle from.
  // 32 x 32 tiles transposed through a per-warp shared scratch (Pn holds 33 r floats, so r / 32
  // warps have room), coalesced on both sides.
  {
    const int nt = (r + 31) / 32, nwm = min(kCholThreads / 32, r / 32);
    if (nwm == 0) {
      for (int64_t e = tid; e < (int64_t)r * r; e += kCholThreads) {
        const int64_t i = e / r, j = e % r;
        if (j > i) S[i * ls + j] = S[j * ls + i];
      }
    } else if (warp < nwm) {
      float *tb = Pn + warp * (32 * 33);
      const int npairs = nt * (nt - 1) / 2;
      for (int u = warp; u < npairs + nt; u += nwm) {
        int bi, bj;  // upper tile (bi, bj), bj >= bi; u < npairs: off-diagonal, else the diagonal tile
        if (u < npairs) {
          bj = (int)tri_row(u) + 1;
          bi = u - (bj - 1) * bj / 2;
        } else {
          bi = bj = u - npairs;
        }
        for (int y = 0; y < 32; ++y) {  // lower tile (bj, bi) -> scratch
          const int gi = bj * 32 + y, gj = bi * 32 + lane;
          tb[y * 33 + lane] = (gi < r && gj < r) ? S[(int64_t)gi * ls + gj] : 0.f;
        }
        __syncwarp();
        for (int y = 0; y < 32; ++y) {  // upper tile (bi, bj) = transpose
          const int gi = bi * 32 + y, gj = bj * 32 + lane;
          if (gi < r && gj < r && gj > gi) S[(int64_t)gi * ls + gj] = tb[lane * 33 + y];
        }
        __syncwarp();
      }
    }
    __syncthreads();
  }
  for (int i = tid; i < r; i += kCholThreads) diag0[i] = S[(int64_t)i * ls + i];
  if (pass >= 1) {
    // ||E||_2 of E = S - I by 8 power iterations (one warp per row, coalesced row reads)
    float *v = Pn, *wv = Pn + r;  // Pn holds at least 33 * r floats
    __shared__ float wn[kCholThreads / 32];
    __shared__ float lam_s;
    for (int i = tid; i < r; i += kCholThreads) v[i] = 1.f + 0.25f * __sinf(0.7f * (float)i);  // fixed start
    __syncthreads();
    float lam = 0.f;
    for (int itp = 0; itp < 8; ++itp) {
      for (int i = warp; i < r; i += kCholThreads / 32) {
        float acc0 = 0.f, acc1 = 0.f;
        int j = lane;
        for (; j + 32 < r; j += 64) {
          acc0 = fmaf(S[(int64_t)i * ls + j] - (i == j ? 1.f : 0.f), v[j], acc0);
          acc1 = fmaf(S[(int64_t)i * ls + j + 32] - (i == j + 32 ? 1.f : 0.f), v[j + 32], acc1);
        }
        if (j < r) acc0 = fmaf(S[(int64_t)i * ls + j] - (i == j ? 1.f : 0.f), v[j], acc0);
        float acc = acc0 + acc1;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
        if (lane == 0) wv[i] = acc;
      }
      __syncthreads();
      float pn = 0.f;
      for (int i = tid; i < r; i += kCholThreads) pn = fmaf(wv[i], wv[i], pn);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) pn += __shfl_xor_sync(0xffffffffu, pn, o);
      if (lane == 0) wn[warp] = pn;
      __syncthreads();
      if (tid == 0) {
        float a = 0.f;
        for (int w = 0; w < kCholThreads / 32; ++w) a += wn[w];
        lam_s = a;  // ||E v||^2
      }
      __syncthreads();
      const float nrm = sqrtf(lam_s);
      // ||E v|| / ||v||: v has unit norm from the second iteration on
      lam = nrm;
      const float inv = (nrm > 0.f && isfinite(nrm)) ? 1.f / nrm : 0.f;
      for (int i = tid; i < r; i += kCholThreads) v[i] = wv[i] * inv;
      __syncthreads();
      if (itp == 0) lam = INFINITY;  // the first product uses an unnormalized start vector
    }
    if (isfinite(lam) && 1.5f * lam < near_identity) {
      for (int64_t e = tid; e < (int64_t)r * r; e += kCholThreads) {
        const int64_t i = e / r, j = e % r;
        const float sij = S[i * ls + j];
        Li[i * ls + j] = (j < i) ? -sij : (j == i ? 1.f - 0.5f * (sij - 1.f) : 0.f);
      }
      return;
    }
  }
  __syncthreads();

  bool ok = cholesky_blocked(S, r, ls, D, Pn, &bad);
  bool shifted = false;
  if (!ok) {  // shifted retry: lower triangle from the untouched upper triangle, shifted diagonal
    if (tid == 0) {
      double tr = 0.0;
      for (int i = 0; i < r; ++i) tr += (double)diag0[i];
      trace_s = tr;
    }
    __syncthreads();
    const double u = 5.9604644775390625e-8;  // 2^-24
    const double shift = 11.0 * ((double)Ly.m * r + (double)r * (r + 1)) * u * trace_s;
    for (int64_t e = tid; e < (int64_t)r * r; e += kCholThreads) {
      const int64_t i = e / r, j = e % r;
      if (j < i) S[i * ls + j] = S[j * ls + i];
      else if (j == i) S[i * ls + j] = (float)((double)diag0[i] + shift);
    }
    __syncthreads();
    shifted = true;
    ok = (trace_s > 0.0) && isfinite(trace_s) && cholesky_blocked(S, r, ls, D, Pn, &bad);
  }
  if (tid == 0) {
    if (pass == 0) sh.orth_shifted[l] = shifted ? 1 : 0;
    else if (shifted) sh.orth_shifted[l] = 1;
  }
  if (!ok) {
    if (tid == 0) set_status(sh.status, ST_BREAKDOWN);
    for (int64_t e = tid; e < (int64_t)r * r; e += kCholThreads) Li[(e / r) * ls + e % r] = 0.f;
    return;
  }

  // ---------------- L^{-1}, block row by block row ----------------
  // Linv[I,I] = L[I,I]^{-1};  Linv[I,J] = -L[I,I]^{-1} sum_{K=J..I-1} L[I,K] Linv[K,J]  (J < I)
  for (int I0 = 0; I0 < r; I0 += CB) {
    const int nb = min(CB, r - I0);
    for (int e = tid; e < CB * CB; e += kCholThreads) {
      const int i = e / CB, j = e % CB;
      float v;
      if (i < nb && j < nb) v = (j <= i) ? S[(int64_t)(I0 + i) * ls + I0 + j] : 0.f;
      else v = (i == j) ? 1.f : 0.f;
      D[i * CBP + j] = v;
    }
    __syncthreads();
    if (warp == 0) {  // lane c solves L_II x = e_c
      float x[CB];
#pragma unroll
      for (int i = 0; i < CB; ++i) {
        float v = (i == lane) ? 1.f : 0.f;
#pragma unroll
        for (int k = 0; k < i; ++k) v -= D[i * CBP + k] * x[k];
        x[i] = v / D[i * CBP + i];
      }
#pragma unroll
      for (int i = 0; i < CB; ++i) DI[i * CBP + lane] = x[i];
    }
    // Row block I of L staged in shared memory: Lb[i][k] = L[I0+i][k], k < I0.
    for (int e = tid; e < CB * I0; e += kCholThreads) {
      const int i = e / I0, k = e % I0;
      Pn[i * I0 + k] = (i < nb) ? S[(int64_t)(I0 + i) * ls + k] : 0.f;
    }
    __syncthreads();
    // Thread c < I0 owns column c: T[i] = sum_{k=c}^{I0-1} Lb[i][k] Linv[k][c] for the 32 rows
    // i of the block (one load of Linv[k][c] feeds 32 FMAs), then Linv[I0+i][c] = -(DI T)[i].
    for (int c = tid; c < I0; c += kCholThreads) {
      float acc[CB];
#pragma unroll
      for (int i = 0; i < CB; ++i) acc[i] = 0.f;
      // Linv[k][c] = 0 for k < c (upper triangle, stored as zeros), so every lane of a warp can
      // start at the warp's first column: uniform trip counts, 8 independent loads in flight.
      const int kbeg = c & ~31;
      int k = kbeg;
      for (; k + 8 <= I0; k += 8) {
        float lk[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) lk[u] = Li[(int64_t)(k + u) * ls + c];
#pragma unroll
        for (int u = 0; u < 8; ++u)
#pragma unroll
          for (int i = 0; i < CB; ++i) acc[i] = fmaf(Pn[i * I0 + k + u], lk[u], acc[i]);
      }
      for (; k < I0; ++k) {
        const float lk = Li[(int64_t)k * ls + c];
#pragma unroll
        for (int i = 0; i < CB; ++i) acc[i] = fmaf(Pn[i * I0 + k], lk, acc[i]);
      }
#pragma unroll
      for (int i = CB - 1; i >= 0; --i) {  // in place: row i needs acc[j] for j <= i only
        float v = 0.f;
#pragma unroll
        for (int j = 0; j <= i; ++j) v = fmaf(DI[i * CBP + j], acc[j], v);
        acc[i] = -v;
      }
#pragma unroll
      for (int i = 0; i < CB; ++i)
        if (i < nb) Li[(int64_t)(I0 + i) * ls + c] = acc[i];
    }
    // diagonal block DI and zeros to its right
    for (int e = tid; e < nb * (r - I0); e += kCholThreads) {
      const int i = e / (r - I0), c = I0 + e % (r - I0);
      float v = 0.f;
      if (c < I0 + nb) {
        const int j = c - I0;
        v = (j <= i) ? DI[i * CBP + j] : 0.f;
      }
      Li[(int64_t)(I0 + i) * ls + c] = v;
    }
    __syncthreads();
  }
}

cudaError_t prepare_chol_inv(int32_t max_r, size_t *smem_out) {
  const int64_t big = (int64_t)max_r * CBP > (int64_t)CB * max_r ? (int64_t)max_r * CBP : (int64_t)CB * max_r;
  const size_t smem = sizeof(float) * (2 * CB * CBP + DION_MAX_RANK_PAD + big);
  *smem_out = smem;
  return cudaFuncSetAttribute(chol_inv_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
}

void launch_chol_inv(const Shared &sh, size_t smem, int32_t pass, float near_identity, cudaStream_t s) {
  if (sh.num_layers > 0) chol_inv_kernel<<<sh.num_layers, kCholThreads, smem, s>>>(sh, pass, near_identity);
}

// ===================================================================== ColumnNormalize ===
// Q_t[:, j] = R[:, j] / (||R[:, j]||_2 + eps_col).  Tile = {layer, 32-column group}; lane =
// column, warps stride over rows; fp32 sums of 16 rows folded into fp64 in a fixed order.
constexpr int kColThreads = 256;

__global__ void __launch_bounds__(kColThreads) colnorm_kernel(Shared sh, const int4 *tiles, float eps_col) {
  const int4 t = tiles[blockIdx.x];
  if (!sh.active[t.x]) return;
  const DevLayer &L = sh.layers[t.x];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t j = (int64_t)t.y * 32 + lane, n = L.n, r = L.r, ldp = L.ldp;
  __shared__ double part[kColThreads / 32][32];
  __shared__ float inv[32];
  double acc = 0.0;
  if (j < r) {
    float f = 0.f;
    int cnt = 0;
    for (int64_t i = warp; i < n; i += kColThreads / 32) {
      const float v = L.R[i * ldp + j];
      f = fmaf(v, v, f);
      if (++cnt == 16) { acc += f; f = 0.f; cnt = 0; }
    }
    acc += f;
  }
  part[warp][lane] = acc;
  __syncthreads();
  if (warp == 0) {
    double s = 0.0;
    for (int w = 0; w < kColThreads / 32; ++w) s += part[w][lane];
    inv[lane] = (float)(1.0 / (sqrt(s) + (double)eps_col));
  }
  __syncthreads();
  if (j < r) {
    const float c = inv[lane];
    for (int64_t i = warp; i < n; i += kColThreads / 32) {
      const float rv = L.R[i * ldp + j], q = rv * c;
      L.Q[i * L.ldq + j] = q;
      if (L.R_hi != nullptr) {  // bf16 operands of the tensor-core update (rounded to nearest)
        L.R_hi[i * ldp + j] = __float2bfloat16_rn(rv);
        L.Qn_hi[i * ldp + j] = __float2bfloat16_rn(q);
      }
    }
  }
}

void launch_colnorm(const Shared &sh, const int4 *tiles, int32_t ntiles, float eps_col, cudaStream_t s) {
  if (ntiles > 0) colnorm_kernel<<<ntiles, kColThreads, 0, s>>>(sh, tiles, eps_col);
}

// =============================================================== error feedback + update ===
// M = B - (1 - mu) P R^T and X = X - eta sqrt(m/n) P Q_t^T in one pass over the tile, plus the
// fp64 partial of ||M_t||^2 for Equation 1.  Tile = {layer, tile row, tile col, slot}.
constexpr int UBM = 64, UBN = 64, UBK = 16, kUpdThreads = 256;

__global__ void __launch_bounds__(kUpdThreads) update_kernel(Shared sh, const int4 *tiles, float mu, float eta) {
  // P, R: ld ldp; Q: ld ldq
  __shared__ float As[UBK][UBM + 4];
  __shared__ float Rs[UBK][UBN + 4];
  __shared__ float Qs[UBK][UBN + 4];
  __shared__ double red[kUpdThreads / 32];
  const int4 t = tiles[blockIdx.x];
  if (!sh.active[t.x]) return;
  const DevLayer &L = sh.layers[t.x];
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  const int64_t i0 = (int64_t)t.y * UBM, j0 = (int64_t)t.z * UBN, r = L.r, ldp = L.ldp;
  float u1[4][4] = {}, u2[4][4] = {};
  for (int64_t k0 = 0; k0 < r; k0 += UBK) {
#pragma unroll
    for (int s = 0; s < (UBM * UBK) / kUpdThreads; ++s) {
      const int idx = tid + s * kUpdThreads;
      const int kk = idx % UBK, ii = idx / UBK;
      const int64_t gk = k0 + kk, gi = i0 + ii, gj = j0 + ii;
      As[kk][ii] = (gi < L.m && gk < r) ? L.P[gi * ldp + gk] : 0.f;
      Rs[kk][ii] = (gj < L.n && gk < r) ? L.R[gj * ldp + gk] : 0.f;
      Qs[kk][ii] = (gj < L.n && gk < r) ? L.Q[gj * L.ldq + gk] : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < UBK; ++kk) {
      float a[4], b[4], q[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = As[kk][ty * 4 + i];
#pragma unroll
      for (int j = 0; j < 4; ++j) { b[j] = Rs[kk][tx * 4 + j]; q[j] = Qs[kk][tx * 4 + j]; }
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          u1[i][j] = fmaf(a[i], b[j], u1[i][j]);
          u2[i][j] = fmaf(a[i], q[j], u2[i][j]);
        }
    }
    __syncthreads();
  }
  const float dec = 1.f - mu, c = eta * L.sqrt_m_over_n;
  float ss = 0.f;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int64_t gi = i0 + ty * 4 + i;
    if (gi >= L.m) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int64_t gj = j0 + tx * 4 + j;
      if (gj >= L.n) continue;
      float *mp = L.M + gi * L.ldm + gj;
      const float mn = fmaf(-dec, u1[i][j], *mp);
      *mp = mn;
      float *xp = L.X + gi * L.ldx + gj;
      *xp = fmaf(-c, u2[i][j], *xp);
      ss = fmaf(mn, mn, ss);
    }
  }
  const double tot = block_sum<kUpdThreads>((double)ss, red);
  if (tid == 0) sh.upart[t.w] = tot;
}

void launch_update(const Shared &sh, const int4 *tiles, int32_t ntiles, float mu, float eta, cudaStream_t s) {
  if (ntiles > 0) update_kernel<<<ntiles, kUpdThreads, 0, s>>>(sh, tiles, mu, eta);
}

// ======================================================================== local branch ===
// Algorithm 2's else-branch: M = B is already in place; X = X - eta_local G.
template <int GT>
__device__ void local_tile(const DevLayer &L, int64_t row0, int64_t nrows, float eta_local) {
  const int64_t n = L.n, n4 = n >> 2;
  for (int64_t rr = 0; rr < nrows; ++rr) {
    const int64_t i = row0 + rr;
    float *Xrow = L.X + i * L.ldx;
    const int64_t goff = i * L.ldg;
    for (int64_t c4 = threadIdx.x; c4 < n4; c4 += kRowThreads) {
      float4 x = *reinterpret_cast<float4 *>(Xrow + 4 * c4);
      float g[4];
      load_g4<GT>(L.G, goff + 4 * c4, g);
      x.x = fmaf(-eta_local, g[0], x.x); x.y = fmaf(-eta_local, g[1], x.y);
      x.z = fmaf(-eta_local, g[2], x.z); x.w = fmaf(-eta_local, g[3], x.w);
      *reinterpret_cast<float4 *>(Xrow + 4 * c4) = x;
    }
    for (int64_t c = 4 * n4 + threadIdx.x; c < n; c += kRowThreads)
      Xrow[c] = fmaf(-eta_local, load_g1<GT>(L.G, goff + c), Xrow[c]);
  }
}

__global__ void __launch_bounds__(kRowThreads) local_kernel(Shared sh, const int4 *tiles, float eta_local) {
  const int4 t = tiles[blockIdx.x];
  if (sh.active[t.x]) return;
  const DevLayer &L = sh.layers[t.x];
  if (L.g_dtype == DT_BF16) local_tile<DT_BF16>(L, t.y, t.z, eta_local);
  else local_tile<DT_FP32>(L, t.y, t.z, eta_local);
}

void launch_local(const Shared &sh, const int4 *tiles, int32_t ntiles, float eta_local, cudaStream_t s) {
  if (ntiles > 0) local_kernel<<<ntiles, kRowThreads, 0, s>>>(sh, tiles, eta_local);
}

// ============================================================================ finalize ===
// Equation 1: | ||M_t|| - ||M_{t-1}|| | / (||M_{t-1}|| + eps).  ||M_t|| comes from the update
// kernel's partials on synchronized layers and equals ||B_t|| on local layers (M = B).
__global__ void __launch_bounds__(kGateThreads) finalize_kernel(Shared sh, StepArgs a) {
  if (a.eq1 == nullptr) return;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int l = warp; l < sh.num_layers; l += kGateThreads / 32) {
    const DevLayer &Ly = sh.layers[l];
    double nm;
    if (sh.active[l]) {
      double s = 0.0;
      for (int k = lane; k < Ly.upart_cnt; k += 32) s += sh.upart[Ly.upart_off + k];
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
      nm = sqrt(s);
    } else {
      nm = sh.norm_b[l];
    }
    if (lane == 0) {
      const double before = sh.norm_m_before[l];
      a.eq1[l] = fabs(nm - before) / (before + (double)a.eps_rmmc);
    }
  }
}

void launch_finalize(const Shared &sh, const StepArgs &a, cudaStream_t s) {
  if (a.eq1 != nullptr) finalize_kernel<<<1, kGateThreads, 0, s>>>(sh, a);
}

}  // namespace cd
