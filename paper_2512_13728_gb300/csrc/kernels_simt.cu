// CUDA-core kernels of the CurvaDion step (fp32 operands, fp32 FMA, fp64 partial sums).
//
// These kernels serve the DION_PREC_FP32 mode end to end, and the buffer, gate, Cholesky,
// column-normalization, local-branch and finalize steps of every mode.  Every kernel reads
// its work list (tiles) from device memory and skips layers whose `active` flag says they
// do not take the Dion branch this step, so one fixed launch sequence serves every gate
// decision without a host round trip.
#include "chol_blocks.cuh"
#include "common.cuh"

#include <algorithm>
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
      if (!HAS_BH || !L.b_deferred) *reinterpret_cast<float4 *>(Mrow + 4 * c4) = m;
      if (HAS_BH) {  // bf16 copy of B (operand of the tensor-core contractions)
        const __nv_bfloat162 h01 = __floats2bfloat162_rn(m.x, m.y), h23 = __floats2bfloat162_rn(m.z, m.w);
        uint2 hv;
        hv.x = *reinterpret_cast<const uint32_t *>(&h01);
        hv.y = *reinterpret_cast<const uint32_t *>(&h23);
        *reinterpret_cast<uint2 *>(L.Bh + i * L.ldbh + 4 * c4) = hv;
        if (L.Bl != nullptr) {  // BF16X3: the low half B - bf16(B), rounded to bf16
          const float2 f01 = __bfloat1622float2(h01), f23 = __bfloat1622float2(h23);
          const __nv_bfloat162 l01 = __floats2bfloat162_rn(m.x - f01.x, m.y - f01.y);
          const __nv_bfloat162 l23 = __floats2bfloat162_rn(m.z - f23.x, m.w - f23.y);
          uint2 lv;
          lv.x = *reinterpret_cast<const uint32_t *>(&l01);
          lv.y = *reinterpret_cast<const uint32_t *>(&l23);
          *reinterpret_cast<uint2 *>(L.Bl + i * L.ldbh + 4 * c4) = lv;
        }
      }
    }
    for (int64_t c = 4 * n4 + threadIdx.x; c < n; c += kRowThreads) {
      const float mo = Mrow[c];
      const float b = mo + load_g1<GT>(L.G, goff + c);
      sm[0] = fmaf(mo, mo, sm[0]);
      sb[0] = fmaf(b, b, sb[0]);
      if (!HAS_BH || !L.b_deferred) Mrow[c] = b;
      if (HAS_BH) {
        const __nv_bfloat16 h = __float2bfloat16_rn(b);
        L.Bh[i * L.ldbh + c] = h;
        if (L.Bl != nullptr) L.Bl[i * L.ldbh + c] = __float2bfloat16_rn(b - __bfloat162float(h));
      }
    }
  }
}

// HALVES: also write the layer's bf16 copy of B (or, in BF16X3, its two halves) where the plan
// keeps one; without, only B (into M) and the norms, the halves following for the Dion-branch
// layers alone once the gate has run (split_b_kernel).
template <bool HALVES>
__global__ void __launch_bounds__(kRowThreads) form_b_kernel(Shared sh, const int4 *tiles) {
  __shared__ double red[kRowThreads / 32];
  const int4 t = tiles[blockIdx.x];
  DION_TILE_CHECK(t.x >= 0 && t.x < sh.num_layers, sh.status);
  const DevLayer &L = sh.layers[t.x];
  DION_TILE_CHECK(t.y >= 0 && t.z >= 1 && (int64_t)t.y + t.z <= L.m, sh.status);
  float sb[4] = {0.f, 0.f, 0.f, 0.f}, sm[4] = {0.f, 0.f, 0.f, 0.f};
  if (HALVES && L.Bh != nullptr) {
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

void launch_form_b(const Shared &sh, const int4 *tiles, int32_t ntiles, cudaStream_t s, bool halves) {
  if (ntiles <= 0) return;
  if (halves) form_b_kernel<true><<<ntiles, kRowThreads, 0, s>>>(sh, tiles);
  else form_b_kernel<false><<<ntiles, kRowThreads, 0, s>>>(sh, tiles);
}

// BF16X3, after the gate: the two bf16 halves of B (already in M) for the Dion-branch layers,
// hi = bf16(B), lo = bf16(B - hi), the same roundings as form_b_tile.  Tile = a buffer-pass
// row tile {layer, first row, rows, slot}.  `needed` false: the buffer pass already wrote them
// (DION_GATE_ALWAYS), and every block returns at once.
__global__ void __launch_bounds__(kRowThreads) split_b_kernel(Shared sh, const int4 *tiles, int needed) {
  if (!needed) return;
  const int4 t = tiles[blockIdx.x];
  DION_TILE_CHECK(t.x >= 0 && t.x < sh.num_layers, sh.status);
  if (!sh.active[t.x]) return;
  const DevLayer &L = sh.layers[t.x];
  DION_TILE_CHECK(t.y >= 0 && t.z >= 1 && (int64_t)t.y + t.z <= L.m && L.Bh != nullptr && L.Bl != nullptr, sh.status);
  const int64_t n = L.n, n4 = n >> 2;
  for (int64_t rr = 0; rr < t.z; ++rr) {
    const int64_t i = t.y + rr;
    const float *Brow = L.M + i * L.ldm;
    __nv_bfloat16 *hrow = L.Bh + i * L.ldbh, *lrow = L.Bl + i * L.ldbh;
    for (int64_t c4 = threadIdx.x; c4 < n4; c4 += kRowThreads) {
      const float4 b = *reinterpret_cast<const float4 *>(Brow + 4 * c4);
      const __nv_bfloat162 h01 = __floats2bfloat162_rn(b.x, b.y), h23 = __floats2bfloat162_rn(b.z, b.w);
      const float2 f01 = __bfloat1622float2(h01), f23 = __bfloat1622float2(h23);
      const __nv_bfloat162 l01 = __floats2bfloat162_rn(b.x - f01.x, b.y - f01.y);
      const __nv_bfloat162 l23 = __floats2bfloat162_rn(b.z - f23.x, b.w - f23.y);
      uint2 hv, lv;
      hv.x = *reinterpret_cast<const uint32_t *>(&h01);
      hv.y = *reinterpret_cast<const uint32_t *>(&h23);
      lv.x = *reinterpret_cast<const uint32_t *>(&l01);
      lv.y = *reinterpret_cast<const uint32_t *>(&l23);
      *reinterpret_cast<uint2 *>(hrow + 4 * c4) = hv;
      *reinterpret_cast<uint2 *>(lrow + 4 * c4) = lv;
    }
    for (int64_t c = 4 * n4 + threadIdx.x; c < n; c += kRowThreads) {
      const float b = Brow[c];
      const __nv_bfloat16 h = __float2bfloat16_rn(b);
      hrow[c] = h;
      lrow[c] = __float2bfloat16_rn(b - __bfloat162float(h));
    }
  }
}

void launch_split_b(const Shared &sh, const int4 *tiles, int32_t ntiles, bool needed, cudaStream_t s) {
  if (ntiles > 0) split_b_kernel<<<ntiles, kRowThreads, 0, s>>>(sh, tiles, needed ? 1 : 0);
}

// =============================================================================== gate ===
// Algorithm 2: RMMC_l = | ||B|| - prev_l | / (prev_l + eps); prev_l = ||B||; global max over
// layers; strict compare with tau (a non-finite RMMC counts as above every threshold); the
// gate mode then decides which layers take the Dion branch.

__device__ __forceinline__ bool above(double v, float tau) {
  return !isfinite(v) || v > (double)tau;
}

// Monotone map of a non-negative double (or +inf) to an unsigned key, so that the maximum can
// be taken with an integer atomic: for x >= 0 the IEEE bit pattern already orders correctly.
__device__ __forceinline__ unsigned long long max_key(double x) {
  return (unsigned long long)__double_as_longlong(x) | (1ull << 63);
}
__device__ __forceinline__ double from_max_key(unsigned long long k) {
  return __longlong_as_double((long long)(k & ~(1ull << 63)));
}

// Algorithm 2 for layer l, by one warp: ||B|| and ||M_{t-1}|| from the buffer pass's tile
// partials (fixed-order fp64 sums), RMMC, prev_norm <- ||B||, the per-layer flag.  Returns
// RMMC (in lane 0; +inf when not finite, which counts as above every threshold).
__device__ double gate_layer(const Shared &sh, const StepArgs &a, int l, int lane) {
  const DevLayer &Ly = sh.layers[l];
  double sb = 0.0, sm = 0.0;
  for (int k = lane; k < Ly.bpart_cnt; k += 32) {  // fixed lane/slot assignment
    sb += __ldcg(&sh.bpart[2 * (Ly.bpart_off + k)]);
    sm += __ldcg(&sh.bpart[2 * (Ly.bpart_off + k) + 1]);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    sb += __shfl_xor_sync(0xffffffffu, sb, o);
    sm += __shfl_xor_sync(0xffffffffu, sm, o);
  }
  double rm = 0.0;
  if (lane == 0) {
    const double nb = sqrt(sb);
    const double prev = a.prev_norm[l];
    rm = fabs(nb - prev) / (prev + (double)a.eps_rmmc);
    if (!isfinite(nb)) set_status(sh.status, ST_NONFINITE);
    a.rmmc[l] = rm;
    a.prev_norm[l] = nb;
    a.flags[l] = above(rm, Ly.tau) ? 1 : 0;
    sh.norm_b[l] = nb;
    sh.norm_m_before[l] = sqrt(sm);
  }
  return isfinite(rm) ? rm : INFINITY;
}

// The gate mode's branch mask from the flags (all blocks' flags are written) and the global
// flag; one block, all threads.  Also counts the Dion-branch layers into the scratch.
__device__ void gate_finish(const Shared &sh, const StepArgs &a, int gflag, int *count_s) {
  const int L = sh.num_layers;
  if (threadIdx.x == 0) *count_s = 0;
  __syncthreads();
  int mine = 0;
  for (int i = threadIdx.x; i < L; i += blockDim.x) {
    int act;
    switch (a.gate_mode) {
      case GATE_ALWAYS: act = 1; break;
      case GATE_GLOBAL: act = gflag; break;
      case GATE_PER_LAYER: act = *reinterpret_cast<const volatile uint8_t *>(&a.flags[i]); break;  // other blocks'
      default: act = (a.step % a.period) == 0; break;
    }
    sh.active[i] = (uint8_t)act;
    mine += act;
  }
  atomicAdd(count_s, mine);
  __syncthreads();
  if (threadIdx.x == 0) {
    sh.gate_scratch[kScratchActive] = (unsigned long long)*count_s;
    sh.gate_scratch[kScratchShifted] = 0ull;  // counted by this step's Cholesky kernels
  }
}

// One warp per layer; the running maximum of RMMC goes to an atomic max (order-independent, so
// deterministic).  The last block to finish sets the global flag and the branch mask of every
// layer and resets the scratch.
constexpr int kGateWarps = 8;
__global__ void __launch_bounds__(kGateWarps * 32) gate_kernel(Shared sh, StepArgs a) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int L = sh.num_layers;
  const int l = blockIdx.x * kGateWarps + warp;
  __shared__ int last_s, gflag_s, count_s;
  if (l < L) {
    const double rm = gate_layer(sh, a, l, lane);
    if (lane == 0) atomicMax(&sh.gate_scratch[0], max_key(rm));
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();  // this block's writes are visible before it is counted
    last_s = atomicAdd(&sh.gate_scratch[1], 1ull) == (unsigned long long)(gridDim.x - 1);
  }
  __syncthreads();
  if (!last_s) return;
  if (threadIdx.x == 0) {
    __threadfence();
    const unsigned long long key = atomicAdd(&sh.gate_scratch[0], 0ull);
    const int gf = (L > 0 && above(from_max_key(key), a.tau_global)) ? 1 : 0;
    a.gflag[0] = (uint8_t)gf;
    gflag_s = gf;
    sh.gate_scratch[0] = 0ull;  // for the next step (kernel boundary orders it)
    sh.gate_scratch[1] = 0ull;
  }
  __syncthreads();
  gate_finish(sh, a, gflag_s, &count_s);
}

void launch_gate(const Shared &sh, const StepArgs &a, cudaStream_t s) {
  gate_kernel<<<std::max(1, (sh.num_layers + kGateWarps - 1) / kGateWarps), kGateWarps * 32, 0, s>>>(sh, a);
}

// Data-parallel steps: Algorithm 2's branch from RMMC values the caller has already reduced
// over the workers (AllReduce_max), in a.rmmc.  One block: every layer's flag, the maximum over
// layers (a non-finite value counts as above every threshold) for the global flag, and the
// branch mask of the gate mode.
constexpr int kGateRedThreads = 256;
__global__ void __launch_bounds__(kGateRedThreads) gate_reduced_kernel(Shared sh, StepArgs a) {
  __shared__ double max_s[kGateRedThreads / 32];
  __shared__ int gflag_s, count_s;
  const int L = sh.num_layers, lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  double mx = -1.0;
  for (int l = threadIdx.x; l < L; l += kGateRedThreads) {
    double v = a.rmmc[l];
    if (!isfinite(v)) v = INFINITY;
    a.flags[l] = above(v, sh.layers[l].tau) ? 1 : 0;
    mx = fmax(mx, v);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) mx = fmax(mx, __shfl_xor_sync(0xffffffffu, mx, o));
  if (lane == 0) max_s[warp] = mx;
  __syncthreads();
  if (threadIdx.x == 0) {
    double g = -1.0;
    for (int w = 0; w < kGateRedThreads / 32; ++w) g = fmax(g, max_s[w]);
    gflag_s = (L > 0 && above(g, a.tau_global)) ? 1 : 0;
    a.gflag[0] = (uint8_t)gflag_s;
  }
  __syncthreads();
  gate_finish(sh, a, gflag_s, &count_s);
}

void launch_gate_reduced(const Shared &sh, const StepArgs &a, cudaStream_t s) {
  gate_reduced_kernel<<<1, kGateRedThreads, 0, s>>>(sh, a);
}

// ==================================================================== norms + gate ===
// Gated modes with the fused buffer + B Q kernel: Algorithm 2 needs ||B|| before it knows which
// layers take the Dion branch, so this pass forms B = M + G into M (read M, G; write M:
// 10 B/element) with the sums of B^2 and M_{t-1}^2 per 128-row tile (the fused kernel's slots),
// and the last block to finish runs the gate.  The fused kernel and everything after it touch
// only the layers that sync and read B from M; the local branch then only updates X.
// Tile = {layer, 128-row block}.
constexpr int kNormThreads = 256;
template <int GT>
__device__ void norms_tile(const DevLayer &L, int64_t row0, int64_t nrows, float sb[4], float sm[4]) {
  float *M = L.M;
  const int64_t n = L.n, n4 = n >> 2;
  // four rows at a time: each thread keeps four independent M and G loads in flight
  int64_t rr = 0;
  for (; rr + 4 <= nrows; rr += 4) {
    const int64_t i = row0 + rr;
    for (int64_t c4 = threadIdx.x; c4 < n4; c4 += kNormThreads) {
      float4 m[4];
      float g[4][4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        m[u] = __ldcs(reinterpret_cast<const float4 *>(L.M + (i + u) * L.ldm + 4 * c4));
        load_g4<GT>(L.G, (i + u) * L.ldg + 4 * c4, g[u]);
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const float b0 = m[u].x + g[u][0], b1 = m[u].y + g[u][1], b2 = m[u].z + g[u][2], b3 = m[u].w + g[u][3];
        sm[0] = fmaf(m[u].x, m[u].x, sm[0]); sm[1] = fmaf(m[u].y, m[u].y, sm[1]);
        sm[2] = fmaf(m[u].z, m[u].z, sm[2]); sm[3] = fmaf(m[u].w, m[u].w, sm[3]);
        sb[0] = fmaf(b0, b0, sb[0]); sb[1] = fmaf(b1, b1, sb[1]);
        sb[2] = fmaf(b2, b2, sb[2]); sb[3] = fmaf(b3, b3, sb[3]);
        *reinterpret_cast<float4 *>(M + (i + u) * L.ldm + 4 * c4) = make_float4(b0, b1, b2, b3);
      }
    }
  }
  for (; rr < nrows; ++rr) {
    const int64_t i = row0 + rr;
    for (int64_t c4 = threadIdx.x; c4 < n4; c4 += kNormThreads) {
      const float4 m = __ldcs(reinterpret_cast<const float4 *>(L.M + i * L.ldm + 4 * c4));
      float g[4];
      load_g4<GT>(L.G, i * L.ldg + 4 * c4, g);
      const float b0 = m.x + g[0], b1 = m.y + g[1], b2 = m.z + g[2], b3 = m.w + g[3];
      sm[0] = fmaf(m.x, m.x, sm[0]); sm[1] = fmaf(m.y, m.y, sm[1]);
      sm[2] = fmaf(m.z, m.z, sm[2]); sm[3] = fmaf(m.w, m.w, sm[3]);
      sb[0] = fmaf(b0, b0, sb[0]); sb[1] = fmaf(b1, b1, sb[1]);
      sb[2] = fmaf(b2, b2, sb[2]); sb[3] = fmaf(b3, b3, sb[3]);
      *reinterpret_cast<float4 *>(M + i * L.ldm + 4 * c4) = make_float4(b0, b1, b2, b3);
    }
  }
  // columns past the last multiple of 4
  for (int64_t e = threadIdx.x; e < nrows * (n - 4 * n4); e += kNormThreads) {
    const int64_t i = row0 + e / (n - 4 * n4), c = 4 * n4 + e % (n - 4 * n4);
    const float mo = M[i * L.ldm + c], b = mo + load_g1<GT>(L.G, i * L.ldg + c);
    sm[0] = fmaf(mo, mo, sm[0]);
    sb[0] = fmaf(b, b, sb[0]);
    M[i * L.ldm + c] = b;
  }
}

__global__ void __launch_bounds__(kNormThreads) norms_gate_kernel(Shared sh, StepArgs a, const int4 *tiles) {
  __shared__ double red[kNormThreads / 32];
  __shared__ int last_s, count_s;
  __shared__ double max_s[kNormThreads / 32];
  const int4 t = tiles[blockIdx.x];  // {layer, 128-row block}
  DION_TILE_CHECK(t.x >= 0 && t.x < sh.num_layers, sh.status);
  const DevLayer &L = sh.layers[t.x];
  DION_TILE_CHECK(t.y >= 0 && (int64_t)t.y * 128 < L.m, sh.status);
  const int64_t row0 = (int64_t)t.y * 128, nrows = min((int64_t)128, L.m - row0);
  float sb[4] = {0.f, 0.f, 0.f, 0.f}, sm[4] = {0.f, 0.f, 0.f, 0.f};
  if (L.g_dtype == DT_BF16) norms_tile<DT_BF16>(L, row0, nrows, sb, sm);
  else norms_tile<DT_FP32>(L, row0, nrows, sb, sm);
  const double b = block_sum<kNormThreads>(((double)sb[0] + sb[1]) + ((double)sb[2] + sb[3]), red);
  const double mo = block_sum<kNormThreads>(((double)sm[0] + sm[1]) + ((double)sm[2] + sm[3]), red);
  if (threadIdx.x == 0) {
    const int slot = L.bpart_off + t.y;
    sh.bpart[2 * slot] = b;
    sh.bpart[2 * slot + 1] = mo;
    __threadfence();  // this block's partials are visible before it is counted
    last_s = atomicAdd(&sh.gate_scratch[2], 1ull) == (unsigned long long)(gridDim.x - 1);
  }
  __syncthreads();
  if (!last_s) return;
  __threadfence();
  // the last block: Algorithm 2 for every layer, one warp per layer, and the maximum of RMMC
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  double mx = -1.0;
  for (int l = warp; l < sh.num_layers; l += kNormThreads / 32) mx = fmax(mx, gate_layer(sh, a, l, lane));
  if (lane == 0) max_s[warp] = mx;
  __syncthreads();
  __shared__ int gflag_s;
  if (threadIdx.x == 0) {
    double g = -1.0;
    for (int w = 0; w < kNormThreads / 32; ++w) g = fmax(g, max_s[w]);
    const int gf = (sh.num_layers > 0 && above(g, a.tau_global)) ? 1 : 0;
    a.gflag[0] = (uint8_t)gf;
    gflag_s = gf;
    sh.gate_scratch[2] = 0ull;  // for the next step (kernel boundary orders it)
  }
  __syncthreads();
  gate_finish(sh, a, gflag_s, &count_s);
}

void launch_norms_gate(const Shared &sh, const StepArgs &a, const int4 *tiles, int32_t ntiles, cudaStream_t s) {
  if (ntiles > 0) norms_gate_kernel<<<ntiles, kNormThreads, 0, s>>>(sh, a, tiles);
}

// ==================================================================== grouped GEMM ===
// C = op(A) op(B) over a list of problems (the FP32 mode's contractions) on CUDA cores: 128 x 128
// output tiles, 8-deep k slices through two shared-memory buffers (the next slice's global loads
// are in flight while the current one is multiplied), 8 x 8 outputs per thread as 2 x 2 blocks
// of 4 x 4 that lie 64 rows / columns apart, so each k step reads 16 bytes per operand block per
// thread without bank conflicts.  Global loads are 16 bytes along whichever dimension of an
// operand is contiguous (zero outside the matrix).  Tile = {problem, tile row, tile col}.
constexpr int GBM = kGemmTile, GBN = kGemmTile, GBK = 8, kGemmThreads = 256;

// Elements (row, col .. col + 3) of a row-major matrix (col a multiple of 4, rows 16-byte
// aligned), zero outside it.
__device__ __forceinline__ float4 ld4_rows(const float *base, int64_t row, int64_t col, int64_t rows, int64_t cols,
                                           int64_t ld) {
  if (row >= rows || col >= cols) return make_float4(0.f, 0.f, 0.f, 0.f);
  const float *p = base + row * ld + col;
  if (col + 4 <= cols) return *reinterpret_cast<const float4 *>(p);
  float v[4] = {0.f, 0.f, 0.f, 0.f};
  for (int e = 0; e < 4; ++e)
    if (col + e < cols) v[e] = p[e];
  return make_float4(v[0], v[1], v[2], v[3]);
}

__global__ void __launch_bounds__(kGemmThreads) gemm_kernel(Shared sh, const GemmProblem *probs,
                                                            const int4 *tiles) {
  const int4 t = tiles[blockIdx.x];
  const GemmProblem p = probs[t.x];
  if (p.mode == GEMM_SHIFTED && sh.gate_scratch[kScratchShifted] == 0ull) return;  // no layer shifted
  DION_TILE_CHECK(p.layer >= 0 && p.layer < sh.num_layers && t.y >= 0 && t.z >= 0 &&
                      (int64_t)t.y * GBM < p.Mrows && (int64_t)t.z * GBN < p.Ncols, sh.status);
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
  __shared__ __align__(16) float As[2][GBK][GBM + 4];
  __shared__ __align__(16) float Bs[2][GBK][GBN + 4];
  // this thread's 16-byte share of a k slice of A (128 x 8) and of B (8 x 128): along the
  // contiguous dimension, 4 consecutive elements of one row / column
  const int a_r = p.transA ? (tid >> 5) : (tid >> 1), a_c = p.transA ? (tid & 31) * 4 : (tid & 1) * 4;
  const int b_r = p.transB ? (tid >> 1) : (tid >> 5), b_c = p.transB ? (tid & 1) * 4 : (tid & 31) * 4;
  auto load = [&](int64_t k0, float4 &av, float4 &bv) {
    av = p.transA ? ld4_rows(p.A, k0 + a_r, i0 + a_c, p.K, p.Mrows, p.lda)   // A^T stored K x M
                  : ld4_rows(p.A, i0 + a_r, k0 + a_c, p.Mrows, p.K, p.lda);  // A stored M x K
    bv = p.transB ? ld4_rows(p.B, j0 + b_r, k0 + b_c, p.Ncols, p.K, p.ldb)   // B^T stored N x K
                  : ld4_rows(p.B, k0 + b_r, j0 + b_c, p.K, p.Ncols, p.ldb);  // B stored K x N
  };
  auto store = [&](int buf, const float4 &av, const float4 &bv) {
    if (p.transA) {
      *reinterpret_cast<float4 *>(&As[buf][a_r][a_c]) = av;
    } else {
      As[buf][a_c + 0][a_r] = av.x; As[buf][a_c + 1][a_r] = av.y;
      As[buf][a_c + 2][a_r] = av.z; As[buf][a_c + 3][a_r] = av.w;
    }
    if (p.transB) {
      Bs[buf][b_c + 0][b_r] = bv.x; Bs[buf][b_c + 1][b_r] = bv.y;
      Bs[buf][b_c + 2][b_r] = bv.z; Bs[buf][b_c + 3][b_r] = bv.w;
    } else {
      *reinterpret_cast<float4 *>(&Bs[buf][b_r][b_c]) = bv;
    }
  };
  float acc[8][8] = {};
  float4 av, bv;
  load(0, av, bv);
  store(0, av, bv);
  __syncthreads();
  int cur = 0;
  for (int64_t k0 = 0; k0 < p.K; k0 += GBK) {
    const bool more = k0 + GBK < p.K;
    if (more) load(k0 + GBK, av, bv);  // in flight during this slice's products
#pragma unroll
    for (int kk = 0; kk < GBK; ++kk) {
      const float4 a0 = *reinterpret_cast<const float4 *>(&As[cur][kk][ty * 4]);
      const float4 a1 = *reinterpret_cast<const float4 *>(&As[cur][kk][64 + ty * 4]);
      const float4 b0 = *reinterpret_cast<const float4 *>(&Bs[cur][kk][tx * 4]);
      const float4 b1 = *reinterpret_cast<const float4 *>(&Bs[cur][kk][64 + tx * 4]);
      const float a[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
      const float b[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
#pragma unroll
      for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    if (more) store(cur ^ 1, av, bv);
    __syncthreads();
    cur ^= 1;
  }
  // output rows ty*4 + (0..3) and 64 + ty*4 + (0..3), columns likewise with tx
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int64_t gi = i0 + (i < 4 ? ty * 4 + i : 64 + ty * 4 + (i - 4));
    if (gi >= p.Mrows) continue;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int64_t gj = j0 + h * 64 + tx * 4;
      float *c = p.C + gi * p.ldc + gj;
      if (gj + 4 <= p.Ncols) {
        *reinterpret_cast<float4 *>(c) = make_float4(acc[i][4 * h], acc[i][4 * h + 1], acc[i][4 * h + 2], acc[i][4 * h + 3]);
      } else {
#pragma unroll
        for (int e = 0; e < 4; ++e)
          if (gj + e < p.Ncols) c[e] = acc[i][4 * h + e];
      }
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
//
// One CTA per layer (r <= 512), 16 warps.  S (full, symmetric) is only read; the factor and
// its inverse are built in place in the L^{-1} buffer W by one right-looking sweep over
// 32-wide block columns k (k0 = 32 k).  Before step k, for rows i >= k0:
//   W[i][j], j >= k0 : the Schur complement S - L[:, :k0] L[:, :k0]^T (lower triangle),
//   W[i][j], j <  k0 : U[i][j] = -sum_{K < k} L[i, K] L^{-1}[K, j],
// and rows above k0 hold their final L^{-1}.  Step k:
//   warp 0     factors the 32 x 32 diagonal block in registers (shuffles) and inverts it
//              (D_k = L_kk^{-1}), while warps 1..15 load the rest of block row k's U and the
//              panel rows below the block;
//   warps 1..  finish block row k: L^{-1}[k, :k0] = D_k U[k, :k0], and form the panel
//              L[i, k] = A[i, k] D_k^T of every row below;
//   all        with Y = [L^{-1}[k, :k0 + 32] | L[k0 + 32 :, k]^T] (32 x r, shared memory),
//              apply W[i][j] -= sum_c Y[c][i] Y[c][j] to every row i below the block and every
//              j <= i: for j >= k0 + 32 this is the trailing Cholesky update, for j < k0 + 32
//              the accumulation of U (whose columns k0 .. k0 + 31 start from zero here).
// The update is a rank-32 outer product over a lower trapezoid, 8 x 8 register tiles fed by
// 128-bit shared loads, so the factorization and the inverse (r^3 / 3 multiply-adds in all)
// run at the FMA rate instead of being serialized behind per-column solves.  A retry starts
// again from S with its diagonal shifted.  If the shifted retry also fails, DION_ERR_BREAKDOWN
// is set and L^{-1} = 0 for the layer, so its P, R and Q become 0, M becomes B and X is
// unchanged (no NaN written).
constexpr int kCholThreads = 512;
constexpr int kFoBatch = 8;  // 16-byte groups each thread has in flight in the first-order factor

// Row i and 16-byte column group j4 (4 j4 <= i) of flat group p of a lower triangle whose rows
// 4 b .. 4 b + 3 hold b + 1 groups each, 2 b (b + 1) groups before them (p < 2^24: the fp32
// estimate of b is off by at most one, corrected in integers; 32-bit division).
__device__ __forceinline__ void lower_group(int64_t p, int &i, int &j4) {
  const uint32_t pu = (uint32_t)p;
  uint32_t b = (uint32_t)((sqrtf(2.f * (float)pu + 1.f) - 1.f) * 0.5f);
  while (2u * (b + 1u) * (b + 2u) <= pu) ++b;
  while (b > 0u && 2u * b * (b + 1u) > pu) --b;
  const uint32_t off = pu - 2u * b * (b + 1u), q = off / (b + 1u);
  i = (int)(4u * b + q);
  j4 = (int)(off - q * (b + 1u));
}

// Column c of Y lives at ysw(c): bit 2 flips when bit 5 is set, so the two 16-byte halves of
// an 8-column group swap in every other 32-column stretch.  Eight consecutive groups read by
// one quarter-warp then fall on distinct banks.
__device__ __forceinline__ int ysw(int c) { return c ^ ((c >> 3) & 4); }
__device__ __forceinline__ void load8y(const float *row, int c0, float w[8]) {  // c0 % 8 == 0
  const int s = (c0 >> 3) & 4;
  const float4 a = *reinterpret_cast<const float4 *>(row + c0 + s), b = *reinterpret_cast<const float4 *>(row + c0 + (s ^ 4));
  w[0] = a.x; w[1] = a.y; w[2] = a.z; w[3] = a.w; w[4] = b.x; w[5] = b.y; w[6] = b.z; w[7] = b.w;
}

// W <- L^{-1} with L L^T = S + shift I (lower triangle of S read).  Returns false, uniformly
// over the block, on a pivot that is not positive and finite.  Shared memory: D (CB x CBP),
// DI (CB x CB), rd (CB reciprocal pivots), Y (CB x ldy, ldy >= r rounded up to 8, columns
// >= r zero).
__device__ bool chol_inverse(const float *__restrict__ S, float *__restrict__ W, int r, int64_t ls, float shift,
                             float *D, float *DI, float *rd, float *Y, int ldy, int *bad) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, q = tid - 32;
  for (int k0 = 0; k0 < r; k0 += CB) {
    const int nb = min(CB, r - k0), R0 = k0 + nb, t = r - R0;
    const float *src = (k0 == 0) ? S : W;
    const float dshift = (k0 == 0) ? shift : 0.f;
    float v[CB];
    if (warp == 0) {
      // ---- diagonal block: lane i holds row k0 + i (identity padding below a short block)
      const int64_t row = k0 + lane;
      if (nb == CB) {
        load8(src + row * ls + k0, v);
        load8(src + row * ls + k0 + 8, v + 8);
        load8(src + row * ls + k0 + 16, v + 16);
        load8(src + row * ls + k0 + 24, v + 24);
      } else {
#pragma unroll
        for (int j = 0; j < CB; ++j) v[j] = (lane < nb && j < nb) ? src[row * ls + k0 + j] : 0.f;
      }
#pragma unroll
      for (int j = 0; j < CB; ++j) {
        if (j > lane) v[j] = 0.f;
        if (j == lane) v[j] = (lane < nb) ? v[j] + dshift : 1.f;
      }
      bool ok = true;
      chol32_col<0>(v, rd, lane, ok);
#pragma unroll
      for (int j = 0; j < CB; ++j) D[lane * CBP + j] = v[j];
      __syncwarp();
      // lane c: column c of D_k = L_kk^{-1} by forward substitution on e_c
      trinv32_row<0>(v, D, rd, lane);
#pragma unroll
      for (int i = 0; i < CB; ++i) DI[i * CB + lane] = v[i];
      if (lane == 0) *bad = ok ? 0 : 1;
    } else if (q < k0) {
      // ---- column q of U[k, :k0]
#pragma unroll
      for (int c = 0; c < CB; ++c) v[c] = (c < nb) ? W[(int64_t)(k0 + c) * ls + q] : 0.f;
    } else if (q < k0 + t) {
      // ---- panel row R0 + q - k0 (a full block: nb = 32 whenever rows remain below it)
      const float *p = src + (int64_t)(R0 + q - k0) * ls + k0;
      load8(p, v);
      load8(p + 8, v + 8);
      load8(p + 16, v + 16);
      load8(p + 24, v + 24);
    }
    __syncthreads();
    if (*bad) return false;
    if (warp > 0 && q < k0 + t) {
      // v <- D_k v (lower triangular, in place from the bottom): the finished L^{-1}[k, q]
      // for a U column, the panel entries L[row, k0 ..] = A[row, k0 ..] D_k^T for a panel row
      trmv32<CB - 1>(v, DI);
      if (q < k0) {
#pragma unroll
        for (int c = 0; c < CB; ++c) {
          if (c < nb) W[(int64_t)(k0 + c) * ls + q] = v[c];
          Y[c * ldy + ysw(q)] = v[c];
        }
      } else {
#pragma unroll
        for (int c = 0; c < CB; ++c) Y[c * ldy + ysw(R0 + q - k0)] = v[c];
      }
    }
    // block row k right of k0: D_k on the diagonal block, zeros beyond
    for (int i = warp; i < nb; i += kCholThreads / 32)
      for (int c = lane; c < r - k0; c += 32) W[(int64_t)(k0 + i) * ls + k0 + c] = (c <= i) ? DI[i * CB + c] : 0.f;
    if (t > 0)
      for (int e = tid; e < CB * CB; e += kCholThreads) Y[(e >> 5) * ldy + ysw(k0 + (e & 31))] = DI[e];
    __syncthreads();
    if (t > 0) {
      // ---- rank-32 update of rows R0 .. r - 1, columns 0 .. i, in 8 x 8 tiles
      const int c1 = R0 / 8 + 1, nbt = (t + 7) / 8;
      const int ntiles = nbt * c1 + nbt * (nbt - 1) / 2;
      for (int p = tid; p < ntiles; p += kCholThreads) {
        const int bi = trap_row(p, c1), bj = p - (bi * c1 + bi * (bi - 1) / 2);
        const int i0 = R0 + 8 * bi, j0 = 8 * bj;
        // the tile starts from the current W (one load latency per tile), or from zero for
        // the U columns of block k, which start here
        const bool fresh = (j0 >= k0 && j0 < R0);
        float acc[8][8];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const int row = i0 + u;
          if (fresh || row >= r) {
#pragma unroll
            for (int w = 0; w < 8; ++w) acc[u][w] = 0.f;
          } else {
            load8(src + (int64_t)row * ls + j0, acc[u]);
#pragma unroll
            for (int w = 0; w < 8; ++w)
              if (j0 + w == row) acc[u][w] += dshift;
          }
        }
#pragma unroll 1
        for (int c = 0; c < CB; ++c) {
          float a[8], b[8];
          load8y(Y + c * ldy, i0, a);
          load8y(Y + c * ldy, j0, b);
#pragma unroll
          for (int u = 0; u < 8; ++u)
#pragma unroll
            for (int w = 0; w < 8; ++w) acc[u][w] = fmaf(-a[u], b[w], acc[u][w]);
        }
#pragma unroll
        for (int u = 0; u < 8; ++u)
          if (i0 + u < r) store8(W + (int64_t)(i0 + u) * ls + j0, acc[u]);
      }
    }
    __syncthreads();
  }
  return true;
}

// ||S - I||_2 estimated by 8 power iterations.  S - I is symmetric, so each product reads only
// the 32 x 32 tiles on and below the diagonal (half of S, which stays in L2 across the
// iterations): warp w takes tiles w, w + 16, ... and adds each tile's row sums (a
// reduce-scatter over the lanes) and, off the diagonal, its column sums into its own partial
// vector; the partials are then summed in warp order, so the estimate is deterministic.
// Shared memory: Y (at least 18 rows of ldy floats).  Called by the whole block.
__device__ __noinline__ float power_norm_sym(const float *__restrict__ S, int r, int64_t ls, float *Y, int ldy) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  __shared__ float wn[kCholThreads / 32];
  __shared__ float lam_s;
  float lam = INFINITY;
  float *part = Y;                  // 16 rows of ldy: one partial vector per warp
  float *pv = Y + 16 * ldy, *wv = Y + 17 * ldy;
  for (int i = tid; i < r; i += kCholThreads) pv[i] = 1.f + 0.25f * __sinf(0.7f * (float)i);  // fixed start
  const int nt = (r + 31) / 32, ntiles = nt * (nt + 1) / 2;
  __syncthreads();
  for (int itp = 0; itp < 8; ++itp) {
    float *mine = part + warp * ldy;
    for (int i = lane; i < r; i += 32) mine[i] = 0.f;
    __syncwarp();
    for (int p = warp; p < ntiles; p += kCholThreads / 32) {
      const int bi = trap_row(p, 1), bj = p - bi * (bi + 1) / 2;  // tile row bi >= tile column bj
      const int c = bj * 32 + lane;
      const float vc = (c < r) ? pv[c] : 0.f;
      float a[32], colsum = 0.f;
#pragma unroll
      for (int y = 0; y < 32; ++y) {
        const int row = bi * 32 + y;
        float e = 0.f;
        if (row < r && c < r) e = S[(int64_t)row * ls + c] - (row == c ? 1.f : 0.f);
        a[y] = e * vc;
        if (bi != bj) colsum = fmaf(e, (row < r) ? pv[row] : 0.f, colsum);
      }
      // reduce-scatter: lane y ends with sum over the lanes of a[y] (row y of the tile)
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const bool upper = (lane & o) != 0;
#pragma unroll
        for (int k = 0; k < o; ++k) {
          const float send = upper ? a[k] : a[k + o];
          const float keep = upper ? a[k + o] : a[k];
          a[k] = keep + __shfl_xor_sync(0xffffffffu, send, o);
        }
      }
      if (bi * 32 + lane < r) mine[bi * 32 + lane] += a[0];
      __syncwarp();
      if (bi != bj && c < r) mine[c] += colsum;
      __syncwarp();
    }
    __syncthreads();
    float pn = 0.f;
    for (int i = tid; i < r; i += kCholThreads) {
      float yv = 0.f;
      for (int w = 0; w < kCholThreads / 32; ++w) yv += part[w * ldy + i];
      wv[i] = yv;
      pn = fmaf(yv, yv, pn);
    }
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
    lam = nrm;  // ||E v|| / ||v||: v has unit norm from the second iteration on
    const float inv = (nrm > 0.f && isfinite(nrm)) ? 1.f / nrm : 0.f;
    for (int i = tid; i < r; i += kCholThreads) pv[i] = wv[i] * inv;
    __syncthreads();
    if (itp == 0) lam = INFINITY;  // the first product uses an unnormalized start vector
  }
  return lam;
}

// pass 0 and 1: every active layer; pass 2: only layers marked by a shifted retry.
// Passes 1 and 2 factor the Gram matrix of an already nearly orthonormal X.  With E = S - I,
// when 1.5 times a bound on ||E||_2 is below near_identity, the factor of S = I + E is taken
// to first order, L = I + F with F = strictly-lower(E) + diag(E) / 2 and L^{-1} = I - F; the
// resulting X L^{-T} is then orthonormal up to O(||E||_2^2).  The bound is ||E||_F when that
// is small enough, else a power-iteration estimate of ||E||_2.
__global__ void __launch_bounds__(kCholThreads, 1) chol_inv_kernel(Shared sh, int pass, float near_identity) {
  const int l = blockIdx.x;
  if (pass == 2 && sh.gate_scratch[kScratchShifted] == 0ull) return;  // no layer took the shifted retry
  if (!sh.active[l]) return;
  if (pass == 2 && !sh.orth_shifted[l]) return;
  const DevLayer &Ly = sh.layers[l];
  const int r = (int)Ly.r;
  const int64_t ls = Ly.ldp;  // leading dimension of S and L^{-1} (a multiple of 8)
  const float *S = Ly.S;
  float *Li = Ly.Linv;
  extern __shared__ __align__(16) float smem[];
  float *D = smem;                 // CB x CBP
  float *rd = D + CB * CBP;        // CB
  float *DI = rd + 32;             // CB x CB (16-byte aligned)
  float *Y = DI + CB * CB;         // CB x ldy
  const int ldy = (r + 7) / 8 * 8;
  __shared__ int bad;
  __shared__ double red[kCholThreads / 32];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

  if (pass >= 1) {
    // ||E||_F^2 from the lower triangle (E symmetric), fixed-order reduction.  The 16-byte
    // groups (i, j4) on or below the diagonal (4 j4 <= i) are taken in a flat order (rows 4 b ..
    // 4 b + 3 hold b + 1 groups each), consecutive threads on consecutive groups, kFoBatch
    // groups per thread in flight, every one of them a load (a group's columns past the
    // diagonal are masked)
    const int r4 = (r + 3) / 4, nb4 = r / 4;
    const int64_t lgroups = 2ll * nb4 * (nb4 + 1) + (int64_t)(r % 4) * (nb4 + 1);
    double fs = 0.0;
    for (int64_t g0 = tid; g0 < lgroups; g0 += (int64_t)kCholThreads * kFoBatch) {
      float4 v[kFoBatch];
      int gi[kFoBatch], gj[kFoBatch];
#pragma unroll
      for (int u = 0; u < kFoBatch; ++u) {
        const int64_t g = g0 + (int64_t)u * kCholThreads;
        lower_group(g, gi[u], gj[u]);
        v[u] = make_float4(0.f, 0.f, 0.f, 0.f);
        if (g < lgroups) v[u] = *reinterpret_cast<const float4 *>(S + (int64_t)gi[u] * ls + 4 * gj[u]);
        else gi[u] = -1;  // past the last group: every column masked below
      }
      float a = 0.f;
#pragma unroll
      for (int u = 0; u < kFoBatch; ++u) {
        const int i = gi[u];
        const float ve[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          const int j = 4 * gj[u] + c;
          const float e = (j <= i) ? ve[c] - (i == j ? 1.f : 0.f) : 0.f;
          a = fmaf((j < i ? 2.f : 1.f) * e, e, a);
        }
      }
      fs += (double)a;
    }
    fs = block_sum<kCholThreads>(fs, red);
    __shared__ float lam_s;
    if (tid == 0) lam_s = (float)sqrt(fs);
    __syncthreads();
    float lam = lam_s;
    if (!(isfinite(lam) && 1.5f * lam < near_identity)) {
      lam = power_norm_sym(S, r, ls, Y, ldy);
    }
    if (isfinite(lam) && 1.5f * lam < near_identity) {
      // the groups on or below the diagonal in the same order, 16-byte loads and stores (a group
      // that straddles column r is stored element-wise), then zeros above them, a warp per row
      for (int64_t g0 = tid; g0 < lgroups; g0 += (int64_t)kCholThreads * kFoBatch) {
        float4 v[kFoBatch];
        int gi[kFoBatch], gj[kFoBatch];
#pragma unroll
        for (int u = 0; u < kFoBatch; ++u) {
          const int64_t g = g0 + (int64_t)u * kCholThreads;
          lower_group(g, gi[u], gj[u]);
          v[u] = g < lgroups ? *reinterpret_cast<const float4 *>(S + (int64_t)gi[u] * ls + 4 * gj[u])
                             : make_float4(0.f, 0.f, 0.f, 0.f);
        }
#pragma unroll
        for (int u = 0; u < kFoBatch; ++u) {
          if (g0 + (int64_t)u * kCholThreads >= lgroups) break;
          const int i = gi[u], j4 = gj[u];
          float o[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
#pragma unroll
          for (int c = 0; c < 4; ++c) {
            const int j = 4 * j4 + c;
            o[c] = (j < i) ? -o[c] : (j == i ? 1.f - 0.5f * (o[c] - 1.f) : 0.f);
          }
          float *dst = Li + (int64_t)i * ls + 4 * j4;
          if (4 * j4 + 4 <= r) {
            *reinterpret_cast<float4 *>(dst) = make_float4(o[0], o[1], o[2], o[3]);
          } else {
#pragma unroll
            for (int c = 0; c < 4; ++c)
              if (4 * j4 + c < r) dst[c] = o[c];
          }
        }
      }
      for (int i = warp; i < r; i += kCholThreads / 32) {
        for (int j4 = i / 4 + 1 + lane; j4 < r4; j4 += 32) {
          float *dst = Li + (int64_t)i * ls + 4 * j4;
          if (4 * j4 + 4 <= r) {
            *reinterpret_cast<float4 *>(dst) = make_float4(0.f, 0.f, 0.f, 0.f);
          } else {
            for (int c = 0; 4 * j4 + c < r; ++c) dst[c] = 0.f;
          }
        }
      }
      return;
    }
  }
  // Y: zero the columns past r once (the update's tiles read up to the next multiple of 8)
  for (int e = tid; e < CB * ldy; e += kCholThreads)
    if (ysw(e % ldy) >= r) Y[e] = 0.f;
  __syncthreads();

  bool ok = chol_inverse(S, Li, r, ls, 0.f, D, DI, rd, Y, ldy, &bad);
  bool shifted = false;
  if (!ok) {  // shifted retry from S + s I
    double tr = 0.0;
    for (int i = tid; i < r; i += kCholThreads) tr += (double)S[(int64_t)i * ls + i];
    tr = block_sum<kCholThreads>(tr, red);
    __shared__ double trace_s;
    if (tid == 0) trace_s = tr;
    __syncthreads();
    const double u = 5.9604644775390625e-8;  // 2^-24
    const double shift = 11.0 * ((double)Ly.m * r + (double)r * (r + 1)) * u * trace_s;
    shifted = true;
    ok = (trace_s > 0.0) && isfinite(trace_s) && chol_inverse(S, Li, r, ls, (float)shift, D, DI, rd, Y, ldy, &bad);
  }
  if (tid == 0) {
    if (pass == 0) sh.orth_shifted[l] = shifted ? 1 : 0;
    else if (shifted) sh.orth_shifted[l] = 1;
    if (shifted) atomicAdd(&sh.gate_scratch[kScratchShifted], 1ull);
  }
  if (!ok) {
    if (tid == 0) set_status(sh.status, ST_BREAKDOWN);
    __syncthreads();
    for (int64_t e = tid; e < (int64_t)r * r; e += kCholThreads) Li[(e / r) * ls + e % r] = 0.f;
  }
}

cudaError_t prepare_chol_inv(int32_t max_r, size_t *smem_out) {
  const int ldy = (max_r + 7) / 8 * 8;
  const size_t smem = sizeof(float) * (CB * CBP + 32 + CB * CB + (size_t)CB * std::max(ldy, 8));
  *smem_out = smem;
  return cudaFuncSetAttribute(chol_inv_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
}

void launch_chol_inv(const Shared &sh, size_t smem, int32_t pass, float near_identity, cudaStream_t s) {
  if (sh.num_layers > 0) chol_inv_kernel<<<sh.num_layers, kCholThreads, smem, s>>>(sh, pass, near_identity);
}

// ===================================================================== ColumnNormalize ===
// Q_t[:, j] = R[:, j] / (||R[:, j]||_2 + eps_col).  Tile = {layer, 32-column group}.  A thread
// owns 4 adjacent columns of every 32nd row (8 threads span the group's 128 bytes of a row, so a
// warp reads 4 full row segments per instruction) and keeps 4 rows' 16-byte loads in flight;
// fp32 sums of 16 rows folded into fp64, the 32 row-group partials added in a fixed order.
constexpr int kColThreads = 256, kColRowGroups = kColThreads / 8, kColUnroll = 4;

__global__ void __launch_bounds__(kColThreads) colnorm_kernel(Shared sh, const int4 *tiles, float eps_col) {
  const int4 t = tiles[blockIdx.x];
  DION_TILE_CHECK(t.x >= 0 && t.x < sh.num_layers && t.y >= 0 && (int64_t)t.y * 32 < sh.layers[t.x].r, sh.status);
  if (!sh.active[t.x]) return;
  const DevLayer &L = sh.layers[t.x];
  const int quad = threadIdx.x & 7, rg = threadIdx.x >> 3;
  const int64_t n = L.n, r = L.r, ldp = L.ldp, ldq = L.ldq;
  const int64_t j = (int64_t)t.y * 32 + 4 * quad;  // first of this thread's columns
  const int nc = r - j >= 4 ? 4 : r - j > 0 ? (int)(r - j) : 0;  // columns of this thread in range
  // rows of R (ldp a multiple of 8, the workspace 256-byte aligned) and of Q (the plan checks
  // the caller's base and ldq against the 16-byte rule) start on 16-byte boundaries
  const float *R = L.R + j;
  auto load = [&](int64_t i) -> float4 {
    if (i >= n || nc == 0) return make_float4(0.f, 0.f, 0.f, 0.f);
    if (nc == 4) return *reinterpret_cast<const float4 *>(R + i * ldp);
    const float *p = R + i * ldp;
    return make_float4(p[0], nc > 1 ? p[1] : 0.f, nc > 2 ? p[2] : 0.f, 0.f);
  };
  __shared__ double part[kColRowGroups][33];
  __shared__ float inv[32];
  double a0 = 0.0, a1 = 0.0, a2 = 0.0, a3 = 0.0;
  float f0 = 0.f, f1 = 0.f, f2 = 0.f, f3 = 0.f;
  int cnt = 0;
  for (int64_t i = rg; i < n; i += kColRowGroups * kColUnroll) {
    float4 v[kColUnroll];
#pragma unroll
    for (int u = 0; u < kColUnroll; ++u) v[u] = load(i + (int64_t)u * kColRowGroups);
#pragma unroll
    for (int u = 0; u < kColUnroll; ++u) {
      f0 = fmaf(v[u].x, v[u].x, f0);
      f1 = fmaf(v[u].y, v[u].y, f1);
      f2 = fmaf(v[u].z, v[u].z, f2);
      f3 = fmaf(v[u].w, v[u].w, f3);
    }
    if (++cnt == 16 / kColUnroll) {
      a0 += f0; a1 += f1; a2 += f2; a3 += f3;
      f0 = f1 = f2 = f3 = 0.f;
      cnt = 0;
    }
  }
  part[rg][4 * quad + 0] = a0 + f0;
  part[rg][4 * quad + 1] = a1 + f1;
  part[rg][4 * quad + 2] = a2 + f2;
  part[rg][4 * quad + 3] = a3 + f3;
  __syncthreads();
  if (threadIdx.x < 32) {
    double s = 0.0;
    for (int g = 0; g < kColRowGroups; ++g) s += part[g][threadIdx.x];
    inv[threadIdx.x] = (float)(1.0 / (sqrt(s) + (double)eps_col));
  }
  __syncthreads();
  if (nc == 0) return;
  const float c0 = inv[4 * quad], c1 = inv[4 * quad + 1], c2 = inv[4 * quad + 2], c3 = inv[4 * quad + 3];
  float *Q = L.Q + j;
  for (int64_t i = rg; i < n; i += kColRowGroups * kColUnroll) {
    float4 v[kColUnroll];
#pragma unroll
    for (int u = 0; u < kColUnroll; ++u) v[u] = load(i + (int64_t)u * kColRowGroups);
#pragma unroll
    for (int u = 0; u < kColUnroll; ++u) {
      const int64_t ii = i + (int64_t)u * kColRowGroups;
      if (ii >= n) break;
      const float4 q = make_float4(v[u].x * c0, v[u].y * c1, v[u].z * c2, v[u].w * c3);
      float *dst = Q + ii * ldq;
      if (nc == 4) {
        *reinterpret_cast<float4 *>(dst) = q;
      } else {
        dst[0] = q.x;
        if (nc > 1) dst[1] = q.y;
        if (nc > 2) dst[2] = q.z;
        if (nc > 3) dst[3] = q.w;
      }
    }
  }
}

void launch_colnorm(const Shared &sh, const int4 *tiles, int32_t ntiles, float eps_col, cudaStream_t s) {
  if (ntiles > 0) colnorm_kernel<<<ntiles, kColThreads, 0, s>>>(sh, tiles, eps_col);
}

// =============================================================== error feedback + update ===
// M = B - (1 - mu) P R^T and X = X - eta sqrt(m/n) P Q_t^T in one pass over the tile, plus the
// fp64 partial of ||M_t||^2 for Equation 1.  128 x 64 tiles, 8-deep k slices through two
// shared-memory buffers (the next slice's 16-byte loads in flight during this one's products),
// 8 x 4 outputs of each product per thread (rows 64 apart, so the 16-byte shared reads are
// conflict-free); the epilogue reads and writes M and X 16 bytes at a time.
// Tile = {layer, tile row, tile col, slot}.
constexpr int UBM = kUpdTileM, UBN = kUpdTileN, UBK = 8, kUpdThreads = 256;

__global__ void __launch_bounds__(kUpdThreads, 2) update_kernel(Shared sh, const int4 *tiles, float mu, float eta,
                                                             float keep) {
  // P, R: ld ldp; Q: ld ldq; k slices stored transposed (K-th row = one k of every tile row)
  __shared__ __align__(16) float As[2][UBK][UBM + 4];
  __shared__ __align__(16) float Rs[2][UBK][UBN + 4];
  __shared__ __align__(16) float Qs[2][UBK][UBN + 4];
  __shared__ double red[kUpdThreads / 32];
  const int4 t = tiles[blockIdx.x];
  DION_TILE_CHECK(t.x >= 0 && t.x < sh.num_layers && t.y >= 0 && t.z >= 0 &&
                      (int64_t)t.y * UBM < sh.layers[t.x].m && (int64_t)t.z * UBN < sh.layers[t.x].n, sh.status);
  if (!sh.active[t.x]) return;
  const DevLayer &L = sh.layers[t.x];
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  const int64_t i0 = (int64_t)t.y * UBM, j0 = (int64_t)t.z * UBN, r = L.r, ldp = L.ldp;
  // this thread's share of a k slice: 4 consecutive k of one row of P, and of one row of R
  // (threads 0..127) or of Q_t (threads 128..255)
  const int pr = tid >> 1, kq = (tid & 1) * 4, br = (tid & 127) >> 1;
  const bool is_q = tid >= 128;
  auto load = [&](int64_t k0, float4 &pv, float4 &bv) {
    pv = ld4_rows(L.P, i0 + pr, k0 + kq, L.m, r, ldp);
    bv = is_q ? ld4_rows(L.Q, j0 + br, k0 + kq, L.n, r, L.ldq) : ld4_rows(L.R, j0 + br, k0 + kq, L.n, r, ldp);
  };
  auto store = [&](int buf, const float4 &pv, const float4 &bv) {
    As[buf][kq + 0][pr] = pv.x; As[buf][kq + 1][pr] = pv.y;
    As[buf][kq + 2][pr] = pv.z; As[buf][kq + 3][pr] = pv.w;
    float(*Bd)[UBN + 4] = is_q ? Qs[buf] : Rs[buf];
    Bd[kq + 0][br] = bv.x; Bd[kq + 1][br] = bv.y;
    Bd[kq + 2][br] = bv.z; Bd[kq + 3][br] = bv.w;
  };
  float u1[8][4] = {}, u2[8][4] = {};
  float4 pv, bv;
  load(0, pv, bv);
  store(0, pv, bv);
  __syncthreads();
  int cur = 0;
  for (int64_t k0 = 0; k0 < r; k0 += UBK) {
    const bool more = k0 + UBK < r;
    if (more) load(k0 + UBK, pv, bv);
#pragma unroll
    for (int kk = 0; kk < UBK; ++kk) {
      const float4 a0 = *reinterpret_cast<const float4 *>(&As[cur][kk][ty * 4]);
      const float4 a1 = *reinterpret_cast<const float4 *>(&As[cur][kk][64 + ty * 4]);
      const float4 b4 = *reinterpret_cast<const float4 *>(&Rs[cur][kk][tx * 4]);
      const float4 q4 = *reinterpret_cast<const float4 *>(&Qs[cur][kk][tx * 4]);
      const float a[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
      const float b[4] = {b4.x, b4.y, b4.z, b4.w}, q[4] = {q4.x, q4.y, q4.z, q4.w};
#pragma unroll
      for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          u1[i][j] = fmaf(a[i], b[j], u1[i][j]);
          u2[i][j] = fmaf(a[i], q[j], u2[i][j]);
        }
    }
    if (more) store(cur ^ 1, pv, bv);
    __syncthreads();
    cur ^= 1;
  }
  const float dec = 1.f - mu, c = eta * L.sqrt_m_over_n;
  float ss = 0.f;
  const int64_t gj = j0 + tx * 4;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int64_t gi = i0 + (i < 4 ? ty * 4 + i : 64 + ty * 4 + (i - 4));
    if (gi >= L.m || gj >= L.n) continue;
    float *mp = L.M + gi * L.ldm + gj, *xp = L.X + gi * L.ldx + gj;
    if (gj + 4 <= L.n) {
      float4 mv = *reinterpret_cast<float4 *>(mp), xv = *reinterpret_cast<float4 *>(xp);
      mv.x = fmaf(-dec, u1[i][0], mv.x); mv.y = fmaf(-dec, u1[i][1], mv.y);
      mv.z = fmaf(-dec, u1[i][2], mv.z); mv.w = fmaf(-dec, u1[i][3], mv.w);
      xv.x = fmaf(-c, u2[i][0], xv.x * keep); xv.y = fmaf(-c, u2[i][1], xv.y * keep);
      xv.z = fmaf(-c, u2[i][2], xv.z * keep); xv.w = fmaf(-c, u2[i][3], xv.w * keep);
      *reinterpret_cast<float4 *>(mp) = mv;
      *reinterpret_cast<float4 *>(xp) = xv;
      ss = fmaf(mv.x, mv.x, ss); ss = fmaf(mv.y, mv.y, ss);
      ss = fmaf(mv.z, mv.z, ss); ss = fmaf(mv.w, mv.w, ss);
    } else {
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        if (gj + j >= L.n) continue;
        const float mn = fmaf(-dec, u1[i][j], mp[j]);
        mp[j] = mn;
        xp[j] = fmaf(-c, u2[i][j], xp[j] * keep);
        ss = fmaf(mn, mn, ss);
      }
    }
  }
  const double tot = block_sum<kUpdThreads>((double)ss, red);
  if (tid == 0) sh.upart[t.w] = tot;
}

void launch_update(const Shared &sh, const int4 *tiles, int32_t ntiles, float mu, float eta, float keep,
                   cudaStream_t s) {
  if (ntiles > 0) update_kernel<<<ntiles, kUpdThreads, 0, s>>>(sh, tiles, mu, eta, keep);
}

// ======================================================================== local branch ===
// Algorithm 2's else-branch: X = X - eta_local G (after decoupled weight decay: X scaled by
// keep = 1 - eta_local * weight_decay), and M = B = M + G (already in place unless the layer
// defers B to the update).
template <int GT>
__device__ void local_tile(const DevLayer &L, int64_t row0, int64_t nrows, float eta_local, float keep, bool b_in_m) {
  const int64_t n = L.n, n4 = n >> 2;
  const bool form_m = L.b_deferred != 0 && !b_in_m;
  for (int64_t rr = 0; rr < nrows; ++rr) {
    const int64_t i = row0 + rr;
    float *Xrow = L.X + i * L.ldx, *Mrow = L.M + i * L.ldm;
    const int64_t goff = i * L.ldg;
    for (int64_t c4 = threadIdx.x; c4 < n4; c4 += kRowThreads) {
      float4 x = *reinterpret_cast<float4 *>(Xrow + 4 * c4);
      float g[4];
      load_g4<GT>(L.G, goff + 4 * c4, g);
      x.x = fmaf(-eta_local, g[0], x.x * keep); x.y = fmaf(-eta_local, g[1], x.y * keep);
      x.z = fmaf(-eta_local, g[2], x.z * keep); x.w = fmaf(-eta_local, g[3], x.w * keep);
      *reinterpret_cast<float4 *>(Xrow + 4 * c4) = x;
      if (form_m) {
        float4 m = *reinterpret_cast<float4 *>(Mrow + 4 * c4);
        m.x += g[0]; m.y += g[1]; m.z += g[2]; m.w += g[3];
        *reinterpret_cast<float4 *>(Mrow + 4 * c4) = m;
      }
    }
    for (int64_t c = 4 * n4 + threadIdx.x; c < n; c += kRowThreads) {
      const float g = load_g1<GT>(L.G, goff + c);
      Xrow[c] = fmaf(-eta_local, g, Xrow[c] * keep);
      if (form_m) Mrow[c] += g;
    }
  }
}

__global__ void __launch_bounds__(kRowThreads) local_kernel(Shared sh, const int4 *tiles, float eta_local, float keep) {
  const int4 t = tiles[blockIdx.x];
  DION_TILE_CHECK(t.x >= 0 && t.x < sh.num_layers && t.y >= 0 && t.z >= 1 &&
                      (int64_t)t.y + t.z <= sh.layers[t.x].m, sh.status);
  if (sh.active[t.x]) return;
  const DevLayer &L = sh.layers[t.x];
  if (L.g_dtype == DT_BF16) local_tile<DT_BF16>(L, t.y, t.z, eta_local, keep, sh.b_in_m != 0);
  else local_tile<DT_FP32>(L, t.y, t.z, eta_local, keep, sh.b_in_m != 0);
}

void launch_local(const Shared &sh, const int4 *tiles, int32_t ntiles, float eta_local, float keep, cudaStream_t s) {
  if (ntiles > 0) local_kernel<<<ntiles, kRowThreads, 0, s>>>(sh, tiles, eta_local, keep);
}

// ============================================================================ finalize ===
// Equation 1: | ||M_t|| - ||M_{t-1}|| | / (||M_{t-1}|| + eps).  ||M_t|| comes from the update
// kernel's partials on synchronized layers and equals ||B_t|| on local layers (M = B).
// One warp per layer: Equation 1 from the update's tile partials of ||M_t||^2.
__global__ void __launch_bounds__(kGateWarps * 32) finalize_kernel(Shared sh, StepArgs a) {
  if (a.eq1 == nullptr) return;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int l = blockIdx.x * kGateWarps + warp; l < sh.num_layers; l += gridDim.x * kGateWarps) {
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
  if (a.eq1 != nullptr)
    finalize_kernel<<<std::max(1, (sh.num_layers + kGateWarps - 1) / kGateWarps), kGateWarps * 32, 0, s>>>(sh, a);
}

}  // namespace cd
