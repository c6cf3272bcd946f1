// dion_buffer_norms_noalloc: the buffer step of a CurvaDion step (B = M + G written back into
// M) and the two norms the RMMC statistics need, ||B|| and ||M_{t-1}||, for callers that must
// not allocate device memory.
//
// Some callers cannot call cudaMalloc: a training framework whose caching allocator has
// reserved the device memory up front and owns every byte of it, or a latency-critical loop
// where cudaMalloc/cudaFree would synchronize the device.  dion_plan_create allocates a
// workspace, so those callers use this entry point instead.  Its scratch (the layer table and
// the per-tile partial sums) lives in one file-scope __device__ array of fixed size that every
// GPU loading this library holds until the process exits.  The caller passes the inputs
// (M, G) and the outputs (the norms); nothing else is allocated.
#include "../../include/curvadion.h"
#include "common.cuh"

#include <algorithm>
#include <cmath>
#include <cstddef>

namespace {

constexpr int kThreads = 256;
constexpr int64_t kTileElems = 65536;  // a tile is whole rows of about this many elements

struct NaLayer {
  int64_t m, n, ldm, ldg;
  float *M;
  const void *G;
  int32_t g_dtype, rows_per_tile;
  int32_t tile_begin, tile_count;  // this layer's tiles (one partial pair each)
};

struct NoAllocScratch {
  NaLayer layers[DION_NOALLOC_MAX_LAYERS];
  double partials[2 * DION_NOALLOC_MAX_TILES];  // per tile: sum B^2, sum M_{t-1}^2
};

// Shared by every call on a device; contents are whatever the last call left.  Every slot a
// call reads is written by the same call first, so nothing has to be cleared between calls.
static __device__ __align__(256) NoAllocScratch g_scratch;

// The device address of g_scratch, resolved once per device (the symbol's name is only a
// host-side stand-in and must not be passed to a kernel).  Fixed size: no host allocation.
constexpr int kMaxDevices = 64;
NoAllocScratch *g_addr[kMaxDevices] = {};

__device__ __forceinline__ float g_at(const NaLayer &L, int64_t off) {
  if (L.g_dtype == cd::DT_BF16) return __bfloat162float(static_cast<const __nv_bfloat16 *>(L.G)[off]);
  return static_cast<const float *>(L.G)[off];
}

// One block per tile; the tile's layer is found by binary search over the tile ranges.
__global__ void __launch_bounds__(kThreads) na_buffer_kernel(NoAllocScratch *sc, int num_layers) {
  __shared__ double red[kThreads / 32];
  const int tile = blockIdx.x;
  int lo = 0, hi = num_layers - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) / 2;
    if (sc->layers[mid].tile_begin <= tile) lo = mid;
    else hi = mid - 1;
  }
  const NaLayer L = sc->layers[lo];
  const int64_t r0 = (int64_t)(tile - L.tile_begin) * L.rows_per_tile;
  const int64_t r1 = r0 + L.rows_per_tile < L.m ? r0 + L.rows_per_tile : L.m;
  float sb = 0.f, sm = 0.f;
  double db = 0.0, dm = 0.0;
  for (int64_t i = r0; i < r1; ++i) {
    for (int64_t c = threadIdx.x; c < L.n; c += kThreads) {
      const float mo = L.M[i * L.ldm + c];
      const float b = mo + g_at(L, i * L.ldg + c);
      L.M[i * L.ldm + c] = b;
      sb = fmaf(b, b, sb);
      sm = fmaf(mo, mo, sm);
    }
    db += (double)sb;  // fp32 sums of at most a row's share per thread, folded into fp64
    dm += (double)sm;
    sb = sm = 0.f;
  }
  db = cd::block_sum<kThreads>(db, red);
  dm = cd::block_sum<kThreads>(dm, red);
  if (threadIdx.x == 0) {
    sc->partials[2 * tile] = db;
    sc->partials[2 * tile + 1] = dm;
  }
}

// One warp per layer: fixed-order fp64 sums of the layer's tile partials.
__global__ void __launch_bounds__(kThreads) na_reduce_kernel(const NoAllocScratch *sc, int num_layers,
                                                             double *norm_b, double *norm_m) {
  const int lane = threadIdx.x & 31;
  const int l = blockIdx.x * (kThreads / 32) + (threadIdx.x >> 5);
  if (l >= num_layers) return;
  const NaLayer &L = sc->layers[l];
  double b = 0.0, m = 0.0;
  for (int k = lane; k < L.tile_count; k += 32) {
    b += sc->partials[2 * (L.tile_begin + k)];
    m += sc->partials[2 * (L.tile_begin + k) + 1];
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    b += __shfl_xor_sync(0xffffffffu, b, o);
    m += __shfl_xor_sync(0xffffffffu, m, o);
  }
  if (lane == 0) {
    norm_b[l] = sqrt(b);
    norm_m[l] = sqrt(m);
  }
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace

extern "C" dion_status dion_buffer_norms_noalloc(const dion_layer *layers, int32_t num_layers, double *norm_b_out,
                                                 double *norm_m_out, void *stream) {
  if (num_layers < 1 || layers == nullptr || norm_b_out == nullptr || norm_m_out == nullptr)
    return DION_ERR_INVALID_ARG;
  if (num_layers > DION_NOALLOC_MAX_LAYERS) return DION_ERR_UNSUPPORTED;
  NaLayer tab[DION_NOALLOC_MAX_LAYERS];  // on the stack: this entry point allocates nothing
  int64_t tiles = 0;
  for (int32_t l = 0; l < num_layers; ++l) {
    const dion_layer &ly = layers[l];
    if (ly.m < 1 || ly.n < 1 || !ly.M || !ly.G) return DION_ERR_INVALID_ARG;
    if (ly.g_dtype != DION_DTYPE_FP32 && ly.g_dtype != DION_DTYPE_BF16) return DION_ERR_INVALID_ARG;
    if (ly.ldm < ly.n || ly.ldg < ly.n) return DION_ERR_INVALID_ARG;
    const int64_t gsz = ly.g_dtype == DION_DTYPE_BF16 ? 2 : 4;
    if (!aligned16(ly.M) || !aligned16(ly.G) || (ly.ldm * 4) % 16 || (ly.ldg * gsz) % 16) return DION_ERR_ALIGNMENT;
    const int64_t rows = std::max<int64_t>(1, std::min<int64_t>(ly.m, kTileElems / ly.n));
    const int64_t cnt = (ly.m + rows - 1) / rows;
    NaLayer &t = tab[l];
    t.m = ly.m; t.n = ly.n; t.ldm = ly.ldm; t.ldg = ly.ldg;
    t.M = ly.M; t.G = ly.G; t.g_dtype = ly.g_dtype;
    t.rows_per_tile = (int32_t)rows;
    t.tile_begin = (int32_t)std::min<int64_t>(tiles, DION_NOALLOC_MAX_TILES);
    t.tile_count = (int32_t)cnt;
    tiles += cnt;
  }
  if (tiles > DION_NOALLOC_MAX_TILES) return DION_ERR_UNSUPPORTED;

  // Set-up, once per device with that device current: the scratch's device address.
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return DION_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return DION_ERR_UNSUPPORTED;
  if (g_addr[dev] == nullptr) {
    void *ptr = nullptr;
    if (cudaGetSymbolAddress(&ptr, g_scratch) != cudaSuccess || ptr == nullptr) return DION_ERR_CUDA;
    g_addr[dev] = static_cast<NoAllocScratch *>(ptr);
  }
  NoAllocScratch *sc = g_addr[dev];
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // The layer table is copied from this call's host array (stream-ordered; pageable source).
  void *dev_layers = reinterpret_cast<char *>(sc) + offsetof(NoAllocScratch, layers);
  if (cudaMemcpyAsync(dev_layers, tab, sizeof(NaLayer) * num_layers, cudaMemcpyHostToDevice, s) != cudaSuccess)
    return DION_ERR_CUDA;
  na_buffer_kernel<<<(unsigned)tiles, kThreads, 0, s>>>(sc, num_layers);
  na_reduce_kernel<<<(num_layers + kThreads / 32 - 1) / (kThreads / 32), kThreads, 0, s>>>(sc, num_layers,
                                                                                          norm_b_out, norm_m_out);
  return cudaGetLastError() == cudaSuccess ? DION_OK : DION_ERR_CUDA;
}
