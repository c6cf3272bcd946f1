// dion_buffer_norms_noalloc: the buffer step of a CurvaDion step (B = M + G written back into
// M) and the two norms the RMMC statistics need, ||B|| and ||M_{t-1}||, for callers that must
// not allocate device memory.
//
// Some callers cannot call cudaMalloc: a training framework whose caching allocator has
// reserved the device memory up front and owns every byte of it, or a latency-critical loop
// where cudaMalloc/cudaFree would synchronize the device.  dion_plan_create allocates a
// workspace, so those callers use this entry point instead.  Its only scratch, the per-tile
// partial sums, lives in one file-scope __device__ array of fixed size that every GPU loading
// this library holds until the process exits.  The layer table travels as a kernel parameter.
// The caller passes the inputs (M, G) and the outputs (the norms); nothing else is allocated.
#include "../../include/curvadion.h"
#include "common.cuh"

#include <cuda.h>

#include <algorithm>
#include <cmath>
#include <cstddef>
#include <mutex>

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

// The layer table as a kernel parameter (16 KB, under the 32 KB parameter limit): nothing is
// copied from host memory, so a call never waits for the host or for a pageable copy.
struct NaTable {
  NaLayer layers[DION_NOALLOC_MAX_LAYERS];
};
static_assert(sizeof(NaTable) <= 24 * 1024, "the table must fit the kernel parameter space");

struct NoAllocScratch {
  double partials[2 * DION_NOALLOC_MAX_TILES];  // per tile: sum B^2, sum M_{t-1}^2
};

// Shared by every call on a device; contents are whatever the last call left.  Every slot a
// call reads is written by the same call first, so nothing has to be cleared between calls.
static __device__ __align__(256) NoAllocScratch g_scratch;

// The device address of g_scratch, resolved at set-up once per device and CUDA context (the
// symbol's name is only a host-side stand-in and must not be passed to a kernel).  A device
// reset creates a new context in which the module, and so the array, may sit elsewhere: the
// context's id is kept with the address and a new id triggers a new lookup.  Fixed-size
// tables guarded by a mutex: no host allocation, safe for concurrent host threads.
constexpr int kMaxDevices = 64;
struct AddrEntry {
  unsigned long long ctx_id = 0;
  bool valid = false;
  NoAllocScratch *ptr = nullptr;
};
AddrEntry g_addr[kMaxDevices];
std::mutex g_addr_mu;

using CtxGetCurrentFn = CUresult (*)(CUcontext *);
using CtxGetIdFn = CUresult (*)(CUcontext, unsigned long long *);

// Id of the calling thread's current context, or false when the driver entry points are
// unavailable or no context is current yet.
bool current_ctx_id(unsigned long long *id) {
  static CtxGetCurrentFn get_current = nullptr;
  static CtxGetIdFn get_id = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q{};
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_current = reinterpret_cast<CtxGetCurrentFn>(p);
    p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_id = reinterpret_cast<CtxGetIdFn>(p);
  });
  if (!get_current || !get_id) return false;
  CUcontext ctx = nullptr;
  if (get_current(&ctx) != CUDA_SUCCESS || ctx == nullptr) return false;
  return get_id(ctx, id) == CUDA_SUCCESS;
}

// The scratch's device address on the current device `dev` (set-up on the first call in each
// context: cudaGetSymbolAddress with that device current, return code checked).
cudaError_t scratch_address(int dev, NoAllocScratch **out) {
  std::lock_guard<std::mutex> lock(g_addr_mu);
  AddrEntry &e = g_addr[dev];
  unsigned long long id = 0;
  const bool have_id = current_ctx_id(&id);
  if (e.valid && have_id && id == e.ctx_id) {
    *out = e.ptr;
    return cudaSuccess;
  }
  void *ptr = nullptr;
  const cudaError_t err = cudaGetSymbolAddress(&ptr, g_scratch);  // also makes the context current
  if (err != cudaSuccess) return err;
  if (ptr == nullptr) return cudaErrorInvalidSymbol;
  unsigned long long id2 = 0;
  e.valid = current_ctx_id(&id2);  // without an id the lookup is repeated on every call
  e.ctx_id = id2;
  e.ptr = static_cast<NoAllocScratch *>(ptr);
  *out = e.ptr;
  return cudaSuccess;
}

__device__ __forceinline__ float g_at(const NaLayer &L, int64_t off) {
  if (L.g_dtype == cd::DT_BF16) return __bfloat162float(static_cast<const __nv_bfloat16 *>(L.G)[off]);
  return static_cast<const float *>(L.G)[off];
}

// One block per tile; the tile's layer is found by binary search over the tile ranges.
__global__ void __launch_bounds__(kThreads) na_buffer_kernel(const __grid_constant__ NaTable tab, int num_layers,
                                                             double *partials) {
  __shared__ double red[kThreads / 32];
  const int tile = blockIdx.x;
  int lo = 0, hi = num_layers - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) / 2;
    if (tab.layers[mid].tile_begin <= tile) lo = mid;
    else hi = mid - 1;
  }
  const NaLayer L = tab.layers[lo];
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
    partials[2 * tile] = db;
    partials[2 * tile + 1] = dm;
  }
}

// One warp per layer: fixed-order fp64 sums of the layer's tile partials (lane k takes tiles
// k, k + 32, ...; then a fixed shuffle tree).
__global__ void __launch_bounds__(kThreads) na_reduce_kernel(const __grid_constant__ NaTable tab, int num_layers,
                                                             const double *partials, double *norm_b, double *norm_m) {
  const int lane = threadIdx.x & 31;
  const int l = blockIdx.x * (kThreads / 32) + (threadIdx.x >> 5);
  if (l >= num_layers) return;
  const NaLayer &L = tab.layers[l];
  double b = 0.0, m = 0.0;
  for (int k = lane; k < L.tile_count; k += 32) {
    b += partials[2 * (L.tile_begin + k)];
    m += partials[2 * (L.tile_begin + k) + 1];
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
  NaTable tab;  // on the stack, then passed by value to the kernels: this entry point allocates nothing
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
    NaLayer &t = tab.layers[l];
    t.m = ly.m; t.n = ly.n; t.ldm = ly.ldm; t.ldg = ly.ldg;
    t.M = ly.M; t.G = ly.G; t.g_dtype = ly.g_dtype;
    t.rows_per_tile = (int32_t)rows;
    t.tile_begin = (int32_t)std::min<int64_t>(tiles, DION_NOALLOC_MAX_TILES);
    t.tile_count = (int32_t)std::min<int64_t>(cnt, DION_NOALLOC_MAX_TILES);
    tiles += cnt;
    if (tiles > DION_NOALLOC_MAX_TILES) return DION_ERR_UNSUPPORTED;  // before any device work
  }

  // Set-up, once per device (and context) with that device current: the scratch's device address.
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return DION_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return DION_ERR_UNSUPPORTED;
  NoAllocScratch *sc = nullptr;
  if (scratch_address(dev, &sc) != cudaSuccess) return DION_ERR_CUDA;
  double *partials = sc->partials;  // address arithmetic only: sc is a device address

  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaLaunchConfig_t cfg{};
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = s;
  // each launch's own status, so an earlier unrelated error is neither reported nor cleared here
  cfg.gridDim = dim3((unsigned)tiles);
  if (cudaLaunchKernelEx(&cfg, na_buffer_kernel, tab, (int)num_layers, partials) != cudaSuccess) return DION_ERR_CUDA;
  cfg.gridDim = dim3((unsigned)((num_layers + kThreads / 32 - 1) / (kThreads / 32)));
  if (cudaLaunchKernelEx(&cfg, na_reduce_kernel, tab, (int)num_layers, (const double *)partials, norm_b_out,
                         norm_m_out) != cudaSuccess)
    return DION_ERR_CUDA;
  return DION_OK;
}
