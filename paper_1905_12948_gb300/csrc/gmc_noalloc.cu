// gmc_topk_noalloc: the top-k compressor of one vector, for callers that must
// not allocate device memory. Its scratch (radix histogram, selection state,
// per-tile counts and offsets) lives in one file-scope __device__ array of a
// fixed size instead of memory the library or the caller allocates. Every GPU
// that loads the library holds that array until the process exits.
//
// Steps: three radix passes over x find the k-th largest magnitude key T
// (digits of 11, 10 and 10 bits; the last block of each pass turns the
// histogram into the next digit), then per-tile counts, one scan over the
// tiles, and an index-ordered write of the k (index, value) pairs. The
// selection is the library's top-k: the first k elements under (|x| bit
// pattern descending, index ascending).
#include <mutex>

#include "gmc.h"
#include "gmc_internal.h"

namespace gmc {
namespace {

constexpr int64_t kNoallocMaxN = int64_t(1) << 26;  // largest n accepted
constexpr int kNaTile = 4096;                         // elements per tile
constexpr int64_t kNaMaxTiles = kNoallocMaxN / kNaTile;
constexpr int kNaThreads = 256;
constexpr int kNaMaxDevices = 64;

// Scratch layout (uint32 words).
constexpr int64_t kOffHist = 0;                          // kHistBins
constexpr int64_t kOffState = kOffHist + kHistBins;      // 16 words
constexpr int64_t kOffGt = kOffState + 16;               // kNaMaxTiles
constexpr int64_t kOffEq = kOffGt + kNaMaxTiles;         // kNaMaxTiles
constexpr int64_t kOffPos = kOffEq + kNaMaxTiles;        // kNaMaxTiles + 1
constexpr int64_t kOffEqb = kOffPos + kNaMaxTiles + 1;   // kNaMaxTiles
constexpr int64_t kScratchWords = kOffEqb + kNaMaxTiles;
// state words
enum { kSPrefix = 0, kSRank = 1, kST = 2, kSNtie = 3, kSDone = 4 /* 3 words */ };

// The shared scratch: kScratchWords * 4 bytes (about 270 KB) per device.
static __device__ __align__(256) uint32_t g_noalloc_scratch[kScratchWords];

template <int PASS>
__global__ void __launch_bounds__(kNaThreads) k_na_pass(const float* __restrict__ x, int64_t n,
                                                       uint32_t k, uint32_t* scratch) {
  constexpr int nbins = PASS == 0 ? 2048 : 1024;
  constexpr int shift = PASS == 0 ? 20 : (PASS == 1 ? 10 : 0);
  __shared__ uint32_t h[nbins];
  __shared__ uint32_t ws[32];
  __shared__ uint32_t s_last, s_bin, s_rank;
  uint32_t* gh = scratch + kOffHist;
  uint32_t* st = scratch + kOffState;
  const uint32_t prefix = st[kSPrefix];
  for (int b = threadIdx.x; b < nbins; b += blockDim.x) h[b] = 0;
  __syncthreads();
  for (int64_t j = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; j < n;
       j += (int64_t)gridDim.x * blockDim.x) {
    const uint32_t key = mag_key(x[j]);
    if (PASS == 0 || (key >> (shift + 10)) == prefix) atomicAdd(&h[(key >> shift) & (nbins - 1)], 1u);
  }
  __syncthreads();
  for (int b = threadIdx.x; b < nbins; b += blockDim.x)
    if (h[b]) atomicAdd(&gh[b], h[b]);
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) s_last = (atomicAdd(&st[kSDone + PASS], 1u) == gridDim.x - 1) ? 1u : 0u;
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  for (int b = threadIdx.x; b < nbins; b += blockDim.x) {
    h[b] = __ldcg(&gh[b]);
    gh[b] = 0;
  }
  if (threadIdx.x == 0) {
    s_bin = 0;
    s_rank = 0;
  }
  __syncthreads();
  block_find_from_top(h, nbins, PASS == 0 ? k : st[kSRank], ws, &s_bin, &s_rank);
  if (threadIdx.x == 0) {
    if (PASS == 0) st[kSPrefix] = s_bin;
    else if (PASS == 1) st[kSPrefix] = (prefix << 10) | s_bin;
    else st[kST] = (prefix << 10) | s_bin;
    if (PASS < 2) st[kSRank] = s_rank;
    else st[kSNtie] = s_rank;
  }
}

// per tile: elements above T and equal to T
__global__ void __launch_bounds__(kNaThreads) k_na_count(const float* __restrict__ x, int64_t n,
                                                        uint32_t* scratch) {
  __shared__ unsigned long long ws[32];
  const uint32_t T = scratch[kOffState + kST];
  const int64_t j0 = (int64_t)blockIdx.x * kNaTile;
  uint32_t g = 0, q = 0;
  for (int i = threadIdx.x; i < kNaTile; i += blockDim.x) {
    const int64_t j = j0 + i;
    if (j < n) {
      const uint32_t key = mag_key(x[j]);
      g += key > T;
      q += key == T;
    }
  }
  unsigned long long tot;
  block_inclusive_scan<unsigned long long>(((unsigned long long)g << 32) | q, ws, &tot);
  if (threadIdx.x == 0) {
    scratch[kOffGt + blockIdx.x] = (uint32_t)(tot >> 32);
    scratch[kOffEq + blockIdx.x] = (uint32_t)tot;
  }
}

// one block: tile offsets of the output and ties before each tile
__global__ void __launch_bounds__(1024) k_na_scan(int64_t n_tiles, uint32_t k, uint32_t* scratch) {
  __shared__ unsigned long long ws[32];
  const uint32_t n_tie = scratch[kOffState + kSNtie];
  uint32_t carry_g = 0, carry_q = 0;
  for (int64_t t0 = 0; t0 < n_tiles; t0 += blockDim.x) {
    const int64_t tile = t0 + threadIdx.x;
    uint32_t g = 0, q = 0;
    if (tile < n_tiles) {
      g = scratch[kOffGt + tile];
      q = scratch[kOffEq + tile];
    }
    const unsigned long long v = ((unsigned long long)g << 32) | q;
    unsigned long long tot;
    const unsigned long long exc = block_inclusive_scan<unsigned long long>(v, ws, &tot) - v;
    const uint32_t gb = carry_g + (uint32_t)(exc >> 32), qb = carry_q + (uint32_t)exc;
    if (tile < n_tiles) {
      scratch[kOffPos + tile] = gb + min(qb, n_tie);
      scratch[kOffEqb + tile] = qb;
    }
    carry_g += (uint32_t)(tot >> 32);
    carry_q += (uint32_t)tot;
  }
  if (threadIdx.x == 0) scratch[kOffPos + n_tiles] = carry_g + min(carry_q, n_tie);
}

// per tile: write the kept elements in index order
__global__ void __launch_bounds__(kNaThreads) k_na_write(const float* __restrict__ x, int64_t n,
                                                        uint32_t k, const uint32_t* scratch,
                                                        uint32_t* idx_out, float* val_out) {
  constexpr int P = kNaTile / kNaThreads;  // consecutive elements per thread
  __shared__ unsigned long long ws[32];
  const uint32_t T = scratch[kOffState + kST];
  const uint32_t n_tie = scratch[kOffState + kSNtie];
  const uint32_t base = scratch[kOffPos + blockIdx.x];
  const uint32_t eqb = scratch[kOffEqb + blockIdx.x];
  const int64_t j0 = (int64_t)blockIdx.x * kNaTile + (int64_t)threadIdx.x * P;
  uint32_t g = 0, q = 0;
  for (int i = 0; i < P; ++i) {
    const int64_t j = j0 + i;
    if (j < n) {
      const uint32_t key = mag_key(x[j]);
      g += key > T;
      q += key == T;
    }
  }
  const unsigned long long v = ((unsigned long long)g << 32) | q;
  unsigned long long tot;
  const unsigned long long exc = block_inclusive_scan<unsigned long long>(v, ws, &tot) - v;
  const uint32_t taken0 = min(eqb, n_tie);
  uint32_t qg = eqb + (uint32_t)exc;
  uint32_t o = base + (uint32_t)(exc >> 32) + (min(qg, n_tie) - taken0);
  for (int i = 0; i < P; ++i) {
    const int64_t j = j0 + i;
    if (j < n) {
      const float xv = x[j];
      const uint32_t key = mag_key(xv);
      const bool take = key > T || (key == T && qg < n_tie);
      if (key == T) ++qg;
      if (take) {
        if (o < k) {
          idx_out[o] = (uint32_t)j;
          val_out[o] = xv;
        }
        ++o;
      }
    }
  }
}

// Set-up of one device: the scratch array's device address and the SM count,
// valid for the CUDA context they were taken in.
struct DeviceSetup {
  unsigned long long ctx_id = 0;  // 0: not set up
  uint32_t* scratch = nullptr;
  int sms = 1;
};
std::mutex g_setup_mutex;
DeviceSetup g_setup[kNaMaxDevices];

using CtxGetCurrentFn = int (*)(void** ctx);
using CtxGetIdFn = int (*)(void* ctx, unsigned long long* id);

// Id of the current thread's CUDA context on the current device (the
// runtime's primary context, made current if it was not), through the driver
// entry points the runtime exposes. 0 on failure.
unsigned long long current_context_id(int dev) {
  static CtxGetCurrentFn get_current = nullptr;
  static CtxGetIdFn get_id = nullptr;
  if (!get_current || !get_id) {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &f, 12000, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess || !f)
      return 0;
    get_current = reinterpret_cast<CtxGetCurrentFn>(f);
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &f, 12000, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess || !f)
      return 0;
    get_id = reinterpret_cast<CtxGetIdFn>(f);
  }
  void* ctx = nullptr;
  if (get_current(&ctx) != 0) return 0;
  if (!ctx) {  // the runtime has not made its context current on this thread yet
    if (cudaSetDevice(dev) != cudaSuccess || get_current(&ctx) != 0 || !ctx) return 0;
  }
  unsigned long long id = 0;
  return get_id(ctx, &id) == 0 ? id : 0;
}

// The scratch array's device address and the SM count of the current device.
// Host code cannot use the array's name as a device address: the address is
// looked up with cudaGetSymbolAddress once per device, with that device
// current, and again only if the device's context was replaced since (e.g.
// after cudaDeviceReset), so that a stale address is never passed on.
cudaError_t device_setup(DeviceSetup* out) {
  int dev = 0;
  cudaError_t err = cudaGetDevice(&dev);
  if (err != cudaSuccess) return err;
  if (dev < 0 || dev >= kNaMaxDevices) return cudaErrorInvalidDevice;
  const unsigned long long ctx = current_context_id(dev);
  if (ctx == 0) return cudaErrorInitializationError;
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  DeviceSetup& st = g_setup[dev];
  if (st.ctx_id != ctx) {
    void* p = nullptr;
    err = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (err != cudaSuccess) return err;
    int sms = 0;
    err = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (err != cudaSuccess) return err;
    st.scratch = static_cast<uint32_t*>(p);
    st.sms = sms > 0 ? sms : 1;
    st.ctx_id = ctx;
  }
  *out = st;
  return cudaSuccess;
}

// One plain launch; returns that launch's own error (it neither reads nor
// clears an error left by earlier, unrelated work).
template <typename... P, typename... Args>
cudaError_t launch(void (*kernel)(P...), unsigned grid, unsigned block, cudaStream_t s, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(block);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = s;
  cfg.attrs = nullptr;
  cfg.numAttrs = 0;
  return cudaLaunchKernelEx(&cfg, kernel, args...);
}

}  // namespace
}  // namespace gmc

extern "C" int gmc_topk_noalloc(const float* x_dev, int64_t n, int64_t k, uint32_t* idx_dev,
                                float* val_dev, void* stream) {
  using namespace gmc;
  if (!x_dev || !idx_dev || !val_dev || n < 1 || k < 1 || k > n) return GMC_EINVAL;
  if (n > kNoallocMaxN) return GMC_ETOOBIG;
  DeviceSetup dv;
  if (device_setup(&dv) != cudaSuccess) return GMC_ECUDA;
  uint32_t* scratch = dv.scratch;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // the histogram and the pass state must start at zero; the tables are
  // fully rewritten by every call
  if (cudaMemsetAsync(scratch, 0, (size_t)(kOffState + 16) * sizeof(uint32_t), s) != cudaSuccess)
    return GMC_ECUDA;
  const int64_t want = (n + kNaThreads * 16 - 1) / (kNaThreads * 16);
  const unsigned grid = (unsigned)(want < 2 * (int64_t)dv.sms ? want : 2 * (int64_t)dv.sms);
  const int64_t n_tiles = (n + kNaTile - 1) / kNaTile;
  const uint32_t kk = (uint32_t)k;
  cudaError_t err = launch(k_na_pass<0>, grid, kNaThreads, s, x_dev, n, kk, scratch);
  if (err == cudaSuccess) err = launch(k_na_pass<1>, grid, kNaThreads, s, x_dev, n, kk, scratch);
  if (err == cudaSuccess) err = launch(k_na_pass<2>, grid, kNaThreads, s, x_dev, n, kk, scratch);
  if (err == cudaSuccess) err = launch(k_na_count, (unsigned)n_tiles, kNaThreads, s, x_dev, n, scratch);
  if (err == cudaSuccess) err = launch(k_na_scan, 1u, 1024u, s, n_tiles, kk, scratch);
  if (err == cudaSuccess)
    err = launch(k_na_write, (unsigned)n_tiles, kNaThreads, s, x_dev, n, kk,
                 static_cast<const uint32_t*>(scratch), idx_dev, val_dev);
  return err == cudaSuccess ? GMC_OK : GMC_ECUDA;
}
