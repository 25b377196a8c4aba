// Device-side definitions shared by the GMC kernels: per-worker selection
// state, step counters, the fp32 accumulator operation, magnitude keys, and
// warp / block scan primitives.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

namespace gmc {

constexpr uint32_t kKeyMask = 0x7fffffffu;   // |v| through its bit pattern
constexpr uint32_t kNoCandidate = 0xffffffffu; // threshold above every key
constexpr int kThreads = 256;                // block size of the streaming kernels
constexpr int kWarps = kThreads / 32;
constexpr int kSampleThreads = 1024;
constexpr int kSampleChunks = 4096;          // sampled 8-element chunks per worker
constexpr int kSampleAll = 32768;            // d at or below which every element is sampled
constexpr int kHistBins = 2048;              // first radix digit: key bits 30..20

// Per-worker top-k selection state, rewritten every step.
struct WorkerSel {
  uint32_t theta;    // candidate threshold key from the sample (kNoCandidate = none)
  uint32_t count;    // candidates appended by the accumulate pass (may exceed cap)
  uint32_t prefix;   // radix digits fixed so far
  uint32_t rank;     // 1-based rank still to find inside the current bucket
  uint32_t T;        // the k-th largest key
  uint32_t n_tie;    // elements equal to T that are kept (lowest indices first)
  uint32_t done[3];  // finished-block counters of the three select passes
  uint32_t pad[7];
};

// Step counters (see GMC_STAT_* in gmc.h), unsigned 64-bit slots.
struct Counters {
  unsigned long long v[8];
};
enum CounterSlot { kSteps = 0, kPairs = 1, kNnz = 2, kUnion = 3, kChanged = 4,
                   kFallbacks = 5, kNonfinite = 6 };

// Device status bits (gmc_check).
constexpr unsigned kStatusNonfinite = 1u;
constexpr unsigned kStatusInternal = 2u;

__device__ __forceinline__ uint32_t mag_key(float v) {
  return __float_as_uint(v) & kKeyMask;
}
__device__ __forceinline__ bool is_nonfinite(float v) {
  return (__float_as_uint(v) & 0x7f800000u) == 0x7f800000u;
}
// e_{t+1/2} = (e + g) - (c * dl): three operations, each rounded once (Alg. 1).
__device__ __forceinline__ float accumulate(float e, float g, float c, float dl) {
  return __fsub_rn(__fadd_rn(e, g), __fmul_rn(c, dl));
}
__device__ __forceinline__ bool needs_dense(const WorkerSel& s, uint32_t ksel, uint32_t cap) {
  return s.count < ksel || s.count > cap;
}
__device__ __forceinline__ uint32_t lanemask_lt() {
  uint32_t m;
  asm("mov.u32 %0, %%lanemask_lt;" : "=r"(m));
  return m;
}

// Inclusive scan of one value per thread over the block (blockDim a multiple
// of 32, at most 1024). `ws` needs 32 words of shared memory. Returns the
// inclusive prefix; *total receives the block total.
template <typename V>
__device__ __forceinline__ V block_inclusive_scan(V x, V* ws, V* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int nwarps = blockDim.x >> 5;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    V y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) ws[warp] = x;
  __syncthreads();
  if (warp == 0) {
    V w = lane < nwarps ? ws[lane] : V(0);
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      V y = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += y;
    }
    ws[lane] = w;  // inclusive warp-total prefix
  }
  __syncthreads();
  V add = warp > 0 ? ws[warp - 1] : V(0);
  V tot = ws[nwarps - 1];
  __syncthreads();  // ws may be reused by the caller
  *total = tot;
  return x + add;
}

// Given a histogram hist[nbins] (shared memory) of keys and a 1-based rank r
// counted from the largest key, find the bucket b that holds the r-th largest
// key and the rank of that key inside b. nbins must be a multiple of
// blockDim.x. All threads receive the result.
__device__ __forceinline__ void block_find_from_top(const uint32_t* hist, int nbins, uint32_t r,
                                                    uint32_t* ws, uint32_t* out_bin,
                                                    uint32_t* out_rank) {
  const int per = nbins / blockDim.x;
  // thread t owns buckets [nbins - (t+1)*per, nbins - t*per): thread 0 the top ones
  const int hi = nbins - threadIdx.x * per;
  uint32_t mine = 0;
  for (int i = 1; i <= per; ++i) mine += hist[hi - i];
  uint32_t total;
  uint32_t incl = block_inclusive_scan<uint32_t>(mine, ws, &total);
  uint32_t above = incl - mine;  // keys in buckets above mine
  if (above < r && r <= incl) {
    for (int i = 1; i <= per; ++i) {
      const uint32_t h = hist[hi - i];
      if (r <= above + h) {
        *out_bin = uint32_t(hi - i);
        *out_rank = r - above;
        break;
      }
      above += h;
    }
  }
  __syncthreads();
}

}  // namespace gmc
