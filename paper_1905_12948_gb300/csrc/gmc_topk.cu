// Top-k path of one GMC step (Alg. 1 with the top-s compressor of Sec. 4).
//
//   sample      per worker, e_{t+1/2} at a stratified sample of 32,768
//               coordinates -> a candidate threshold key theta below the k-th
//               largest |v| with overwhelming probability (one thread-block
//               cluster per worker)
//   accumulate  ONE dense pass: v = (e + g) - c*(w_t - w_{t-1}) written over e;
//               every v with key >= theta is appended to its worker's part of
//               the candidate buffer (a tile's candidates in sub-chunks, in
//               index order) and counted into a histogram relative to theta;
//               the bulk version also applies the previous step's aggregation
//   select      the bin of that histogram holding the k-th key, its candidates
//               ranked in shared memory: the k-th largest key T and the ties at
//               T that are kept (the lowest indices: the largest kept, t_idx)
//   dense       for a worker whose filter missed (too few or too many
//               candidates): exact radix select over dense v, sub-chunks rewritten
//   aggregate   a candidate is sent iff selected(key, j, T, t_idx): e = +0 where
//               sent, the sent values summed in ascending worker order from +0,
//               w -= (eta/K) * sum on the union, w_{t+1} - w_t kept -- in the
//               next step's bulk pass, or at once (k_mark, k_owner_sum)
//
// Keys are the fp32 bit patterns with the sign cleared (monotone in |v|); the
// selected set is the first k elements under (key descending, index ascending).
#include <algorithm>

#include <cooperative_groups.h>

#include "gmc_internal.h"

namespace gmc {
namespace {

constexpr int kMaxK = 32;  // workers supported by the top-k kernels (one lane or mask bit each)

__device__ __forceinline__ float4 load_g4(const float* __restrict__ g, int64_t j, int64_t d,
                                          int mode) {
  if (j + 3 < d) {
    if (mode == 4) return __ldcs(reinterpret_cast<const float4*>(g + j));
    if (mode == 2) {
      const float2 a = __ldcs(reinterpret_cast<const float2*>(g + j));
      const float2 b = __ldcs(reinterpret_cast<const float2*>(g + j + 2));
      return make_float4(a.x, a.y, b.x, b.y);
    }
    return make_float4(__ldcs(g + j), __ldcs(g + j + 1), __ldcs(g + j + 2), __ldcs(g + j + 3));
  }
  float4 r = make_float4(0.f, 0.f, 0.f, 0.f);
  if (j < d) r.x = g[j];
  if (j + 1 < d) r.y = g[j + 1];
  if (j + 2 < d) r.z = g[j + 2];
  return r;
}

// The local momentum of worker k at sampled coordinate j, formed from g
// (m_{t+1} = beta*m_t + eta*g, Sec. 2.3 eq. (3)) without storing it.
__device__ __forceinline__ float local_m(const TopkArgs& A, int k, int64_t j, float g) {
  return __fadd_rn(__fmul_rn(A.beta, A.lm[(int64_t)k * A.ld + j]), __fmul_rn(A.gs, g));
}
// The local-momentum baseline: m = beta*m + eta*g over 4 coordinates (m
// loaded from p beforehand, p 16-byte aligned inside ld), stored back at p;
// returns it for the accumulator in place of g.
__device__ __forceinline__ float4 local_m4(const TopkArgs& A, float* p, float4 m, float4 g) {
  float4 r;
  r.x = __fadd_rn(__fmul_rn(A.beta, m.x), __fmul_rn(A.gs, g.x));
  r.y = __fadd_rn(__fmul_rn(A.beta, m.y), __fmul_rn(A.gs, g.y));
  r.z = __fadd_rn(__fmul_rn(A.beta, m.z), __fmul_rn(A.gs, g.z));
  r.w = __fadd_rn(__fmul_rn(A.beta, m.w), __fmul_rn(A.gs, g.w));
  __stcs(reinterpret_cast<float4*>(p), r);
  return r;
}

// Alg. 4 feeds eta * g into the accumulator: one more rounded product.
__device__ __forceinline__ float4 scale_g(const TopkArgs& A, float4 g) {
  if (A.gscale) {
    g.x = __fmul_rn(A.gs, g.x);
    g.y = __fmul_rn(A.gs, g.y);
    g.z = __fmul_rn(A.gs, g.z);
    g.w = __fmul_rn(A.gs, g.w);
  }
  return g;
}

__device__ __forceinline__ int g_mode(const float* p) {
  const uintptr_t a = reinterpret_cast<uintptr_t>(p);
  return (a & 15) == 0 ? 4 : ((a & 7) == 0 ? 2 : 1);
}


__device__ __forceinline__ uint32_t warp_excl_scan(uint32_t x, uint32_t* total) {
  const int lane = threadIdx.x & 31;
  uint32_t incl = x;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += y;
  }
  *total = __shfl_sync(0xffffffffu, incl, 31);
  return incl - x;
}

// Sampled coordinate of slot i. Exact top-k: kSampleRun (16) consecutive
// coordinates from (c * d / chunks) rounded down to a multiple of kSampleRun,
// c = 0 .. chunks-1 (every coordinate when chunks = 0); this sample only sets
// the candidate threshold, never the result. Approximate top-s (Sec. 5.1): run i/8 of the
// n = n_sample/8 runs of 8 consecutive coordinates, one per stratum
// [r d / n, (r+1) d / n), starting on a multiple of 8 inside it at the slot
// the r-th draw of the step's shared stream `key` picks (d < 8: slot i).
__device__ __forceinline__ int64_t sample_coord(const TopkArgs& A, uint64_t key, int i) {
  if (A.approx) {
    if (A.d < 8) return i;
    const uint64_t n = A.n_sample >> 3, d = (uint64_t)A.d, run = (uint64_t)i >> 3;
    const uint64_t lo = run * d / n, hi = (run + 1) * d / n;
    const uint64_t a = (lo + 7) & ~uint64_t(7);
    return (int64_t)(a + 8 * (uint64_t)below(draw(key, run), (hi - a) >> 3) + (i & 7));
  }
  if (!A.sample_chunks) return i;
  // sample_chunks is kSampleChunks, a power of two: floor(ch * d / kSampleChunks)
  // by a shift (a 64-bit division would cost more than the slot's loads)
  static_assert((kSampleChunks & (kSampleChunks - 1)) == 0, "kSampleChunks must be a power of two");
  constexpr int kChunkShift = __builtin_ctz(kSampleChunks);
  static_assert((1 << kChunkShift) == kSampleChunks, "shift of kSampleChunks");
  constexpr int kRunShift = __builtin_ctz(kSampleRun);
  const int64_t ch = i >> kRunShift;
  return (((ch * A.d) >> kChunkShift) & ~int64_t(kSampleRun - 1)) + (i & (kSampleRun - 1));
}
__device__ __forceinline__ uint64_t sample_key(const TopkArgs& A) {
  return A.approx ? stream_key(A.seed, A.t, 0) : 0ull;
}

// The previous step's aggregation at the sampled coordinates, when it is
// still pending, once for all workers: the senders of coordinate j are the
// workers whose value there (still in e: it was their accumulator) was
// selected; w still holds w_t. For slot i: the senders' mask, and
// w_{t+1}[j] - w_t[j] -- their values summed in ascending worker order from
// +0 (Alg. 1). The approximate top-s runs it every step: it also stores each
// slot's coordinate, and the step's w_t - w_{t-1} there (from dlt when no
// aggregation is pending), for k_sample to read in order.
constexpr int kTailBlocks = 4;  // blocks of tiles the bulk pass ends with: the coldest (tile_order)

__global__ void __launch_bounds__(kThreads) k_sample_pending(TopkArgs A) {
  griddep_wait();
  __shared__ uint32_t Tp[kMaxK], tip[kMaxK];
  for (int kk = threadIdx.x; kk < A.K; kk += blockDim.x) {  // the previous step's selections
    Tp[kk] = A.sel[kk].T;
    tip[kk] = A.sel[kk].t_idx;
  }
  __syncthreads();
  if (A.use_order && blockIdx.x == gridDim.x - 1) {  // the launch's extra block
    // The block order of this step's bulk pass (tile_order): the blocks in
    // the golden-stride sequence (b * blk_mul) mod nb, which spreads every run
    // of neighbouring blocks evenly over the pass, except the kTailBlocks
    // blocks that produced the fewest candidates since the last order was
    // made, which go last (the coldest at the very end): the pass then ends
    // on light tiles. Deterministic: minima by (count, block), one scan.
    __shared__ unsigned long long ws64[32];
    __shared__ unsigned long long s_pick[kTailBlocks];
    const uint32_t nb = A.n_blk, per = (nb + blockDim.x - 1) / blockDim.x;
    const uint32_t lo = min(nb, threadIdx.x * per), hi = min(nb, lo + per);
    for (int r = 0; r < kTailBlocks; ++r) {
      unsigned long long m = ~0ull;
      for (uint32_t b = lo; b < hi; ++b) {
        const unsigned long long key = ((unsigned long long)A.blk_cost[b] << 32) | b;
        bool taken = false;
        for (int q = 0; q < r; ++q) taken |= s_pick[q] == key;
        if (!taken && key < m) m = key;
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const unsigned long long y = __shfl_xor_sync(0xffffffffu, m, o);
        m = y < m ? y : m;
      }
      if ((threadIdx.x & 31) == 0) ws64[threadIdx.x >> 5] = m;
      __syncthreads();
      if (threadIdx.x == 0) {
        unsigned long long mm = ~0ull;
        for (int w = 0; w < (int)(blockDim.x >> 5); ++w) mm = ws64[w] < mm ? ws64[w] : mm;
        s_pick[r] = mm;
      }
      __syncthreads();
    }
    uint32_t pick[kTailBlocks];
#pragma unroll
    for (int r = 0; r < kTailBlocks; ++r) pick[r] = (uint32_t)s_pick[r];
    auto picked = [&](uint32_t b) {
      bool t = false;
#pragma unroll
      for (int r = 0; r < kTailBlocks; ++r) t |= pick[r] == b;
      return t;
    };
    // positions q of the sequence in this thread's chunk, less the picked blocks before
    unsigned long long skip = 0, n_skip;
    for (uint32_t q = lo; q < hi; ++q) skip += picked((uint32_t)(((unsigned long long)q * A.blk_mul) % nb));
    uint32_t pos = lo - (uint32_t)(block_inclusive_scan<unsigned long long>(skip, ws64, &n_skip) - skip);
    for (uint32_t q = lo; q < hi; ++q) {
      const uint32_t b = (uint32_t)(((unsigned long long)q * A.blk_mul) % nb);
      if (!picked(b)) A.blk_order[pos++] = b;
    }
    if (threadIdx.x < kTailBlocks) A.blk_order[nb - 1 - threadIdx.x] = pick[threadIdx.x];
    __syncthreads();  // every cost read: this step's pass counts afresh
    for (uint32_t b = lo; b < hi; ++b) A.blk_cost[b] = 0u;
    return;
  }
  const int n_s = (int)A.n_sample;
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n_s) return;
  const int64_t j = sample_coord(A, sample_key(A), i);
  uint32_t m = 0;
  float dd = 0.f;
  if (A.pending) {
    float x[kMaxK];
#pragma unroll
    for (int b = 0; b < kMaxK; ++b) x[b] = b < A.K ? __ldcg(A.e + (int64_t)b * A.ld + j) : 0.f;
    const float wo = A.w[j];  // loaded with the residuals, used only where a worker sent
    float sum = 0.f;
#pragma unroll
    for (int b = 0; b < kMaxK; ++b) {
      if (b < A.K && selected(mag_key(x[b]), (uint32_t)j, Tp[b], tip[b])) {
        sum = __fadd_rn(sum, x[b]);
        m |= 1u << b;
      }
    }
    if (m) dd = __fsub_rn(__fsub_rn(wo, __fmul_rn(A.a_prev, sum)), wo);
  }
  if (A.approx) {
    if (!m) dd = A.dlt[j];
    A.sample_pend[2 * A.sample_stride + i] = (uint32_t)j;
  }
  A.sample_pend[i] = m;
  A.sample_pend[A.sample_stride + i] = __float_as_uint(dd);
}

// Bin of a candidate key in the relative histogram: (key - theta) >> shift,
// the top bin also taking everything further up (candidate keys are >= theta).
__device__ __forceinline__ int rel_bin(uint32_t key, uint32_t theta, int shift) {
  const uint32_t b = (key > theta ? key - theta : 0u) >> shift;
  return b < (uint32_t)kRelBins ? (int)b : kRelBins - 1;
}

// ---------------------------------------------------------------------------
// Sample of the approximate top-s (Sec. 5.1): blocks spread over the workers'
// samples store every sampled key and add its first radix digit to the
// worker's histogram, for k_sample_theta. The accumulator at a sampled
// coordinate is formed as if the previous step's aggregation had been applied
// (residual +0 where the worker sent, the pending delta).
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kThreads) k_sample(TopkArgs A) {
  griddep_wait();
  __shared__ uint32_t hist[kHistBins];
  const int k = blockIdx.y;
  WorkerSel& S = A.sel[k];
  if (blockIdx.x == 0 && k == 0 && threadIdx.x == 0) {
    A.big_tiles[0] = 0;
    *A.tile_ctr = 0u;  // the bulk pass claims its tiles from zero
  }
  if (blockIdx.x == 0)  // this step's candidate histogram starts empty
    for (int b = threadIdx.x; b < kRelBins; b += blockDim.x) A.chist[(int64_t)k * kRelBins + b] = 0u;
  if (A.dense_mode) {
    if (blockIdx.x == 0 && threadIdx.x == 0) {
      S.theta = kNoCandidate;
      S.count = 0;
      S.dense = 0;
    }
    return;
  }
  const float* ek = A.e + (int64_t)k * A.ld;
  const float* gk = A.grads + (int64_t)k * A.d;
  const uint16_t* gk16 = A.grads16 + (int64_t)k * A.d;
  uint32_t* keys = A.sample_keys + (int64_t)k * A.sample_stride;
  const int n_s = (int)A.n_sample;
  for (int b = threadIdx.x; b < kHistBins; b += blockDim.x) hist[b] = 0;
  __syncthreads();
  const int per = (n_s + gridDim.x - 1) / gridDim.x;
  const int i_lo = blockIdx.x * per;
  const int i_hi = min(n_s, i_lo + per);
  for (int i0 = i_lo; i0 < i_hi; i0 += 8 * blockDim.x) {
    float ev[8], gv[8], dv[8];
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      const int i = i0 + q * blockDim.x + threadIdx.x;
      ev[q] = gv[q] = dv[q] = 0.f;
      if (i < i_hi) {  // coordinate, senders and w_t - w_{t-1} from k_sample_pending
        const int64_t j = A.sample_pend[2 * A.sample_stride + i];
        const uint32_t m = A.sample_pend[i];
        const float e = ek[j];  // loaded whatever m holds: no load waits on another but j
        ev[q] = ((m >> k) & 1u) ? 0.f : e;
        const float g = A.bf16 ? bf16_f32(gk16[j]) : gk[j];
        gv[q] = A.local_mom ? local_m(A, k, j, g) : (A.gscale ? __fmul_rn(A.gs, g) : g);
        dv[q] = __uint_as_float(A.sample_pend[A.sample_stride + i]);
      }
    }
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      const int i = i0 + q * blockDim.x + threadIdx.x;
      int bin = -1;
      if (i < i_hi) {
        const uint32_t key = mag_key(accumulate(ev[q], gv[q], A.c, dv[q]));
        keys[i] = key;
        bin = (int)(key >> 20);
      }
      warp_hist_add(hist, bin);
    }
  }
  __syncthreads();
  uint32_t* gh = A.ghist + (int64_t)k * kHistBins;
  for (int b = threadIdx.x; b < kHistBins; b += blockDim.x)
    if (hist[b]) atomicAdd(&gh[b], hist[b]);
  // k_sample_theta fixes theta exactly from the keys and this histogram
}

// Radix select in shared memory over values below 2^bits (bits <= 31), taken
// relative to `base` (x[i] - base): digits of at most 11 bits from the top.
// Returns base + the r-th largest; rank_out = its rank among the values equal
// to it. With bits = 31 and base = 0 this is a select over whole keys.
__device__ __forceinline__ uint32_t smem_select_bits(const uint32_t* x, uint32_t n, uint32_t r, int bits,
                                                     uint32_t base, uint32_t* h, uint32_t* ws,
                                                     uint32_t* s_bin, uint32_t* s_rank, uint32_t* rank_out) {
  uint32_t prefix = 0;  // the digits fixed so far
  int done = 0;         // bits fixed so far (from the top)
  while (done < bits) {
    const int width = min(11, bits - done), shift = bits - done - width, nbins = 1 << width;
    for (int b = threadIdx.x; b < nbins; b += blockDim.x) h[b] = 0;
    if (threadIdx.x == 0) {
      *s_bin = 0;
      *s_rank = 0;
    }
    __syncthreads();
    for (uint32_t i0 = 0; i0 < n; i0 += blockDim.x) {
      const uint32_t i = i0 + threadIdx.x;
      if (i < n) {
        const uint32_t v = x[i] - base;
        // the digits above this one must match the prefix (a shift by 32 is
        // avoided: no digit is fixed before the first pass)
        if (done == 0 || (v >> (shift + width)) == prefix) atomicAdd(&h[(v >> shift) & (uint32_t)(nbins - 1)], 1u);
      }
    }
    __syncthreads();
    block_find_from_top_any(h, nbins, r, ws, s_bin, s_rank);
    prefix = (prefix << width) | *s_bin;
    r = *s_rank;
    done += width;
    __syncthreads();
  }
  *rank_out = r;
  return base + prefix;
}

// Radix select in shared memory: the r-th largest of n values (digits 11/10/10).
__device__ __forceinline__ uint32_t smem_select(const uint32_t* x, uint32_t n, uint32_t r,
                                                uint32_t* h, uint32_t* ws, uint32_t* s_bin,
                                                uint32_t* s_rank, uint32_t* rank_out) {
  uint32_t prefix = 0;
  for (int pass = 0; pass < 3; ++pass) {
    const int nbins = pass == 0 ? 2048 : 1024;
    const int shift = pass == 0 ? 20 : (pass == 1 ? 10 : 0);
    for (int b = threadIdx.x; b < nbins; b += blockDim.x) h[b] = 0;
    if (threadIdx.x == 0) {
      *s_bin = 0;
      *s_rank = 0;
    }
    __syncthreads();
    for (uint32_t i0 = 0; i0 < n; i0 += blockDim.x) {
      const uint32_t i = i0 + threadIdx.x;
      int bin = -1;
      if (i < n) {
        const uint32_t v = x[i];
        if (pass == 0 || (v >> (shift + 10)) == prefix) bin = (int)((v >> shift) & (uint32_t)(nbins - 1));
      }
      if (bin >= 0) atomicAdd(&h[bin], 1u);  // plain atomics measured faster than match_any here
    }
    __syncthreads();
    block_find_from_top(h, nbins, r, ws, s_bin, s_rank);
    prefix = pass == 0 ? *s_bin : ((prefix << 10) | *s_bin);
    r = *s_rank;
    __syncthreads();
  }
  *rank_out = r;
  return prefix;
}

// ---------------------------------------------------------------------------
// The exact top-k's sample with one thread-block cluster per worker (its CTAs
// are co-scheduled by the hardware). Each CTA forms v at its slots (up to 8 per
// thread, kept in registers) and adds its keys' first radix digit (bits
// 30..20) into the histogram held in the shared memory of the cluster's first
// CTA; after a cluster barrier every CTA reads it back and finds the bin of
// the r-th largest key, adds the second digit (bits 19..10) of its keys in
// that bin into a second histogram there, and after another barrier the first
// CTA reads off theta = the two digits: a lower bound of the r-th largest
// sampled key within 2^10 keys. Distributed shared memory and hardware
// barriers only: no global scratch, no spin-wait.
// ---------------------------------------------------------------------------
// Eight consecutive values from p: two 16-byte loads when p is 16-byte
// aligned, else eight 4-byte (or 2-byte) loads.
__device__ __forceinline__ void load8(const float* p, float (&v)[8]) {
  if ((reinterpret_cast<uintptr_t>(p) & 15u) == 0) {
    const float4 a = *reinterpret_cast<const float4*>(p), b = *reinterpret_cast<const float4*>(p + 4);
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
    v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
  } else {
#pragma unroll
    for (int q = 0; q < 8; ++q) v[q] = p[q];
  }
}
__device__ __forceinline__ void load8u(const uint32_t* p, uint32_t (&v)[8]) {
  if ((reinterpret_cast<uintptr_t>(p) & 15u) == 0) {
    const uint4 a = *reinterpret_cast<const uint4*>(p), b = *reinterpret_cast<const uint4*>(p + 4);
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
    v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
  } else {
#pragma unroll
    for (int q = 0; q < 8; ++q) v[q] = p[q];
  }
}
__device__ __forceinline__ void load8_bf16(const uint16_t* p, float (&v)[8]) {
  if ((reinterpret_cast<uintptr_t>(p) & 15u) == 0) {
    const uint4 a = *reinterpret_cast<const uint4*>(p);
    const uint32_t w[4] = {a.x, a.y, a.z, a.w};
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      v[2 * q] = bf16_f32((uint16_t)(w[q] & 0xffffu));
      v[2 * q + 1] = bf16_f32((uint16_t)(w[q] >> 16));
    }
  } else {
#pragma unroll
    for (int q = 0; q < 8; ++q) v[q] = bf16_f32(p[q]);
  }
}

namespace scl {
// Four CTAs of 1024 threads per worker: clusters of eight CTAs left the
// sixteenth worker's cluster waiting for a second wave at K = 16 (only
// fifteen were co-resident on GB300), which doubled the sample's time
constexpr int kCtas = 4;                                    // CTAs per cluster, one cluster per worker
constexpr int kThreadsC = 1024;
constexpr int kSlots = kSampleSlots / (kCtas * kThreadsC);  // sampled slots per thread
static_assert(kSlots * kCtas * kThreadsC == kSampleSlots, "the cluster covers the whole sample");
static_assert(kSlots == 8 && kSampleRun % kSlots == 0,
              "a thread's slots are 8 consecutive coordinates of one sampled run (load8)");
static_assert(kHistBins % kThreadsC == 0 && 1024 % kThreadsC == 0, "histograms split evenly over a block");
}  // namespace scl

__global__ void __cluster_dims__(scl::kCtas, 1, 1) __launch_bounds__(scl::kThreadsC)
    k_sample_cluster(TopkArgs A) {
  using namespace scl;
  griddep_wait();
  namespace cg = cooperative_groups;
  cg::cluster_group cl = cg::this_cluster();
  __shared__ uint32_t hist[kHistBins];  // this CTA's counts
  __shared__ uint32_t red1[kHistBins];  // first CTA: the cluster's first-digit counts
  __shared__ uint32_t red2[1024];       // first CTA: the cluster's second digits in the bin b1
  __shared__ uint32_t ws[32];
  __shared__ uint32_t s_bin, s_rank;
  const int k = blockIdx.y;
  const unsigned crank = cl.block_rank();
  WorkerSel& S = A.sel[k];
  if (crank == 0 && k == 0) {  // the step's first kernel that counts: its counters start at zero
    if (threadIdx.x == 0) {
      A.big_tiles[0] = 0;
      *A.tile_ctr = 0u;  // and the bulk pass claims its tiles from zero
    }
    if (threadIdx.x < 8) A.step_ctr->v[threadIdx.x] = 0ull;
  }
  if (crank == 0)  // this step's candidate histogram starts empty
    for (int b = threadIdx.x; b < kRelBins; b += blockDim.x) A.chist[(int64_t)k * kRelBins + b] = 0u;
  if (A.dense_mode) {  // uniform over the grid: no CTA reaches a cluster barrier
    if (crank == 0 && threadIdx.x == 0) {
      S.theta = kNoCandidate;
      S.count = 0;
      S.dense = 0;
    }
    return;
  }
  for (int b = threadIdx.x; b < kHistBins; b += blockDim.x) {
    hist[b] = 0;
    red1[b] = 0;
  }
  for (int b = threadIdx.x; b < 1024; b += blockDim.x) red2[b] = 0;
  const float* ek = A.e + (int64_t)k * A.ld;
  const float* gk = A.grads + (int64_t)k * A.d;
  const uint16_t* gk16 = A.grads16 + (int64_t)k * A.d;
  const int n_s = (int)A.n_sample;  // at most kSampleSlots
  // this thread's slots: kSlots consecutive coordinates j0 .. j0 + 7 of one
  // run (every coordinate when the sample is the whole vector), read with 16-byte
  // loads where the rows allow; every load is issued before any value is
  // used, then v is formed as if the previous step's aggregation were applied
  const int i0 = ((int)crank * kThreadsC + (int)threadIdx.x) * kSlots;
  const int nv = max(0, min(kSlots, n_s - i0));  // valid slots
  float ev[kSlots], gv[kSlots], dv[kSlots], lv[kSlots];
  uint32_t pm[kSlots], pd[kSlots];
#pragma unroll
  for (int q = 0; q < kSlots; ++q) {
    ev[q] = gv[q] = dv[q] = lv[q] = 0.f;
    pm[q] = pd[q] = 0u;
  }
  if (nv == kSlots) {
    const int64_t j0 = sample_coord(A, 0ull, i0);  // a multiple of kSlots (runs start on kSampleRun)
    load8(ek + j0, ev);  // rows of e, lm and dlt start on 16 bytes (ld: whole tiles)
    load8(A.dlt + j0, dv);
    if (A.local_mom) load8(A.lm + (int64_t)k * A.ld + j0, lv);
    if (A.bf16) load8_bf16(gk16 + j0, gv);
    else load8(gk + j0, gv);  // a row of g starts on 4 bytes: 16-byte loads only where aligned
    if (A.pending) {
      load8u(A.sample_pend + i0, pm);
      load8u(A.sample_pend + A.sample_stride + i0, pd);
    }
  } else {
#pragma unroll
    for (int q = 0; q < kSlots; ++q) {
      if (q < nv) {
        const int64_t j = sample_coord(A, 0ull, i0 + q);
        ev[q] = ek[j];
        gv[q] = A.bf16 ? bf16_f32(gk16[j]) : gk[j];
        dv[q] = A.dlt[j];
        if (A.local_mom) lv[q] = A.lm[(int64_t)k * A.ld + j];
        if (A.pending) {
          pm[q] = A.sample_pend[i0 + q];
          pd[q] = A.sample_pend[A.sample_stride + i0 + q];
        }
      }
    }
  }
  uint32_t key[kSlots];
#pragma unroll
  for (int q = 0; q < kSlots; ++q) {
    const float g = A.local_mom ? __fadd_rn(__fmul_rn(A.beta, lv[q]), __fmul_rn(A.gs, gv[q]))
                                : (A.gscale ? __fmul_rn(A.gs, gv[q]) : gv[q]);
    const float e = ((pm[q] >> k) & 1u) ? 0.f : ev[q];
    const float dl = pm[q] ? __uint_as_float(pd[q]) : dv[q];
    key[q] = q < nv ? mag_key(accumulate(e, g, A.c, dl)) : 0xffffffffu;
    // plain shared-memory atomics: a warp's keys spread over a few dozen bins,
    // and the warp-aggregated form (match_any) measured slower here
    if (key[q] != 0xffffffffu) atomicAdd(&hist[key[q] >> 20], 1u);
  }
  // every CTA of the cluster runs and has zeroed its histograms before any remote add
  cl.sync();
  uint32_t* r1 = cl.map_shared_rank(red1, 0);
  for (int b = threadIdx.x; b < kHistBins; b += blockDim.x)
    if (hist[b]) atomicAdd(&r1[b], hist[b]);
  cl.sync();
  // the bin of the r-th largest key and its rank there (every CTA alike)
  for (int b = threadIdx.x; b < kHistBins; b += blockDim.x) hist[b] = r1[b];
  if (threadIdx.x == 0) {
    s_bin = 0;
    s_rank = 0;
  }
  __syncthreads();
  const uint32_t r = A.sample_rank < (uint32_t)n_s ? A.sample_rank : (uint32_t)n_s;
  block_find_from_top(hist, kHistBins, r, ws, &s_bin, &s_rank);
  const uint32_t b1 = s_bin, rr = s_rank;
  for (int b = threadIdx.x; b < 1024; b += blockDim.x) hist[b] = 0;
  __syncthreads();
#pragma unroll
  for (int q = 0; q < kSlots; ++q)
    if (key[q] != 0xffffffffu && (key[q] >> 20) == b1) atomicAdd(&hist[(key[q] >> 10) & 1023u], 1u);
  __syncthreads();
  uint32_t* r2 = cl.map_shared_rank(red2, 0);
  for (int b = threadIdx.x; b < 1024; b += blockDim.x)
    if (hist[b]) atomicAdd(&r2[b], hist[b]);
  // after this barrier no CTA touches another's shared memory
  cl.sync();
  if (crank != 0) return;
  if (threadIdx.x == 0) {
    s_bin = 0;
    s_rank = 0;
  }
  __syncthreads();
  block_find_from_top(red2, 1024, rr, ws, &s_bin, &s_rank);
  if (threadIdx.x == 0) {
    // capped at the Inf key: every non-finite value is a candidate (and counted there)
    S.theta = min((b1 << 20) | (s_bin << 10), 0x7f800000u);
    S.count = 0;
    S.dense = 0;
  }
}

// ---------------------------------------------------------------------------
// Approximate top-s (Sec. 5.1): theta is the exact r-th largest sampled key.
// Every block finds, from the sample's first-digit histogram, the bin that
// holds it and collects that bin's keys from its slice of the sample (128 a
// round, one bucket reservation); the last block ranks the bucket in shared
// memory. A bin too crowded for the bucket is resolved by the last block's
// two remaining radix digits over the whole sample.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kThreads) k_sample_theta(TopkArgs A) {
  griddep_wait();
  extern __shared__ __align__(16) uint32_t fin[];  // kBucketCap keys
  __shared__ uint32_t h[kHistBins];
  __shared__ uint32_t ws[32];
  __shared__ uint32_t s_last, s_bin, s_rank, s_n;
  const int k = blockIdx.y;
  WorkerSel& S = A.sel[k];
  uint32_t* gh = A.ghist + (int64_t)k * kHistBins;
  for (int b = threadIdx.x; b < kHistBins; b += blockDim.x) h[b] = __ldcg(&gh[b]);
  if (threadIdx.x == 0) {
    s_bin = 0;
    s_rank = 0;
  }
  __syncthreads();
  const uint32_t n_s = A.n_sample;
  const uint32_t r = A.sample_rank < n_s ? A.sample_rank : n_s;
  block_find_from_top(h, kHistBins, r, ws, &s_bin, &s_rank);
  const uint32_t b1 = s_bin, r1 = s_rank;
  const uint32_t* keys = A.sample_keys + (int64_t)k * A.sample_stride;
  uint32_t* bk = A.bucket + (int64_t)k * 2 * kBucketCap;
  const int lane = threadIdx.x & 31;
  const uint32_t lt = lanemask_lt();
  const uint32_t per = (n_s + gridDim.x - 1) / gridDim.x;
  const uint32_t i_lo = min(n_s, blockIdx.x * per), i_hi = min(n_s, i_lo + per);
  for (uint32_t i0 = i_lo + (threadIdx.x >> 5) * 128; i0 < i_hi; i0 += kWarps * 128) {
    uint32_t key[4], m[4], n = 0;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const uint32_t i = i0 + q * 32 + lane;
      key[q] = i < i_hi ? __ldcg(keys + i) : 0u;
      m[q] = __ballot_sync(0xffffffffu, i < i_hi && (key[q] >> 20) == b1);
      n += __popc(m[q]);
    }
    if (n) {
      uint32_t base = 0;
      if (lane == 0) base = atomicAdd(&S.count_bucket, n);
      base = __shfl_sync(0xffffffffu, base, 0);
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const uint32_t o = base + __popc(m[q] & lt);
        if (((m[q] >> lane) & 1u) && o < (uint32_t)kBucketCap) bk[o] = key[q];
        base += __popc(m[q]);
      }
    }
  }
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) s_last = (atomicAdd(&S.done[2], 1u) == gridDim.x - 1) ? 1u : 0u;
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  if (threadIdx.x == 0) {
    s_n = __ldcg(&S.count_bucket);
    S.count_bucket = 0;
    S.done[2] = 0;
  }
  for (int b = threadIdx.x; b < kHistBins; b += blockDim.x) gh[b] = 0;  // zero between uses
  __syncthreads();
  const uint32_t n = s_n;
  uint32_t theta;
  if (n <= (uint32_t)kBucketCap) {
    for (uint32_t i = threadIdx.x; i < n; i += blockDim.x) fin[i] = __ldcg(&bk[i]);
    __syncthreads();
    uint32_t unused;
    theta = smem_select(fin, n, r1, h, ws, &s_bin, &s_rank, &unused);
  } else {
    // the remaining digits (bits 19..10, then 9..0) over every sampled key
    uint32_t prefix = b1, rr = r1;
    for (int pass = 1; pass < 3; ++pass) {
      const int shift = pass == 1 ? 10 : 0;
      for (int b = threadIdx.x; b < 1024; b += blockDim.x) h[b] = 0;
      if (threadIdx.x == 0) {
        s_bin = 0;
        s_rank = 0;
      }
      __syncthreads();
      for (uint32_t i0 = 0; i0 < n_s; i0 += blockDim.x) {
        const uint32_t i = i0 + threadIdx.x;
        int bin = -1;
        if (i < n_s) {
          const uint32_t v = __ldcg(keys + i);
          if ((v >> (shift + 10)) == prefix) bin = (int)((v >> shift) & 1023u);
        }
        warp_hist_add(h, bin);
      }
      __syncthreads();
      block_find_from_top(h, 1024, rr, ws, &s_bin, &s_rank);
      prefix = (prefix << 10) | s_bin;
      rr = s_rank;
      __syncthreads();
    }
    theta = prefix;
  }
  if (threadIdx.x == 0) {
    // capped at the Inf key: every non-finite value is a candidate (and counted there)
    S.theta = min(theta, 0x7f800000u);
    S.count = 0;
    S.dense = 0;
    S.nsel = 0;
  }
}

// ---------------------------------------------------------------------------
// accumulate + filter. Each warp owns one sub-tile (1/kChunksPerTile) of every
// tile; for each worker it writes v over e and appends its candidates as one
// index-sorted sub-chunk, reserved at once -- warps never wait for each other.
// ---------------------------------------------------------------------------
// A restored state (gmc_load_state): w_t - w_{t-1} is in dlt over the whole
// range, with no pair lists of the step before. Read it densely for one warp's
// sub-tile [sub0, sub0 + n) (n a multiple of 4, sub0 16-byte aligned, inside
// ld) and clear it, as the listed path does.
__device__ __forceinline__ void stage_delta_dense(const TopkArgs& A, uint32_t sub0, int n, float* dlw,
                                                  int lane) {
  for (int i = lane; i < n / 4; i += 32) {
    float4* p = reinterpret_cast<float4*>(A.dlt + sub0) + i;
    const float4 x = *p;
    reinterpret_cast<float4*>(dlw)[i] = x;
    if ((__float_as_uint(x.x) | __float_as_uint(x.y) | __float_as_uint(x.z) | __float_as_uint(x.w)) != 0u)
      *p = make_float4(0.f, 0.f, 0.f, 0.f);
  }
  __syncwarp();
}

// w_t - w_{t-1} on one warp's sub-tile [sub0, sub0 + n) into dlw: non-zero only
// where the previous step sent pairs, listed by its sub-chunks (k', tile, w).
__device__ __forceinline__ void stage_delta_warp(const TopkArgs& A, int64_t tile, int w,
                                                 uint32_t sub0, int n, float* dlw, int lane) {
  if (A.dense_prev) {
    stage_delta_dense(A, sub0, n, dlw, lane);
    return;
  }
  for (int i = lane; i < n / 4; i += 32)
    reinterpret_cast<float4*>(dlw)[i] = make_float4(0.f, 0.f, 0.f, 0.f);
  __syncwarp();
  if (A.has_prev) {
    for (int k0 = 0; k0 < A.K; k0 += 32) {
      const int kk = k0 + lane;
      uint32_t base = 0, cnt = 0;
      if (kk < A.K) {
        const uint2 bc = A.chunk_prev[chunk_at(A, kk, tile, w)];
        base = bc.x;
        cnt = bc.y;
      }
      uint32_t total;
      const uint32_t pre = warp_excl_scan(cnt, &total);
      for (uint32_t e0 = 0; e0 < total; e0 += 32) {
        const uint32_t e = e0 + lane;
        int src = 0;  // the last lane whose non-empty sub-chunk starts at or before e
#pragma unroll 1
        for (int l = 1; l < 32; ++l) {
          const uint32_t pl = __shfl_sync(0xffffffffu, pre, l);
          const uint32_t cl = __shfl_sync(0xffffffffu, cnt, l);
          if (cl && pl <= e) src = l;
        }
        const uint32_t b = __shfl_sync(0xffffffffu, base, src);
        const uint32_t p = __shfl_sync(0xffffffffu, pre, src);
        if (e < total) {
          const uint32_t at = b + (e - p);
          if (at < A.cap) {
            const int64_t q = (int64_t)(k0 + src) * A.cap + at;
            const uint32_t j = A.cand_idx_prev[q];
            const WorkerSel& Sp = A.sel[k0 + src];  // the previous step's selection
            if (selected(mag_key(A.cand_val_prev[q]), j, Sp.T, Sp.t_idx)) {
              const int64_t l = (int64_t)j - sub0;
              if (l >= 0 && l < n) dlw[l] = A.dlt[j];
              else atomicOr(A.status, kStatusInternal);
            }
          }
        }
      }
    }
    __syncwarp();
    // w_t - w_{t-1} has been read for this sub-tile; clear it here (this step's
    // aggregate writes w_{t+1} - w_t)
    for (int l = lane; l < n; l += 32)
      if (dlw[l] != 0.f) A.dlt[sub0 + l] = 0.f;
  }
  __syncwarp();
}

// The previous step's aggregation (Alg. 1: w_{t+1} = w_t - (eta/K) sum_k C_k(.),
// e_{t+1,k} = e_{t+1/2,k} - C_k(.)) applied on one warp's sub-tile
// [sub0, sub0 + n), n <= 512, when it was left pending: from the previous
// step's sent pairs of this sub-tile (sub-chunks (k', tile, w)) it records the
// senders of every coordinate in mkw, sums their values in ascending worker
// order from +0, writes w_{t+1} over w_t there and leaves w_{t+1} - w_t in dlw.
// The residuals are not touched: the caller takes e = +0 where mkw has its bit.
__device__ __forceinline__ void stage_pending_warp(const TopkArgs& A, int64_t tile, int w,
                                                   uint32_t sub0, int n, float* dlw, uint32_t* mkw,
                                                   int lane, uint32_t& uni, uint32_t& chg) {
  for (int i = lane; i < n / 4; i += 32) {
    reinterpret_cast<float4*>(dlw)[i] = make_float4(0.f, 0.f, 0.f, 0.f);
    reinterpret_cast<uint4*>(mkw)[i] = make_uint4(0u, 0u, 0u, 0u);
  }
  __syncwarp();
  const uint32_t lt = lanemask_lt();
  for (int k0 = 0; k0 < A.K; k0 += 32) {
    const int kk = k0 + lane;
    uint32_t base = 0, cnt = 0;
    if (kk < A.K) {
      const uint2 bc = A.chunk_prev[chunk_at(A, kk, tile, w)];
      base = bc.x;
      cnt = bc.y;
    }
    uint32_t total;
    const uint32_t pre = warp_excl_scan(cnt, &total);
    // entries run through the workers in ascending order, 32 per round
    for (uint32_t e0 = 0; e0 < total; e0 += 32) {
      const uint32_t e = e0 + lane;
      int src = 0;
#pragma unroll 1
      for (int l = 1; l < 32; ++l) {
        const uint32_t pl = __shfl_sync(0xffffffffu, pre, l);
        const uint32_t cl = __shfl_sync(0xffffffffu, cnt, l);
        if (cl && pl <= e) src = l;
      }
      const uint32_t b = __shfl_sync(0xffffffffu, base, src);
      const uint32_t p = __shfl_sync(0xffffffffu, pre, src);
      bool act = false;
      uint32_t l = 0;
      float v = 0.f;
      if (e < total) {
        const uint32_t at = b + (e - p);
        if (at < A.cap) {
          const int64_t q = (int64_t)(k0 + src) * A.cap + at;
          const uint32_t j = A.cand_idx_prev[q];
          const float vq = A.cand_val_prev[q];
          const WorkerSel& Sp = A.sel[k0 + src];  // the previous step's selection
          if (selected(mag_key(vq), j, Sp.T, Sp.t_idx)) {
            const int64_t ll = (int64_t)j - sub0;
            if (ll >= 0 && ll < n) {
              act = true;
              l = (uint32_t)ll;
              v = vq;
              atomicOr(&mkw[l], 1u << (k0 + src));
            } else {
              atomicOr(A.status, kStatusInternal);
            }
          }
        }
      }
      // lanes holding the same coordinate add one at a time, in lane (= worker) order
      const uint32_t peers = __match_any_sync(0xffffffffu, act ? (int)l : -1 - lane);
      const uint32_t r = __popc(peers & lt);
      const uint32_t rmax = __reduce_max_sync(0xffffffffu, act ? r : 0u);
      for (uint32_t turn = 0; turn <= rmax; ++turn) {
        if (act && r == turn) dlw[l] = __fadd_rn(dlw[l], v);
        __syncwarp();
      }
    }
  }
  __syncwarp();
  // coordinates of the union: w_{t+1} = w_t - a * sum (all loads issued first)
  float wo[16];
  uint32_t has = 0;
#pragma unroll
  for (int i = 0; i < 16; ++i) {
    const int l = lane + 32 * i;
    wo[i] = 0.f;
    if (l < n && mkw[l]) {
      has |= 1u << i;
      wo[i] = A.w[sub0 + l];
    }
  }
#pragma unroll
  for (int i = 0; i < 16; ++i) {
    if ((has >> i) & 1u) {
      const int l = lane + 32 * i;
      const float wn = __fsub_rn(wo[i], __fmul_rn(A.a_prev, dlw[l]));
      A.w[sub0 + l] = wn;
      const float dd = __fsub_rn(wn, wo[i]);
      dlw[l] = dd;
      ++uni;
      chg += dd != 0.f;
    }
  }
  __syncwarp();
}

// Candidate flags (bit i: value i is a candidate) of 4 consecutive values at
// sub-tile offset l; `lim` = valid values in the sub-tile (all when it is full).
__device__ __forceinline__ uint32_t cand_bits(const float v[4], int l, int lim, uint32_t theta) {
  uint32_t bits = 0;
#pragma unroll
  for (int i = 0; i < 4; ++i)
    bits |= ((mag_key(v[i]) >= theta) && (l + i < lim) ? 1u : 0u) << i;
  return bits;
}

// Write one group's candidates (index order: lane-major, element-minor) at
// pos; counts the non-finite ones (theta never exceeds the Inf key).
__device__ __forceinline__ void write_group(const float v[4], uint32_t j, uint32_t bits, uint32_t lt,
                                            uint32_t& pos, uint32_t end, uint32_t* ci, float* cv,
                                            uint32_t& nonfinite) {
  const uint32_t n = __popc(bits);
  if (!__any_sync(0xffffffffu, n != 0)) return;
  uint32_t incl = n;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_up_sync(0xffffffffu, incl, o);
    if ((int)(threadIdx.x & 31) >= o) incl += y;
  }
  uint32_t o = pos + incl - n;
  pos += __shfl_sync(0xffffffffu, incl, 31);
  (void)lt;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    if ((bits >> i) & 1u) {
      if (o < end) {
        ci[o] = j + i;
        cv[o] = v[i];
      }
      nonfinite += is_nonfinite(v[i]) ? 1u : 0u;
      ++o;
    }
  }
}

// load/store version for small tiles; candidates share one region per worker
// kLocal: the local-momentum baseline's instantiation (its momentum loads
// need registers the other forms do without).
template <int U, bool kLocal, bool kBf16>
__global__ void __launch_bounds__(kThreads) k_accumulate(TopkArgs A) {
  griddep_wait();
  constexpr int SUB = 128 * U;       // elements per warp and worker
  constexpr int T = kWarps * SUB;    // elements per tile
  extern __shared__ __align__(16) unsigned char smem[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  float* dlw = reinterpret_cast<float*>(smem) + warp * SUB;
  const uint32_t lt = lanemask_lt();
  uint32_t nonfinite = 0;

  for (int64_t tile = blockIdx.x; tile < A.n_tiles; tile += gridDim.x) {
    const uint32_t s0 = (uint32_t)(tile * T) + warp * SUB;
    stage_delta_warp(A, tile, warp, s0, SUB, dlw, lane);
    const int64_t rem = A.d - (int64_t)s0;
    const int lim = rem < SUB ? (int)rem : SUB;
    for (int k = 0; k < A.K; ++k) {
      const uint32_t theta = A.sel[k].theta;
      float* ekt = A.e + (int64_t)k * A.ld + s0;
      const float* gk = A.grads + (int64_t)k * A.d;
      const uint16_t* gk16 = A.grads16 + (int64_t)k * A.d;
      const int gm = g_mode(gk);
      float4 ev[U], gv[U], mv[U];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int l = u * 128 + lane * 4;
        ev[u] = __ldcs(reinterpret_cast<const float4*>(ekt + l));
        gv[u] = scale_g(A, kBf16 ? load_g4_bf16(gk16, (int64_t)s0 + l, A.d)
                                 : load_g4(gk, (int64_t)s0 + l, A.d, gm));
        if (kLocal) mv[u] = __ldcs(reinterpret_cast<const float4*>(A.lm + (int64_t)k * A.ld + s0 + l));
      }
      if (kLocal) {
#pragma unroll
        for (int u = 0; u < U; ++u)
          gv[u] = local_m4(A, A.lm + (int64_t)k * A.ld + s0 + u * 128 + lane * 4, mv[u], gv[u]);
      }
      float v[U][4];
      uint32_t bits[U];
      uint32_t nloc = 0;
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int l = u * 128 + lane * 4;
        const float4 d4 = *reinterpret_cast<const float4*>(dlw + l);
        v[u][0] = accumulate(ev[u].x, gv[u].x, A.c, d4.x);
        v[u][1] = accumulate(ev[u].y, gv[u].y, A.c, d4.y);
        v[u][2] = accumulate(ev[u].z, gv[u].z, A.c, d4.z);
        v[u][3] = accumulate(ev[u].w, gv[u].w, A.c, d4.w);
        __stcs(reinterpret_cast<float4*>(ekt + l), make_float4(v[u][0], v[u][1], v[u][2], v[u][3]));
        bits[u] = cand_bits(v[u], l, lim, theta);
        nloc += __popc(bits[u]);
      }
      const uint32_t cnt = __reduce_add_sync(0xffffffffu, nloc);
      uint32_t base = 0;
      if (lane == 0 && cnt) base = atomicAdd(&A.sel[k].count, cnt);
      base = __shfl_sync(0xffffffffu, base, 0);
      if (cnt) {
        uint32_t pos = base;
        uint32_t* ci = A.cand_idx + (int64_t)k * A.cap;
        float* cv = A.cand_val + (int64_t)k * A.cap;
#pragma unroll
        for (int u = 0; u < U; ++u)
          write_group(v[u], s0 + u * 128 + lane * 4, bits[u], lt, pos, A.cap, ci, cv, nonfinite);
      }
      if (lane == 0) A.chunk[chunk_at(A, k, tile, warp)] = make_uint2(base, cnt);
    }
  }
  if (nonfinite) {
    atomicOr(A.status, kStatusNonfinite);
    atomicAdd(&A.step_ctr->v[kNonfinite], (unsigned long long)nonfinite);
  }
}

// ---------------------------------------------------------------------------
// bulk-copy version (tiles of 4096). One persistent CTA per SM. A producer
// thread streams each (tile, worker) item's e and g into a ring of shared-
// memory stages with cp.async.bulk; sixteen consumer warps, two per 512-
// element sub-tile of every tile (one for the workers of even index, one for
// the odd), read their part, release the stage, store v over e and append
// their candidates to their sub-tile's part of this CTA's region of the
// candidate buffer (one part per sub-tile and worker). Candidates are staged
// in shared memory and leave in whole 128-byte lines. Producer and consumers
// meet only at mbarriers (every wait bounded); the two warps of a sub-tile
// meet at a named barrier twice per tile.
//
// The even warp of a sub-tile forms its w_t - w_{t-1} (and applies the
// previous step's aggregation when it was left pending) from the previous
// step's sent pairs. Those are reached through two dependent loads -- the
// sub-chunk table, then the pairs -- and the pending case reads w at the
// pairs' coordinates: a chain of three memory latencies. The warp runs that
// chain as a pipeline, so that no latency lies on its path. With few workers
// (K <= 5, short tiles), and in the bf16 and local-momentum forms, the
// pipeline spans tiles: while the warp works on
// tile n it loads w for tile n+1, the pairs of tile n+2 and the sub-chunk
// entries of tile n+3. With more workers a tile lasts long enough for the
// whole chain of tile n+1: its entries at the start of tile n, its pairs
// after the warp's first item, w after its second. A sub-tile with more than
// 32 pairs takes the direct path (stage_pending_warp / stage_delta_warp).
//
// A CTA's first tiles are fixed and every later one is claimed from a counter
// (tile_at_n, tile_claim_n), so that CTAs whose streams run faster take more
// tiles and all of them finish together. A claim is made a few tiles before
// the CTA starts it (the pipeline must know its tiles ahead), so when the
// counter runs out each CTA still holds those tiles; the SMs' streaming rates
// differ by up to a fifth, and the CTAs' finishing times spread by that share
// of the tiles they hold. The shallow pipeline lets a CTA claim two tiles
// ahead instead of four, which halves that spread.
// ---------------------------------------------------------------------------
namespace bulk {
constexpr int kT = kBulkTile;
constexpr int kStages = 4;                 // shared-memory ring of (e, g) tiles
// Each worker-parity warp group has its own kGroupStages of the ring, which it
// reads in order: an mbarrier wait by phase parity can only tell the phase it
// waits for from the one before, so no warp may wait on a stage two phases
// ahead, as it could if the groups shared stages (an odd K, or a ring whose
// size is not twice a group's share).
constexpr int kGroupStages = kStages / 2;
constexpr int kSubTiles = kChunksPerTile;  // 8 sub-tiles of 512 elements
constexpr int kSub = kT / kSubTiles;       // 512
constexpr int kConsumers = 2 * kSubTiles;  // warps 0..15: sub-tile w & 7, workers of parity w >> 3
constexpr int kGLen = kT + 8;              // g stage: up to 3 leading floats of misalignment
constexpr int kProducer = kConsumers;      // warp 16
constexpr int kThreadsAll = (kConsumers + 1) * 32;
struct Smem {
  float e[kStages][kT];
  float g[kStages][kGLen];
  float dl[kSubTiles][kSub];               // w_t - w_{t-1} of a sub-tile
  uint32_t mk[kSubTiles][kSub];            // senders of the pending aggregation (bit k)
  uint8_t own[kConsumers][32];             // scratch of each consumer warp: worker of each listed pair
  uint32_t upos[kSubTiles][32];            // union coordinates of a sub-tile, one per lane
  uint32_t pflag[kSubTiles];               // per sub-tile: more than 32 pairs (per-element masks)
  uint64_t full[kStages];                  // e, g landed (1 arrival + tx bytes)
  uint64_t empty[kStages];                 // all consumer warps read the stage (8 arrivals)
  int32_t gmeta[kStages];                  // leading floats in the g stage, -1 = not copied
  uint32_t theta[kMaxK];
  uint32_t Tp[kMaxK], tip[kMaxK];          // the previous step's selection (T, t_idx) per worker
  uint32_t tq[16];                         // claimed tiles (tile_at)
  uint32_t next[kSubTiles];                // per sub-tile: the next tile of its two warps
  // followed by the candidate staging lines: per consumer warp and worker, 32
  // indices then 32 values (staging_bytes)
};
// Tiles: a CTA's first F fixed, the rest claimed F - 1 tiles ahead of the
// producer's start of the tile before it (tile_claim_n publishes the claim of
// tile n - 1 into slot n - 1 + F when it starts tile n). Only the lead warp of
// a sub-tile (it has worker 0's items) reads the queue; the earliest read of a
// slot is that of tile n + D (D: the pipeline's depth, 3 or 1) during tile n,
// after it waited on an item of tile n - 1, whose issue followed the
// producer's publishing of slots up to n - 2 + F: so F = D + 2. The producer
// runs at most kStages items (tiles, for K <= 2) ahead of the slowest consumer.
constexpr int kFixedDeep = 5;     // K <= kDeepMaxK: depth 3
constexpr int kFixedShallow = 3;  // more workers: depth 1
constexpr int kDeepMaxK = 5;      // from K = 6 the lead warp has three items a tile or more
constexpr int kQ = 16;
static_assert(kQ > kStages + kFixedDeep, "the producer may overwrite a claimed tile not yet read");
// Dynamic shared memory of the bulk pass for K workers.
__host__ __device__ constexpr int smem_bytes(int K) {
  return (int)((sizeof(Smem) + 127) / 128 * 128) + kSubTiles * K * 64 * 4;
}
static_assert(smem_bytes(kBulkMaxK) <= 232448, "bulk pass shared memory above the 227 KB a block may use");

// The first (up to 32) sent pairs of one sub-tile of the previous step, lane e
// holding pair e of the list that runs through the workers in ascending order.
struct Pairs {
  uint32_t j;      // coordinate, or kNone
  float v;         // value
  int kw;          // worker
  uint32_t total;  // pairs in the sub-tile (warp-uniform)
};
}  // namespace bulk

// Sub-chunk entry (k = lane, tile, w) of the previous step, or none.
__device__ __forceinline__ uint2 pipe_chunk(const TopkArgs& A, int64_t tile, int w, int lane) {
  return (A.has_prev && tile < A.n_tiles && lane < A.K) ? A.chunk_prev[chunk_at(A, lane, tile, w)]
                                                         : make_uint2(0u, 0u);
}

// Issue the loads of a sub-tile's first 32 pairs from its sub-chunk entries.
__device__ __forceinline__ bulk::Pairs pipe_pairs(const TopkArgs& A, uint2 cb, uint8_t* own, int lane) {
  bulk::Pairs P;
  const uint32_t pre = warp_excl_scan(cb.y, &P.total);
  for (uint32_t i = 0; i < cb.y && pre + i < 32u; ++i) own[pre + i] = (uint8_t)lane;
  __syncwarp();
  const bool has = (uint32_t)lane < P.total;
  const int src = has ? own[lane] : 0;
  __syncwarp();
  const uint32_t b = __shfl_sync(0xffffffffu, cb.x, src);
  const uint32_t p = __shfl_sync(0xffffffffu, pre, src);
  P.j = kNone;
  P.v = 0.f;
  P.kw = src;
  const uint32_t at = b + ((uint32_t)lane - p);
  if (has && at < A.cap) {
    const int64_t q = (int64_t)src * A.cap + at;
    P.j = A.cand_idx_prev[q];
    P.v = A.cand_val_prev[q];
  }
  return P;
}

// The pair was sent: selected under its worker's selection of the previous step.
__device__ __forceinline__ bool pair_sent(const bulk::Pairs& P, const uint32_t* Tp, const uint32_t* tip) {
  return P.j != kNone && selected(mag_key(P.v), P.j, Tp[P.kw], tip[P.kw]);
}

// Issue the load of w (pending aggregation) or of w_t - w_{t-1} (applied) at a sent pair.
__device__ __forceinline__ float pipe_w(const TopkArgs& A, const bulk::Pairs& P, const uint32_t* Tp,
                                        const uint32_t* tip) {
  if (!pair_sent(P, Tp, tip) || P.j >= (uint32_t)A.d) return 0.f;
  return A.pending ? A.w[P.j] : A.dlt[P.j];
}

// A sub-tile's w_t - w_{t-1} into dlw and the pending senders into mkw from
// its pairs (all of them: total <= 32) and the loaded wv. Pending
// aggregation (Alg. 1, last line): the senders' values summed in ascending
// worker order from +0, w_{t+1} = w_t - a * sum written over w, and
// Δ = w_{t+1} - w_t. Applied before: Δ was left in dlt; read, then cleared.
// Returns the union coordinate this lane listed (its first sender), or ~0u.
__device__ __forceinline__ uint32_t apply_pairs(const TopkArgs& A, uint32_t sub0, const bulk::Pairs& P,
                                                const uint32_t* Tp, const uint32_t* tip, float wv,
                                                float* dlw, uint32_t* mkw, int lane, uint32_t lt,
                                                uint32_t& uni, uint32_t& chg) {
  using bulk::kSub;
  for (int i = lane; i < kSub / 4; i += 32) {
    reinterpret_cast<float4*>(dlw)[i] = make_float4(0.f, 0.f, 0.f, 0.f);
    reinterpret_cast<uint4*>(mkw)[i] = make_uint4(0u, 0u, 0u, 0u);
  }
  __syncwarp();
  bool act = false;
  uint32_t l = 0;
  if (pair_sent(P, Tp, tip)) {
    const int64_t ll = (int64_t)P.j - sub0;
    if (ll >= 0 && ll < kSub) {
      act = true;
      l = (uint32_t)ll;
    } else {
      atomicOr(A.status, kStatusInternal);
    }
  }
  const bool first = act && atomicOr(&mkw[l], 1u << P.kw) == 0u;  // the coordinate's first sender
  if (A.pending) {
    // lanes holding the same coordinate add one at a time, in lane (= worker) order
    const uint32_t peers = __match_any_sync(0xffffffffu, act ? (int)l : -1 - lane);
    const uint32_t rk = __popc(peers & lt);
    const uint32_t rmax = __reduce_max_sync(0xffffffffu, act ? rk : 0u);
    for (uint32_t turn = 0; turn <= rmax; ++turn) {
      if (act && rk == turn) dlw[l] = __fadd_rn(dlw[l], P.v);
      __syncwarp();
    }
  }
  __syncwarp();
  if (first) {
    if (A.pending) {
      const float wn = __fsub_rn(wv, __fmul_rn(A.a_prev, dlw[l]));
      A.w[P.j] = wn;
      const float dd = __fsub_rn(wn, wv);
      dlw[l] = dd;
      ++uni;
      chg += dd != 0.f;
    } else {
      dlw[l] = wv;          // w_t - w_{t-1}, read once
      A.dlt[P.j] = 0.f;     // and cleared: this step's aggregate writes the next one
    }
  }
  __syncwarp();
  return first ? l : ~0u;
}

template <bool kLocal, bool kBf16>
__global__ void __launch_bounds__(bulk::kThreadsAll, 1) k_accumulate_bulk(TopkArgs A) {
  griddep_wait();
  using namespace bulk;
  extern __shared__ __align__(128) unsigned char smem_raw[];
  Smem& sm = *reinterpret_cast<Smem*>(smem_raw);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // the lead warp's pipeline spans three tiles: for few workers, and for the
  // bf16 and local-momentum forms, where the one-tile pipeline measured slower
  // (vgg16_bf16 1.98 -> 1.93 ms, vgg16_local 3.51 -> 3.45 ms with it spanning three)
  const bool deep = (kLocal || kBf16) ? true : A.K <= kDeepMaxK;
  const uint32_t F = deep ? kFixedDeep : kFixedShallow;
  const uint32_t* order = A.use_order ? A.blk_order : nullptr;  // the tiles' order (tile_order)
  const uint32_t G = gridDim.x, nbw = (uint32_t)(A.n_tiles / G);  // whole blocks of G tiles
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&sm.full[s], 1);
      mbar_init(&sm.empty[s], kSubTiles);  // the eight warps of the stage's worker parity
    }
    fence_mbar_init();
  }
  for (int kk = threadIdx.x; kk < kMaxK; kk += blockDim.x) {
    sm.theta[kk] = kk < A.K ? A.sel[kk].theta : kNoCandidate;
    sm.Tp[kk] = kk < A.K ? A.sel[kk].T : 0u;  // this step's select runs after this pass
    sm.tip[kk] = kk < A.K ? A.sel[kk].t_idx : 0u;
  }
  __syncthreads();

  if (warp == kProducer) {
    // ---- producer ----
    if (lane != 0) return;
    // gradient rows of es-byte elements (fp32, or bf16 from gmc_step_bf16)
    constexpr int es = kBf16 ? 2 : 4;
    const char* g_lo = kBf16 ? reinterpret_cast<const char*>(A.grads16) : reinterpret_cast<const char*>(A.grads);
    const char* g_hi = g_lo + (int64_t)A.K * A.d * es;
    uint32_t issued[2] = {0u, 0u};  // items issued to each worker-parity group
    uint32_t held = ~0u;            // test hook: (group << 31) | count of the item not copied
    uint32_t claim = 0;
    bool ok = true;
    for (uint32_t n = 0; ok; ++n) {
      const int64_t tile =
          tile_order(tile_claim_n<kQ>(sm.tq, n, F, A.tile_ctr, claim, A.n_tiles), A.n_tiles, order);
      if (tile >= A.n_tiles) break;
      const int64_t j0 = tile * kT;
      const int64_t nvalid = A.d - j0 < kT ? A.d - j0 : kT;
      for (int k = 0; k < A.K; ++k) {
        const uint32_t grp = (uint32_t)k & 1u, c = issued[grp];
        const uint32_t s = grp * kGroupStages + c % kGroupStages, r = c / kGroupStages;
        if (r > 0 && !wait_bounded(&sm.empty[s], (r - 1) & 1, A.wait_ns)) {
          ok = false;
          break;
        }
        issued[grp] = c + 1;
        if (tile == A.hold_tile && k == A.hold_k) {  // the stage's phase never completes
          held = (grp << 31) | c;
          continue;
        }
        const float* esrc = A.e + (int64_t)k * A.ld + j0;
        const uintptr_t ga = reinterpret_cast<uintptr_t>(g_lo + ((int64_t)k * A.d + j0) * es);
        const uint32_t off = (uint32_t)(ga & 15) / es;  // leading elements before the row's tile
        const char* gsrc = reinterpret_cast<const char*>(ga - off * es);
        const uint32_t gbytes = (uint32_t)(((nvalid + off) * es + 15) & ~int64_t(15));
        const bool gbulk = !A.g_direct && (ga % es) == 0 && gsrc >= g_lo && gsrc + gbytes <= g_hi;
        sm.gmeta[s] = gbulk ? (int32_t)off : -1;
        mbar_arrive_expect_tx(&sm.full[s], kT * 4 + (gbulk ? gbytes : 0));
        bulk_load(sm.e[s], esrc, kT * 4, &sm.full[s]);
        if (gbulk) bulk_load(sm.g[s], gsrc, gbytes, &sm.full[s]);
      }
    }
    if (!ok) atomicOr(A.status, kStatusTimeout);
    // Every copy issued lands before the CTA's shared memory goes away, even
    // when the consumers gave up on their waits: the last kGroupStages items
    // of each group (the earlier ones were read, as their stages' empty
    // barriers showed) read valid global memory and complete without any
    // other warp's help. No later phase is armed on their stages, so each
    // parity wait is for exactly that copy.
    for (uint32_t grp = 0; grp < 2; ++grp) {
      const uint32_t c1 = issued[grp], c0 = c1 > (uint32_t)kGroupStages ? c1 - kGroupStages : 0u;
      for (uint32_t c = c0; c < c1; ++c)
        if (((grp << 31) | c) != held &&
            !wait_bounded(&sm.full[grp * kGroupStages + c % kGroupStages], (c / kGroupStages) & 1, kWaitLimitNs))
          atomicOr(A.status, kStatusTimeout | kStatusInternal);
    }
    return;
  }

  // ---- consumers ----
  const uint32_t lt = lanemask_lt();
  const int sw = warp & (kSubTiles - 1);  // sub-tile
  const int gp = warp / kSubTiles;         // workers k = gp, gp + 2, ...
  float* dlw = sm.dl[sw];
  uint32_t* mkw = sm.mk[sw];
  uint8_t* own = sm.own[warp];
  // the sub-tile's part of the CTA's region, per worker: slots [part0, part0 + cap_part);
  // lane k counts worker k's candidates so far
  const uint32_t part0 = (blockIdx.x * kSubTiles + sw) * A.cap_part;
  uint32_t* stg = reinterpret_cast<uint32_t*>(smem_raw + (sizeof(Smem) + 127) / 128 * 128) +
                  sw * A.K * 64;
  uint32_t run = 0;
  uint32_t taken = 0;  // items of this warp's group read so far (its stages, in order)
  uint32_t nonfinite = 0, uni = 0, chg = 0;
  bool ok = true;  // false after a bounded wait gave up: the items are skipped, the tile loop
                   // still runs (its named barriers need both warps of the sub-tile)
  // The sub-tile's w_t - w_{t-1} is formed by one of its two warps, the lead
  // (the warp of the even workers), from the pairs pc and w at them wc of its
  // tile, which it loaded while working on the tiles before (see above):
  // deep, pn and cx are the pairs of tile n + 1 and the entries of tile n + 2;
  // shallow, cx, pn and wn are the entries, pairs and w of tile n + 1.
  const bool lead = gp == 0;
  // the CTA's n-th tile (tile_order)
  auto tile_n = [&](uint32_t n) { return tile_order(tile_at_n<kQ>(sm.tq, n, F), A.n_tiles, order); };
  Pairs pc{kNone, 0.f, 0, 0u}, pn{kNone, 0.f, 0, 0u};
  float wc = 0.f;
  uint2 cx = make_uint2(0u, 0u);
  if (lead) {  // fill: the first tiles' chains
    pc = pipe_pairs(A, pipe_chunk(A, tile_n(0), sw, lane), own, lane);
    if (deep) pn = pipe_pairs(A, pipe_chunk(A, tile_n(1), sw, lane), own, lane);
    wc = pipe_w(A, pc, sm.Tp, sm.tip);
    if (deep) cx = pipe_chunk(A, tile_n(2), sw, lane);
  }
  const uint32_t pair_bar = 1 + sw;  // named barrier of the sub-tile's two warps
  // The sub-tile's two warps take their next tile from one read of its
  // queue slot (sm.next), so that both leave the loop together: the named
  // barriers need both. A warp whose wait gave up ends the CTA's tiles.
  int64_t tile = tile_n(0);
  for (uint32_t n = 0; tile < A.n_tiles; ++n) {  // n: tiles done
    const uint32_t s0 = (uint32_t)(tile * kT) + sw * kSub;
    // this sub-tile's w_t - w_{t-1}, and the pending senders (their residual
    // is +0): at most 32 union coordinates, one per lane (upos, umask), are
    // zeroed in each worker's stage before it is read; more use per-element masks
    if (lead) {
      uint32_t up = ~0u;
      bool many = false;
      if (A.dense_prev) {  // restored state: no pairs, w_t - w_{t-1} read densely
        stage_delta_dense(A, s0, kSub, dlw, lane);
      } else if (pc.total <= 32u) {
        up = apply_pairs(A, s0, pc, sm.Tp, sm.tip, wc, dlw, mkw, lane, lt, uni, chg);
      } else if (A.pending) {
        stage_pending_warp(A, tile, sw, s0, kSub, dlw, mkw, lane, uni, chg);
        many = true;
      } else {
        stage_delta_warp(A, tile, sw, s0, kSub, dlw, lane);
      }
      sm.upos[sw][lane] = up;
      if (lane == 0) sm.pflag[sw] = many ? 1u : 0u;
    }
    asm volatile("bar.sync %0, 64;" ::"r"(pair_bar) : "memory");
    const bool many = sm.pflag[sw] != 0u;
    const uint32_t upos = sm.upos[sw][lane];
    const uint32_t umask = (A.pending && upos != ~0u) ? mkw[upos] : 0u;
    const bool patch = __any_sync(0xffffffffu, umask != 0u);
    float4 dl4[kSub / 128];
#pragma unroll
    for (int u = 0; u < kSub / 128; ++u) dl4[u] = *reinterpret_cast<const float4*>(dlw + u * 128 + lane * 4);
    if (lead && lane == 0)  // the slot of tile n + 1 was published before tile n - 3's items
      sm.next[sw] = (!ok || n + 1 >= (uint64_t)A.n_tiles) ? (uint32_t)A.n_tiles
                                                          : (uint32_t)tile_n(n + 1);
    // the lead warp rewrites the sub-tile's buffers for the next tile only after this
    asm volatile("bar.sync %0, 64;" ::"r"(pair_bar) : "memory");
    float wn = 0.f;
    Pairs pnn{kNone, 0.f, 0, 0u};
    uint2 cxn = make_uint2(0u, 0u);
    if (lead) {  // the next tiles' loads, in flight while this tile is processed
      if (deep) {
        wn = pipe_w(A, pn, sm.Tp, sm.tip);
        pnn = pipe_pairs(A, cx, own, lane);
        cxn = pipe_chunk(A, tile_n(n + 3), sw, lane);
      } else {
        cx = pipe_chunk(A, tile_n(n + 1), sw, lane);
      }
    }
    uint32_t item = 0;  // this warp's items of the tile so far
    const int64_t rem = A.d - (int64_t)s0;
    const int lim = rem < kSub ? (int)rem : kSub;
    // candidate flags of this lane's 16 values (bit 4u + i: value u*128 + lane*4 + i)
    uint32_t valid = 0;
#pragma unroll
    for (int u = 0; u < kSub / 128; ++u)
#pragma unroll
      for (int i = 0; i < 4; ++i) valid |= (u * 128 + lane * 4 + i < lim ? 1u : 0u) << (4 * u + i);
    uint2 bc_lane = make_uint2(0u, 0u);
    uint32_t tcnt = 0;  // this warp's candidates of the tile (the block's cost, tile_order)
    for (int k = gp; ok && k < A.K; k += 2) {
      const uint32_t s = gp * kGroupStages + taken % kGroupStages, r = taken / kGroupStages;
      ++taken;
      float4 mv[kSub / 128];  // the local-momentum baseline: m loaded while the stage lands
      if (kLocal) {
#pragma unroll
        for (int u = 0; u < kSub / 128; ++u)
          mv[u] = __ldcs(reinterpret_cast<const float4*>(A.lm + (int64_t)k * A.ld + s0 + u * 128 + lane * 4));
      }
      if (!__all_sync(0xffffffffu, wait_bounded(&sm.full[s], r & 1, A.wait_ns))) {  // warp-uniform
        ok = false;
        break;
      }
      const int32_t off = sm.gmeta[s];
      float* se = sm.e[s] + sw * kSub;
      const float* sg = sm.g[s] + (off > 0 ? off : 0) + sw * kSub;
      if (patch) {
        if ((umask >> k) & 1u) {
          se[upos] = 0.f;
          fence_proxy_async();  // before the stage is refilled by the bulk copy
        }
        __syncwarp();
      }
      float v[kSub / 128][4];
#pragma unroll
      for (int u = 0; u < kSub / 128; ++u) {
        const int l = u * 128 + lane * 4;
        float4 e4 = *reinterpret_cast<const float4*>(se + l);
        float4 g4;
        if constexpr (kBf16) {
          if (off >= 0)
            g4 = bf16x4(reinterpret_cast<const uint16_t*>(sm.g[s]) + off + sw * kSub + l);
          else
            g4 = load_g4_bf16(A.grads16 + (int64_t)k * A.d, (int64_t)s0 + l, A.d);
        } else if (off == 0) {
          g4 = *reinterpret_cast<const float4*>(sg + l);
        } else if (off == 2) {
          const float2 a = *reinterpret_cast<const float2*>(sg + l);
          const float2 b = *reinterpret_cast<const float2*>(sg + l + 2);
          g4 = make_float4(a.x, a.y, b.x, b.y);
        } else if (off > 0) {
          g4 = make_float4(sg[l], sg[l + 1], sg[l + 2], sg[l + 3]);
        } else {
          const float* gk = A.grads + (int64_t)k * A.d;
          g4 = load_g4(gk, (int64_t)s0 + l, A.d, g_mode(gk));
        }
        if (lim < kSub && off >= 0) {  // past d the stage holds bytes of no meaning
          if (l >= lim) g4.x = 0.f;
          if (l + 1 >= lim) g4.y = 0.f;
          if (l + 2 >= lim) g4.z = 0.f;
          if (l + 3 >= lim) g4.w = 0.f;
        }
        g4 = scale_g(A, g4);
        if (kLocal) g4 = local_m4(A, A.lm + (int64_t)k * A.ld + s0 + l, mv[u], g4);
        if (many) {  // more union coordinates than lanes: per-element sender masks
          const uint4 m4 = *reinterpret_cast<const uint4*>(mkw + l);
          if ((m4.x >> k) & 1u) e4.x = 0.f;
          if ((m4.y >> k) & 1u) e4.y = 0.f;
          if ((m4.z >> k) & 1u) e4.z = 0.f;
          if ((m4.w >> k) & 1u) e4.w = 0.f;
        }
        const float4 d4 = dl4[u];
        v[u][0] = accumulate(e4.x, g4.x, A.c, d4.x);
        v[u][1] = accumulate(e4.y, g4.y, A.c, d4.y);
        v[u][2] = accumulate(e4.z, g4.z, A.c, d4.z);
        v[u][3] = accumulate(e4.w, g4.w, A.c, d4.w);
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&sm.empty[s]);  // this warp is done reading stage s
      // candidates: |v| >= theta, or NaN (its key is above every threshold);
      // theta is at most the Inf key, or kNoCandidate for none
      const uint32_t th = sm.theta[k];
      const float tf = __uint_as_float(th);
      float* ekt = A.e + (int64_t)k * A.ld + s0;
      uint32_t bits = 0;
#pragma unroll
      for (int u = 0; u < kSub / 128; ++u) {
        const int l = u * 128 + lane * 4;
        __stcs(reinterpret_cast<float4*>(ekt + l), make_float4(v[u][0], v[u][1], v[u][2], v[u][3]));
#pragma unroll
        for (int i = 0; i < 4; ++i) bits |= (!(fabsf(v[u][i]) < tf) ? 1u : 0u) << (4 * u + i);
      }
      bits &= th == kNoCandidate ? 0u : valid;
      const uint32_t cnt = __reduce_add_sync(0xffffffffu, __popc(bits));
      tcnt += cnt;
      const uint32_t run_k = __shfl_sync(0xffffffffu, run, k);  // worker k's candidates so far
      if (cnt) {
        if (lane == 0 && run_k + cnt > A.cap_part) A.sel[k].dense = 1;  // part full: dense path
        // rank in index order (group u, then lane, then value): the four
        // groups' counts, one byte each, scanned over the lanes at once
        uint32_t packed = 0;
#pragma unroll
        for (int u = 0; u < kSub / 128; ++u) packed |= (uint32_t)__popc((bits >> (4 * u)) & 0xfu) << (8 * u);
        uint32_t incl = packed;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const uint32_t y = __shfl_up_sync(0xffffffffu, incl, o);
          if (lane >= o) incl += y;
        }
        const uint32_t tot = __shfl_sync(0xffffffffu, incl, 31);
        const uint32_t excl = incl - packed;
        uint32_t gbase[kSub / 128];  // rank of the lane's first candidate in each group
        uint32_t acc = run_k;
#pragma unroll
        for (int u = 0; u < kSub / 128; ++u) {
          gbase[u] = acc + ((excl >> (8 * u)) & 0xffu);
          acc += (tot >> (8 * u)) & 0xffu;
        }
        uint32_t* ci = A.cand_idx + (int64_t)k * A.cap + part0;
        float* cv = A.cand_val + (int64_t)k * A.cap + part0;
        uint32_t* si = stg + k * 64;
        float* sv = reinterpret_cast<float*>(si + 32);
        const uint32_t end = run_k + cnt;
        for (uint32_t line = run_k >> 5; line <= (end - 1) >> 5; ++line) {
#pragma unroll
          for (int u = 0; u < kSub / 128; ++u) {
            uint32_t o = gbase[u];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              if ((bits >> (4 * u + i)) & 1u) {
                if ((o >> 5) == line && o < A.cap_part) {
                  si[o & 31] = s0 + u * 128 + lane * 4 + i;
                  sv[o & 31] = v[u][i];
                }
                ++o;
              }
            }
          }
          __syncwarp();
          const uint32_t line_end = (line + 1) * 32;
          if (line_end <= end && line_end <= A.cap_part) {  // a whole line: one coalesced store per array
            const float x = sv[lane];
            ci[line * 32 + lane] = si[lane];
            cv[line * 32 + lane] = x;
            nonfinite += is_nonfinite(x) ? 1u : 0u;
            atomicAdd(&A.chist[(int64_t)k * kRelBins + rel_bin(mag_key(x), th, A.sel_shift)], 1u);
          }
          __syncwarp();
        }
        if (lane == k) run += cnt;
      }
      if (lane == k) bc_lane = make_uint2(part0 + run_k, cnt);
      if (lead && !deep) {  // the next tile's chain, one link per item
        if (item == 0) pn = pipe_pairs(A, cx, own, lane);
        else if (item == 1) wn = pipe_w(A, pn, sm.Tp, sm.tip);
      }
      ++item;
    }
    if (lead && !deep && item < 2) {  // a wait gave up before the chain was complete
      if (item == 0) pn = pipe_pairs(A, cx, own, lane);
      wn = pipe_w(A, pn, sm.Tp, sm.tip);
    }
    // the tile's sub-chunk entries of this warp's workers: lane k holds worker k's
    if (ok && lane < A.K && (lane & 1) == gp) A.chunk[chunk_at(A, lane, tile, sw)] = bc_lane;
    if (A.blk_cost && lane == 0 && tcnt && tile < (int64_t)nbw * G) atomicAdd(&A.blk_cost[tile / G], tcnt);
    if (lead) {
      pc = pn;
      wc = wn;
      if (deep) {
        pn = pnn;
        cx = cxn;
      }
    }
    // the per-element masks of a many-sender sub-tile stay in use until both warps are done
    if (many) asm volatile("bar.sync %0, 64;" ::"r"(pair_bar) : "memory");
    tile = (int64_t)sm.next[sw];  // written before this tile's second barrier, rewritten after the next one's first
  }
  if (!ok) atomicOr(A.status, kStatusTimeout);
  if (A.pending) {  // the previous step's counts, straight into the totals
    const uint32_t u_w = __reduce_add_sync(0xffffffffu, uni);
    const uint32_t c_w = __reduce_add_sync(0xffffffffu, chg);
    if (lane == 0 && u_w) atomicAdd(&A.total_ctr->v[kUnion], (unsigned long long)u_w);
    if (lane == 0 && c_w) atomicAdd(&A.total_ctr->v[kChanged], (unsigned long long)c_w);
  }
  // the staged tail of each worker's part, and the part's count
  for (int k = gp; k < A.K; k += 2) {
    const uint32_t run_k = __shfl_sync(0xffffffffu, run, k);
    const uint32_t line = run_k >> 5;
    if (run_k <= A.cap_part && (uint32_t)lane < (run_k & 31)) {
      const uint32_t* si = stg + k * 64;
      const float x = reinterpret_cast<const float*>(si + 32)[lane];
      A.cand_idx[(int64_t)k * A.cap + part0 + line * 32 + lane] = si[lane];
      A.cand_val[(int64_t)k * A.cap + part0 + line * 32 + lane] = x;
      nonfinite += is_nonfinite(x) ? 1u : 0u;
      atomicAdd(&A.chist[(int64_t)k * kRelBins + rel_bin(mag_key(x), sm.theta[k], A.sel_shift)], 1u);
    }
  }
  if (nonfinite) {
    atomicOr(A.status, kStatusNonfinite);
    atomicAdd(&A.step_ctr->v[kNonfinite], (unsigned long long)nonfinite);
  }
  if (lane < A.K && (lane & 1) == gp) {
    A.rcount[(int64_t)lane * A.regions * kSubTiles + blockIdx.x * kSubTiles + sw] =
        run < A.cap_part ? run : A.cap_part;
    if (run) atomicAdd(&A.sel[lane].count, run);
  }
}

// ---------------------------------------------------------------------------
// Candidate ranges of a worker, visited one warp per part: the parts of the
// bulk pass (one per CTA and warp), or [0, count) split evenly when the
// candidates share one region. nparts = candidate_parts(A); a warp of a block
// visits parts blockIdx.x * kWarps + warp, then every gridDim.x * kWarps.
// ---------------------------------------------------------------------------
__device__ __forceinline__ int candidate_parts(const TopkArgs& A) {
  return A.regions > 1 ? A.regions * kChunksPerTile : (int)gridDim.x * kWarps;
}
__device__ __forceinline__ void candidate_part(const TopkArgs& A, int k, int p, int nparts,
                                               uint32_t* lo, uint32_t* hi) {
  if (A.regions == 1) {
    const uint32_t cnt = min(A.sel[k].count, A.cap);
    const uint32_t per = ((cnt + nparts - 1) / nparts + 3) & ~3u;
    *lo = min(cnt, (uint32_t)p * per);
    *hi = min(cnt, *lo + per);
  } else {
    *lo = (uint32_t)p * A.cap_part;
    *hi = *lo + A.rcount[(int64_t)k * nparts + p];
  }
}

// ---------------------------------------------------------------------------
// exact select among candidates, two passes:
//   hist    a kRelBins-bin histogram of the candidates' keys above theta, in
//           bins of 2^sel_shift keys (sel_shift is chosen from k so that the
//           k-th key's bin holds about 2048 candidates on smooth data); the
//           last block finds the bin holding the k-th key
//   finish  the candidates of that bin are collected (key, index); the last
//           block ranks them in shared memory: the k-th key T, how many keys
//           equal T are kept, and -- when fewer are kept than there are -- the
//           largest index kept (ties go to the lower index)
// ---------------------------------------------------------------------------
// The candidate histogram of the load/store pass (the bulk pass counts its
// candidates into chist as they leave its staging lines).
__global__ void __launch_bounds__(kThreads) k_select_hist(TopkArgs A) {
  griddep_wait();
  __shared__ uint32_t h[kRelBins];
  const int k = blockIdx.y;
  WorkerSel& S = A.sel[k];
  if (needs_dense(S, A.ksel, A.cap)) return;
  const uint32_t theta = S.theta;
  for (int b = threadIdx.x; b < kRelBins; b += blockDim.x) h[b] = 0;
  __syncthreads();
  const float* cv = A.cand_val + (int64_t)k * A.cap;
  const int nparts = candidate_parts(A);
  const int lane = threadIdx.x & 31;
  for (int part = blockIdx.x * kWarps + (threadIdx.x >> 5); part < nparts; part += gridDim.x * kWarps) {
    uint32_t lo, hi;
    candidate_part(A, k, part, nparts, &lo, &hi);
    for (uint32_t i0 = lo; i0 < hi; i0 += 4 * 32) {
      uint32_t kv[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const uint32_t i = i0 + q * 32 + lane;
        kv[q] = i < hi ? mag_key(cv[i]) : 0xffffffffu;
      }
#pragma unroll
      for (int q = 0; q < 4; ++q) warp_hist_add(h, kv[q] != 0xffffffffu ? rel_bin(kv[q], theta, A.sel_shift) : -1);
    }
  }
  __syncthreads();
  uint32_t* gh = A.chist + (int64_t)k * kRelBins;
  for (int b = threadIdx.x; b < kRelBins; b += blockDim.x)
    if (h[b]) atomicAdd(&gh[b], h[b]);
}

__global__ void __launch_bounds__(kThreads) k_select_finish(TopkArgs A) {
  griddep_wait();
  // kBucketCap keys (the indices stay in the global bucket): 48 KB, so that
  // four blocks fit on an SM and the grid runs in one wave
  extern __shared__ __align__(16) uint32_t fin[];
  __shared__ uint32_t h[kHistBins];
  __shared__ uint32_t ws[32];
  __shared__ uint32_t s_last, s_bin, s_rank, s_n;
  const int k = blockIdx.y;
  WorkerSel& S = A.sel[k];
  if (needs_dense(S, A.ksel, A.cap)) return;
  const uint32_t theta = S.theta;
  // the bin holding the k-th key, and its rank there (every block, from the histogram)
  for (int b = threadIdx.x; b < kRelBins; b += blockDim.x) h[b] = __ldcg(&A.chist[(int64_t)k * kRelBins + b]);
  if (threadIdx.x == 0) {
    s_bin = 0;
    s_rank = 0;
  }
  __syncthreads();
  block_find_from_top(h, kRelBins, A.ksel, ws, &s_bin, &s_rank);
  const int want = (int)s_bin;
  const uint32_t want_rank = s_rank;
  if (want_rank == 0) {  // fewer candidates than k counted: the dense path decides
    if (blockIdx.x == 0 && threadIdx.x == 0) S.dense = 1;
    return;
  }
  const int lane = threadIdx.x & 31;
  const uint32_t lt = lanemask_lt();
  uint32_t* bk = A.bucket + (int64_t)k * 2 * kBucketCap;  // keys, then indices
  const uint32_t* ci = A.cand_idx + (int64_t)k * A.cap;
  const float* cv = A.cand_val + (int64_t)k * A.cap;
  const int nparts = candidate_parts(A);
  // kQ * 32 candidates a round (slots slot[q]), their keys and indices loaded
  // together, one bucket reservation per round
  constexpr int kQ = 8;
  auto collect = [&](const uint32_t (&slot)[kQ], const bool (&in)[kQ]) {
    uint32_t key[kQ], idx[kQ], m[kQ], n = 0;
#pragma unroll
    for (int q = 0; q < kQ; ++q) key[q] = in[q] ? mag_key(cv[slot[q]]) : 0u;
    // the index only of a candidate in the k-th key's bin (about 2,048 of a
    // worker's candidates), loaded while the bucket is reserved: about half
    // the bytes of loading every candidate's index
#pragma unroll
    for (int q = 0; q < kQ; ++q) {
      const bool mine = in[q] && rel_bin(key[q], theta, A.sel_shift) == want;
      idx[q] = mine ? ci[slot[q]] : 0u;
      m[q] = __ballot_sync(0xffffffffu, mine);
      n += __popc(m[q]);
    }
    if (n) {
      uint32_t base = 0;
      if (lane == 0) base = atomicAdd(&S.count_bucket, n);
      base = __shfl_sync(0xffffffffu, base, 0);
#pragma unroll
      for (int q = 0; q < kQ; ++q) {
        const uint32_t o = base + __popc(m[q] & lt);
        if (((m[q] >> lane) & 1u) && o < (uint32_t)kBucketCap) {
          bk[o] = key[q];
          bk[kBucketCap + o] = idx[q];
        }
        base += __popc(m[q]);
      }
    }
  };
  if (A.regions > 1) {
    // bulk path: the warp takes a run of at most 32 consecutive parts, lane l
    // reading the count of part p_lo + l, and walks their candidates as one
    // list (each candidate's part by a binary search over the lanes' counts),
    // so its loads do not wait for one part after another
    const int nw = (int)gridDim.x * kWarps;
    const int per = (nparts + nw - 1) / nw;  // at most 32 (sel_blocks)
    const int p_lo = min(nparts, (int)(blockIdx.x * kWarps + (threadIdx.x >> 5)) * per);
    const int p_hi = min(nparts, p_lo + per);
    const uint32_t cnt = p_lo + lane < p_hi ? A.rcount[(int64_t)k * nparts + p_lo + lane] : 0u;
    uint32_t incl = cnt;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t y = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += y;
    }
    const uint32_t total = __shfl_sync(0xffffffffu, incl, 31);
    for (uint32_t i0 = 0; i0 < total; i0 += kQ * 32) {
      uint32_t slot[kQ];
      bool in[kQ];
#pragma unroll
      for (int q = 0; q < kQ; ++q) {
        const uint32_t i = i0 + q * 32 + lane;
        in[q] = i < total;
        int lo = 0, hi = 32;  // the first lane whose inclusive count exceeds i (six halvings of 32)
#pragma unroll
        for (int it = 0; it < 6; ++it) {
          const int mid = min((lo + hi) >> 1, 31);
          const uint32_t v = __shfl_sync(0xffffffffu, incl, mid);
          if (lo < hi) {
            if (v <= i) lo = mid + 1; else hi = mid;
          }
        }
        const int L = lo < 32 ? lo : 31;
        const uint32_t before = __shfl_sync(0xffffffffu, incl - cnt, L);
        slot[q] = in[q] ? (uint32_t)(p_lo + L) * A.cap_part + (i - before) : 0u;
      }
      collect(slot, in);
    }
  } else {
    for (int part = blockIdx.x * kWarps + (threadIdx.x >> 5); part < nparts; part += gridDim.x * kWarps) {
      uint32_t lo, hi;
      candidate_part(A, k, part, nparts, &lo, &hi);
      for (uint32_t i0 = lo; i0 < hi; i0 += kQ * 32) {
        uint32_t slot[kQ];
        bool in[kQ];
#pragma unroll
        for (int q = 0; q < kQ; ++q) {
          slot[q] = i0 + q * 32 + lane;
          in[q] = slot[q] < hi;
        }
        collect(slot, in);
      }
    }
  }
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) s_last = (atomicAdd(&S.done[1], 1u) == gridDim.x - 1) ? 1u : 0u;
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  if (threadIdx.x == 0) {
    s_n = __ldcg(&S.count_bucket);
    S.count_bucket = 0;
    S.done[1] = 0;
  }
  __syncthreads();
  const uint32_t n = s_n;
  if (n > (uint32_t)kBucketCap) {  // the k-th key's bin is too crowded: the dense path decides
    if (threadIdx.x == 0) S.dense = 1;
    return;
  }
  uint32_t* keys = fin;
  for (uint32_t i = threadIdx.x; i < n; i += blockDim.x) keys[i] = __ldcg(&bk[i]);
  __syncthreads();
  uint32_t n_tie;
  // every key of the bucket lies in the bin `want`: below the top bin its
  // keys are theta + want * 2^s + [0, 2^s), and only those low s bits are ranked
  const bool bounded = want < kRelBins - 1;
  const uint32_t T = bounded ? smem_select_bits(keys, n, want_rank, A.sel_shift,
                                                theta + ((uint32_t)want << A.sel_shift), h, ws, &s_bin,
                                                &s_rank, &n_tie)
                             : smem_select(keys, n, want_rank, h, ws, &s_bin, &s_rank, &n_tie);
  // ties: gather the indices of the keys equal to T over the keys, in place;
  // a round writes below the end of what the block has read so far
  if (threadIdx.x == 0) s_n = 0;
  __syncthreads();
  for (uint32_t i0 = 0; i0 < n; i0 += blockDim.x) {
    const uint32_t i = i0 + threadIdx.x;
    const bool tie = i < n && keys[i] == T;
    const uint32_t j = tie ? __ldcg(&bk[kBucketCap + i]) : 0u;
    __syncthreads();
    if (tie) keys[atomicAdd(&s_n, 1u)] = j;
  }
  __syncthreads();
  const uint32_t ties = s_n;
  uint32_t t_idx = 0xffffffffu;
  if (ties > n_tie) {  // keep the n_tie lowest indices: t_idx = (ties - n_tie + 1)-th largest
    uint32_t unused;
    t_idx = smem_select(keys, ties, ties - n_tie + 1, h, ws, &s_bin, &s_rank, &unused);
  }
  if (threadIdx.x == 0) {
    S.T = T;
    S.n_tie = n_tie;
    S.ties = ties;
    S.t_idx = t_idx;
    // ||C_k||_0: every key sent is >= T; only when T is the zero key are the
    // n_tie ties kept zeros
    atomicAdd(&A.step_ctr->v[kNnz], (unsigned long long)(A.ksel - (T == 0u ? n_tie : 0u)));
  }
}

// ---------------------------------------------------------------------------
// Approximate top-s (Sec. 5.1): the candidates are C(v) itself -- every key
// >= theta, all ties kept. One block per worker records T = theta and the
// count, and counts the pairs and the non-zero ones (zeros are sent only when
// theta is the zero key). More than `limit` candidates, or a part that
// overflowed, leaves the worker to the dense path.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kThreads) k_select_approx(TopkArgs A) {
  griddep_wait();
  __shared__ uint32_t s_zero;
  const int k = blockIdx.y;
  WorkerSel& S = A.sel[k];
  const uint32_t count = S.count;
  if (S.dense || count > A.limit || count > A.cap) {
    if (threadIdx.x == 0) S.dense = 1;
    return;
  }
  const uint32_t T = S.theta;
  if (threadIdx.x == 0) s_zero = 0;
  __syncthreads();
  if (T == 0u) {
    const float* cv = A.cand_val + (int64_t)k * A.cap;
    const int nparts = candidate_parts(A);
    uint32_t z = 0;
    for (int part = threadIdx.x >> 5; part < nparts; part += kWarps) {
      uint32_t lo, hi;
      candidate_part(A, k, part, nparts, &lo, &hi);
      for (uint32_t i = lo + (threadIdx.x & 31); i < hi; i += 32) z += mag_key(cv[i]) == 0u;
    }
    if (z) atomicAdd(&s_zero, z);
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    S.T = T;
    S.t_idx = 0xffffffffu;
    S.n_tie = 0;
    S.nsel = count;
    atomicAdd(&A.step_ctr->v[kPairs], (unsigned long long)count);
    atomicAdd(&A.step_ctr->v[kNnz], (unsigned long long)(count - s_zero));
  }
}

// ---------------------------------------------------------------------------
// dense exact select + chunk rewrite for workers whose filter missed; one
// block per worker (a rare path: correct for any input, not fast). For the
// approximate top-s: every key >= theta when at most `limit` reach it, else
// the exact top-`limit`.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void select_dense_worker(const TopkArgs& A, const int k) {
  WorkerSel& S = A.sel[k];
  if (A.approx ? S.dense == 0 : !needs_dense(S, A.ksel, A.cap)) return;
  __shared__ uint32_t h[kHistBins];
  __shared__ uint32_t ws[32];
  __shared__ unsigned long long ws64[32];
  __shared__ uint32_t s_bin, s_rank;
  __shared__ unsigned long long s_reach;
  const float* vk = A.e + (int64_t)k * A.ld;
  const int64_t d = A.d;
  uint32_t r = A.ksel, prefix = 0;
  uint32_t nsel = A.ksel;
  bool all_ties = false;  // approximate top-s below its limit: T = theta, every tie kept
  unsigned long long reach = 0;  // approximate: (components above theta) << 32 | (equal to it)
  if (A.approx) {
    const uint32_t theta = S.theta;
    unsigned long long x = 0;
    for (int64_t j = threadIdx.x; j < d; j += blockDim.x) {
      const uint32_t key = mag_key(vk[j]);
      x += key > theta ? (1ull << 32) : (key == theta ? 1ull : 0ull);
    }
    unsigned long long tot;
    block_inclusive_scan<unsigned long long>(x, ws64, &tot);
    if (threadIdx.x == 0) s_reach = tot;
    __syncthreads();
    reach = s_reach;
    const unsigned long long n_reach = (reach >> 32) + (reach & 0xffffffffull);
    if (n_reach <= A.limit) {
      all_ties = true;
      nsel = (uint32_t)n_reach;
    } else {
      r = A.limit;
      nsel = A.limit;
    }
  }
  for (int pass = 0; pass < 3 && !all_ties; ++pass) {
    const int nbins = pass == 0 ? 2048 : 1024;
    const int shift = pass == 0 ? 20 : (pass == 1 ? 10 : 0);
    for (int b = threadIdx.x; b < nbins; b += blockDim.x) h[b] = 0;
    if (threadIdx.x == 0) {
      s_bin = 0;
      s_rank = 0;
    }
    __syncthreads();
    for (int64_t j0 = 0; j0 < d; j0 += blockDim.x) {
      const int64_t j = j0 + threadIdx.x;
      int bin = -1;
      if (j < d) {
        const uint32_t key = mag_key(vk[j]);
        if (pass == 0 || (key >> (shift + 10)) == prefix)
          bin = (int)((key >> shift) & (uint32_t)(nbins - 1));
      }
      warp_hist_add(h, bin);
    }
    __syncthreads();
    block_find_from_top(h, nbins, r, ws, &s_bin, &s_rank);
    prefix = pass == 0 ? s_bin : ((prefix << 10) | s_bin);
    r = s_rank;
    __syncthreads();
  }
  const uint32_t T = all_ties ? S.theta : prefix;
  const uint32_t n_tie = all_ties ? 0xffffffffu : r;
  if (all_ties && threadIdx.x == 0) S.t_idx = 0xffffffffu;

  const int P = A.tile / (int)blockDim.x;  // consecutive elements per thread
  const int per_sub = (int)blockDim.x / kChunksPerTile;  // threads per sub-tile
  __shared__ uint32_t sb[kChunksPerTile + 1];
  uint32_t* oi = A.cand_idx + (int64_t)k * A.cap;
  float* ov = A.cand_val + (int64_t)k * A.cap;
  uint32_t running = 0, eqrun = 0;
  for (int64_t tile = 0; tile < A.n_tiles; ++tile) {
    const int64_t j0 = tile * A.tile + (int64_t)threadIdx.x * P;
    uint32_t g = 0, q = 0;
    for (int i = 0; i < P; ++i) {
      const int64_t j = j0 + i;
      if (j < d) {
        const uint32_t key = mag_key(vk[j]);
        g += key > T;
        q += key == T;
      }
    }
    const unsigned long long x = ((unsigned long long)g << 32) | q;
    unsigned long long tot;
    const unsigned long long exc = block_inclusive_scan<unsigned long long>(x, ws64, &tot) - x;
    const uint32_t taken0 = min(eqrun, n_tie);
    uint32_t qg = eqrun + (uint32_t)exc;
    uint32_t o = running + (uint32_t)(exc >> 32) + (min(qg, n_tie) - taken0);
    if (threadIdx.x % per_sub == 0) sb[threadIdx.x / per_sub] = o;
    for (int i = 0; i < P; ++i) {
      const int64_t j = j0 + i;
      if (j < d) {
        const float v = vk[j];
        const uint32_t key = mag_key(v);
        const bool take = key > T || (key == T && qg < n_tie);
        if (key == T && qg + 1 == n_tie) S.t_idx = (uint32_t)j;  // the last tie kept
        if (key == T) ++qg;
        if (take) {
          if (o < nsel && o < A.cap) {
            oi[o] = (uint32_t)j;
            ov[o] = v;
          }
          ++o;
        }
      }
    }
    const uint32_t in_tile = (uint32_t)(tot >> 32) + (min(eqrun + (uint32_t)tot, n_tie) - taken0);
    if (threadIdx.x == 0) sb[kChunksPerTile] = running + in_tile;
    __syncthreads();
    if (threadIdx.x < kChunksPerTile)
      A.chunk[chunk_at(A, k, tile, threadIdx.x)] =
          make_uint2(sb[threadIdx.x], sb[threadIdx.x + 1] - sb[threadIdx.x]);
    running += in_tile;
    eqrun += (uint32_t)tot;
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    if (running != nsel) atomicOr(A.status, kStatusInternal);
    // the sub-chunks now hold exactly C(v), [0, nsel) of the candidate buffer;
    // zeros are sent only when T is the zero key: n_tie of them, or every tie
    const uint32_t zeros = T != 0u ? 0u : (all_ties ? (uint32_t)(reach & 0xffffffffull) : n_tie);
    S.T = T;
    S.n_tie = n_tie;
    S.nsel = nsel;
    S.dense = 1;
    atomicAdd(&A.step_ctr->v[kFallbacks], 1ull);
    atomicAdd(&A.step_ctr->v[kNnz], (unsigned long long)(nsel - zeros));
    if (A.approx) atomicAdd(&A.step_ctr->v[kPairs], (unsigned long long)nsel);
  }
}

// One block per worker. When it is the step's last launch (A.finalize), the
// last block out also adds the step's counters to the totals (k_finalize's
// work, one launch fewer).
__global__ void __launch_bounds__(1024) k_select_dense(TopkArgs A) {
  griddep_wait();
  select_dense_worker(A, blockIdx.x);
  if (!A.finalize) return;
  __shared__ uint32_t s_last;
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    s_last = atomicAdd(&A.sel[0].done[3], 1u) == gridDim.x - 1 ? 1u : 0u;
  }
  __syncthreads();
  if (s_last && threadIdx.x == 0) {
    __threadfence();
    A.sel[0].done[3] = 0;
    finalize_counters(A.step_ctr, A.total_ctr, A.pairs_add);
  }
}

// ---------------------------------------------------------------------------
// aggregate + update, over all candidates in parallel (no per-tile order),
// when it is applied at once (an eager step, or reading the state):
//   mark  a sent candidate sets its worker's bit in the coordinate's mask
//   sum   the sent candidate of the lowest worker in the mask (the owner) adds
//         the workers' values in ascending worker order from +0 -- each value
//         is still in e[k][j], where the accumulate pass wrote it -- sets those
//         e to +0, and applies w -= (eta/K) * sum, keeping w_{t+1} - w_t.
// A candidate is sent iff selected(key, index, T, t_idx) under its worker's
// selection of that step.
// ---------------------------------------------------------------------------
// Candidates of worker k, part p of nparts: the dense path's [0, k) when it
// decided this worker, else a region of the bulk pass or a slice of [0, count).
__device__ __forceinline__ void sent_part(const TopkArgs& A, int k, int p, int nparts,
                                          uint32_t* lo, uint32_t* hi) {
  if (A.sel[k].dense || A.regions == 1) {
    const uint32_t n = A.sel[k].dense ? (A.approx ? A.sel[k].nsel : A.ksel) : min(A.sel[k].count, A.cap);
    const uint32_t per = (n + nparts - 1) / nparts;
    *lo = min(n, (uint32_t)p * per);
    *hi = min(n, *lo + per);
  } else {
    *lo = (uint32_t)p * A.cap_part;
    *hi = *lo + A.rcount[(int64_t)k * nparts + p];
  }
}

__global__ void __launch_bounds__(kThreads) k_mark(TopkArgs A) {
  griddep_wait();
  const int k = blockIdx.y;
  const uint32_t T = A.sel[k].T, tidx = A.sel[k].t_idx;
  const uint32_t bit = 1u << k;
  const uint32_t* ci = A.cand_idx + (int64_t)k * A.cap;
  const float* cv = A.cand_val + (int64_t)k * A.cap;
  const int nparts = candidate_parts(A);
  const int lane = threadIdx.x & 31;
  for (int part = blockIdx.x * kWarps + (threadIdx.x >> 5); part < nparts; part += gridDim.x * kWarps) {
    uint32_t lo, hi;
    sent_part(A, k, part, nparts, &lo, &hi);
    for (uint32_t i0 = lo; i0 < hi; i0 += 4 * 32) {
      uint32_t jq[4];
      float vq[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const uint32_t i = i0 + q * 32 + lane;
        jq[q] = i < hi ? ci[i] : kNone;
        vq[q] = i < hi ? cv[i] : 0.f;
      }
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const uint32_t j = jq[q];
        if (j < (uint32_t)A.d && selected(mag_key(vq[q]), j, T, tidx)) atomicOr(&A.mask[j], bit);
      }
    }
  }
}

__global__ void __launch_bounds__(kThreads) k_owner_sum(TopkArgs A) {
  griddep_wait();
  const int k = blockIdx.y;
  const uint32_t* ci = A.cand_idx + (int64_t)k * A.cap;
  const float* cv = A.cand_val + (int64_t)k * A.cap;
  const uint32_t T = A.sel[k].T, tidx = A.sel[k].t_idx;
  const uint32_t mine = 1u << k, lower = mine - 1u;
  const int nparts = candidate_parts(A);
  unsigned long long uni = 0, changed = 0;
  for (int part = blockIdx.x * kWarps + (threadIdx.x >> 5); part < nparts; part += gridDim.x * kWarps) {
    uint32_t lo, hi;
    sent_part(A, k, part, nparts, &lo, &hi);
    for (uint32_t i = lo + (threadIdx.x & 31); i < hi; i += 32) {
      const uint32_t j = __ldcg(ci + i);
      if (j >= (uint32_t)A.d || !selected(mag_key(__ldcg(cv + i)), j, T, tidx)) continue;  // not sent
      const uint32_t m = A.mask[j];
      if (!(m & mine) || (m & lower)) continue;  // a lower worker owns j (or done)
      // every sender's value is still in e[b][j]: load them all at once, then
      // add in ascending worker order from +0
      const float wo = A.w[j];
      float vals[32];
#pragma unroll
      for (int b = 0; b < 32; ++b)
        vals[b] = ((m >> b) & 1u) ? __ldcg(A.e + (int64_t)b * A.ld + j) : 0.f;
      float sum = 0.f;
#pragma unroll
      for (int b = 0; b < 32; ++b) {
        if ((m >> b) & 1u) {
          sum = __fadd_rn(sum, vals[b]);
          A.e[(int64_t)b * A.ld + j] = 0.f;  // e_{t+1,b} = e_{t+1/2,b} - C(.) = +0 where sent
          if (A.mfm) A.lm[(int64_t)b * A.ld + j] = 0.f;  // momentum factor masking
        }
      }
      A.mask[j] = 0u;
      ++uni;
      if (A.server_mom) {  // Alg. 3: k_server_update applies the sum with the momentum term
        A.dlt[j] = sum;
        continue;
      }
      const float wn = __fsub_rn(wo, __fmul_rn(A.a_prev, sum));
      A.w[j] = wn;
      const float dd = __fsub_rn(wn, wo);
      A.dlt[j] = dd;
      changed += (dd != 0.f);
    }
  }
  uni = warp_sum(uni);
  changed = warp_sum(changed);
  if ((threadIdx.x & 31) == 0) {
    for (Counters* c : {A.step_ctr, A.total_ctr}) {
      if (!c) continue;
      if (uni) atomicAdd(&c->v[kUnion], uni);
      if (changed) atomicAdd(&c->v[kChanged], changed);
    }
  }
}

// Alg. 3, the server with the momentum term, over every coordinate:
// w_{t+1} = (w_t - a*s) + beta*(w_t - w_{t-1}), s the workers' sum (left in
// dlt by the aggregate on the union, +0 elsewhere); then mom = w_{t+1} - w_t
// (what fl(w_{t+1} - w_t) gives the next step) and dlt back to zero.
__global__ void __launch_bounds__(kThreads) k_server_update(TopkArgs A) {
  griddep_wait();
  unsigned long long changed = 0;
  const int64_t n4 = A.d >> 2;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t q = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; q < n4; q += stride) {
    const float4 s4 = __ldcs(reinterpret_cast<const float4*>(A.dlt) + q);
    const float4 w4 = __ldcs(reinterpret_cast<const float4*>(A.w) + q);
    const float4 m4 = __ldcs(reinterpret_cast<const float4*>(A.mom) + q);
    const float s[4] = {s4.x, s4.y, s4.z, s4.w}, wo[4] = {w4.x, w4.y, w4.z, w4.w};
    const float mo[4] = {m4.x, m4.y, m4.z, m4.w};
    float wn[4], mn[4];
    bool nz = false;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      wn[i] = __fadd_rn(__fsub_rn(wo[i], __fmul_rn(A.a, s[i])), __fmul_rn(A.beta, mo[i]));
      mn[i] = __fsub_rn(wn[i], wo[i]);
      changed += mn[i] != 0.f;
      nz |= __float_as_uint(s[i]) != 0u;
    }
    __stcs(reinterpret_cast<float4*>(A.w) + q, make_float4(wn[0], wn[1], wn[2], wn[3]));
    __stcs(reinterpret_cast<float4*>(A.mom) + q, make_float4(mn[0], mn[1], mn[2], mn[3]));
    if (nz) reinterpret_cast<float4*>(A.dlt)[q] = make_float4(0.f, 0.f, 0.f, 0.f);
  }
  for (int64_t j = (n4 << 2) + (int64_t)blockIdx.x * blockDim.x + threadIdx.x; j < A.d; j += stride) {
    const float s = A.dlt[j], wo = A.w[j];
    const float wn = __fadd_rn(__fsub_rn(wo, __fmul_rn(A.a, s)), __fmul_rn(A.beta, A.mom[j]));
    const float mn = __fsub_rn(wn, wo);
    A.w[j] = wn;
    A.mom[j] = mn;
    changed += mn != 0.f;
    if (__float_as_uint(s) != 0u) A.dlt[j] = 0.f;
  }
  changed = warp_sum(changed);
  if ((threadIdx.x & 31) == 0 && changed) atomicAdd(&A.step_ctr->v[kChanged], changed);
}

// (index, value) pairs of worker k's last C(.) in ascending index order: its
// sent candidates, tile by tile, sub-chunk by sub-chunk.
__global__ void __launch_bounds__(1024) k_gather_selected(TopkArgs A, int k, uint32_t* idx_out,
                                                          float* val_out) {
  griddep_wait();
  __shared__ uint32_t ws[32];
  const uint32_t* ci = A.cand_idx + (int64_t)k * A.cap;
  const float* cv = A.cand_val + (int64_t)k * A.cap;
  const uint32_t T = A.sel[k].T, tidx = A.sel[k].t_idx;
  const uint32_t want = A.approx ? A.sel[k].nsel : A.ksel;
  uint32_t carry = 0;
  for (int64_t t0 = 0; t0 < A.n_tiles; t0 += blockDim.x) {
    const int64_t tile = t0 + threadIdx.x;
    uint32_t cnt = 0;
    if (tile < A.n_tiles) {
      for (int w = 0; w < kChunksPerTile; ++w) {
        const uint2 bc = A.chunk[chunk_at(A, k, tile, w)];
        const uint32_t base = bc.x, n = bc.y;
        for (uint32_t i = 0; i < n && base + i < A.cap; ++i)
          cnt += selected(mag_key(cv[base + i]), ci[base + i], T, tidx) ? 1u : 0u;
      }
    }
    uint32_t tot;
    uint32_t pos = carry + block_inclusive_scan<uint32_t>(cnt, ws, &tot) - cnt;
    if (cnt) {
      for (int w = 0; w < kChunksPerTile; ++w) {
        const uint2 bc = A.chunk[chunk_at(A, k, tile, w)];
        const uint32_t base = bc.x, n = bc.y;
        for (uint32_t i = 0; i < n && base + i < A.cap; ++i) {
          const uint32_t j = ci[base + i];
          if (!selected(mag_key(cv[base + i]), j, T, tidx)) continue;
          if (pos < want) {
            idx_out[pos] = j;
            val_out[pos] = cv[base + i];
          }
          ++pos;
        }
      }
    }
    carry += tot;
  }
  if (threadIdx.x == 0 && carry != want) atomicOr(A.status, kStatusInternal);
}

int tile_u(int tile) { return tile / (kWarps * 128); }

bool use_bulk(int tile) { return tile == bulk::kT; }

}  // namespace

// Dynamic shared memory of the accumulate pass for tiles of `tile` and K workers.
int accumulate_smem_bytes(int tile, int K) {
  return use_bulk(tile) ? bulk::smem_bytes(K) : tile * 12;
}

cudaError_t configure_topk_kernels() {
  cudaError_t err = cudaSuccess;
  auto set = [&](const void* f, int bytes) {
    const cudaError_t e2 = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (err == cudaSuccess) err = e2;
  };
  set((const void*)k_accumulate<1, false, false>, 1024 * 12);
  set((const void*)k_accumulate<2, false, false>, 2048 * 12);
  set((const void*)k_accumulate<4, false, false>, 4096 * 12);
  set((const void*)k_accumulate<1, true, false>, 1024 * 12);
  set((const void*)k_accumulate<2, true, false>, 2048 * 12);
  set((const void*)k_accumulate<4, true, false>, 4096 * 12);
  set((const void*)k_accumulate<1, false, true>, 1024 * 12);
  set((const void*)k_accumulate<2, false, true>, 2048 * 12);
  set((const void*)k_accumulate<4, false, true>, 4096 * 12);
  set((const void*)k_accumulate<1, true, true>, 1024 * 12);
  set((const void*)k_accumulate<2, true, true>, 2048 * 12);
  set((const void*)k_accumulate<4, true, true>, 4096 * 12);
  set((const void*)k_accumulate_bulk<false, false>, bulk::smem_bytes(kBulkMaxK));
  set((const void*)k_accumulate_bulk<true, false>, bulk::smem_bytes(kBulkMaxK));
  set((const void*)k_accumulate_bulk<false, true>, bulk::smem_bytes(kBulkMaxK));
  set((const void*)k_accumulate_bulk<true, true>, bulk::smem_bytes(kBulkMaxK));
  set((const void*)k_select_finish, kBucketCap * 4);
  set((const void*)k_sample_theta, kBucketCap * 4);
  return err;
}

int select_blocks_per_sm() {
  int n = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, k_select_finish, kThreads, kBucketCap * 4) != cudaSuccess)
    cudaGetLastError();
  return n > 0 ? n : 1;
}

int accumulate_blocks_per_sm(int tile) {
  if (use_bulk(tile)) return 1;  // one persistent CTA per SM
  int n = 0;
  const int smem = accumulate_smem_bytes(tile, kMaxK);
  switch (tile_u(tile)) {
    case 1: cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, k_accumulate<1, false, false>, kThreads, smem); break;
    case 2: cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, k_accumulate<2, false, false>, kThreads, smem); break;
    default: cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, k_accumulate<4, false, false>, kThreads, smem); break;
  }
  return n > 0 ? n : 1;
}

cudaError_t launch_sample(const TopkArgs& A, cudaStream_t s) {
  if ((A.pending || A.approx) && !A.dense_mode) {
    const int n_s = (int)A.n_sample;
    const unsigned grid = (unsigned)((n_s + kThreads - 1) / kThreads) + (A.use_order ? 1u : 0u);
    const cudaError_t err = launch_pdl(k_sample_pending, dim3(grid), dim3(kThreads), 0, s, A);
    if (err != cudaSuccess) return err;
  }
  if (!A.approx) return launch_pdl(k_sample_cluster, dim3(scl::kCtas, A.K), dim3(scl::kThreadsC), 0, s, A);
  const cudaError_t err = launch_pdl(k_sample, dim3(A.sample_blocks, A.K), dim3(kThreads), 0, s, A);
  if (err != cudaSuccess || !A.approx) return err;
  return launch_pdl(k_sample_theta, dim3(A.theta_blocks, A.K), dim3(kThreads), kBucketCap * 4, s, A);
}

// The load/store pass's instantiation for the step's form and gradient type.
template <int U>
cudaError_t launch_ls(const TopkArgs& A, int grid, int smem, cudaStream_t s) {
  if (A.local_mom && A.bf16) return launch_pdl(k_accumulate<U, true, true>, dim3(grid), dim3(kThreads), smem, s, A);
  if (A.local_mom) return launch_pdl(k_accumulate<U, true, false>, dim3(grid), dim3(kThreads), smem, s, A);
  if (A.bf16) return launch_pdl(k_accumulate<U, false, true>, dim3(grid), dim3(kThreads), smem, s, A);
  return launch_pdl(k_accumulate<U, false, false>, dim3(grid), dim3(kThreads), smem, s, A);
}

cudaError_t launch_accumulate(const TopkArgs& A, int grid, cudaStream_t s) {
  const int smem = accumulate_smem_bytes(A.tile, A.K);
  if (use_bulk(A.tile)) {
    const dim3 g(grid), b(bulk::kThreadsAll);
    if (A.local_mom && A.bf16) return launch_pdl(k_accumulate_bulk<true, true>, g, b, smem, s, A);
    if (A.local_mom) return launch_pdl(k_accumulate_bulk<true, false>, g, b, smem, s, A);
    if (A.bf16) return launch_pdl(k_accumulate_bulk<false, true>, g, b, smem, s, A);
    return launch_pdl(k_accumulate_bulk<false, false>, g, b, smem, s, A);
  }
  switch (tile_u(A.tile)) {
    case 1: return launch_ls<1>(A, grid, smem, s);
    case 2: return launch_ls<2>(A, grid, smem, s);
    default: return launch_ls<4>(A, grid, smem, s);
  }
}

cudaError_t launch_select(const TopkArgs& A, int blocks_per_worker, cudaStream_t s) {
  const dim3 grid(blocks_per_worker, A.K);
  if (A.regions == 1) {  // the bulk pass histogrammed its candidates already
    const cudaError_t err = launch_pdl(k_select_hist, grid, dim3(kThreads), 0, s, A);
    if (err != cudaSuccess) return err;
  }
  return launch_pdl(k_select_finish, grid, dim3(kThreads), kBucketCap * 4, s, A);
}

cudaError_t launch_select_approx(const TopkArgs& A, cudaStream_t s) {
  return launch_pdl(k_select_approx, dim3(1, A.K), dim3(kThreads), 0, s, A);
}

cudaError_t launch_select_dense(const TopkArgs& A, cudaStream_t s) {
  return launch_pdl(k_select_dense, dim3(A.K), dim3(1024), 0, s, A);
}

cudaError_t launch_mark(const TopkArgs& A, int grid, cudaStream_t s) {
  return launch_pdl(k_mark, dim3(grid, A.K), dim3(kThreads), 0, s, A);
}

cudaError_t launch_owner_sum(const TopkArgs& A, int grid, cudaStream_t s) {
  return launch_pdl(k_owner_sum, dim3(grid, A.K), dim3(kThreads), 0, s, A);
}

cudaError_t launch_server_update(const TopkArgs& A, cudaStream_t s) {
  int n = 0;
  cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, k_server_update, kThreads, 0);
  int dev = 0, sms = 1;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int64_t want = (A.d / 4 + kThreads - 1) / kThreads;
  const int grid = (int)std::max<int64_t>(1, std::min<int64_t>(want, (int64_t)sms * std::max(n, 1)));
  return launch_pdl(k_server_update, dim3(grid), dim3(kThreads), 0, s, A);
}

cudaError_t launch_gather_selected(const TopkArgs& A, int k, uint32_t* idx_out, float* val_out,
                                   cudaStream_t s) {
  k_gather_selected<<<1, 1024, 0, s>>>(A, k, idx_out, val_out);
  return cudaGetLastError();
}

}  // namespace gmc
