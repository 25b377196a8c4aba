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
constexpr int kSampleRun = 16;               // consecutive coordinates per sampled run (power of two):
                                             // 64 bytes of a row, one DRAM burst
constexpr int kSampleAll = 32768;            // d at or below which every element is sampled
constexpr int kSampleSlots = 32768;          // sampled positions per worker (= kSampleAll)
constexpr int kSampleChunks = kSampleSlots / kSampleRun;  // sampled runs per worker
static_assert((kSampleRun & (kSampleRun - 1)) == 0 && kSampleRun <= 32, "kSampleRun: a power of two, at most a warp");
constexpr int kHistBins = 2048;              // first radix digit: key bits 30..20
constexpr int kRelBins = 2048;               // bins of the candidates' relative histogram
constexpr int kBucketCap = 12288;            // candidates of one bin ranked in shared memory

// Per-worker top-k selection state, rewritten every step.
struct WorkerSel {
  uint32_t theta;    // candidate threshold key from the sample (kNoCandidate = none)
  uint32_t count;    // candidates appended by the accumulate pass (may exceed cap)
  uint32_t prefix;   // select: relative-histogram bin holding the k-th key
  uint32_t rank;     // select: the k-th key's 1-based rank inside that bin
  uint32_t T;        // the k-th largest key
  uint32_t n_tie;    // elements equal to T that are kept (lowest indices first)
  uint32_t ties;     // candidates equal to T
  uint32_t t_idx;    // a candidate equal to T is kept iff its index <= t_idx
  uint32_t dense;    // 1: this worker's selection is made by the dense path
  uint32_t done[4];  // finished-block counters: -, the select finish, the approximate
                     // top-s threshold, and (worker 0's) the dense select's blocks
  uint32_t count_bucket;  // candidates collected from the k-th key's bin
  uint32_t nsel;     // approximate top-s: components sent (the count varies by step)
  uint32_t pad;
};

// Step counters (see GMC_STAT_* in gmc.h), unsigned 64-bit slots.
struct Counters {
  unsigned long long v[8];
};
enum CounterSlot { kSteps = 0, kPairs = 1, kNnz = 2, kUnion = 3, kChanged = 4,
                   kFallbacks = 5, kNonfinite = 6 };
// The end of a step (one thread, after every kernel of the step that counts):
// the pairs counted on the host, the step mark, and the step into the totals.
// The step's counts may come from other blocks of the calling kernel: they
// are read from L2.
__device__ __forceinline__ void finalize_counters(Counters* step, Counters* total,
                                                  unsigned long long pairs_add) {
  step->v[kPairs] = __ldcg(&step->v[kPairs]) + pairs_add;
  step->v[kSteps] = 1;
  for (int i = 0; i < 8; ++i) total->v[i] += __ldcg(&step->v[i]);
}

// Device status bits (gmc_check).
constexpr unsigned kStatusNonfinite = 1u;
constexpr unsigned kStatusInternal = 2u;
constexpr unsigned kStatusTimeout = 4u;     // a bounded wait gave up (see wait_bounded): tiles were skipped
constexpr int kChunksPerTile = 8;           // candidate sub-chunks per tile: one per warp
constexpr uint32_t kNone = 0xffffffffu;     // no coordinate

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
// The dense path decides this worker's C(v) when its sampled filter missed:
// fewer candidates than k, a candidate region overflowed, or too many ties.
__device__ __forceinline__ bool needs_dense(const WorkerSel& s, uint32_t ksel, uint32_t cap) {
  return s.count < ksel || s.count > cap || s.dense != 0;
}
// bfloat16 gradients: the upper 16 bits of an fp32 pattern, widened exactly.
__device__ __forceinline__ float bf16_f32(uint32_t b) { return __uint_as_float(b << 16); }
// Four consecutive bf16 values at p (2-byte aligned, shared or global memory).
__device__ __forceinline__ float4 bf16x4(const uint16_t* p) {
  const uintptr_t a = reinterpret_cast<uintptr_t>(p);
  uint32_t lo, hi;
  if ((a & 7) == 0) {
    const uint2 x = *reinterpret_cast<const uint2*>(p);
    lo = x.x;
    hi = x.y;
  } else if ((a & 3) == 0) {
    lo = *reinterpret_cast<const uint32_t*>(p);
    hi = *reinterpret_cast<const uint32_t*>(p + 2);
  } else {
    lo = (uint32_t)p[0] | ((uint32_t)p[1] << 16);
    hi = (uint32_t)p[2] | ((uint32_t)p[3] << 16);
  }
  return make_float4(__uint_as_float(lo << 16), __uint_as_float(lo & 0xffff0000u),
                     __uint_as_float(hi << 16), __uint_as_float(hi & 0xffff0000u));
}
// Elements j .. j+3 of a bf16 row of d, zeros past d.
__device__ __forceinline__ float4 load_g4_bf16(const uint16_t* g, int64_t j, int64_t d) {
  if (j + 3 < d) return bf16x4(g + j);
  float4 r = make_float4(0.f, 0.f, 0.f, 0.f);
  if (j < d) r.x = bf16_f32(g[j]);
  if (j + 1 < d) r.y = bf16_f32(g[j + 1]);
  if (j + 2 < d) r.z = bf16_f32(g[j + 2]);
  return r;
}

// SplitMix64 (Steele, Lea & Flood, OOPSLA 2014): output function, the key of
// step t's stream (stream 0 = shared by all workers, k+1 = worker k), the
// stream's i-th draw, and [0, n) from a draw's top 32 bits by multiply-shift.
constexpr uint64_t kGamma = 0x9E3779B97F4A7C15ull;
__device__ __forceinline__ uint64_t sm64_mix(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}
__device__ __forceinline__ uint64_t stream_key(uint64_t seed, int64_t t, uint64_t stream) {
  const uint64_t k1 = sm64_mix(seed + kGamma * (uint64_t)(t + 1));
  return sm64_mix(k1 + kGamma * (stream + 1));
}
__device__ __forceinline__ uint64_t draw(uint64_t key, uint64_t i) {
  return sm64_mix(key + kGamma * (i + 1));
}
__device__ __forceinline__ uint32_t below(uint64_t x, uint64_t n) {
  return (uint32_t)(((x >> 32) * n) >> 32);
}
// Membership of a candidate in C(v): above the k-th key, or equal to it with
// an index no larger than the last tie kept (ties go to the lower index).
__device__ __forceinline__ bool selected(uint32_t key, uint32_t j, uint32_t T, uint32_t t_idx) {
  return key > T || (key == T && j <= t_idx);
}
// Shared-memory histogram increment, aggregated over the lanes of a warp that
// hit the same bucket (all lanes of the warp must call it; inactive: bin < 0).
__device__ __forceinline__ void warp_hist_add(uint32_t* hist, int bin) {
  const uint32_t peers = __match_any_sync(0xffffffffu, bin);
  const int leader = __ffs(peers) - 1;
  if (bin >= 0 && (int)(threadIdx.x & 31) == leader) atomicAdd(&hist[bin], (uint32_t)__popc(peers));
}
// Sum over the 32 lanes of a warp (all lanes must call it).
template <typename V>
__device__ __forceinline__ V warp_sum(V x) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
  return x;
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

// The same for any power-of-two nbins, also fewer bins than threads (a thread
// owns at most max(1, nbins / blockDim.x) of them; the others none).
__device__ __forceinline__ void block_find_from_top_any(const uint32_t* hist, int nbins, uint32_t r,
                                                        uint32_t* ws, uint32_t* out_bin,
                                                        uint32_t* out_rank) {
  const int per = nbins >= (int)blockDim.x ? nbins / (int)blockDim.x : 1;
  const int hi = nbins - (int)threadIdx.x * per;  // this thread's bins: [hi - per, hi), none when hi <= 0
  uint32_t mine = 0;
  for (int i = 1; i <= per && hi - i >= 0; ++i) mine += hist[hi - i];
  uint32_t total;
  const uint32_t incl = block_inclusive_scan<uint32_t>(mine, ws, &total);
  uint32_t above = incl - mine;
  if (above < r && r <= incl) {
    for (int i = 1; i <= per && hi - i >= 0; ++i) {
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

// ---------------------------------------------------------------------------
// mbarrier and bulk-copy primitives (inline PTX, sm_90+ / sm_103a)
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_addr(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.release.cta.shared::cta.b64 _, [%0], %1;"
               ::"r"(smem_addr(bar)), "r"(bytes) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.release.cta.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cta.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_addr(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ uint64_t global_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
// Bound of every mbarrier wait of the bulk passes (a test may shorten it for
// one step), and of the wait for a CTA's own copies in flight before it exits.
constexpr uint64_t kWaitLimitNs = 2000000000ull;
// Wait for the phase with the given parity to complete, giving up after
// limit_ns (returns false): a wait never hangs the GPU.
__device__ __forceinline__ bool wait_bounded(uint64_t* bar, uint32_t parity, uint64_t limit_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (global_ns() - t0 > limit_ns) return false;
  }
  return true;
}
// Programmatic dependent launch: a step's kernels are launched with
// programmatic stream serialization, so one may be scheduled while the one
// before it finishes; each waits here, before it touches memory, until its
// predecessor's writes are visible. Without that launch attribute it returns
// at once.
__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// Tiles of a persistent streaming pass. A CTA's first kFixed tiles are fixed,
// blockIdx.x + n * gridDim.x; every later one is claimed from a counter that
// the step's previous kernel zeroed, kFixed - 1 tiles before the CTA starts
// it, so that a CTA whose streams run faster takes more tiles and all of them
// finish together. The CTA's producer thread, when it starts its tile n,
// publishes the claim it made at tile n - 1 (for tile n - 1 + kFixed) in
// tq[(n - 1 + kFixed) % kQ], and then claims the next one; a thread reads
// tq[m % kQ] only after it has synchronised with the producer's start of tile
// m + 1 - kFixed. kQ must exceed the tiles between the oldest slot a thread
// may still read and the newest the producer may write.
// The number of fixed tiles may also be chosen at run time (uniform over the
// grid): tile_at_n / tile_claim_n.
template <int kQ>
__device__ __forceinline__ int64_t tile_at_n(const uint32_t* tq, uint32_t n, uint32_t fixed) {
  return n < fixed ? (int64_t)blockIdx.x + (int64_t)n * gridDim.x : (int64_t)tq[n % kQ];
}
// The order in which a pass visits its tiles, in blocks of G = gridDim.x
// consecutive tiles: the i-th tile claimed is order[i / G] * G + i mod G over
// the nb = n_tiles / G whole blocks (the partial block at the end stays last;
// order: a permutation of [0, nb), or NULL for index order; i >= n_tiles: past
// the last, unchanged). Within a block consecutive tiles still go to
// different CTAs at about the same time, so a layer's tiles spread over the
// CTAs' candidate parts as in index order.
__device__ __forceinline__ int64_t tile_order(int64_t i, int64_t n_tiles, const uint32_t* order) {
  if (i >= n_tiles || !order) return i;
  const uint32_t G = gridDim.x, nb = (uint32_t)(n_tiles / G);
  if ((uint64_t)i >= (uint64_t)nb * G) return i;
  const uint32_t b = (uint32_t)i / G, o = (uint32_t)i - b * G;
  const uint32_t ob = __ldg(order + b);
  return (int64_t)(ob < nb ? ob : b) * G + o;
}
template <int kFixed, int kQ>
__device__ __forceinline__ int64_t tile_at(const uint32_t* tq, uint32_t n) {
  return tile_at_n<kQ>(tq, n, (uint32_t)kFixed);
}
// The producer's part at the start of its tile n: returns the tile.
template <int kQ>
__device__ __forceinline__ int64_t tile_claim_n(uint32_t* tq, uint32_t n, uint32_t fixed, uint32_t* ctr,
                                                uint32_t& claim, int64_t n_tiles) {
  if (n > 0) tq[(n - 1 + fixed) % kQ] = fixed * gridDim.x + claim;
  const int64_t tile = tile_at_n<kQ>(tq, n, fixed);
  if (tile < n_tiles) claim = atomicAdd(ctr, 1u);
  return tile;
}
template <int kFixed, int kQ>
__device__ __forceinline__ int64_t tile_claim(uint32_t* tq, uint32_t n, uint32_t* ctr, uint32_t& claim,
                                              int64_t n_tiles) {
  return tile_claim_n<kQ>(tq, n, (uint32_t)kFixed, ctr, claim, n_tiles);
}

// Order this thread's generic-proxy shared-memory accesses before later
// async-proxy (bulk copy) accesses to the same memory.
__device__ __forceinline__ void fence_proxy_async() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
// Bulk copy global -> this CTA's shared memory, completing on `bar` (tx bytes).
// dst, src 16-byte aligned; bytes a multiple of 16.
__device__ __forceinline__ void bulk_load(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
      ::"r"(smem_addr(dst)), "l"(src), "r"(bytes), "r"(smem_addr(bar))
      : "memory");
}

// Prefetch [src, src + bytes) of global memory into L2 (no completion to wait
// for). src 16-byte aligned; bytes a multiple of 16.
__device__ __forceinline__ void bulk_prefetch_l2(const void* src, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(src), "r"(bytes) : "memory");
}

}  // namespace gmc
