// RBGS path of one GMC / GMC+ step (Alg. 1 / Alg. 2 with the random-block
// compressor of Sec. 4 and Sec. 5.2), and the small kernels shared by both
// compressors (GMC+ detach, counters).
//
//   pick   per block-choice stream (one shared by all workers, or one per
//          worker): m distinct blocks out of nb by Floyd's sampling driven by a
//          SplitMix64 counter stream keyed by (seed, t[, k]); writes the sorted
//          block list, a block -> slot map and the union flags
//   step   ONE dense pass per tile for all K workers in ascending order:
//          v = (e + g) - c*(w_t - w_{t-1}); inside chosen blocks v is sent
//          (copied to the worker's slab), summed into the aggregate and its
//          residual set to +0, elsewhere v is the residual; then, on the union,
//          w -= (eta/K) * sum and w_{t+1} - w_t is stored for the next step.
#include "gmc_internal.h"

namespace gmc {
namespace {

constexpr int kPickSmemWords = 12288;  // bitmap words kept in shared memory

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

__device__ __forceinline__ int g_mode(const float* p) {
  const uintptr_t a = reinterpret_cast<uintptr_t>(p);
  return (a & 15) == 0 ? 4 : ((a & 7) == 0 ? 2 : 1);
}

__device__ __forceinline__ uint32_t block_of(int64_t j, const RbgsArgs& A) {
  return A.B_shift != 0xffffffffu ? (uint32_t)(j >> A.B_shift) : (uint32_t)(j / A.B);
}

// ---------------------------------------------------------------------------
// pick: one block per stream
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kThreads) k_rbgs_pick(RbgsArgs A) {
  griddep_wait();
  if (blockIdx.x == 0 && threadIdx.x == 0) *A.tile_ctr = 0u;  // the fused pass claims its tiles from it
  extern __shared__ uint32_t bm_s[];
  __shared__ uint32_t ws[32];
  const int s = blockIdx.x;
  const int64_t nbw = (A.nb + 31) / 32;
  const bool in_smem = nbw <= kPickSmemWords;
  uint32_t* bm = in_smem ? bm_s : A.bitmap + (int64_t)s * nbw;
  if (in_smem) {
    for (int64_t i = threadIdx.x; i < nbw; i += blockDim.x) bm_s[i] = 0;
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    // Floyd: for j = nb-m .. nb-1, r = uniform[0, j]; keep j if r was taken, else r
    const uint64_t key = stream_key(A.seed, A.t, A.per_worker ? (uint64_t)s + 1 : 0ull);
    uint64_t i = 0;
    for (int64_t jj = A.nb - A.m; jj < A.nb; ++jj, ++i) {
      const uint32_t r = below(draw(key, i), (uint64_t)jj + 1);
      const uint32_t pick = ((bm[r >> 5] >> (r & 31)) & 1u) ? (uint32_t)jj : r;
      bm[pick >> 5] |= 1u << (pick & 31);
    }
  }
  __syncthreads();
  int32_t* rank = A.rank + (int64_t)s * A.nb;
  int32_t* blk = A.blocks + (int64_t)s * A.m;
  uint32_t carry = 0;
  for (int64_t w0 = 0; w0 < nbw; w0 += blockDim.x) {
    const int64_t wi = w0 + threadIdx.x;
    const uint32_t word = wi < nbw ? bm[wi] : 0u;
    uint32_t tot;
    const uint32_t inc = block_inclusive_scan<uint32_t>((uint32_t)__popc(word), ws, &tot);
    uint32_t q = carry + inc - (uint32_t)__popc(word);
    if (wi < nbw) {
      for (int bit = 0; bit < 32; ++bit) {
        const int64_t b = wi * 32 + bit;
        if (b >= A.nb) break;
        if ((word >> bit) & 1u) {
          rank[b] = (int32_t)q;
          blk[q] = (int32_t)b;
          A.uflag_cur[b] = 1;
          ++q;
        } else {
          rank[b] = -1;
        }
      }
      if (!in_smem) bm[wi] = 0u;  // the global bitmap stays zero between steps
    }
    carry += tot;
  }
}

// ---------------------------------------------------------------------------
// fused step: persistent blocks walk tiles of kRbgsTile elements
// ---------------------------------------------------------------------------
template <bool kBf16>
__global__ void __launch_bounds__(kThreads) k_rbgs_step(RbgsArgs A) {
  griddep_wait();
  constexpr int U = kRbgsTile / (kThreads * 4);  // float4 groups per thread
  __shared__ unsigned long long ws[32];
  uint32_t nonfinite = 0;
  unsigned long long pairs = 0, nnz = 0, uni = 0, changed = 0;
  const int64_t slab_ld = A.m * A.B;

  for (int64_t tile = blockIdx.x; tile < A.n_tiles; tile += gridDim.x) {
    const int64_t t0 = tile * kRbgsTile;
    const int64_t last = (t0 + kRbgsTile < A.d ? t0 + kRbgsTile : A.d) - 1;
    const int64_t b_lo = block_of(t0, A), b_hi = block_of(last, A);
    int tp = 0, tc = 0;
    for (int64_t b = b_lo + threadIdx.x; b <= b_hi; b += kThreads) {
      tp |= A.has_prev ? A.uflag_prev[b] : 0;
      tc |= A.uflag_cur[b];
    }
    tp = __syncthreads_or(tp);
    tc = __syncthreads_or(tc);

    uint32_t bid[U][4];
    float dlv[U][4], acc[U][4];
    uint32_t inU = 0;  // bit (u*4+i): coordinate in this step's union
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int64_t j = t0 + u * (kThreads * 4) + threadIdx.x * 4;
      float4 d4 = make_float4(0.f, 0.f, 0.f, 0.f);
      if (tp) d4 = *reinterpret_cast<const float4*>(A.dlt + j);
      dlv[u][0] = d4.x; dlv[u][1] = d4.y; dlv[u][2] = d4.z; dlv[u][3] = d4.w;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        acc[u][i] = 0.f;
        const bool in = j + i < A.d;
        bid[u][i] = in ? block_of(j + i, A) : 0u;
        if (in && tc && A.uflag_cur[bid[u][i]]) inU |= 1u << (u * 4 + i);
      }
    }

    for (int k = 0; k < A.K; ++k) {
      const int32_t* rk = A.rank + (A.per_worker ? (int64_t)k * A.nb : 0);
      float* ek = A.e + (int64_t)k * A.ld;
      const float* gk = A.grads + (int64_t)k * A.d;
      const uint16_t* gk16 = A.grads16 + (int64_t)k * A.d;
      float* sk = A.slab + (int64_t)k * slab_ld;
      const int gm = g_mode(gk);
      float4 ev[U], gv[U];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int64_t j = t0 + u * (kThreads * 4) + threadIdx.x * 4;
        ev[u] = __ldcs(reinterpret_cast<const float4*>(ek + j));
        gv[u] = kBf16 ? load_g4_bf16(gk16, j, A.d) : load_g4(gk, j, A.d, gm);
      }
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int64_t j = t0 + u * (kThreads * 4) + threadIdx.x * 4;
        float v[4] = {accumulate(ev[u].x, gv[u].x, A.c, dlv[u][0]),
                      accumulate(ev[u].y, gv[u].y, A.c, dlv[u][1]),
                      accumulate(ev[u].z, gv[u].z, A.c, dlv[u][2]),
                      accumulate(ev[u].w, gv[u].w, A.c, dlv[u][3])};
        float en[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          en[i] = v[i];
          if (j + i < A.d) {
            nonfinite += is_nonfinite(v[i]) ? 1u : 0u;
            if (tc) {
              const int32_t q = rk[bid[u][i]];
              if (q >= 0) {
                acc[u][i] = __fadd_rn(acc[u][i], v[i]);
                sk[(int64_t)q * A.B + (j + i - (int64_t)bid[u][i] * A.B)] = v[i];
                en[i] = 0.f;  // e_{t+1,k} = +0 where sent
                ++pairs;
                nnz += (v[i] != 0.f);
              }
            }
          }
        }
        __stcs(reinterpret_cast<float4*>(ek + j), make_float4(en[0], en[1], en[2], en[3]));
      }
    }

    if (tp || tc) {
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int64_t j = t0 + u * (kThreads * 4) + threadIdx.x * 4;
        float dd[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          if (inU & (1u << (u * 4 + i))) {
            const float wo = A.w[j + i];
            const float wn = __fsub_rn(wo, __fmul_rn(A.a, acc[u][i]));
            A.w[j + i] = wn;
            dd[i] = __fsub_rn(wn, wo);
            changed += (dd[i] != 0.f);
            ++uni;
          }
        }
        *reinterpret_cast<float4*>(A.dlt + j) = make_float4(dd[0], dd[1], dd[2], dd[3]);
      }
    }
  }
  unsigned long long tot;
  block_inclusive_scan<unsigned long long>(pairs, ws, &tot);
  if (threadIdx.x == 0 && tot) atomicAdd(&A.step_ctr->v[kPairs], tot);
  block_inclusive_scan<unsigned long long>(nnz, ws, &tot);
  if (threadIdx.x == 0 && tot) atomicAdd(&A.step_ctr->v[kNnz], tot);
  block_inclusive_scan<unsigned long long>(uni, ws, &tot);
  if (threadIdx.x == 0 && tot) atomicAdd(&A.step_ctr->v[kUnion], tot);
  block_inclusive_scan<unsigned long long>(changed, ws, &tot);
  if (threadIdx.x == 0 && tot) atomicAdd(&A.step_ctr->v[kChanged], tot);
  if (nonfinite) {
    atomicOr(A.status, kStatusNonfinite);
    atomicAdd(&A.step_ctr->v[kNonfinite], (unsigned long long)nonfinite);
  }
}

// (index, value) pairs of worker k's last C(.), in ascending index order.
__global__ void k_rbgs_expand(RbgsArgs A, int k, uint32_t* idx_out, float* val_out) {
  griddep_wait();
  const int64_t n = A.m * A.B;
  const int32_t* blk = A.blocks + (A.per_worker ? (int64_t)k * A.m : 0);
  const float* sk = A.slab + (int64_t)k * n;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t q = i / A.B, off = i - q * A.B;
    const int64_t j = (int64_t)blk[q] * A.B + off;
    if (j < A.d) {
      idx_out[i] = (uint32_t)j;
      val_out[i] = sk[i];
    }
  }
}

// GMC+ detach: out[k][j] = w[j] - b * e[k][j] (Alg. 2).
__global__ void k_detach(DetachArgs A) {
  griddep_wait();
  const int k = A.k0 + blockIdx.y;
  const float* ek = A.e + (int64_t)k * A.ld;
  float* ok = A.out + (int64_t)(k - A.k0) * A.out_ld;
  for (int64_t j = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; j < A.d;
       j += (int64_t)gridDim.x * blockDim.x)
    ok[j] = __fsub_rn(A.w[j], __fmul_rn(A.b, ek[j]));
}

__global__ void k_finalize(Counters* step, Counters* total, unsigned long long pairs_add) {
  griddep_wait();
  if (threadIdx.x == 0) finalize_counters(step, total, pairs_add);
}


// ---------------------------------------------------------------------------
// The same step as k_rbgs_step, with e and g streamed through a shared-memory
// ring by bulk copies. One persistent CTA per SM: a producer thread issues
// each (tile, worker) item's cp.async.bulk copies of e and g into the ring;
// sixteen consumer warps each own 256 elements of every tile and run through
// the K workers in ascending order (the aggregate adds in that order).
// Producer and consumers meet only at mbarriers; every wait is bounded. A
// CTA's first two tiles are fixed and every later one is claimed from a
// counter (tile_at, tile_claim), so that CTAs whose streams run faster take
// more tiles and all of them finish together.
// ---------------------------------------------------------------------------
namespace rbulk {
constexpr int kT = kRbgsTile;
constexpr int kStages = 4;
constexpr int kConsumers = 16;
constexpr int kSub = kT / kConsumers;      // 256 elements per consumer warp
constexpr int kGLen = kT + 8;              // g stage: up to 3 leading floats of misalignment
constexpr int kThreadsAll = (kConsumers + 1) * 32;
constexpr int kG = kSub / 128;             // float4 groups per lane
struct Smem {
  float e[kStages][kT];
  float g[kStages][kGLen];
  uint64_t full[kStages];                  // e, g landed (1 arrival + tx bytes)
  uint64_t empty[kStages];                 // all consumer warps read the stage
  int32_t gmeta[kStages];                  // leading floats in the g stage, -1 = not copied
  uint32_t tq[8];                          // claimed tiles (tile_at)
};
// Tiles: the first two of a CTA fixed, the rest claimed one tile ahead of the
// producer's start of the tile before it. A consumer reads a tile's slot at
// its start, after waiting on the previous tile's items (the producer's start
// of that tile is two tiles on from the claim's); the producer runs at most
// kStages items (tiles, for K = 1) ahead of the slowest consumer.
constexpr int kFixed = 2;
constexpr int kQ = 8;
static_assert(kQ > kStages + kFixed, "the producer may overwrite a claimed tile not yet read");
}  // namespace rbulk

template <bool kBf16>
__global__ void __launch_bounds__(rbulk::kThreadsAll, 1) k_rbgs_bulk(RbgsArgs A) {
  griddep_wait();
  using namespace rbulk;
  extern __shared__ __align__(128) unsigned char smem_raw[];
  Smem& sm = *reinterpret_cast<Smem*>(smem_raw);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&sm.full[s], 1);
      mbar_init(&sm.empty[s], kConsumers);
    }
    fence_mbar_init();
  }
  __syncthreads();

  if (warp == kConsumers) {
    // ---- producer ----
    if (lane != 0) return;
    // gradient rows of es-byte elements (fp32, or bf16 from gmc_step_bf16)
    constexpr int es = kBf16 ? 2 : 4;
    const char* g_lo = kBf16 ? reinterpret_cast<const char*>(A.grads16) : reinterpret_cast<const char*>(A.grads);
    const char* g_hi = g_lo + (int64_t)A.K * A.d * es;
    uint32_t item = 0, claim = 0;
    uint32_t held = ~0u;  // test hook: the item not copied
    bool ok = true;
    for (uint32_t n = 0; ok; ++n) {
      const int64_t tile = tile_claim<kFixed, kQ>(sm.tq, n, A.tile_ctr, claim, A.n_tiles);
      if (tile >= A.n_tiles) break;
      const int64_t j0 = tile * kT;
      const int64_t nvalid = A.d - j0 < kT ? A.d - j0 : kT;
      for (int k = 0; k < A.K; ++k, ++item) {
        const uint32_t s = item % kStages, r = item / kStages;
        if (r > 0 && !wait_bounded(&sm.empty[s], (r - 1) & 1, A.wait_ns)) {
          ok = false;
          break;
        }
        if (tile == A.hold_tile && k == A.hold_k) {  // the stage's phase never completes
          held = item;
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
    // when the consumers gave up on their waits: the last kStages items (the
    // earlier ones were read, as their stages' empty barriers showed) read
    // valid global memory and complete without any other warp's help; no
    // later phase is armed on their stages.
    const uint32_t first = item > (uint32_t)kStages ? item - kStages : 0u;
    for (uint32_t i = first; i < item; ++i)
      if (i != held && !wait_bounded(&sm.full[i % kStages], (i / kStages) & 1, kWaitLimitNs))
        atomicOr(A.status, kStatusTimeout | kStatusInternal);
    return;
  }

  // ---- consumers ----
  const int64_t slab_ld = A.m * A.B;
  uint32_t nonfinite = 0;
  unsigned long long pairs = 0, nnz = 0, uni = 0, changed = 0;
  uint32_t item = 0;
  bool ok = true;
  for (uint32_t n = 0; ok; ++n) {
    const int64_t tile = tile_at<kFixed, kQ>(sm.tq, n);
    if (tile >= A.n_tiles) break;
    const int64_t s0 = tile * kT + warp * kSub;
    const int64_t rem = A.d - s0;
    const int lim = rem < kSub ? (rem > 0 ? (int)rem : 0) : kSub;
    // does the sub-tile touch the last step's union (tp) or this step's (tc)?
    int tp = 0, tc = 0;
    if (lim > 0) {
      const int64_t b_lo = block_of(s0, A), b_hi = block_of(s0 + lim - 1, A);
      for (int64_t b = b_lo + lane; b <= b_hi; b += 32) {
        tp |= A.has_prev ? A.uflag_prev[b] : 0;
        tc |= A.uflag_cur[b];
      }
    }
    tp = __any_sync(0xffffffffu, tp);
    tc = __any_sync(0xffffffffu, tc);
    float dl[kG][4], acc[kG][4];
    uint32_t bid[kG][4];
    uint32_t inU = 0;  // bit (u*4+i): coordinate in this step's union
#pragma unroll
    for (int u = 0; u < kG; ++u) {
      const int l = u * 128 + lane * 4;
      float4 d4 = make_float4(0.f, 0.f, 0.f, 0.f);
      if (tp && l < lim) d4 = *reinterpret_cast<const float4*>(A.dlt + s0 + l);
      dl[u][0] = d4.x; dl[u][1] = d4.y; dl[u][2] = d4.z; dl[u][3] = d4.w;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        acc[u][i] = 0.f;
        const bool in = l + i < lim;
        bid[u][i] = (in && tc) ? block_of(s0 + l + i, A) : 0u;
        if (in && tc && A.uflag_cur[bid[u][i]]) inU |= 1u << (u * 4 + i);
      }
    }
    for (int k = 0; k < A.K; ++k, ++item) {
      const uint32_t s = item % kStages, r = item / kStages;
      if (!__all_sync(0xffffffffu, wait_bounded(&sm.full[s], r & 1, A.wait_ns))) {  // warp-uniform
        ok = false;
        break;
      }
      const int32_t off = sm.gmeta[s];
      const float* se = sm.e[s] + warp * kSub;
      const float* sg = sm.g[s] + (off > 0 ? off : 0) + warp * kSub;
      float v[kG][4];
#pragma unroll
      for (int u = 0; u < kG; ++u) {
        const int l = u * 128 + lane * 4;
        const float4 e4 = *reinterpret_cast<const float4*>(se + l);
        float4 g4;
        if constexpr (kBf16) {
          if (off >= 0)
            g4 = bf16x4(reinterpret_cast<const uint16_t*>(sm.g[s]) + off + warp * kSub + l);
          else
            g4 = load_g4_bf16(A.grads16 + (int64_t)k * A.d, s0 + l, A.d);
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
          g4 = load_g4(gk, s0 + l, A.d, g_mode(gk));
        }
        if (lim < kSub && off >= 0) {  // past d the stage holds bytes of no meaning
          if (l >= lim) g4.x = 0.f;
          if (l + 1 >= lim) g4.y = 0.f;
          if (l + 2 >= lim) g4.z = 0.f;
          if (l + 3 >= lim) g4.w = 0.f;
        }
        v[u][0] = accumulate(e4.x, g4.x, A.c, dl[u][0]);
        v[u][1] = accumulate(e4.y, g4.y, A.c, dl[u][1]);
        v[u][2] = accumulate(e4.z, g4.z, A.c, dl[u][2]);
        v[u][3] = accumulate(e4.w, g4.w, A.c, dl[u][3]);
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&sm.empty[s]);  // this warp is done reading stage s
      float* ek = A.e + (int64_t)k * A.ld + s0;
      const int32_t* rk = A.rank + (A.per_worker ? (int64_t)k * A.nb : 0);
      float* sk = A.slab + (int64_t)k * slab_ld;
#pragma unroll
      for (int u = 0; u < kG; ++u) {
        const int l = u * 128 + lane * 4;
        float en[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          en[i] = v[u][i];
          if (l + i < lim) {
            nonfinite += is_nonfinite(v[u][i]) ? 1u : 0u;
            if (tc) {
              const int32_t q = rk[bid[u][i]];
              if (q >= 0) {  // in one of worker k's chosen blocks: sent
                acc[u][i] = __fadd_rn(acc[u][i], v[u][i]);
                sk[(int64_t)q * A.B + (s0 + l + i - (int64_t)bid[u][i] * A.B)] = v[u][i];
                en[i] = 0.f;  // e_{t+1,k} = +0 where sent
                ++pairs;
                nnz += (v[u][i] != 0.f);
              }
            }
          }
        }
        __stcs(reinterpret_cast<float4*>(ek + l), make_float4(en[0], en[1], en[2], en[3]));
      }
    }
    if (ok && (tp || tc)) {  // the union: w_{t+1} = w_t - a * sum, and w_{t+1} - w_t for the next step
#pragma unroll
      for (int u = 0; u < kG; ++u) {
        const int l = u * 128 + lane * 4;
        if (l >= lim) continue;
        float dd[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          if (inU & (1u << (u * 4 + i))) {
            const float wo = A.w[s0 + l + i];
            const float wn = __fsub_rn(wo, __fmul_rn(A.a, acc[u][i]));
            A.w[s0 + l + i] = wn;
            dd[i] = __fsub_rn(wn, wo);
            changed += (dd[i] != 0.f);
            ++uni;
          }
        }
        *reinterpret_cast<float4*>(A.dlt + s0 + l) = make_float4(dd[0], dd[1], dd[2], dd[3]);
      }
    }
  }
  if (!ok) atomicOr(A.status, kStatusTimeout);
  pairs = warp_sum(pairs);
  nnz = warp_sum(nnz);
  uni = warp_sum(uni);
  changed = warp_sum(changed);
  if (lane == 0) {
    if (pairs) atomicAdd(&A.step_ctr->v[kPairs], pairs);
    if (nnz) atomicAdd(&A.step_ctr->v[kNnz], nnz);
    if (uni) atomicAdd(&A.step_ctr->v[kUnion], uni);
    if (changed) atomicAdd(&A.step_ctr->v[kChanged], changed);
  }
  if (nonfinite) {
    atomicOr(A.status, kStatusNonfinite);
    atomicAdd(&A.step_ctr->v[kNonfinite], (unsigned long long)nonfinite);
  }
}

}  // namespace

cudaError_t configure_rbgs_kernels() {
  cudaError_t err = cudaFuncSetAttribute((const void*)k_rbgs_pick,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, kPickSmemWords * 4);
  const cudaError_t e2 = cudaFuncSetAttribute((const void*)k_rbgs_bulk<false>,
                                              cudaFuncAttributeMaxDynamicSharedMemorySize,
                                              (int)sizeof(rbulk::Smem));
  const cudaError_t e3 = cudaFuncSetAttribute((const void*)k_rbgs_bulk<true>,
                                              cudaFuncAttributeMaxDynamicSharedMemorySize,
                                              (int)sizeof(rbulk::Smem));
  return err != cudaSuccess ? err : (e2 != cudaSuccess ? e2 : e3);
}

int rbgs_blocks_per_sm() {
  int n = 0;
  cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, k_rbgs_step<false>, kThreads, 0);
  return n > 0 ? n : 1;
}

cudaError_t launch_rbgs_pick(const RbgsArgs& A, cudaStream_t s) {
  const int64_t nbw = (A.nb + 31) / 32;
  const int smem = nbw <= kPickSmemWords ? (int)(nbw * 4) : 0;
  const cudaError_t err = launch_pdl(k_rbgs_pick, dim3(A.per_worker ? A.K : 1), dim3(kThreads), smem, s, A);
  if (err != cudaSuccess) return err;
  return cudaGetLastError();
}

cudaError_t launch_rbgs_step(const RbgsArgs& A, int grid, cudaStream_t s) {
  if (A.bulk) {
    return launch_pdl(A.bf16 ? k_rbgs_bulk<true> : k_rbgs_bulk<false>, dim3(grid), dim3(rbulk::kThreadsAll),
                      sizeof(rbulk::Smem), s, A);
  }
  return launch_pdl(A.bf16 ? k_rbgs_step<true> : k_rbgs_step<false>, dim3(grid), dim3(kThreads), 0, s, A);
}

cudaError_t launch_rbgs_expand(const RbgsArgs& A, int k, uint32_t* idx_out, float* val_out,
                               cudaStream_t s) {
  const int64_t n = A.m * A.B;
  const int grid = (int)((n + 255) / 256 < 4096 ? (n + 255) / 256 : 4096);
  k_rbgs_expand<<<grid > 0 ? grid : 1, 256, 0, s>>>(A, k, idx_out, val_out);
  return cudaGetLastError();
}

cudaError_t launch_detach(const DetachArgs& A, cudaStream_t s) {
  const int64_t blocks = (A.d + 255) / 256;
  const dim3 grid((unsigned)(blocks < 1024 ? blocks : 1024), (unsigned)(A.k1 - A.k0));
  const cudaError_t err = launch_pdl(k_detach, dim3(grid), dim3(256), 0, s, A);
  if (err != cudaSuccess) return err;
  return cudaGetLastError();
}

cudaError_t launch_finalize(Counters* step, Counters* total, unsigned long long pairs_add,
                            cudaStream_t s) {
  const cudaError_t err = launch_pdl(k_finalize, dim3(1), dim3(32), 0, s, step, total, pairs_add);
  if (err != cudaSuccess) return err;
  return cudaGetLastError();
}

}  // namespace gmc
