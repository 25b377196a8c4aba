// Top-k path of one GMC step (Alg. 1 with the top-s compressor of Sec. 4):
//
//   sample      per worker, e_{t+1/2} at a stratified sample -> a threshold key
//               theta below the k-th largest |v| with overwhelming probability
//   accumulate  ONE dense pass: v = (e + g) - c*(w_t - w_{t-1}) written over e,
//               and every v with key >= theta appended to the worker's candidate
//               list in per-tile chunks that are sorted by index
//   select x3   exact k-th largest key T among the candidates (radix digits of
//               11, 10 and 10 bits), and how many ties at T are kept
//   dense       for a worker whose filter missed (too few or too many
//               candidates): the exact select and compaction over dense v
//   compact x3  per-tile counts, per-worker scan, index-ordered write of
//               C(v) = (index, value) pairs
//   aggregate   per tile: sum the workers' values in ascending worker order,
//               e = 0 at sent coordinates, w -= (eta/K) * sum on the union,
//               store w_{t+1} - w_t for the next step's accumulator
//
// Keys are the fp32 bit patterns with the sign cleared (monotone in |v|); the
// selected set is the first k elements under (key descending, index ascending).
#include "gmc_internal.h"

namespace gmc {
namespace {

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

template <typename V>
__device__ __forceinline__ V warp_sum(V x) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
  return x;
}

// ---------------------------------------------------------------------------
// sample: one block per worker
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kSampleThreads) k_sample(TopkArgs A) {
  extern __shared__ uint32_t keys[];
  __shared__ uint32_t hist[kHistBins];
  __shared__ uint32_t ws[32];
  __shared__ uint32_t s_bin, s_rank;
  const int k = blockIdx.x;
  WorkerSel& S = A.sel[k];
  if (A.dense_mode) {
    if (threadIdx.x == 0) {
      S.theta = kNoCandidate;
      S.count = 0;
    }
    return;
  }
  const float* ek = A.e + (int64_t)k * A.ld;
  const float* gk = A.grads + (int64_t)k * A.d;
  int n_s;
  if (A.sample_chunks == 0) {
    n_s = (int)A.d;
    for (int j = threadIdx.x; j < n_s; j += blockDim.x)
      keys[j] = mag_key(accumulate(ek[j], gk[j], A.c, A.dlt[j]));
  } else {
    n_s = A.sample_chunks * 8;
    for (int ch = threadIdx.x; ch < A.sample_chunks; ch += blockDim.x) {
      const int64_t p = ((int64_t)ch * A.d / A.sample_chunks) & ~int64_t(7);
#pragma unroll
      for (int i = 0; i < 8; ++i)
        keys[ch * 8 + i] = mag_key(accumulate(ek[p + i], gk[p + i], A.c, A.dlt[p + i]));
    }
  }
  for (int b = threadIdx.x; b < kHistBins; b += blockDim.x) hist[b] = 0;
  if (threadIdx.x == 0) {
    s_bin = 0;
    s_rank = 0;
  }
  __syncthreads();
  uint32_t r = A.sample_rank < (uint32_t)n_s ? A.sample_rank : (uint32_t)n_s;
  for (int i = threadIdx.x; i < n_s; i += blockDim.x) atomicAdd(&hist[keys[i] >> 20], 1u);
  __syncthreads();
  block_find_from_top(hist, kHistBins, r, ws, &s_bin, &s_rank);
  const uint32_t b1 = s_bin;
  r = s_rank;
  __syncthreads();
  for (int b = threadIdx.x; b < 1024; b += blockDim.x) hist[b] = 0;
  __syncthreads();
  for (int i = threadIdx.x; i < n_s; i += blockDim.x) {
    const uint32_t key = keys[i];
    if ((key >> 20) == b1) atomicAdd(&hist[(key >> 10) & 1023u], 1u);
  }
  __syncthreads();
  block_find_from_top(hist, 1024, r, ws, &s_bin, &s_rank);
  if (threadIdx.x == 0) {
    S.theta = (b1 << 20) | (s_bin << 10);
    S.count = 0;
  }
}

// ---------------------------------------------------------------------------
// accumulate + filter: the one dense pass. Persistent blocks walk the tiles;
// each tile is done for all K workers so the staged w_t - w_{t-1} is reused.
// ---------------------------------------------------------------------------
template <int U>
__global__ void __launch_bounds__(kThreads) k_accumulate(TopkArgs A) {
  constexpr int SUB = 128 * U;       // elements per warp and worker
  constexpr int T = kWarps * SUB;    // elements per tile
  extern __shared__ __align__(16) unsigned char smem[];
  float* dl = reinterpret_cast<float*>(smem);
  uint32_t* st_idx = reinterpret_cast<uint32_t*>(dl + T);
  float* st_val = reinterpret_cast<float*>(st_idx + T);
  __shared__ uint32_t s_wcnt[kWarps], s_woff[kWarps], s_base;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t lt = lanemask_lt();
  uint32_t nonfinite = 0;

  for (int64_t tile = blockIdx.x; tile < A.n_tiles; tile += gridDim.x) {
    const int64_t t0 = tile * T;
    for (int i = threadIdx.x; i < T / 4; i += kThreads)
      reinterpret_cast<float4*>(dl)[i] = make_float4(0.f, 0.f, 0.f, 0.f);
    __syncthreads();
    if (A.has_prev) {
      // w_t - w_{t-1} is non-zero only on the previous step's union of sent
      // coordinates; scatter it into the tile from the previous sorted lists.
      for (int kk = 0; kk < A.K; ++kk) {
        const uint32_t* pp = A.pos_prev + (int64_t)kk * (A.n_tiles + 1);
        const uint32_t lo = pp[tile], hi = pp[tile + 1];
        const uint32_t* ip = A.idx_prev + (int64_t)kk * A.ksel;
        for (uint32_t i = lo + threadIdx.x; i < hi && i < A.ksel; i += kThreads) {
          const uint32_t j = ip[i];
          if ((uint64_t)(j - t0) < (uint64_t)T) dl[j - t0] = A.dlt[j];
          else atomicOr(A.status, kStatusInternal);
        }
      }
    }
    __syncthreads();

    for (int k = 0; k < A.K; ++k) {
      const uint32_t theta = A.sel[k].theta;
      float* ek = A.e + (int64_t)k * A.ld;
      const float* gk = A.grads + (int64_t)k * A.d;
      const int gm = g_mode(gk);
      const int64_t wbase = t0 + warp * SUB;
      float4 ev[U], gv[U];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int64_t j = wbase + u * 128 + lane * 4;
        ev[u] = __ldcs(reinterpret_cast<const float4*>(ek + j));
        gv[u] = load_g4(gk, j, A.d, gm);
      }
      uint32_t wcnt = 0;
      uint32_t* sti = st_idx + warp * SUB;
      float* stv = st_val + warp * SUB;
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int64_t j = wbase + u * 128 + lane * 4;
        const float4 d4 = *reinterpret_cast<const float4*>(dl + (j - t0));
        float v[4];
        v[0] = accumulate(ev[u].x, gv[u].x, A.c, d4.x);
        v[1] = accumulate(ev[u].y, gv[u].y, A.c, d4.y);
        v[2] = accumulate(ev[u].z, gv[u].z, A.c, d4.z);
        v[3] = accumulate(ev[u].w, gv[u].w, A.c, d4.w);
        __stcs(reinterpret_cast<float4*>(ek + j), make_float4(v[0], v[1], v[2], v[3]));
        bool f[4];
        uint32_t bal[4];
        uint32_t before = 0, total = 0;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const bool in = j + i < A.d;
          f[i] = in && mag_key(v[i]) >= theta;
          nonfinite += (in && is_nonfinite(v[i])) ? 1u : 0u;
          bal[i] = __ballot_sync(0xffffffffu, f[i]);
          before += __popc(bal[i] & lt);
          total += __popc(bal[i]);
        }
        uint32_t o = wcnt + before;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          if (f[i]) {
            sti[o] = (uint32_t)(j + i);
            stv[o] = v[i];
            ++o;
          }
        }
        wcnt += total;
      }
      if (lane == 0) s_wcnt[warp] = wcnt;
      __syncthreads();
      if (threadIdx.x == 0) {
        uint32_t tot = 0;
#pragma unroll
        for (int w = 0; w < kWarps; ++w) {
          s_woff[w] = tot;
          tot += s_wcnt[w];
        }
        const uint32_t base = tot ? atomicAdd(&A.sel[k].count, tot) : 0u;
        s_base = base;
        A.chunk_base[(int64_t)k * A.n_tiles + tile] = base;
        A.chunk_cnt[(int64_t)k * A.n_tiles + tile] = tot;
      }
      __syncthreads();
      const uint32_t base = s_base + s_woff[warp];
      uint32_t* ci = A.cand_idx + (int64_t)k * A.cap;
      float* cv = A.cand_val + (int64_t)k * A.cap;
      for (uint32_t i = lane; i < wcnt; i += 32) {
        const uint32_t p = base + i;
        if (p < A.cap) {
          ci[p] = sti[i];
          cv[p] = stv[i];
        }
      }
      __syncwarp();
    }
    __syncthreads();
  }
  if (nonfinite) {
    atomicOr(A.status, kStatusNonfinite);
    atomicAdd(&A.step_ctr->v[kNonfinite], (unsigned long long)nonfinite);
  }
}

// ---------------------------------------------------------------------------
// exact select among candidates: three radix passes; the last block of each
// worker turns the global histogram into the next digit.
// ---------------------------------------------------------------------------
template <int PASS>
__global__ void __launch_bounds__(kThreads) k_select_pass(TopkArgs A) {
  constexpr int nbins = PASS == 0 ? 2048 : 1024;
  constexpr int shift = PASS == 0 ? 20 : (PASS == 1 ? 10 : 0);
  __shared__ uint32_t h[nbins];
  __shared__ uint32_t ws[32];
  __shared__ uint32_t s_last, s_bin, s_rank;
  const int k = blockIdx.y;
  WorkerSel& S = A.sel[k];
  if (needs_dense(S, A.ksel, A.cap)) return;
  const uint32_t cnt = S.count;
  const uint32_t prefix = S.prefix;
  for (int b = threadIdx.x; b < nbins; b += blockDim.x) h[b] = 0;
  __syncthreads();
  const float* cv = A.cand_val + (int64_t)k * A.cap;
  for (uint32_t i = blockIdx.x * blockDim.x + threadIdx.x; i < cnt; i += gridDim.x * blockDim.x) {
    const uint32_t key = mag_key(cv[i]);
    if (PASS == 0 || (key >> (shift + 10)) == prefix)
      atomicAdd(&h[(key >> shift) & (nbins - 1)], 1u);
  }
  __syncthreads();
  uint32_t* gh = A.ghist + (int64_t)k * kHistBins;
  for (int b = threadIdx.x; b < nbins; b += blockDim.x)
    if (h[b]) atomicAdd(&gh[b], h[b]);
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) s_last = (atomicAdd(&S.done[PASS], 1u) == gridDim.x - 1) ? 1u : 0u;
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
    S.done[PASS] = 0;
  }
  __syncthreads();
  const uint32_t r = PASS == 0 ? A.ksel : S.rank;
  block_find_from_top(h, nbins, r, ws, &s_bin, &s_rank);
  if (threadIdx.x == 0) {
    if (s_rank == 0) atomicOr(A.status, kStatusInternal);
    if (PASS == 0) {
      S.prefix = s_bin;
      S.rank = s_rank;
    } else if (PASS == 1) {
      S.prefix = (prefix << 10) | s_bin;
      S.rank = s_rank;
    } else {
      S.T = (prefix << 10) | s_bin;
      S.n_tie = s_rank;
    }
  }
}

// ---------------------------------------------------------------------------
// dense exact select + compaction for workers whose filter missed; one block
// per worker (a rare path: correct for any input, not fast).
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(1024) k_select_dense(TopkArgs A) {
  const int k = blockIdx.x;
  WorkerSel& S = A.sel[k];
  if (!needs_dense(S, A.ksel, A.cap)) return;
  __shared__ uint32_t h[kHistBins];
  __shared__ uint32_t ws[32];
  __shared__ unsigned long long ws64[32];
  __shared__ uint32_t s_bin, s_rank;
  const float* vk = A.e + (int64_t)k * A.ld;
  const int64_t d = A.d;
  uint32_t r = A.ksel, prefix = 0;
  for (int pass = 0; pass < 3; ++pass) {
    const int nbins = pass == 0 ? 2048 : 1024;
    const int shift = pass == 0 ? 20 : (pass == 1 ? 10 : 0);
    for (int b = threadIdx.x; b < nbins; b += blockDim.x) h[b] = 0;
    if (threadIdx.x == 0) {
      s_bin = 0;
      s_rank = 0;
    }
    __syncthreads();
    for (int64_t j = threadIdx.x; j < d; j += blockDim.x) {
      const uint32_t key = mag_key(vk[j]);
      if (pass == 0 || (key >> (shift + 10)) == prefix)
        atomicAdd(&h[(key >> shift) & (uint32_t)(nbins - 1)], 1u);
    }
    __syncthreads();
    block_find_from_top(h, nbins, r, ws, &s_bin, &s_rank);
    prefix = pass == 0 ? s_bin : ((prefix << 10) | s_bin);
    r = s_rank;
    __syncthreads();
  }
  const uint32_t T = prefix, n_tie = r;

  const int P = A.tile / (int)blockDim.x;  // consecutive elements per thread
  uint32_t* pos = A.pos_cur + (int64_t)k * (A.n_tiles + 1);
  uint32_t* oi = A.idx_cur + (int64_t)k * A.ksel;
  float* ov = A.val_cur + (int64_t)k * A.ksel;
  uint32_t running = 0, eqrun = 0;
  for (int64_t tile = 0; tile < A.n_tiles; ++tile) {
    if (threadIdx.x == 0) pos[tile] = running;
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
    for (int i = 0; i < P; ++i) {
      const int64_t j = j0 + i;
      if (j < d) {
        const float v = vk[j];
        const uint32_t key = mag_key(v);
        const bool take = key > T || (key == T && qg < n_tie);
        if (key == T) ++qg;
        if (take) {
          if (o < A.ksel) {
            oi[o] = (uint32_t)j;
            ov[o] = v;
          }
          ++o;
        }
      }
    }
    running += (uint32_t)(tot >> 32) + (min(eqrun + (uint32_t)tot, n_tie) - taken0);
    eqrun += (uint32_t)tot;
  }
  if (threadIdx.x == 0) {
    pos[A.n_tiles] = running;
    if (running != A.ksel) atomicOr(A.status, kStatusInternal);
    S.T = T;
    S.n_tie = n_tie;
    atomicAdd(&A.step_ctr->v[kFallbacks], 1ull);
  }
}

// ---------------------------------------------------------------------------
// compaction: per-tile counts, per-worker scan, index-ordered write
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kThreads) k_chunk_count(TopkArgs A) {
  const int k = blockIdx.y;
  const WorkerSel& S = A.sel[k];
  if (needs_dense(S, A.ksel, A.cap)) return;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t tile = (int64_t)blockIdx.x * kWarps + warp;
  if (tile >= A.n_tiles) return;
  const int64_t ct = (int64_t)k * A.n_tiles + tile;
  const uint32_t base = A.chunk_base[ct], cnt = A.chunk_cnt[ct], T = S.T;
  const float* cv = A.cand_val + (int64_t)k * A.cap + base;
  uint32_t g = 0, q = 0;
  for (uint32_t i = lane; i < cnt; i += 32) {
    const uint32_t key = mag_key(cv[i]);
    g += key > T;
    q += key == T;
  }
  g = warp_sum(g);
  q = warp_sum(q);
  if (lane == 0) {
    A.gt_cnt[ct] = g;
    A.eq_cnt[ct] = q;
  }
}

__global__ void __launch_bounds__(1024) k_chunk_scan(TopkArgs A) {
  const int k = blockIdx.x;
  const WorkerSel& S = A.sel[k];
  if (needs_dense(S, A.ksel, A.cap)) return;
  __shared__ unsigned long long ws[32];
  const uint32_t n_tie = S.n_tie;
  uint32_t* pos = A.pos_cur + (int64_t)k * (A.n_tiles + 1);
  const int64_t row = (int64_t)k * A.n_tiles;
  uint32_t carry_g = 0, carry_q = 0;
  for (int64_t t0 = 0; t0 < A.n_tiles; t0 += blockDim.x) {
    const int64_t tile = t0 + threadIdx.x;
    uint32_t g = 0, q = 0;
    if (tile < A.n_tiles) {
      g = A.gt_cnt[row + tile];
      q = A.eq_cnt[row + tile];
    }
    const unsigned long long x = ((unsigned long long)g << 32) | q;
    unsigned long long tot;
    const unsigned long long exc = block_inclusive_scan<unsigned long long>(x, ws, &tot) - x;
    const uint32_t gb = carry_g + (uint32_t)(exc >> 32);
    const uint32_t qb = carry_q + (uint32_t)exc;
    if (tile < A.n_tiles) {
      pos[tile] = gb + min(qb, n_tie);
      A.eq_before[row + tile] = qb;
    }
    carry_g += (uint32_t)(tot >> 32);
    carry_q += (uint32_t)tot;
  }
  if (threadIdx.x == 0) {
    const uint32_t total = carry_g + min(carry_q, n_tie);
    pos[A.n_tiles] = total;
    if (total != A.ksel) atomicOr(A.status, kStatusInternal);
  }
}

__global__ void __launch_bounds__(kThreads) k_chunk_write(TopkArgs A) {
  const int k = blockIdx.y;
  const WorkerSel& S = A.sel[k];
  if (needs_dense(S, A.ksel, A.cap)) return;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t tile = (int64_t)blockIdx.x * kWarps + warp;
  if (tile >= A.n_tiles) return;
  const uint32_t lt = lanemask_lt();
  const int64_t ct = (int64_t)k * A.n_tiles + tile;
  const uint32_t base = A.chunk_base[ct], cnt = A.chunk_cnt[ct];
  const uint32_t T = S.T, n_tie = S.n_tie;
  const uint32_t p = A.pos_cur[(int64_t)k * (A.n_tiles + 1) + tile];
  const uint32_t eb = A.eq_before[ct];
  uint32_t* oi = A.idx_cur + (int64_t)k * A.ksel + p;
  float* ov = A.val_cur + (int64_t)k * A.ksel + p;
  const uint32_t* ci = A.cand_idx + (int64_t)k * A.cap + base;
  const float* cv = A.cand_val + (int64_t)k * A.cap + base;
  uint32_t written = 0, eqseen = 0;
  for (uint32_t i0 = 0; i0 < cnt; i0 += 32) {
    const uint32_t i = i0 + lane;
    const bool valid = i < cnt;
    float v = 0.f;
    uint32_t idx = 0, key = 0;
    if (valid) {
      v = cv[i];
      idx = ci[i];
      key = mag_key(v);
    }
    const bool gt = valid && key > T;
    const bool eq = valid && key == T;
    const uint32_t em = __ballot_sync(0xffffffffu, eq);
    const bool take = gt || (eq && eb + eqseen + __popc(em & lt) < n_tie);
    const uint32_t tm = __ballot_sync(0xffffffffu, take);
    if (take) {
      const uint32_t o = written + __popc(tm & lt);
      if (p + o < A.ksel) {
        oi[o] = idx;
        ov[o] = v;
      } else {
        atomicOr(A.status, kStatusInternal);
      }
    }
    written += __popc(tm);
    eqseen += __popc(em);
  }
}

// ---------------------------------------------------------------------------
// aggregate + update, one tile at a time (persistent blocks)
// ---------------------------------------------------------------------------
template <int U>
__global__ void __launch_bounds__(kThreads) k_aggregate(TopkArgs A) {
  constexpr int T = kWarps * 128 * U;
  extern __shared__ __align__(16) unsigned char smem[];
  float* s_acc = reinterpret_cast<float*>(smem);
  uint16_t* ulist = reinterpret_cast<uint16_t*>(s_acc + T);
  uint8_t* flag = reinterpret_cast<uint8_t*>(ulist + T);
  __shared__ uint32_t s_ucnt;
  __shared__ unsigned long long ws[32];
  for (int i = threadIdx.x; i < T; i += kThreads) {
    s_acc[i] = 0.f;
    flag[i] = 0;
  }
  if (threadIdx.x == 0) s_ucnt = 0;
  __syncthreads();
  unsigned long long nnz = 0, uni = 0, changed = 0;
  for (int64_t tile = blockIdx.x; tile < A.n_tiles; tile += gridDim.x) {
    const int64_t t0 = tile * T;
    if (A.has_prev) {
      // w_t - w_{t-1} is rebuilt below: clear it on the previous union first
      for (int kk = 0; kk < A.K; ++kk) {
        const uint32_t* pp = A.pos_prev + (int64_t)kk * (A.n_tiles + 1);
        const uint32_t lo = pp[tile], hi = pp[tile + 1];
        const uint32_t* ip = A.idx_prev + (int64_t)kk * A.ksel;
        for (uint32_t i = lo + threadIdx.x; i < hi && i < A.ksel; i += kThreads) {
          const uint32_t j = ip[i];
          if (j < (uint32_t)A.d) A.dlt[j] = 0.f;
        }
      }
    }
    // workers in ascending order: sum_k C(e_{t+1/2,k}) starting from +0
    for (int k = 0; k < A.K; ++k) {
      const uint32_t* pc = A.pos_cur + (int64_t)k * (A.n_tiles + 1);
      const uint32_t lo = pc[tile], hi = pc[tile + 1];
      const uint32_t* ic = A.idx_cur + (int64_t)k * A.ksel;
      const float* vc = A.val_cur + (int64_t)k * A.ksel;
      float* ek = A.e + (int64_t)k * A.ld;
      for (uint32_t i = lo + threadIdx.x; i < hi && i < A.ksel; i += kThreads) {
        const uint32_t j = ic[i];
        const float v = vc[i];
        const uint32_t l = j - (uint32_t)t0;
        if (l >= (uint32_t)T || j >= (uint32_t)A.d) {
          atomicOr(A.status, kStatusInternal);
          continue;
        }
        s_acc[l] = __fadd_rn(s_acc[l], v);
        if (!flag[l]) {
          flag[l] = 1;
          ulist[atomicAdd(&s_ucnt, 1u)] = (uint16_t)l;
        }
        ek[j] = 0.f;  // e_{t+1,k} = e_{t+1/2,k} - C(e_{t+1/2,k}) = +0 where sent
        nnz += (v != 0.f);
      }
      __syncthreads();
    }
    const uint32_t n = s_ucnt;
    for (uint32_t u = threadIdx.x; u < n; u += kThreads) {
      const uint32_t l = ulist[u];
      const int64_t j = t0 + l;
      const float wo = A.w[j];
      const float wn = __fsub_rn(wo, __fmul_rn(A.a, s_acc[l]));
      A.w[j] = wn;
      const float dd = __fsub_rn(wn, wo);
      A.dlt[j] = dd;
      changed += (dd != 0.f);
      s_acc[l] = 0.f;
      flag[l] = 0;
    }
    if (threadIdx.x == 0) uni += n;
    __syncthreads();
    if (threadIdx.x == 0) s_ucnt = 0;
    __syncthreads();
  }
  unsigned long long tot;
  nnz = block_inclusive_scan<unsigned long long>(nnz, ws, &tot);
  if (threadIdx.x == 0 && tot) atomicAdd(&A.step_ctr->v[kNnz], tot);
  block_inclusive_scan<unsigned long long>(changed, ws, &tot);
  if (threadIdx.x == 0 && tot) atomicAdd(&A.step_ctr->v[kChanged], tot);
  if (threadIdx.x == 0 && uni) atomicAdd(&A.step_ctr->v[kUnion], uni);
}

int tile_u(int tile) { return tile / (kWarps * 128); }

}  // namespace

int accumulate_smem_bytes(int tile) { return tile * 12; }
int aggregate_smem_bytes(int tile) { return tile * 7; }

cudaError_t configure_topk_kernels() {
  cudaError_t err = cudaSuccess;
  auto set = [&](const void* f, int bytes) {
    const cudaError_t e2 = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (err == cudaSuccess) err = e2;
  };
  set((const void*)k_sample, kSampleAll * 4);
  set((const void*)k_accumulate<1>, accumulate_smem_bytes(1024));
  set((const void*)k_accumulate<2>, accumulate_smem_bytes(2048));
  set((const void*)k_accumulate<4>, accumulate_smem_bytes(4096));
  set((const void*)k_accumulate<8>, accumulate_smem_bytes(8192));
  set((const void*)k_aggregate<1>, aggregate_smem_bytes(1024));
  set((const void*)k_aggregate<2>, aggregate_smem_bytes(2048));
  set((const void*)k_aggregate<4>, aggregate_smem_bytes(4096));
  set((const void*)k_aggregate<8>, aggregate_smem_bytes(8192));
  return err;
}

int accumulate_blocks_per_sm(int tile) {
  int n = 0;
  const int smem = accumulate_smem_bytes(tile);
  switch (tile_u(tile)) {
    case 1: cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, k_accumulate<1>, kThreads, smem); break;
    case 2: cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, k_accumulate<2>, kThreads, smem); break;
    case 4: cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, k_accumulate<4>, kThreads, smem); break;
    default: cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, k_accumulate<8>, kThreads, smem); break;
  }
  return n > 0 ? n : 1;
}

int aggregate_blocks_per_sm(int tile) {
  int n = 0;
  const int smem = aggregate_smem_bytes(tile);
  switch (tile_u(tile)) {
    case 1: cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, k_aggregate<1>, kThreads, smem); break;
    case 2: cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, k_aggregate<2>, kThreads, smem); break;
    case 4: cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, k_aggregate<4>, kThreads, smem); break;
    default: cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, k_aggregate<8>, kThreads, smem); break;
  }
  return n > 0 ? n : 1;
}

cudaError_t launch_sample(const TopkArgs& A, cudaStream_t s) {
  const int n_s = A.sample_chunks == 0 ? (int)A.d : A.sample_chunks * 8;
  const int smem = A.dense_mode ? 0 : n_s * 4;
  k_sample<<<A.K, kSampleThreads, smem, s>>>(A);
  return cudaGetLastError();
}

cudaError_t launch_accumulate(const TopkArgs& A, int grid, cudaStream_t s) {
  const int smem = accumulate_smem_bytes(A.tile);
  switch (tile_u(A.tile)) {
    case 1: k_accumulate<1><<<grid, kThreads, smem, s>>>(A); break;
    case 2: k_accumulate<2><<<grid, kThreads, smem, s>>>(A); break;
    case 4: k_accumulate<4><<<grid, kThreads, smem, s>>>(A); break;
    default: k_accumulate<8><<<grid, kThreads, smem, s>>>(A); break;
  }
  return cudaGetLastError();
}

cudaError_t launch_select_pass(const TopkArgs& A, int pass, int blocks_per_worker, cudaStream_t s) {
  const dim3 grid(blocks_per_worker, A.K);
  if (pass == 0) k_select_pass<0><<<grid, kThreads, 0, s>>>(A);
  else if (pass == 1) k_select_pass<1><<<grid, kThreads, 0, s>>>(A);
  else k_select_pass<2><<<grid, kThreads, 0, s>>>(A);
  return cudaGetLastError();
}

cudaError_t launch_select_dense(const TopkArgs& A, cudaStream_t s) {
  k_select_dense<<<A.K, 1024, 0, s>>>(A);
  return cudaGetLastError();
}

cudaError_t launch_chunk_count(const TopkArgs& A, cudaStream_t s) {
  const dim3 grid((unsigned)((A.n_tiles + kWarps - 1) / kWarps), A.K);
  k_chunk_count<<<grid, kThreads, 0, s>>>(A);
  return cudaGetLastError();
}

cudaError_t launch_chunk_scan(const TopkArgs& A, cudaStream_t s) {
  k_chunk_scan<<<A.K, 1024, 0, s>>>(A);
  return cudaGetLastError();
}

cudaError_t launch_chunk_write(const TopkArgs& A, cudaStream_t s) {
  const dim3 grid((unsigned)((A.n_tiles + kWarps - 1) / kWarps), A.K);
  k_chunk_write<<<grid, kThreads, 0, s>>>(A);
  return cudaGetLastError();
}

cudaError_t launch_aggregate(const TopkArgs& A, int grid, cudaStream_t s) {
  const int smem = aggregate_smem_bytes(A.tile);
  switch (tile_u(A.tile)) {
    case 1: k_aggregate<1><<<grid, kThreads, smem, s>>>(A); break;
    case 2: k_aggregate<2><<<grid, kThreads, smem, s>>>(A); break;
    case 4: k_aggregate<4><<<grid, kThreads, smem, s>>>(A); break;
    default: k_aggregate<8><<<grid, kThreads, smem, s>>>(A); break;
  }
  return cudaGetLastError();
}

}  // namespace gmc
