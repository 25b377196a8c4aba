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

constexpr uint64_t kGamma = 0x9E3779B97F4A7C15ull;
constexpr int kPickSmemWords = 12288;  // bitmap words kept in shared memory

// SplitMix64 output function (Steele, Lea & Flood, OOPSLA 2014).
__device__ __forceinline__ uint64_t sm64_mix(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}
// Key of step t's block-choice stream; stream 0 = shared, k+1 = worker k.
__device__ __forceinline__ uint64_t stream_key(uint64_t seed, int64_t t, uint64_t stream) {
  const uint64_t k1 = sm64_mix(seed + kGamma * (uint64_t)(t + 1));
  return sm64_mix(k1 + kGamma * (stream + 1));
}
__device__ __forceinline__ uint64_t draw(uint64_t key, uint64_t i) {
  return sm64_mix(key + kGamma * (i + 1));
}
// [0, n) from the top 32 bits of a draw (multiply-shift).
__device__ __forceinline__ uint32_t below(uint64_t x, uint64_t n) {
  return (uint32_t)(((x >> 32) * n) >> 32);
}

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
__global__ void __launch_bounds__(kThreads) k_rbgs_step(RbgsArgs A) {
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
      float* sk = A.slab + (int64_t)k * slab_ld;
      const int gm = g_mode(gk);
      float4 ev[U], gv[U];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int64_t j = t0 + u * (kThreads * 4) + threadIdx.x * 4;
        ev[u] = __ldcs(reinterpret_cast<const float4*>(ek + j));
        gv[u] = load_g4(gk, j, A.d, gm);
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
  const int k = A.k0 + blockIdx.y;
  const float* ek = A.e + (int64_t)k * A.ld;
  float* ok = A.out + (int64_t)(k - A.k0) * A.out_ld;
  for (int64_t j = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; j < A.d;
       j += (int64_t)gridDim.x * blockDim.x)
    ok[j] = __fsub_rn(A.w[j], __fmul_rn(A.b, ek[j]));
}

__global__ void k_finalize(Counters* step, Counters* total, unsigned long long pairs_add) {
  if (threadIdx.x == 0) {
    step->v[kPairs] += pairs_add;
    step->v[kSteps] = 1;
    for (int i = 0; i < 8; ++i) total->v[i] += step->v[i];
  }
}

}  // namespace

cudaError_t configure_rbgs_kernels() {
  return cudaFuncSetAttribute((const void*)k_rbgs_pick,
                              cudaFuncAttributeMaxDynamicSharedMemorySize, kPickSmemWords * 4);
}

int rbgs_blocks_per_sm() {
  int n = 0;
  cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, k_rbgs_step, kThreads, 0);
  return n > 0 ? n : 1;
}

cudaError_t launch_rbgs_pick(const RbgsArgs& A, cudaStream_t s) {
  const int64_t nbw = (A.nb + 31) / 32;
  const int smem = nbw <= kPickSmemWords ? (int)(nbw * 4) : 0;
  k_rbgs_pick<<<A.per_worker ? A.K : 1, kThreads, smem, s>>>(A);
  return cudaGetLastError();
}

cudaError_t launch_rbgs_step(const RbgsArgs& A, int grid, cudaStream_t s) {
  k_rbgs_step<<<grid, kThreads, 0, s>>>(A);
  return cudaGetLastError();
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
  k_detach<<<grid, 256, 0, s>>>(A);
  return cudaGetLastError();
}

cudaError_t launch_finalize(Counters* step, Counters* total, unsigned long long pairs_add,
                            cudaStream_t s) {
  k_finalize<<<1, 32, 0, s>>>(step, total, pairs_add);
  return cudaGetLastError();
}

}  // namespace gmc
