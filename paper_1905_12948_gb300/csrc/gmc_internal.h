// Host-side internals of libgmc: the handle, the kernel argument blocks and the
// launch wrappers implemented by the kernel translation units.
#pragma once

#include <cstdint>
#include <vector>
#include <cuda_runtime.h>

#include "gmc_device.cuh"

namespace gmc {

// Arguments of the top-k kernels (one block describing the step).
//
// C(e_{t+1/2,k}) is kept as index-sorted (index, value) pairs in sub-chunks:
// sub-chunk (k, tile, w) holds worker k's candidates of the w-th of the
// kChunksPerTile equal parts of the tile, in ascending index order, at
// cand_idx/cand_val[k*cap + base .. + cnt). The accumulate pass writes every
// candidate; the select fixes the k-th key T and the last tie kept t_idx, and
// a candidate is sent iff selected(key, index, T, t_idx): the exact top-k, for
// candidates and for every other coordinate alike.
// Buffers alternate between steps:
// the previous step's sent pairs give the non-zero positions of w_t - w_{t-1}.
struct TopkArgs {
  float* e;                  // residuals / accumulator, K rows of ld floats
  int64_t ld;                // row stride of e (multiple of the tile)
  const float* grads;        // K x d, row stride d (caller memory)
  const uint16_t* grads16;   // the same in bfloat16 (gmc_step_bf16), when bf16
  int bf16;
  int64_t d;
  float* dlt;                // w_t - w_{t-1}, dense, zero outside the last union
  float* w;                  // parameters (ld floats)
  float c, a;                // fl(beta/eta), fl(eta/K) (Alg. 4: beta and fl(1/K); Alg. 3: c = 0)
  // The appendix variants: Alg. 4 scales the gradient by eta in the
  // accumulator (gscale, gs = eta); Alg. 3 adds beta (w_t - w_{t-1}) on the
  // server, densely (server_mom: the aggregate leaves the sum in dlt, and
  // k_server_update applies w_{t+1} = (w_t - a*s) + beta*mom, mom = w_t - w_{t-1}).
  int gscale;
  float gs;
  int server_mom;
  float beta;
  float* mom;                // Alg. 3: w_t - w_{t-1} over [0, d)
  // The local-momentum baseline (Sec. 2.3 eq. (3) with error feedback): each
  // worker's m = beta*m + eta*g (lm, K rows of ld) replaces g in the
  // accumulator (c = 0, a = fl(1/K)); mfm: m = 0 where the worker sent.
  int local_mom;
  int mfm;
  float* lm;
  int K;
  int64_t n_tiles;
  int tile;                  // elements per tile
  uint32_t ksel;             // k
  uint32_t cap;              // candidate slots per worker = regions * cap_region
  int regions;               // candidate regions per worker: one per accumulate CTA (1 = shared)
  uint32_t cap_region;       // slots per region: kChunksPerTile warp parts of cap_part
  uint32_t cap_part;         // slots per warp part (a multiple of 32: whole 128-byte lines)
  uint32_t* rcount;          // K x regions x kChunksPerTile: candidates written in each part
  uint32_t sample_rank;      // rank of the sampled threshold
  int sample_chunks;         // 0 = sample every element (or the approximate top-s sample)
  int sample_blocks;         // blocks per worker of the approximate top-s sample (k_sample)
  uint32_t n_sample;         // sampled positions per worker
  uint32_t sample_stride;    // per-worker stride of sample_keys; offset of the delta half of sample_pend
  // Approximate top-s (Sec. 5.1): the sample is one position per stratum of
  // d / n_sample drawn from the shared SplitMix64 stream of (seed, t); theta
  // is the exact sample_rank-th largest sampled key and C(v) = {key >= theta},
  // or the exact top-`limit` when more than `limit` components reach theta.
  int approx;
  uint64_t seed;
  int64_t t;
  uint32_t limit;
  int theta_blocks;          // blocks per worker of k_sample_theta
  int has_prev;              // a previous step's pair lists exist (t > 0, not just restored)
  int dense_prev;            // restored state: w_t - w_{t-1} is in dlt over [0, d), no pair lists
  int dense_mode;            // GMC_SELECT_DENSE
  WorkerSel* sel;            // K entries
  uint32_t* ghist;           // K x kHistBins: the approximate top-s sample's histogram (zero between uses)
  uint32_t* chist;           // K x kRelBins: the candidates' relative histogram (zeroed by the sample)
  uint32_t* bucket;          // K x 2*kBucketCap: keys, then indices of the k-th key's bin
  int sel_shift;             // log2 of the relative-histogram bin width (in keys)
  uint32_t* sample_keys;     // K x sample_stride
  uint32_t* big_tiles;       // [0]: count, then tile ids left to the block aggregate
  uint32_t* cand_idx;        // current chunks: K x cap
  float* cand_val;
  uint2* chunk;              // sub-chunk (base, count): n_tiles x kChunksPerTile x K, see chunk_at
  uint32_t* mask;            // d: workers that sent each coordinate (bit k), zero between steps
  int g_direct;              // grads is mapped host memory: read it with loads, not bulk copies
  const uint32_t* cand_idx_prev;    // previous step's sub-chunks
  const float* cand_val_prev;
  const uint2* chunk_prev;
  // Deferred aggregation: the sum of a step's sent pairs into w and the
  // zeroing of its residuals can be left to the next step's bulk pass, which
  // streams every coordinate anyway (see k_accumulate_bulk).
  int pending;               // the previous step's aggregation is still to be applied
  float a_prev;              // fl(eta/K) of that step
  uint32_t* sample_pend;     // 3 x sample_stride: its senders' mask and w_{t+1} - w_t at the
                             // sampled coordinates (k_sample_pending, for k_sample); the
                             // approximate top-s adds the coordinates
  Counters* total_ctr;       // running totals: the deferred aggregation counts there
  Counters* step_ctr;
  unsigned* status;
  uint32_t* tile_ctr;        // tiles claimed by k_accumulate_bulk (zeroed by the sample kernel)
  // k_accumulate_bulk's tile order (tile_order): blk_cost accumulates the
  // candidates each block of gridDim.x tiles produced; k_sample_pending turns
  // it into blk_order -- the golden-stride sequence of blocks (b * blk_mul)
  // mod n_blk with the coldest few moved to the end -- and clears it.
  uint32_t* blk_cost;        // n_tiles / grid blocks (bulk top-k only, else NULL)
  uint32_t* blk_order;       // the same count
  uint32_t n_blk;            // whole blocks of the bulk pass's grid of tiles: n_tiles / grid
  uint32_t blk_mul;          // the golden stride, coprime to n_blk
  int use_order;             // this step's pass follows blk_order (it was built this step)
  uint64_t wait_ns;          // bound of the bulk pass's mbarrier waits (kWaitLimitNs)
  int64_t hold_tile;         // test hook: the bulk pass issues no copy for item (hold_tile, hold_k),
  int hold_k;                // so that the waits on it give up; hold_tile = -1: none
  int finalize;              // k_select_dense ends the step: adds step_ctr (+ pairs_add pairs) to the totals
  unsigned long long pairs_add;
};

// Slot of sub-chunk (k, tile, w) in the sub-chunk tables: a tile's entries are
// contiguous, each eighth of the tile holding its K workers side by side, so
// one warp writes the K entries of its eighth with one store.
__host__ __device__ __forceinline__ int64_t chunk_at(const TopkArgs& A, int k, int64_t tile, int w) {
  return (tile * kChunksPerTile + w) * A.K + k;
}

// Arguments of the RBGS kernels.
struct RbgsArgs {
  float* e;
  int64_t ld;
  const float* grads;
  const uint16_t* grads16;   // bfloat16 gradients (gmc_step_bf16), when bf16
  int bf16;
  int64_t d;
  float* dlt;
  float* w;
  float c, a;
  int K;
  int64_t n_tiles;
  int64_t B;                 // block size
  uint32_t B_shift;          // log2(B) if B is a power of two, else 0xffffffff
  int64_t nb, m;             // blocks, blocks kept
  int per_worker;
  uint64_t seed;
  int64_t t;
  uint32_t* bitmap;          // streams x ceil(nb/32) words, kept zero between steps
  int32_t* rank;             // streams x nb: slot of a chosen block, -1 otherwise
  int32_t* blocks;           // streams x m: chosen blocks ascending
  uint8_t* uflag_prev;       // nb: union of the previous step's blocks
  uint8_t* uflag_cur;        // nb: union of this step's blocks
  float* slab;               // K x (m*B): C(e_{t+1/2,k}) values, block slot major
  int has_prev;
  int bulk;                  // k_rbgs_bulk (bulk copies through shared memory), else k_rbgs_step
  int g_direct;              // grads is mapped host memory: read it with loads, not bulk copies
  uint32_t* tile_ctr;        // tiles claimed by k_rbgs_bulk (zeroed by k_rbgs_pick)
  uint64_t wait_ns;          // bound of the bulk pass's mbarrier waits (kWaitLimitNs)
  int64_t hold_tile;         // test hook, as in TopkArgs: no copy for item (hold_tile, hold_k)
  int hold_k;
  Counters* step_ctr;
  unsigned* status;
};

struct DetachArgs {
  const float* w;
  const float* e;
  int64_t ld;
  int64_t d;
  float b;                   // fl(lambda*eta)
  float* out;
  int64_t out_ld;
  int k0, k1;                // workers [k0, k1)
};

// Launch with programmatic stream serialization (the kernel begins with
// griddep_wait): its scheduling overlaps the end of the kernel before it.
template <typename... P, typename... Args>
cudaError_t launch_pdl(void (*kernel)(P...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                       Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, args...);
}

// Launch wrappers (each returns the cudaGetLastError of its launches).
cudaError_t launch_sample(const TopkArgs& A, cudaStream_t s);
cudaError_t launch_accumulate(const TopkArgs& A, int grid, cudaStream_t s);
cudaError_t launch_select(const TopkArgs& A, int blocks_per_worker, cudaStream_t s);
// Approximate top-s: T = theta, every tie kept, the count; or the dense path.
cudaError_t launch_select_approx(const TopkArgs& A, cudaStream_t s);
// Alg. 3's server step over [0, d): w_{t+1} = (w_t - a*s) + beta*(w_t - w_{t-1}).
cudaError_t launch_server_update(const TopkArgs& A, cudaStream_t s);
cudaError_t launch_select_dense(const TopkArgs& A, cudaStream_t s);
constexpr int kBulkTile = 4096;  // tile of the bulk-copy accumulate pass (k_accumulate_bulk)
constexpr int kBulkMaxK = 16;    // workers the bulk-copy pass takes (its shared memory grows with K)

// k_mark: the senders of every coordinate into mask (for k_owner_sum).
cudaError_t launch_mark(const TopkArgs& A, int grid, cudaStream_t s);
// Sum of the sent pairs into w (with a_prev), residuals to +0 where sent,
// w_{t+1} - w_t into dlt, mask cleared; counts into step_ctr and total_ctr
// (either may be null).
cudaError_t launch_owner_sum(const TopkArgs& A, int grid, cudaStream_t s);
cudaError_t launch_gather_selected(const TopkArgs& A, int k, uint32_t* idx_out, float* val_out,
                                   cudaStream_t s);
cudaError_t launch_rbgs_pick(const RbgsArgs& A, cudaStream_t s);
cudaError_t launch_rbgs_step(const RbgsArgs& A, int grid, cudaStream_t s);
cudaError_t launch_rbgs_expand(const RbgsArgs& A, int k, uint32_t* idx_out, float* val_out,
                               cudaStream_t s);
cudaError_t launch_detach(const DetachArgs& A, cudaStream_t s);
cudaError_t launch_finalize(Counters* step, Counters* total, unsigned long long pairs_add,
                            cudaStream_t s);

// Occupancy-derived persistent grid sizes.
int accumulate_blocks_per_sm(int tile);
int rbgs_blocks_per_sm();
int select_blocks_per_sm();  // resident k_select_finish blocks per SM (its grid is one wave)
int accumulate_smem_bytes(int tile, int K);
cudaError_t configure_topk_kernels();
cudaError_t configure_rbgs_kernels();

constexpr int kRbgsTile = 4096;  // elements per tile of the fused RBGS kernel

}  // namespace gmc
