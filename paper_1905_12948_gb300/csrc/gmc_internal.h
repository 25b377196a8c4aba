// Host-side internals of libgmc: the handle, the kernel argument blocks and the
// launch wrappers implemented by the kernel translation units.
#pragma once

#include <cstdint>
#include <vector>
#include <cuda_runtime.h>

#include "gmc_device.cuh"

namespace gmc {

// Arguments of the top-k kernels (one block describing the step).
struct TopkArgs {
  float* e;                  // residuals / accumulator, K rows of ld floats
  int64_t ld;                // row stride of e (multiple of the tile)
  const float* grads;        // K x d, row stride d (caller memory)
  int64_t d;
  float* dlt;                // w_t - w_{t-1}, dense, zero outside the last union
  float* w;                  // parameters (ld floats)
  float c, a;                // fl(beta/eta), fl(eta/K)
  int K;
  int64_t n_tiles;
  int tile;                  // elements per tile
  uint32_t ksel;             // k
  uint32_t cap;              // candidate capacity per worker
  uint32_t sample_rank;      // rank of the sampled threshold
  int sample_chunks;         // 0 = sample every element
  int has_prev;              // a previous step exists (t > 0)
  int dense_mode;            // GMC_SELECT_DENSE
  WorkerSel* sel;            // K entries
  uint32_t* cand_idx;        // K x cap
  float* cand_val;           // K x cap
  uint32_t* chunk_base;      // K x n_tiles
  uint32_t* chunk_cnt;       // K x n_tiles
  uint32_t* gt_cnt;          // K x n_tiles
  uint32_t* eq_cnt;          // K x n_tiles
  uint32_t* eq_before;       // K x n_tiles
  uint32_t* ghist;           // K x kHistBins
  const uint32_t* pos_prev;  // K x (n_tiles+1): previous step's per-tile offsets
  const uint32_t* idx_prev;  // K x ksel: previous step's sorted indices
  uint32_t* pos_cur;         // K x (n_tiles+1)
  uint32_t* idx_cur;         // K x ksel
  float* val_cur;            // K x ksel
  Counters* step_ctr;
  unsigned* status;
};

// Arguments of the RBGS kernels.
struct RbgsArgs {
  float* e;
  int64_t ld;
  const float* grads;
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

// Launch wrappers (each returns the cudaGetLastError of its launches).
cudaError_t launch_sample(const TopkArgs& A, cudaStream_t s);
cudaError_t launch_accumulate(const TopkArgs& A, int grid, cudaStream_t s);
cudaError_t launch_select_pass(const TopkArgs& A, int pass, int blocks_per_worker, cudaStream_t s);
cudaError_t launch_select_dense(const TopkArgs& A, cudaStream_t s);
cudaError_t launch_chunk_count(const TopkArgs& A, cudaStream_t s);
cudaError_t launch_chunk_scan(const TopkArgs& A, cudaStream_t s);
cudaError_t launch_chunk_write(const TopkArgs& A, cudaStream_t s);
cudaError_t launch_aggregate(const TopkArgs& A, int grid, cudaStream_t s);
cudaError_t launch_rbgs_pick(const RbgsArgs& A, cudaStream_t s);
cudaError_t launch_rbgs_step(const RbgsArgs& A, int grid, cudaStream_t s);
cudaError_t launch_rbgs_expand(const RbgsArgs& A, int k, uint32_t* idx_out, float* val_out,
                               cudaStream_t s);
cudaError_t launch_detach(const DetachArgs& A, cudaStream_t s);
cudaError_t launch_finalize(Counters* step, Counters* total, unsigned long long pairs_add,
                            cudaStream_t s);

// Occupancy-derived persistent grid sizes.
int accumulate_blocks_per_sm(int tile);
int aggregate_blocks_per_sm(int tile);
int rbgs_blocks_per_sm();
int accumulate_smem_bytes(int tile);
int aggregate_smem_bytes(int tile);
cudaError_t configure_topk_kernels();
cudaError_t configure_rbgs_kernels();

constexpr int kRbgsTile = 4096;  // elements per tile of the fused RBGS kernel

}  // namespace gmc
