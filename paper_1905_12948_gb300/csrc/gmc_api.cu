// C ABI of libgmc (declared in include/gmc.h): handle lifecycle, argument
// validation, device state, and the orchestration of one GMC / GMC+ step on a
// caller-given stream. Only host code lives here; the kernels are in
// gmc_topk.cu and gmc_rbgs.cu.
#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <new>
#include <vector>

#include "gmc.h"
#include "gmc_internal.h"

using namespace gmc;

namespace {

struct ProfRec {
  int kernel;
  cudaEvent_t start, stop;
};

}  // namespace

struct gmc_ctx {
  int device = 0;
  int num_sms = 1;
  // problem
  int64_t d = 0;
  int K = 0;
  float beta = 0.f, eta = 0.f, lambda = 0.f;
  int compressor = GMC_TOPK;
  double ratio = 0.0;
  int64_t block = 0;
  uint64_t seed = 0;
  int per_worker = 0;
  int select_mode = GMC_SELECT_SAMPLED;
  int variant = GMC_VARIANT_GMC;  // Alg. 1, or the appendix's Alg. 3 / Alg. 4
  float* mom = nullptr;           // Alg. 3: w_t - w_{t-1} (allocated by gmc_set_variant)
  float* lm = nullptr;            // local momentum: K rows of ld (allocated by gmc_set_variant)
  float* detach_out = nullptr;
  int64_t detach_ld = 0;
  // geometry
  int tile = 0;
  int64_t n_tiles = 0, ld = 0;
  uint32_t ksel = 0, cap = 0, sample_rank = 0;
  int sample_chunks = 0;
  int64_t nb = 0, m = 0;
  uint32_t B_shift = 0xffffffffu;
  int grid_acc = 1, grid_agg = 1, grid_rbgs = 1, sel_blocks = 1;
  bool rbgs_bulk = false;
  // state
  int64_t t = 0;
  bool initialized = false;
  bool restored = false;  // gmc_load_state: the next step reads w_t - w_{t-1} densely
  float* e = nullptr;
  float* w = nullptr;
  float* dlt = nullptr;
  WorkerSel* sel = nullptr;
  uint32_t* ghist = nullptr;
  uint32_t* chist = nullptr;
  uint32_t* bucket = nullptr;  // K x 2*kBucketCap
  int sel_shift = 20;
  uint32_t* sample_keys = nullptr;
  uint32_t* big_tiles = nullptr;
  uint32_t* rcount = nullptr;
  int regions = 1;
  uint32_t cap_region = 0, cap_part = 0;
  int sample_blocks = 1;
  uint32_t* cand_idx[2] = {nullptr, nullptr};
  float* cand_val[2] = {nullptr, nullptr};
  uint2* chunk[2] = {nullptr, nullptr};
  uint32_t* mask = nullptr;
  uint32_t* sample_pend = nullptr;  // 3 x sample_stride
  // sample geometry; approximate top-s: its limit and theta blocks
  uint32_t n_sample = 0, sample_stride = 0, limit = 0;
  int theta_blocks = 1;
  // deferred aggregation (bulk top-k pass): the last step's sent pairs are
  // summed into w by the next step's bulk pass, or by flush() when state is read
  bool agg_pending = false;
  float a_pending = 0.f;       // fl(eta/K) of that step
  cudaStream_t aux = nullptr;  // library stream for flushes outside a caller stream
  cudaEvent_t ev_step = nullptr, ev_flush = nullptr;
  bool wait_flush = false;     // the next launch waits for ev_flush
  uint32_t* bitmap = nullptr;
  int32_t* rank = nullptr;
  int32_t* blocks = nullptr;
  uint8_t* uflag[2] = {nullptr, nullptr};
  float* slab = nullptr;
  Counters* step_ctr = nullptr;
  uint32_t* tile_ctr = nullptr;  // tiles claimed by the persistent passes
  uint32_t* blk_cost = nullptr;  // the bulk top-k pass's tile order (tile_order): costs, order
  uint32_t* blk_order = nullptr;
  uint32_t n_blk = 0, blk_mul = 1;
  Counters* total_ctr = nullptr;
  unsigned* status = nullptr;
  // test hook (gmc_test_withhold_copy): the next step's bulk pass withholds
  // the copy of item (hold_tile, hold_k) and bounds its waits by hold_wait_ns
  int64_t hold_tile = -1;
  int hold_k = 0;
  uint64_t hold_wait_ns = 0;
  float* gstage = nullptr;
  std::vector<void*> allocations;
  // profiling
  bool prof = false;
  uint32_t prof_mask = 0xffffffffu;  // kernel ids bracketed by events while profiling
  std::vector<ProfRec> pending;
  std::vector<cudaEvent_t> free_events;
  double prof_ms[GMC_KERNEL_COUNT] = {};
  int64_t prof_launches[GMC_KERNEL_COUNT] = {};
  double prof_bytes[GMC_KERNEL_COUNT] = {};
};

namespace {

class DeviceGuard {
 public:
  explicit DeviceGuard(int dev) {
    cudaGetDevice(&prev_);
    if (prev_ != dev) cudaSetDevice(dev);
    dev_ = dev;
  }
  ~DeviceGuard() {
    if (prev_ != dev_) cudaSetDevice(prev_);
  }

 private:
  int prev_ = 0, dev_ = 0;
};

// Test hook (gmc_test_fail_alloc): the device allocation that finds the
// countdown at 0 fails as cudaMalloc does when memory runs out; -1 = off.
std::atomic<int64_t> g_fail_countdown{-1};
std::atomic<int64_t> g_live_allocations{0};  // device allocations held by all handles

bool injected_alloc_failure() {
  int64_t c = g_fail_countdown.load();
  while (c >= 0 && !g_fail_countdown.compare_exchange_weak(c, c - 1)) {
  }
  return c == 0;
}

template <typename T>
cudaError_t dalloc(gmc_ctx* h, T** p, size_t count) {
  void* q = nullptr;
  *p = nullptr;
  const size_t bytes = std::max<size_t>(count, 1) * sizeof(T);
  if (injected_alloc_failure()) return cudaErrorMemoryAllocation;
  cudaError_t err = cudaMalloc(&q, bytes);
  if (err != cudaSuccess) return err;
  h->allocations.push_back(q);
  g_live_allocations.fetch_add(1);
  *p = static_cast<T*>(q);
  return cudaMemset(q, 0, bytes);
}

void free_all(gmc_ctx* h) {
  for (void* p : h->allocations) cudaFree(p);
  g_live_allocations.fetch_sub((int64_t)h->allocations.size());
  h->allocations.clear();
  if (h->ev_step) cudaEventDestroy(h->ev_step);
  if (h->ev_flush) cudaEventDestroy(h->ev_flush);
  if (h->aux) cudaStreamDestroy(h->aux);
  h->ev_step = h->ev_flush = nullptr;
  h->aux = nullptr;
  for (auto& r : h->pending) {
    cudaEventDestroy(r.start);
    cudaEventDestroy(r.stop);
  }
  h->pending.clear();
  for (cudaEvent_t e : h->free_events) cudaEventDestroy(e);
  h->free_events.clear();
}

int status_of(cudaError_t err) {
  if (err == cudaSuccess) return GMC_OK;
  if (err == cudaErrorMemoryAllocation) return GMC_ENOMEM;
  return GMC_ECUDA;
}

cudaEvent_t take_event(gmc_ctx* h) {
  if (!h->free_events.empty()) {
    cudaEvent_t e = h->free_events.back();
    h->free_events.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  cudaEventCreate(&e);
  return e;
}

// Enqueue one kernel launch, bracketed by events when profiling is on.
template <typename F>
cudaError_t timed(gmc_ctx* h, int kernel, double bytes, cudaStream_t s, F&& launch) {
  if (!h->prof || !((h->prof_mask >> kernel) & 1u)) return launch();
  ProfRec r{kernel, take_event(h), take_event(h)};
  cudaEventRecord(r.start, s);
  cudaError_t err = launch();
  cudaEventRecord(r.stop, s);
  h->pending.push_back(r);
  h->prof_bytes[kernel] += bytes;
  return err;
}

void drain_profile(gmc_ctx* h) {
  for (auto& r : h->pending) {
    cudaEventSynchronize(r.stop);
    float ms = 0.f;
    if (cudaEventElapsedTime(&ms, r.start, r.stop) == cudaSuccess) {
      h->prof_ms[r.kernel] += ms;
      h->prof_launches[r.kernel] += 1;
    }
    h->free_events.push_back(r.start);
    h->free_events.push_back(r.stop);
  }
  h->pending.clear();
}

bool local_variant(const gmc_ctx* h) {
  return h->variant == GMC_VARIANT_LOCAL_MOMENTUM || h->variant == GMC_VARIANT_LOCAL_MOMENTUM_MFM;
}
// Detach coefficient: fl(lambda*eta) (Alg. 2); lambda for the local-momentum
// baseline, whose residual already carries eta.
float detach_b(const gmc_ctx* h) { return local_variant(h) ? h->lambda : h->lambda * h->eta; }

void set_constants(gmc_ctx* h, TopkArgs* A) {
  A->c = h->beta / h->eta;
  A->a = h->eta / (float)h->K;
  A->beta = h->beta;
  A->mom = h->mom;
  if (h->variant == GMC_VARIANT_SERVER_MOMENTUM) {  // Alg. 3: e + g; the momentum is the server's
    A->c = 0.f;
    A->server_mom = 1;
  } else if (h->variant == GMC_VARIANT_LR_IN_RESIDUAL) {  // Alg. 4: e + eta*g - beta*dw, w -= (1/K) sum
    A->c = h->beta;
    A->a = 1.f / (float)h->K;
    A->gscale = 1;
    A->gs = h->eta;
  } else if (h->variant == GMC_VARIANT_LOCAL_MOMENTUM || h->variant == GMC_VARIANT_LOCAL_MOMENTUM_MFM) {
    A->c = 0.f;  // e + m, m = beta*m + eta*g; w -= (1/K) sum
    A->a = 1.f / (float)h->K;
    A->gs = h->eta;
    A->local_mom = 1;
    A->mfm = h->variant == GMC_VARIANT_LOCAL_MOMENTUM_MFM ? 1 : 0;
    A->lm = h->lm;
  }
}

// Arguments of step t's top-k kernels; chunk buffers alternate with the parity of t.
TopkArgs topk_args_at(gmc_ctx* h, const float* grads, int64_t t) {
  TopkArgs A{};
  std::memset(&A, 0, sizeof(A));
  const int cur = (int)(t & 1), prev = cur ^ 1;
  A.e = h->e;
  A.ld = h->ld;
  A.grads = grads;
  A.d = h->d;
  A.dlt = h->dlt;
  A.w = h->w;
  set_constants(h, &A);
  A.K = h->K;
  A.n_tiles = h->n_tiles;
  A.tile = h->tile;
  A.ksel = h->ksel;
  A.cap = h->cap;
  A.sample_rank = h->sample_rank;
  A.sample_chunks = h->sample_chunks;
  A.sample_blocks = h->sample_blocks;
  A.dense_prev = h->restored && t == h->t ? 1 : 0;
  A.has_prev = t > 0 && !A.dense_prev;
  A.dense_mode = h->select_mode == GMC_SELECT_DENSE;
  A.sel = h->sel;
  A.ghist = h->ghist;
  A.chist = h->chist;
  A.bucket = h->bucket;
  A.sel_shift = h->sel_shift;
  A.sample_keys = h->sample_keys;
  A.n_sample = h->n_sample;
  A.sample_stride = h->sample_stride;
  A.approx = h->compressor == GMC_TOPK_APPROX ? 1 : 0;
  A.seed = h->seed;
  A.t = t;
  A.limit = h->limit;
  A.theta_blocks = h->theta_blocks;
  A.big_tiles = h->big_tiles;
  A.g_direct = 0;
  A.regions = h->regions;
  A.cap_region = h->cap_region;
  A.cap_part = h->cap_part;
  A.rcount = h->rcount;
  A.cand_idx = h->cand_idx[cur];
  A.cand_val = h->cand_val[cur];
  A.chunk = h->chunk[cur];
  A.mask = h->mask;
  A.cand_idx_prev = h->cand_idx[prev];
  A.cand_val_prev = h->cand_val[prev];
  A.sample_pend = h->sample_pend;
  A.total_ctr = h->total_ctr;
  A.pending = 0;
  A.a_prev = A.a;
  A.chunk_prev = h->chunk[prev];
  A.step_ctr = h->step_ctr;
  A.tile_ctr = h->tile_ctr;
  A.blk_cost = h->blk_cost;
  A.blk_order = h->blk_order;
  A.n_blk = h->n_blk;
  A.blk_mul = h->blk_mul;
  A.use_order = 0;
  A.wait_ns = kWaitLimitNs;
  A.hold_tile = -1;
  A.status = h->status;
  return A;
}

TopkArgs topk_args(gmc_ctx* h, const float* grads) { return topk_args_at(h, grads, h->t); }

// The stride of the bulk top-k pass's block order (tile_order): the first
// integer from nb times the golden ratio's fractional part that is coprime to
// nb, so that (b * stride) mod nb visits every block once.
uint32_t golden_stride(int64_t nb) {
  if (nb < 3) return 1;
  int64_t m = (int64_t)std::llround(0.6180339887498949 * (double)nb);
  for (;; ++m) {
    int64_t a = m, b = nb;
    while (b) {
      const int64_t r = a % b;
      a = b;
      b = r;
    }
    if (a == 1) return (uint32_t)(m % nb);
  }
}


RbgsArgs rbgs_args(gmc_ctx* h, const float* grads) {
  RbgsArgs A;
  std::memset(&A, 0, sizeof(A));
  const int cur = (int)(h->t & 1), prev = cur ^ 1;
  A.e = h->e;
  A.ld = h->ld;
  A.grads = grads;
  A.d = h->d;
  A.dlt = h->dlt;
  A.w = h->w;
  A.c = h->beta / h->eta;
  A.a = h->eta / (float)h->K;
  A.K = h->K;
  A.bulk = h->rbgs_bulk ? 1 : 0;
  A.n_tiles = h->n_tiles;
  A.B = h->block;
  A.B_shift = h->B_shift;
  A.nb = h->nb;
  A.m = h->m;
  A.per_worker = h->per_worker;
  A.seed = h->seed;
  A.t = h->t;
  A.bitmap = h->bitmap;
  A.rank = h->rank;
  A.blocks = h->blocks;
  A.uflag_prev = h->uflag[prev];
  A.uflag_cur = h->uflag[cur];
  A.slab = h->slab;
  A.has_prev = h->t > 0;
  A.step_ctr = h->step_ctr;
  A.tile_ctr = h->tile_ctr;
  A.wait_ns = kWaitLimitNs;
  A.hold_tile = -1;
  A.status = h->status;
  return A;
}

#define GMC_TRY(expr)                          \
  do {                                         \
    const cudaError_t err_ = (expr);           \
    if (err_ != cudaSuccess) return status_of(err_); \
  } while (0)

// Work on s that reads or writes the state waits for a flush that may have
// been enqueued on another stream since the last step; a step (clear = true)
// resets the flag, later work is ordered after that step by the caller.
cudaError_t order_after_flush(gmc_ctx* h, cudaStream_t s, bool clear) {
  if (!h->wait_flush) return cudaSuccess;
  if (clear) h->wait_flush = false;
  return cudaStreamWaitEvent(s, h->ev_flush, 0);
}

// One step of Alg. 1 / Alg. 2 on stream s. With the bulk top-k pass the
// step's aggregation (sum of the sent pairs into w, residuals to +0 where
// sent) is left pending unless `eager`: the next step's bulk pass applies it
// while it streams the tile, or flush() does when the state is read.
// `direct`: grads is mapped host memory, read in place by the kernels.
int enqueue_step(gmc_ctx* h, const void* grads_any, cudaStream_t s, bool eager, bool direct = false,
                 bool bf16 = false) {
  // fp32 rows, or bfloat16 rows (gmc_step_bf16) widened exactly as they are read
  const float* grads = bf16 ? nullptr : static_cast<const float*>(grads_any);
  const uint16_t* grads16 = bf16 ? static_cast<const uint16_t*>(grads_any) : nullptr;
  const double Kd = (double)h->K * (double)h->d;
  GMC_TRY(order_after_flush(h, s, true));
  // the exact top-k's sample kernel clears the step's counters itself (a
  // memset between two kernels would keep the second from starting early)
  if (h->compressor != GMC_TOPK) GMC_TRY(cudaMemsetAsync(h->step_ctr, 0, sizeof(Counters), s));
  unsigned long long pairs_add = 0;
  bool finalized = false;  // the step's counters already added up by its last kernel
  if (h->compressor != GMC_RBGS) {
    const bool approx = h->compressor == GMC_TOPK_APPROX;
    TopkArgs A = topk_args(h, grads);
    A.grads16 = grads16;
    A.bf16 = bf16 ? 1 : 0;
    A.g_direct = direct ? 1 : 0;
    if (h->hold_tile >= 0) {  // test hook, one step
      A.hold_tile = h->hold_tile;
      A.hold_k = h->hold_k;
      A.wait_ns = h->hold_wait_ns;
      h->hold_tile = -1;
    }
    A.pending = h->agg_pending ? 1 : 0;
    A.a_prev = h->a_pending;
    // the tile order is built by k_sample_pending, which runs on these steps
    A.use_order = (h->blk_order && (A.pending || approx) && !A.dense_mode) ? 1 : 0;
    const bool defer = h->tile == kBulkTile && !eager && !h->detach_out && !A.server_mom && !A.mfm;
    const double kk = (double)h->K * (double)h->ksel;
    pairs_add = approx ? 0ull : (unsigned long long)h->K * h->ksel;  // approximate: counted on the device
    // deferred: the dense select is the step's last launch and ends it
    A.finalize = defer ? 1 : 0;
    A.pairs_add = pairs_add;
    finalized = defer;
    GMC_TRY(timed(h, GMC_KERNEL_SAMPLE, 0.0, s, [&] { return launch_sample(A, s); }));
    // read g, e (and the local momentum), write v over e (and the momentum)
    GMC_TRY(timed(h, GMC_KERNEL_ACCUMULATE, ((A.local_mom ? 20.0 : 12.0) - (bf16 ? 2.0 : 0.0)) * Kd, s,
                  [&] { return launch_accumulate(A, h->grid_acc, s); }));
    h->agg_pending = false;
    GMC_TRY(timed(h, GMC_KERNEL_SELECT, 0.0, s, [&] {
      return approx ? launch_select_approx(A, s) : launch_select(A, h->sel_blocks, s);
    }));
    GMC_TRY(timed(h, GMC_KERNEL_DENSE, 0.0, s, [&] { return launch_select_dense(A, s); }));
    if (defer) {
      // the next step's sample and bulk pass apply the aggregation
      h->agg_pending = true;
      h->a_pending = A.a;
    } else {
      TopkArgs B = A;
      B.a_prev = A.a;
      B.total_ctr = nullptr;  // k_finalize adds the step's counts to the totals
      GMC_TRY(timed(h, GMC_KERNEL_AGGREGATE, 24.0 * kk + (B.server_mom ? 20.0 * h->d : 0.0), s, [&] {
        cudaError_t err = launch_mark(B, h->grid_agg, s);
        if (err == cudaSuccess) err = launch_owner_sum(B, h->grid_agg, s);
        if (err == cudaSuccess && B.server_mom) err = launch_server_update(B, s);  // Alg. 3
        return err;
      }));
    }
  } else {
    RbgsArgs A = rbgs_args(h, grads);
    A.grads16 = grads16;
    A.bf16 = bf16 ? 1 : 0;
    A.g_direct = direct ? 1 : 0;
    if (h->hold_tile >= 0) {  // test hook, one step
      A.hold_tile = h->hold_tile;
      A.hold_k = h->hold_k;
      A.wait_ns = h->hold_wait_ns;
      h->hold_tile = -1;
    }
    // restored state: w_t - w_{t-1} may be non-zero in any block (zero outside
    // the last union, where dlt holds it): flag every block as the last union's
    if (h->restored && h->t > 0) GMC_TRY(cudaMemsetAsync(A.uflag_prev, 1, (size_t)h->nb, s));
    GMC_TRY(cudaMemsetAsync(A.uflag_cur, 0, (size_t)h->nb, s));
    GMC_TRY(timed(h, GMC_KERNEL_RBGS_PICK, 0.0, s, [&] { return launch_rbgs_pick(A, s); }));
    GMC_TRY(timed(h, GMC_KERNEL_RBGS_STEP, (bf16 ? 10.0 : 12.0) * Kd, s,
                  [&] { return launch_rbgs_step(A, h->grid_rbgs, s); }));
  }
  if (h->detach_out) {
    DetachArgs D{h->w, h->e, h->ld, h->d, detach_b(h), h->detach_out, h->detach_ld, 0, h->K};
    GMC_TRY(timed(h, GMC_KERNEL_DETACH, 8.0 * Kd + 4.0 * h->d, s, [&] { return launch_detach(D, s); }));
  }
  if (!finalized)
    GMC_TRY(timed(h, GMC_KERNEL_OTHER, 0.0, s,
                  [&] { return launch_finalize(h->step_ctr, h->total_ctr, pairs_add, s); }));
  if (h->ev_step) GMC_TRY(cudaEventRecord(h->ev_step, s));
  h->t += 1;
  h->restored = false;
  return GMC_OK;
}

// Apply a pending aggregation on stream s (ordered after the last step):
// the senders of every coordinate into mask, then k_owner_sum.
int flush(gmc_ctx* h, cudaStream_t s) {
  if (!h->agg_pending) return GMC_OK;
  GMC_TRY(cudaStreamWaitEvent(s, h->ev_step, 0));
  TopkArgs A = topk_args_at(h, nullptr, h->t - 1);
  A.a_prev = h->a_pending;
  A.step_ctr = h->step_ctr;    // the counts belong to the last step
  A.total_ctr = h->total_ctr;  // which k_finalize has already added up
  GMC_TRY(launch_mark(A, h->grid_agg, s));
  GMC_TRY(launch_owner_sum(A, h->grid_agg, s));
  GMC_TRY(cudaEventRecord(h->ev_flush, s));
  h->wait_flush = true;
  h->agg_pending = false;
  return GMC_OK;
}

#define GMC_TRY_ST(expr)                 \
  do {                                   \
    const int st_ = (expr);              \
    if (st_ != GMC_OK) return st_;       \
  } while (0)

bool finite_f(float x) { return std::isfinite(x); }

}  // namespace

extern "C" {

const char* gmc_strerror(int status) {
  switch (status) {
    case GMC_OK: return "success";
    case GMC_EINVAL: return "invalid argument";
    case GMC_ENOMEM: return "out of memory";
    case GMC_ECUDA: return "CUDA error";
    case GMC_ENONFINITE: return "non-finite accumulator value";
    case GMC_ESTATE: return "call out of order";
    case GMC_EINTERNAL: return "internal consistency check failed";
    case GMC_ETOOBIG: return "size exceeds the fixed scratch of gmc_topk_noalloc (n <= 2^26)";
    case GMC_ETIMEOUT: return "a bounded wait in a step's kernel gave up: the step skipped work and its state is invalid";
    default: return "unknown status";
  }
}

const char* gmc_kernel_name(int32_t kernel) {
  static const char* names[GMC_KERNEL_COUNT] = {
      "accumulate", "rbgs_step", "sample", "select", "dense_select",
      "compact", "aggregate", "rbgs_pick", "detach", "other"};
  return (kernel >= 0 && kernel < GMC_KERNEL_COUNT) ? names[kernel] : "?";
}

int gmc_create(gmc_t* out, int64_t d, int32_t K, float beta, float eta, int32_t compressor,
               double ratio, int64_t block) {
  if (!out) return GMC_EINVAL;
  *out = nullptr;
  if (d < 1 || d >= (int64_t(1) << 31) - (int64_t(1) << 16)) return GMC_EINVAL;
  if (K < 1) return GMC_EINVAL;
  if (!finite_f(beta) || !(beta >= 0.f) || !(beta < 1.f)) return GMC_EINVAL;
  if (!finite_f(eta) || !(eta > 0.f)) return GMC_EINVAL;
  if (!std::isfinite(ratio) || !(ratio > 0.0) || !(ratio <= 1.0)) return GMC_EINVAL;
  if (compressor != GMC_TOPK && compressor != GMC_RBGS && compressor != GMC_TOPK_APPROX) return GMC_EINVAL;
  if (compressor == GMC_RBGS && block < 1) return GMC_EINVAL;
  if (K > 32) return GMC_EINVAL;

  gmc_ctx* h = new (std::nothrow) gmc_ctx();
  if (!h) return GMC_ENOMEM;
  cudaGetDevice(&h->device);
  cudaDeviceGetAttribute(&h->num_sms, cudaDevAttrMultiProcessorCount, h->device);
  if (h->num_sms < 1) h->num_sms = 1;
  h->d = d;
  h->K = K;
  h->beta = beta;
  h->eta = eta;
  h->compressor = compressor;
  h->ratio = ratio;
  h->block = block;
  h->lambda = compressor == GMC_RBGS ? 0.5f : 0.f;

  auto fail = [&](cudaError_t err) {
    free_all(h);
    delete h;
    cudaGetLastError();
    return status_of(err);
  };
  cudaError_t err = configure_topk_kernels();
  if (err == cudaSuccess) err = configure_rbgs_kernels();
  if (err != cudaSuccess) return fail(err);

  const int64_t streams_wide = 2 * (int64_t)h->num_sms;
  if (compressor != GMC_RBGS) {
    // tiles of 4096 take the bulk-copy pass, for up to kBulkMaxK workers (its
    // shared memory grows with K); otherwise the load/store pass
    int U = K <= kBulkMaxK ? 4 : 2;
    if (d < 4096 * streams_wide) U = 2;
    if (d < 2048 * streams_wide) U = 1;
    h->tile = 1024 * U;
    h->n_tiles = (d + h->tile - 1) / h->tile;
    h->ld = h->n_tiles * h->tile;
    const int64_t ks = std::max<int64_t>(1, (int64_t)std::floor(ratio * (double)d));
    h->ksel = (uint32_t)ks;
    if (compressor == GMC_TOPK_APPROX) {
      // Sec. 5.1: |S| = about d/100 sampled components (runs of 8, one per
      // stratum of d / floor(d/800)), theta such that ratio*|S| of them reach
      // it; at most limit = min(d, 4 s + 4096) are sent
      h->sample_chunks = 0;
      h->n_sample = d < 8 ? (uint32_t)d : (uint32_t)(8 * std::max<int64_t>(1, d / 800));
      h->sample_rank = (uint32_t)std::max<int64_t>(1, (int64_t)std::floor(ratio * (double)h->n_sample));
      h->limit = (uint32_t)std::min<int64_t>(d, 4 * ks + 4096);
      // candidate parts: the expected count s with a 5-sigma margin of the
      // sample's spread (relative sd 1/sqrt(r)); the dense path rewrites up to limit
      const double r = (double)h->sample_rank;
      const double capd = std::ceil((double)ks * (1.0 + 5.0 / std::sqrt(r))) + 4096.0;
      h->cap = (uint32_t)std::min<double>((double)d, capd);
    } else if (d <= kSampleAll) {
      h->sample_chunks = 0;
      h->sample_rank = h->ksel;
      h->cap = (uint32_t)d;
    } else {
      h->sample_chunks = kSampleChunks;
      const double ns = (double)kSampleSlots;
      const double mean = ns * (double)ks / (double)d;
      const double r = std::min(ns, std::ceil(mean + 5.0 * std::sqrt(mean) + 8.0));
      h->sample_rank = (uint32_t)r;
      const double capd = std::ceil((double)d * (r + 8.0 * std::sqrt(r) + 16.0) / ns) + 4096.0;
      h->cap = (uint32_t)std::min<double>((double)d, capd);
    }
    h->grid_acc = (int)std::min<int64_t>(h->n_tiles, (int64_t)h->num_sms * accumulate_blocks_per_sm(h->tile));
    h->grid_agg = 0;  // set below from the candidate regions
    // candidate slots: the bulk pass gives every CTA its own region per worker,
    // one part per consumer warp (twice its share of the expected candidates,
    // plus slack, in whole 128-byte lines); otherwise one region
    const uint32_t cap0 = h->cap;
    if (h->tile == kBulkTile) {
      h->n_blk = (uint32_t)(h->n_tiles / h->grid_acc);
      h->blk_mul = golden_stride(h->n_blk);
      h->regions = h->grid_acc;
      const uint64_t share = (2ull * cap0 + h->regions * kChunksPerTile - 1) / (h->regions * kChunksPerTile);
      h->cap_part = (uint32_t)((share + 128 + 31) & ~31ull);
      h->cap_region = h->cap_part * kChunksPerTile;
    } else {
      h->regions = 1;
      h->cap_region = (cap0 + 3) & ~3u;
      h->cap_part = h->cap_region;
    }
    h->cap = (uint32_t)std::min<uint64_t>(
        std::max<uint64_t>((uint64_t)h->regions * h->cap_region, h->limit), 0xfffffff0ull);
    const int64_t per = (h->cap + 8191) / 8192;
    h->grid_agg = h->regions > 1 ? h->regions : (int)std::max<int64_t>(1, 4 * (int64_t)h->num_sms / K);
    // select: on the bulk path a warp walks the candidates of a run of at most
    // 32 parts as one list; the grid is one wave of as many blocks as fit on
    // an SM (each holds kBucketCap keys of shared memory: three on GB300), for
    // all the workers -- a second, partial wave cost about 10 us
    const int64_t nparts = (int64_t)h->regions * kChunksPerTile;
    const int64_t sel_wave = (int64_t)select_blocks_per_sm() * h->num_sms;
    h->sel_blocks = h->regions > 1 ? (int)std::min<int64_t>(
                                         h->regions, std::max<int64_t>((nparts + 32 * kWarps - 1) / (32 * kWarps),
                                                                       std::max<int64_t>(1, sel_wave / K)))
                                   : (int)std::max<int64_t>(1, std::min<int64_t>(per, std::max<int64_t>(1, streams_wide / K)));
    if (compressor == GMC_TOPK) h->n_sample = (uint32_t)(h->sample_chunks ? kSampleSlots : d);
    h->sample_stride = std::max<uint32_t>(kSampleSlots, (h->n_sample + 3) & ~3u);
    h->sample_blocks = (int)std::max<int64_t>(1, ((int64_t)h->n_sample + 2047) / 2048);
    h->theta_blocks = (int)std::max<int64_t>(1, std::min<int64_t>(2 * h->num_sms / K + 1,
                                                                  ((int64_t)h->n_sample + 8191) / 8192));
    // relative-histogram bin width 2^sel_shift keys: near the k-th key a key
    // step of 2^23 is an octave of |v|, and a Gaussian-like tail puts about
    // 11 ln2 * k * 2^s / 2^23 candidates in one bin; aim at 2048 (the bin is
    // ranked in shared memory when it holds at most kBucketCap)
    {
      const double w = 2048.0 * 8388608.0 / (11.0 * std::log(2.0) * (double)h->ksel);
      h->sel_shift = (int)std::min(20.0, std::max(0.0, std::floor(std::log2(w))));
    }
    const int64_t Kt = (int64_t)K * h->n_tiles;
    if ((err = dalloc(h, &h->e, (size_t)K * h->ld)) != cudaSuccess ||
        (err = dalloc(h, &h->w, (size_t)h->ld)) != cudaSuccess ||
        (err = dalloc(h, &h->dlt, (size_t)h->ld)) != cudaSuccess ||
        (err = dalloc(h, &h->sel, (size_t)K)) != cudaSuccess ||
        (err = dalloc(h, &h->ghist, (size_t)K * kHistBins)) != cudaSuccess ||
        (err = dalloc(h, &h->chist, (size_t)K * kRelBins)) != cudaSuccess ||
        (err = dalloc(h, &h->bucket, (size_t)K * 2 * kBucketCap)) != cudaSuccess ||
        (err = dalloc(h, &h->sample_keys, (size_t)K * h->sample_stride)) != cudaSuccess ||
        (err = dalloc(h, &h->big_tiles, (size_t)h->n_tiles + 1)) != cudaSuccess ||
        (err = dalloc(h, &h->rcount, (size_t)K * h->regions * kChunksPerTile)) != cudaSuccess ||
        (err = dalloc(h, &h->mask, (size_t)h->ld)) != cudaSuccess ||
        (err = dalloc(h, &h->sample_pend, (size_t)3 * h->sample_stride)) != cudaSuccess)
      return fail(err);
    if (h->n_blk >= 8 && ((err = dalloc(h, &h->blk_cost, (size_t)h->n_blk)) != cudaSuccess ||
                          (err = dalloc(h, &h->blk_order, (size_t)h->n_blk)) != cudaSuccess))
      return fail(err);
    if ((err = cudaStreamCreateWithFlags(&h->aux, cudaStreamNonBlocking)) != cudaSuccess ||
        (err = cudaEventCreateWithFlags(&h->ev_step, cudaEventDisableTiming)) != cudaSuccess ||
        (err = cudaEventCreateWithFlags(&h->ev_flush, cudaEventDisableTiming)) != cudaSuccess)
      return fail(err);
    for (int p = 0; p < 2; ++p) {
      if ((err = dalloc(h, &h->cand_idx[p], (size_t)K * h->cap)) != cudaSuccess ||
          (err = dalloc(h, &h->cand_val[p], (size_t)K * h->cap)) != cudaSuccess ||
          (err = dalloc(h, &h->chunk[p], (size_t)Kt * kChunksPerTile)) != cudaSuccess)
        return fail(err);
    }
  } else {
    h->tile = kRbgsTile;
    h->n_tiles = (d + h->tile - 1) / h->tile;
    h->ld = h->n_tiles * h->tile;
    h->nb = (d + block - 1) / block;
    h->m = std::max<int64_t>(1, (int64_t)std::floor(ratio * (double)h->nb));
    if (h->nb >= (int64_t(1) << 31)) return fail(cudaErrorInvalidValue);
    if ((block & (block - 1)) == 0) {
      uint32_t sh = 0;
      while ((int64_t(1) << sh) < block) ++sh;
      h->B_shift = sh;
    }
    // enough tiles for one per SM: the bulk-copy kernel (one persistent CTA per SM)
    h->rbgs_bulk = h->n_tiles >= h->num_sms;
    h->grid_rbgs = h->rbgs_bulk ? h->num_sms
                                : (int)std::min<int64_t>(h->n_tiles, (int64_t)h->num_sms * rbgs_blocks_per_sm());
    const int64_t nbw = (h->nb + 31) / 32;
    if ((err = dalloc(h, &h->e, (size_t)K * h->ld)) != cudaSuccess ||
        (err = dalloc(h, &h->w, (size_t)h->ld)) != cudaSuccess ||
        (err = dalloc(h, &h->dlt, (size_t)h->ld)) != cudaSuccess ||
        (err = dalloc(h, &h->bitmap, (size_t)K * nbw)) != cudaSuccess ||
        (err = dalloc(h, &h->rank, (size_t)K * h->nb)) != cudaSuccess ||
        (err = dalloc(h, &h->blocks, (size_t)K * h->m)) != cudaSuccess ||
        (err = dalloc(h, &h->uflag[0], (size_t)h->nb)) != cudaSuccess ||
        (err = dalloc(h, &h->uflag[1], (size_t)h->nb)) != cudaSuccess ||
        (err = dalloc(h, &h->slab, (size_t)K * h->m * block)) != cudaSuccess)
      return fail(err);
  }
  if ((err = dalloc(h, &h->step_ctr, 1)) != cudaSuccess ||
      (err = dalloc(h, &h->tile_ctr, 1)) != cudaSuccess ||
      (err = dalloc(h, &h->total_ctr, 1)) != cudaSuccess ||
      (err = dalloc(h, &h->status, 1)) != cudaSuccess)
    return fail(err);
  if ((err = cudaDeviceSynchronize()) != cudaSuccess) return fail(err);
  *out = h;
  return GMC_OK;
}

void gmc_destroy(gmc_t h) {
  if (!h) return;
  DeviceGuard g(h->device);
  cudaDeviceSynchronize();
  free_all(h);
  delete h;
}

int gmc_set_lambda(gmc_t h, float lambda) {
  if (!h || !finite_f(lambda) || lambda < 0.f || lambda > 1.f) return GMC_EINVAL;
  // GMC+ detaches Alg. 1; the local-momentum baseline detaches as DEF-A does
  if (lambda != 0.f && (h->variant == GMC_VARIANT_SERVER_MOMENTUM || h->variant == GMC_VARIANT_LR_IN_RESIDUAL))
    return GMC_EINVAL;
  h->lambda = lambda;
  return GMC_OK;
}

int gmc_set_rbgs_mode(gmc_t h, int32_t per_worker) {
  if (!h || (per_worker != 0 && per_worker != 1)) return GMC_EINVAL;
  h->per_worker = per_worker;
  return GMC_OK;
}

int gmc_set_seed(gmc_t h, uint64_t seed) {
  if (!h) return GMC_EINVAL;
  h->seed = seed;
  return GMC_OK;
}

int gmc_set_eta(gmc_t h, float eta) {
  if (!h || !finite_f(eta) || !(eta > 0.f)) return GMC_EINVAL;
  h->eta = eta;
  return GMC_OK;
}

int gmc_set_variant(gmc_t h, int32_t variant) {
  if (!h) return GMC_EINVAL;
  if (variant < GMC_VARIANT_GMC || variant > GMC_VARIANT_LOCAL_MOMENTUM_MFM) return GMC_EINVAL;
  if (variant != GMC_VARIANT_GMC && h->compressor == GMC_RBGS) return GMC_EINVAL;
  if ((variant == GMC_VARIANT_SERVER_MOMENTUM || variant == GMC_VARIANT_LR_IN_RESIDUAL) && h->lambda != 0.f)
    return GMC_EINVAL;
  if (h->initialized && h->t > 0) return GMC_ESTATE;  // the residuals mean another thing
  if (variant == GMC_VARIANT_SERVER_MOMENTUM && !h->mom) {
    DeviceGuard g(h->device);
    cudaError_t err = dalloc(h, &h->mom, (size_t)h->ld);
    if (err == cudaSuccess) err = cudaMemset(h->mom, 0, (size_t)h->ld * sizeof(float));
    if (err != cudaSuccess) return status_of(err);
  }
  if ((variant == GMC_VARIANT_LOCAL_MOMENTUM || variant == GMC_VARIANT_LOCAL_MOMENTUM_MFM) && !h->lm) {
    DeviceGuard g(h->device);
    cudaError_t err = dalloc(h, &h->lm, (size_t)h->K * h->ld);
    if (err != cudaSuccess) return status_of(err);
  }
  h->variant = variant;
  return GMC_OK;
}

int gmc_set_select_mode(gmc_t h, int32_t mode) {
  if (!h || (mode != GMC_SELECT_SAMPLED && mode != GMC_SELECT_DENSE)) return GMC_EINVAL;
  // the approximate top-s is defined by its sample: it has no dense engine
  if (h->compressor == GMC_TOPK_APPROX && mode != GMC_SELECT_SAMPLED) return GMC_EINVAL;
  h->select_mode = mode;
  return GMC_OK;
}

int gmc_set_detach_output(gmc_t h, float* out_dev, int64_t ld) {
  if (!h) return GMC_EINVAL;
  if (out_dev && ld < h->d) return GMC_EINVAL;
  h->detach_out = out_dev;
  h->detach_ld = out_dev ? ld : 0;
  return GMC_OK;
}

}  // extern "C"

namespace {
// Everything but w back to the start of Alg. 1 (e = 0, w_{-1} = w_0, t = 0,
// counters cleared), on stream s.
int reset_state(gmc_ctx* h, cudaStream_t s) {
  GMC_TRY(order_after_flush(h, s, true));
  h->agg_pending = false;  // a pending aggregation of the old state is dropped
  GMC_TRY(cudaMemsetAsync(h->e, 0, (size_t)h->K * h->ld * sizeof(float), s));
  GMC_TRY(cudaMemsetAsync(h->dlt, 0, (size_t)h->ld * sizeof(float), s));
  if (h->mom) GMC_TRY(cudaMemsetAsync(h->mom, 0, (size_t)h->ld * sizeof(float), s));
  if (h->lm) GMC_TRY(cudaMemsetAsync(h->lm, 0, (size_t)h->K * h->ld * sizeof(float), s));
  if (h->compressor != GMC_RBGS) {
    for (int p = 0; p < 2; ++p)
      GMC_TRY(cudaMemsetAsync(h->chunk[p], 0, (size_t)h->K * h->n_tiles * kChunksPerTile * sizeof(uint2), s));
    GMC_TRY(cudaMemsetAsync(h->sel, 0, (size_t)h->K * sizeof(WorkerSel), s));
    GMC_TRY(cudaMemsetAsync(h->mask, 0, (size_t)h->ld * sizeof(uint32_t), s));
    if (h->blk_cost) GMC_TRY(cudaMemsetAsync(h->blk_cost, 0, (size_t)h->n_blk * sizeof(uint32_t), s));
  } else {
    for (int p = 0; p < 2; ++p) GMC_TRY(cudaMemsetAsync(h->uflag[p], 0, (size_t)h->nb, s));
  }
  GMC_TRY(cudaMemsetAsync(h->step_ctr, 0, sizeof(Counters), s));
  GMC_TRY(cudaMemsetAsync(h->total_ctr, 0, sizeof(Counters), s));
  GMC_TRY(cudaMemsetAsync(h->status, 0, sizeof(unsigned), s));
  h->t = 0;
  h->restored = false;
  h->initialized = true;
  return GMC_OK;
}

// gmc_step_host for fp32 or bf16 gradient rows.
int step_host(gmc_ctx* h, const void* grads_host, uint64_t* step_stats_host, cudaStream_t s, bool bf16) {
  // page-locked host memory is mapped into the device's address space: the
  // kernels read the gradients in place, each crossing the host link once
  // while the pass runs; other host memory is copied to a staging buffer first
  const void* mapped = nullptr;
  int st;
  if (cudaHostGetDevicePointer(const_cast<void**>(&mapped), const_cast<void*>(grads_host), 0) == cudaSuccess) {
    st = enqueue_step(h, mapped, s, true, true, bf16);
  } else {
    cudaGetLastError();
    const size_t n = (size_t)h->K * (size_t)h->d;
    if (!h->gstage) {
      cudaError_t err = dalloc(h, &h->gstage, n);
      if (err != cudaSuccess) return status_of(err);
    }
    GMC_TRY(cudaMemcpyAsync(h->gstage, grads_host, n * (bf16 ? 2 : 4), cudaMemcpyHostToDevice, s));
    st = enqueue_step(h, h->gstage, s, true, false, bf16);
  }
  if (st != GMC_OK) return st;
  if (step_stats_host)
    GMC_TRY(cudaMemcpyAsync(step_stats_host, h->step_ctr, sizeof(Counters), cudaMemcpyDeviceToHost, s));
  return GMC_OK;
}
}  // namespace

extern "C" {

int gmc_set_params(gmc_t h, const float* w0_dev, void* stream) {
  if (!h || !w0_dev) return GMC_EINVAL;
  DeviceGuard g(h->device);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  GMC_TRY_ST(reset_state(h, s));
  GMC_TRY(cudaMemcpyAsync(h->w, w0_dev, (size_t)h->d * sizeof(float), cudaMemcpyDeviceToDevice, s));
  return GMC_OK;
}

int gmc_step(gmc_t h, const float* grads_dev, void* stream) {
  if (!h || !grads_dev) return GMC_EINVAL;
  if (!h->initialized) return GMC_ESTATE;
  DeviceGuard g(h->device);
  return enqueue_step(h, grads_dev, static_cast<cudaStream_t>(stream), false);
}


int gmc_step_host(gmc_t h, const float* grads_host, uint64_t* step_stats_host, void* stream) {
  if (!h || !grads_host) return GMC_EINVAL;
  if (!h->initialized) return GMC_ESTATE;
  DeviceGuard g(h->device);
  return step_host(h, grads_host, step_stats_host, static_cast<cudaStream_t>(stream), false);
}

int gmc_step_bf16(gmc_t h, const uint16_t* grads_bf16_dev, void* stream) {
  if (!h || !grads_bf16_dev || (reinterpret_cast<uintptr_t>(grads_bf16_dev) & 1)) return GMC_EINVAL;
  if (!h->initialized) return GMC_ESTATE;
  DeviceGuard g(h->device);
  return enqueue_step(h, grads_bf16_dev, static_cast<cudaStream_t>(stream), false, false, true);
}

int gmc_step_host_bf16(gmc_t h, const uint16_t* grads_bf16_host, uint64_t* step_stats_host, void* stream) {
  if (!h || !grads_bf16_host || (reinterpret_cast<uintptr_t>(grads_bf16_host) & 1)) return GMC_EINVAL;
  if (!h->initialized) return GMC_ESTATE;
  DeviceGuard g(h->device);
  return step_host(h, grads_bf16_host, step_stats_host, static_cast<cudaStream_t>(stream), true);
}

int gmc_get_params(gmc_t h, float* w_dev_out, void* stream) {
  if (!h || !w_dev_out) return GMC_EINVAL;
  if (!h->initialized) return GMC_ESTATE;
  DeviceGuard g(h->device);
  GMC_TRY_ST(flush(h, static_cast<cudaStream_t>(stream)));
  GMC_TRY(order_after_flush(h, static_cast<cudaStream_t>(stream), false));
  GMC_TRY(cudaMemcpyAsync(w_dev_out, h->w, (size_t)h->d * sizeof(float), cudaMemcpyDeviceToDevice,
                          static_cast<cudaStream_t>(stream)));
  return GMC_OK;
}

int gmc_get_residual(gmc_t h, int32_t k, float* e_dev_out, void* stream) {
  if (!h || !e_dev_out || k < 0 || k >= h->K) return GMC_EINVAL;
  if (!h->initialized) return GMC_ESTATE;
  DeviceGuard g(h->device);
  GMC_TRY_ST(flush(h, static_cast<cudaStream_t>(stream)));
  GMC_TRY(order_after_flush(h, static_cast<cudaStream_t>(stream), false));
  GMC_TRY(cudaMemcpyAsync(e_dev_out, h->e + (int64_t)k * h->ld, (size_t)h->d * sizeof(float),
                          cudaMemcpyDeviceToDevice, static_cast<cudaStream_t>(stream)));
  return GMC_OK;
}

int64_t gmc_selected_capacity(gmc_t h) {
  if (!h) return -1;
  if (h->compressor == GMC_TOPK_APPROX) return (int64_t)h->limit;
  return h->compressor == GMC_TOPK ? (int64_t)h->ksel : h->m * h->block;
}

int gmc_get_selected(gmc_t h, int32_t k, uint32_t* idx_dev, float* val_dev, int64_t capacity,
                     int64_t* count_host, void* stream) {
  if (!h || !idx_dev || !val_dev || !count_host || k < 0 || k >= h->K) return GMC_EINVAL;
  if (!h->initialized || h->t == 0 || h->restored) return GMC_ESTATE;
  DeviceGuard g(h->device);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (h->compressor != GMC_RBGS) {
    int64_t count = h->ksel;
    if (h->compressor == GMC_TOPK_APPROX) {  // the count varies by step: read it
      uint32_t nsel = 0;
      GMC_TRY(cudaMemcpyAsync(&nsel, &h->sel[k].nsel, sizeof(uint32_t), cudaMemcpyDeviceToHost, s));
      GMC_TRY(cudaStreamSynchronize(s));
      count = nsel;
    }
    *count_host = count;
    if (capacity < count) return GMC_EINVAL;
    const TopkArgs A = topk_args_at(h, nullptr, h->t - 1);
    GMC_TRY(launch_gather_selected(A, k, idx_dev, val_dev, s));
  } else {
    int32_t last_block = 0;
    const int32_t* blk = h->blocks + (h->per_worker ? (int64_t)k * h->m : 0) + (h->m - 1);
    GMC_TRY(cudaMemcpyAsync(&last_block, blk, sizeof(int32_t), cudaMemcpyDeviceToHost, s));
    GMC_TRY(cudaStreamSynchronize(s));
    int64_t count = h->m * h->block;
    if (last_block == h->nb - 1) count -= h->nb * h->block - h->d;
    *count_host = count;
    if (capacity < count) return GMC_EINVAL;
    RbgsArgs A = rbgs_args(h, nullptr);
    GMC_TRY(launch_rbgs_expand(A, k, idx_dev, val_dev, s));
  }
  GMC_TRY(cudaStreamSynchronize(s));
  return GMC_OK;
}

int gmc_get_worker_params(gmc_t h, int32_t k, float* out_dev, void* stream) {
  if (!h || !out_dev || k < 0 || k >= h->K) return GMC_EINVAL;
  if (!h->initialized) return GMC_ESTATE;
  DeviceGuard g(h->device);
  GMC_TRY_ST(flush(h, static_cast<cudaStream_t>(stream)));
  GMC_TRY(order_after_flush(h, static_cast<cudaStream_t>(stream), false));
  DetachArgs D{h->w, h->e, h->ld, h->d, detach_b(h), out_dev, h->d, k, k + 1};
  GMC_TRY(launch_detach(D, static_cast<cudaStream_t>(stream)));
  return GMC_OK;
}

int gmc_get_stats(gmc_t h, uint64_t* counters_host, int32_t n, double* rcc_host) {
  if (!h || n < 0 || n > GMC_STAT_COUNT || (n > 0 && !counters_host)) return GMC_EINVAL;
  if (!h->initialized) return GMC_ESTATE;
  DeviceGuard g(h->device);
  GMC_TRY_ST(flush(h, h->aux));
  GMC_TRY(cudaDeviceSynchronize());
  Counters c;
  GMC_TRY(cudaMemcpy(&c, h->total_ctr, sizeof(Counters), cudaMemcpyDeviceToHost));
  for (int i = 0; i < n; ++i) counters_host[i] = c.v[i];
  if (rcc_host) {
    const double T = (double)c.v[kSteps];
    double r = 0.0;
    if (T > 0) {
      r = ((double)h->K * (double)c.v[kChanged] + (double)c.v[kNnz]) /
          ((double)h->d * (double)h->K * T);
      if (h->compressor == GMC_RBGS) r *= 0.5;
    }
    *rcc_host = r;
  }
  return GMC_OK;
}

// ---------------------------------------------------------------------------
// checkpoint / resume
// ---------------------------------------------------------------------------
namespace {
// Fixed-layout header of a saved state, followed by w (d floats), w_t - w_{t-1}
// (d floats), the K residual rows (d floats each) and, for Alg. 3, the server's
// w_t - w_{t-1} (d floats); all little-endian fp32 as the GPU holds them.
struct StateHeader {
  char magic[8];
  uint32_t version, header_bytes;
  int64_t d;
  int32_t K, compressor;
  double ratio;
  int64_t block;
  int32_t variant, per_worker;
  uint64_t seed;
  int64_t t;
  float beta, eta, lambda;
  int32_t select_mode;
  uint64_t totals[8];
  uint32_t status, has_mom, lm_rows, pad;
};
constexpr char kMagic[8] = {'G', 'M', 'C', 'S', 'T', 'A', 'T', 'E'};
constexpr uint32_t kStateVersion = 1;

int64_t state_bytes(const gmc_ctx* h) {
  const int64_t rows = (int64_t)(2 + h->K) + (h->variant == GMC_VARIANT_SERVER_MOMENTUM ? 1 : 0) +
                       (local_variant(h) ? h->K : 0);
  return (int64_t)sizeof(StateHeader) + rows * h->d * (int64_t)sizeof(float);
}
}  // namespace

int64_t gmc_state_bytes(gmc_t h) {
  if (!h) return -1;
  return state_bytes(h);
}

int gmc_save_state(gmc_t h, void* host_out, int64_t capacity) {
  if (!h || !host_out) return GMC_EINVAL;
  if (!h->initialized) return GMC_ESTATE;
  if (capacity < state_bytes(h)) return GMC_EINVAL;
  DeviceGuard g(h->device);
  GMC_TRY_ST(flush(h, h->aux));  // the state Alg. 1 defines: no aggregation left pending
  GMC_TRY(cudaDeviceSynchronize());
  StateHeader H;
  std::memset(&H, 0, sizeof(H));
  std::memcpy(H.magic, kMagic, sizeof(kMagic));
  H.version = kStateVersion;
  H.header_bytes = (uint32_t)sizeof(StateHeader);
  H.d = h->d;
  H.K = h->K;
  H.compressor = h->compressor;
  H.ratio = h->ratio;
  H.block = h->block;
  H.variant = h->variant;
  H.per_worker = h->per_worker;
  H.seed = h->seed;
  H.t = h->t;
  H.beta = h->beta;
  H.eta = h->eta;
  H.lambda = h->lambda;
  H.select_mode = h->select_mode;
  Counters c;
  GMC_TRY(cudaMemcpy(&c, h->total_ctr, sizeof(Counters), cudaMemcpyDeviceToHost));
  for (int i = 0; i < 8; ++i) H.totals[i] = c.v[i];
  GMC_TRY(cudaMemcpy(&H.status, h->status, sizeof(unsigned), cudaMemcpyDeviceToHost));
  H.has_mom = h->variant == GMC_VARIANT_SERVER_MOMENTUM ? 1u : 0u;
  H.lm_rows = local_variant(h) ? (uint32_t)h->K : 0u;
  char* out = static_cast<char*>(host_out);
  std::memcpy(out, &H, sizeof(H));
  const size_t row = (size_t)h->d * sizeof(float);
  char* p = out + sizeof(H);
  GMC_TRY(cudaMemcpy(p, h->w, row, cudaMemcpyDeviceToHost));
  p += row;
  // w_t - w_{t-1}: where the step left it (dlt, zero outside the last union),
  // or, for Alg. 3, the server's dense copy (dlt is zero between its steps)
  GMC_TRY(cudaMemcpy(p, h->dlt, row, cudaMemcpyDeviceToHost));
  p += row;
  GMC_TRY(cudaMemcpy2D(p, row, h->e, (size_t)h->ld * sizeof(float), row, (size_t)h->K,
                       cudaMemcpyDeviceToHost));
  p += row * h->K;
  if (H.has_mom) {
    GMC_TRY(cudaMemcpy(p, h->mom, row, cudaMemcpyDeviceToHost));
    p += row;
  }
  if (H.lm_rows)
    GMC_TRY(cudaMemcpy2D(p, row, h->lm, (size_t)h->ld * sizeof(float), row, (size_t)h->K,
                         cudaMemcpyDeviceToHost));
  return GMC_OK;
}

int gmc_load_state(gmc_t h, const void* host_in, int64_t bytes) {
  if (!h || !host_in || bytes < (int64_t)sizeof(StateHeader)) return GMC_EINVAL;
  StateHeader H;
  std::memcpy(&H, host_in, sizeof(H));
  if (std::memcmp(H.magic, kMagic, sizeof(kMagic)) != 0 || H.version != kStateVersion ||
      H.header_bytes != sizeof(StateHeader))
    return GMC_EINVAL;
  // the handle must have been created for the same problem and form
  if (H.d != h->d || H.K != h->K || H.compressor != h->compressor || H.ratio != h->ratio ||
      (h->compressor == GMC_RBGS && H.block != h->block) || H.variant != h->variant ||
      H.t < 0 || H.has_mom != (h->variant == GMC_VARIANT_SERVER_MOMENTUM ? 1u : 0u) ||
      H.lm_rows != (local_variant(h) ? (uint32_t)h->K : 0u))
    return GMC_EINVAL;
  if (bytes < state_bytes(h)) return GMC_EINVAL;
  if (!finite_f(H.eta) || !(H.eta > 0.f) || !finite_f(H.lambda) || H.lambda < 0.f || H.lambda > 1.f ||
      (H.per_worker != 0 && H.per_worker != 1) ||
      (H.select_mode != GMC_SELECT_SAMPLED && H.select_mode != GMC_SELECT_DENSE))
    return GMC_EINVAL;
  DeviceGuard g(h->device);
  GMC_TRY(cudaDeviceSynchronize());
  const char* p = static_cast<const char*>(host_in) + sizeof(H);
  GMC_TRY_ST(reset_state(h, h->aux));  // as gmc_set_params: e, dlt, mom, tables, counters cleared
  GMC_TRY(cudaStreamSynchronize(h->aux));
  const size_t row = (size_t)h->d * sizeof(float);
  GMC_TRY(cudaMemcpy(h->w, p, row, cudaMemcpyHostToDevice));
  p += row;
  GMC_TRY(cudaMemcpy(h->dlt, p, row, cudaMemcpyHostToDevice));
  p += row;
  GMC_TRY(cudaMemcpy2D(h->e, (size_t)h->ld * sizeof(float), p, row, row, (size_t)h->K,
                       cudaMemcpyHostToDevice));
  p += row * h->K;
  if (H.has_mom) {
    GMC_TRY(cudaMemcpy(h->mom, p, row, cudaMemcpyHostToDevice));
    p += row;
  }
  if (H.lm_rows)
    GMC_TRY(cudaMemcpy2D(h->lm, (size_t)h->ld * sizeof(float), p, row, row, (size_t)h->K,
                         cudaMemcpyHostToDevice));
  Counters c;
  for (int i = 0; i < 8; ++i) c.v[i] = H.totals[i];
  GMC_TRY(cudaMemcpy(h->total_ctr, &c, sizeof(Counters), cudaMemcpyHostToDevice));
  unsigned st = H.status;
  GMC_TRY(cudaMemcpy(h->status, &st, sizeof(unsigned), cudaMemcpyHostToDevice));
  h->seed = H.seed;
  h->per_worker = H.per_worker;
  h->eta = H.eta;
  h->lambda = H.lambda;
  h->select_mode = H.select_mode;
  h->t = H.t;
  h->restored = H.t > 0;
  GMC_TRY(cudaDeviceSynchronize());
  return GMC_OK;
}

int gmc_check(gmc_t h) {
  if (!h) return GMC_EINVAL;
  if (!h->initialized) return GMC_OK;
  DeviceGuard g(h->device);
  cudaError_t err = cudaDeviceSynchronize();
  if (err != cudaSuccess) return GMC_ECUDA;
  unsigned st = 0;
  err = cudaMemcpy(&st, h->status, sizeof(unsigned), cudaMemcpyDeviceToHost);
  if (err != cudaSuccess) return GMC_ECUDA;
  if (st & kStatusInternal) return GMC_EINTERNAL;
  if (st & kStatusTimeout) return GMC_ETIMEOUT;
  if (st & kStatusNonfinite) return GMC_ENONFINITE;
  return GMC_OK;
}

int gmc_test_withhold_copy(gmc_t h, int64_t tile, int32_t k, uint64_t wait_limit_ns) {
  if (!h || k < 0 || k >= h->K || wait_limit_ns == 0 || wait_limit_ns > kWaitLimitNs) return GMC_EINVAL;
  const bool bulk = h->compressor == GMC_RBGS ? h->rbgs_bulk : h->tile == kBulkTile;
  if (!bulk || tile < 0 || tile >= h->n_tiles) return GMC_EINVAL;
  h->hold_tile = tile;
  h->hold_k = k;
  h->hold_wait_ns = wait_limit_ns;
  return GMC_OK;
}

int64_t gmc_test_fail_alloc(int64_t fail_at) {
  g_fail_countdown.store(fail_at < 0 ? -1 : fail_at);
  return g_live_allocations.load();
}

int gmc_profile_enable(gmc_t h, int32_t on) {
  if (!h) return GMC_EINVAL;
  DeviceGuard g(h->device);
  if (on && !h->prof) {
    drain_profile(h);
    for (int i = 0; i < GMC_KERNEL_COUNT; ++i) {
      h->prof_ms[i] = 0.0;
      h->prof_launches[i] = 0;
      h->prof_bytes[i] = 0.0;
    }
  }
  h->prof = on != 0;
  return GMC_OK;
}

int gmc_profile_kernels(gmc_t h, uint32_t kernel_mask) {
  if (!h) return GMC_EINVAL;
  h->prof_mask = kernel_mask;
  return GMC_OK;
}

int gmc_profile_read(gmc_t h, int32_t kernel, double* total_ms, int64_t* launches,
                     double* algorithmic_bytes) {
  if (!h || kernel < 0 || kernel >= GMC_KERNEL_COUNT) return GMC_EINVAL;
  DeviceGuard g(h->device);
  drain_profile(h);
  if (total_ms) *total_ms = h->prof_ms[kernel];
  if (launches) *launches = h->prof_launches[kernel];
  if (algorithmic_bytes) *algorithmic_bytes = h->prof_bytes[kernel];
  return GMC_OK;
}

}  // extern "C"
