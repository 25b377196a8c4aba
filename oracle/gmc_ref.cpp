// GMC / GMC+ oracle in plain C++: the paper's update rules written out with
// dense arrays, one worker per thread.
//
// TEST INFRASTRUCTURE. Only the tests, __graft_entry__.smoke() and the CPU
// baseline / reference arm of bench.py may load this library. The product path
// (the CUDA library and its Python binding) never loads it and shares no code
// with it: nothing here includes a header of the CUDA library.
//
// What it follows (Shi et al., "Global Momentum Compression for Sparse
// Communication in Distributed Learning", arXiv 1905.12948):
//   Algorithm 1 (GMC, Sec. 3.1), for every worker k at step t:
//     e_{t+1/2,k} = e_{t,k} + g_{t,k} - (beta/eta) (w_t - w_{t-1})
//     e_{t+1,k}   = e_{t+1/2,k} - C(e_{t+1/2,k})
//     w_{t+1}     = w_t - (eta/K) sum_k C(e_{t+1/2,k})
//   with w_{-1} = w_0 and e_{0,k} = 0; Algorithm 2 (GMC+, Sec. 4) adds the
//   detached point w_{t,k} = w_t - lambda*eta*e_{t,k}, an output here.
//   Compressors (Sec. 4): top-s, the s components of largest magnitude; RBGS,
//   random blocks with one seed shared by all workers (Sec. 5.2), or one per
//   worker.
//   Relative communication cost (Sec. 5), halved for RBGS (Sec. 5.2).
//
// Precision: fp32 state, each operation one IEEE round-to-nearest-even fp32
// operation in the order the algorithm writes it (compiled without FMA
// contraction or fast-math): v = (e + g) - (c * (w - w_prev)), c = fl(beta/eta);
// the aggregate adds the workers' values in ascending worker order from +0;
// w_next = w - (a * sum), a = fl(eta/K); detach w - (b * e), b = fl(lambda*eta).
//
// Readings where the paper is silent (the same as the numpy oracle's):
//   * top-s: magnitudes compare through the fp32 bit pattern with the sign
//     cleared (+0 and -0 tie); ties go to the lower index;
//     s = max(1, floor(ratio * d));
//   * RBGS: aligned blocks of B (the last may be short), m = max(1,
//     floor(ratio * nb)) distinct blocks drawn by Floyd's sampling (Bentley &
//     Floyd, CACM 1987) from a SplitMix64 counter stream (Steele, Lea & Flood,
//     OOPSLA 2014) keyed by (seed, t) -- or (seed, t, k) per worker -- with
//     multiply-shift range reduction;
//   * the residual at a sent coordinate is +0 exactly.
//
// Threads: the accumulator, the compressor and the residual of each worker
// depend on that worker's rows alone (Alg. 1's worker part), so workers run
// on separate threads; the server part (aggregate and update) runs on one
// thread in ascending worker order.
#include <algorithm>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <new>
#include <thread>
#include <vector>

namespace {

constexpr uint64_t kGolden = 0x9E3779B97F4A7C15ull;

// SplitMix64 output function (Steele, Lea & Flood 2014).
uint64_t splitmix64_mix(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

// Key of the block-choice stream of step t (stream 0: shared by all workers;
// k + 1: worker k), and the stream's i-th draw.
uint64_t stream_key(uint64_t seed, int64_t t, uint64_t stream) {
  const uint64_t k1 = splitmix64_mix(seed + kGolden * (uint64_t)(t + 1));
  return splitmix64_mix(k1 + kGolden * (stream + 1));
}
uint64_t stream_draw(uint64_t key, uint64_t i) { return splitmix64_mix(key + kGolden * (i + 1)); }

// [0, n) from a draw's top 32 bits, by multiply-shift.
uint64_t below(uint64_t x, uint64_t n) { return ((x >> 32) * n) >> 32; }

// m distinct blocks of [0, nb) by Floyd's sampling, ascending.
std::vector<int64_t> floyd_blocks(uint64_t key, int64_t nb, int64_t m) {
  std::vector<char> chosen((size_t)nb, 0);
  int64_t i = 0;
  for (int64_t j = nb - m; j < nb; ++j, ++i) {
    const int64_t r = (int64_t)below(stream_draw(key, (uint64_t)i), (uint64_t)(j + 1));
    chosen[(size_t)(chosen[(size_t)r] ? j : r)] = 1;
  }
  std::vector<int64_t> out;
  out.reserve((size_t)m);
  for (int64_t b = 0; b < nb; ++b)
    if (chosen[(size_t)b]) out.push_back(b);
  return out;
}

uint32_t magnitude_key(float x) {
  uint32_t u;
  std::memcpy(&u, &x, 4);
  return u & 0x7fffffffu;
}

// Support of top-s (Sec. 4): the s components of largest magnitude key, ties
// to the lower index, ascending. From the definition: kth = the s-th largest
// key (a selection, std::nth_element); every component above kth, then the
// lowest-index components equal to kth until s are taken.
std::vector<int64_t> top_s_support(const float* x, int64_t n, int64_t s) {
  std::vector<uint32_t> keys((size_t)n);
  for (int64_t j = 0; j < n; ++j) keys[(size_t)j] = magnitude_key(x[j]);
  std::nth_element(keys.begin(), keys.begin() + (n - s), keys.end());
  const uint32_t kth = keys[(size_t)(n - s)];
  keys.clear();
  keys.shrink_to_fit();
  int64_t above = 0;
  for (int64_t j = 0; j < n; ++j) above += magnitude_key(x[j]) > kth;
  int64_t ties_left = s - above;
  std::vector<int64_t> out;
  out.reserve((size_t)s);
  for (int64_t j = 0; j < n; ++j) {
    const uint32_t kj = magnitude_key(x[j]);
    if (kj > kth) {
      out.push_back(j);
    } else if (kj == kth && ties_left > 0) {
      out.push_back(j);
      --ties_left;
    }
  }
  return out;
}

struct Ref {
  int64_t d = 0;
  int K = 0;
  float beta = 0.f, eta = 0.f, lambda = 0.f;
  float c = 0.f, a = 0.f, b = 0.f;  // fl(beta/eta), fl(eta/K), fl(lambda*eta)
  int compressor = 0;                // 0 top-s, 1 RBGS
  double ratio = 0.0;
  int64_t s = 0;                     // top-s count
  int64_t B = 0, nb = 0, m = 0;      // RBGS geometry
  uint64_t seed = 0;
  int per_worker = 0;
  int threads = 1;
  int64_t t = 0;
  bool ready = false;
  std::vector<float> w, w_prev, e;   // e: K rows of d
  std::vector<std::vector<int64_t>> support;  // last step's supports
  std::vector<std::vector<float>> values;     // and values
  uint64_t totals[5] = {0, 0, 0, 0, 0};       // steps, pairs, nnz, union, changed

  void set_eta(float eta_) {
    eta = eta_;
    c = beta / eta;
    a = eta / (float)K;
    b = lambda * eta;
  }

  // Alg. 1's worker part for worker k: accumulator, compressor, residual.
  void worker(int k, const float* g, const std::vector<std::vector<int64_t>>& blocks) {
    float* ek = e.data() + (size_t)k * d;
    const float* gk = g + (size_t)k * d;
    for (int64_t j = 0; j < d; ++j) {
      const float dw = w[(size_t)j] - w_prev[(size_t)j];
      const float eg = ek[j] + gk[j];
      const float cd = c * dw;
      ek[j] = eg - cd;  // e_{t+1/2,k}, held in place
    }
    std::vector<int64_t> sup;
    if (compressor == 0) {
      sup = top_s_support(ek, d, s);
    } else {
      for (int64_t blk : blocks[per_worker ? (size_t)k : 0])
        for (int64_t j = blk * B; j < std::min((blk + 1) * B, d); ++j) sup.push_back(j);
    }
    std::vector<float> val(sup.size());
    for (size_t i = 0; i < sup.size(); ++i) {
      val[i] = ek[sup[i]];
      ek[sup[i]] = 0.0f;  // e_{t+1,k} = e_{t+1/2,k} - C(e_{t+1/2,k}): +0 where sent
    }
    support[(size_t)k] = std::move(sup);
    values[(size_t)k] = std::move(val);
  }

  void step(const float* g) {
    std::vector<std::vector<int64_t>> blocks;
    if (compressor == 1) {
      const int streams = per_worker ? K : 1;
      for (int st = 0; st < streams; ++st)
        blocks.push_back(floyd_blocks(stream_key(seed, t, per_worker ? (uint64_t)(st + 1) : 0u), nb, m));
    }
    // the workers, `threads` at a time
    std::vector<std::thread> pool;
    for (int k0 = 0; k0 < K; k0 += threads) {
      const int k1 = std::min(K, k0 + threads);
      for (int k = k0 + 1; k < k1; ++k) pool.emplace_back([this, k, g, &blocks] { worker(k, g, blocks); });
      worker(k0, g, blocks);
      for (auto& th : pool) th.join();
      pool.clear();
    }
    // the server: sum of the workers' C in ascending worker order from +0, then
    // w_{t+1} = w_t - (eta/K) * sum over every coordinate
    std::vector<float> total((size_t)d, 0.0f);
    std::vector<char> in_union((size_t)d, 0);
    uint64_t pairs = 0, nnz = 0;
    for (int k = 0; k < K; ++k) {
      const auto& sup = support[(size_t)k];
      const auto& val = values[(size_t)k];
      for (size_t i = 0; i < sup.size(); ++i) {
        total[(size_t)sup[i]] = total[(size_t)sup[i]] + val[i];
        in_union[(size_t)sup[i]] = 1;
        nnz += val[i] != 0.0f;
      }
      pairs += sup.size();
    }
    uint64_t uni = 0, changed = 0;
    for (int64_t j = 0; j < d; ++j) {
      const float wn = w[(size_t)j] - a * total[(size_t)j];
      changed += (wn - w[(size_t)j]) != 0.0f;
      uni += in_union[(size_t)j];
      w_prev[(size_t)j] = w[(size_t)j];
      w[(size_t)j] = wn;
    }
    totals[0] += 1;
    totals[1] += pairs;
    totals[2] += nnz;
    totals[3] += uni;
    totals[4] += changed;
    t += 1;
  }
};

}  // namespace

extern "C" {

// A new oracle instance (compressor 0: top-s, 1: RBGS), or NULL for invalid
// arguments. threads <= 0: one per worker, at most the host's hardware threads.
void* gmcref_create(int64_t d, int32_t K, float beta, float eta, int32_t compressor, double ratio,
                    int64_t block, float lambda, uint64_t seed, int32_t per_worker, int32_t threads) {
  if (d < 1 || K < 1 || !(beta >= 0.f && beta < 1.f) || !(eta > 0.f) || !(ratio > 0.0 && ratio <= 1.0))
    return nullptr;
  if (compressor != 0 && compressor != 1) return nullptr;
  if (compressor == 1 && block < 1) return nullptr;
  Ref* r = new (std::nothrow) Ref();
  if (!r) return nullptr;
  r->d = d;
  r->K = K;
  r->beta = beta;
  r->lambda = lambda;
  r->compressor = compressor;
  r->ratio = ratio;
  r->seed = seed;
  r->per_worker = per_worker ? 1 : 0;
  r->s = std::max<int64_t>(1, (int64_t)std::floor(ratio * (double)d));
  if (compressor == 1) {
    r->B = block;
    r->nb = (d + block - 1) / block;
    r->m = std::max<int64_t>(1, (int64_t)std::floor(ratio * (double)r->nb));
  }
  int hw = (int)std::thread::hardware_concurrency();
  if (hw < 1) hw = 1;
  r->threads = threads > 0 ? std::min(threads, K) : std::min(hw, K);
  r->set_eta(eta);
  r->support.resize((size_t)K);
  r->values.resize((size_t)K);
  return r;
}

void gmcref_destroy(void* h) { delete static_cast<Ref*>(h); }

int32_t gmcref_threads(void* h) { return h ? static_cast<Ref*>(h)->threads : 0; }

// w_{-1} = w_0, e_{0,k} = 0, t = 0, counters cleared (Alg. 1 initialisation).
int gmcref_set_params(void* h, const float* w0) {
  Ref* r = static_cast<Ref*>(h);
  if (!r || !w0) return 1;
  r->w.assign(w0, w0 + r->d);
  r->w_prev = r->w;
  r->e.assign((size_t)r->K * (size_t)r->d, 0.0f);
  for (auto& s : r->support) s.clear();
  for (auto& v : r->values) v.clear();
  std::memset(r->totals, 0, sizeof(r->totals));
  r->t = 0;
  r->ready = true;
  return 0;
}

int gmcref_set_eta(void* h, float eta) {
  Ref* r = static_cast<Ref*>(h);
  if (!r || !(eta > 0.f)) return 1;
  r->set_eta(eta);
  return 0;
}

// One step of Alg. 1 with g_{t,k} = grads[k*d .. k*d + d).
int gmcref_step(void* h, const float* grads) {
  Ref* r = static_cast<Ref*>(h);
  if (!r || !grads || !r->ready) return 1;
  r->step(grads);
  return 0;
}

int64_t gmcref_support_size(void* h, int32_t k) {
  Ref* r = static_cast<Ref*>(h);
  if (!r || k < 0 || k >= r->K) return -1;
  return (int64_t)r->support[(size_t)k].size();
}

// The last step's C(e_{t-1/2,k}): its support (ascending) and values.
int gmcref_support(void* h, int32_t k, int64_t* idx, float* val) {
  Ref* r = static_cast<Ref*>(h);
  if (!r || k < 0 || k >= r->K) return 1;
  const auto& s = r->support[(size_t)k];
  const auto& v = r->values[(size_t)k];
  if (idx) std::copy(s.begin(), s.end(), idx);
  if (val) std::copy(v.begin(), v.end(), val);
  return 0;
}

// The state arrays, owned by the instance: w_t (d floats) and the residuals
// e_{t,k} (K rows of d floats), valid until the next step or set_params.
const float* gmcref_w(void* h) { return h && static_cast<Ref*>(h)->ready ? static_cast<Ref*>(h)->w.data() : nullptr; }
const float* gmcref_e(void* h) { return h && static_cast<Ref*>(h)->ready ? static_cast<Ref*>(h)->e.data() : nullptr; }

// GMC+ detached point of worker k: out = w_t - (lambda*eta) * e_{t,k} (Alg. 2).
int gmcref_worker_params(void* h, int32_t k, float* out) {
  Ref* r = static_cast<Ref*>(h);
  if (!r || !r->ready || k < 0 || k >= r->K || !out) return 1;
  const float* ek = r->e.data() + (size_t)k * r->d;
  for (int64_t j = 0; j < r->d; ++j) out[j] = r->w[(size_t)j] - r->b * ek[j];
  return 0;
}

// Cumulative counters: steps, pairs, nnz, union, changed.
int gmcref_totals(void* h, uint64_t* out) {
  Ref* r = static_cast<Ref*>(h);
  if (!r || !out) return 1;
  std::copy(r->totals, r->totals + 5, out);
  return 0;
}

// Stand-alone pieces, for the pins: top-s of one vector, and the RBGS blocks.
int gmcref_top_s(const float* x, int64_t n, int64_t s, int64_t* idx) {
  if (!x || !idx || n < 1 || s < 1 || s > n) return 1;
  const auto sup = top_s_support(x, n, s);
  std::copy(sup.begin(), sup.end(), idx);
  return 0;
}

int gmcref_rbgs_blocks(uint64_t seed, int64_t t, uint64_t stream, int64_t nb, int64_t m, int64_t* out) {
  if (!out || nb < 1 || m < 1 || m > nb) return 1;
  const auto b = floyd_blocks(stream_key(seed, t, stream), nb, m);
  std::copy(b.begin(), b.end(), out);
  return 0;
}

uint64_t gmcref_splitmix64_next(uint64_t* state) {
  *state += kGolden;
  return splitmix64_mix(*state);
}

}  // extern "C"
