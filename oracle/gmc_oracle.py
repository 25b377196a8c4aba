"""GMC / GMC+ oracle: a plain, slow, CPU statement of the paper's update rules.

TEST INFRASTRUCTURE. Only the tests, ``__graft_entry__.smoke()`` and the CPU
baseline / reference arm of ``bench.py`` may import this module. The product
path (the CUDA library and its Python binding) never imports it and shares no
code with it.

What it follows (Shi et al., "Global Momentum Compression for Sparse
Communication in Distributed Learning", arXiv 1905.12948):
  * Algorithm 1 (GMC), Sec. 3.1: w_{-1} = w_0, e_{0,k} = 0;
        e_{t+1/2,k} = e_{t,k} + g_{t,k} - (beta/eta) (w_t - w_{t-1})
        e_{t+1,k}   = e_{t+1/2,k} - C(e_{t+1/2,k})
        w_{t+1}     = w_t - (eta/K) sum_k C(e_{t+1/2,k})
  * Algorithm 2 (GMC+), Sec. 4: the same step plus the detach
        w_{t+1,k}   = w_{t+1} - lambda*eta*e_{t+1,k},   w_{0,k} = w_0.
    Gradients are inputs here, so the detached points are an output only.
  * Compressors (Sec. 4): top-s (the s components of largest magnitude) and
    RBGS (random blocks chosen with one seed shared by all workers, Sec. 5.2);
    the approximate top-s of Sec. 5.1 (after DGC): a threshold theta taken
    from a random sample S of d/100 components, such that |S|/1024 -- the
    compression ratio times |S| -- sampled magnitudes reach it; every
    component with |a| >= theta is sent.
  * Relative communication cost (Sec. 5, RCC), halved for RBGS (Sec. 5.2).
  * The appendix's other ways to combine momentum and error feedback, as
    variants of the same step:
      Alg. 3 (momentum on the server): e_{t+1/2,k} = e_{t,k} + g_{t,k};
        w_{t+1} = w_t - (eta/K) sum_k C(e_{t+1/2,k}) + beta (w_t - w_{t-1});
      Alg. 4 (learning rate inside the residual):
        e_{t+1/2,k} = e_{t,k} + eta g_{t,k} - beta (w_t - w_{t-1});
        w_{t+1} = w_t - (1/K) sum_k C(e_{t+1/2,k}).
  * The local-momentum baseline the paper compares against (Sec. 2.3, eq. (3),
    with error feedback: DGC without momentum factor masking, Sec. 3.1):
        m_{t+1,k} = beta m_{t,k} + eta g_{t,k},  m_{0,k} = 0
        e_{t+1/2,k} = e_{t,k} + m_{t+1,k}; C and the residual as in Alg. 1;
        w_{t+1} = w_t - (1/K) sum_k C(e_{t+1/2,k});
    with masking (DGC w/ mfm), m_{t+1,k} is also set to 0 where worker k sent;
    the detached point of the DEF-A-like form is w_{t,k} = w_t - lambda e_{t,k}
    (the residual already carries eta).

Precision. The paper fixes none. Top-s turns floating-point magnitudes into an
integer decision (which indices are sent), so that decision is taken in the
kernel's precision, fp32; every later state depends on those decisions, so the
whole state (w, w_{t-1}, e) is fp32. Each elementary operation is one IEEE-754
round-to-nearest-even fp32 operation, evaluated in the order the algorithm
writes it: e_{t+1/2} = ((e + g) - (c * (w_t - w_{t-1}))) with c = fl(beta/eta);
the aggregate sums the workers' values in ascending worker order starting from
+0; w_{t+1} = w_t - (a * sum) with a = fl(eta/K); the detach is
w - (b * e) with b = fl(lambda*eta). numpy float32 ufuncs round each operation
once and never fuse a multiply into an add, which is exactly that.

Readings where the paper is silent:
  * top-s ties: the lower index wins; magnitudes compare through the IEEE bit
    pattern with the sign cleared, so +0 and -0 tie;
  * s = max(1, floor(ratio * d)) for a compression ratio;
  * RBGS: d is cut into aligned blocks of B (the last one may be short),
    m = max(1, floor(ratio * nb)) distinct blocks are drawn with Floyd's
    sampling (Bentley & Floyd, CACM 1987) from a SplitMix64 counter stream
    (Steele, Lea & Flood, OOPSLA 2014) keyed by (seed, t) -- or (seed, t, k)
    in the per-worker mode -- with multiply-shift range reduction;
  * the residual at a sent coordinate is +0 exactly (v - v for finite v);
  * approximate top-s: S is drawn afresh each step, the same for all
    workers, as n = max(1, floor(d/800)) runs of 8 consecutive components
    (|S| = 8n, about d/100), one run per stratum [floor(i d/n),
    floor((i+1) d/n)), starting at a multiple of 8 inside it picked by the
    i-th draw of the SplitMix64 stream keyed by (seed, t) with
    multiply-shift reduction (d < 8: S = [0, d));
    theta is the r-th largest sampled magnitude key, r = max(1,
    floor(ratio |S|)); a component is sent iff its key is >= theta's; when
    more than M = min(d, 4 s + 4096) components reach theta (s the nominal
    count of top-s), the exact top-M is sent instead.
"""
from __future__ import annotations

import math
from typing import List, Optional

import numpy as np

F32 = np.float32
U32 = np.uint32

TOPK = "topk"
RBGS = "rbgs"
TOPK_APPROX = "topk_approx"

ALG1 = "gmc"               # Algorithm 1 (the method)
ALG3 = "server_momentum"   # Algorithm 3: momentum term on the server
ALG4 = "lr_in_residual"    # Algorithm 4: learning rate inside the residual
LOCAL = "local_momentum"   # local momentum with error feedback (DGC w/o mfm)
LOCAL_MFM = "local_momentum_mfm"  # the same with momentum factor masking (DGC w/ mfm)

APPROX_SAMPLE_DIV = 100  # |S| = d/100 (Sec. 5.1)

# ---------------------------------------------------------------------------
# Compressors
# ---------------------------------------------------------------------------


def magnitude_key(x: np.ndarray) -> np.ndarray:
    """|x| as an unsigned integer that orders like |x|: the fp32 bit pattern
    with the sign bit cleared (monotone for non-negative floats)."""
    return np.ascontiguousarray(x, F32).view(U32) & U32(0x7FFFFFFF)


def topk_count(d: int, ratio: float) -> int:
    """s = max(1, floor(ratio * d)), the number of components top-s keeps."""
    return max(1, math.floor(ratio * d))


def top_s_support(x: np.ndarray, s: int) -> np.ndarray:
    """Support of the top-s compressor (Sec. 4): the s components of largest
    |x|, ties going to the lower index. Returned in ascending index order.

    Written from the definition: let kth be the s-th largest magnitude key;
    every component above kth is kept, then the lowest-index components equal
    to kth until s are kept.
    """
    d = x.size
    if not 1 <= s <= d:
        raise ValueError("s must be in [1, d]")
    key = magnitude_key(x)
    kth = np.partition(key, d - s)[d - s]
    above = np.flatnonzero(key > kth)
    ties = np.flatnonzero(key == kth)[: s - above.size]
    return np.sort(np.concatenate([above, ties]))


GOLDEN_GAMMA = 0x9E3779B97F4A7C15
_M64 = (1 << 64) - 1


def splitmix64_mix(z: int) -> int:
    """SplitMix64 output function (Steele, Lea & Flood 2014): two
    xor-shift-multiply rounds and a final xor-shift on a 64-bit word."""
    z &= _M64
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & _M64
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & _M64
    return z ^ (z >> 31)


def splitmix64_sequence(seed: int, n: int) -> List[int]:
    """The first n outputs of a SplitMix64 generator whose state starts at
    ``seed``: the state advances by the golden gamma, then is mixed."""
    out, state = [], seed & _M64
    for _ in range(n):
        state = (state + GOLDEN_GAMMA) & _M64
        out.append(splitmix64_mix(state))
    return out


def rbgs_stream_key(seed: int, t: int, stream: int) -> int:
    """Key of the block-choice stream of step t. ``stream`` is 0 when all
    workers share the choice (the paper's setting) and k+1 for worker k in the
    per-worker mode."""
    k1 = splitmix64_mix((seed + GOLDEN_GAMMA * (t + 1)) & _M64)
    return splitmix64_mix((k1 + GOLDEN_GAMMA * (stream + 1)) & _M64)


def rbgs_draw(key: int, i: int) -> int:
    """The i-th 64-bit draw of a stream: SplitMix64 in counter form."""
    return splitmix64_mix((key + GOLDEN_GAMMA * (i + 1)) & _M64)


def below(x: int, n: int) -> int:
    """Map a 64-bit draw to [0, n) by multiply-shift on its top 32 bits."""
    return ((x >> 32) * n) >> 32


def floyd_blocks(key: int, nb: int, m: int) -> np.ndarray:
    """m distinct block ids out of [0, nb), Floyd's sampling without
    replacement, returned sorted ascending."""
    chosen = set()
    for i, j in enumerate(range(nb - m, nb)):
        r = below(rbgs_draw(key, i), j + 1)
        chosen.add(j if r in chosen else r)
    return np.array(sorted(chosen), np.int64)


APPROX_RUN = 8  # consecutive components per run of the sample


def approx_runs(d: int) -> int:
    """Runs of the sample: max(1, floor(d/800)), so that |S| is about d/100."""
    return max(1, d // (APPROX_SAMPLE_DIV * APPROX_RUN))


def approx_sample_size(d: int) -> int:
    """|S| = 8 * runs (all of [0, d) when d < 8), about d/100 (Sec. 5.1)."""
    return d if d < APPROX_RUN else APPROX_RUN * approx_runs(d)


def approx_rank(n_sample: int, ratio: float) -> int:
    """r = max(1, floor(ratio * |S|)): how many sampled magnitudes reach theta
    (|S|/1024 in Sec. 5.1, where the ratio is 1/1024)."""
    return max(1, math.floor(ratio * n_sample))


def approx_limit(d: int, ratio: float) -> int:
    """M = min(d, 4 s + 4096): the most components the approximate top-s sends
    (beyond it, the exact top-M)."""
    return min(d, 4 * topk_count(d, ratio) + 4096)


def approx_sample_positions(seed: int, t: int, d: int) -> np.ndarray:
    """The sample S of step t, ascending. Stratum i = [floor(i d/n),
    floor((i+1) d/n)) of the n runs contributes the 8 components from
    a_i + 8 * below(draw_i, m_i), where a_i is lo_i rounded up to a multiple of
    8, m_i the number of whole runs of 8 from a_i inside the stratum, and
    draw_i the i-th draw of the stream keyed by (seed, t) (the shared RBGS
    stream). d < 8: all of [0, d). Python integers throughout."""
    if d < APPROX_RUN:
        return np.arange(d, dtype=np.int64)
    n = approx_runs(d)
    key = rbgs_stream_key(seed, t, 0)
    out = np.empty(APPROX_RUN * n, np.int64)
    for i in range(n):
        lo, hi = i * d // n, (i + 1) * d // n
        a = -(-lo // APPROX_RUN) * APPROX_RUN
        m = (hi - a) // APPROX_RUN
        start = a + APPROX_RUN * below(rbgs_draw(key, i), m)
        out[APPROX_RUN * i: APPROX_RUN * (i + 1)] = np.arange(start, start + APPROX_RUN)
    return out


def approx_top_s_support(x: np.ndarray, sample: np.ndarray, r: int, limit: int):
    """Support of the approximate top-s (Sec. 5.1) and its threshold key:
    theta = the r-th largest magnitude key among x[sample]; every component
    whose key is >= theta is sent, unless more than `limit` are, in which case
    the exact top-`limit` is. Returned in ascending index order."""
    key = magnitude_key(x)
    sampled = np.sort(key[sample])[::-1]
    theta = int(sampled[r - 1])
    support = np.flatnonzero(key >= U32(theta))
    if support.size > limit:
        support = top_s_support(x, limit)
    return support, theta


def rbgs_support(blocks: np.ndarray, B: int, d: int) -> np.ndarray:
    """Coordinates covered by the chosen blocks, ascending."""
    if blocks.size == 0:
        return np.zeros(0, np.int64)
    return np.concatenate([np.arange(b * B, min((b + 1) * B, d)) for b in blocks])


# ---------------------------------------------------------------------------
# GMC / GMC+ state and step
# ---------------------------------------------------------------------------


class StepResult:
    """What one step produced (kept for the tests)."""

    def __init__(self, e_half, supports, values, w_next, blocks, stats, sample=None,
                 thresholds=None):
        self.sample = sample          # approximate top-s: the sampled positions S
        self.thresholds = thresholds  # approximate top-s: theta's key per worker
        self.e_half = e_half          # e_{t+1/2,k}, float32 [K, d]
        self.supports = supports      # list of K int64 index arrays (ascending)
        self.values = values          # list of K float32 arrays: C(e_{t+1/2,k}) on its support
        self.w_next = w_next          # w_{t+1}
        self.blocks = blocks          # RBGS: list of chosen block arrays (per stream), else None
        self.stats = stats            # dict of per-step counters


class GMC:
    """Algorithm 1 (GMC) and Algorithm 2 (GMC+) for K workers, dense arrays."""

    def __init__(self, d: int, K: int, beta: float, eta: float, compressor: str = TOPK,
                 ratio: float = 0.01, block: int = 4096, lam: float = 0.0, seed: int = 0,
                 per_worker: bool = False, variant: str = ALG1):
        if d < 1 or K < 1:
            raise ValueError("d and K must be >= 1")
        if not 0.0 <= beta < 1.0:
            raise ValueError("beta must be in [0, 1)")
        if not eta > 0.0:
            raise ValueError("eta must be > 0")
        if not 0.0 < ratio <= 1.0:
            raise ValueError("ratio must be in (0, 1]")
        if compressor not in (TOPK, RBGS, TOPK_APPROX):
            raise ValueError("unknown compressor")
        if variant not in (ALG1, ALG3, ALG4, LOCAL, LOCAL_MFM):
            raise ValueError("unknown variant")
        if variant != ALG1 and compressor == RBGS:
            raise ValueError("the variants take a top-s compressor")
        if variant in (ALG3, ALG4) and lam != 0.0:
            raise ValueError("GMC+ detaches Alg. 1 only")
        self.variant = variant
        self.d, self.K = d, K
        self.beta = F32(beta)
        self.lam = F32(lam)
        self.compressor = compressor
        self.ratio = ratio
        self.seed = seed
        self.per_worker = per_worker
        if compressor == TOPK:
            self.s = topk_count(d, ratio)
        elif compressor == TOPK_APPROX:
            self.s = topk_count(d, ratio)
            self.n_sample = approx_sample_size(d)
            self.r_sample = approx_rank(self.n_sample, ratio)
            self.limit = approx_limit(d, ratio)
        else:
            if block < 1:
                raise ValueError("block must be >= 1")
            self.B = block
            self.nb = -(-d // block)
            self.m = max(1, math.floor(ratio * self.nb))
        self.set_eta(eta)
        self.w = None

    def set_eta(self, eta: float) -> None:
        """Constants of the step, each one fp32 rounding of the paper's ratio.
        Alg. 4 scales the residual update by 1/K instead of eta/K."""
        self.eta = F32(eta)
        self.c = F32(self.beta / self.eta)          # beta / eta
        self.a = F32(self.eta / F32(self.K))        # eta / K
        if self.variant in (ALG4, LOCAL, LOCAL_MFM):
            self.a = F32(F32(1.0) / F32(self.K))    # 1 / K
        self.b = F32(self.lam * self.eta)           # lambda * eta
        if self.variant in (LOCAL, LOCAL_MFM):
            self.b = self.lam                       # lambda (e carries eta)

    def set_params(self, w0: np.ndarray) -> None:
        """Initial state: w_{-1} = w_0 and e_{0,k} = 0 (Alg. 1 and Alg. 2)."""
        w0 = np.asarray(w0, F32)
        if w0.shape != (self.d,):
            raise ValueError("w0 must have shape (d,)")
        self.w = w0.copy()
        self.w_prev = w0.copy()
        self.e = np.zeros((self.K, self.d), F32)
        self.u = np.zeros((self.K, self.d), F32)    # local momentum m_{t,k} (local variants)
        self.t = 0
        self.totals = dict(steps=0, pairs=0, nnz=0, union=0, changed=0)

    # -- compressor support for worker k at the current step -----------------
    def _blocks(self) -> List[np.ndarray]:
        streams = range(1, self.K + 1) if self.per_worker else [0]
        return [floyd_blocks(rbgs_stream_key(self.seed, self.t, s), self.nb, self.m)
                for s in streams]

    def step(self, grads: np.ndarray) -> StepResult:
        """One iteration t of Algorithm 1 / 2 with g_{t,k} = grads[k]."""
        if self.w is None:
            raise RuntimeError("set_params first")
        g = np.asarray(grads, F32)
        if g.shape != (self.K, self.d):
            raise ValueError("grads must have shape (K, d)")
        K = self.K

        # workers: e_{t+1/2,k} = e_{t,k} + g_{t,k} - (beta/eta)(w_t - w_{t-1})
        if self.variant == ALG1:
            e_half = (self.e + g) - self.c * (self.w - self.w_prev)
        elif self.variant == ALG3:   # e_{t,k} + g_{t,k}
            e_half = self.e + g
        elif self.variant == ALG4:   # e_{t,k} + eta g_{t,k} - beta (w_t - w_{t-1})
            e_half = (self.e + self.eta * g) - self.beta * (self.w - self.w_prev)
        else:                        # m = beta m + eta g; e_{t,k} + m_{t+1,k}
            m_next = self.beta * self.u + self.eta * g
            e_half = self.e + m_next

        # workers: C(e_{t+1/2,k}) -- its support and values
        blocks = sample = thresholds = None
        if self.compressor == TOPK:
            supports = [top_s_support(e_half[k], self.s) for k in range(K)]
        elif self.compressor == TOPK_APPROX:
            sample = approx_sample_positions(self.seed, self.t, self.d)
            picked = [approx_top_s_support(e_half[k], sample, self.r_sample, self.limit)
                      for k in range(K)]
            supports = [p[0] for p in picked]
            thresholds = [p[1] for p in picked]
        else:
            blocks = self._blocks()
            per_stream = [rbgs_support(b, self.B, self.d) for b in blocks]
            supports = [per_stream[k if self.per_worker else 0] for k in range(K)]
        values = [e_half[k, supports[k]].copy() for k in range(K)]

        # workers: e_{t+1,k} = e_{t+1/2,k} - C(e_{t+1/2,k})
        e_next = e_half.copy()
        for k in range(K):
            e_next[k, supports[k]] = F32(0.0)
        if self.variant in (LOCAL, LOCAL_MFM):
            if self.variant == LOCAL_MFM:  # momentum factor masking
                for k in range(K):
                    m_next[k, supports[k]] = F32(0.0)
            self.u = m_next

        # server: w_{t+1} = w_t - (eta/K) sum_k C(e_{t+1/2,k}), workers summed in order
        # (Alg. 4: 1/K in a; Alg. 3 adds beta (w_t - w_{t-1}))
        total = np.zeros(self.d, F32)
        for k in range(K):
            total[supports[k]] = total[supports[k]] + values[k]
        w_next = self.w - self.a * total
        if self.variant == ALG3:
            w_next = w_next + self.beta * (self.w - self.w_prev)

        in_union = np.zeros(self.d, bool)
        for k in range(K):
            in_union[supports[k]] = True
        stats = dict(
            pairs=int(sum(s.size for s in supports)),
            nnz=int(sum(np.count_nonzero(v) for v in values)),
            union=int(np.count_nonzero(in_union)),
            changed=int(np.count_nonzero(w_next - self.w)),
        )
        for key, val in stats.items():
            self.totals[key] += val
        self.totals["steps"] += 1

        self.w_prev, self.w, self.e = self.w, w_next, e_next
        self.t += 1
        return StepResult(e_half, supports, values, w_next, blocks, stats, sample, thresholds)

    def worker_params(self, k: int) -> np.ndarray:
        """GMC+ detached point of worker k: w_{t,k} = w_t - lambda*eta*e_{t,k}."""
        return self.w - self.b * self.e[k]

    def rcc(self) -> float:
        """Relative communication cost over the steps so far (Sec. 5):
        (1/(d K T)) sum_t (K ||w_{t+1}-w_t||_0 + sum_k ||C_k||_0), halved for
        RBGS, whose messages carry no indices (Sec. 5.2)."""
        T = self.totals["steps"]
        if T == 0:
            return 0.0
        num = self.K * self.totals["changed"] + self.totals["nnz"]
        r = num / (self.d * self.K * T)
        return r / 2 if self.compressor == RBGS else r
