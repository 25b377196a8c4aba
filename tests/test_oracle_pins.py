"""Pins of the oracle against what the paper and the mathematics fix.

Each test checks the oracle (oracle/gmc_oracle.py) against something other
than itself: a reduction to a textbook method in float64, a closed form, an
identity the paper derives (Sec. 3.3 update rule, Lemma 1, the GMC+ mean-iterate
recursion of Sec. 4), brute force on tiny inputs, published generator outputs
or a value the paper prints. Together they are chosen so that a dropped term,
a wrong sign or coefficient, a wrong index or a transposed operand in the oracle
fails at least one of them.
"""
import itertools
import json
import math
import os

import numpy as np
import pytest

import oracle
from oracle import GMC, RBGS, TOPK, TOPK_APPROX

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
U = 2.0 ** -24  # unit roundoff of fp32


def _golden(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


def _grads(rng, T, K, d, scale=1.0):
    return [(rng.standard_normal((K, d)) * scale).astype(np.float32) for _ in range(T)]


# ---------------------------------------------------------------------------
# P1: beta = 0 and no compression -> distributed SGD (Sec. 2.3, Sec. 3.3)
# ---------------------------------------------------------------------------

def test_p1_sgd_reduction():
    rng = np.random.default_rng(1)
    d, K, T, eta = 257, 3, 20, 0.1
    o = GMC(d, K, beta=0.0, eta=eta, compressor=TOPK, ratio=1.0)
    w0 = rng.standard_normal(d).astype(np.float32)
    o.set_params(w0)
    grads = _grads(rng, T, K, d)
    w_ref = w0.astype(np.float64)
    tol = np.zeros(d)
    eta32 = float(np.float32(eta))
    for g in grads:
        o.step(g)
        assert not np.any(o.e), "with no compression the residual must stay exactly 0"
        g64 = g.astype(np.float64)
        w_ref = w_ref - eta32 / K * g64.sum(0)
        tol += (K + 3) * U * eta32 / K * np.abs(g64).sum(0) + 2 * U * np.abs(o.w)
        np.testing.assert_array_less(np.abs(o.w - w_ref), 2 * tol + 1e-30)


# ---------------------------------------------------------------------------
# P2: no compression, beta > 0 -> heavy-ball MSGD (Sec. 2.3, eq. (2))
# ---------------------------------------------------------------------------

def _heavy_ball(w0, grads, eta, beta):
    """w_{t+1} = w_t - eta*mean_k g_{t,k} + beta*(w_t - w_{t-1}), w_{-1} = w_0, in float64."""
    w_prev, w = w0.copy(), w0.copy()
    out = [w.copy()]
    for g in grads:
        w_next = w - eta * g.mean(0) + beta * (w - w_prev)
        w_prev, w = w, w_next
        out.append(w.copy())
    return out


def test_p2_heavy_ball_closed_form():
    """The float64 recursion itself against the textbook closed form for a
    constant gradient: w_t = w_0 - eta*g/(1-beta) * [t - beta(1-beta^t)/(1-beta)]."""
    eta, beta, T = 0.05, 0.9, 60
    g = np.array([[0.3, -1.2, 2.0]])
    w0 = np.array([1.0, -2.0, 0.5])
    traj = _heavy_ball(w0, [g] * T, eta, beta)
    for t in range(T + 1):
        closed = w0 - eta * g[0] / (1 - beta) * (t - beta * (1 - beta ** t) / (1 - beta))
        np.testing.assert_allclose(traj[t], closed, rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("K", [1, 4])
def test_p2_heavy_ball_reduction(K):
    rng = np.random.default_rng(2 + K)
    d, T, eta, beta = 129, 40, 0.05, 0.9
    o = GMC(d, K, beta=beta, eta=eta, compressor=TOPK, ratio=1.0)
    w0 = rng.standard_normal(d).astype(np.float32)
    o.set_params(w0)
    grads = _grads(rng, T, K, d)
    eta32, beta32 = float(np.float32(eta)), float(np.float32(beta))
    ref = _heavy_ball(w0.astype(np.float64), [g.astype(np.float64) for g in grads], eta32, beta32)
    budget = np.zeros(d)
    w_prev = w0.astype(np.float64)
    for t, g in enumerate(grads):
        w_t = o.w.astype(np.float64)
        o.step(g)
        assert not np.any(o.e)
        w_next = o.w.astype(np.float64)
        dlt = np.abs(w_t - w_prev)
        local = 6 * U * (np.abs(w_next) + np.abs(w_t) + (K + 3) * eta32 / K *
                         (np.abs(g.astype(np.float64)).sum(0) + K * beta32 / eta32 * dlt) + beta32 * dlt)
        budget += local
        err = np.abs(w_next - ref[t + 1])
        np.testing.assert_array_less(err, 2 * budget / (1 - beta32) + 1e-30)
        w_prev = w_t


def test_p2_constant_gradient_against_closed_form():
    """The fp32 oracle (ratio = 1, K workers with the same constant gradient)
    tracks the closed form of P2 to fp32 accuracy."""
    d, K, T, eta, beta = 5, 2, 50, 0.05, 0.9
    g = np.array([0.3, -1.2, 2.0, 0.0, 1e-3], np.float32)
    w0 = np.array([1.0, -2.0, 0.5, 3.0, 0.0], np.float32)
    o = GMC(d, K, beta=beta, eta=eta, compressor=TOPK, ratio=1.0)
    o.set_params(w0)
    eta64, beta64 = float(np.float32(eta)), float(np.float32(beta))
    for t in range(1, T + 1):
        o.step(np.stack([g] * K))
        closed = w0 - eta64 * g / (1 - beta64) * (t - beta64 * (1 - beta64 ** t) / (1 - beta64))
        np.testing.assert_allclose(o.w, closed, rtol=2e-5, atol=2e-6)


# ---------------------------------------------------------------------------
# P3: C(v) + e = v exactly, for every worker, coordinate and step (Alg. 1)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("compressor", [TOPK, RBGS, TOPK_APPROX])
def test_p3_exact_split(compressor):
    rng = np.random.default_rng(3)
    d, K, T = 1000, 4, 12
    o = GMC(d, K, beta=0.9, eta=0.1, compressor=compressor, ratio=0.05, block=64, seed=5,
            per_worker=True)
    o.set_params(rng.standard_normal(d).astype(np.float32))
    for g in _grads(rng, T, K, d):
        r = o.step(g)
        for k in range(K):
            S = r.supports[k]
            sel = np.zeros(d, bool)
            sel[S] = True
            vbits = r.e_half[k].view(np.uint32)
            ebits = o.e[k].view(np.uint32)
            assert np.all(ebits[sel] == 0), "sent coordinates leave +0 behind"
            assert np.all(ebits[~sel] == vbits[~sel]), "unsent coordinates keep v bitwise"
            assert np.all(r.values[k].view(np.uint32) == vbits[S]), "C(v) carries v bitwise"
            np.testing.assert_array_equal(S, np.sort(S))


# ---------------------------------------------------------------------------
# P4: top-s by brute force on tiny inputs, ties and signed zeros included
# ---------------------------------------------------------------------------

def _brute_top_s(x, s):
    order = sorted(range(x.size), key=lambda j: (-abs(float(x[j])), j))
    return np.array(sorted(order[:s]), np.int64)


def _tiny_inputs(rng, n_cases):
    kinds = ["normal", "small_set", "all_equal", "zeros", "signed_zero", "wide"]
    for case in range(n_cases):
        d = int(rng.integers(1, 257))
        kind = kinds[case % len(kinds)]
        if kind == "normal":
            x = rng.standard_normal(d)
        elif kind == "small_set":
            x = rng.choice([-2.0, -1.0, -0.0, 0.0, 1.0, 2.0], size=d)
        elif kind == "all_equal":
            x = np.full(d, rng.choice([-3.5, 0.25, 7.0]))
        elif kind == "zeros":
            x = np.zeros(d)
        elif kind == "signed_zero":
            x = rng.choice([-0.0, 0.0, 1e-45, -1e-45, 1.0], size=d)
        else:
            x = rng.standard_normal(d) * np.exp(rng.uniform(-80, 80, size=d))
        s = int(rng.integers(1, d + 1))
        yield x.astype(np.float32), s


def test_p4_top_s_brute_force():
    rng = np.random.default_rng(4)
    for x, s in _tiny_inputs(rng, 10_000):
        got = oracle.top_s_support(x, s)
        np.testing.assert_array_equal(got, _brute_top_s(x, s))


def test_p4_top_s_properties():
    """min kept |x| >= max dropped |x|, and the delta-approximate bound of
    Assumption 1 with delta = s/d holds deterministically for top-s."""
    rng = np.random.default_rng(44)
    for x, s in _tiny_inputs(rng, 2_000):
        S = oracle.top_s_support(x, s)
        keep = np.zeros(x.size, bool)
        keep[S] = True
        a = np.abs(x.astype(np.float64))
        if keep.all():
            continue
        assert a[keep].min() >= a[~keep].max()
        cx = np.where(keep, x.astype(np.float64), 0.0)
        lhs = np.sum((cx - x) ** 2)
        assert lhs <= (1 - s / x.size) * np.sum(x.astype(np.float64) ** 2) * (1 + 1e-12) + 1e-300


def test_magnitude_key_orders_like_abs():
    rng = np.random.default_rng(45)
    x = np.concatenate([rng.standard_normal(500) * np.exp(rng.uniform(-85, 85, 500)),
                        [0.0, -0.0, 1e-45, -1e-45, np.inf, -np.inf, 3.0e38]]).astype(np.float32)
    key = oracle.magnitude_key(x)
    a = np.abs(x.astype(np.float64))
    for i, j in itertools.combinations(range(x.size), 2):
        assert (key[i] < key[j]) == (a[i] < a[j])
        assert (key[i] == key[j]) == (a[i] == a[j])


def test_full_ratio_is_identity():
    x = np.random.default_rng(46).standard_normal(77).astype(np.float32)
    np.testing.assert_array_equal(oracle.top_s_support(x, x.size), np.arange(x.size))


def test_topk_count():
    """s = max(1, floor(ratio*d)) gives the configured sizes."""
    assert oracle.topk_count(65_536, 0.01) == 655
    assert oracle.topk_count(272_474, 0.01) == 2_724
    assert oracle.topk_count(11_173_962, 0.001) == 11_173
    assert oracle.topk_count(138_357_544, 0.001) == 138_357
    assert oracle.topk_count(10, 0.01) == 1


# ---------------------------------------------------------------------------
# P5, P6: the update rule with C eliminated (Sec. 3.3) and Lemma 1
# ---------------------------------------------------------------------------

def _update_rule_residual(o, grads):
    """Yield, after each step: both sides of w_{t+1} - w_t = -eta*gbar - eta*ebar_t +
    eta*ebar_{t+1} + beta*(w_t - w_{t-1}), with an fp32 rounding budget."""
    eta = float(o.eta)
    beta = float(o.beta)
    K = o.K
    c = float(o.c)
    w_prev = o.w.astype(np.float64)
    for g in grads:
        w_t = o.w.astype(np.float64)
        e_t = o.e.astype(np.float64)
        r = o.step(g)
        w_n = o.w.astype(np.float64)
        e_n = o.e.astype(np.float64)
        g64 = g.astype(np.float64)
        lhs = w_n - w_t
        rhs = -eta * g64.mean(0) - eta * e_t.mean(0) + eta * e_n.mean(0) + beta * (w_t - w_prev)
        dl = np.abs(w_t - w_prev)
        v = np.abs(r.e_half.astype(np.float64))
        scale = (np.abs(e_t) + np.abs(g64) + c * dl + v + np.abs(e_n)).sum(0)
        budget = 8 * U * (np.abs(w_n) + np.abs(w_t) + (K + 3) * eta / K * scale + beta * dl)
        yield lhs, rhs, budget, w_t, w_prev, e_t, e_n, g64
        w_prev = w_t


@pytest.mark.parametrize("compressor", [TOPK, RBGS, TOPK_APPROX])
def test_p5_update_rule(compressor):
    rng = np.random.default_rng(5)
    d, K, T = 600, 4, 30
    o = GMC(d, K, beta=0.9, eta=0.1, compressor=compressor, ratio=0.05, block=16, seed=9)
    o.set_params(rng.standard_normal(d).astype(np.float32))
    for lhs, rhs, budget, *_ in _update_rule_residual(o, _grads(rng, T, K, d)):
        np.testing.assert_array_less(np.abs(lhs - rhs), budget + 1e-30)


@pytest.mark.parametrize("compressor", [TOPK, RBGS, TOPK_APPROX])
def test_p6_lemma1_z_sequence(compressor):
    """z_t = w_t + beta/(1-beta)(w_t - w_{t-1}) - eta/(1-beta) ebar_t obeys
    z_{t+1} = z_t - eta/(1-beta) gbar_t for any compressor (Lemma 1)."""
    rng = np.random.default_rng(6)
    d, K, T = 400, 3, 25
    o = GMC(d, K, beta=0.9, eta=0.1, compressor=compressor, ratio=0.02, block=8, seed=3)
    o.set_params(rng.standard_normal(d).astype(np.float32))
    beta, eta = float(o.beta), float(o.eta)
    for lhs, rhs, budget, w_t, w_prev, e_t, e_n, g in _update_rule_residual(o, _grads(rng, T, K, d)):
        w_n = w_t + lhs
        z_t = w_t + beta / (1 - beta) * (w_t - w_prev) - eta / (1 - beta) * e_t.mean(0)
        z_n = w_n + beta / (1 - beta) * (w_n - w_t) - eta / (1 - beta) * e_n.mean(0)
        err = np.abs(z_n - (z_t - eta / (1 - beta) * g.mean(0)))
        np.testing.assert_array_less(err, 2 * budget / (1 - beta) + 1e-30)


# ---------------------------------------------------------------------------
# P6b, P7: GMC+ (Alg. 2) -- the mean-iterate recursion and lambda = 0
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("compressor", [RBGS, TOPK, TOPK_APPROX])
def test_p6b_gmcplus_mean_iterate(compressor):
    """With wbar_t = mean_k w_{t,k} (the detached points), Sec. 4's
    zbar_t = wbar_t + beta/(1-beta)(wbar_t - wbar_{t-1})
             - [(1-lam) eta ebar_t + beta lam eta ebar_{t-1}] / (1-beta)
    obeys zbar_{t+1} = zbar_t - eta/(1-beta) * mean_k g_{t,k}."""
    rng = np.random.default_rng(7)
    d, K, T, lam = 300, 4, 25, 0.5
    o = GMC(d, K, beta=0.9, eta=0.1, compressor=compressor, ratio=0.05, block=10, lam=lam, seed=1)
    o.set_params(rng.standard_normal(d).astype(np.float32))
    beta, eta = float(o.beta), float(o.eta)
    lam = float(o.lam)

    def wbar():
        return np.mean([o.worker_params(k).astype(np.float64) for k in range(K)], axis=0)

    wb_prev = o.w.astype(np.float64)       # wbar_{-1} = w_0
    eb_prev = np.zeros(d)                  # ebar_{-1} = 0
    wb = wbar()
    eb = o.e.astype(np.float64).mean(0)
    z = wb + beta / (1 - beta) * (wb - wb_prev) - ((1 - lam) * eta * eb + beta * lam * eta * eb_prev) / (1 - beta)
    for lhs, rhs, budget, w_t, w_prev, e_t, e_n, g in _update_rule_residual(o, _grads(rng, T, K, d)):
        wb_n = wbar()
        eb_n = o.e.astype(np.float64).mean(0)
        z_n = wb_n + beta / (1 - beta) * (wb_n - wb) - ((1 - lam) * eta * eb_n + beta * lam * eta * eb) / (1 - beta)
        err = np.abs(z_n - (z - eta / (1 - beta) * g.mean(0)))
        detach_budget = 4 * U * (np.abs(wb) + np.abs(wb_n) + lam * eta * (np.abs(e_t) + np.abs(e_n)).sum(0))
        np.testing.assert_array_less(err, 2 * (budget + detach_budget) / (1 - beta) + 1e-30)
        wb, eb, z = wb_n, eb_n, z_n


def test_p7_lambda_zero_is_gmc():
    rng = np.random.default_rng(8)
    d, K, T = 200, 3, 10
    runs = []
    for lam in (0.0, 0.5):
        o = GMC(d, K, beta=0.9, eta=0.1, compressor=RBGS, ratio=0.1, block=7, lam=lam, seed=2)
        o.set_params(np.ones(d, np.float32))
        for g in _grads(np.random.default_rng(80), T, K, d):
            o.step(g)
        runs.append(o)
    a, b = runs
    assert np.array_equal(a.w.view(np.uint32), b.w.view(np.uint32))
    assert np.array_equal(a.e.view(np.uint32), b.e.view(np.uint32))
    for k in range(K):
        assert np.array_equal(a.worker_params(k).view(np.uint32), a.w.view(np.uint32))
    assert not np.array_equal(b.worker_params(0), b.w)
    del rng


# ---------------------------------------------------------------------------
# P8: RBGS -- generator, sampler, counts, RCC
# ---------------------------------------------------------------------------

def test_splitmix64_published_outputs():
    gold = _golden("splitmix64.json")
    for seed, key in ((0, "seed_0"), (1234567, "seed_1234567")):
        want = [int(h, 16) for h in gold[key]]
        assert oracle.splitmix64_sequence(seed, len(want)) == want


def test_below_range():
    for n in (1, 2, 3, 6240, 2 ** 32):
        for x in (0, 1, 2 ** 32 - 1, 2 ** 63, 2 ** 64 - 1, 0x123456789ABCDEF0):
            assert 0 <= oracle.below(x, n) < n
    assert oracle.below(2 ** 64 - 1, 6240) == 6239


def test_floyd_uniform_over_subsets():
    """Floyd's sampler fed by the generator hits every m-subset of [0, nb)
    equally often (chi-square, 20 subsets of 3 out of 6)."""
    nb, m, n = 6, 3, 20_000
    counts = {}
    for i in range(n):
        key = oracle.rbgs_stream_key(12345, i, 0)
        sub = tuple(oracle.floyd_blocks(key, nb, m))
        assert len(set(sub)) == m and list(sub) == sorted(sub)
        counts[sub] = counts.get(sub, 0) + 1
    assert len(counts) == math.comb(nb, m)
    expected = n / len(counts)
    chi2 = sum((c - expected) ** 2 / expected for c in counts.values())
    assert chi2 < 60.0  # 19 degrees of freedom; p < 1e-5 beyond this


@pytest.mark.parametrize("per_worker", [False, True])
def test_p8_rbgs_counts(per_worker):
    rng = np.random.default_rng(9)
    d, K, B, ratio = 1000, 5, 64, 0.2     # nb = 16 (last block 40 long), m = 3
    o = GMC(d, K, beta=0.9, eta=0.1, compressor=RBGS, ratio=ratio, block=B, seed=77,
            per_worker=per_worker)
    o.set_params(rng.standard_normal(d).astype(np.float32))
    assert (o.nb, o.m) == (16, 3)
    for t in range(6):
        r = o.step(rng.standard_normal((K, d)).astype(np.float32))
        assert len(r.blocks) == (K if per_worker else 1)
        for blocks in r.blocks:
            assert blocks.size == o.m and np.unique(blocks).size == o.m
            assert blocks.min() >= 0 and blocks.max() < o.nb
        for k in range(K):
            blocks = r.blocks[k if per_worker else 0]
            size = sum(min((b + 1) * B, d) - b * B for b in blocks)
            assert r.supports[k].size == size
            assert np.count_nonzero(r.values[k]) == size
        if not per_worker:
            for k in range(1, K):
                np.testing.assert_array_equal(r.supports[k], r.supports[0])
    if per_worker:
        assert any(not np.array_equal(r.supports[k], r.supports[0]) for k in range(1, K))


def test_p8_rbgs_rcc_matches_paper():
    """One shared block of d/1024 components: RCC = 1/1024 (Sec. 5.2)."""
    gold = _golden("rcc_rbgs.json")
    d, K = 1024 * 37, 4
    B = d // 1024
    nb = -(-d // B)
    ratio = 1.0 / nb                       # m = max(1, floor(ratio * nb)) = 1
    o = GMC(d, K, beta=0.9, eta=0.1, compressor=RBGS, ratio=ratio, block=B, seed=4)
    assert o.m == gold["blocks_chosen"]
    rng = np.random.default_rng(10)
    o.set_params(rng.standard_normal(d).astype(np.float32))
    for _ in range(5):
        o.step((rng.standard_normal((K, d)) + 3.0).astype(np.float32))
    assert o.rcc() == pytest.approx(gold["rcc"], rel=0, abs=1e-15)


def test_rcc_dense_pairs():
    """No compression with (index, value) pairs: every component is sent by
    every worker and every parameter changes, so RCC = 2 (Sec. 5 accounting)."""
    rng = np.random.default_rng(11)
    d, K = 50, 3
    o = GMC(d, K, beta=0.5, eta=0.1, compressor=TOPK, ratio=1.0)
    o.set_params(rng.standard_normal(d).astype(np.float32))
    for _ in range(4):
        o.step((rng.standard_normal((K, d)) + 5.0).astype(np.float32))
    assert o.rcc() == 2.0


# ---------------------------------------------------------------------------
# The appendix variants: Alg. 3 (momentum on the server) and Alg. 4 (learning
# rate inside the residual)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("variant", [oracle.ALG3, oracle.ALG4])
def test_variants_without_compression_are_heavy_ball(variant):
    """ratio = 1: both variants leave e = 0 exactly and follow the heavy-ball
    recursion of eq. (2) in float64 (the appendix: they differ from GMC only
    in how the compression error is fed back)."""
    rng = np.random.default_rng(21)
    d, K, T, eta, beta = 129, 3, 40, 0.05, 0.9
    o = GMC(d, K, beta=beta, eta=eta, compressor=TOPK, ratio=1.0, variant=variant)
    w0 = rng.standard_normal(d).astype(np.float32)
    o.set_params(w0)
    grads = _grads(rng, T, K, d)
    eta32, beta32 = float(np.float32(eta)), float(np.float32(beta))
    ref = _heavy_ball(w0.astype(np.float64), [g.astype(np.float64) for g in grads], eta32, beta32)
    budget = np.zeros(d)
    w_prev = w0.astype(np.float64)
    for t, g in enumerate(grads):
        w_t = o.w.astype(np.float64)
        o.step(g)
        assert not np.any(o.e)
        w_next = o.w.astype(np.float64)
        dlt = np.abs(w_t - w_prev)
        local = 6 * U * (np.abs(w_next) + np.abs(w_t) + (K + 3) * eta32 / K *
                         (np.abs(g.astype(np.float64)).sum(0) + K * beta32 / eta32 * dlt) + beta32 * dlt)
        budget += local
        np.testing.assert_array_less(np.abs(w_next - ref[t + 1]), 2 * budget / (1 - beta32) + 1e-30)
        w_prev = w_t


def test_alg3_update_rule_is_gmcs():
    """Eliminating C from Alg. 3 gives GMC's update rule (the appendix): the
    P5 identity holds for Alg. 3's residuals."""
    rng = np.random.default_rng(22)
    d, K, T = 600, 4, 30
    o = GMC(d, K, beta=0.9, eta=0.1, compressor=TOPK, ratio=0.05, variant=oracle.ALG3)
    o.set_params(rng.standard_normal(d).astype(np.float32))
    for lhs, rhs, budget, *_ in _update_rule_residual(o, _grads(rng, T, K, d)):
        np.testing.assert_array_less(np.abs(lhs - rhs), budget + 1e-30)


def test_alg4_update_rule():
    """Alg. 4 with C eliminated: w_{t+1} - w_t = -eta gbar - ebar_t + ebar_{t+1}
    + beta (w_t - w_{t-1}) (its residual carries the learning rate)."""
    rng = np.random.default_rng(23)
    d, K, T, eta, beta = 600, 4, 30, 0.1, 0.9
    o = GMC(d, K, beta=beta, eta=eta, compressor=TOPK, ratio=0.05, variant=oracle.ALG4)
    o.set_params(rng.standard_normal(d).astype(np.float32))
    eta32, beta32 = float(np.float32(eta)), float(np.float32(beta))
    w_prev = o.w.astype(np.float64)
    for g in _grads(rng, T, K, d):
        w_t, e_t = o.w.astype(np.float64), o.e.astype(np.float64)
        r = o.step(g)
        w_n, e_n, g64 = o.w.astype(np.float64), o.e.astype(np.float64), g.astype(np.float64)
        lhs = w_n - w_t
        rhs = -eta32 * g64.mean(0) - e_t.mean(0) + e_n.mean(0) + beta32 * (w_t - w_prev)
        dl = np.abs(w_t - w_prev)
        scale = (np.abs(e_t) + eta32 * np.abs(g64) + beta32 * dl + np.abs(r.e_half) + np.abs(e_n)).sum(0)
        budget = 8 * U * (np.abs(w_n) + np.abs(w_t) + (K + 3) / K * scale + beta32 * dl)
        np.testing.assert_array_less(np.abs(lhs - rhs), budget + 1e-30)
        w_prev = w_t


@pytest.mark.parametrize("variant", [oracle.ALG3, oracle.ALG4])
def test_variants_reduce_to_gmc(variant):
    """Bitwise: with beta = 0 Alg. 3 is GMC; with beta = 0 and eta = 1 Alg. 4
    is GMC (the learning-rate factor and the 1/K scale coincide)."""
    rng = np.random.default_rng(24)
    d, K, T = 500, 3, 10
    eta = 1.0 if variant == oracle.ALG4 else 0.1
    a = GMC(d, K, beta=0.0, eta=eta, compressor=TOPK, ratio=0.05)
    b = GMC(d, K, beta=0.0, eta=eta, compressor=TOPK, ratio=0.05, variant=variant)
    w0 = rng.standard_normal(d).astype(np.float32)
    a.set_params(w0)
    b.set_params(w0)
    for g in _grads(rng, T, K, d):
        ra, rb = a.step(g), b.step(g)
        for k in range(K):
            np.testing.assert_array_equal(ra.supports[k], rb.supports[k])
        assert np.array_equal(a.w.view(np.uint32), b.w.view(np.uint32))
        assert np.array_equal(a.e.view(np.uint32), b.e.view(np.uint32))


def test_alg4_is_gmc_scaled_under_constant_eta():
    """The appendix: with a constant learning rate Alg. 4 is Alg. 1, its
    residual being eta times GMC's. Same supports, e4 = eta e1 and w4 = w1 up
    to fp32 rounding."""
    rng = np.random.default_rng(25)
    d, K, T, eta = 800, 4, 12, 0.25
    a = GMC(d, K, beta=0.9, eta=eta, compressor=TOPK, ratio=0.02)
    b = GMC(d, K, beta=0.9, eta=eta, compressor=TOPK, ratio=0.02, variant=oracle.ALG4)
    w0 = rng.standard_normal(d).astype(np.float32)
    a.set_params(w0)
    b.set_params(w0)
    for g in _grads(rng, T, K, d):
        ra, rb = a.step(g), b.step(g)
        for k in range(K):
            np.testing.assert_array_equal(ra.supports[k], rb.supports[k])
        np.testing.assert_allclose(b.e, float(a.eta) * a.e.astype(np.float64), rtol=1e-4, atol=1e-6)
        np.testing.assert_allclose(b.w, a.w, rtol=1e-5, atol=1e-6)


# ---------------------------------------------------------------------------
# The local-momentum baseline (Sec. 2.3 eq. (3) with error feedback: DGC w/o
# and w/ momentum factor masking)
# ---------------------------------------------------------------------------

def test_local_momentum_without_compression_is_serial_msgd():
    """Sec. 2.3: local momentum without sparsification is serial MSGD (the
    heavy-ball recursion), with e = 0 exactly."""
    rng = np.random.default_rng(41)
    d, K, T, eta, beta = 129, 4, 40, 0.05, 0.9
    o = GMC(d, K, beta=beta, eta=eta, compressor=TOPK, ratio=1.0, variant=oracle.LOCAL)
    w0 = rng.standard_normal(d).astype(np.float32)
    o.set_params(w0)
    grads = _grads(rng, T, K, d)
    eta32, beta32 = float(np.float32(eta)), float(np.float32(beta))
    ref = _heavy_ball(w0.astype(np.float64), [g.astype(np.float64) for g in grads], eta32, beta32)
    m_abs = np.zeros((K, d))
    budget = np.zeros(d)
    for t, g in enumerate(grads):
        w_t = o.w.astype(np.float64)
        o.step(g)
        assert not np.any(o.e)
        m_abs = beta32 * m_abs + eta32 * np.abs(g.astype(np.float64))
        budget += 6 * U * (np.abs(o.w.astype(np.float64)) + np.abs(w_t) + (K + 3) / K * m_abs.sum(0))
        np.testing.assert_array_less(np.abs(o.w - ref[t + 1]), 2 * budget / (1 - beta32) + 1e-30)


def test_momentum_factor_masking_without_compression_is_sgd():
    """Sec. 3.1's remark: with momentum factor masking and no sparsification,
    every coordinate is sent each step, the momentum is reset, and the method
    is plain distributed SGD: w_{t+1} = w_t - eta * mean_k g_{t,k}."""
    rng = np.random.default_rng(42)
    d, K, T, eta = 257, 3, 20, 0.1
    o = GMC(d, K, beta=0.9, eta=eta, compressor=TOPK, ratio=1.0, variant=oracle.LOCAL_MFM)
    w0 = rng.standard_normal(d).astype(np.float32)
    o.set_params(w0)
    w_ref = w0.astype(np.float64)
    tol = np.zeros(d)
    eta32 = float(np.float32(eta))
    for g in _grads(rng, T, K, d):
        o.step(g)
        assert not np.any(o.e) and not np.any(o.u)
        g64 = g.astype(np.float64)
        w_ref = w_ref - eta32 / K * g64.sum(0)
        tol += (K + 3) * U * eta32 / K * np.abs(g64).sum(0) + 2 * U * np.abs(o.w)
        np.testing.assert_array_less(np.abs(o.w - w_ref), 2 * tol + 1e-30)


@pytest.mark.parametrize("variant", [oracle.LOCAL, oracle.LOCAL_MFM])
def test_local_momentum_update_rule(variant):
    """With C eliminated: w_{t+1} - w_t = -ebar_t - mbar_{t+1} + ebar_{t+1},
    and the momentum follows m_{t+1} = beta m_t + eta g off the sent
    coordinates (and is 0 on them with masking)."""
    rng = np.random.default_rng(43)
    d, K, T, eta, beta = 500, 4, 25, 0.1, 0.9
    o = GMC(d, K, beta=beta, eta=eta, compressor=TOPK, ratio=0.03, variant=variant)
    o.set_params(rng.standard_normal(d).astype(np.float32))
    eta32, beta32 = float(np.float32(eta)), float(np.float32(beta))
    for g in _grads(rng, T, K, d):
        w_t, e_t, m_t = (x.astype(np.float64) for x in (o.w, o.e, o.u))
        r = o.step(g)
        w_n, e_n, m_n = (x.astype(np.float64) for x in (o.w, o.e, o.u))
        m_new = beta32 * m_t + eta32 * g.astype(np.float64)
        sent = np.zeros((K, d), bool)
        for k in range(K):
            sent[k, r.supports[k]] = True
        mb = 4 * U * (beta32 * np.abs(m_t) + eta32 * np.abs(g))
        want = np.where(sent, 0.0, m_new) if variant == oracle.LOCAL_MFM else m_new
        np.testing.assert_array_less(np.abs(m_n - want), mb + 1e-30)
        lhs = w_n - w_t
        rhs = -e_t.mean(0) - m_new.mean(0) + e_n.mean(0)
        scale = (np.abs(e_t) + np.abs(m_new) + np.abs(r.e_half) + np.abs(e_n)).sum(0)
        budget = 8 * U * (np.abs(w_n) + np.abs(w_t) + (K + 3) / K * scale)
        np.testing.assert_array_less(np.abs(lhs - rhs), budget + 1e-30)


def test_local_momentum_at_beta_zero_is_alg4():
    """Bitwise: with beta = 0 the local momentum is eta g and the step is
    Alg. 4's (which then has no momentum term either)."""
    rng = np.random.default_rng(44)
    d, K = 400, 3
    a = GMC(d, K, beta=0.0, eta=0.3, compressor=TOPK, ratio=0.05, variant=oracle.ALG4)
    b = GMC(d, K, beta=0.0, eta=0.3, compressor=TOPK, ratio=0.05, variant=oracle.LOCAL)
    w0 = rng.standard_normal(d).astype(np.float32)
    a.set_params(w0)
    b.set_params(w0)
    for g in _grads(rng, 8, K, d):
        ra, rb = a.step(g), b.step(g)
        for k in range(K):
            np.testing.assert_array_equal(ra.supports[k], rb.supports[k])
        assert np.array_equal(a.w.view(np.uint32), b.w.view(np.uint32))
        assert np.array_equal(a.e.view(np.uint32), b.e.view(np.uint32))


def test_variants_refuse_gmcplus_and_rbgs():
    with pytest.raises(ValueError):
        GMC(10, 2, 0.9, 0.1, compressor=RBGS, block=2, variant=oracle.ALG3)
    with pytest.raises(ValueError):
        GMC(10, 2, 0.9, 0.1, lam=0.5, variant=oracle.ALG4)


# ---------------------------------------------------------------------------
# Approximate top-s (Sec. 5.1): sample, threshold, selection
# ---------------------------------------------------------------------------

def test_approx_sizes():
    """|S| is about d/100 in runs of 8 (|S| = 8 floor(d/800)); r = ratio |S|,
    |S|/1024 at the paper's ratio s/d = 1/1024 (Sec. 5.1)."""
    d = 102_400 * 13
    n = oracle.approx_sample_size(d)
    assert n == 8 * (d // 800) == 13_312
    assert abs(n - d / 100) <= 8
    assert oracle.approx_rank(n, 1 / 1024) == 13
    assert oracle.approx_sample_size(799) == 8 and oracle.approx_sample_size(5) == 5
    assert oracle.approx_rank(8, 1 / 1024) == 1
    assert oracle.approx_limit(138_357_544, 0.001) == 4 * 138_357 + 4096
    assert oracle.approx_limit(1000, 0.001) == 1000


def test_approx_sample_positions_from_the_generator():
    """One run of 8 per stratum, starting on a multiple of 8 at the offset the
    published generator's outputs give (the stream's draws are SplitMix64
    outputs from its key)."""
    for d, seed, t in ((1000, 0, 0), (1_000_003, 99, 7), (8_000, 5, 3), (15, 0, 1), (805, 2, 2)):
        pos = oracle.approx_sample_positions(seed, t, d)
        n = oracle.approx_runs(d)
        key = oracle.rbgs_stream_key(seed, t, 0)
        draws = oracle.splitmix64_sequence(key, n)
        assert pos.size == oracle.approx_sample_size(d) == 8 * n
        for i in range(n):
            lo, hi = i * d // n, (i + 1) * d // n
            run = pos[8 * i: 8 * i + 8]
            a = -(-lo // 8) * 8
            m = (hi - a) // 8
            assert m >= 1 and run[0] % 8 == 0 and lo <= run[0] and run[-1] < hi
            assert run[0] == a + 8 * (((draws[i] >> 32) * m) >> 32)
            np.testing.assert_array_equal(run, np.arange(run[0], run[0] + 8))
    np.testing.assert_array_equal(oracle.approx_sample_positions(3, 0, 5), np.arange(5))
    a = oracle.approx_sample_positions(1, 0, 100_000)
    assert not np.array_equal(a, oracle.approx_sample_positions(1, 1, 100_000))
    assert not np.array_equal(a, oracle.approx_sample_positions(2, 0, 100_000))


def test_approx_sample_offsets_uniform():
    """The run's slot inside a stratum of 100 slots is uniform (chi-square
    over 100 cells)."""
    counts = np.zeros(100, np.int64)
    d = 800 * 4000
    for t in range(5):
        pos = oracle.approx_sample_positions(31, t, d)[::8]
        np.add.at(counts, (pos - np.arange(pos.size) * 800) // 8, 1)
    expected = counts.sum() / 100
    chi2 = float(((counts - expected) ** 2 / expected).sum())
    assert chi2 < 180.0  # 99 degrees of freedom; p < 1e-5 beyond this


def _brute_approx(x, sample, r, limit):
    mags = sorted((abs(float(x[p])) for p in sample), reverse=True)
    theta = mags[r - 1]
    sup = [j for j in range(x.size) if abs(float(x[j])) >= theta]
    if len(sup) > limit:
        sup = sorted(sorted(range(x.size), key=lambda j: (-abs(float(x[j])), j))[:limit])
    return np.array(sup, np.int64)


def test_approx_brute_force():
    """Theta and the support against a plain loop over |x| (ties, signed
    zeros and the exact top-M beyond the limit included)."""
    rng = np.random.default_rng(12)
    for case, (x, _) in enumerate(_tiny_inputs(rng, 3_000)):
        d = x.size
        n = int(rng.integers(1, d + 1))
        sample = np.sort(rng.choice(d, size=n, replace=False))
        r = int(rng.integers(1, n + 1))
        limit = int(rng.integers(1, d + 1)) if case % 3 == 0 else d
        got, theta = oracle.approx_top_s_support(x, sample, r, limit)
        np.testing.assert_array_equal(got, _brute_approx(x, sample, r, limit))
        mags = sorted((abs(float(x[p])) for p in sample), reverse=True)
        assert abs(float(np.array([theta], np.uint32).view(np.float32)[0])) == mags[r - 1]


def test_approx_threshold_properties():
    """A threshold set: everything sent is at least as large as everything
    kept back, and at least r sampled components are sent (below the limit)."""
    rng = np.random.default_rng(13)
    for _ in range(200):
        d = int(rng.integers(200, 5000))
        x = (rng.standard_normal(d) * np.exp(rng.uniform(-3, 3, d))).astype(np.float32)
        n = oracle.approx_sample_size(d)
        r = oracle.approx_rank(n, 0.05)
        sample = oracle.approx_sample_positions(int(rng.integers(0, 2 ** 63)), 0, d)
        S, _ = oracle.approx_top_s_support(x, sample, r, d)
        keep = np.zeros(d, bool)
        keep[S] = True
        a = np.abs(x.astype(np.float64))
        if not keep.all():
            assert a[keep].min() >= a[~keep].max()
        assert np.count_nonzero(keep[sample]) >= r


def test_approx_count_near_ratio():
    """On Gaussian data the number sent is ratio*d up to the sample's spread
    (about 1/sqrt(r)): within 40% per draw, within 8% on average."""
    rng = np.random.default_rng(14)
    d, ratio = 1 << 20, 0.01
    n = oracle.approx_sample_size(d)
    r = oracle.approx_rank(n, ratio)
    assert r == 104
    rel = []
    for t in range(20):
        x = rng.standard_normal(d).astype(np.float32)
        S, _ = oracle.approx_top_s_support(x, oracle.approx_sample_positions(3, t, d), r, d)
        rel.append(S.size / (ratio * d))
    assert all(0.6 < q < 1.4 for q in rel)
    assert abs(np.mean(rel) - 1.0) < 0.08


def test_approx_limit_takes_exact_top():
    """All-zero accumulators: theta is the zero key, every component reaches
    it, and the limit leaves the M lowest indices (ties to the lower index)."""
    d, K = 20_000, 2
    o = GMC(d, K, beta=0.0, eta=0.1, compressor=TOPK_APPROX, ratio=0.001)
    assert o.limit == 4 * 20 + 4096
    o.set_params(np.zeros(d, np.float32))
    r = o.step(np.zeros((K, d), np.float32))
    for k in range(K):
        np.testing.assert_array_equal(r.supports[k], np.arange(o.limit))
        assert r.thresholds[k] == 0
    assert r.stats["pairs"] == K * o.limit and r.stats["nnz"] == 0


# ---------------------------------------------------------------------------
# P9: the two-worker quadratic of Sec. 3.2 (qualitative; parity unpinned)
# ---------------------------------------------------------------------------

def test_p9_toy_quadratic_converges():
    cfg = _golden("toy_quadratic.json")
    d, K = cfg["d"], cfg["K"]
    i = np.arange(d)
    wgt = (d - i).astype(np.float64)
    o = GMC(d, K, beta=cfg["beta"], eta=cfg["eta"], compressor=TOPK, ratio=cfg["s_fraction"])
    o.set_params(np.array(cfg["start"], np.float32))
    dist = []
    for _ in range(3000):
        w = o.w.astype(np.float64)
        g = np.stack([2 * wgt * (w - (i + 1)), 2 * wgt * (w + (i + 1))]).astype(np.float32)
        o.step(g)
        dist.append(float(np.linalg.norm(o.w)))
    d0 = float(np.linalg.norm(cfg["start"]))
    assert dist[500] < 1e-3 * d0
    assert max(dist[-1000:]) < 1e-4 * d0


def _toy_distances(variant, d, s_fraction, start, steps=3000):
    """Distances to the optimum w* = 0 of the two-worker quadratic of Sec. 3.2
    (beta = 0.9, eta = 0.005, top-s), for one form of the step."""
    i = np.arange(d)
    wgt = (d - i).astype(np.float64)
    o = GMC(d, 2, beta=0.9, eta=0.005, compressor=TOPK, ratio=s_fraction, variant=variant)
    o.set_params(np.array(start, np.float32))
    dist = []
    for _ in range(steps):
        w = o.w.astype(np.float64)
        o.step(np.stack([2 * wgt * (w - (i + 1)), 2 * wgt * (w + (i + 1))]).astype(np.float32))
        dist.append(float(np.linalg.norm(o.w.astype(np.float64))))
    return np.array(dist)


def test_p9b_toy_global_beats_local_momentum():
    """Sec. 3.2, Figs. 1 and 2 (qualitative; parity unpinned: the figures carry
    no numbers): GMC ends closer to the optimum than the local-momentum method
    without masking, masking slows convergence down (d = 2, s = 0.5 d), and
    for d = 20 GMC stays nearer the optimum than both local-momentum methods
    at s = 0.1 d, 0.5 d and 0.8 d. The d = 20 start is not given in the paper;
    this test reads it as 20 points evenly spaced from -1 to 2."""
    cfg = _golden("toy_quadratic.json")
    gmc = _toy_distances(oracle.ALG1, 2, 0.5, cfg["start"])
    local = _toy_distances(oracle.LOCAL, 2, 0.5, cfg["start"])
    mfm = _toy_distances(oracle.LOCAL_MFM, 2, 0.5, cfg["start"])
    assert gmc[-1] < local[-1]
    assert mfm[300] > gmc[300] and mfm[300] > local[300]
    start = list(np.linspace(-1.0, 2.0, 20))
    for s in (0.1, 0.5, 0.8):
        tail = {v: _toy_distances(v, 20, s, start)[-1000:].mean()
                for v in (oracle.ALG1, oracle.LOCAL, oracle.LOCAL_MFM)}
        assert tail[oracle.ALG1] < tail[oracle.LOCAL] and tail[oracle.ALG1] < tail[oracle.LOCAL_MFM], (s, tail)


# ---------------------------------------------------------------------------
# The appendix's comparison of Alg. 4 with GMC under a decaying learning rate
# ---------------------------------------------------------------------------

def _cosine_etas(eta0, T):
    """Sec. 5.1's cosine annealing without restarts, per step:
    eta_t = eta0 * 0.5 * (1 + cos(t pi / (T + 1))), each rounded to fp32."""
    return [float(np.float32(eta0 * 0.5 * (1.0 + math.cos(t * math.pi / (T + 1))))) for t in range(T)]


def _top_s_64(x, s):
    """Top-s of a float64 vector: largest |x|, ties to the lower index, ascending."""
    order = np.lexsort((np.arange(x.size), -np.abs(x)))
    return np.sort(order[:s])


def _toy_grads(w, d):
    """The two workers' gradients of Sec. 3.2's quadratic at w (optimum 0)."""
    i = np.arange(d)
    wgt = (d - i).astype(np.float64)
    return np.stack([2 * wgt * (w - (i + 1)), 2 * wgt * (w + (i + 1))]).astype(np.float32)


@pytest.mark.parametrize("variant", [oracle.ALG1, oracle.ALG4])
@pytest.mark.parametrize("problem", ["gaussian", "toy_quadratic"])
def test_appendix_rewriting_under_decaying_eta(variant, problem):
    """The appendix ("Other Ways for Combining Momentum and Error Feedback")
    writes both forms with one scaled accumulator, under a learning rate eta_t:
        a_{t,k} = r_{t,k} + eta_t g_{t,k} - beta (w_t - w_{t-1}),
        w_{t+1} = w_t - (1/K) sum_k C(a_{t,k}),
        r_{t+1,k} = rho_{t+1} (a_{t,k} - C(a_{t,k})),
    where r is eta_t e_t for GMC (the residual rescaled, rho_{t+1} =
    eta_{t+1}/eta_t) and Alg. 4's own residual (rho = 1): Alg. 4's residual
    enters the next step with the larger coefficient, since eta_t does not
    increase. Checked in float64 on the fp32 oracle's own state at every step
    of Sec. 5.1's cosine schedule: the oracle sends top-s of a (compressors
    are scale-invariant, C(eta x) = eta C(x)), its update is -(1/K) sum C(a),
    and the residual it carries is rho (a - C(a)) with rho as stated; the
    factor changes by up to a few per cent a step here, far above rounding."""
    rng = np.random.default_rng(61)
    if problem == "gaussian":
        d, K, ratio, eta0, T = 2000, 4, 0.01, 0.1, 40
    else:
        d, K, ratio, eta0, T = 20, 2, 0.1, 0.005, 60
    beta = 0.9
    s = oracle.topk_count(d, ratio)
    o = GMC(d, K, beta=beta, eta=eta0, compressor=TOPK, ratio=ratio, variant=variant)
    o.set_params((rng.standard_normal(d) if problem == "gaussian"
                  else np.linspace(-1.0, 2.0, d)).astype(np.float32))
    etas = _cosine_etas(eta0, T)
    b32 = float(np.float32(beta))
    carry = None  # a_{t-1} - C(a_{t-1}), float64
    w_prev = o.w.astype(np.float64)
    for t, eta_t in enumerate(etas):
        o.set_eta(eta_t)
        w_t, e_t = o.w.astype(np.float64), o.e.astype(np.float64)
        r_t = eta_t * e_t if variant == oracle.ALG1 else e_t  # the scaled residual
        if carry is not None:
            rho = eta_t / etas[t - 1] if variant == oracle.ALG1 else 1.0
            if variant == oracle.ALG1:
                assert rho < 1.0 - 1e-3 or t < 3
            # the oracle formed a_{t-1} in fp32 (three roundings, c = fl(beta/eta)):
            # a budget on the size of its terms, as in P5
            np.testing.assert_array_less(np.abs(r_t - rho * carry), 8 * U * rho * carry_mag + 1e-30)
        g = (_grads(rng, 1, K, d)[0] if problem == "gaussian" else _toy_grads(w_t, d))
        a = r_t + eta_t * g.astype(np.float64) - b32 * (w_t - w_prev)
        r = o.step(g)
        C = np.zeros_like(a)
        for k in range(K):
            np.testing.assert_array_equal(r.supports[k], _top_s_64(a[k], s))
            C[k, r.supports[k]] = a[k, r.supports[k]]
        step = o.w.astype(np.float64) - w_t
        budget = 8 * U * (np.abs(o.w) + np.abs(w_t) + np.abs(a).sum(0) / K * (K + 3))
        np.testing.assert_array_less(np.abs(step + C.sum(0) / K), budget + 1e-30)
        carry = a - C
        carry_mag = np.abs(r_t) + eta_t * np.abs(g.astype(np.float64)) + b32 * np.abs(w_t - w_prev)
        w_prev = w_t
