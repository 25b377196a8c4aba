"""Pins of the C++ oracle (oracle/gmc_ref.cpp) against what the paper and the
mathematics fix, the same as the numpy oracle's (test_oracle_pins.py): the
reductions to distributed SGD and to heavy-ball momentum in float64 and the
closed form for a constant gradient, the exact split C(v) + e = v, top-s
against brute force on tiny inputs, the update rule with C eliminated and
Lemma 1 (Sec. 3.3), the GMC+ mean-iterate recursion (Sec. 4), lambda = 0,
and RBGS (published SplitMix64 outputs, Floyd's uniformity, block counts,
the paper's RCC). A last test runs both oracles -- two independent
statements of Alg. 1 / Alg. 2 -- on the same inputs and compares every
result bitwise.
"""
import math

import numpy as np
import pytest

import oracle
from oracle import cref
from test_oracle_pins import (U, _brute_top_s, _golden, _grads, _heavy_ball, _tiny_inputs,
                              _update_rule_residual)

TOPK, RBGS = "topk", "rbgs"


def CG(*a, **kw):
    kw.setdefault("keep_half", True)
    kw.setdefault("threads", 3)
    return cref.CGMC(*a, **kw)


def test_p1_sgd_reduction():
    rng = np.random.default_rng(1)
    d, K, T, eta = 257, 3, 20, 0.1
    o = CG(d, K, beta=0.0, eta=eta, compressor=TOPK, ratio=1.0)
    w0 = rng.standard_normal(d).astype(np.float32)
    o.set_params(w0)
    w_ref = w0.astype(np.float64)
    tol = np.zeros(d)
    eta32 = float(np.float32(eta))
    for g in _grads(rng, T, K, d):
        o.step(g)
        assert not np.any(o.e), "with no compression the residual must stay exactly 0"
        g64 = g.astype(np.float64)
        w_ref = w_ref - eta32 / K * g64.sum(0)
        tol += (K + 3) * U * eta32 / K * np.abs(g64).sum(0) + 2 * U * np.abs(o.w)
        np.testing.assert_array_less(np.abs(o.w - w_ref), 2 * tol + 1e-30)


@pytest.mark.parametrize("K", [1, 4])
def test_p2_heavy_ball_reduction(K):
    rng = np.random.default_rng(2 + K)
    d, T, eta, beta = 129, 40, 0.05, 0.9
    o = CG(d, K, beta=beta, eta=eta, compressor=TOPK, ratio=1.0)
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
    d, K, T, eta, beta = 5, 2, 50, 0.05, 0.9
    g = np.array([0.3, -1.2, 2.0, 0.0, 1e-3], np.float32)
    w0 = np.array([1.0, -2.0, 0.5, 3.0, 0.0], np.float32)
    o = CG(d, K, beta=beta, eta=eta, compressor=TOPK, ratio=1.0)
    o.set_params(w0)
    eta64, beta64 = float(np.float32(eta)), float(np.float32(beta))
    for t in range(1, T + 1):
        o.step(np.stack([g] * K))
        closed = w0 - eta64 * g / (1 - beta64) * (t - beta64 * (1 - beta64 ** t) / (1 - beta64))
        np.testing.assert_allclose(o.w, closed, rtol=2e-5, atol=2e-6)


@pytest.mark.parametrize("compressor,per_worker", [(TOPK, False), (RBGS, False), (RBGS, True)])
def test_p3_exact_split(compressor, per_worker):
    """Sent coordinates leave +0 and carry v; the others keep v: checked
    against v formed directly from the definition in numpy float32."""
    rng = np.random.default_rng(3)
    d, K, T = 1000, 4, 12
    o = CG(d, K, beta=0.9, eta=0.1, compressor=compressor, ratio=0.05, block=64, seed=5,
           per_worker=per_worker)
    o.set_params(rng.standard_normal(d).astype(np.float32))
    c = np.float32(np.float32(0.9) / np.float32(0.1))
    w_prev = o.w.copy()
    for g in _grads(rng, T, K, d):
        w_t, e_t = o.w.copy(), o.e.copy()
        v = (e_t + g) - c * (w_t - w_prev)
        r = o.step(g)
        for k in range(K):
            S = r.supports[k]
            sel = np.zeros(d, bool)
            sel[S] = True
            ebits = o.e[k].view(np.uint32)
            assert np.all(ebits[sel] == 0), "sent coordinates leave +0 behind"
            assert np.all(ebits[~sel] == v[k].view(np.uint32)[~sel]), "unsent coordinates keep v"
            assert np.all(r.values[k].view(np.uint32) == v[k].view(np.uint32)[S]), "C(v) carries v"
            np.testing.assert_array_equal(S, np.sort(S))
        w_prev = w_t


def test_p4_top_s_brute_force():
    rng = np.random.default_rng(4)
    for x, s in _tiny_inputs(rng, 10_000):
        np.testing.assert_array_equal(cref.top_s_support(x, s), _brute_top_s(x, s))


@pytest.mark.parametrize("compressor", [TOPK, RBGS])
def test_p5_update_rule(compressor):
    rng = np.random.default_rng(5)
    d, K, T = 600, 4, 30
    o = CG(d, K, beta=0.9, eta=0.1, compressor=compressor, ratio=0.05, block=16, seed=9)
    o.set_params(rng.standard_normal(d).astype(np.float32))
    for lhs, rhs, budget, *_ in _update_rule_residual(o, _grads(rng, T, K, d)):
        np.testing.assert_array_less(np.abs(lhs - rhs), budget + 1e-30)


@pytest.mark.parametrize("compressor", [TOPK, RBGS])
def test_p6_lemma1_z_sequence(compressor):
    rng = np.random.default_rng(6)
    d, K, T = 400, 3, 25
    o = CG(d, K, beta=0.9, eta=0.1, compressor=compressor, ratio=0.02, block=8, seed=3)
    o.set_params(rng.standard_normal(d).astype(np.float32))
    beta, eta = float(o.beta), float(o.eta)
    for lhs, rhs, budget, w_t, w_prev, e_t, e_n, g in _update_rule_residual(o, _grads(rng, T, K, d)):
        w_n = w_t + lhs
        z_t = w_t + beta / (1 - beta) * (w_t - w_prev) - eta / (1 - beta) * e_t.mean(0)
        z_n = w_n + beta / (1 - beta) * (w_n - w_t) - eta / (1 - beta) * e_n.mean(0)
        err = np.abs(z_n - (z_t - eta / (1 - beta) * g.mean(0)))
        np.testing.assert_array_less(err, 2 * budget / (1 - beta) + 1e-30)


@pytest.mark.parametrize("compressor", [RBGS, TOPK])
def test_p6b_gmcplus_mean_iterate(compressor):
    rng = np.random.default_rng(7)
    d, K, T, lam = 300, 4, 25, 0.5
    o = CG(d, K, beta=0.9, eta=0.1, compressor=compressor, ratio=0.05, block=10, lam=lam, seed=1)
    o.set_params(rng.standard_normal(d).astype(np.float32))
    beta, eta, lam = float(o.beta), float(o.eta), float(o.lam)

    def wbar():
        return np.mean([o.worker_params(k).astype(np.float64) for k in range(K)], axis=0)

    wb_prev = o.w.astype(np.float64)
    eb_prev = np.zeros(d)
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
    d, K, T = 200, 3, 10
    runs = []
    for lam in (0.0, 0.5):
        o = CG(d, K, beta=0.9, eta=0.1, compressor=RBGS, ratio=0.1, block=7, lam=lam, seed=2)
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


def test_p8_splitmix64_published_outputs():
    gold = _golden("splitmix64.json")
    for seed, key in ((0, "seed_0"), (1234567, "seed_1234567")):
        want = [int(h, 16) for h in gold[key]]
        assert cref.splitmix64_sequence(seed, len(want)) == want


def test_p8_floyd_uniform_over_subsets():
    nb, m, n = 6, 3, 20_000
    counts = {}
    for i in range(n):
        sub = tuple(cref.rbgs_blocks(12345, i, 0, nb, m))
        assert len(set(sub)) == m and list(sub) == sorted(sub)
        counts[sub] = counts.get(sub, 0) + 1
    assert len(counts) == math.comb(nb, m)
    expected = n / len(counts)
    assert sum((c - expected) ** 2 / expected for c in counts.values()) < 60.0


@pytest.mark.parametrize("per_worker", [False, True])
def test_p8_rbgs_counts(per_worker):
    rng = np.random.default_rng(9)
    d, K, B, ratio = 1000, 5, 64, 0.2     # nb = 16 (last block 40 long), m = 3
    o = CG(d, K, beta=0.9, eta=0.1, compressor=RBGS, ratio=ratio, block=B, seed=77,
           per_worker=per_worker)
    o.set_params(rng.standard_normal(d).astype(np.float32))
    for t in range(6):
        r = o.step(rng.standard_normal((K, d)).astype(np.float32))
        for k in range(K):
            blocks = np.unique(r.supports[k] // B)
            assert blocks.size == 3 and blocks.max() < 16
            size = sum(min((b + 1) * B, d) - b * B for b in blocks)
            assert r.supports[k].size == size
            np.testing.assert_array_equal(
                blocks, cref.rbgs_blocks(77, t, k + 1 if per_worker else 0, 16, 3))
        if not per_worker:
            for k in range(1, K):
                np.testing.assert_array_equal(r.supports[k], r.supports[0])
    if per_worker:
        assert any(not np.array_equal(r.supports[k], r.supports[0]) for k in range(1, K))


def test_p8_rbgs_rcc_matches_paper():
    gold = _golden("rcc_rbgs.json")
    d, K = 1024 * 37, 4
    B = d // 1024
    nb = -(-d // B)
    o = CG(d, K, beta=0.9, eta=0.1, compressor=RBGS, ratio=1.0 / nb, block=B, seed=4)
    rng = np.random.default_rng(10)
    o.set_params(rng.standard_normal(d).astype(np.float32))
    for _ in range(5):
        o.step((rng.standard_normal((K, d)) + 3.0).astype(np.float32))
    assert o.rcc() == pytest.approx(gold["rcc"], rel=0, abs=1e-15)


@pytest.mark.parametrize("compressor,per_worker,d,K,threads", [
    (TOPK, False, 100_003, 5, 2), (TOPK, False, 4_099, 16, 16), (RBGS, False, 100_003, 5, 3),
    (RBGS, True, 50_001, 7, 0)])
def test_both_oracles_agree_bitwise(compressor, per_worker, d, K, threads):
    """Two independent statements of Alg. 1 / Alg. 2, on the same inputs and
    with eta changed between steps: every selection, value, w, residual,
    detached point and counter equal bit for bit."""
    rng = np.random.default_rng(d + K)
    a = oracle.GMC(d, K, 0.9, 0.1, compressor=compressor, ratio=0.01, block=997, lam=0.5, seed=7,
                   per_worker=per_worker)
    b = cref.CGMC(d, K, 0.9, 0.1, compressor=compressor, ratio=0.01, block=997, lam=0.5, seed=7,
                  per_worker=per_worker, threads=threads)
    w0 = (rng.standard_normal(d) * 0.01).astype(np.float32)
    a.set_params(w0)
    b.set_params(w0)
    for t in range(6):
        if t == 3:
            a.set_eta(0.05)
            b.set_eta(0.05)
        g = (rng.standard_normal((K, d)) * 0.1).astype(np.float32)
        ra, rb = a.step(g), b.step(g)
        for k in range(K):
            np.testing.assert_array_equal(ra.supports[k], rb.supports[k])
            assert np.array_equal(ra.values[k].view(np.uint32), rb.values[k].view(np.uint32))
        assert np.array_equal(a.w.view(np.uint32), b.w.view(np.uint32))
        assert np.array_equal(a.e.view(np.uint32), b.e.view(np.uint32))
    for k in (0, K - 1):
        assert np.array_equal(a.worker_params(k).view(np.uint32), b.worker_params(k).view(np.uint32))
    assert a.totals == b.totals
    assert a.rcc() == b.rcc()
