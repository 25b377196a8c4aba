"""The deferred aggregation of the bulk top-k pass against the oracle.

With the bulk pass (d of a million and more) a step leaves the sum of its sent
pairs into w, and the zeroing of the senders' residuals, to the next step's
pass over the tiles; reading the state (w, a residual, the worker parameters,
the counters) applies it first. These tests run several steps in a row with
only the selections read in between, so each step applies the previous one's
aggregation inside its own pass and its sampled threshold sees it through the
sampled senders; then they compare w, every residual and the counters.
"""
import math

import numpy as np
import pytest

from parity_util import Pair

pytestmark = pytest.mark.gpu

D_BULK = 1_300_001  # above the bulk-pass size; odd, so rows start at every alignment


def _grads(rng, K, d):
    return (rng.standard_normal((K, d)) * np.exp(rng.uniform(-3, 0, size=d))).astype(np.float32)


def test_deferred_steps_in_a_row_with_eta_schedule():
    K, steps = 4, 6
    rng = np.random.default_rng(31)
    p = Pair(D_BULK, K, 0.9, 0.1, ratio=0.002, seed=4)
    for t in range(steps):
        eta = max(0.1 * 0.5 * (1 + math.cos(t * math.pi / steps)), 1e-3)  # Sec. 5.1 schedule
        p.gpu.set_eta(eta)  # between a step and the application of its aggregation
        p.ref.set_eta(eta)
        r = p.step(_grads(rng, K, D_BULK))
        p.compare(r, state=False)
    p.compare(r)  # applies the last aggregation, then w and every residual
    s = p.compare_stats()
    assert s["fallbacks"] == 0, "the sampled threshold must see the pending aggregation"
    assert p.gpu.check() == 0


def test_state_read_on_another_stream_between_deferred_steps():
    import torch
    K = 3
    rng = np.random.default_rng(32)
    p = Pair(D_BULK, K, 0.8, 0.05, ratio=0.003, seed=5)
    side = torch.cuda.Stream()
    for t in range(4):
        r = p.step(_grads(rng, K, D_BULK))
        p.compare(r, state=False)
        if t == 1:  # the aggregation is applied on `side`; the next step must wait for it
            with torch.cuda.stream(side):
                w = p.gpu.params(stream=side)
            side.synchronize()
            np.testing.assert_array_equal(w.cpu().numpy().view(np.uint32),
                                          p.ref.w.astype(np.float32).view(np.uint32))
    p.compare(r)
    p.compare_stats()


def test_deferred_steps_mixed_with_host_steps_and_detach():
    """gmc_step (deferred), gmc_step_host (applies its aggregation in the step
    and reports its counters), then GMC+ detached outputs switched on."""
    import torch
    K = 3
    rng = np.random.default_rng(33)
    p = Pair(D_BULK, K, 0.9, 0.1, ratio=0.002, seed=6)
    stats = torch.zeros(8, dtype=torch.int64).pin_memory()
    for t in range(3):
        r = p.step(_grads(rng, K, D_BULK))
        p.compare(r, state=False)
    g = _grads(rng, K, D_BULK)
    p.gpu.step_host(torch.from_numpy(g).pin_memory(), stats)
    r = p.ref.step(g)
    torch.cuda.synchronize()
    assert int(stats[3]) == r.stats["union"] and int(stats[4]) == r.stats["changed"]
    p.compare(r, state=False)
    out = torch.empty((K, D_BULK), dtype=torch.float32, device=p.dev)
    p.gpu.set_detach_output(out)
    for t in range(2):
        r = p.step(_grads(rng, K, D_BULK))
        torch.cuda.synchronize()
        for k in range(K):  # lambda = 0: w_{t+1,k} = w_{t+1}
            np.testing.assert_array_equal(out[k].cpu().numpy().view(np.uint32),
                                          p.ref.w.astype(np.float32).view(np.uint32))
        p.compare(r, state=False)
    p.compare(r)
    p.compare_stats()


@pytest.mark.parametrize("pinned", [True, False])
def test_host_steps_pinned_and_pageable(pinned):
    """gmc_step_host on the bulk pass: pinned (mapped) host gradients are read
    in place by the kernels, pageable ones copied to a staging buffer first.
    Several host steps in a row, then device steps, against the oracle."""
    import torch
    K = 5
    rng = np.random.default_rng(34 + pinned)
    p = Pair(D_BULK, K, 0.9, 0.1, ratio=0.003, seed=8)
    stats = torch.zeros(8, dtype=torch.int64).pin_memory()
    for t in range(3):
        g = _grads(rng, K, D_BULK)
        host = torch.from_numpy(g)
        if pinned:
            host = host.pin_memory()
        p.gpu.step_host(host, stats)
        r = p.ref.step(g)
        torch.cuda.synchronize()
        assert int(stats[1]) == r.stats["pairs"] and int(stats[2]) == r.stats["nnz"]
        assert int(stats[3]) == r.stats["union"] and int(stats[4]) == r.stats["changed"]
        p.compare(r, residuals=(t == 2))
    for t in range(2):
        r = p.step(_grads(rng, K, D_BULK))
        p.compare(r, state=(t == 1))
    p.compare_stats()
    assert p.gpu.stats()["fallbacks"] == 0
    assert p.gpu.check() == 0


def test_dense_sub_tiles_and_ties_on_the_bulk_pass():
    """Many sent pairs per 512-coordinate sub-tile (more than one per lane:
    the per-element sender masks), K = 1, an odd K and K = 12, ties across
    tiles, deferred and host (applied at once) steps alternating."""
    import torch
    for K, ratio in ((1, 0.05), (7, 0.02), (12, 0.01)):
        rng = np.random.default_rng(40 + K)
        p = Pair(D_BULK, K, 0.9, 0.1, ratio=ratio, seed=9)
        stats = torch.zeros(8, dtype=torch.int64).pin_memory()
        for t in range(4):
            g = _grads(rng, K, D_BULK)
            g[:, rng.integers(0, D_BULK, size=4000)] = np.float32(0.75)  # ties across tiles
            if t % 2:
                p.gpu.step_host(torch.from_numpy(g).pin_memory(), stats)
                r = p.ref.step(g)
                torch.cuda.synchronize()
            else:
                r = p.step(g)
            p.compare(r, state=(t == 3))
        p.compare_stats()
        assert p.gpu.check() == 0
        p.gpu.close()


def test_bulk_pass_reports_non_finite_values():
    """NaN and Inf gradients on the bulk pass: the step completes, counts
    them, and gmc_check reports GMC_ENONFINITE."""
    import torch
    K = 2
    rng = np.random.default_rng(44)
    p = Pair(D_BULK, K, 0.9, 0.1, ratio=0.002, seed=10)
    g = _grads(rng, K, D_BULK)
    g[0, 12345] = np.nan
    g[1, 999_999] = np.inf
    p.gpu.step(torch.from_numpy(g).to(p.dev))
    torch.cuda.synchronize()
    assert p.gpu.stats()["nonfinite"] == 2
    assert p.gpu.check() == 4  # GMC_ENONFINITE


@pytest.mark.parametrize("K,tail", [(1, 1001), (2, 1001), (5, 1001), (6, 1001), (7, 1001), (16, 1001),
                                    (6, 3001)])
def test_claimed_tiles_and_odd_worker_counts(K, tail):
    """Several tiles per CTA beyond its fixed ones, so the bulk pass claims
    the rest from its tile counter; the worker-parity warp groups each read
    their own stages of the ring, in order, for every K (odd K gives the two
    groups different item counts per tile, K = 1 leaves one group without
    items). K <= 5 runs the three-tile pipeline of w_t - w_{t-1}, K >= 6 the
    one-tile pipeline with two tiles claimed ahead. The ragged last tile's
    last four sub-tiles lie past d (tail 1001) or hold its last 953
    coordinates (tail 3001)."""
    d = 152 * 4096 * 9 + tail  # about nine tiles per CTA
    rng = np.random.default_rng(40 + K)
    p = Pair(d, K, 0.9, 0.1, ratio=0.001, seed=9, ref="cpp")
    for t in range(3):
        r = p.step(_grads(rng, K, d))
        p.compare(r, state=False)
    p.compare(r)
    s = p.compare_stats()
    assert s["fallbacks"] == 0
    assert p.gpu.check() == 0
