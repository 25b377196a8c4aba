"""gmc_topk_noalloc against the regular top-k path and the oracle.

Some callers cannot allocate device memory: for example code whose device
memory is all owned by another allocator, such as a framework's caching pool
or a serving process with a fixed memory budget. gmc_topk_noalloc gives them
the library's top-k compressor with its scratch in a fixed array inside the
library, so neither the library nor the caller allocates anything per call.

These tests call it through the C ABI. The first checks it against the
regular entry point (gmc_step of a handle with one worker, beta = 0 and a zero
state, whose accumulator is then exactly the input vector) on two calls in a
row with different inputs and sizes, so the second call also shows that the
shared scratch is reset between calls. The others check it against the
oracle's top-s (Sec. 4: the s largest magnitudes, ties to the lower index),
indices exactly and values bitwise, on the cases where the tie handling and
the tile scan are most exposed: a tie group that straddles the k-th value
over many tiles, all-equal and all-zero (+0 and -0) vectors, k = n, n = 1,
n below one tile, non-finite values, and the largest n the scratch takes.

This file is collected last (pytest orders files by name), so a run that
stops at the first failure has run every other test before it.
"""
import numpy as np
import pytest

import oracle
from parity_util import ATOL, RTOL, bits

pytestmark = pytest.mark.gpu

GMC_EINVAL, GMC_ETOOBIG = 1, 7
MAX_N = 1 << 26


def _regular_topk(x, k):
    """Top-k of x through gmc_step + gmc_get_selected (the existing path)."""
    import torch
    from paper_1905_12948_gb300 import GMC
    n = x.numel()
    ratio = (k + 0.5) / n  # k = floor(ratio * n)
    h = GMC(n, 1, beta=0.0, eta=1.0, compressor="topk", ratio=ratio, device=x.device)
    h.set_params(torch.zeros(n, dtype=torch.float32, device=x.device))
    h.step(x.view(1, n))
    idx, val = h.selected(0)
    assert h.check() == 0
    h.close()
    return idx.cpu().numpy(), val.cpu().numpy()


def _noalloc_topk(x, k):
    import torch
    from paper_1905_12948_gb300 import gmc
    lib = gmc.load()
    n = x.numel()
    idx = torch.full((k,), -1, dtype=torch.int32, device=x.device)
    val = torch.empty(k, dtype=torch.float32, device=x.device)
    stream = torch.cuda.current_stream().cuda_stream
    st = lib.gmc_topk_noalloc(x.data_ptr(), n, k, idx.data_ptr(), val.data_ptr(), stream)
    assert st == 0, lib.gmc_strerror(st)
    torch.cuda.synchronize()
    return idx.cpu().numpy().astype(np.int64), val.cpu().numpy()


def _check_against_oracle(x_np, k):
    import torch
    x = torch.from_numpy(x_np).cuda()
    got_idx, got_val = _noalloc_topk(x, k)
    want = oracle.top_s_support(x_np, k)
    assert np.array_equal(got_idx, want), (
        f"indices differ: {np.setdiff1d(got_idx, want)[:5]} vs {np.setdiff1d(want, got_idx)[:5]}")
    assert np.array_equal(bits(got_val), bits(x_np[want])), "values differ bitwise"


def _heavy(rng, n):
    return (rng.standard_normal(n) * np.exp(rng.uniform(-4, 0, size=n))).astype(np.float32)


def test_noalloc_topk_matches_regular_path_twice():
    import torch
    rng = np.random.default_rng(2024)
    dev = torch.device("cuda")
    cases = [(1_000_003, 1_000), (70_001, 700)]
    for n, k in cases:  # two calls in a row
        x_np = _heavy(rng, n)
        x_np[rng.integers(0, n, size=50)] = 0.5  # equal values across tiles
        x = torch.from_numpy(x_np).to(dev)
        want_idx, want_val = _regular_topk(x, k)
        got_idx, got_val = _noalloc_topk(x, k)
        np.testing.assert_array_equal(got_idx, want_idx)
        np.testing.assert_allclose(got_val, want_val, rtol=RTOL, atol=ATOL)
        assert np.array_equal(bits(got_val), bits(want_val))
        assert np.array_equal(got_idx, oracle.top_s_support(x_np, k))


def _tie_group(rng, n, k, above, ties):
    """`above` components at +-9 (all kept) and `ties` at +-7 over many tiles,
    above every other magnitude: the k-th key is 7's, and k - above of the
    ties are kept, the lowest indices first."""
    x = _heavy(rng, n)
    pos = rng.choice(n, size=above + ties, replace=False)
    sign = np.where(rng.random(above + ties) < 0.5, -1.0, 1.0).astype(np.float32)
    x[pos[:above]] = 9.0 * sign[:above]
    x[pos[above:]] = 7.0 * sign[above:]
    return x


CASES = {
    "tie_group_straddles_T": lambda rng: (_tie_group(rng, 1_000_003, 1_000, 0, 3_000), 1_000),
    "ties_below_kept_values": lambda rng: (_tie_group(rng, 2_000_001, 1_000, 500, 3_000), 1_000),
    "all_equal": lambda rng: (np.full(10_000, 0.25, np.float32), 3_000),
    "all_zero_signed": lambda rng: (np.where(rng.random(5_000) < 0.5, -0.0, 0.0).astype(np.float32), 4_999),
    "k_equals_n": lambda rng: (_heavy(rng, 70_001), 70_001),
    "n_is_1": lambda rng: (np.array([-3.5], np.float32), 1),
    "below_one_tile": lambda rng: (_heavy(rng, 1_000), 10),
    "one_tile_plus_one": lambda rng: (_heavy(rng, 4_097), 4_097 // 2),
    "non_finite": lambda rng: (np.concatenate([_heavy(rng, 100_000),
                                               np.array([np.inf, -np.inf, np.nan], np.float32)]), 5),
}


@pytest.mark.parametrize("case", list(CASES))
def test_noalloc_edge_cases_match_the_oracle(case):
    rng = np.random.default_rng(sum(map(ord, case)))
    x_np, k = CASES[case](rng)
    _check_against_oracle(np.ascontiguousarray(x_np, np.float32), k)


@pytest.mark.parametrize("n", [MAX_N - 1, MAX_N])
def test_noalloc_largest_sizes(n):
    rng = np.random.default_rng(n)
    x_np = rng.standard_normal(n, dtype=np.float32)
    x_np[rng.integers(0, n, size=20_000)] = 3.0  # a tie group over the whole range
    k = int(np.count_nonzero(np.abs(x_np) > 3.0)) + 10_000  # the k-th value falls inside it
    _check_against_oracle(x_np, k)


def test_noalloc_rejects_sizes_above_its_scratch():
    import torch
    from paper_1905_12948_gb300 import gmc
    lib = gmc.load()
    x = torch.zeros(4, dtype=torch.float32, device="cuda")
    out_i = torch.empty(4, dtype=torch.int32, device="cuda")
    out_v = torch.empty(4, dtype=torch.float32, device="cuda")
    assert lib.gmc_topk_noalloc(x.data_ptr(), MAX_N + 1, 4, out_i.data_ptr(),
                                out_v.data_ptr(), None) == GMC_ETOOBIG
    assert lib.gmc_topk_noalloc(x.data_ptr(), 4, 5, out_i.data_ptr(), out_v.data_ptr(), None) == GMC_EINVAL
    assert lib.gmc_topk_noalloc(x.data_ptr(), 4, 0, out_i.data_ptr(), out_v.data_ptr(), None) == GMC_EINVAL
    assert b"2^26" in lib.gmc_strerror(GMC_ETOOBIG)
