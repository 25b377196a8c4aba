"""Oracle for the GMC / GMC+ step -- test infrastructure only.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU baseline
(and its reference arm) may import this package. See ``gmc_oracle`` for what it
computes and which passages of the paper each part follows.
"""
from .gmc_oracle import (ALG1, ALG3, ALG4, GMC, LOCAL, LOCAL_MFM, RBGS, TOPK,  # noqa: F401
                         TOPK_APPROX,
                         approx_limit, approx_rank,
                         approx_runs,
                         approx_sample_positions, approx_sample_size, approx_top_s_support,
                         below, floyd_blocks, magnitude_key, rbgs_draw, rbgs_stream_key,
                         rbgs_support, splitmix64_mix, splitmix64_sequence, top_s_support,
                         topk_count)
