"""fp64 CPU oracle of the ReSA decode-time attention path (arXiv 2506.04108).

TEST INFRASTRUCTURE ONLY: imported by ``tests/``, ``__graft_entry__.smoke()``
and the CPU-baseline leg of ``bench.py``; never by the library. It shares no
code with the CUDA path. Every function is pinned by ``tests/test_oracle.py``
against closed forms, brute force, library routines or hand-worked examples
(``tests/golden/``); no function is "parity unpinned".
"""
from .resa_oracle import *  # noqa: F401,F403
from .resa_oracle import (ResaParams, SequenceState, attend_positions, attend_prefix, block_positions, block_summaries,
                          dense_attention, gbsa_attention, memory_access_ratio, online_summary_update,
                          pooled_query, quest_scores, rectify_attention, rectify_step, select_blocks,
                          select_for_group, selection_budget, sparse_decode_step, split_combine_attention,
                          widen_bf16)
