"""CommitKV CPU oracle — TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s cpu_baseline
and reference legs may import this package.  It shares no code, header,
table or helper with the CUDA library in ``paper_2608_07855_gb300``, and
the library never imports it.

Contents
  core   fp64 page/set deletion effects (explicit deletion and Eq. 6 closed
         form, in C), row statistics, the greedy joint test, lifecycle
         classification (Eq. 9-10), pending protection and retained-index
         selection (Eq. 12-13), the compaction gather (Eq. 4), and a
         per-token window-attention fill score (a reading: the paper
         defines no fill score).
  brute  an independent pure-Python brute force over every page subset for
         tiny problems, used to pin ``core``.

Parity status: the paper prints no worked numeric example.  Effect values
are pinned by exact identities (explicit deletion = Eq. 6), hand-derived
cases, invariants and brute force; the percentile convention, the pending
prefix rule and the fill rule are readings of silent passages and are
"parity unpinned" against the paper itself (they are pinned only against
hand tables written from those readings).
"""
from .core import (  # noqa: F401
    Problem,
    build,
    classify,
    effects,
    gather,
    greedy,
    page_effects,
    row_stats,
    select_indices,
    set_effect,
    token_scores,
    STATE_NONE,
    STATE_CANDIDATE,
    STATE_DORMANT,
    STATE_NEWLY_ACTIVE,
    STATE_STILL_ACTIVE,
    STATE_UNCERTAIN,
)
