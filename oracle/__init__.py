"""CPU oracle for the gs-SGD gradient-compression step (test infrastructure only).

This package is a plain, slow, obviously-correct restatement of what the GPU library
computes, written from the paper (global-sketching SGD, arXiv 2108.06004) and kept
independent of the CUDA path: it shares no code, headers, tables or helpers with
``paper_2108_06004_gb300`` and never imports it.  Only ``tests/``, the ``smoke()`` check
in ``__graft_entry__`` and the CPU-baseline leg of ``bench.py`` may import it; the product
path never routes through it.

Arithmetic conventions
  * momentum / error accumulators follow fp32 round-to-nearest semantics exactly (each
    operation is done in fp64 and rounded once to fp32, which equals the IEEE fp32
    result of that single operation);
  * sketch cells, the tree merge, the median estimate and the gathered values are fp64;
  * hash buckets and signs are exact integers (Python big ints are the ground truth, a
    numpy limb-split evaluation is the fast path and is checked against them).

Modules
  ``countsketch``  hash family h_j / s_j and the seeded coefficient derivation.
  ``gssgd``        accumulate, sketch, tree merge, median query, top-k, gather-and-zero,
                   and one full step (Alg. 1 steps 5-24 with Alg. 2).

Parity status: every function here is pinned by a CPU test against a property fixed by
the paper or by mathematics (see ``tests/test_oracle_pins.py``); the paper prints no
worked numeric example, so no absolute end-to-end value is pinned by the paper itself.
"""

from .countsketch import (  # noqa: F401
    MERSENNE_P,
    splitmix64,
    derive_coefficients,
    bucket_exact,
    sign_exact,
    hash_rows,
    splitmix64_at,
)
from .gssgd import (  # noqa: F401
    accumulate,
    sketch,
    merge_schedule,
    merge_tree,
    query,
    cell_band,
    topk,
    topk_by_threshold,
    heavymix,
    heavymix_select,
    heavymix_members,
    heavymix_select_from,
    gather_and_zero,
    apply_update,
    query_at,
    sketch_sparse,
    sketched_state_step,
    SketchedStateResult,
    step,
    StepResult,
)
