"""CPU oracle for batched multi-draft speculative verification (arXiv 2410.18234).

TEST INFRASTRUCTURE ONLY.  This package is a plain, slow, fp64 restatement of
what the verification path computes, written from the paper and kept separate
from the CUDA path: the two share no code, no headers and no tables.  Only the
test suite, ``__graft_entry__.smoke()`` and ``bench.py`` (its ``cpu_baseline``
leg and its ``--impl reference`` arm) may import anything from here.  The
product path never routes through it.

Modules
-------
philox   Philox4x32-10 counter-based generator (Salmon et al., SC'11) and the
         draw layout shared in definition (not in code) with the device side.
verify   the token-level selection schemes and the walk along the draft tree
         (Section 3 Definition 1 and Theorem 1, Section 4, Appendix A
         Algorithm 1, Appendix "Variant of Truncated LP", Remark 4).
theory   brute-force linear programs and closed forms used as pins
         (Problem 1, Theorem 1, Theorem 2, Example 1, Theorem 3, Remark 2,
         the truncation bound of Section 4).
enum     exhaustive enumeration of selection rules over Omega^K (tiny
         vocabularies), used to pin the induced distribution p_I.
truncated  the truncated-alphabet scheme (Section 4) and top-k / top-p
         preprocessing (Section 5), with the enumerated law that pins it.
sorted_lp  the truncated LP with the sorted rule on Omega_2 (Section 4 Eq.
         heur, Algorithm 2, App. I): no device counterpart yet.
acceptance  analytic acceptance probability of each scheme on one row, and the
         optimum of Theorem 3 (K = 2; Remark 2's conjectured form for K > 2)
         for any vocabulary size.

Parity status: every function here is pinned by a ``-m "not gpu"`` test
(see tests/test_oracle_*.py) except the SpecTr-style sequential-rejection
baseline, whose definition is not printed in the paper: it is pinned only by
target preservation (exact enumeration), "parity unpinned" against SpecTr's
own publication.
"""
