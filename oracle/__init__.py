"""CPU oracle for the concurrent-GEMM hot path — TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py`` (its
``cpu_baseline`` leg and its ``--impl reference`` arm) may import anything
from this package.  The product package ``paper_2409_02227_gb300`` never
imports it, and the oracle imports nothing from the product package: the two
share no kernels, helpers, tables or constants.  Inputs reach both sides as
raw bf16 bit patterns made by the seeded generator module
``paper_2409_02227_gb300.workloads``, which holds no GEMM arithmetic.

Contents (each module cites the passage it follows):

* ``gemm``         — fp64 GEMM over bf16 inputs (Sec. 2.1.2), a plain C loop
                      nest in ``oracle_gemm.c`` behind ctypes, plus a pure
                      Python triple loop for tiny cases.
* ``schedule``     — brute-force makespan search over every way of running a
                      small GEMM set as consecutive concurrent groups: the
                      paper's "Oracle" configuration that always picks the
                      right concurrency degree, sequential included (Sec. 5.5).
* ``planner_ref``  — an independent restatement of the dynamic logic's table
                      lookup (bucketize, preferred CD, min(CD, available),
                      heterogeneous split; Sec. 4.3 and Sec. 6.7), used to check
                      the product planner byte for byte.

Parity status: ``gemm`` is pinned (identity, permutation, small-integer
closed forms, pure-Python triple loop, numpy float64); ``schedule`` is pinned
(Bell numbers, hand-solved tables, an independent subset DP);
``planner_ref`` is pinned by hand-solved special cases of the paper's rules.
"""
