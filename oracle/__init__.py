"""fp64 CPU oracle for the CyFA core operator -- TEST INFRASTRUCTURE ONLY.

This package is the slow, obviously-correct reference that the CUDA library
is checked against.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import it.
The product path (``paper_2609_36259_gb300``) never imports it, and it never
imports the product path: the two share no code.

Everything is float64 numpy, written from the paper (CyFA: Linear Sequence
Modeling with Relative-Time-Partitioned Memory):

* ``basis``      -- Phi, U(tau), P(tau), b, the Dirichlet shift kernel
                    (Sec. 3.1, App. A.1-A.2).
* ``gates``      -- clock / decay / write-strength activations and the
                    cumulative clock (Sec. 3.1, Sec. 3.4).
* ``forward``    -- four independent forward forms: relative-time recurrence
                    (Eq. cyfa-physical-recurrence), absolute-clock recurrence
                    (Eq. cyfa-absolute-recurrence / cyfa-absolute-readout),
                    the quadratic unrolled form (Prop. 3) and the chunk form
                    (App. B).
* ``backward``   -- reverse-mode gradient of the absolute-clock token
                    recurrence, with the clock gradient of Eq.
                    app-clock-gradient-accumulation.

Parity status of each function is stated in its module header; every
function is pinned by ``tests/test_oracle_*.py`` against closed forms,
special cases, the paper's printed objects or finite differences.
"""
