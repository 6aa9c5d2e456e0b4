"""fp64 CPU oracle for the BGPO masked-diffusion ELBO hot path.

TEST INFRASTRUCTURE ONLY. This package is the slow, obviously correct statement
of what the GPU path computes. Only ``tests/``, ``__graft_entry__.smoke()`` and
the CPU-baseline / reference leg of ``bench.py`` may import it. The product
package ``paper_2510_11683_gb300`` never imports it, and it never imports the
product package: the two share no code, no constants and no helpers.

Modules
-------
philox       Philox4x64-10 counter-based generator (Salmon et al., SC'11).
bgpo_oracle  forward masking (Sec. 2.1), per-step ELBO term (Eq. 4), MC ELBO
             (Eq. 5), BGPO bound (Eq. 10, 13, 14), loss (Eq. 19 / Algorithm 1),
             analytic gradients, the VRPO objective (Eq. 7) used for the
             Equivalence pin (Sec. 3.2), and group advantages (Eq. 18).

Every function is pinned by ``tests/test_oracle_*.py`` against something other
than itself: published known-answer vectors, an independent library (numpy's
Philox, torch's log_softmax), brute-force enumeration of all masks, fp64 finite
differences, closed forms and the paper's inequalities. No function is
"parity unpinned".
"""
