"""CPU oracle for ReSS (Residual-Restoring Sparse Attention).

TEST INFRASTRUCTURE ONLY.  Nothing in the product path imports, links or executes this
package: only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline / reference legs
may use it.  It shares no code with the CUDA library (paper_2609_35593_gb300); the two
meet only through the arrays made by the seeded generator in `synth`.

The oracle is a plain, slow restatement in float64 of what the paper defines, step by
step, in the paper's order and notation (see `ress_oracle` for the citations).  Every
function is pinned by tests/test_oracle_*.py against identities, closed forms, brute force
and library routines; the decision margins (which rows a comparison may excuse) are pinned
by rows whose keys and gains have closed forms worked out by hand.  The one quantity with
no external pin is named below.

parity unpinned: the absolute values of J on the synthetic inputs and the drift-vs-rounds
curve (the paper prints no worked example); only invariants pin them.
"""
from .ress_oracle import *  # noqa: F401,F403
