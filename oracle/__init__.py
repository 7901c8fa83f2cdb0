"""fp64 CPU oracle for the REAL-Q per-layer quantization sweep.

TEST INFRASTRUCTURE ONLY.  Nothing in the product path may import, call, link
or execute anything in this package: only the tests, ``__graft_entry__.smoke``
and the CPU-baseline leg of ``bench.py`` use it.  It shares no code with the
CUDA path (``paper_2609_00049_gb300``); the two meet only through the seeded
input generators in ``synth``.

Contents
--------
realq.py   the sweep in the paper's order and notation, fp64 throughout except
           where a floating-point value decides an integer (the int4 code and
           the zero point), which is taken in fp32 on both sides.
brute.c    exhaustive search over all int4 codes of a tiny layer (the
           brute-force pin of the quantizer + surrogate), built by build.py.
block.py   one synthetic decoder block in fp64 with its backward, the
           exact two-block sliding-window loss (Sec. 4.4) of any linear
           module of the block, and the final block's true KL at the LM head
           with the Fisher of Eq. (fisher_full), and Alg. 1's loop over the
           block's modules with those losses; imported as ``oracle.block``.
"""
from .realq import *  # noqa: F401,F403
