"""Plain CPU oracle of the Seer hot path (numpy, fp64).

TEST INFRASTRUCTURE ONLY.  Nothing in the product package imports this tree;
only ``tests/``, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` /
``--impl reference`` legs of ``bench.py`` may call it.  It shares no code,
constants or helpers with the CUDA path: it is a slow, obviously correct
restatement of what the paper defines, so a reader can check it by eye.

Every function cites the passage it follows (Seer, arXiv 2607.14557):

* Sec. 3.2 / Sec. 1 -- step-0 text-side MLP activation sparsity with an
  absolute near-zero threshold;
* Sec. 3.3 -- the SNR boundary criterion (jump / noise over a short look-ahead
  window, ``L* = i* + 1``);
* Sec. 3.4, Eqs. 3-4 -- batch max, static micro-buckets, padding waste ratio
  and the three execution paths;
* Sec. 3.5 -- device-side compaction (slice, repack, bucket-align, pad, mask);
* Sec. 3.1 Eq. 2 and Sec. 3.6 Eqs. 6-7, 9-10 -- bidirectional softmax
  attention over the retained multimodal context.

Parity status: every function here is pinned by ``tests/test_oracle_*.py``
(hand-derived fixtures under ``tests/golden/``, closed forms, invariants,
library routines of torch/numpy on special cases).  None is "parity unpinned".
"""
from .seer_oracle import *  # noqa: F401,F403
from .seer_oracle import __all__  # noqa: F401
