"""CPU oracle for acoustic-to-text KV eviction and retained-cache attention.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this package.  The CUDA library
never calls it, and it shares no code with the CUDA path: the two meet only
through the seeded inputs of ``synth``.

What it computes, in plain, slow Python/numpy (float64 for floating point):

* ``policy``     - the online eviction rule of Sec. 3.3, executed literally:
                   after a unit, while the resident count exceeds B, drop the
                   acoustic and structural states of the oldest unit outside
                   the W most recent units; transcript, response text and the
                   system prefix always stay; positions never change.
* ``layout``     - the paged layout contract of the library (two regions per
                   session, lowest-free page allocation), restated as lists so
                   page tables can be compared bit for bit.
* ``rope``       - rotate-half rotary embedding at the original positions.
* ``attention``  - exact softmax attention over the retained keys.
* ``cache``      - the above combined behind calls that mirror the library.

Readings of the paper that the oracle fixes (where the text is silent or
ambiguous) are listed in the module that applies each of them.

Parity pins: every function here is pinned by ``tests/test_oracle_*.py``
against brute force, closed forms, invariants and hand-worked examples.  One
part is "parity unpinned": nothing in the paper fixes the real per-unit token
counts beyond "about ten audio tokens" and "17 versus about three positions
per second", so the synthetic token counts are a workload choice, not a pin.
"""
