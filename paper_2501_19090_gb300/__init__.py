"""PIFA (Pivoting Factorization) layer forward pass for GB300 (sm_103a).

``paper_2501_19090_gb300.inputs`` draws seeded synthetic layers and activations.
``paper_2501_19090_gb300.pifa`` is the thin ctypes binding over the C-ABI library ``libpifa.so``
(built from ``csrc/`` by ``paper_2501_19090_gb300.build``); it loads the library on first use and
raises if the library is missing.
"""
