"""Oracle for the MoARa-on-GaLore step: TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` import this package.  It shares no code with the CUDA library and
imports nothing from it.  ``moara_ref`` is the float64 NumPy oracle;
``brute`` is its loop-only twin for tiny inputs, used to pin it.
"""
