"""Event-factorized parallel decode attention for GB300 (sm_103a).

The compute path is the CUDA library ``libpad.so`` built from ``csrc/``; the
Python layer in ``binding`` only marshals arguments to its C ABI.
"""
