"""GB300-native INT8 encoder-decoder translation path (MobileNMT, arXiv 2306.04235).

The compute path is the C-ABI library ``libmnmt.so`` (hand-written sm_103a
CUDA); :mod:`paper_2306_04235_gb300.mnmt` is its thin ctypes binding and
:mod:`paper_2306_04235_gb300.synth` the seeded synthetic-input generator.
Importing the package itself loads nothing.
"""
