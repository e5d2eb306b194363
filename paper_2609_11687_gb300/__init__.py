"""GB300-native Kashin-DCT decomposition and 2-bit coding.

``paper_2609_11687_gb300.kashin`` binds the C-ABI library ``libkashin.so`` built
from ``csrc/`` (hand-written sm_103a CUDA).  Importing this package does not load
the library; importing ``.kashin`` does, and fails loudly if it is missing.
``paper_2609_11687_gb300.synth`` draws the seeded synthetic weight matrices.
"""
