"""GB300-native EmTrackMichelId hit identification (arXiv:2009.04509).

The compute path is the C-ABI library ``libemtk.so`` (hand-written sm_103a
CUDA); ``emtk`` is its thin ctypes binding.  ``synth`` draws the seeded
synthetic inputs.
"""
