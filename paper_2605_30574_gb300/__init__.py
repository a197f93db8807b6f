"""GB300-native spliced decode attention (arxiv 2605.30574, §3 splice intervention).

Submodules are imported lazily: ``splice`` binds the CUDA library
``libsplice.so``; ``synth`` generates seeded inputs.
"""
