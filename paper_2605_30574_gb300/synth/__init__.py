"""Seeded synthetic inputs for the spliced decode-attention workloads.

``workloads`` fixes the sweep shapes; ``host`` regenerates any input slice on
the CPU; ``device`` (ctypes over ``libsplice_synth.so``) fills whole device
stores with the same values.  This package holds none of the method's
arithmetic and is the only code shared by the CUDA path and the oracle.
"""
