"""GB300 (sm_103a) implementation of JARQ layer-wise refinement.

``paper_2609_38599_gb300.jarq`` is the Python binding of the C ABI declared in
``include/jarq.h``; ``paper_2609_38599_gb300.build`` compiles ``libjarq.so``.
Importing the binding loads the CUDA library and raises if it is missing.
"""
