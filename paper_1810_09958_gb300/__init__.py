"""GB300 (sm_103a) hot path of the ISA Mapper paper (Sotoudeh et al., SysML 2019):
tcgen05 GEMM, a persistent GRU forward and a fused separable depthwise
convolution behind the C ABI in include/isam.h.

``paper_1810_09958_gb300.isam`` is the binding; ``paper_1810_09958_gb300.synth``
draws the seeded synthetic inputs.  Importing the package loads nothing; the
library is loaded on first use and must have been built (``build.build()``).
"""
__all__ = ["isam", "synth", "build"]
