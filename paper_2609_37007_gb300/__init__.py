"""GB300-native RVQ-position-aware speculative decoding of the MultiCodeDecoder
(arXiv 2609.37007).  The decoding path is the CUDA library libmcd.so (include/mcd.h);
`mcd` is its thin ctypes binding and `synth` draws synthetic workloads."""
from . import synth  # noqa: F401
