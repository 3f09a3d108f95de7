"""GB300-native Residual Fallback Quantization (RFQ) linear layer.

The compute path lives in ``librfq.so`` (hand-written sm_103a CUDA behind a
C ABI, declared in ``include/rfq.h``); :mod:`.rfq` is its thin ctypes binding
and :mod:`.synth` generates seeded synthetic inputs.  Importing this package
loads nothing; the first call through :mod:`.rfq` loads the library and
raises if it has not been built.
"""
