"""GB300-native (sm_103a) 4-bit weight-streaming GEMV for LLM decoding.

The hot path of token decoding of 4-bit quantized models (the workload of
Table 1 of the WebLLM paper): the fused dequantize-and-multiply of packed
int4 group-quantized weights against the activation vector(s), and the
per-token chain of those projections.  The compute lives in the CUDA library
``libwq4.so`` behind ``include/wq4.h``; ``wq4`` is its Python binding,
``model`` builds device-resident synthetic decoders, ``synth`` draws seeded
inputs.
"""
