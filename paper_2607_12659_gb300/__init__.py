"""GB300-native flow-matching denoise of a pi0.5-style action expert, with the parts of Jetson-PI
around it.

The computation lives in CUDA libraries built in-tree (``build``):
  ``libjpi.so``          the action expert (C-ABI ``include/jpi.h``, binding ``jpi``) and the
                         future correction module with its Q-Former compressor
                         (``include/jpi_corr.h``, binding ``corr``);
  ``libjpi_prefill.so``  the LLM prefill that fills the expert's KV store
                         (``include/jpi_prefill.h``, binding ``prefill``).
``scheduler`` is the host-side confidence-based scheduling of App. C Alg. 1 around them.
Nothing here computes the model on the CPU.
"""

__all__ = ["jpi", "corr", "prefill", "scheduler", "build"]
