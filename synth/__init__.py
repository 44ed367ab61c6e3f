"""Seeded synthetic inputs for the action-expert denoise.

This package draws weights, prefix KV caches, robot states, action noise, correction items, the LLM
prefill's and the correction module's weights and inputs from a seeded
numpy PCG64 generator. It is shared by the CPU oracle and by the CUDA path's tests and bench,
and it holds none of the method's arithmetic: only shapes, draws and the bf16 rounding of the
drawn values (input preparation, so that both sides consume bit-identical numbers).
"""

from .inputs import (  # noqa: F401
    ExpertConfig,
    TINY,
    PI05,
    LAYER_WEIGHTS,
    GLOBAL_WEIGHTS,
    round_to_bf16,
    make_weights,
    make_requests,
    make_correction,
    weight_shapes,
)
from .correction import (  # noqa: F401
    PI05_CORRECTION,
    CorrectionConfig,
    correction_param_count,
    correction_weight_shapes,
    make_correction_inputs,
    make_correction_weights,
)
from .llm import (  # noqa: F401
    GEMMA2B,
    LLM_LAYER_WEIGHTS,
    LLMConfig,
    llm_weight_shapes,
    make_llm_weights,
    make_prefix_embeddings,
)
