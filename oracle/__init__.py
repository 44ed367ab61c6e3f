"""CPU oracle (test infrastructure only).

Plain fp64 numpy restatement of the action expert's flow-matching denoise (`expert`) and of
the VLM's LLM prefill that produces the KV cache it attends over (`prefill`), and of the future
correction module with its Q-Former state compressor (`correction`). It is imported
only by the tests, by the smoke check and by the bench's CPU-baseline leg; the library and
its CUDA kernels never import it and share no code with it.
"""

from .expert import (  # noqa: F401
    sinusoidal_time_embedding, swish, time_conditioning, rms_modulate, rope, suffix_mask,
    attention, gelu_tanh, layer_mods, expert_forward, flow_times, denoise, denoise_batch,
    forward_batch, to_f64,
)
