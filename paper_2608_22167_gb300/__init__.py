"""GB300-native (sm_103a) paged-attention hot path of the MCP-Universe RL
rollout step: KV append and causal / sliding-window attention over ragged,
paged bf16 KV caches with split-KV decode, a shared-prefix cascade pass for
GRPO groups and a tensor-core append-chunk kernel.

The C ABI is include/mcpu.h; ``paper_2608_22167_gb300.mcpu`` is its ctypes
binding (importing it loads libmcpu.so and fails loudly if it is missing).
"""

__all__ = ["mcpu", "build"]
