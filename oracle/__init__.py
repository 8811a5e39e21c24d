"""CPU oracle for the LLM-prefix hot path — TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline / reference arm
may import or run this package. The product path (``paper_2608_14586_gb300``) never imports
it, and it never imports the product path: the two share nothing but the seeded input
generator in ``synth/``.

What it computes: the plain definition of a contiguous range of LLaMA-style pre-norm decoder
blocks in float64, with inputs and weights taken exactly as their bf16 values. The paper
(Sec. IV-B, Eq. 5 and Eq. 6) treats each Transformer block as an indivisible unit and states
that splitting the ordered block list at a partition point p leaves the network function
unchanged: the GPU runs blocks 1..p and hands the boundary hidden state h^(p) to the
remaining blocks. The paper names the block's stages (normalisation, projection, attention,
feed-forward; Sec. IV-B) but not their formulas; the block is read as RMSNorm -> QKV
projection -> rotary embedding -> causal grouped-query attention with KV-cache write ->
output projection + residual -> RMSNorm -> SwiGLU MLP + residual.

Every function is pinned by tests in ``tests/test_oracle_pins.py`` against closed forms,
hand-worked examples (``tests/golden/``), invariants and brute force.
"""
from .decoder import (  # noqa: F401
    KVCache,
    LayerWeights,
    apply_rope,
    attention_weights,
    block_forward,
    block_forward_rows,
    boundary_bytes,
    boundary_transfer,
    bf16_to_f64,
    causal_gqa_attention,
    decode_step,
    prefix_forward,
    rms_norm,
    rope_cos_sin,
    silu,
    swiglu,
    to_bf16_bits,
)
