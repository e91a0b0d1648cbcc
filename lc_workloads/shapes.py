"""Parameter layouts of the synthetic workloads (Llama-style decoders).

The layer partition follows §2.2: embed_tokens, each transformer block, the
final normalization and lm_head are the layers, N = B + 3, and a tied
lm_head is the embedding itself (so N = B + 2).  Every projection matrix and
every RMSNorm vector is its own tensor.  With ``per_tensor=True`` every
tensor is its own selection unit instead (the per-tensor stress layout).
"""
from dataclasses import dataclass, field
from typing import List


@dataclass(frozen=True)
class TensorSpec:
    name: str
    layer: int
    numel: int
    dtype: str = "bf16"


@dataclass
class ModelShape:
    name: str
    blocks: int
    d_model: int
    ffn: int
    n_heads: int
    n_kv_heads: int
    head_dim: int
    vocab: int
    tied: bool
    per_tensor: bool = False
    tensors: List[TensorSpec] = field(default_factory=list)
    nlayers: int = 0
    layer_names: List[str] = field(default_factory=list)

    @property
    def numel(self):
        return sum(t.numel for t in self.tensors)


def decoder_shape(name, blocks, d_model, ffn, n_heads, n_kv_heads, head_dim, vocab, tied,
                  per_tensor=False):
    d, q, kv = d_model, n_heads * head_dim, n_kv_heads * head_dim
    groups = [("embed_tokens", [("embed_tokens.weight", vocab * d)])]
    for b in range(blocks):
        p = "layers.%d." % b
        groups.append(("block%d" % b, [
            (p + "self_attn.q_proj.weight", q * d),
            (p + "self_attn.k_proj.weight", kv * d),
            (p + "self_attn.v_proj.weight", kv * d),
            (p + "self_attn.o_proj.weight", d * q),
            (p + "mlp.gate_proj.weight", ffn * d),
            (p + "mlp.up_proj.weight", ffn * d),
            (p + "mlp.down_proj.weight", d * ffn),
            (p + "input_layernorm.weight", d),
            (p + "post_attention_layernorm.weight", d),
        ]))
    groups.append(("norm", [("norm.weight", d)]))
    if not tied:
        groups.append(("lm_head", [("lm_head.weight", vocab * d)]))
    tensors, names = [], []
    for gname, members in groups:
        for tname, n in members:
            if per_tensor:
                names.append(tname)
                tensors.append(TensorSpec(tname, len(names) - 1, n))
            else:
                tensors.append(TensorSpec(tname, len(names), n))
        if not per_tensor:
            names.append(gname)
    return ModelShape(name, blocks, d_model, ffn, n_heads, n_kv_heads, head_dim, vocab, tied,
                      per_tensor, tensors, len(names), names)


def tiny():
    """4 blocks, d=256, ffn=1024, 4 heads of 64 (MHA), vocab 8000, tied head."""
    return decoder_shape("tiny-4x256", 4, 256, 1024, 4, 4, 64, 8000, tied=True)


def llama32_1b():
    """Llama-3.2-1B shape: 16 blocks, d=2048, ffn=8192, 32 q / 8 kv heads of 64,
    vocab 128256, tied head (18 layers, as Table 1 lists for it)."""
    return decoder_shape("llama3.2-1b", 16, 2048, 8192, 32, 8, 64, 128256, tied=True)


def llama3_8b(per_tensor=False):
    """Llama-3-8B shape: 32 blocks, d=4096, ffn=14336, 32 q / 8 kv heads of 128,
    vocab 128256, untied head (35 layers; 291 tensors)."""
    return decoder_shape("llama3-8b" + ("-per-tensor" if per_tensor else ""), 32, 4096, 14336,
                         32, 8, 128, 128256, tied=False, per_tensor=per_tensor)


def first_blocks(shape, nblocks):
    """The first `nblocks` transformer blocks of a shape as a shape of their
    own (layers renumbered from 0), and the original layer ids kept."""
    blocks = [l for l in range(shape.nlayers) if shape.layer_names[l].startswith("block")]
    keep = blocks[:nblocks] if blocks else list(range(min(nblocks, shape.nlayers)))
    ts = [TensorSpec(t.name, keep.index(t.layer), t.numel, t.dtype)
          for t in shape.tensors if t.layer in keep]
    sub = ModelShape("%s-first%d" % (shape.name, len(keep)), 0, 0, 0, 0, 0, 0, 0, False, False,
                     ts, len(keep), [shape.layer_names[l] for l in keep])
    return sub, keep
