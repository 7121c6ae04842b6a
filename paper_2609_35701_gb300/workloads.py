"""Seeded synthetic inputs: hidden-weight shape lists and gradient generators.

This module holds shapes and random numbers only, none of the optimizer's
arithmetic. Both the CUDA path (tests, bench) and the CPU oracle receive the
tensors it makes, so the two sides always see identical fp32 inputs.

Shapes follow the paper's PyTorch layout (rows = output features, columns =
input features, Section 3.1). The hidden 2D weights of one Llama-style layer
are q/k/v/o (hidden x hidden for multi-head attention), gate/up (ffn x hidden)
and down (hidden x ffn) (Section 1 and Table 11). The Llama-130M and
Llama-350M sets below are exactly the paper's N_h of Section 4 ("Memory
overhead"), which the tests check against Table 5.

Workloads (the paper trains on C4, which is not used here: these seeded
gradients stand in for its Llama pretraining gradients):
  single256  1 x 256x256; N(0, 0.02^2) times log-uniform [0.1, 10] row and
             column scales; lr 0.02, mu 0.95, wd 0.1, 5 NS iterations.
  llama130m  Llama-130M hidden weights (12 layers, d 768, ffn 2048); base
             N(0, 0.01^2); layers 0-5 row-imbalanced, 6-11 column-imbalanced,
             log-uniform [0.1, 10] scales.
  llama350m  Llama-350M hidden weights (24 layers, d 1024, ffn 2736); base
             N(0, 0.01^2); per-matrix pattern row / column / none by seed.
  llama1b    24 layers, d 2048, ffn 5461; base N(0, 0.01^2); |t_3| row and
             column scales (Student-t, nu = 3).
  llama7b    32 layers, d 4096, ffn 11008; base N(0, 0.005^2); per-matrix
             row / column / both imbalance, log-uniform [0.05, 20].
  llama60m_full / llama130m_full
             every trainable parameter of Llama-60M / Llama-130M (hidden 2D
             weights, 32000 x d token embedding and LM head, RMSNorm weights),
             the llama130m recipe on each.
Imbalance scales are fixed per (seed, matrix); base noise is drawn per
(seed, step, matrix). Initial weights are N(0, 0.02^2) per (seed, matrix).
"""
from __future__ import annotations

from dataclasses import dataclass, field

import torch

MODULES = ("q_proj", "k_proj", "v_proj", "o_proj", "gate_proj", "up_proj", "down_proj")


def hidden_shapes(layers, hidden, ffn, q_heads=None, kv_heads=None, head_dim=64):
    """(name, rows, cols) of every 2D hidden weight, layer by layer."""
    q = hidden if q_heads is None else q_heads * head_dim
    kv = q if kv_heads is None else kv_heads * head_dim
    out = []
    for l in range(layers):
        out += [
            (f"layers.{l}.q_proj", q, hidden),
            (f"layers.{l}.k_proj", kv, hidden),
            (f"layers.{l}.v_proj", kv, hidden),
            (f"layers.{l}.o_proj", hidden, q),
            (f"layers.{l}.gate_proj", ffn, hidden),
            (f"layers.{l}.up_proj", ffn, hidden),
            (f"layers.{l}.down_proj", hidden, ffn),
        ]
    return out


HIDDEN, REMAINING_2D, VECTOR = 0, 1, 2   # parameter types of Algorithm 1


def full_model_params(layers, hidden, ffn, vocab, q_heads, kv_heads, head_dim=64, tied=False, qkv_bias=False):
    """(name, rows, cols, kind) of every trainable parameter of a
    pre-norm SwiGLU decoder (Table 11 architectures): the hidden 2D weights,
    the token embedding and LM head (one matrix when tied), two RMSNorm
    weights per layer and a final one, and q/k/v biases when present
    (Qwen2). 1D parameters are given as (1, d)."""
    out = [(n, r, c, HIDDEN) for n, r, c in hidden_shapes(layers, hidden, ffn, q_heads, kv_heads, head_dim)]
    out.append(("embed_tokens", vocab, hidden, REMAINING_2D))
    if not tied:
        out.append(("lm_head", vocab, hidden, REMAINING_2D))
    q, kv = q_heads * head_dim, kv_heads * head_dim
    for l in range(layers):
        out.append((f"layers.{l}.input_layernorm", 1, hidden, VECTOR))
        out.append((f"layers.{l}.post_attention_layernorm", 1, hidden, VECTOR))
        if qkv_bias:
            out += [(f"layers.{l}.q_proj.bias", 1, q, VECTOR), (f"layers.{l}.k_proj.bias", 1, kv, VECTOR),
                    (f"layers.{l}.v_proj.bias", 1, kv, VECTOR)]
    out.append(("norm", 1, hidden, VECTOR))
    return out


@dataclass
class Workload:
    name: str
    shapes: list                      # [(name, rows, cols)]
    base_sigma: float
    pattern: str                      # how imbalance patterns are assigned
    scale_lo: float = 0.1
    scale_hi: float = 10.0
    steps: int = 10
    lr: float = 0.02
    momentum: float = 0.95
    weight_decay: float = 0.1
    eps: float = 1e-7
    seed: int = 0
    extra: dict = field(default_factory=dict)

    kinds: list = None                # one parameter type per shape (None: all hidden)

    @property
    def numel(self):
        return sum(r * c for _, r, c in self.shapes)

    def kind_list(self):
        return [HIDDEN] * len(self.shapes) if self.kinds is None else list(self.kinds)


def _llama(layers, hidden, ffn):
    return hidden_shapes(layers, hidden, ffn)


WORKLOADS = {
    "single256": Workload("single256", [("w", 256, 256)], 0.02, "both", steps=1),
    "llama130m": Workload("llama130m", _llama(12, 768, 2048), 0.01, "half_row_half_col", steps=10),
    "llama350m": Workload("llama350m", _llama(24, 1024, 2736), 0.01, "row_col_none", steps=10),
    "llama1b": Workload("llama1b", _llama(24, 2048, 5461), 0.01, "t3_both", steps=10),
    "llama7b": Workload("llama7b", _llama(32, 4096, 11008), 0.005, "row_col_both",
                        scale_lo=0.05, scale_hi=20.0, steps=5),
}


def _full(name, layers, hidden, ffn, vocab, heads, steps=10):
    params = full_model_params(layers, hidden, ffn, vocab, heads, heads)
    return Workload(name, [(n, r, c) for n, r, c, _ in params], 0.01, "half_row_half_col", steps=steps,
                    kinds=[k for _, _, _, k in params])


# Every trainable parameter of Llama-60M / Llama-130M (Table 11), as one
# optimizer state (Algorithm 1 over all three parameter types).
WORKLOADS["llama60m_full"] = _full("llama60m_full", 8, 512, 1376, 32000, 8)
WORKLOADS["llama130m_full"] = _full("llama130m_full", 12, 768, 2048, 32000, 12)


def get_workload(name):
    return WORKLOADS[name]


def first_layers(w: Workload, layers: int):
    """The same workload over its first `layers` layers only (entries that
    belong to no layer are kept): a smaller case of the same kernels, e.g. to
    profile a model too large to capture whole."""
    keep = [k for k, (n, _, _) in enumerate(w.shapes)
            if not n.startswith("layers.") or int(n.split(".")[1]) < layers]
    kinds = None if w.kinds is None else [w.kinds[k] for k in keep]
    return Workload(f"{w.name}[:{layers} layers]", [w.shapes[k] for k in keep], w.base_sigma, w.pattern,
                    scale_lo=w.scale_lo, scale_hi=w.scale_hi, steps=w.steps, lr=w.lr, momentum=w.momentum,
                    weight_decay=w.weight_decay, eps=w.eps, seed=w.seed, extra=dict(w.extra), kinds=kinds)


def custom_workload(shapes, pattern="both", base_sigma=0.01, seed=0, **kw):
    """A workload over an arbitrary list of (rows, cols) shapes (tests)."""
    sh = [(f"m{i}", int(r), int(c)) for i, (r, c) in enumerate(shapes)]
    return Workload("custom", sh, base_sigma, pattern, seed=seed, **kw)


def _gen(device, *key):
    g = torch.Generator(device=device)
    s = 0x9E3779B1
    for k in key:
        s = (s * 1000003 + int(k) + 1) % (2 ** 63 - 1)
    g.manual_seed(s)
    return g


def _pattern_of(w: Workload, i: int, layer: int):
    p = w.pattern
    if p == "half_row_half_col":
        n_layers = max(1, sum(1 for n, _, _ in w.shapes if n.endswith("q_proj")))
        return "row" if layer < n_layers // 2 else "col"
    if p in ("row_col_none", "row_col_both"):
        choices = ("row", "col", "none") if p == "row_col_none" else ("row", "col", "both")
        g = _gen("cpu", w.seed, 17, i)
        return choices[int(torch.randint(0, 3, (1,), generator=g))]
    return p  # "both", "row", "col", "none", "t3_both"


def _loguniform(n, lo, hi, g, device):
    u = torch.rand(n, generator=g, device=device, dtype=torch.float32)
    return torch.exp(torch.log(torch.tensor(lo)) + u * (torch.log(torch.tensor(hi)) - torch.log(torch.tensor(lo))))


def _abs_t3(n, g, device):
    # Student-t with nu = 3: Z / sqrt(V / 3), V ~ chi^2_3 = sum of 3 squared normals.
    z = torch.randn(n, generator=g, device=device, dtype=torch.float32)
    v = torch.randn(3, n, generator=g, device=device, dtype=torch.float32).pow(2).sum(0)
    return (z / torch.sqrt(v / 3.0)).abs()


def scales(w: Workload, i: int, device="cpu"):
    """Per-row and per-column imbalance scales of matrix i (None = 1)."""
    _, m, n = w.shapes[i]
    layer = int(w.shapes[i][0].split(".")[1]) if w.shapes[i][0].startswith("layers.") else 0
    pat = _pattern_of(w, i, layer)
    g = _gen(device, w.seed, 1, i)
    if pat == "t3_both":
        return _abs_t3(m, g, device), _abs_t3(n, g, device)
    rs = _loguniform(m, w.scale_lo, w.scale_hi, g, device) if pat in ("row", "both") else None
    cs = _loguniform(n, w.scale_lo, w.scale_hi, g, device) if pat in ("col", "both") else None
    return rs, cs


def gradient(w: Workload, i: int, step: int, device="cpu", scale_cache=None):
    """fp32 gradient of matrix i at a given step."""
    _, m, n = w.shapes[i]
    g = _gen(device, w.seed, 2, step, i)
    G = torch.randn(m, n, generator=g, device=device, dtype=torch.float32) * w.base_sigma
    rs, cs = scale_cache[i] if scale_cache is not None else scales(w, i, device)
    if rs is not None:
        G.mul_(rs[:, None])
    if cs is not None:
        G.mul_(cs[None, :])
    return G


def gradients(w: Workload, step: int, device="cpu", scale_cache=None):
    return [gradient(w, i, step, device, scale_cache) for i in range(len(w.shapes))]


def scale_table(w: Workload, device="cpu"):
    return [scales(w, i, device) for i in range(len(w.shapes))]


def initial_weights(w: Workload, device="cpu"):
    """W_0 ~ N(0, 0.02^2), seeded per matrix (the paper trains from random
    initialisation, Section 4; the 0.02 scale is the usual Llama init)."""
    out = []
    for i, (_, m, n) in enumerate(w.shapes):
        g = _gen(device, w.seed, 3, i)
        out.append(torch.randn(m, n, generator=g, device=device, dtype=torch.float32) * 0.02)
    return out
