"""Seeded synthetic inputs shared by the oracle tests, the GPU tests and the benchmark.

This module holds the model shapes, the weight generator and the prompt generator.
It contains none of the method's arithmetic: it only draws random numbers and
rounds them to the storage precision.  Both the CUDA path and the fp64 oracle
receive exactly the tensors produced here.

Recipe (the paper's workloads, synthetic stand-ins):
  * every matrix and embedding ~ N(0, 0.02), drawn in fp32 and rounded to the
    storage dtype (bf16 for the Vicuna-shaped configs, fp32 for "tiny");
  * every RMSNorm gain = 1.0;
  * prompts are uniform-random token ids in [0, vocab).
The paper's backbones (Table 1) are Vicuna-7B/13B; its prompts come from
MT-bench / Vicuna-bench, which are not used here: seeded uniform ids stand in.
"""
from __future__ import annotations

import copy

import torch

WEIGHT_SEED = 1234
PROMPT_SEED = 0
INIT_STD = 0.02

# Shapes: Table 1 (layers, hidden size, heads) plus the Llama FFN / vocab sizes.
_BASE = dict(rms_eps=1e-6, rope_theta=10000.0, n_draft_heads=4, kv_block=16)

CONFIGS = {
    # correctness config, fp32 everywhere
    "tiny": dict(_BASE, n_layers=2, d_model=256, n_heads=4, head_dim=64, ffn_dim=688,
                 vocab=1024, dtype="fp32", tree_nodes=16, topk=[4, 2, 1, 1],
                 batch=1, prompt_len=64, gen_tokens=32),
    # small bf16 config that exercises every bf16 kernel at ragged sizes
    "mini": dict(_BASE, n_layers=2, d_model=512, n_heads=4, head_dim=128, ffn_dim=1408,
                 vocab=2048, dtype="bf16", tree_nodes=64, topk=[5, 5, 5, 5],
                 batch=1, prompt_len=100, gen_tokens=24),
    # ragged batch of the small bf16 config
    "mini_b4": dict(_BASE, n_layers=2, d_model=512, n_heads=4, head_dim=128, ffn_dim=1408,
                    vocab=2048, dtype="bf16", tree_nodes=32, topk=[5, 5, 5, 5],
                    batch=4, prompt_lens=[37, 100, 64, 129], gen_tokens=16),
    "7b": dict(_BASE, n_layers=32, d_model=4096, n_heads=32, head_dim=128, ffn_dim=11008,
               vocab=32000, dtype="bf16", tree_nodes=64, topk=[5, 5, 5, 5],
               batch=1, prompt_len=512, gen_tokens=256),
    "13b": dict(_BASE, n_layers=40, d_model=5120, n_heads=40, head_dim=128, ffn_dim=13824,
                vocab=32000, dtype="bf16", tree_nodes=64, topk=[5, 5, 5, 5],
                batch=1, prompt_len=2048, gen_tokens=256),
    "7b_16k": dict(_BASE, n_layers=32, d_model=4096, n_heads=32, head_dim=128, ffn_dim=11008,
                   vocab=32000, dtype="bf16", tree_nodes=64, topk=[5, 5, 5, 5],
                   batch=1, prompt_len=16384, gen_tokens=128 * 5, steps=128),
    "7b_b8": dict(_BASE, n_layers=32, d_model=4096, n_heads=32, head_dim=128, ffn_dim=11008,
                  vocab=32000, dtype="bf16", tree_nodes=32, topk=[5, 5, 5, 5],
                  batch=8, prompt_len_range=[256, 4096], gen_tokens=128 * 5, steps=128),
}


def get_config(name: str) -> dict:
    cfg = copy.deepcopy(CONFIGS[name])
    cfg["name"] = name
    return cfg


def prompt_lengths(cfg: dict, seed: int = PROMPT_SEED) -> list[int]:
    """Per-sequence prompt lengths of a config (ragged ones drawn with the prompt seed)."""
    if "prompt_lens" in cfg:
        return list(cfg["prompt_lens"])
    if "prompt_len_range" in cfg:
        lo, hi = cfg["prompt_len_range"]
        g = torch.Generator().manual_seed(seed)
        return [int(v) for v in torch.randint(lo, hi + 1, (cfg["batch"],), generator=g)]
    return [cfg["prompt_len"]] * cfg["batch"]


def make_prompts(cfg: dict, seed: int = PROMPT_SEED) -> list[list[int]]:
    """Uniform-random token ids in [0, vocab), one list per sequence."""
    lens = prompt_lengths(cfg, seed)
    g = torch.Generator().manual_seed(seed + 1)
    return [torch.randint(0, cfg["vocab"], (n,), generator=g).tolist() for n in lens]


def weight_shapes(cfg: dict) -> list[tuple[str, tuple[int, ...]]]:
    """Canonical weight names and shapes, in generation order.

    Matrices are stored [out][in] (row-major, one output feature per row), so
    y = W @ x.  Names follow the paper: the base LLM (embed, per-layer block,
    final norm, LM head), the trigram encoder W1/W2, the draft's full-context
    Transformer block ("draft.*") and the K residual decoding heads Theta_k.
    """
    d, f, v, hd, h = (cfg["d_model"], cfg["ffn_dim"], cfg["vocab"], cfg["head_dim"],
                      cfg["n_heads"])
    assert h * hd == d
    out: list[tuple[str, tuple[int, ...]]] = [("embed", (v, d))]

    def block(prefix: str) -> None:
        out.extend([
            (f"{prefix}.attn_norm", (d,)),
            (f"{prefix}.wqkv", (3 * d, d)),
            (f"{prefix}.wo", (d, d)),
            (f"{prefix}.ffn_norm", (d,)),
            (f"{prefix}.w_gate", (f, d)),
            (f"{prefix}.w_up", (f, d)),
            (f"{prefix}.w_down", (d, f)),
        ])

    for i in range(cfg["n_layers"]):
        block(f"layers.{i}")
    out += [("final_norm", (d,)), ("lm_head", (v, d))]
    out += [("tri_w1", (d, 3 * d)), ("tri_w2", (d, d))]
    block("draft")
    head_in = d if cfg.get("draft_mode", 0) & 2 else 2 * d  # no-residual heads read h_full alone
    for k in range(cfg["n_draft_heads"]):
        out.append((f"heads.{k}", (v, head_in)))
    return out


def storage_dtype(cfg: dict) -> torch.dtype:
    return torch.float32 if cfg["dtype"] == "fp32" else torch.bfloat16


def make_weights(cfg: dict, seed: int = WEIGHT_SEED, device: str = "cpu") -> dict:
    """Random-init weights: N(0, 0.02) drawn in fp32, rounded to the storage dtype.

    The generator is torch's (CPU generator on "cpu", Philox on "cuda"); the values
    depend on (seed, device).  Norm gains are exactly 1.
    """
    dt = storage_dtype(cfg)
    g = torch.Generator(device=device).manual_seed(seed)
    w = {}
    for name, shape in weight_shapes(cfg):
        if name.endswith("norm"):
            w[name] = torch.ones(shape, dtype=dt, device=device)
        else:
            t = torch.randn(shape, generator=g, device=device, dtype=torch.float32)
            t.mul_(INIT_STD)
            w[name] = t.to(dt)
            del t
    return w


def weight_bytes(cfg: dict) -> dict:
    """Bytes of each weight group, for roofline accounting."""
    esz = 4 if cfg["dtype"] == "fp32" else 2
    tot: dict[str, int] = {}
    for name, shape in weight_shapes(cfg):
        n = 1
        for s in shape:
            n *= s
        grp = name.split(".")[0]
        tot[grp] = tot.get(grp, 0) + n * esz
    return tot
