"""Seeded synthetic workloads shaped like the paper's memory layers.

This module holds shapes, distributions and seeds only -- none of the layer's
arithmetic -- so that the CUDA library and the CPU oracle can be fed the very
same stored arrays.  The paper trains on RedPajama through trained 151M-1.6B
models (Sec. 5.1); none of that is needed to exercise the layer, so every
tensor here is drawn from a seeded Gaussian with the scale the layer sees:

  x      ~ N(0, 1)                [B, D_i]
  W_q    ~ N(0, 1/D_i)  variance  [H*D_k, D_i]   (query variance ~1)
  K_row, K_col ~ N(0, 1/D_k) variance [H, K, D_k]  K = sqrt(E) * n
  C      ~ N(0, 1)                [H, r, r]      Tucker cores; with h > 1
                                  component cores (MCS) [H, h, r, r] ~ N(0, 1/h)
  V      ~ N(0, 0.02^2)  (std 0.02) [N, D_v]     N = n * n physical rows
  W_p    ~ N(0, 1/(E*D_v)) variance [E, D_v, D'_v]
  query-side extras, when enabled (Tricks 2 and 4):
  conv taps ~ N(0, 1/conv_k) variance [conv_k, D_i], conv bias ~ N(0, 0.1^2)
  query LayerNorm gain ~ 1 + N(0, 0.1^2), bias ~ N(0, 0.1^2)  [A, H*D_k]
  conv state (the inputs before each sequence) ~ N(0, 1) like the tokens

Draw order from one generator seeded with the workload seed: W_q, (W_q_col),
K_row, K_col, C, W_p, then the conv taps and bias and the LayerNorm gain and
bias (when enabled).  V has a generator of its own.  Token batches come from a second generator seeded
with ``seed + 10_000 + 7919 * batch_index``.  Tables above 256 Mi elements
are drawn on the GPU (when one is used) in chunks, seeded the same way.
"""
from __future__ import annotations

import math

import numpy as np
import torch

# name -> layer shape (field names follow the C ABI's ultramem_config)
CONFIGS = {
    # tiny fp32 layer: 16 tokens, 256x256 grid, no IVE
    "tiny_fp32": dict(d_in=256, d_k=64, heads=2, rank=2, n=256, expand_e=1, d_v=256,
                      d_out=256, topk=16, topm=16, has_proj=0, share_query=1, act=0,
                      dtype="f32", seed=0, batches=(16,)),
    # decode-shaped layer: 64 tokens, 1024x1024 physical grid, E=4
    "decode_1m": dict(d_in=1024, d_k=128, heads=2, rank=2, n=1024, expand_e=4, d_v=256,
                      d_out=1024, topk=32, topm=32, has_proj=1, share_query=1, act=0,
                      dtype="bf16", seed=1, batches=(64,)),
    # mid-size layer: 2048x2048 physical grid (2 GiB bf16 table), decode sweep
    "mid_4m": dict(d_in=2048, d_k=128, heads=4, rank=2, n=2048, expand_e=4, d_v=256,
                   d_out=2048, topk=64, topm=64, has_proj=1, share_query=1, act=0,
                   dtype="bf16", seed=2, batches=(1, 8, 32, 128)),
    # largest paper-scale table: 4480x4480 ~ 20.07M rows (9.6 GiB bf16)
    "large_20m": dict(d_in=2048, d_k=128, heads=4, rank=2, n=4480, expand_e=4, d_v=256,
                      d_out=2048, topk=64, topm=64, has_proj=1, share_query=1, act=0,
                      dtype="bf16", seed=3, batches=(1, 64, 256)),
    # prefill chunk: 16384 tokens (4 sequences x 4096) on the 2048x2048 grid
    "prefill_16k": dict(d_in=2048, d_k=128, heads=4, rank=2, n=2048, expand_e=4, d_v=256,
                        d_out=2048, topk=64, topm=64, has_proj=1, share_query=1, act=0,
                        dtype="bf16", seed=4, batches=(16384,)),
}

# the batch the decode-shaped layer is quoted at
HEADLINE = ("decode_1m", 64)


def layer_config(name: str, **overrides) -> dict:
    """The config dict of a named workload, ints only, with overrides applied.

    ``dtype`` becomes 0 (fp32) / 1 (bf16); ``shuffle_seed`` defaults to the
    workload seed + 1000."""
    base = dict(CONFIGS[name])
    base.update(overrides)
    cfg = {k: v for k, v in base.items() if k != "batches"}
    if isinstance(cfg["dtype"], str):
        cfg["dtype"] = {"f32": 0, "bf16": 1}[cfg["dtype"]]
    cfg.setdefault("shuffle_seed", cfg["seed"] + 1000)
    return cfg


def small_config(**kw) -> dict:
    """A small layer for fast tests; any field can be overridden."""
    cfg = dict(d_in=96, d_k=32, heads=2, rank=2, n=24, expand_e=4, d_v=64, d_out=80,
               topk=8, topm=8, has_proj=1, share_query=1, act=0, dtype=1, seed=11,
               shuffle_seed=12345)
    cfg.update(kw)
    return cfg


def keys_per_axis(cfg: dict) -> int:
    s = int(round(math.sqrt(cfg["expand_e"])))
    return s * int(cfg["n"])


def torch_dtype(cfg: dict):
    return torch.float32 if int(cfg["dtype"]) == 0 else torch.bfloat16


def _randn(gen, shape, std, dtype, device="cpu"):
    t = torch.randn(*shape, generator=gen, dtype=torch.float32, device=device)
    if std != 1.0:
        t.mul_(std)
    return t.to(dtype)


def _table(cfg, seed, dtype, device):
    """V [N, D_v] with std 0.02, drawn in chunks of rows."""
    N = int(cfg["n"]) ** 2
    dv = int(cfg["d_v"])
    big = N * dv > (1 << 28) and device != "cpu" and torch.cuda.is_available()
    gdev = device if big else "cpu"
    gen = torch.Generator(device=gdev)
    gen.manual_seed(seed + 20_000)
    out = torch.empty((N, dv), dtype=dtype, device=device)
    rows = max(1, (1 << 26) // dv)
    for r0 in range(0, N, rows):
        r1 = min(N, r0 + rows)
        out[r0:r1].copy_(_randn(gen, (r1 - r0, dv), 0.02, dtype, gdev))
    return out


def make_weights(cfg: dict, device="cpu", with_table=True) -> dict:
    """All parameters of one layer as torch tensors on ``device``."""
    seed = int(cfg["seed"])
    dt = torch_dtype(cfg)
    gen = torch.Generator().manual_seed(seed)
    H, dk, din = int(cfg["heads"]), int(cfg["d_k"]), int(cfg["d_in"])
    K, r = keys_per_axis(cfg), int(cfg["rank"])
    E, dv, do = int(cfg["expand_e"]), int(cfg["d_v"]), int(cfg["d_out"])
    w = {}
    w["w_q"] = _randn(gen, (H * dk, din), 1.0 / math.sqrt(din), dt)
    w["w_q_col"] = None if int(cfg["share_query"]) else \
        _randn(gen, (H * dk, din), 1.0 / math.sqrt(din), dt)
    w["k_row"] = _randn(gen, (H, K, dk), 1.0 / math.sqrt(dk), dt)
    w["k_col"] = _randn(gen, (H, K, dk), 1.0 / math.sqrt(dk), dt)
    h = int(cfg.get("cores", 0))
    w["core"] = _randn(gen, (H, h, r, r), 1.0 / math.sqrt(h), torch.float32) if h > 1 \
        else _randn(gen, (H, r, r), 1.0, torch.float32)
    w["w_proj"] = _randn(gen, (E, dv, do), 1.0 / math.sqrt(E * dv), dt) \
        if int(cfg["has_proj"]) else None
    kc = int(cfg.get("conv_k", 0))
    if kc > 0:   # Trick 4: causal depthwise convolution of x
        w["conv_w"] = _randn(gen, (kc, din), 1.0 / math.sqrt(kc), torch.float32)
        w["conv_b"] = _randn(gen, (din,), 0.1, torch.float32)
    if int(cfg.get("query_ln", 0)):   # Trick 2: query LayerNorm per head
        A = 1 if int(cfg["share_query"]) else 2
        w["ln_g"] = 1.0 + _randn(gen, (A, H * dk), 0.1, torch.float32)
        w["ln_b"] = _randn(gen, (A, H * dk), 0.1, torch.float32)
    w = {k: (None if v is None else v.to(device)) for k, v in w.items()}
    w["values"] = _table(cfg, seed, dt, device) if with_table else None
    return w


def make_tokens(cfg: dict, B: int, batch_index: int = 0, device="cpu") -> torch.Tensor:
    """One batch x [B, D_i] ~ N(0, 1) in the layer's storage type."""
    gen = torch.Generator().manual_seed(int(cfg["seed"]) + 10_000 + 7919 * batch_index)
    return _randn(gen, (B, int(cfg["d_in"])), 1.0, torch_dtype(cfg)).to(device)


def make_conv_state(cfg: dict, n_seq: int, batch_index: int = 0, device="cpu"):
    """The conv_k - 1 inputs before each of n_seq sequences, [n_seq, conv_k-1,
    D_i] ~ N(0, 1) in the storage type (Trick 4's decode state)."""
    kc = int(cfg["conv_k"])
    gen = torch.Generator().manual_seed(int(cfg["seed"]) + 30_000 + 7919 * batch_index)
    return _randn(gen, (n_seq, kc - 1, int(cfg["d_in"])), 1.0, torch_dtype(cfg)).to(device)


def stored_numpy(t):
    """A torch tensor as the oracle reads it: fp32 as float32, bf16 as raw
    uint16 bit patterns (exact)."""
    if t is None:
        return None
    t = t.detach().cpu().contiguous()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view(np.uint16)
    return t.numpy().astype(np.float32, copy=False)
