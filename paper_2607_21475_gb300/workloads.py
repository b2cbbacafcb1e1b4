"""Seeded synthetic workloads shaped like the paper's decode settings.

This module only draws inputs (keys, values, queries, importance scores) and
names the configurations; it holds none of the method's arithmetic, so the
float64 oracle and the CUDA path can both be fed from it.

The paper evaluates on 7B-class grouped-query-attention models with
6k-32k-token contexts and 10-50% cache budgets (LongBench at 6k and 16k,
thirty-turn agent dialogues).  Those datasets and weights are not used here:
the inputs below are random tensors with the shapes, dtypes and score
distributions of those workloads.

Design parameters per workload: budget_tokens = round(budget * N) (expected
retained tokens per KV head), k_head = round(0.2 * budget_tokens) (score top
slice; the tiny case uses 2% of N), 4 sinks and 32 recent positions, floor
eps = 1e-6, and a compact-cache capacity that is a multiple of 64 and
leaves about 8 standard deviations of Poisson head-room above the budget.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field, replace

import torch

__all__ = ["Workload", "WORKLOADS", "sweep_workloads", "make_layer_inputs",
           "peaked_attention_inputs", "unit_seed"]


@dataclass(frozen=True)
class Workload:
    name: str
    n_layers: int
    batch: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    n_ctx: int
    dtype: str                 # "f32" or "bf16" for K, V and the decode query
    budget: float              # fraction of N retained in expectation
    score_kind: str            # "lognormal" | "attention" | "pareto" | "segments"
    seed: int
    k_head_of_ctx: float = 0.0  # if > 0: k_head = round(k_head_of_ctx * N)
    n_obs: int = 64             # observation positions for "attention" scores
    outlier_channels: int = 0   # per KV head, scaled in K and V
    outlier_scale: float = 8.0
    philox_seed: int = 0
    n_sink: int = 4
    n_recent: int = 32
    eps: float = 1e-6
    bisect_iters: int = 40

    @property
    def group(self) -> int:
        return self.n_q_heads // self.n_kv_heads

    @property
    def budget_tokens(self) -> int:
        return int(round(self.budget * self.n_ctx))

    @property
    def k_head(self) -> int:
        if self.k_head_of_ctx > 0:
            return int(round(self.k_head_of_ctx * self.n_ctx))
        return int(round(0.2 * self.budget_tokens))

    @property
    def capacity(self) -> int:
        bt = self.budget_tokens
        cap = bt + 8.0 * math.sqrt(max(bt, 1)) + 64
        cap = int(math.ceil(cap / 64.0)) * 64
        return min(cap, ((self.n_ctx + 63) // 64) * 64)

    @property
    def elem_bytes(self) -> int:
        return 4 if self.dtype == "f32" else 2

    @property
    def torch_dtype(self):
        return torch.float32 if self.dtype == "f32" else torch.bfloat16

    def with_(self, **kw) -> "Workload":
        return replace(self, **kw)


WORKLOADS = {
    # one layer, MHA 4 heads, head_dim 64, N=512, fp32, budget 10%
    "tiny": Workload("tiny", 1, 1, 4, 4, 64, 512, "f32", 0.10, "lognormal", 1001,
                     k_head_of_ctx=0.02),
    # Qwen2.5-7B-shaped: 28 layers, 28/4 heads, d=128, B=8, N=6144, bf16, 25%
    "qwen7b_6k": Workload("qwen7b_6k", 28, 8, 28, 4, 128, 6144, "bf16", 0.25, "attention",
                          1002, outlier_channels=4),
    # same GQA shape, N=16384, B=16, heavy-tailed scores, three budgets
    "qwen7b_16k_b10": Workload("qwen7b_16k_b10", 28, 16, 28, 4, 128, 16384, "bf16", 0.10,
                               "pareto", 1003),
    "qwen7b_16k_b25": Workload("qwen7b_16k_b25", 28, 16, 28, 4, 128, 16384, "bf16", 0.25,
                               "pareto", 1003),
    "qwen7b_16k_b50": Workload("qwen7b_16k_b50", 28, 16, 28, 4, 128, 16384, "bf16", 0.50,
                               "pareto", 1003),
    # long dialogue: 32/8 heads, d=128, B=32, N=32768 = 30 segments, 10%
    "dialogue_32k": Workload("dialogue_32k", 1, 32, 32, 8, 128, 32768, "bf16", 0.10,
                             "segments", 1004),
}


def sweep_workloads():
    """Batch {1,8,32,64} x N {4k,16k,64k,128k} x budget {5,10,25,50}% on 28/4, d=128."""
    out = []
    for b in (1, 8, 32, 64):
        for n in (4096, 16384, 65536, 131072):
            for beta in (0.05, 0.10, 0.25, 0.50):
                out.append(Workload(f"sweep_b{b}_n{n // 1024}k_p{int(beta * 100)}", 1, b, 28, 4,
                                    128, n, "bf16", beta, "lognormal", 1005))
    return out


def unit_seed(w: Workload, layer: int, salt: int) -> int:
    """Deterministic generator seed for one tensor of one layer."""
    return (w.seed * 1_000_003 + layer * 7919 + salt * 104_729) & 0x7FFFFFFFFFFFFFFF


def _gen(device, seed):
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return g


def _segment_decay(n_ctx: int, device) -> torch.Tensor:
    """Per-token factor 0.5^((29 - seg)/10) for 30 segments (29 x 1092 + rest)."""
    seg_len = 1092
    pos = torch.arange(n_ctx, device=device)
    seg = torch.clamp(pos // seg_len, max=29).to(torch.float64)
    return torch.pow(0.5, (29.0 - seg) / 10.0).to(torch.float32)


def make_layer_inputs(w: Workload, layer: int = 0, device="cpu", batch=None):
    """Inputs of one layer: dict with K, V [B,Hkv,N,d], Q [B,Hq,d] (w.dtype),
    and either ``scores`` [B,Hkv,N] fp32 or ``q_obs`` [B,Hkv,n_obs*G,d].

    ``batch`` restricts to the first rows (same values as the full draw for
    K/V/Q only when the full batch is drawn; callers that need identical
    bits on both sides draw once and slice).
    """
    B = w.batch if batch is None else batch
    Hkv, N, d, G = w.n_kv_heads, w.n_ctx, w.head_dim, w.group
    dt = w.torch_dtype
    out = {}
    gk = _gen(device, unit_seed(w, layer, 1))
    K = torch.randn((B, Hkv, N, d), generator=gk, device=device, dtype=torch.float32)
    gv = _gen(device, unit_seed(w, layer, 2))
    V = torch.randn((B, Hkv, N, d), generator=gv, device=device, dtype=torch.float32)
    if w.outlier_channels > 0:
        go = _gen("cpu", unit_seed(w, layer, 3))
        for h in range(Hkv):
            ch = torch.randperm(d, generator=go)[: w.outlier_channels].to(device)
            K[:, h, :, ch] *= w.outlier_scale
            V[:, h, :, ch] *= w.outlier_scale
    out["K"] = K.to(dt).contiguous()
    del K
    out["V"] = V.to(dt).contiguous()
    del V
    gq = _gen(device, unit_seed(w, layer, 4))
    out["Q"] = torch.randn((B, w.n_q_heads, d), generator=gq, device=device,
                           dtype=torch.float32).to(dt).contiguous()
    gs = _gen(device, unit_seed(w, layer, 5))
    if w.score_kind == "attention":
        out["q_obs"] = torch.randn((B, Hkv, w.n_obs * G, d), generator=gs, device=device,
                                   dtype=torch.float32).to(dt).contiguous()
    else:
        if w.score_kind == "lognormal":
            z = torch.randn((B, Hkv, N), generator=gs, device=device, dtype=torch.float32)
            s = torch.exp(1.5 * z)
        elif w.score_kind == "pareto":
            # Pareto(alpha=1.2, x_m=1): x_m * U^(-1/alpha), U in (0, 1]
            u = torch.rand((B, Hkv, N), generator=gs, device=device, dtype=torch.float32)
            s = torch.pow(1.0 - u, -1.0 / 1.2)
        elif w.score_kind == "segments":
            z = torch.randn((B, Hkv, N), generator=gs, device=device, dtype=torch.float32)
            s = torch.exp(1.5 * z) * _segment_decay(N, device)
        else:
            raise ValueError(w.score_kind)
        out["scores"] = s.contiguous()
    return out


def peaked_attention_inputs(w: Workload, layer: int = 0, device="cpu", q_scale: float = 3.0,
                            obs_noise: float = 0.5, n_obs: int = 64):
    """A workload's K, V with decode queries sharpened and observation queries
    that resemble them, for measuring the certificate where attention is
    concentrated (with K, Q ~ N(0, 1) at d = 128 each query spreads its mass
    over thousands of tokens and the full-cache output is close to 0).

    Q = q_scale * Q0 (Q0 the workload's queries); ``q_obs`` [B,Hkv,n_obs*G,d]:
    row r of KV head h is q_scale * (Q0[h*G + r // n_obs] + obs_noise * z),
    z ~ N(0, 1), so scores accumulated from them rank tokens the way the
    decode queries weight them.  Returns the dict of make_layer_inputs with
    Q replaced, ``q_obs`` added and ``scores`` removed."""
    inp = make_layer_inputs(w, layer, device)
    inp.pop("scores", None)
    B, Hkv, G, d = w.batch, w.n_kv_heads, w.group, w.head_dim
    q0 = inp["Q"].float()
    gz = _gen(device, unit_seed(w, layer, 6))
    z = torch.randn((B, Hkv, n_obs * G, d), generator=gz, device=device, dtype=torch.float32)
    base = q0.view(B, Hkv, G, 1, d).expand(B, Hkv, G, n_obs, d).reshape(B, Hkv, G * n_obs, d)
    inp["q_obs"] = (q_scale * (base + obs_noise * z)).to(w.torch_dtype).contiguous()
    inp["Q"] = (q_scale * q0).to(w.torch_dtype).contiguous()
    return inp
