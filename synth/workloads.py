"""Synthetic workloads: the five Llama-shaped decoder configurations, their
prompts, generation lengths and LEDE policy grids.

The paper evaluates LayerSkip-pretrained Llama checkpoints on CNN/DM, TOPv2,
Alpaca and HumanEval at batch 1 with up to 512 new tokens (§4.1, Evaluation
Setup).  Neither checkpoints nor datasets are used here: random-init weights
of the same architectures (seeded, see synth.h) and uniform random prompts
stand in for them.  Layers in the second half get their attention-output and
FFN-down projections scaled down, so that early exits agree with the full
model at a controllable rate.

Candidate exit layers and draft caps follow the paper's online procedure
(§3.1.2 Action Space, §3.3) with the maximum speculation length of 12 per
round (§4.1, Baselines); the 70B shape allows 16.
"""
from __future__ import annotations

from dataclasses import dataclass, field

SEED_WEIGHTS = 0
SEED_PROMPT = 1
SEED_QNET = 2

# tensor ids of synth.h
TID_EMBED = 1
TID_LMHEAD = 2
TID_LAYER_BASE = 16
LT_WQKV, LT_WO, LT_WGU, LT_WDOWN = 0, 1, 2, 3


def layer_tid(layer: int, which: int) -> int:
    return TID_LAYER_BASE + 4 * layer + which


TRACE_T = 20  # C_trace window (§3.1.1, T = 20)
TOPK_CONF = 5  # token confidence C_k uses the top-5 probabilities (§3.1.1, k = 5)
QNET_IN = 3  # state s = (C_5, H, C_trace)
QNET_OUT = 2  # Q(continue), Q(exit) (§3.1.2: continue = 0, exit = 1)


@dataclass(frozen=True)
class ModelShape:
    name: str
    n_layers: int
    d_model: int
    n_heads: int
    n_kv_heads: int
    head_dim: int
    ffn_dim: int
    vocab: int
    rms_eps: float
    rope_theta: float
    dtype: str  # "f32" or "bf16": weight, KV-cache and embedding storage
    sigma: float = 0.02
    late_scale: float = 0.2  # on wo / wdown of layers >= n_layers // 2 (0-indexed)

    @property
    def qkv_rows(self) -> int:
        return (self.n_heads + 2 * self.n_kv_heads) * self.head_dim

    @property
    def elt_bytes(self) -> int:
        return 4 if self.dtype == "f32" else 2

    def layer_weight_elems(self) -> int:
        d, f = self.d_model, self.ffn_dim
        return self.qkv_rows * d + d * self.n_heads * self.head_dim + 2 * f * d + d * f

    def layer_weight_bytes(self) -> int:
        return self.layer_weight_elems() * self.elt_bytes

    def lm_head_bytes(self) -> int:
        return self.vocab * self.d_model * self.elt_bytes

    def kv_bytes_per_pos_layer(self) -> int:
        return 2 * self.n_kv_heads * self.head_dim * self.elt_bytes


@dataclass(frozen=True)
class Workload:
    shape: ModelShape
    prompt_len: int
    gen_len: int
    candidates: tuple
    kmax: int
    qnet_hidden: int
    static_grid_l: tuple = field(default=())

    @property
    def name(self) -> str:
        return self.shape.name

    @property
    def max_seq(self) -> int:
        need = self.prompt_len + self.gen_len + self.kmax + 2
        return (need + 63) // 64 * 64


TINY = Workload(
    ModelShape("tiny", 4, 256, 4, 4, 64, 688, 1024, 1e-5, 10000.0, "f32", late_scale=0.1),
    prompt_len=32, gen_len=64, candidates=(1, 2, 3), kmax=4, qnet_hidden=64)

LLAMA2_7B = Workload(
    ModelShape("llama2-7b", 32, 4096, 32, 32, 128, 11008, 32000, 1e-5, 10000.0, "bf16"),
    prompt_len=512, gen_len=256, candidates=tuple(range(4, 29, 4)), kmax=12, qnet_hidden=256)

LLAMA3_8B = Workload(
    ModelShape("llama3-8b", 32, 4096, 32, 8, 128, 14336, 128256, 1e-5, 500000.0, "bf16"),
    prompt_len=1024, gen_len=512, candidates=tuple(range(4, 29, 4)), kmax=12, qnet_hidden=256)

LLAMA2_13B = Workload(
    ModelShape("llama2-13b", 40, 5120, 40, 40, 128, 13824, 32000, 1e-5, 10000.0, "bf16"),
    prompt_len=2048, gen_len=256, candidates=tuple(range(5, 36, 5)), kmax=12, qnet_hidden=256)

LLAMA2_70B = Workload(
    ModelShape("llama2-70b", 80, 8192, 64, 8, 128, 28672, 32000, 1e-5, 10000.0, "bf16"),
    prompt_len=1024, gen_len=256, candidates=tuple(range(8, 73, 8)), kmax=16, qnet_hidden=256)

WORKLOADS = {w.name: w for w in (TINY, LLAMA2_7B, LLAMA3_8B, LLAMA2_13B, LLAMA2_70B)}


def scaled_down(w: Workload, n_layers: int, d_model: int, n_heads: int, n_kv_heads: int,
                ffn_dim: int, vocab: int, prompt_len: int, gen_len: int, name: str | None = None,
                head_dim: int | None = None) -> Workload:
    """A smaller model of the same family (dtype, theta, scaling) for tests
    that the oracle must finish in seconds.  Candidates are rescaled to the
    new depth."""
    s = w.shape
    hd = head_dim if head_dim is not None else s.head_dim
    shape = ModelShape(name or f"{s.name}-small", n_layers, d_model, n_heads, n_kv_heads, hd,
                       ffn_dim, vocab, s.rms_eps, s.rope_theta, s.dtype, s.sigma, s.late_scale)
    cands = tuple(sorted({max(1, min(n_layers - 1, round(c * n_layers / s.n_layers)))
                          for c in w.candidates}))
    return Workload(shape, prompt_len, gen_len, cands, w.kmax, w.qnet_hidden)
