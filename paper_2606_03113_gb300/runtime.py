"""Device model and engine on top of the C ABI.

`DeviceModel` allocates a Llama-shaped decoder's weights with PyTorch on one
GPU and fills them with the library's seeded synthetic-weight fixture (the
same generator the CPU oracle reads).  `Engine` owns one ssd_ctx: workspace
(KV cache, activations, control block) from PyTorch, work on a PyTorch stream.
"""
from __future__ import annotations

import ctypes as C

import numpy as np
import torch

import synth
from synth.workloads import ModelShape, Workload

from . import ssd as S


def _dt(shape: ModelShape):
    return (torch.bfloat16, S.SSD_DTYPE_BF16) if shape.dtype == "bf16" else (torch.float32,
                                                                            S.SSD_DTYPE_F32)


class DeviceModel:
    """Synthetic weights of `shape` on `device`: N(0, sigma^2)-like matrices
    (synth.h), out/down projections of the second half of the layers scaled by
    late_scale, unit norm weights."""

    def __init__(self, shape: ModelShape, device: str = "cuda:0", seed: int = synth.SEED_WEIGHTS):
        self.shape = shape
        self.device = torch.device(device)
        dt, code = _dt(shape)
        self.dtype_code = code
        s = shape
        stream = torch.cuda.current_stream(self.device).cuda_stream

        def mat(rows, cols, tid, sigma):
            t = torch.empty((rows, cols), dtype=dt, device=self.device)
            S.ssd_synth_fill(t.data_ptr(), code, t.numel(), seed, tid, sigma, stream)
            return t

        def ones(n):
            return torch.ones(n, dtype=dt, device=self.device)

        self.embed = mat(s.vocab, s.d_model, synth.TID_EMBED, s.sigma)
        self.lm_head = mat(s.vocab, s.d_model, synth.TID_LMHEAD, s.sigma)
        self.final_norm = ones(s.d_model)
        self.layers = []
        qd = s.n_heads * s.head_dim
        for l in range(s.n_layers):
            late = s.late_scale if l >= s.n_layers // 2 else 1.0
            base = synth.layer_tid(l, 0)
            self.layers.append(dict(
                attn_norm=ones(s.d_model),
                wqkv=mat(s.qkv_rows, s.d_model, base + 0, s.sigma),
                wo=mat(s.d_model, qd, base + 1, s.sigma * late),
                ffn_norm=ones(s.d_model),
                w_gate_up=mat(2 * s.ffn_dim, s.d_model, base + 2, s.sigma),
                w_down=mat(s.d_model, s.ffn_dim, base + 3, s.sigma * late)))
        torch.cuda.current_stream(self.device).synchronize()

    def weight_bytes(self) -> int:
        n = self.embed.numel() + self.lm_head.numel()
        for L in self.layers:
            n += sum(t.numel() for t in L.values())
        return n * self.embed.element_size()


class Engine:
    def __init__(self, model: DeviceModel, max_seq: int, stream: torch.cuda.Stream | None = None):
        s = model.shape
        self.model = model
        self.shape = s
        self.max_seq = max_seq
        self.stream = stream or torch.cuda.current_stream(model.device)
        cfg = S.ssd_model_cfg(s.n_layers, s.d_model, s.n_heads, s.n_kv_heads, s.head_dim, s.ffn_dim,
                              s.vocab, max_seq, s.rms_eps, s.rope_theta, model.dtype_code)
        self.cfg = cfg
        nbytes = S.ssd_workspace_bytes(cfg)
        if nbytes == 0:
            raise S.SsdError(S.SSD_ERR_INVALID_ARG, "ssd_workspace_bytes", "invalid configuration")
        self.workspace = torch.empty(nbytes + 256, dtype=torch.uint8, device=model.device)
        base = self.workspace.data_ptr()
        ptr = (base + 255) // 256 * 256
        L = s.n_layers
        arrs = {}
        for key in ("attn_norm", "wqkv", "wo", "ffn_norm", "w_gate_up", "w_down"):
            a = (C.c_void_p * L)(*[lw[key].data_ptr() for lw in model.layers])
            arrs[key] = a
        self._arrs = arrs
        w = S.ssd_weights(model.embed.data_ptr(), model.lm_head.data_ptr(),
                          model.final_norm.data_ptr(),
                          *[C.cast(arrs[k], C.POINTER(C.c_void_p))
                            for k in ("attn_norm", "wqkv", "wo", "ffn_norm", "w_gate_up", "w_down")])
        self.ctx = S.ssd_init_model(cfg, w, ptr, nbytes, self.stream.cuda_stream)
        self.policy_kind = None
        self.kmax = 0

    # ----------------------------------------------------------- policies
    def set_policy(self, kind: int, cand=(), kmax: int = 0, static_l: int = 0, static_k: int = 0,
                   qnet_params: np.ndarray | None = None, qnet_hidden: int = 0, trace_T: int = 20,
                   topk: int = 5, fixed_k: int = 0, conf_threshold: float = 0.0,
                   temperature: float = 0.0, sample_seed: int = 0, qnet_in: int = 3,
                   discard_on_continue: bool = False):
        """temperature > 0 turns on speculative sampling at that temperature
        (drafts drawn from the exit distribution, emitted tokens distributed
        as the full model's), with uniforms keyed by sample_seed."""
        cand_arr = (C.c_int32 * max(1, len(cand)))(*cand)
        qp = None
        if qnet_params is not None:
            arr = np.ascontiguousarray(qnet_params, dtype=np.float32).ravel()
            # the library copies W1[hidden][in], b1, W2[2][hidden], b2 from this pointer
            need = qnet_hidden * (qnet_in + 3) + 2
            if kind == S.SSD_POLICY_LEDE and arr.size != need:
                raise ValueError(f"qnet_params holds {arr.size} floats; a network with "
                                 f"{qnet_in} inputs and {qnet_hidden} hidden units needs {need}")
            self._qp = arr
            qp = self._qp.ctypes.data_as(C.POINTER(C.c_float))
        p = S.ssd_policy(kind, len(cand), C.cast(cand_arr, C.POINTER(C.c_int32)), kmax, static_l,
                         static_k, qnet_in, qnet_hidden, qp, trace_T, topk, fixed_k, conf_threshold,
                         temperature, sample_seed, 1 if discard_on_continue else 0)
        S.ssd_set_policy(self.ctx, p)
        self.policy_kind = kind
        self.kmax = 0 if kind == S.SSD_POLICY_AR else kmax

    # Each setter takes temperature= and sample_seed= (sampled decoding).
    def set_ar(self, **sampling):
        self.set_policy(S.SSD_POLICY_AR, **sampling)

    def set_static(self, l: int, k: int, kmax: int | None = None, **sampling):
        self.set_policy(S.SSD_POLICY_STATIC, kmax=kmax or k, static_l=l, static_k=k, **sampling)

    def set_lede(self, w: Workload, qnet_params: np.ndarray | None = None, kmax: int | None = None,
                 cand=None, fixed_k: int = 0, state: str = "paper",
                 discard_on_continue: bool = False, **sampling):
        """LEDE (§3.3); one candidate is the ablation without dynamic exit,
        fixed_k > 0 the one without adaptive drafting (Table 3).  state
        "paper": the network reads (C_5, H, C_trace); "pooled": the mean
        final-normed exit state of the round's rows and the max-probability
        (d_model + 1 inputs)."""
        if state not in ("paper", "pooled"):
            raise ValueError(f"unknown state {state!r}")
        q_in = 3 if state == "paper" else w.shape.d_model + 1
        qp = (qnet_params if qnet_params is not None
              else synth.qnet_hidden_params(q_in, w.qnet_hidden))
        self.set_policy(S.SSD_POLICY_LEDE, cand=tuple(cand or w.candidates), kmax=kmax or w.kmax,
                        qnet_params=qp, qnet_hidden=w.qnet_hidden, fixed_k=fixed_k,
                        qnet_in=q_in, discard_on_continue=discard_on_continue, **sampling)

    def set_threshold(self, l: int, tau: float, kmax: int, **sampling):
        """Fixed exit layer l; drafting goes on while a draft's max-probability
        is >= tau (a Draft & Verify-style rule, §4.1 baselines)."""
        self.set_policy(S.SSD_POLICY_THRESHOLD, kmax=kmax, static_l=l, conf_threshold=tau,
                        **sampling)

    # ------------------------------------------------------------ running
    def prefill(self, ids) -> int:
        return S.ssd_prefill(self.ctx, ids)

    def resume(self, ids):
        S.ssd_resume(self.ctx, ids)

    def step(self, cap: int):
        return S.ssd_step(self.ctx, cap)

    def generate(self, n: int, rounds: bool = False):
        out, nr, infos = S.ssd_generate(self.ctx, n, rounds_cap=n if rounds else 0)
        return out, nr, infos

    def generate_async(self, n: int, out: torch.Tensor | None = None):
        S.ssd_generate_async(self.ctx, n, out.data_ptr() if out is not None else 0)

    def generate_result(self, traces: bool = False, cap: int = 4096):
        return S.ssd_generate_result(self.ctx, cap if traces else 0)

    def traces(self, cap: int = 4096):
        return S.ssd_read_traces(self.ctx, cap)

    def forward_exit(self, ids, pos0: int, l_exit: int, topk: int = 5, logits: bool = True):
        return S.ssd_forward_exit(self.ctx, ids, pos0, l_exit, topk, logits, self.shape.vocab)

    def qnet_eval(self, states):
        return S.ssd_qnet_eval(self.ctx, states)

    def read_kv(self, layer, kind, head, p0, n):
        return S.ssd_read_kv(self.ctx, layer, kind, head, p0, n, self.shape.head_dim)

    def read_state(self):
        return S.ssd_read_state(self.ctx)

    def op_gemv(self, which: int, layer: int, x: torch.Tensor, y: torch.Tensor, stream=None):
        M = x.shape[0]
        st = (stream or self.stream).cuda_stream
        S.ssd_op_gemv(self.ctx, which, layer, M, x.data_ptr(), y.data_ptr(), st)

    def op_layer(self, kernel: int, layer: int, M: int, pos0: int, stream=None):
        st = (stream or self.stream).cuda_stream
        S.ssd_op_layer(self.ctx, kernel, layer, M, pos0, st)

    def close(self):
        if getattr(self, "ctx", None):
            S.ssd_destroy(self.ctx)
            self.ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def pass_launches(n_layers: int, bf16: bool = True) -> int:
    """Kernel launches of a pass over n layers: bf16 runs the first QKV, then
    per layer attention and one chained launch (O, gate/up, down, next QKV);
    fp32 launches the five layer kernels per layer."""
    if n_layers <= 0:
        return 0
    return 2 * n_layers + 1 if bf16 else S.KERNELS_PER_LAYER * n_layers


def kernels_per_round(trace: dict, n_layers: int, kind: int, bf16: bool = True) -> int:
    """Kernel launches of one round of the round graph, from its record:
    round_begin, walk (embed; per visited segment its layers, head, decide),
    draft_begin, drafts (embed, layers 1..l*, head, decide), verify (embed,
    all layers, head), accept."""
    n = 1  # round_begin
    if trace["kcap"] > 0:
        prev = 0
        n += 1  # embed
        for c in trace["visited"]:
            n += pass_launches(c - prev, bf16) + 2
            prev = c
        n += 1  # draft_begin
        n += (trace["k"] - 1) * (1 + pass_launches(trace["lstar"], bf16) + 2)
    n += 1 + pass_launches(n_layers, bf16) + 1 + 1
    return n
