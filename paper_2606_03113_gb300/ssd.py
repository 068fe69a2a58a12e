"""Python binding of libssd.so (include/ssd.h, include/ssd_ops.h).

The functions keep the C names and only marshal arguments; every step of the
decoding path runs in the library's CUDA kernels.  PyTorch provides device
memory and streams.  Importing needs no GPU; calls that launch work do.
"""
from __future__ import annotations

import ctypes as C
import os
import threading

import numpy as np

from . import _build

SSD_OK, SSD_ERR_INVALID_ARG, SSD_ERR_CUDA, SSD_ERR_CAPACITY = 0, 1, 2, 3
SSD_ERR_STATE, SSD_ERR_DEVICE_FLAG, SSD_ERR_UNSUPPORTED = 4, 5, 6
STATUS_NAMES = {0: "SSD_OK", 1: "SSD_ERR_INVALID_ARG", 2: "SSD_ERR_CUDA", 3: "SSD_ERR_CAPACITY",
                4: "SSD_ERR_STATE", 5: "SSD_ERR_DEVICE_FLAG", 6: "SSD_ERR_UNSUPPORTED"}
SSD_DTYPE_F32, SSD_DTYPE_BF16 = 0, 1
SSD_POLICY_AR, SSD_POLICY_STATIC, SSD_POLICY_LEDE, SSD_POLICY_THRESHOLD = 0, 1, 2, 3
TRACE_MAXK, TRACE_MAXQ, TRACE_MAXC = 16, 48, 16
MAX_M = 17
KERNELS_PER_LAYER = 5


class ssd_model_cfg(C.Structure):
    _fields_ = [("n_layers", C.c_int32), ("d_model", C.c_int32), ("n_heads", C.c_int32),
                ("n_kv_heads", C.c_int32), ("head_dim", C.c_int32), ("ffn_dim", C.c_int32),
                ("vocab", C.c_int32), ("max_seq", C.c_int32), ("rms_eps", C.c_float),
                ("rope_theta", C.c_float), ("dtype", C.c_int32)]


class ssd_weights(C.Structure):
    _fields_ = [("embed", C.c_void_p), ("lm_head", C.c_void_p), ("final_norm", C.c_void_p),
                ("attn_norm", C.POINTER(C.c_void_p)), ("wqkv", C.POINTER(C.c_void_p)),
                ("wo", C.POINTER(C.c_void_p)), ("ffn_norm", C.POINTER(C.c_void_p)),
                ("w_gate_up", C.POINTER(C.c_void_p)), ("w_down", C.POINTER(C.c_void_p))]


class ssd_policy(C.Structure):
    _fields_ = [("kind", C.c_int32), ("n_cand", C.c_int32),
                ("cand_layers", C.POINTER(C.c_int32)), ("kmax", C.c_int32),
                ("static_l", C.c_int32), ("static_k", C.c_int32), ("qnet_in", C.c_int32),
                ("qnet_hidden", C.c_int32), ("qnet_params", C.POINTER(C.c_float)),
                ("trace_T", C.c_int32), ("topk", C.c_int32), ("fixed_k", C.c_int32),
                ("conf_threshold", C.c_float), ("temperature", C.c_float),
                ("sample_seed", C.c_uint32), ("discard_on_continue", C.c_int32)]


class ssd_round_info(C.Structure):
    _fields_ = [("exit_layer", C.c_int32), ("n_drafted", C.c_int32), ("n_accepted", C.c_int32),
                ("n_visited", C.c_int32), ("n_emitted", C.c_int32), ("pos", C.c_int32)]


class ssd_round_trace(C.Structure):
    _fields_ = [("pos", C.c_int32), ("x", C.c_int32), ("kcap", C.c_int32),
                ("n_visited", C.c_int32), ("lstar", C.c_int32), ("k", C.c_int32),
                ("a", C.c_int32), ("n_emit", C.c_int32), ("n_q", C.c_int32), ("pad", C.c_int32),
                ("visited", C.c_int32 * TRACE_MAXC), ("drafts", C.c_int32 * TRACE_MAXK),
                ("verify_tok", C.c_int32 * (TRACE_MAXK + 1)),
                ("emitted", C.c_int32 * (TRACE_MAXK + 1)), ("q_action", C.c_int32 * TRACE_MAXQ),
                ("draft_margin", C.c_float * TRACE_MAXK),
                ("verify_margin", C.c_float * (TRACE_MAXK + 1)),
                ("verify_pmax", C.c_float * (TRACE_MAXK + 1)),
                ("q_val", (C.c_float * 2) * TRACE_MAXQ), ("q_state", (C.c_float * 3) * TRACE_MAXQ),
                ("sampled", C.c_int32), ("pad2", C.c_int32),
                ("accept_margin", C.c_float * TRACE_MAXK), ("fix_margin", C.c_float)]

    def as_dict(self) -> dict:
        k, a, n = self.k, self.a, self.n_emit
        nq = min(self.n_q, TRACE_MAXQ)
        return dict(pos=self.pos, x=self.x, kcap=self.kcap, lstar=self.lstar, k=k, a=a,
                    n_emit=n, visited=list(self.visited[:self.n_visited]),
                    drafts=list(self.drafts[:k]), verify_tok=list(self.verify_tok[:k + 1]),
                    emitted=list(self.emitted[:n]), draft_margin=list(self.draft_margin[:k]),
                    verify_margin=list(self.verify_margin[:k + 1]),
                    verify_pmax=list(self.verify_pmax[:k + 1]), q_action=list(self.q_action[:nq]),
                    q_val=[tuple(self.q_val[i]) for i in range(nq)],
                    q_state=[tuple(self.q_state[i]) for i in range(nq)],
                    sampled=bool(self.sampled), accept_margin=list(self.accept_margin[:k]),
                    fix_margin=self.fix_margin)


class ssd_exit_stats(C.Structure):
    _fields_ = [("argmax", C.c_int32), ("top_idx", C.c_int32 * 8), ("top_logit", C.c_float * 8),
                ("zmax", C.c_float), ("lse", C.c_float), ("entropy", C.c_float),
                ("conf_k", C.c_float), ("pmax", C.c_float), ("margin", C.c_float)]

    def as_dict(self) -> dict:
        return dict(argmax=self.argmax, top_idx=list(self.top_idx), top_logit=list(self.top_logit),
                    zmax=self.zmax, lse=self.lse, entropy=self.entropy, conf_k=self.conf_k,
                    pmax=self.pmax, margin=self.margin)


# Every exported entry point with its ctypes signature (restype, argtypes).
_P, _I32, _U32, _U64, _SZ = C.c_void_p, C.c_int32, C.c_uint32, C.c_uint64, C.c_size_t
SIGNATURES = {
    "ssd_workspace_bytes": (_SZ, [C.POINTER(ssd_model_cfg)]),
    "ssd_init_model": (C.c_int, [C.POINTER(ssd_model_cfg), C.POINTER(ssd_weights), _P, _SZ, _P,
                                 C.POINTER(_P)]),
    "ssd_set_policy": (C.c_int, [_P, C.POINTER(ssd_policy)]),
    "ssd_prefill": (C.c_int, [_P, _P, _I32, _P]),
    "ssd_resume": (C.c_int, [_P, _P, _I32]),
    "ssd_step": (C.c_int, [_P, _P, _I32, _P, C.POINTER(ssd_round_info)]),
    "ssd_generate": (C.c_int, [_P, _I32, _P, _P, _P, _I32, _P]),
    "ssd_generate_async": (C.c_int, [_P, _I32, _P]),
    "ssd_generate_result": (C.c_int, [_P, _P, _P, _P, _I32]),
    "ssd_read_traces": (C.c_int, [_P, _P, _I32, _P]),
    "ssd_last_error": (C.c_char_p, [_P]),
    "ssd_destroy": (None, [_P]),
    "ssd_forward_exit": (C.c_int, [_P, _P, _I32, _I32, _I32, _I32, _P, _P]),
    "ssd_qnet_eval": (C.c_int, [_P, _P, _I32, _P]),
    "ssd_read_kv": (C.c_int, [_P, _I32, _I32, _I32, _I32, _I32, _P]),
    "ssd_read_state": (C.c_int, [_P, _P, _P, _P, _I32, _P]),
    "ssd_op_gemv": (C.c_int, [_P, _I32, _I32, _I32, _P, _P, _P]),
    "ssd_op_layer": (C.c_int, [_P, _I32, _I32, _I32, _I32, _P]),
    "ssd_gemv_noalloc": (C.c_int, [_P, _I32, _I32, _I32, _P, _I32, _P, _P, _P]),
    "ssd_synth_fill": (C.c_int, [_P, _I32, _U64, _U32, _U32, C.c_double, _P]),
    "ssd_read_probe": (C.c_int, [_P, _U64, _P, _P]),
}

_lock = threading.Lock()
_lib = None


def lib() -> C.CDLL:
    """Loads libssd.so (building it in-tree first if absent).  Raises if the
    CUDA toolkit or the library is unavailable: there is no fallback."""
    global _lib
    with _lock:
        if _lib is None:
            path = _build.LIB_PATH
            if not os.path.exists(path):
                _build.build()
            L = C.CDLL(path)
            for name, (res, args) in SIGNATURES.items():
                f = getattr(L, name)
                f.restype = res
                f.argtypes = args
            _lib = L
    return _lib


class SsdError(RuntimeError):
    def __init__(self, status: int, where: str, msg: str):
        super().__init__(f"{where}: {STATUS_NAMES.get(status, status)}: {msg}")
        self.status = status


def _check(status: int, where: str, ctx=None):
    if status != SSD_OK:
        msg = lib().ssd_last_error(ctx)
        raise SsdError(status, where, msg.decode() if msg else "")


def _ptr(a: np.ndarray) -> int:
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data


# ------------------------------------------------------------- same-name API

def ssd_workspace_bytes(cfg: ssd_model_cfg) -> int:
    return lib().ssd_workspace_bytes(C.byref(cfg))


def ssd_init_model(cfg: ssd_model_cfg, weights: ssd_weights, workspace_ptr: int,
                   workspace_bytes: int, stream_ptr: int) -> int:
    out = C.c_void_p()
    _check(lib().ssd_init_model(C.byref(cfg), C.byref(weights), workspace_ptr, workspace_bytes,
                                stream_ptr, C.byref(out)), "ssd_init_model")
    return out.value


def ssd_set_policy(ctx: int, policy: ssd_policy):
    _check(lib().ssd_set_policy(ctx, C.byref(policy)), "ssd_set_policy", ctx)


def ssd_prefill(ctx: int, ids) -> int:
    ids = np.ascontiguousarray(ids, dtype=np.int32)
    first = np.zeros(1, dtype=np.int32)
    _check(lib().ssd_prefill(ctx, _ptr(ids), ids.size, _ptr(first)), "ssd_prefill", ctx)
    return int(first[0])


def ssd_resume(ctx: int, ids):
    ids = np.ascontiguousarray(ids, dtype=np.int32)
    _check(lib().ssd_resume(ctx, _ptr(ids), ids.size), "ssd_resume", ctx)


def ssd_step(ctx: int, cap: int):
    out = np.zeros(cap, dtype=np.int32)
    n = np.zeros(1, dtype=np.int32)
    info = ssd_round_info()
    _check(lib().ssd_step(ctx, _ptr(out), cap, _ptr(n), C.byref(info)), "ssd_step", ctx)
    return out[:int(n[0])].copy(), info


def ssd_generate(ctx: int, max_new: int, out: np.ndarray | None = None, rounds_cap: int = 0):
    out = np.zeros(max_new, dtype=np.int32) if out is None else out
    n = np.zeros(2, dtype=np.int32)
    rounds = (ssd_round_info * rounds_cap)() if rounds_cap > 0 else None
    _check(lib().ssd_generate(ctx, max_new, _ptr(out), _ptr(n[0:1]),
                              C.cast(rounds, C.c_void_p) if rounds is not None else None,
                              rounds_cap, n[1:2].ctypes.data), "ssd_generate", ctx)
    nr = int(n[1])
    infos = [rounds[i] for i in range(min(nr, rounds_cap))] if rounds is not None else []
    return out, nr, infos


def ssd_generate_async(ctx: int, max_new: int, out_dev_ptr: int = 0):
    _check(lib().ssd_generate_async(ctx, max_new, out_dev_ptr or None), "ssd_generate_async", ctx)


def ssd_generate_result(ctx: int, traces_cap: int = 0):
    n = np.zeros(2, dtype=np.int32)
    tr = (ssd_round_trace * traces_cap)() if traces_cap > 0 else None
    _check(lib().ssd_generate_result(ctx, _ptr(n[0:1]), n[1:2].ctypes.data,
                                     C.cast(tr, C.c_void_p) if tr is not None else None,
                                     traces_cap), "ssd_generate_result", ctx)
    nr = int(n[0])
    return nr, int(n[1]), ([tr[i].as_dict() for i in range(min(nr, traces_cap))] if tr else [])


def ssd_read_traces(ctx: int, cap: int):
    tr = (ssd_round_trace * max(cap, 1))()
    n = np.zeros(1, dtype=np.int32)
    _check(lib().ssd_read_traces(ctx, C.cast(tr, C.c_void_p), cap, _ptr(n)), "ssd_read_traces", ctx)
    return [tr[i].as_dict() for i in range(min(int(n[0]), cap))]


def ssd_destroy(ctx: int):
    if ctx:
        lib().ssd_destroy(ctx)


def ssd_forward_exit(ctx: int, ids, pos0: int, l_exit: int, topk: int = 5, want_logits: bool = True,
                     vocab: int = 0):
    ids = np.ascontiguousarray(ids, dtype=np.int32)
    M = ids.size
    logits = np.zeros((M, vocab), dtype=np.float32) if want_logits else None
    st = (ssd_exit_stats * M)()
    _check(lib().ssd_forward_exit(ctx, _ptr(ids), M, pos0, l_exit, topk,
                                  _ptr(logits) if logits is not None else None,
                                  C.cast(st, C.c_void_p)), "ssd_forward_exit", ctx)
    return logits, [st[i].as_dict() for i in range(M)]


def ssd_qnet_eval(ctx: int, states) -> np.ndarray:
    s = np.ascontiguousarray(states, dtype=np.float32).reshape(-1, 3)
    q = np.zeros((s.shape[0], 2), dtype=np.float32)
    _check(lib().ssd_qnet_eval(ctx, _ptr(s), s.shape[0], _ptr(q)), "ssd_qnet_eval", ctx)
    return q


def ssd_read_kv(ctx: int, layer: int, kind: int, head: int, p0: int, n: int, head_dim: int):
    out = np.zeros((n, head_dim), dtype=np.float32)
    _check(lib().ssd_read_kv(ctx, layer, kind, head, p0, n, _ptr(out)), "ssd_read_kv", ctx)
    return out


def ssd_read_state(ctx: int, cap: int = 64):
    x = np.zeros(3, dtype=np.int32)
    tr = np.zeros(cap, dtype=np.float32)
    _check(lib().ssd_read_state(ctx, _ptr(x[0:1]), x[1:2].ctypes.data, _ptr(tr), cap,
                                x[2:3].ctypes.data), "ssd_read_state", ctx)
    return int(x[0]), int(x[1]), tr[:min(int(x[2]), cap)].copy()


def ssd_op_gemv(ctx: int, which: int, layer: int, M: int, x_ptr: int, y_ptr: int,
                stream_ptr: int = 0):
    _check(lib().ssd_op_gemv(ctx, which, layer, M, x_ptr, y_ptr, stream_ptr or None),
           "ssd_op_gemv", ctx)


def ssd_op_layer(ctx: int, kernel: int, layer: int, M: int, pos0: int, stream_ptr: int = 0):
    _check(lib().ssd_op_layer(ctx, kernel, layer, M, pos0, stream_ptr or None), "ssd_op_layer", ctx)


def ssd_gemv_noalloc(w_ptr: int, dtype: int, rows: int, cols: int, x_ptr: int, M: int, y_ptr: int,
                     err_ptr: int = 0, stream_ptr: int = 0):
    """y = W x without a context or any device allocation (see ssd_ops.h);
    err_ptr (device int32, optional) receives the kernel's error word."""
    _check(lib().ssd_gemv_noalloc(w_ptr, dtype, rows, cols, x_ptr, M, y_ptr, err_ptr or None,
                                  stream_ptr or None), "ssd_gemv_noalloc")


def ssd_synth_fill(dst_ptr: int, dtype: int, n: int, seed: int, tid: int, sigma: float,
                   stream_ptr: int = 0):
    _check(lib().ssd_synth_fill(dst_ptr, dtype, n, seed, tid, sigma, stream_ptr or None),
           "ssd_synth_fill")


def ssd_read_probe(src_ptr: int, nbytes: int, sink_ptr: int, stream_ptr: int = 0):
    _check(lib().ssd_read_probe(src_ptr, nbytes, sink_ptr, stream_ptr or None), "ssd_read_probe")
