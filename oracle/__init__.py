"""TEST INFRASTRUCTURE: Python access to the plain fp64 CPU oracle of LEDE's
self-speculative decoding loop (lede_oracle.c).

Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline / reference
leg may import this package.  It shares no code with the CUDA path; both read
their inputs from synth/ (seeded weights, prompts and Q-network parameters).
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
import threading

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
REPO = os.path.dirname(HERE)
BUILD_DIR = os.path.join(HERE, "_build")
LIB_PATH = os.path.join(BUILD_DIR, "liboracle.so")

MAX_CAND, MAX_K, MAX_Q, TOPK_MAX = 32, 32, 64, 8
POLICY_AR, POLICY_STATIC, POLICY_LEDE, POLICY_THRESHOLD = 0, 1, 2, 3
T_EMBED, T_LMHEAD, T_FINAL_NORM, T_ATTN_NORM, T_FFN_NORM, T_WQKV, T_WO, T_WGU, T_WDOWN = range(9)


class Cfg(C.Structure):
    _fields_ = [("n_layers", C.c_int32), ("d_model", C.c_int32), ("n_heads", C.c_int32),
                ("n_kv_heads", C.c_int32), ("head_dim", C.c_int32), ("ffn_dim", C.c_int32),
                ("vocab", C.c_int32), ("bf16", C.c_int32), ("rms_eps", C.c_double),
                ("rope_theta", C.c_double), ("sigma", C.c_double), ("late_scale", C.c_double),
                ("seed", C.c_uint32), ("synth", C.c_int32)]


class Stats(C.Structure):
    _fields_ = [("argmax", C.c_int32), ("topk", C.c_int32), ("top_idx", C.c_int32 * TOPK_MAX),
                ("top_logit", C.c_double * TOPK_MAX), ("zmax", C.c_double), ("lse", C.c_double),
                ("entropy", C.c_double), ("conf_k", C.c_double), ("pmax", C.c_double),
                ("margin", C.c_double)]


class Policy(C.Structure):
    _fields_ = [("kind", C.c_int32), ("n_cand", C.c_int32), ("cand", C.c_int32 * MAX_CAND),
                ("kmax", C.c_int32), ("static_l", C.c_int32), ("static_k", C.c_int32),
                ("q_in", C.c_int32), ("q_hidden", C.c_int32), ("trace_T", C.c_int32),
                ("topk", C.c_int32), ("q_params", C.c_void_p), ("fixed_k", C.c_int32),
                ("conf_threshold", C.c_double), ("temperature", C.c_double),
                ("sample_seed", C.c_uint32), ("discard_on_continue", C.c_int32)]


class RoundLog(C.Structure):
    _fields_ = [("pos", C.c_int32), ("x", C.c_int32), ("kcap", C.c_int32),
                ("n_visited", C.c_int32), ("lstar", C.c_int32), ("k", C.c_int32), ("a", C.c_int32),
                ("n_emit", C.c_int32), ("n_q", C.c_int32), ("visited", C.c_int32 * MAX_CAND),
                ("drafts", C.c_int32 * MAX_K), ("verify_tok", C.c_int32 * (MAX_K + 1)),
                ("emitted", C.c_int32 * (MAX_K + 1)), ("q_action", C.c_int32 * MAX_Q),
                ("draft_margin", C.c_double * MAX_K), ("verify_margin", C.c_double * (MAX_K + 1)),
                ("verify_pmax", C.c_double * (MAX_K + 1)), ("q_val", (C.c_double * 2) * MAX_Q),
                ("q_state", (C.c_double * 3) * MAX_Q), ("sampled", C.c_int32),
                ("accept_margin", C.c_double * MAX_K), ("fix_margin", C.c_double)]

    def as_dict(self) -> dict:
        k, a, n = self.k, self.a, self.n_emit
        nq = min(self.n_q, MAX_Q)
        return dict(pos=self.pos, x=self.x, kcap=self.kcap, lstar=self.lstar, k=k, a=a,
                    n_emit=n, visited=list(self.visited[:self.n_visited]),
                    drafts=list(self.drafts[:k]), verify_tok=list(self.verify_tok[:k + 1]),
                    emitted=list(self.emitted[:n]), draft_margin=list(self.draft_margin[:k]),
                    verify_margin=list(self.verify_margin[:k + 1]),
                    verify_pmax=list(self.verify_pmax[:k + 1]),
                    q_action=list(self.q_action[:nq]),
                    q_val=[tuple(self.q_val[i]) for i in range(nq)],
                    q_state=[tuple(self.q_state[i]) for i in range(nq)],
                    sampled=bool(self.sampled), accept_margin=list(self.accept_margin[:k]),
                    fix_margin=self.fix_margin)


_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile liboracle.so (gcc, OpenMP, no FMA contraction so x86 and Arm
    builds round identically; -O3 keeps IEEE semantics, so every result is
    the same bit for bit as at -O2, only faster)."""
    src = os.path.join(HERE, "lede_oracle.c")
    deps = [src, os.path.join(HERE, "lede_oracle.h"), os.path.join(REPO, "synth", "synth.h")]
    os.makedirs(BUILD_DIR, exist_ok=True)
    newest = max(os.path.getmtime(p) for p in deps)
    if force or not os.path.exists(LIB_PATH) or os.path.getmtime(LIB_PATH) < newest:
        tmp = LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O3", "-std=c11", "-fopenmp", "-ffp-contract=off", "-fPIC",
                               "-shared", src, "-o", tmp, "-lm"])
        os.replace(tmp, LIB_PATH)
    return LIB_PATH


def lib():
    global _lib
    with _lock:
        if _lib is None:
            build()
            L = C.CDLL(LIB_PATH)
            p, i32 = C.c_void_p, C.c_int
            L.orc_model_create.argtypes = [C.POINTER(Cfg)]
            L.orc_model_create.restype = p
            L.orc_model_free.argtypes = [p]
            L.orc_model_free.restype = None
            L.orc_model_set.argtypes = [p, i32, i32, p, C.c_int64]
            L.orc_model_get.argtypes = [p, i32, i32, C.c_int64]
            L.orc_model_get.restype = C.c_double
            L.orc_sess_create.argtypes = [p, i32]
            L.orc_sess_create.restype = p
            L.orc_sess_free.argtypes = [p]
            L.orc_sess_free.restype = None
            L.orc_sess_kv_len.argtypes = [p]
            L.orc_sess_x.argtypes = [p]
            L.orc_sess_kv.argtypes = [p, i32, i32, i32, i32, i32]
            L.orc_sess_kv.restype = C.c_double
            L.orc_forward.argtypes = [p, p, i32, i32, i32, i32, p]
            L.orc_logits.argtypes = [p, p, p]
            L.orc_matvec.argtypes = [p, i32, i32, p, p]
            L.orc_matvec_synth.argtypes = [C.c_uint32, C.c_uint32, C.c_double, i32, C.c_int64,
                                           C.c_int64, C.c_int64, p, p]
            L.orc_stats_from_logits.argtypes = [p, i32, i32, C.POINTER(Stats)]
            L.orc_stats_from_logits.restype = None
            L.orc_exit_head.argtypes = [p, p, p, i32, C.POINTER(Stats)]
            L.orc_qnet.argtypes = [p, i32, i32, p, p]
            L.orc_qnet.restype = None
            L.orc_trace_conf.argtypes = [p, i32]
            L.orc_trace_conf.restype = C.c_double
            L.orc_trace_push.argtypes = [p, C.c_double]
            L.orc_trace_push.restype = None
            L.orc_prefill.argtypes = [p, p, i32, i32, p]
            L.orc_resume.argtypes = [p, p, i32, i32]
            L.orc_prefill_sampled.argtypes = [p, p, i32, i32, C.c_double, C.c_uint32, p, p]
            L.orc_tempered.argtypes = [p, i32, C.c_double, p]
            L.orc_tempered.restype = None
            L.orc_draw.argtypes = [p, i32, C.c_double, p]
            L.orc_spec_step.argtypes = [p, p, i32, i32, C.c_double, C.c_double, p, p, p, p]
            L.orc_round.argtypes = [p, C.POINTER(Policy), i32, C.POINTER(RoundLog)]
            L.orc_generate.argtypes = [p, C.POINTER(Policy), i32, p, p, i32, p]
            L.orc_num_threads.argtypes = []
            _lib = L
    return _lib


def _ptr(a: np.ndarray) -> int:
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data


class OracleError(RuntimeError):
    pass


def _check(rc: int, what: str):
    if rc != 0:
        raise OracleError(f"{what} failed with status {rc}")


def stats_from_logits(z, topk: int = 5) -> dict:
    z = np.ascontiguousarray(z, dtype=np.float64)
    st = Stats()
    lib().orc_stats_from_logits(_ptr(z), z.size, topk, C.byref(st))
    return stats_dict(st)


def stats_dict(st: Stats) -> dict:
    k = st.topk
    return dict(argmax=st.argmax, top_idx=list(st.top_idx[:k]), top_logit=list(st.top_logit[:k]),
                zmax=st.zmax, lse=st.lse, entropy=st.entropy, conf_k=st.conf_k, pmax=st.pmax,
                margin=st.margin)


def qnet(params: np.ndarray, hidden: int, s) -> np.ndarray:
    params = np.ascontiguousarray(params, dtype=np.float32)
    sv = np.ascontiguousarray(s, dtype=np.float64)
    q = np.zeros(2, dtype=np.float64)
    lib().orc_qnet(_ptr(params), sv.size, hidden, _ptr(sv), _ptr(q))
    return q


def make_policy(kind: int, cand=(), kmax: int = 0, static_l: int = 0, static_k: int = 0,
                q_params: np.ndarray | None = None, q_hidden: int = 0, trace_T: int = 20,
                topk: int = 5, fixed_k: int = 0, conf_threshold: float = 0.0,
                temperature: float = 0.0, sample_seed: int = 0, q_in: int = 3,
                discard_on_continue: bool = False) -> Policy:
    """q_in = 3: the paper's state (C_5, H, C_trace); q_in = d_model + 1: the
    pooled state (mean final-normed exit state of the round's rows, pmax)."""
    P = Policy()
    P.kind = kind
    P.n_cand = len(cand)
    for i, c in enumerate(cand):
        P.cand[i] = c
    P.kmax, P.static_l, P.static_k = kmax, static_l, static_k
    P.q_in, P.q_hidden, P.trace_T, P.topk = q_in, q_hidden, trace_T, topk
    P.fixed_k, P.conf_threshold = fixed_k, conf_threshold
    P.temperature, P.sample_seed = temperature, sample_seed
    P.discard_on_continue = 1 if discard_on_continue else 0
    if q_params is not None:
        arr = np.ascontiguousarray(q_params, dtype=np.float32)
        P._keep = arr  # keep alive
        P.q_params = arr.ctypes.data
    return P


class Model:
    """Oracle model; weights come from synth.h unless `synth=False`."""

    def __init__(self, shape, seed: int = 0, synth: bool = True):
        self.shape = shape
        c = Cfg()
        c.n_layers, c.d_model, c.n_heads = shape.n_layers, shape.d_model, shape.n_heads
        c.n_kv_heads, c.head_dim, c.ffn_dim = shape.n_kv_heads, shape.head_dim, shape.ffn_dim
        c.vocab, c.bf16 = shape.vocab, 1 if shape.dtype == "bf16" else 0
        c.rms_eps, c.rope_theta = shape.rms_eps, shape.rope_theta
        c.sigma, c.late_scale = shape.sigma, shape.late_scale
        c.seed, c.synth = seed, 1 if synth else 0
        self._cfg = c
        self.h = lib().orc_model_create(C.byref(c))
        if not self.h:
            raise OracleError("orc_model_create failed (bad shape or out of memory)")

    def close(self):
        if self.h:
            lib().orc_model_free(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def set(self, which: int, layer: int, data):
        a = np.ascontiguousarray(data, dtype=np.float64).ravel()
        _check(lib().orc_model_set(self.h, which, layer, _ptr(a), a.size), "orc_model_set")

    def get(self, which: int, layer: int, idx: int) -> float:
        return lib().orc_model_get(self.h, which, layer, idx)

    def matvec(self, which: int, layer: int, x) -> np.ndarray:
        x = np.ascontiguousarray(x, dtype=np.float64)
        rows = {T_EMBED: self.shape.vocab, T_LMHEAD: self.shape.vocab, T_WQKV: self.shape.qkv_rows,
                T_WO: self.shape.d_model, T_WGU: 2 * self.shape.ffn_dim,
                T_WDOWN: self.shape.d_model}[which]
        y = np.zeros(rows, dtype=np.float64)
        _check(lib().orc_matvec(self.h, which, layer, _ptr(x), _ptr(y)), "orc_matvec")
        return y

    def logits(self, h) -> np.ndarray:
        h = np.ascontiguousarray(h, dtype=np.float64)
        z = np.zeros(self.shape.vocab, dtype=np.float64)
        _check(lib().orc_logits(self.h, _ptr(h), _ptr(z)), "orc_logits")
        return z

    def exit_head(self, h, topk: int = 5):
        h = np.ascontiguousarray(h, dtype=np.float64)
        z = np.zeros(self.shape.vocab, dtype=np.float64)
        st = Stats()
        _check(lib().orc_exit_head(self.h, _ptr(h), _ptr(z), topk, C.byref(st)), "orc_exit_head")
        return z, stats_dict(st)

    def session(self, max_seq: int) -> "Session":
        return Session(self, max_seq)


class Session:
    def __init__(self, model: Model, max_seq: int):
        self.model = model
        self.max_seq = max_seq
        self.h = lib().orc_sess_create(model.h, max_seq)
        if not self.h:
            raise OracleError("orc_sess_create failed")

    def close(self):
        if self.h:
            lib().orc_sess_free(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    @property
    def kv_len(self) -> int:
        return lib().orc_sess_kv_len(self.h)

    @property
    def x(self) -> int:
        return lib().orc_sess_x(self.h)

    def kv(self, layer, which, head, pos, i) -> float:
        return lib().orc_sess_kv(self.h, layer, which, head, pos, i)

    def forward(self, tokens, pos0: int, l_from: int, l_to: int, h=None) -> np.ndarray:
        tok = np.ascontiguousarray(tokens, dtype=np.int32)
        M, d = tok.size, self.model.shape.d_model
        hh = (np.zeros((M, d)) if h is None else np.array(h, dtype=np.float64, copy=True))
        hh = np.ascontiguousarray(hh)
        _check(lib().orc_forward(self.h, _ptr(tok), M, pos0, l_from, l_to, _ptr(hh)), "orc_forward")
        return hh

    def trace_conf(self, T: int = 20) -> float:
        return lib().orc_trace_conf(self.h, T)

    def trace_push(self, p: float):
        lib().orc_trace_push(self.h, p)

    def prefill(self, ids, trace_T: int = 20, temperature: float = 0.0, seed: int = 0) -> int:
        """Prompt prefill; the first token is greedy, or drawn at `temperature`
        (> 0) with the uniform keyed by (seed, n - 1); its draw margin is
        left in `self.prefill_margin`."""
        ids = np.ascontiguousarray(ids, dtype=np.int32)
        first = np.zeros(1, dtype=np.int32)
        mg = np.zeros(1, dtype=np.float64)
        _check(lib().orc_prefill_sampled(self.h, _ptr(ids), ids.size, trace_T, temperature, seed,
                                         _ptr(first), _ptr(mg)), "orc_prefill")
        self.prefill_margin = float(mg[0])
        return int(first[0])

    def resume(self, ids, trace_T: int = 20):
        ids = np.ascontiguousarray(ids, dtype=np.int32)
        _check(lib().orc_resume(self.h, _ptr(ids), ids.size, trace_T), "orc_resume")

    def round(self, policy: Policy, cap: int) -> dict:
        lg = RoundLog()
        _check(lib().orc_round(self.h, C.byref(policy), cap, C.byref(lg)), "orc_round")
        return lg.as_dict()

    def generate(self, policy: Policy, n_new: int, logs_cap: int = 4096):
        out = np.zeros(n_new, dtype=np.int32)
        logs = (RoundLog * logs_cap)()
        nr = np.zeros(1, dtype=np.int32)
        _check(lib().orc_generate(self.h, C.byref(policy), n_new, _ptr(out), logs, logs_cap,
                                  _ptr(nr)), "orc_generate")
        return out, [logs[i].as_dict() for i in range(min(int(nr[0]), logs_cap))]


def matvec_synth(seed: int, tid: int, sigma: float, bf16: bool, row0: int, nrows: int, x) -> np.ndarray:
    x = np.ascontiguousarray(x, dtype=np.float64)
    y = np.zeros(nrows, dtype=np.float64)
    _check(lib().orc_matvec_synth(seed, tid, sigma, 1 if bf16 else 0, row0, nrows, x.size, _ptr(x),
                                  _ptr(y)), "orc_matvec_synth")
    return y


def tempered(z, temperature: float) -> np.ndarray:
    """softmax(z / temperature) (orc_tempered)."""
    z = np.ascontiguousarray(z, dtype=np.float64)
    p = np.zeros_like(z)
    lib().orc_tempered(_ptr(z), z.size, temperature, _ptr(p))
    return p


def draw(w, u: float):
    """Inverse-CDF draw of orc_draw: (token, margin); token -1 when w has no mass."""
    w = np.ascontiguousarray(w, dtype=np.float64)
    mg = np.zeros(1, dtype=np.float64)
    t = lib().orc_draw(_ptr(w), w.size, u, _ptr(mg))
    return int(t), float(mg[0])


def spec_step(p, q, d: int, r: float, u: float):
    """One speculative-sampling acceptance test (orc_spec_step):
    (emitted token, kept, accept margin, draw margin)."""
    p = np.ascontiguousarray(p, dtype=np.float64)
    q = np.ascontiguousarray(q, dtype=np.float64)
    res = np.zeros_like(p)
    kept = np.zeros(1, dtype=np.int32)
    am = np.zeros(1, dtype=np.float64)
    dm = np.zeros(1, dtype=np.float64)
    t = lib().orc_spec_step(_ptr(p), _ptr(q), p.size, d, r, u, _ptr(res), _ptr(kept), _ptr(am),
                            _ptr(dm))
    return int(t), bool(kept[0]), float(am[0]), float(dm[0])


def num_threads() -> int:
    return lib().orc_num_threads()
