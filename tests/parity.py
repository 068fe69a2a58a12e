"""Parity helpers shared by the GPU tests.

Generation parity follows a segment-and-resync protocol.  The oracle
generates the whole sequence once, logging every decision with its margin
(token decisions: top-1 minus top-2 logit; Q decisions: |Q_exit - Q_continue|).
The GPU replays it round by round from the same state.  A round whose
decisions all have margins above the tolerance must match exactly (walk,
exit layer, drafts, verification tokens, acceptance count, emitted tokens,
Q actions; Q values within q_val_tol).  A round with a near-tie is not
compared: both sides then restart from the oracle's emitted sequence
(ssd_resume), which reproduces the oracle's state exactly (KV, trace window,
pending token).
"""
from __future__ import annotations

import numpy as np

import oracle
import synth


def has_gpu() -> bool:
    try:
        import torch
        return torch.cuda.is_available()
    except Exception:
        return False


def oracle_policy(kind: str, w, qp=None, l=0, k=0, kmax=None, cand=None):
    if kind == "ar":
        return oracle.make_policy(oracle.POLICY_AR)
    if kind == "static":
        return oracle.make_policy(oracle.POLICY_STATIC, kmax=kmax or k, static_l=l, static_k=k)
    return oracle.make_policy(oracle.POLICY_LEDE, tuple(cand or w.candidates), kmax=kmax or w.kmax,
                              q_params=qp, q_hidden=w.qnet_hidden)


def set_gpu_policy(eng, kind: str, w, qp=None, l=0, k=0, kmax=None, cand=None):
    if kind == "ar":
        eng.set_ar()
    elif kind == "static":
        eng.set_static(l, k, kmax=kmax or k)
    else:
        eng.set_lede(w, qp, kmax=kmax, cand=cand)


def round_is_clear(lg: dict, tol_tok: float, tol_q: float) -> bool:
    margins = list(lg["draft_margin"]) + list(lg["verify_margin"])
    if margins and min(margins) <= tol_tok:
        return False
    return all(abs(q1 - q0) > tol_q for q0, q1 in lg["q_val"])


def first_token_margin(om, ids) -> float:
    s = om.session(len(ids) + 1)
    h = s.forward(ids, 0, 0, om.shape.n_layers)
    _, st = om.exit_head(h[-1])
    return st["margin"]


def generation_parity(eng, om, w, ids, kind: str, n_new: int, tol_tok: float, tol_q: float,
                      q_val_tol: float, qp=None, l=0, k=0, kmax=None, cand=None) -> dict:
    """Returns counts of compared / skipped rounds; asserts on every compared one."""
    P = oracle_policy(kind, w, qp, l, k, kmax, cand)
    s = om.session(eng.max_seq)
    ofirst = s.prefill(ids)
    otoks, logs = s.generate(P, n_new)
    set_gpu_policy(eng, kind, w, qp, l, k, kmax, cand)
    gfirst = eng.prefill(ids)
    seq = list(ids) + [ofirst]
    if gfirst != ofirst:
        assert first_token_margin(om, ids) <= tol_tok, (gfirst, ofirst)
        eng.resume(seq)
    compared = skipped = 0
    q_err = 0.0
    done = 0
    for lg in logs:
        cap = n_new - done
        clear = round_is_clear(lg, tol_tok, tol_q)
        if clear:
            toks, info = eng.step(cap)
            g = eng.traces(1)[0]
            ctx = f"round at pos {lg['pos']}: gpu {g} oracle {lg}"
            assert g["pos"] == lg["pos"] and g["x"] == lg["x"] and g["kcap"] == lg["kcap"], ctx
            for key in ("visited", "lstar", "k", "a", "drafts", "verify_tok", "emitted", "q_action"):
                assert g[key] == lg[key], (key, ctx)
            assert list(toks) == lg["emitted"], ctx
            for (a0, a1), (b0, b1) in zip(g["q_val"], lg["q_val"]):
                q_err = max(q_err, abs(a0 - b0), abs(a1 - b1))
            assert q_err <= q_val_tol, (q_err, ctx)
            compared += 1
        else:
            skipped += 1
        seq += lg["emitted"]
        done += lg["n_emit"]
        if not clear and done < n_new:
            eng.resume(seq)
    assert done == n_new and seq[len(ids):] == [ofirst] + list(otoks)
    return dict(compared=compared, skipped=skipped, rounds=len(logs), q_err=q_err)


def rel_err(a, b) -> float:
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    return float(np.abs(a - b).max() / max(np.abs(b).max(), 1e-30))


def prompt(w, n=None):
    return synth.prompt_ids(n or w.prompt_len, w.shape.vocab)
