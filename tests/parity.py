"""Parity helpers shared by the GPU tests.

Generation parity follows a segment-and-resync protocol.  The oracle
generates the whole sequence once, logging every decision with its margin
(token decisions: top-1 minus top-2 logit; Q decisions: |Q_exit - Q_continue|).
The GPU replays it round by round from the same state.  Within a round the
decisions are compared in the order they are taken, up to the first one the
oracle takes with a margin at or below the tolerance: Q actions (values within
q_val_tol), drafts, verification tokens, and the walk's exit layer once its
decisions are all compared.  A round without a near-tie must match entirely
(drafts, acceptance count, emitted tokens).  After a round with a near-tie
the GPU restarts from the oracle's emitted sequence (ssd_resume), which
reproduces the oracle's state (KV, trace window, pending token).

Sampled decoding (temperature > 0) adds, after the verification tokens, the
acceptance tests in the order taken (margin (p - r q) / max(p, r q); the
kept/rejected outcome must match) and the round's last draw; a draw's margin
(drafts and the last draw) is the distance of u S to the nearer end of the
drawn token's CDF interval, relative to the mass S.
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


# Policy kinds: "ar", "static" (l, k), "lede" (cand; fixed_k > 0 drafts a
# fixed length), "threshold" (l, tau).
def oracle_policy(kind: str, w, qp=None, l=0, k=0, kmax=None, cand=None, fixed_k=0, tau=0.0,
                  temperature=0.0, seed=0, state="paper", discard=False):
    smp = dict(temperature=temperature, sample_seed=seed)
    if kind == "ar":
        return oracle.make_policy(oracle.POLICY_AR, **smp)
    if kind == "static":
        return oracle.make_policy(oracle.POLICY_STATIC, kmax=kmax or k, static_l=l, static_k=k,
                                  **smp)
    if kind == "threshold":
        return oracle.make_policy(oracle.POLICY_THRESHOLD, kmax=kmax or w.kmax, static_l=l,
                                  conf_threshold=tau, **smp)
    q_in = 3 if state == "paper" else w.shape.d_model + 1
    return oracle.make_policy(oracle.POLICY_LEDE, tuple(cand or w.candidates), kmax=kmax or w.kmax,
                              q_params=qp, q_hidden=w.qnet_hidden, fixed_k=fixed_k, q_in=q_in,
                              discard_on_continue=discard, **smp)


def set_gpu_policy(eng, kind: str, w, qp=None, l=0, k=0, kmax=None, cand=None, fixed_k=0, tau=0.0,
                   temperature=0.0, seed=0, state="paper", discard=False):
    smp = dict(temperature=temperature, sample_seed=seed)
    if kind == "ar":
        eng.set_ar(**smp)
    elif kind == "static":
        eng.set_static(l, k, kmax=kmax or k, **smp)
    elif kind == "threshold":
        eng.set_threshold(l, tau, kmax or w.kmax, **smp)
    else:
        eng.set_lede(w, qp, kmax=kmax, cand=cand, fixed_k=fixed_k, state=state,
                     discard_on_continue=discard, **smp)


def decision_mode(kind: str, fixed_k: int = 0) -> str:
    """"q": decisions in the walk and after every draft (LEDE, threshold);
    "walk": in the walk only (LEDE with a fixed draft length); "none"."""
    if kind == "threshold" or (kind == "lede" and not fixed_k):
        return "q"
    return "walk" if kind == "lede" else "none"


def decisions(lg: dict, mode, thr: bool = False) -> list:
    """The round's decisions in the order they are taken: the walk's Q
    decisions, d_1, then each further draft followed by the decision after
    it (mode "q"), then the verification tokens g_0..g_k.  Each entry is
    (kind, index, margin).  Threshold decisions are logged as (tau, pmax);
    their margin is |pmax - tau| / tau."""
    if mode is True:
        mode = "q"
    elif mode is False:
        mode = "none"
    out = []

    def margin(i):
        q0, q1 = lg["q_val"][i]
        return abs(q1 - q0) / q0 if thr else abs(q1 - q0)

    nv = len(lg["visited"]) if mode != "none" else 0
    if thr:
        nv = 1 if lg["kcap"] > 0 else 0
    for i in range(nv):
        out.append(("q", i, margin(i)))
    k = lg["k"]
    for i in range(k):
        out.append(("d", i, lg["draft_margin"][i]))
        if mode == "q" and i >= 1:
            out.append(("q", nv + i - 1, margin(nv + i - 1)))
    if lg.get("sampled"):
        # the verification rows' argmax decides nothing here
        for i in range(min(lg["a"] + 1, k)):
            out.append(("acc", i, abs(lg["accept_margin"][i])))
        out.append(("fix", lg["a"], lg["fix_margin"]))
        return out
    for i in range(k + 1):
        out.append(("v", i, lg["verify_margin"][i]))
    return out


def compare_round(g: dict, lg: dict, lede, tol_tok: float, tol_q: float,
                  q_val_tol: float, thr: bool = False, tol_draw: float = 0.0,
                  tol_acc: float = 0.0):
    """Compares the GPU round g with the oracle round lg decision by decision
    up to the first decision the oracle takes with a margin at or below the
    tolerance.  Returns (compared, total, clear, max Q-value error)."""
    ctx = f"round at pos {lg['pos']}: gpu {g} oracle {lg}"
    assert g["pos"] == lg["pos"] and g["x"] == lg["x"] and g["kcap"] == lg["kcap"], ctx
    assert g.get("sampled", False) == lg.get("sampled", False), ctx
    sampled = lg.get("sampled", False)
    ds = decisions(lg, lede, thr)
    n = 0
    q_err = 0.0
    for kind, i, margin in ds:
        tol = {"q": tol_q, "acc": tol_acc, "fix": tol_draw,
               "d": tol_draw if sampled else tol_tok}.get(kind, tol_tok)
        if margin <= tol:
            break
        if kind == "acc":
            assert (g["accept_margin"][i] > 0) == (lg["accept_margin"][i] > 0), ("acc", i, ctx)
            n += 1
            continue
        if kind == "fix":
            assert g["a"] == lg["a"] and g["emitted"][i] == lg["emitted"][i], ("fix", ctx)
            n += 1
            continue
        if kind == "q":
            assert g["q_action"][i] == lg["q_action"][i], ("q", i, ctx)
            q_err = max(q_err, *(abs(a - b) for a, b in zip(g["q_val"][i], lg["q_val"][i])))
            assert q_err <= q_val_tol, (q_err, ctx)
        elif kind == "d":
            assert g["drafts"][i] == lg["drafts"][i], ("d", i, ctx)
        else:
            assert g["verify_tok"][i] == lg["verify_tok"][i], ("v", i, ctx)
        n += 1
    clear = n == len(ds)
    walk_done = lede in (False, "none") or n >= len(lg["visited"])
    if walk_done and lg["kcap"] > 0:
        assert g["visited"] == lg["visited"] and g["lstar"] == lg["lstar"], ctx
    if clear:
        for key in ("k", "a", "emitted", "q_action"):
            assert g[key] == lg[key], (key, ctx)
    return n, len(ds), clear, q_err


def first_token_margin(om, ids) -> float:
    s = om.session(len(ids) + 1)
    h = s.forward(ids, 0, 0, om.shape.n_layers)
    _, st = om.exit_head(h[-1])
    return st["margin"]


def generation_parity(eng, om, w, ids, kind: str, n_new: int, tol_tok: float, tol_q: float,
                      q_val_tol: float, qp=None, l=0, k=0, kmax=None, cand=None, fixed_k=0,
                      tau=0.0, temperature=0.0, seed=0, tol_draw=0.0, tol_acc=0.0,
                      state="paper", discard=False, osess=None, first_margin=None) -> dict:
    """Returns decision counts; asserts on every compared decision.  osess:
    an oracle session already prefilled (greedy) with ids, so that a long
    prompt is not run through the oracle twice; first_margin: the oracle's
    top-1/top-2 margin of the token after the prompt, when already known."""
    P = oracle_policy(kind, w, qp, l, k, kmax, cand, fixed_k, tau, temperature, seed, state,
                      discard)
    if osess is not None:
        assert temperature == 0 and osess.kv_len == len(ids)
        s, ofirst = osess, osess.x
    else:
        s = om.session(eng.max_seq)
        ofirst = s.prefill(ids, temperature=temperature, seed=seed)
    if temperature > 0:
        first_margin = s.prefill_margin
    otoks, logs = s.generate(P, n_new)
    set_gpu_policy(eng, kind, w, qp, l, k, kmax, cand, fixed_k, tau, temperature, seed, state,
                   discard)
    gfirst = eng.prefill(ids)
    seq = list(ids) + [ofirst]
    if gfirst != ofirst:
        if temperature > 0:
            assert first_margin <= tol_draw, (gfirst, ofirst, first_margin)
        else:
            fm = first_margin if first_margin is not None else first_token_margin(om, ids)
            assert fm <= tol_tok, (gfirst, ofirst)
        eng.resume(seq)
    compared = total = clear_rounds = 0
    q_err = 0.0
    done = 0
    mode = decision_mode(kind, fixed_k)
    thr = kind == "threshold"
    for lg in logs:
        cap = n_new - done
        eng.step(cap)
        g = eng.traces(1)[0]
        n, t, clear, qe = compare_round(g, lg, mode, tol_tok, tol_q, q_val_tol, thr, tol_draw,
                                        tol_acc)
        compared += n
        total += t
        clear_rounds += int(clear)
        q_err = max(q_err, qe)
        seq += lg["emitted"]
        done += lg["n_emit"]
        if not clear and done < n_new:
            eng.resume(seq)
    assert done == n_new and seq[len(ids):] == [ofirst] + list(otoks)
    return dict(compared=compared, decisions=total, clear_rounds=clear_rounds, rounds=len(logs),
                q_err=q_err)


def rel_err(a, b) -> float:
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    return float(np.abs(a - b).max() / max(np.abs(b).max(), 1e-30))


def prompt(w, n=None):
    return synth.prompt_ids(n or w.prompt_len, w.shape.vocab)
