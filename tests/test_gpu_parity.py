"""GPU parity: the CUDA path (through the C ABI) against the CPU oracle on the
same seeded inputs.

Tolerances: the tiny configuration is fp32 end to end, so its tolerances are
far tighter than the bf16 ones.  bf16 configurations follow the stated
targets: logits within 2e-2 max relative error (teacher forced), tokens and
accepted counts exact wherever the oracle's top-1/top-2 margin exceeds 5e-2,
Q-values within 1e-3 when the GPU Q-network is fed the oracle's state.
"""
import numpy as np
import pytest

import oracle
import synth
from parity import generation_parity, has_gpu, prompt, rel_err
from synth.workloads import LLAMA2_7B, LLAMA2_13B, LLAMA2_70B, LLAMA3_8B, TINY, scaled_down

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not has_gpu(), reason="needs a CUDA GPU")]

# Smaller members of each family (same dtype, theta, GQA ratio, late scaling,
# head_dim 128), small enough for the oracle to finish in seconds.
SMALL = {
    "tiny": TINY,
    "7b": scaled_down(LLAMA2_7B, 8, 1024, 8, 8, 2816, 4096, 96, 40, name="7b-small"),
    "8b": scaled_down(LLAMA3_8B, 8, 1024, 8, 2, 3584, 8192, 80, 40, name="8b-small"),
    "13b": scaled_down(LLAMA2_13B, 6, 640, 5, 5, 1728, 4096, 420, 24, name="13b-long"),
    "70b": scaled_down(LLAMA2_70B, 8, 1024, 8, 1, 3584, 4096, 64, 40, name="70b-small"),
}
TOL = {  # (token margin, Q margin, logits rel, e2e Q value)
    "f32": (1e-3, 1e-4, 1e-4, 1e-3),
    "bf16": (5e-2, 1e-2, 2e-2, 2e-2),
}

_cache = {}


def setup(name):
    """(workload, device model, engine, oracle model), cached per module."""
    if name not in _cache:
        from paper_2606_03113_gb300.runtime import DeviceModel, Engine
        w = SMALL[name]
        dm = DeviceModel(w.shape)
        eng = Engine(dm, w.max_seq)
        om = oracle.Model(w.shape)
        _cache[name] = (w, dm, eng, om)
    return _cache[name]


def teardown_module(module):
    for w, dm, eng, om in _cache.values():
        eng.close()
    _cache.clear()


# ------------------------------------------------------------------ fixtures


@pytest.mark.parametrize("name", ["tiny", "7b"])
def test_synth_fill_bitwise(name):
    import torch
    from paper_2606_03113_gb300 import ssd as S
    w, dm, eng, om = setup(name)
    s = w.shape
    gpu = dm.layers[s.n_layers - 1]["wo"].float().cpu().numpy().ravel()
    n = gpu.size
    idx = np.r_[0:64, n - 64:n, np.random.default_rng(0).integers(0, n, 256)]
    ref = np.array([om.get(oracle.T_WO, s.n_layers - 1, int(i)) for i in idx])
    assert np.array_equal(gpu[idx].astype(np.float64), ref)
    e = dm.embed.float().cpu().numpy().ravel()
    assert np.array_equal(e[:512].astype(np.float64),
                          np.array([om.get(oracle.T_EMBED, 0, i) for i in range(512)]))
    # the raw fixture entry point against the host generator, odd length
    buf = torch.empty(1001, dtype=torch.float32, device="cuda")
    S.ssd_synth_fill(buf.data_ptr(), S.SSD_DTYPE_F32, 1001, 9, 77, 0.5, 0)
    torch.cuda.synchronize()
    assert np.array_equal(buf.cpu().numpy(), synth.weights_f32(9, 77, 0, 1001, 0.5))


# ---------------------------------------------------------- kernel parity


@pytest.mark.parametrize("name", ["tiny", "7b", "8b"])
@pytest.mark.parametrize("M", [1, 3, 17])
def test_gemv_matches_oracle(name, M):
    import torch
    w, dm, eng, om = setup(name)
    s = w.shape
    rng = np.random.default_rng(M)
    shapes = {0: (s.qkv_rows, s.d_model), 1: (s.d_model, s.n_heads * s.head_dim),
              2: (2 * s.ffn_dim, s.d_model), 3: (s.d_model, s.ffn_dim), 4: (s.vocab, s.d_model)}
    which_o = {0: oracle.T_WQKV, 1: oracle.T_WO, 2: oracle.T_WGU, 3: oracle.T_WDOWN,
               4: oracle.T_LMHEAD}
    for which, (rows, cols) in shapes.items():
        for layer in ([0] if which == 4 else [0, s.n_layers - 1]):
            x = rng.normal(size=(M, cols)).astype(np.float32)
            xd = torch.from_numpy(x).cuda()
            yd = torch.empty((M, rows), dtype=torch.float32, device="cuda")
            eng.op_gemv(which, layer, xd, yd)
            torch.cuda.synchronize()
            y = yd.cpu().numpy()
            for m in range(M):
                ref = om.matvec(which_o[which], layer, x[m].astype(np.float64))
                assert rel_err(y[m], ref) < 1e-5, (which, layer, m)


@pytest.mark.parametrize("name", ["tiny", "7b", "8b", "13b", "70b"])
def test_prefill_kv_and_trace(name):
    w, dm, eng, om = setup(name)
    s = w.shape
    ids = prompt(w)
    eng.set_ar()
    first = eng.prefill(ids)
    sess = om.session(w.max_seq)
    ofirst = sess.prefill(ids)
    tol = 1e-5 if s.dtype == "f32" else 1e-2
    for layer in (0, s.n_layers // 2, s.n_layers - 1):
        for kind in (0, 1):
            for head in sorted({0, s.n_kv_heads - 1}):
                g = eng.read_kv(layer, kind, head, 0, len(ids))
                ref = np.array([[sess.kv(layer, kind, head, p, i) for i in range(s.head_dim)]
                                for p in range(len(ids))])
                assert rel_err(g, ref) < tol, (layer, kind, head, rel_err(g, ref))
    x, pos, tr = eng.read_state()
    assert pos == len(ids) and x == first
    h_last = om.session(w.max_seq).forward(ids, 0, 0, s.n_layers)[-1]
    if om.exit_head(h_last)[1]["margin"] > TOL[s.dtype][0]:
        assert first == ofirst
    # trace window: full-model max-probabilities of the last 20 prompt rows
    h = om.session(w.max_seq).forward(ids, 0, 0, s.n_layers)
    ref_tr = [om.exit_head(h[r])[1]["pmax"] for r in range(len(ids) - 20, len(ids))]
    assert len(tr) == 20 and rel_err(tr, ref_tr) < (1e-5 if s.dtype == "f32" else 2e-2)


@pytest.mark.parametrize("name", ["tiny", "7b", "8b", "13b", "70b"])
def test_teacher_forced_logits_and_stats(name):
    w, dm, eng, om = setup(name)
    s = w.shape
    _, _, tol_logit, _ = TOL[s.dtype]
    tol_tok = TOL[s.dtype][0]
    ids = prompt(w)
    n0 = len(ids) - 17
    eng.set_ar()
    eng.prefill(ids[:n0])
    sess = om.session(w.max_seq)
    worst = 0.0
    for l_exit in sorted({1, max(1, s.n_layers // 2), s.n_layers}):
        for M in (1, 17):
            z, st = eng.forward_exit(ids[n0:n0 + M], n0, l_exit)
            h = sess.forward(ids[:n0 + M], 0, 0, l_exit)
            for i in range(M):
                zr, sr = om.exit_head(h[n0 + i])
                worst = max(worst, rel_err(z[i], zr))
                assert rel_err(z[i], zr) < tol_logit, (l_exit, M, i, rel_err(z[i], zr))
                g = st[i]
                if sr["margin"] > tol_tok:
                    assert g["argmax"] == sr["argmax"]
                for key in ("entropy", "conf_k", "lse", "zmax"):
                    assert abs(g[key] - sr[key]) <= tol_logit * max(1.0, abs(sr[key])), key
                assert abs(g["pmax"] - sr["pmax"]) <= tol_logit * sr["pmax"]
                # the top-5 list where it is unambiguous: clear gaps between the
                # six largest logits (a tie of the 5th and 6th changes the list)
                if np.all(-np.diff(np.sort(zr)[::-1][:6]) > tol_tok):
                    assert g["top_idx"][:5] == sr["top_idx"][:5]
    print(name, "max relative logit error", worst)


def test_qnet_values_on_oracle_states():
    w, dm, eng, om = setup("7b")
    qp = synth.qnet_hidden_params(3, w.qnet_hidden, seed=4)
    eng.set_lede(w, qp)
    rng = np.random.default_rng(1)
    states = np.c_[rng.uniform(2, 12, 200), rng.uniform(1, 10, 200), rng.uniform(0, 8, 200)]
    q = eng.qnet_eval(states)
    for i in range(200):
        ref = oracle.qnet(qp, w.qnet_hidden, states[i].astype(np.float32).astype(np.float64))
        assert np.abs(q[i] - ref).max() <= 1e-3


# ------------------------------------------------------- generation parity


@pytest.mark.parametrize("name", ["tiny", "7b", "8b", "13b", "70b"])
@pytest.mark.parametrize("kind", ["ar", "static", "lede"])
def test_generation_matches_oracle(name, kind):
    w, dm, eng, om = setup(name)
    tol_tok, tol_q, _, q_val_tol = TOL[w.shape.dtype]
    qp = synth.qnet_hidden_params(3, w.qnet_hidden, seed=2)
    L = w.shape.n_layers
    kw = dict(l=max(1, L // 2), k=min(4, w.kmax)) if kind == "static" else {}
    r = generation_parity(eng, om, w, prompt(w), kind, w.gen_len, tol_tok, tol_q, q_val_tol,
                          qp=qp, **kw)
    print(name, kind, r)
    # A near-tie (about one bf16 decision in seven on these random-init
    # models) ends the comparison of its round, so only a share of all
    # decisions is compared: every compared one must match, and the share
    # must not be vacuous (far larger for fp32).
    need = 0.5 if w.shape.dtype == "f32" else 0.1
    assert r["compared"] >= need * r["decisions"] and r["compared"] >= min(20, r["decisions"]), r


def test_lede_always_exit_policy_drafts_to_cap():
    """A Q-network that always prefers exit drafts kmax tokens at the first
    candidate; one that never does walks every candidate and drafts once."""
    w, dm, eng, om = setup("7b")
    H = w.qnet_hidden
    for qc, qe in ((0.0, 1.0), (1.0, 0.0)):
        qp = np.zeros(6 * H + 2, dtype=np.float32)
        qp[-2], qp[-1] = qc, qe
        r = generation_parity(eng, om, w, prompt(w), "lede", 24, *TOL["bf16"][:2], 1e-3, qp=qp)
        assert r["compared"] >= 0.1 * r["decisions"], r
        for t in eng.traces(64):
            if t["kcap"] > 0:
                if qe > qc:
                    assert t["visited"] == [w.candidates[0]] and t["k"] == t["kcap"]
                else:
                    assert t["visited"] == list(w.candidates) and t["k"] == 1


@pytest.mark.parametrize("name", ["tiny", "7b"])
def test_pooled_state_generation_matches_oracle(name):
    """LEDE whose Q-network reads the pooled state (the tiny configuration's
    state: mean final-normed exit state of the round's rows, then pmax;
    d_model + 1 inputs) under the segment-and-resync protocol."""
    w, dm, eng, om = setup(name)
    tol_tok, tol_q, _, q_val_tol = TOL[w.shape.dtype]
    qp = synth.qnet_hidden_params(w.shape.d_model + 1, w.qnet_hidden, seed=2)
    r = generation_parity(eng, om, w, prompt(w), "lede", w.gen_len, tol_tok, tol_q, q_val_tol,
                          qp=qp, state="pooled")
    print(name, "pooled", r)
    need = 0.5 if w.shape.dtype == "f32" else 0.1
    assert r["compared"] >= need * r["decisions"] and r["compared"] >= min(20, r["decisions"]), r
    # the last round (the protocol steps round by round): logged pooled state
    # is (pmax, rows pooled, |mean|), one row in the walk, one more per draft
    t = eng.traces(1)[0]
    nv = len(t["visited"])
    assert all(t["q_state"][i][1] == 1 for i in range(nv))
    assert all(t["q_state"][nv + i - 1][1] == i + 1 for i in range(1, t["k"]))


def test_discard_reading_matches_oracle():
    """The "discard" reading of adaptive drafting (a continue action drops
    the draft it was taken on) with a pooled-state network that exits iff
    the draft's max-probability exceeds tau: drafts are dropped in many
    rounds, and the GPU follows the oracle decision by decision."""
    w, dm, eng, om = setup("tiny")
    D, H, tau = w.shape.d_model, w.qnet_hidden, 0.003
    # unit 0 = pmax, unit 1 = 1; Q(continue) = tau, Q(exit) = pmax
    W1, b1, W2 = np.zeros((H, D + 1)), np.zeros(H), np.zeros((2, H))
    W1[0, D], b1[1], W2[0, 1], W2[1, 0] = 1.0, 1.0, tau, 1.0
    qp = np.concatenate([W1.ravel(), b1, W2.ravel(), np.zeros(2)]).astype(np.float32)
    s = om.session(w.max_seq)
    s.prefill(prompt(w))
    P = oracle.make_policy(oracle.POLICY_LEDE, w.candidates, kmax=w.kmax, q_params=qp,
                           q_hidden=H, q_in=D + 1, discard_on_continue=True)
    _, logs = s.generate(P, w.gen_len)
    dropped = sum(1 for lg in logs
                  if lg["kcap"] and lg["q_action"][len(lg["visited"]):][-1:] == [0])
    assert dropped >= 3
    tol_tok, tol_q, _, q_val_tol = TOL[w.shape.dtype]
    r = generation_parity(eng, om, w, prompt(w), "lede", w.gen_len, tol_tok, tol_q, q_val_tol,
                          qp=qp, state="pooled", discard=True)
    # the network's margin is |pmax - tau|, often below the 1e-4 Q tolerance
    # on this flat tiny model (about 60 % of the decisions are compared)
    assert r["compared"] >= 0.4 * r["decisions"], r


# --------------------------------------------- policy variants (Table 3, §4.1)


def _median_exit_pmax(om, w, l):
    """Median max-probability of the exit distribution at layer l over the
    prompt (teacher forced): a threshold that splits the drafting decisions."""
    s = om.session(w.max_seq)
    ids = prompt(w)
    h = s.forward(ids, 0, 0, l)
    return float(np.median([om.exit_head(h[i])[1]["pmax"] for i in range(len(ids))]))


@pytest.mark.parametrize("name", ["tiny", "7b", "8b"])
@pytest.mark.parametrize("variant", ["no_dynamic_exit", "no_adaptive_drafting", "threshold",
                                     "discard_on_continue"])
def test_policy_variants_match_oracle(name, variant):
    """The ablations of Table 3 (a single candidate exit layer; a fixed draft
    length after the walk) and a Draft & Verify-style confidence threshold
    run through the same graphs and kernels and match the oracle under the
    same segment-and-resync protocol."""
    w, dm, eng, om = setup(name)
    tol_tok, tol_q, _, q_val_tol = TOL[w.shape.dtype]
    qp = synth.qnet_hidden_params(3, w.qnet_hidden, seed=2)
    L = w.shape.n_layers
    if variant == "no_dynamic_exit":
        kind, kw = "lede", dict(cand=(w.candidates[len(w.candidates) // 2],))
    elif variant == "no_adaptive_drafting":
        kind, kw = "lede", dict(fixed_k=min(4, w.kmax))
    elif variant == "discard_on_continue":
        kind, kw = "lede", dict(discard=True)
    else:
        l = max(1, L // 2)
        kind, kw = "threshold", dict(l=l, tau=_median_exit_pmax(om, w, l))
    r = generation_parity(eng, om, w, prompt(w), kind, w.gen_len, tol_tok, tol_q, q_val_tol,
                          qp=qp, **kw)
    print(name, variant, r)
    need = 0.5 if w.shape.dtype == "f32" else 0.1
    assert r["compared"] >= need * r["decisions"] and r["compared"] >= min(20, r["decisions"]), r
    tr = eng.traces(4096)
    if variant == "no_adaptive_drafting":
        assert all(t["k"] == t["kcap"] for t in tr if t["kcap"] > 0)


# ------------------------------------------- experience for the offline DQN


def test_exit_table_collection_matches_oracle():
    """Experience for the offline DQN (§3.2) read through the C ABI: the
    greedy continuation is the oracle's where its decisions are clear, and
    each sampled position's exit statistics (C_5, H, exit token) at every
    candidate equal the oracle's teacher-forced exit head within the logits
    tolerance; C_trace follows the full-model max-probabilities."""
    from paper_2606_03113_gb300 import policy as P
    w, dm, eng, om = setup("7b")
    ids = prompt(w, 40)
    n_gen = 24
    tab = P.collect_exit_table(eng, w.candidates, [ids], n_gen)
    J = len(w.candidates)
    assert tab.conf.shape == (n_gen, J) and tab.correct.shape == (n_gen, J)
    # the same positions through the oracle, teacher-forced on the GPU's own
    # greedy continuation
    seq = tab.seqs[0]
    assert seq[:len(ids)] == list(ids) and len(seq) == len(ids) + n_gen + 1
    L = w.shape.n_layers
    hL = om.session(w.max_seq).forward(seq[:len(ids) + n_gen], 0, 0, L)
    for j, c in enumerate(w.candidates):
        h = om.session(w.max_seq).forward(seq[:len(ids) + n_gen], 0, 0, c)
        for t in range(0, n_gen, 5):
            _, sr = om.exit_head(h[len(ids) + t])
            _, sf = om.exit_head(hL[len(ids) + t])
            assert abs(tab.conf[t, j] - sr["conf_k"]) <= 2e-2 * max(1.0, sr["conf_k"])
            assert abs(tab.ent[t, j] - sr["entropy"]) <= 2e-2 * max(1.0, sr["entropy"])
            if sr["margin"] > 5e-2 and sf["margin"] > 5e-2:
                assert tab.correct[t, j] == (sr["argmax"] == sf["argmax"]), (c, t)
    # C_trace at the first generated position: the prompt's last 20 full-model rows
    tr0 = -np.mean([np.log(om.exit_head(hL[r])[1]["pmax"]) for r in range(len(ids) - 20, len(ids))])
    assert abs(tab.trace[0] - tr0) <= 2e-2 * max(1.0, tr0)
