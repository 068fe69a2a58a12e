"""Properties of the GPU path that hold at any size (checked here on the small
models and, for the largest ones, in the full-size tests): greedy
self-speculative decoding reproduces greedy autoregressive decoding token for
token; exiting at the last layer accepts every draft; step-by-step and
one-shot generation agree; resuming from the emitted sequence reproduces the
next round; and every bad call returns a status without launching work."""
import numpy as np
import pytest

import synth
from parity import has_gpu, prompt
from paper_2606_03113_gb300 import ssd as S

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not has_gpu(), reason="needs a CUDA GPU")]

from test_gpu_parity import SMALL, setup  # noqa: E402  (shared model cache)


def test_ssd_equals_ar_bitwise_on_gpu():
    # the GPU path is deterministic and row-independent, so every policy must
    # emit exactly the autoregressive tokens
    for name in ("tiny", "7b", "8b", "70b"):
        w, dm, eng, om = setup(name)
        ids = prompt(w)
        eng.set_ar()
        eng.prefill(ids)
        ar, _, _ = eng.generate(w.gen_len)
        L = w.shape.n_layers
        for seed in (2, 3):
            eng.set_lede(w, synth.qnet_hidden_params(3, w.qnet_hidden, seed=seed))
            eng.prefill(ids)
            le, _, _ = eng.generate(w.gen_len)
            assert np.array_equal(ar, le), name
        for l, k in ((1, 2), (max(1, L // 2), w.kmax), (L - 1, 3)):
            eng.set_static(l, k, kmax=w.kmax)
            eng.prefill(ids)
            st, _, _ = eng.generate(w.gen_len)
            assert np.array_equal(ar, st), (name, l, k)
        # the ablations of Table 3 and a confidence-threshold drafting rule
        qp = synth.qnet_hidden_params(3, w.qnet_hidden, seed=2)
        qpp = synth.qnet_hidden_params(w.shape.d_model + 1, w.qnet_hidden, seed=2)
        for setp in (lambda: eng.set_lede(w, qp, fixed_k=3),
                     lambda: eng.set_lede(w, qp, cand=(w.candidates[0],)),
                     lambda: eng.set_threshold(max(1, L // 2), 0.05, w.kmax),
                     lambda: eng.set_lede(w, qpp, state="pooled"),
                     lambda: eng.set_lede(w, qp, discard_on_continue=True)):
            setp()
            eng.prefill(ids)
            va, _, _ = eng.generate(w.gen_len)
            assert np.array_equal(ar, va), name


def test_full_depth_exit_accepts_every_draft():
    for name in ("tiny", "8b"):
        w, dm, eng, om = setup(name)
        L = w.shape.n_layers
        eng.set_static(L, 4, kmax=4)
        eng.prefill(prompt(w))
        _, nr, _ = eng.generate(w.gen_len)
        tr = eng.traces(nr)
        assert all(t["a"] == t["k"] and t["lstar"] == L for t in tr if t["kcap"] > 0)
        assert sum(t["n_emit"] for t in tr) == w.gen_len


def test_step_and_generate_agree_and_resume():
    w, dm, eng, om = setup("7b")
    ids = prompt(w)
    eng.set_lede(w, synth.qnet_hidden_params(3, w.qnet_hidden))
    first = eng.prefill(ids)
    gen, nr, infos = eng.generate(30, rounds=True)
    assert sum(i.n_emitted for i in infos) == 30 and len(infos) == nr
    eng.prefill(ids)
    seq, steps = [], 0
    while len(seq) < 30:
        toks, info = eng.step(30 - len(seq))
        assert len(toks) == info.n_emitted == info.n_accepted + 1
        seq += list(toks)
        steps += 1
    assert seq == list(gen) and steps == nr
    # resume from the emitted prefix: the next round equals the continued one
    full = list(ids) + [first] + seq
    nxt, _ = eng.step(8)
    tr_next = eng.traces(1)[0]
    eng.resume(full)
    again, _ = eng.step(8)
    assert list(again) == list(nxt) and eng.traces(1)[0]["drafts"] == tr_next["drafts"]


def test_error_paths_return_status():
    from paper_2606_03113_gb300.runtime import Engine
    w, dm, _, om = setup("tiny")
    eng = Engine(dm, w.max_seq)  # fresh context: no sequence yet
    with pytest.raises(S.SsdError) as e:
        eng.step(4)  # no policy
    assert e.value.status == S.SSD_ERR_STATE
    eng.set_ar()
    with pytest.raises(S.SsdError) as e:
        eng.prefill(np.zeros(w.max_seq, dtype=np.int32))  # no room for the pending token
    assert e.value.status == S.SSD_ERR_CAPACITY
    with pytest.raises(S.SsdError) as e:
        eng.step(4)  # nothing prefilled yet
    assert e.value.status == S.SSD_ERR_STATE
    with pytest.raises(S.SsdError) as e:
        eng.prefill(np.array([0, w.shape.vocab], dtype=np.int32))
    assert e.value.status == S.SSD_ERR_INVALID_ARG
    eng.prefill(prompt(w))
    with pytest.raises(S.SsdError) as e:
        eng.generate(w.max_seq)  # beyond the KV capacity
    assert e.value.status == S.SSD_ERR_CAPACITY
    for bad in (dict(kind=S.SSD_POLICY_STATIC, static_l=0, static_k=1, kmax=1),
                dict(kind=S.SSD_POLICY_LEDE, cand=(2, 1), kmax=2,
                     qnet_params=np.zeros(6 * 8 + 2, np.float32), qnet_hidden=8),
                dict(kind=S.SSD_POLICY_STATIC, static_l=1, static_k=1, kmax=17),
                dict(kind=9)):
        with pytest.raises(S.SsdError) as e:
            eng.set_policy(**bad)
        assert e.value.status == S.SSD_ERR_INVALID_ARG
    # the context still works afterwards
    eng.set_ar()
    eng.prefill(prompt(w))
    toks, _, _ = eng.generate(4)
    assert len(toks) == 4
    eng.close()


def test_chained_layer_launch_equals_one_launch_per_matrix():
    """The persistent launch that runs a layer's O, gate/up and down and the
    next layer's QKV as phases computes exactly what one launch per matrix
    computes: teacher-forced logits and statistics at every exit depth are
    equal bit for bit, for one row and for a verification tile."""
    import os
    from paper_2606_03113_gb300.runtime import Engine
    w, dm, eng_chain, om = setup("7b")
    ids = prompt(w)
    n0 = len(ids) - 13
    old = os.environ.get("SSD_NO_CHAIN")
    os.environ["SSD_NO_CHAIN"] = "1"
    try:
        eng_plain = Engine(dm, w.max_seq)
        outs = {}
        for name, e in (("plain", eng_plain), ("chain", None)):
            if e is None:
                os.environ["SSD_NO_CHAIN"] = "0"
                e = Engine(dm, w.max_seq)  # re-reads the switch
            e.set_ar()
            e.prefill(ids[:n0])
            res = []
            for l_exit in (1, w.shape.n_layers // 2, w.shape.n_layers):
                for M in (1, 13):
                    z, st = e.forward_exit(ids[n0:n0 + M], n0, l_exit)
                    res.append((z, [s["argmax"] for s in st], [s["entropy"] for s in st]))
            e.prefill(ids)
            toks, _, _ = e.generate(24)
            outs[name] = (res, toks)
            e.close()
    finally:
        if old is None:
            os.environ.pop("SSD_NO_CHAIN", None)
        else:
            os.environ["SSD_NO_CHAIN"] = old
    for (za, aa, ea), (zb, ab, eb) in zip(outs["plain"][0], outs["chain"][0]):
        assert np.array_equal(za, zb) and aa == ab and ea == eb
    assert np.array_equal(outs["plain"][1], outs["chain"][1])
