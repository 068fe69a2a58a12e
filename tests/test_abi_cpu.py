"""The C-ABI library loads without a GPU, exports every symbol the headers
declare, and rejects bad arguments on the host before touching CUDA."""
import ctypes as C
import os
import re

import pytest

from paper_2606_03113_gb300 import ssd as S

INCLUDE = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include")


def declared_functions():
    names = set()
    for f in os.listdir(INCLUDE):
        if not f.endswith(".h"):
            continue
        src = open(os.path.join(INCLUDE, f)).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        for m in re.finditer(r"\b(ssd_[a-z0-9_]+)\s*\(", src):
            names.add(m.group(1))
    return names


def test_every_declared_symbol_is_exported():
    names = declared_functions()
    assert "ssd_init_model" in names and "ssd_generate" in names and len(names) >= 19
    lib = S.lib()
    missing = [n for n in sorted(names) if not hasattr(lib, n)]
    assert not missing, missing
    assert names == set(S.SIGNATURES), names ^ set(S.SIGNATURES)


def cfg(**kw):
    base = dict(n_layers=4, d_model=256, n_heads=4, n_kv_heads=4, head_dim=64, ffn_dim=688,
                vocab=1024, max_seq=128, rms_eps=1e-5, rope_theta=1e4, dtype=S.SSD_DTYPE_F32)
    base.update(kw)
    return S.ssd_model_cfg(**base)


def test_workspace_bytes_and_validation():
    n = S.ssd_workspace_bytes(cfg())
    assert n > 0 and n % 256 == 0
    assert S.ssd_workspace_bytes(cfg(max_seq=256)) > n  # KV grows with capacity
    for bad in (dict(d_model=250), dict(n_heads=3), dict(head_dim=6), dict(vocab=1023),
                dict(ffn_dim=0), dict(max_seq=1), dict(dtype=7), dict(head_dim=512)):
        assert S.ssd_workspace_bytes(cfg(**bad)) == 0, bad


def test_init_rejects_bad_arguments_on_host():
    lib = S.lib()
    out = C.c_void_p()
    w = S.ssd_weights()
    rc = lib.ssd_init_model(C.byref(cfg(d_model=250)), C.byref(w), None, 0, None, C.byref(out))
    assert rc == S.SSD_ERR_INVALID_ARG and out.value is None
    assert b"d_model" in lib.ssd_last_error(None)
    rc = lib.ssd_init_model(C.byref(cfg()), C.byref(w), None, 0, None, C.byref(out))
    assert rc == S.SSD_ERR_INVALID_ARG  # NULL weights
    assert lib.ssd_set_policy(None, None) == S.SSD_ERR_INVALID_ARG
    assert lib.ssd_prefill(None, None, 0, None) == S.SSD_ERR_INVALID_ARG
    assert lib.ssd_step(None, None, 0, None, None) == S.SSD_ERR_INVALID_ARG
    assert lib.ssd_synth_fill(None, 0, 1, 0, 0, 1.0, None) == S.SSD_ERR_INVALID_ARG
    assert lib.ssd_read_probe(None, 16, None, None) == S.SSD_ERR_INVALID_ARG
    lib.ssd_destroy(None)  # no-op


def test_struct_layouts_match_header():
    # sizes the C side relies on (all fields are 4-byte ints / floats or pointers)
    assert C.sizeof(S.ssd_model_cfg) == 11 * 4
    assert C.sizeof(S.ssd_round_info) == 6 * 4
    t = S.ssd_round_trace
    expect = (10 + 16 + 16 + 17 + 17 + 48) * 4 + (16 + 17 + 17) * 4 + 48 * 2 * 4 + 48 * 3 * 4
    expect += (2 + 16 + 1) * 4  # sampled, pad2, accept_margin[16], fix_margin
    assert C.sizeof(t) == expect
    assert C.sizeof(S.ssd_exit_stats) == (1 + 8 + 8 + 6) * 4


def test_product_path_has_no_oracle_import():
    pkg = os.path.dirname(S.__file__)
    for root, _, files in os.walk(pkg):
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h")):
                src = open(os.path.join(root, f)).read()
                assert "import oracle" not in src and "from oracle" not in src, f
                assert "lede_oracle" not in src, f


def test_struct_layouts_match_the_c_compiler(tmp_path):
    """Every field of every struct the binding mirrors sits at the offset the
    C compiler gives it from include/ssd.h and include/ssd_ops.h."""
    import subprocess
    structs = [S.ssd_model_cfg, S.ssd_weights, S.ssd_policy, S.ssd_round_info,
               S.ssd_round_trace, S.ssd_exit_stats]
    lines = ['#include <stdio.h>', '#include "ssd_ops.h"', "int main(void) {"]
    for st in structs:
        name = st.__name__
        lines.append(f'  printf("{name} sizeof %zu\\n", sizeof({name}));')
        for field, _ in st._fields_:
            lines.append(f'  printf("{name} {field} %zu\\n", offsetof({name}, {field}));')
    lines += ["  return 0;", "}"]
    src = tmp_path / "layout.c"
    src.write_text("\n".join(lines) + "\n")
    exe = tmp_path / "layout"
    inc = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include")
    subprocess.check_call(["gcc", "-std=c11", "-I", inc, str(src), "-o", str(exe)])
    out = subprocess.check_output([str(exe)], text=True).split("\n")
    got = {tuple(l.split()[:2]): int(l.split()[2]) for l in out if l.strip()}
    for st in structs:
        name = st.__name__
        assert got[(name, "sizeof")] == C.sizeof(st), name
        for field, _ in st._fields_:
            assert got[(name, field)] == getattr(st, field).offset, (name, field)


def test_binding_checks_the_q_network_size_before_the_call():
    """The binding refuses a parameter array whose size does not match the
    network's shape before the library would read past it."""
    import numpy as np
    from paper_2606_03113_gb300.runtime import Engine

    class NoCtx:  # no device context: the check must come first
        pass

    for q_in, hidden, size in ((3, 8, 8 * 6 + 2 - 1), (257, 4, 3 * 6 + 2)):
        with pytest.raises(ValueError):
            Engine.set_policy(NoCtx(), S.SSD_POLICY_LEDE, cand=(1, 2), kmax=4,
                              qnet_params=np.zeros(size, np.float32), qnet_hidden=hidden,
                              qnet_in=q_in)
