"""Seeded synthetic inputs shared by the oracle and the CUDA path.

`synth.h` maps (seed, tensor id, element index) to a weight, token id or
Q-network parameter; `libsynth` exposes it to Python.  Nothing here computes
any step of the decoding method.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

from .workloads import (LT_WDOWN, LT_WGU, LT_WO, LT_WQKV, QNET_IN, QNET_OUT, SEED_PROMPT,
                        SEED_QNET, SEED_WEIGHTS, TID_EMBED, TID_LMHEAD, TOPK_CONF, TRACE_T,
                        WORKLOADS, ModelShape, Workload, layer_tid, scaled_down)

HERE = os.path.dirname(os.path.abspath(__file__))
BUILD_DIR = os.path.join(HERE, "_build")
LIB_PATH = os.path.join(BUILD_DIR, "libsynth.so")
HEADER = os.path.join(HERE, "synth.h")

_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile libsynth.so with gcc (no FMA contraction: identical on x86 and Arm)."""
    src = os.path.join(HERE, "synth_host.c")
    os.makedirs(BUILD_DIR, exist_ok=True)
    newest = max(os.path.getmtime(src), os.path.getmtime(HEADER))
    if force or not os.path.exists(LIB_PATH) or os.path.getmtime(LIB_PATH) < newest:
        tmp = LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fPIC", "-shared",
                               src, "-o", tmp])
        os.replace(tmp, LIB_PATH)
    return LIB_PATH


def lib():
    global _lib
    with _lock:
        if _lib is None:
            build()
            L = ctypes.CDLL(LIB_PATH)
            u32, u64, dbl, p = ctypes.c_uint32, ctypes.c_uint64, ctypes.c_double, ctypes.c_void_p
            L.synth_philox.argtypes = [p, p, p]
            L.synth_fill_f32.argtypes = [u32, u32, u64, u64, dbl, p]
            L.synth_fill_bf16.argtypes = [u32, u32, u64, u64, dbl, p]
            L.synth_prompt.argtypes = [u32, u64, u32, p]
            L.synth_qnet_params.argtypes = [u32, ctypes.c_int, ctypes.c_int, ctypes.c_int, p]
            L.synth_sample_uniforms.argtypes = [u32, u32, u32, u32, p]
            for f in (L.synth_philox, L.synth_fill_f32, L.synth_fill_bf16, L.synth_prompt,
                      L.synth_qnet_params, L.synth_sample_uniforms):
                f.restype = None
            _lib = L
    return _lib


def _ptr(a: np.ndarray) -> int:
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data


def philox4x32_10(ctr, key) -> np.ndarray:
    c = np.asarray(ctr, dtype=np.uint32)
    k = np.asarray(key, dtype=np.uint32)
    out = np.zeros(4, dtype=np.uint32)
    lib().synth_philox(_ptr(c), _ptr(k), _ptr(out))
    return out


def sample_uniforms(seed: int, pos: int, purpose: int, n: int) -> np.ndarray:
    """Uniforms in (0, 1) of sampled decoding for the round at `pos`:
    purpose 0 draws of drafts, 1 acceptance tests, 2 the round's last draw."""
    out = np.zeros(n, dtype=np.float32)
    lib().synth_sample_uniforms(seed, pos, purpose, n, _ptr(out))
    return out


def prompt_ids(n: int, vocab: int, seed: int = SEED_PROMPT) -> np.ndarray:
    out = np.zeros(n, dtype=np.int32)
    lib().synth_prompt(seed, n, vocab, _ptr(out))
    return out


def qnet_hidden_params(in_dim: int, hidden: int, out_dim: int = QNET_OUT,
                       seed: int = SEED_QNET) -> np.ndarray:
    n = hidden * in_dim + hidden + out_dim * hidden + out_dim
    out = np.zeros(n, dtype=np.float32)
    lib().synth_qnet_params(seed, in_dim, hidden, out_dim, _ptr(out))
    return out


def weights_f32(seed: int, tid: int, start: int, n: int, sigma_scaled: float) -> np.ndarray:
    out = np.zeros(n, dtype=np.float32)
    lib().synth_fill_f32(seed, tid, start, n, sigma_scaled, _ptr(out))
    return out


def weights_bf16_bits(seed: int, tid: int, start: int, n: int, sigma_scaled: float) -> np.ndarray:
    out = np.zeros(n, dtype=np.uint16)
    lib().synth_fill_bf16(seed, tid, start, n, sigma_scaled, _ptr(out))
    return out


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (b.astype(np.uint32) << 16).view(np.float32)


__all__ = ["build", "lib", "philox4x32_10", "prompt_ids", "sample_uniforms", "qnet_hidden_params",
           "weights_f32", "weights_bf16_bits", "bf16_bits_to_f32", "WORKLOADS", "ModelShape", "Workload",
           "scaled_down", "SEED_WEIGHTS", "SEED_PROMPT", "SEED_QNET", "TRACE_T", "TOPK_CONF",
           "QNET_IN", "QNET_OUT", "HEADER", "TID_EMBED", "TID_LMHEAD", "layer_tid",
           "LT_WQKV", "LT_WO", "LT_WGU", "LT_WDOWN"]
