"""ssd_gemv_noalloc: the allocation-free matrix-vector product, for callers
that cannot allocate device memory (code running during CUDA-graph capture,
hosts whose framework owns the device memory pool).  It must give the same
products as ssd_op_gemv, the context-based entry point, on consecutive calls
that share its static scratch, and the oracle's fp64 products of the same
generated weights on sampled rows; its error word must read zero.
Self-contained, so it passes alone in a fresh process as well as after the
other GPU tests; collected last on purpose."""
import numpy as np
import pytest

import oracle
import synth
from parity import has_gpu, rel_err

pytestmark = [pytest.mark.gpu, pytest.mark.skipif(not has_gpu(), reason="needs a CUDA GPU")]


def _sampled_rows(n: int) -> np.ndarray:
    return np.unique(np.r_[0:16, n // 2:n // 2 + 16, n - 16:n])


def test_noalloc_matches_context_gemv_and_oracle_on_consecutive_calls():
    import torch

    from paper_2606_03113_gb300 import ssd as S
    from paper_2606_03113_gb300.runtime import DeviceModel, Engine
    from synth.workloads import LLAMA2_7B, scaled_down

    w = scaled_down(LLAMA2_7B, 2, 1024, 8, 8, 2816, 4096, 32, 8, name="noalloc-small")
    dm = DeviceModel(w.shape)
    eng = Engine(dm, w.max_seq)
    s = w.shape
    cases = [  # (which, layer, W, tensor id, rows, cols, M): two calls in a row, then a third
        (2, 1, dm.layers[1]["w_gate_up"], synth.layer_tid(1, synth.LT_WGU), 2 * s.ffn_dim,
         s.d_model, 1),
        (3, 0, dm.layers[0]["w_down"], synth.layer_tid(0, synth.LT_WDOWN), s.d_model, s.ffn_dim, 5),
        (4, 0, dm.lm_head, synth.TID_LMHEAD, s.vocab, s.d_model, 17),
    ]
    rng = np.random.default_rng(7)
    stream = torch.cuda.current_stream().cuda_stream
    err = torch.full((1,), -1, dtype=torch.int32, device="cuda")
    for which, layer, W, tid, rows, cols, M in cases:
        x = torch.from_numpy(rng.normal(size=(M, cols)).astype(np.float32)).cuda()
        y_ref = torch.zeros((M, rows), dtype=torch.float32, device="cuda")
        y_na = torch.full((M, rows), float("nan"), dtype=torch.float32, device="cuda")
        eng.op_gemv(which, layer, x, y_ref, stream=torch.cuda.current_stream())
        S.ssd_gemv_noalloc(W.data_ptr(), S.SSD_DTYPE_BF16, rows, cols, x.data_ptr(), M,
                           y_na.data_ptr(), err.data_ptr(), stream)
        torch.cuda.synchronize()
        assert int(err.item()) == 0
        a, b = y_na.cpu().numpy(), y_ref.cpu().numpy()
        assert np.isfinite(a).all()
        assert rel_err(a, b) < 1e-5, (which, M, rel_err(a, b))
        # the oracle's fp64 rows of the same generated matrix.  The kernel
        # multiplies bf16 weights by fp32 inputs on the CUDA cores (products
        # exact in an FMA) and rounds each of the K - 1 additions once, so
        # |y - ref| <= gamma_(K-1) sum_k |w_k x_k|, gamma_n = n u / (1 - n u),
        # u = 2^-24, in any summation order.
        rws = _sampled_rows(rows)
        xs = x.cpu().numpy().astype(np.float64)
        for m in sorted({0, M - 1}):
            ref = np.concatenate([oracle.matvec_synth(synth.SEED_WEIGHTS, tid, s.sigma, True, int(r),
                                                      1, xs[m]) for r in rws])
            wabs = np.stack([np.abs(synth.bf16_bits_to_f32(synth.weights_bf16_bits(
                synth.SEED_WEIGHTS, tid, int(r) * cols, cols, s.sigma))).astype(np.float64)
                for r in rws])
            nu = (cols - 1) * 2.0 ** -24
            bound = nu / (1 - nu) * (wabs @ np.abs(xs[m]))
            assert np.all(np.abs(a[m, rws] - ref) <= bound), (which, m)
    # sizes beyond the static scratch are refused before any work is enqueued
    with pytest.raises(S.SsdError) as e:
        S.ssd_gemv_noalloc(dm.lm_head.data_ptr(), S.SSD_DTYPE_BF16, 131072 + 32, s.d_model,
                           x.data_ptr(), 1, y_na.data_ptr(), 0, stream)
    assert e.value.status == S.SSD_ERR_CAPACITY
    with pytest.raises(S.SsdError) as e:
        S.ssd_gemv_noalloc(dm.lm_head.data_ptr(), S.SSD_DTYPE_BF16, s.vocab, s.d_model,
                           x.data_ptr(), 18, y_na.data_ptr(), 0, stream)
    assert e.value.status == S.SSD_ERR_CAPACITY
    eng.close()
