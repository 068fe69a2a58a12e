"""ssd_gemv_noalloc: the allocation-free matrix-vector product, for callers
that cannot allocate device memory (code running during CUDA-graph capture,
hosts whose framework owns the device memory pool).  It must give the same
products as ssd_op_gemv, the context-based entry point, on consecutive calls
that share its static scratch.  Self-contained, so it passes alone in a fresh
process as well as after the other GPU tests; collected last on purpose."""
import numpy as np
import pytest

from parity import has_gpu, rel_err

pytestmark = [pytest.mark.gpu, pytest.mark.skipif(not has_gpu(), reason="needs a CUDA GPU")]


def test_noalloc_matches_context_gemv_on_consecutive_calls():
    import torch

    from paper_2606_03113_gb300 import ssd as S
    from paper_2606_03113_gb300.runtime import DeviceModel, Engine
    from synth.workloads import LLAMA2_7B, scaled_down

    w = scaled_down(LLAMA2_7B, 2, 1024, 8, 8, 2816, 4096, 32, 8, name="noalloc-small")
    dm = DeviceModel(w.shape)
    eng = Engine(dm, w.max_seq)
    s = w.shape
    cases = [  # (which, layer, W, rows, cols, M): two calls in a row, then a third shape
        (2, 1, dm.layers[1]["w_gate_up"], 2 * s.ffn_dim, s.d_model, 1),
        (3, 0, dm.layers[0]["w_down"], s.d_model, s.ffn_dim, 5),
        (4, 0, dm.lm_head, s.vocab, s.d_model, 17),
    ]
    rng = np.random.default_rng(7)
    stream = torch.cuda.current_stream().cuda_stream
    for which, layer, W, rows, cols, M in cases:
        x = torch.from_numpy(rng.normal(size=(M, cols)).astype(np.float32)).cuda()
        y_ref = torch.zeros((M, rows), dtype=torch.float32, device="cuda")
        y_na = torch.full((M, rows), float("nan"), dtype=torch.float32, device="cuda")
        eng.op_gemv(which, layer, x, y_ref, stream=torch.cuda.current_stream())
        S.ssd_gemv_noalloc(W.data_ptr(), S.SSD_DTYPE_BF16, rows, cols, x.data_ptr(), M,
                           y_na.data_ptr(), stream)
        torch.cuda.synchronize()
        a, b = y_na.cpu().numpy(), y_ref.cpu().numpy()
        assert np.isfinite(a).all()
        assert rel_err(a, b) < 1e-5, (which, M, rel_err(a, b))
    # sizes beyond the static scratch are refused before any work is enqueued
    with pytest.raises(S.SsdError) as e:
        S.ssd_gemv_noalloc(dm.lm_head.data_ptr(), S.SSD_DTYPE_BF16, 131072 + 32, s.d_model,
                           x.data_ptr(), 1, y_na.data_ptr(), stream)
    assert e.value.status == S.SSD_ERR_CAPACITY
    with pytest.raises(S.SsdError) as e:
        S.ssd_gemv_noalloc(dm.lm_head.data_ptr(), S.SSD_DTYPE_BF16, s.vocab, s.d_model,
                           x.data_ptr(), 18, y_na.data_ptr(), stream)
    assert e.value.status == S.SSD_ERR_CAPACITY
    eng.close()
