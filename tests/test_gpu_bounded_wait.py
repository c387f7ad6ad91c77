"""The unwind path of a bounded device wait, run on the GPU without a fault:
a wait on an mbarrier that nothing arrives at gives up after the library's
limit, records a timeout in the error word, and the CTA still waits for its
own bulk copy and frees its tensor memory. The host sees UNISVQ_ERR_TIMEOUT
once; afterwards the context, the error word and tensor memory serve a
tcgen05 layer call as before."""
import numpy as np
import pytest

import oracle
import synth

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("no CUDA device", allow_module_level=True)

from paper_2606_10520_gb300 import binding  # noqa: E402


def test_wait_runs_out_and_the_context_stays_usable():
    assert binding.sync_status() == binding.OK
    src = torch.arange(16, dtype=torch.uint8, device="cuda") + 7
    out = torch.full((3,), -5, dtype=torch.int32, device="cuda")
    assert binding.wait_timeout_probe_ptr(src.data_ptr(), out.data_ptr()) == binding.OK
    assert binding.sync_status() == binding.ERR_TIMEOUT
    assert out.tolist() == [0, 1, 7]          # the wait gave up; the own copy landed
    assert binding.sync_status() == binding.OK   # the error word was cleared
    # a layer on the tcgen05 path (it allocates tensor memory) runs and is right
    N, K = 16384, 4096
    codes, A, B = synth.layer_inputs(9, 95, 0, 0, N, K, 2)
    layer = binding.UniSVQLinear(codes, A, B)
    assert layer.query(4)["kernel"] == binding.KERNEL_SKINNY
    xb = synth.activations(9, 95, 1, 4, K)
    x = torch.from_numpy(xb.view(np.int16)).view(torch.bfloat16).cuda()
    y = layer.forward(x)
    assert binding.sync_status() == binding.OK
    rows = np.unique(np.concatenate([synth.rng(9, N, K).choice(N, 64, replace=False), [0, N - 1]]))
    yr, S = oracle.linear(xb, codes[rows], A, B)
    res = oracle.compare(y.float().cpu().numpy().astype(np.float64)[:, rows], yr, S)
    assert res["ok"], res
    layer.close()


def test_wait_probe_rejects_bad_pointers():
    out = torch.zeros(3, dtype=torch.int32, device="cuda")
    src = torch.zeros(32, dtype=torch.uint8, device="cuda")
    assert binding.wait_timeout_probe_ptr(0, out.data_ptr()) == binding.ERR_INVALID_ARG
    assert binding.wait_timeout_probe_ptr(src.data_ptr() + 1, out.data_ptr()) == binding.ERR_INVALID_ARG
