"""Failure detection on the GPU without a fault: a bounded device-side wait
on an mbarrier that nothing completes gives up, the host reads
MOE_ERR_TIMEOUT, and the context keeps working."""
import numpy as np
import pytest
import torch

import oracle
from paper_2506_23635_gb300 import inputs as gen
from tests.gpu_util import assert_parity, dev, need_gpu, to_numpy

pytestmark = pytest.mark.gpu


def test_bounded_wait_times_out_and_context_survives():
    need_gpu()
    from paper_2506_23635_gb300 import moe

    assert moe.get_last_error() == 0
    assert moe.selftest_wait_timeout(20_000_000)  # 20 ms
    assert moe.get_last_error() == 5  # MOE_ERR_TIMEOUT
    assert moe.get_last_error() == 0  # read once, then cleared
    # the context still runs the layer correctly
    L = gen.host_layer(gen.LayerShape(64, 96, 8, 2, "bf16"), 5, 9)
    want, _, _ = oracle.layer_tokens(L.x, L.w_r, L.w1, L.v1, L.w2, "bf16", 2)
    d = moe.dims(64, 96, 8, 2)
    out = moe.layer_forward(d, *[dev(a, "bf16") for a in (L.x, L.w_r, L.w1, L.v1, L.w2)])
    assert moe.get_last_error() == 0
    assert_parity(to_numpy(out), want, "bf16", "after a timeout")


def test_injected_failure_raises_in_binding(monkeypatch):
    need_gpu()
    from paper_2506_23635_gb300 import moe

    monkeypatch.setenv("MOE_INJECT_FAILURE", "moe_layer_forward:4")
    d = moe.dims(64, 64, 4, 2)
    x = torch.zeros((2, 64), dtype=torch.bfloat16, device="cuda")
    w = torch.zeros((64, 4), dtype=torch.bfloat16, device="cuda")
    w1 = torch.zeros((4, 64, 64), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(moe.MoeError) as ei:
        moe.layer_forward(d, x, w, w1, w1, w1)
    assert ei.value.status == 4
