"""moe_layer_forward_noalloc: the layer for callers that cannot allocate
device memory (a framework that owns every device buffer, a plugin handed
only its inputs and outputs, a runtime that forbids allocation after
start-up).  Its scratch space is a fixed array inside the library.

The entry point is called through the C ABI and its output is compared with
moe_layer_forward's (which takes a caller workspace) on two calls in a row,
within the bf16 layer tolerance the other tests use.  This file is collected
last so that a run stopping at the first failure has run everything else."""
import ctypes

import numpy as np
import pytest
import torch

from paper_2506_23635_gb300 import inputs as gen
from tests.gpu_util import assert_parity, dev, need_gpu, to_numpy

pytestmark = pytest.mark.gpu


def _layer(T, seed):
    sh = gen.LayerShape(512, 1024, 8, 2, "bf16")
    L = gen.host_layer(sh, T, seed)
    return sh, [dev(a, "bf16") for a in (L.x, L.w_r, L.w1, L.v1, L.w2)]


def _call_noalloc(moe, d, x, w_r, w1, v1, w2, out):
    ptr = lambda t: ctypes.c_void_p(t.data_ptr())
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    return moe.lib().moe_layer_forward_noalloc(ctypes.byref(d), x.shape[0], ptr(x), ptr(w_r),
                                               ptr(w1), ptr(v1), ptr(w2), None, ptr(out),
                                               stream)


def test_noalloc_matches_workspace_path_twice():
    need_gpu()
    from paper_2506_23635_gb300 import moe

    sh, (x, w_r, w1, v1, w2) = _layer(24, 41)
    d = moe.dims(sh.d_model, sh.ffn_hidden, sh.n_experts, sh.top_k)
    # second call: different tokens, same weights (the scratch keeps the
    # first call's contents, which must not leak into the second result)
    x2 = dev(gen.host_normal((24, sh.d_model), 1.0, "bf16", 42, "x2"), "bf16")
    for xi in (x, x2):
        want = moe.layer_forward(d, xi, w_r, w1, v1, w2)
        out = torch.empty_like(want)
        assert _call_noalloc(moe, d, xi, w_r, w1, v1, w2, out) == 0
        torch.cuda.synchronize()
        assert moe.get_last_error() == 0
        assert_parity(to_numpy(out), to_numpy(want), "bf16", "noalloc vs workspace path")


def test_noalloc_one_token_twice():
    """One token (the decode path that streams the selected experts' rows):
    two calls in a row against the workspace path."""
    need_gpu()
    from paper_2506_23635_gb300 import moe

    sh, (x, w_r, w1, v1, w2) = _layer(1, 45)
    d = moe.dims(sh.d_model, sh.ffn_hidden, sh.n_experts, sh.top_k)
    x2 = dev(gen.host_normal((1, sh.d_model), 1.0, "bf16", 46, "x2"), "bf16")
    for xi in (x, x2):
        want = moe.layer_forward(d, xi, w_r, w1, v1, w2)
        out = torch.empty_like(want)
        assert _call_noalloc(moe, d, xi, w_r, w1, v1, w2, out) == 0
        torch.cuda.synchronize()
        assert moe.get_last_error() == 0
        assert_parity(to_numpy(out), to_numpy(want), "bf16", "noalloc vs workspace path, T=1")


def test_noalloc_rejects_sizes_beyond_its_scratch():
    need_gpu()
    from paper_2506_23635_gb300 import moe

    sh, (x, w_r, w1, v1, w2) = _layer(4, 43)
    d = moe.dims(sh.d_model, sh.ffn_hidden, sh.n_experts, sh.top_k)
    # the largest T whose workspace fits in the fixed scratch array
    T_max = max(t for t in range(1, 4096) if moe.workspace_size(d, t) <= moe.NOALLOC_SCRATCH_BYTES)
    big = torch.zeros((T_max + 1, sh.d_model), dtype=torch.bfloat16, device="cuda")
    out = torch.empty_like(big)
    assert _call_noalloc(moe, d, big, w_r, w1, v1, w2, out) == 3  # MOE_ERR_WORKSPACE
    xs = big[:T_max]
    xs.copy_(dev(gen.host_normal((T_max, sh.d_model), 1.0, "bf16", 44, "x"), "bf16"))
    want = moe.layer_forward(d, xs, w_r, w1, v1, w2)
    got = torch.empty_like(want)
    assert _call_noalloc(moe, d, xs, w_r, w1, v1, w2, got) == 0
    torch.cuda.synchronize()
    assert_parity(to_numpy(got), to_numpy(want), "bf16", "noalloc at its limit")
