"""The C ABI library builds, loads and exports every function include/moe.h
declares; host-side validation returns the documented status before any
launch (CPU only -- no compute call is made)."""
import ctypes
import os
import re

import pytest
import torch

from paper_2506_23635_gb300 import build as moe_build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "moe.h")


@pytest.fixture(scope="module")
def lib():
    moe_build.build()
    from paper_2506_23635_gb300 import moe
    return moe


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(moe_[a-z_]+)\s*\(", text)))


def test_header_declares_the_five_steps():
    names = declared_functions()
    for n in ("moe_route", "moe_dispatch", "moe_expert_ffn", "moe_combine",
              "moe_layer_forward"):
        assert n in names


def test_every_declared_symbol_is_exported(lib):
    L = lib.lib()
    names = declared_functions()
    assert names, "no declarations parsed"
    for n in names:
        assert hasattr(L, n), f"{n} not exported by libmoe.so"
    assert set(names) == set(lib.EXPORTS)


def test_status_strings(lib):
    for code in range(7):
        s = lib.status_string(code)
        assert s.startswith("MOE_")
    assert "unknown" in lib.status_string(99)


DBRX = dict(d_model=6144, ffn_hidden=10752, n_experts=16, top_k=4)


def test_workspace_size(lib):
    d = lib.dims(**DBRX)
    n1 = lib.workspace_size(d, 1)
    n64 = lib.workspace_size(d, 64)
    n2048 = lib.workspace_size(d, 2048)
    assert 0 < n1 < n64 < n2048
    # the GLU hidden vectors (T*K x F fp32) dominate the decode workspace
    assert n64 >= 64 * 4 * 10752 * 4
    assert lib.workspace_size(d, 0) >= 0


@pytest.mark.parametrize("bad", [
    dict(d_model=6143), dict(d_model=0), dict(ffn_hidden=10), dict(n_experts=0),
    dict(n_experts=257, top_k=4), dict(top_k=0), dict(top_k=17),
])
def test_workspace_size_rejects_bad_dims(lib, bad):
    d = lib.dims(**{**DBRX, **bad})
    with pytest.raises(lib.MoeError) as ei:
        lib.workspace_size(d, 8)
    assert ei.value.status == 1


# Validation returns before anything touches the device, so these calls are
# made with placeholder addresses.  They are skipped where a GPU is present
# (the GPU tests cover the same cases with real tensors) so that a validation
# bug could never launch a kernel on a placeholder address.
no_gpu = pytest.mark.skipif(torch.cuda.is_available(),
                            reason="placeholder addresses only where no GPU exists")

A = ctypes.c_void_p(0x10000)  # 16-byte aligned placeholder
MIS = ctypes.c_void_p(0x10004)  # misaligned placeholder


@no_gpu
def test_route_validation(lib):
    L = lib.lib()
    d = lib.dims(**DBRX)
    r = lambda T, x=A, w=A, lg=None, i=A, g=A: L.moe_route(ctypes.byref(d), T, x, w, lg, i, g, None)
    assert r(1, x=None) == 1
    assert r(1, w=None) == 1
    assert r(1, i=None) == 1
    assert r(1, g=None) == 1
    assert r(1, x=MIS) == 1
    assert r(-1) == 1
    assert r(1 << 21) == 1
    assert r(0) == 0  # nothing to do
    bad = lib.dims(**{**DBRX, "top_k": 17})
    assert L.moe_route(ctypes.byref(bad), 1, A, A, None, A, A, None) == 1
    mixed = lib.dims(**DBRX, w_dtype=torch.bfloat16, x_dtype=torch.float32)
    assert L.moe_route(ctypes.byref(mixed), 1, A, A, None, A, A, None) == 2


@no_gpu
def test_layer_and_ffn_validation(lib):
    L = lib.lib()
    d = lib.dims(**DBRX)
    need = lib.workspace_size(d, 8)
    f = lambda T, ws=A, n=need, x=A: L.moe_layer_forward(ctypes.byref(d), T, x, A, A, A, A,
                                                          None, A, ws, n, None)
    assert f(8, ws=None) == 3
    assert f(8, n=need - 1) == 3
    assert f(8, ws=MIS) == 3
    assert f(8, x=None) == 1
    assert f(0) == 0
    g = lambda T, ws=A, n=need: L.moe_expert_ffn(ctypes.byref(d), T, A, A, A, A, A, A, A, ws, n, None)
    assert g(8, n=0) == 3
    assert L.moe_expert_ffn(ctypes.byref(d), 8, A, None, A, A, A, A, A, A, need, None) == 1
    assert L.moe_combine(ctypes.byref(d), 8, A, A, A, MIS, A, None) == 1
    assert L.moe_combine(ctypes.byref(d), 8, A, None, A, None, A, None) == 1
    assert L.moe_dispatch(ctypes.byref(d), 8, None, A, A, A, A, None) == 1
    assert L.moe_dispatch(ctypes.byref(d), 8, A, None, A, A, A, None) == 1


@no_gpu
def test_expert_range_validation(lib):
    L = lib.lib()
    d = lib.dims(**DBRX)
    need = lib.workspace_size(d, 8)
    f = lambda b, e, T=8, ws=A, n=need, x=A, out=A: L.moe_layer_forward_experts(
        ctypes.byref(d), T, x, A, b, e, A, A, A, None, out, ws, n, None)
    for b, e in ((0, 0), (4, 3), (-1, 4), (0, 17), (16, 16)):
        assert f(b, e) == 1, (b, e)
    assert f(0, 0, T=0) == 1  # the range is checked even when there is no token
    assert f(0, 16, T=0) == 0
    assert f(0, 8, x=None) == 1
    assert f(0, 8, out=MIS) == 1
    assert f(0, 8, ws=None) == 3
    assert f(8, 16, n=need - 1) == 3


@no_gpu
def test_noalloc_validation(lib):
    L = lib.lib()
    d = lib.dims(**DBRX)
    call = lambda T, x=A: L.moe_layer_forward_noalloc(ctypes.byref(d), T, x, A, A, A, A, None, A, None)
    assert call(100000) == 3  # beyond the fixed scratch array
    assert call(-1) == 1
    assert call(0) == 0
    assert call(1, x=None) == 1


def test_noalloc_limit_holds_the_dbrx_decode_range(lib):
    """The no-allocation entry point's scratch array holds the DBRX-shaped
    layer's workspace at every decode batch the header promises (1..64
    tokens); the binding's constant is the header's."""
    hdr = open(os.path.join(ROOT, "include", "moe.h")).read()
    m = re.search(r"#define MOE_NOALLOC_SCRATCH_BYTES \((\d+)u \* 1024u \* 1024u\)", hdr)
    assert m is not None
    assert int(m.group(1)) * 1024 * 1024 == lib.NOALLOC_SCRATCH_BYTES
    d = lib.dims(**DBRX)
    sizes = [lib.workspace_size(d, T) for T in range(1, 65)]
    assert max(sizes) <= lib.NOALLOC_SCRATCH_BYTES, max(sizes)


def test_noalloc_injected_failure(lib):
    """MOE_INJECT_FAILURE reaches the no-allocation entry point by its own
    name (a caller's error path can be tested without a GPU)."""
    code = (
        "import ctypes, sys; sys.path.insert(0, %r)\n"
        "from paper_2506_23635_gb300 import moe\n"
        "L = moe.lib(); d = moe.dims(64, 64, 4, 2)\n"
        "print(L.moe_layer_forward_noalloc(ctypes.byref(d), 4, None, None, None, None, None,\n"
        "                                  None, None, None))\n" % ROOT)
    import subprocess
    import sys
    env = dict(os.environ, MOE_INJECT_FAILURE="moe_layer_forward_noalloc:5")
    out = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, env=env,
                         timeout=120)
    assert out.returncode == 0, out.stderr
    assert int(out.stdout.split()[0]) == 5


def test_launch_count_starts_at_zero_without_launches(lib):
    assert lib.launch_count() >= 0


def test_fault_injection_env(lib):
    """MOE_INJECT_FAILURE makes the named entry return the given status before
    anything is validated or launched (null pointers: nothing could launch)."""
    code = (
        "import ctypes, sys; sys.path.insert(0, %r)\n"
        "from paper_2506_23635_gb300 import moe\n"
        "L = moe.lib(); d = moe.dims(64, 64, 4, 2)\n"
        "print(L.moe_route(ctypes.byref(d), 4, None, None, None, None, None, None),\n"
        "      L.moe_layer_forward(ctypes.byref(d), 4, None, None, None, None, None, None, None,\n"
        "                          None, 0, None))\n" % ROOT)
    import subprocess
    import sys
    env = dict(os.environ, MOE_INJECT_FAILURE="moe_layer_forward:4")
    out = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, env=env,
                         timeout=120)
    assert out.returncode == 0, out.stderr
    route_status, layer_status = map(int, out.stdout.split())
    assert route_status == 1  # not injected: ordinary validation of the nulls
    assert layer_status == 4  # injected MOE_ERR_CUDA
    env["MOE_INJECT_FAILURE"] = "moe_route:5"
    out = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, env=env,
                         timeout=120)
    assert list(map(int, out.stdout.split())) == [5, 1]


@no_gpu
def test_attention_and_decoder_validation(lib):
    """The self-attention and decoder entry points reject bad shapes,
    pointers and workspaces before touching the device."""
    L = lib.lib()
    a = lib.sa_dims(6144, 48, 8)
    n = ctypes.c_size_t(0)
    size = lambda dims, T=1: L.moe_sa_workspace_size(ctypes.byref(dims), T, ctypes.byref(n))
    assert size(a) == 0 and n.value > 0
    one = n.value
    assert size(a, 2048) == 0 and n.value > one
    assert size(lib.sa_dims(6144, 48, 8, head_dim=64)) == 2
    assert size(lib.sa_dims(6144, 48, 7)) == 1          # 7 does not divide 48
    assert size(lib.sa_dims(6144, 48, 4)) == 2          # 12 query heads per group
    assert size(lib.sa_dims(6144, 48, 8, rope_base=1.0)) == 1
    assert size(lib.sa_dims(6100, 48, 8)) == 1          # D not a multiple of 8
    assert size(a, 65537) == 1
    fwd = lambda T, resid=A, ws=A, nb=one, seq=A, n_seq=1, ln=8: L.moe_sa_forward(
        ctypes.byref(a), T, seq, A, n_seq, ln, resid, A, A, A, A, 1e-6, ws, nb, None)
    assert fwd(0) == 0
    assert fwd(1, resid=None) == 1
    assert fwd(1, seq=None) == 1
    assert fwd(1, n_seq=0) == 1
    assert fwd(1, ln=0) == 1
    assert fwd(1, resid=MIS) == 1
    assert fwd(1, ws=None) == 3
    assert fwd(1, nb=one - 1) == 3
    assert L.moe_sa_attend(ctypes.byref(a), 1, A, A, A, 1, 8, A, A, None, A, one, None) == 1
    assert L.moe_sa_qkv(ctypes.byref(a), 1, A, A, A, A, 1, 8, A, A, A, A, 0, None) == 3
    d = lib.dims(**DBRX, out_dtype=torch.float32)
    P = ctypes.c_void_p
    arr = (P * 1)(A)
    dec = lambda dims, attn=a: L.moe_decoder_forward(
        ctypes.byref(attn), ctypes.byref(dims), 1, 1, A, A, 1, 8, A, arr, arr, arr, arr, arr,
        arr, arr, arr, 1e-6, A, 1 << 30, None)
    assert dec(lib.dims(**DBRX)) == 1                   # the residual stream must be fp32
    assert dec(d, attn=lib.sa_dims(4096, 32, 8)) == 1   # widths differ
    assert L.moe_decoder_workspace_size(ctypes.byref(a), ctypes.byref(d), 8, ctypes.byref(n)) == 0
    assert n.value >= one


def test_fault_injection_reaches_the_attention_entries(lib):
    code = (
        "import ctypes, sys; sys.path.insert(0, %r)\n"
        "from paper_2506_23635_gb300 import moe\n"
        "L = moe.lib(); a = moe.sa_dims(256, 4, 2)\n"
        "print(L.moe_sa_forward(ctypes.byref(a), 1, None, None, 1, 8, None, None, None, None,\n"
        "                       None, 1e-6, None, 0, None))\n" % ROOT)
    import subprocess
    import sys
    for env_value, want in (("moe_sa_forward:5", 5), ("moe_sa_qkv:5", 1)):
        env = dict(os.environ, MOE_INJECT_FAILURE=env_value)
        out = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True,
                             env=env, timeout=120)
        assert out.returncode == 0, out.stderr
        assert int(out.stdout) == want
