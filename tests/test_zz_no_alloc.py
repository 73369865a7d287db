"""The allocation-free attention entry point (ress_sparse_attn_noalloc) gives the same output
as ress_sparse_attn with a caller-provided workspace.

It exists for callers that cannot allocate device memory when they call in (a framework
that owns all device memory through its own pool, a runtime that reserves everything at
start-up); its scratch is a fixed device array inside the library.  This file is collected
last so that a run stopping at the first failure has run every other test first; it also
passes on its own in a fresh process.
"""
import ctypes

import pytest

import synth

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("no CUDA device", allow_module_level=True)

import gpu_harness as G  # noqa: E402


def _call(layer, O, col_capacity=None, wait=1):
    """ress_sparse_attn_noalloc through the C ABI (ctypes, no binding wrapper)."""
    lib = layer.ress._lib
    b = layer.buf
    p = lambda t: ctypes.c_void_p(t.data_ptr())
    cap = b.col_idx.numel() if col_capacity is None else col_capacity
    return lib.ress_sparse_attn_noalloc(ctypes.byref(layer.d), p(layer.Q), p(layer.K), p(layer.V),
                                        p(b.row_ptr), p(b.col_idx), cap, p(O), wait,
                                        ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))


@pytest.mark.parametrize("name", ["tiny_v2", "vggt_v8"])
def test_noalloc_matches_workspace_entry_point(name):
    wl = synth.WORKLOADS[name]
    layer = G.Layer(synth.make_inputs(wl), wl.n_special, wl.budgets(), wl.rounds, wl.rho).run()
    ref = layer.buf.O.float()
    for call in range(2):  # the shared scratch keeps the previous call's contents
        O = torch.full_like(layer.buf.O, float("nan"))
        rc = _call(layer, O)
        assert rc == 0, layer.ress._lib.ress_last_error()
        torch.cuda.synchronize()
        got = O.float()
        assert not torch.isnan(got).any()
        diff = (got - ref).abs()
        assert diff.max().item() <= G.ATT_MAX_ABS, (call, diff.max().item())
        assert diff.sum().item() / ref.abs().sum().item() <= G.ATT_MEAN_REL
        # same kernel, same arithmetic: the two entry points agree bit for bit
        assert torch.equal(O.view(torch.int16), layer.buf.O.view(torch.int16))


def test_noalloc_rejects_requests_beyond_its_scratch():
    wl = synth.WORKLOADS["tiny_v2"]
    layer = G.Layer(synth.make_inputs(wl), wl.n_special, wl.budgets(), wl.rounds, wl.rho).run()
    O = torch.empty_like(layer.buf.O)
    rc = _call(layer, O, col_capacity=(4 << 20) // 4)
    assert rc == -2  # RESS_EWORKSPACE, nothing launched
    msg = layer.ress._lib.ress_last_error().decode()
    assert "scratch" in msg and "ress_sparse_attn" in msg


def test_noalloc_asynchronous_call_then_waiting_call():
    """wait == 0 returns without synchronising; a following call with wait != 0 on the same
    stream gives the same bits (the shared scratch is rewritten by every call)."""
    wl = synth.WORKLOADS["tiny_v2"]
    layer = G.Layer(synth.make_inputs(wl), wl.n_special, wl.budgets(), wl.rounds, wl.rho).run()
    O1 = torch.full_like(layer.buf.O, float("nan"))
    O2 = torch.full_like(layer.buf.O, float("nan"))
    assert _call(layer, O1, wait=0) == 0, layer.ress._lib.ress_last_error()
    assert _call(layer, O2, wait=1) == 0, layer.ress._lib.ress_last_error()
    torch.cuda.synchronize()
    assert torch.equal(O1.view(torch.int16), layer.buf.O.view(torch.int16))
    assert torch.equal(O2.view(torch.int16), layer.buf.O.view(torch.int16))


def test_noalloc_device_error_is_reported_once():
    """A CSR entry out of range (caught by the union kernel's own bounds check, no memory
    access past the arrays) is reported as RESS_EDEVICE by the waiting call, and the next
    call on a good CSR returns RESS_OK: the recorded failure was cleared."""
    wl = synth.WORKLOADS["tiny_v2"]
    layer = G.Layer(synth.make_inputs(wl), wl.n_special, wl.budgets(), wl.rounds, wl.rho).run()
    good = layer.buf.col_idx.clone()
    layer.buf.col_idx[5] = layer.nb + 100
    O = torch.empty_like(layer.buf.O)
    assert _call(layer, O, wait=1) == -6  # RESS_EDEVICE
    layer.buf.col_idx.copy_(good)
    assert _call(layer, O, wait=1) == 0, layer.ress._lib.ress_last_error()
    assert torch.equal(O.view(torch.int16), layer.buf.O.view(torch.int16))
