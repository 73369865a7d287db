"""The C-ABI library loads, exports every function include/ress.h declares, and validates its
arguments on the host before any launch (no GPU needed: every call below fails validation
or only computes sizes)."""
import ctypes

import numpy as np
import pytest

import oracle as O
import synth
import __graft_entry__

__graft_entry__._build_module().build()
import paper_2609_35593_gb300 as ress  # noqa: E402

EINVAL, EWORKSPACE, EUNSUPPORTED = -1, -2, -3


def test_every_declared_function_is_exported():
    names = ress.exported_names_in_header()
    assert len(names) >= 12
    for n in names:
        assert hasattr(ress._lib, n), n
    for n in ("ress_score", "ress_restore", "ress_sparse_attn", "ress_forward"):
        assert n in names
    assert ress._lib.ress_abi_version() == 6


@pytest.mark.parametrize("name", list(synth.WORKLOADS))
def test_shape_helpers_match_the_oracle(name):
    wl = synth.WORKLOADS[name]
    d = ress.dims(wl.n_tokens, wl.heads, wl.n_special, wl.d_model)
    assert ress.num_blocks(d) == O.n_blocks(wl.n_tokens)
    assert ress.num_candidates(d) == O.n_candidates(wl.n_tokens, wl.n_special)
    c = wl.budgets()
    nb, nc = wl.n_blocks, wl.n_candidates
    expect = wl.heads * (nc * (int(c[0]) + nb - nc) + (nb - nc) * nb)
    assert ress.csr_capacity(d, c) == expect
    L = ress.workspace_layout(d)
    assert L.total == ress.workspace_bytes(d)
    names = [f[0] for f in ress.WsLayout._fields_]
    offs = sorted(getattr(L, n) for n in names[:names.index("ld")])
    assert all(o % 256 == 0 for o in offs) and len(set(offs)) == len(offs)
    assert L.ld >= nb and L.ld % 32 == 0 and L.words == -(-nb // 32)


def test_csr_capacity_matches_oracle_lists():
    X = {k: synth.bf16_to_f32(v).astype(np.float64) for k, v in synth.make_random_layer(778, 2, 128, 1).items()}
    pooled = O.pool(X["Q"], X["K"], X["V"], 10)
    c = [3, 7]
    sel = O.ress_select(pooled, X["W_o"], c, 1)
    rp, ci = O.csr_from_selection(sel, 2, pooled.nb)
    assert ress.csr_capacity(ress.dims(778, 2, 10, 128), c) == ci.size


@pytest.mark.parametrize("field,value,code", [
    ("head_dim", 128, EUNSUPPORTED), ("block", 128, EUNSUPPORTED), ("n_heads", 0, EUNSUPPORTED),
    ("n_heads", 33, EUNSUPPORTED), ("n_tokens", 0, EINVAL), ("n_special", -1, EINVAL),
    ("d_model", 0, EINVAL), ("n_tokens", 64 * 4096 + 1, EUNSUPPORTED)])
def test_invalid_dims_are_rejected(field, value, code):
    d = ress.dims(2748, 4, 10, 256)
    setattr(d, field, value)
    assert ress._lib.ress_workspace_bytes(ctypes.byref(d)) == 0
    L = ress.WsLayout()
    assert ress._lib.ress_workspace_layout(ctypes.byref(d), ctypes.byref(L)) == code
    assert ress._lib.ress_last_error()


def _fake(addr):
    return ctypes.c_void_p(addr)


def test_score_validation_happens_before_launch():
    d = ress.dims(2748, 4, 10, 256)
    c = (ctypes.c_int32 * 4)(21, 21, 21, 21)
    ws_n = ress.workspace_bytes(d)
    A = 1 << 40  # never dereferenced: every call below fails validation
    lib = ress._lib
    args = lambda Q=A, c=c, ws=A, n=ws_n: (ctypes.byref(d), _fake(Q), _fake(A), _fake(A), _fake(A),
                                           ctypes.cast(c, ctypes.c_void_p), _fake(ws), n, None)
    assert lib.ress_score(*args(Q=0)) == EINVAL                  # NULL
    assert lib.ress_score(*args(Q=A + 2)) == EINVAL              # not 16-byte aligned
    assert lib.ress_score(*args(ws=A + 16)) == EINVAL            # workspace not 256-aligned
    assert lib.ress_score(*args(n=ws_n - 1)) == EWORKSPACE
    bad = (ctypes.c_int32 * 4)(21, 0, 21, 21)
    assert lib.ress_score(*args(c=bad)) == EINVAL                # c_h < 1
    big = (ctypes.c_int32 * 4)(21, 43, 21, 21)
    assert lib.ress_score(*args(c=big)) == EINVAL                # c_h > |P| = 42
    assert b"c_h[1]" in lib.ress_last_error()


def test_restore_and_attention_validation():
    d = ress.dims(2748, 4, 10, 256)
    c = (ctypes.c_int32 * 4)(21, 21, 21, 21)
    cp = ctypes.cast(c, ctypes.c_void_p)
    ws_n = ress.workspace_bytes(d)
    cap = ress.csr_capacity(d, [21] * 4)
    A = 1 << 40
    lib = ress._lib
    assert lib.ress_restore(ctypes.byref(d), cp, -1, 0.5, _fake(A), ws_n, _fake(A), _fake(A), cap,
                            None, None, None) == EINVAL
    assert lib.ress_restore(ctypes.byref(d), cp, 3, 1.5, _fake(A), ws_n, _fake(A), _fake(A), cap,
                            None, None, None) == EINVAL
    assert lib.ress_restore(ctypes.byref(d), cp, 3, 0.5, _fake(A), ws_n, _fake(A), _fake(A), cap - 1,
                            None, None, None) == EWORKSPACE
    assert lib.ress_restore(ctypes.byref(d), cp, 3, 0.5, _fake(A), ws_n, _fake(A), _fake(A + 2), cap,
                            None, None, None) == EINVAL
    assert lib.ress_sparse_attn(ctypes.byref(d), _fake(A), _fake(A), _fake(A), _fake(A), _fake(A), cap,
                                _fake(0), _fake(A), ws_n, None) == EINVAL
    assert lib.ress_sparse_attn(ctypes.byref(d), _fake(A), _fake(A), _fake(A), _fake(A), _fake(A), -1,
                                _fake(A), _fake(A), ws_n, None) == EINVAL
    assert lib.ress_forward(ctypes.byref(d), _fake(A), _fake(A), _fake(A), _fake(A), cp, 3, 0.5,
                            _fake(A), ws_n, _fake(A), _fake(A), cap - 1, _fake(A), None, None) == EWORKSPACE


def test_binding_refuses_host_tensors():
    torch = pytest.importorskip("torch")
    d = ress.dims(2748, 4, 10, 256)
    x = torch.zeros(2748, 4, 64, dtype=torch.bfloat16)
    with pytest.raises(ValueError):
        ress.sparse_attn(d, x, x, x, torch.zeros(3, dtype=torch.int32), torch.zeros(3, dtype=torch.int32),
                         x, torch.zeros(8, dtype=torch.uint8))


def test_launch_counter_is_exported_and_monotone():
    a = ress.kernel_launches()
    assert a >= 0 and ress.kernel_launches() >= a


def test_variant_names_map_to_the_header_values():
    v = ress.variant("random", "full", seed=9)
    assert (v.key, v.direction, v.seed) == (2, 2, 9)
    assert ress.variant(cdf=0.75).cdf == 0.75 and ctypes.sizeof(ress.Variant) == 24
    assert (ress.variant().key, ress.variant().direction) == (0, 0)


def test_wait_selftest_validates_before_launch():
    """The bounded-wait self-test rejects a bad limit or workspace on the host."""
    ptr = ctypes.c_void_p(1 << 20)
    assert ress._lib.ress_wait_selftest(ptr, 4096, 0, None) == EINVAL
    assert ress._lib.ress_wait_selftest(ptr, 4096, 100001, None) == EINVAL
    assert ress._lib.ress_wait_selftest(ptr, 16, 1000, None) == EWORKSPACE
    assert ress._lib.ress_wait_selftest(None, 4096, 1000, None) == EINVAL


def test_cdf_variant_capacity_and_validation():
    """A CDF threshold may keep every block: the capacity is H * nq * nb.  Out-of-range
    thresholds, a maximising direction, a nonzero reserved field and restoration rounds
    are rejected on the host (fake device pointers: nothing is launched)."""
    wl = synth.WORKLOADS["vggt_v8"]
    c = wl.budgets()
    for qb in (64, 128):
        d = ress.dims(wl.n_tokens, wl.heads, wl.n_special, wl.d_model, qb)
        nq, nb = ress.num_query_blocks(d), ress.num_blocks(d)
        assert ress.csr_capacity(d, c, ress.variant(cdf=0.9)) == wl.heads * nq * nb
        assert ress.csr_capacity(d, c, ress.variant(key="probability")) == ress.csr_capacity(d, c)
    d = ress.dims(wl.n_tokens, wl.heads, wl.n_special, wl.d_model)
    bad = [ress.variant(cdf=1.5), ress.variant(cdf=-0.1), ress.variant(maximize="swap", cdf=0.5),
           ress.variant(cdf=float("nan"))]
    r = ress.variant(cdf=0.5)
    r.reserved = 1
    bad.append(r)
    for v in bad:
        with pytest.raises(ress.RessError):
            ress.csr_capacity(d, c, v)
    L = ress.workspace_layout(d)
    cap = ress.csr_capacity(d, c, ress.variant(cdf=0.9))
    ptr = ctypes.c_void_p(1 << 20)
    budgets = (ctypes.c_int32 * len(c))(*[int(x) for x in c])
    def restore(v, rounds, capacity):
        return ress._lib.ress_restore_variant(ctypes.byref(d), ctypes.cast(budgets, ctypes.c_void_p),
                                              rounds, 0.5, ctypes.byref(v), ptr, L.total, ptr,
                                              ptr, capacity, None, None, None)
    assert restore(ress.variant(cdf=0.9), 1, cap) == EINVAL
    assert restore(ress.variant(cdf=0.9), 0, cap - 1) == EWORKSPACE
    assert restore(ress.variant(cdf=2.0), 0, cap) == EINVAL
    assert L.kcount > 0


@pytest.mark.parametrize("name", ["tiny_v2", "vggt_v8", "vggt_v32"])
def test_query_block_128_shapes(name):
    """On the paper's grid the selection and CSR rows are 128-token query blocks: their
    count, the sparsified ones, and the CSR capacity match the oracle's row structure."""
    wl = synth.WORKLOADS[name]
    d = ress.dims(wl.n_tokens, wl.heads, wl.n_special, wl.d_model, 128)
    nq = -(-wl.n_tokens // 128)
    nqc = (wl.n_tokens - wl.n_special) // 128
    assert ress.num_query_blocks(d) == nq and ress.num_query_candidates(d) == nqc
    nb, nc = ress.num_blocks(d), ress.num_candidates(d)
    c = wl.budgets()
    assert ress.csr_capacity(d, c) == sum(nqc * (ch + nb - nc) + (nq - nqc) * nb for ch in c)
    L = ress.workspace_layout(d)
    assert L.total == ress.workspace_bytes(d)
    d64 = ress.dims(wl.n_tokens, wl.heads, wl.n_special, wl.d_model)
    assert ress.workspace_bytes(d) < ress.workspace_bytes(d64)  # half the selection rows


def test_query_block_must_be_64_or_128():
    d = ress.dims(1000, 2, 0, 128, 96)
    assert ress.num_query_blocks(d) == -1
