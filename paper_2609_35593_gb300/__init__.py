"""Python binding of the ReSS C-ABI library (libress.so).

Argument marshalling only: every function here checks the tensors it is given (device,
dtype, contiguity), passes raw pointers and the current CUDA stream to the function of the
same name in include/ress.h, and turns a negative return code into RessError.  All
arithmetic runs in the library's CUDA kernels; if libress.so is missing the import fails
(build it with `python -m paper_2609_35593_gb300.build` or __graft_entry__.build()).
"""
from __future__ import annotations

import ctypes
import os
import re

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libress.so")
HEADER = os.path.join(os.path.dirname(HERE), "include", "ress.h")

if not os.path.exists(LIB_PATH):
    raise ImportError(f"{LIB_PATH} is not built; run paper_2609_35593_gb300.build.build() first")
_lib = ctypes.CDLL(LIB_PATH)

HEAD_DIM = 64
BLOCK = 64
MAX_HEADS = 32
MAX_BLOCKS = 4096

STATUS = {0: "RESS_OK", -1: "RESS_EINVAL", -2: "RESS_EWORKSPACE", -3: "RESS_EUNSUPPORTED",
          -4: "RESS_ECUDA", -5: "RESS_ETIMEOUT", -6: "RESS_EDEVICE"}


class RessError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"{STATUS.get(code, code)}: {msg}")
        self.code = code


class Dims(ctypes.Structure):
    """ress_dims: one global-attention layer."""
    _fields_ = [("n_tokens", ctypes.c_int32), ("n_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("block", ctypes.c_int32),
                ("n_special", ctypes.c_int32), ("d_model", ctypes.c_int32),
                ("q_block", ctypes.c_int32)]


class Variant(ctypes.Structure):
    """ress_variant: selection variant of the ablations (key: 0 drift, 1 probability,
    2 random; direction: 0 minimise, 1 restoration maximises, 2 everything maximises;
    cdf: 0, or the threshold tau of the CDF rule, which keeps further candidates until the
    kept pooled mass reaches tau)."""
    _fields_ = [("key", ctypes.c_int32), ("direction", ctypes.c_int32), ("seed", ctypes.c_uint64),
                ("cdf", ctypes.c_float), ("reserved", ctypes.c_int32)]


_KEYS = {"drift": 0, "probability": 1, "random": 2}
_DIRECTIONS = {"none": 0, "swap": 1, "full": 2}


def variant(key: str = "drift", maximize: str = "none", seed: int = 0, cdf: float = 0.0) -> Variant:
    """A ress_variant from names: key in {drift, probability, random}, maximize in
    {none, swap, full}; cdf the CDF threshold tau (0: off)."""
    return Variant(_KEYS[key], _DIRECTIONS[maximize], seed, cdf, 0)


class WsLayout(ctypes.Structure):
    """ress_ws_layout: byte offsets of the workspace arrays."""
    _fields_ = [(n, ctypes.c_int64) for n in
                ("status", "counter", "qbar", "kbar", "vbar", "ztil", "ytil", "gtil", "P", "q", "t",
                 "K", "G", "J", "Jbest", "J0", "dmask", "bmask", "plen", "asplit", "ksplit", "zsplit",
                 "cdot", "ny", "nz", "lstat", "kcount", "prow", "ld", "words", "total")]


_c = ctypes
_P = _c.c_void_p
_SIGS = {
    "ress_last_error": (_c.c_char_p, []),
    "ress_abi_version": (_c.c_int32, []),
    "ress_kernel_launches": (_c.c_uint64, []),
    "ress_num_blocks": (_c.c_int32, [_c.POINTER(Dims)]),
    "ress_num_candidates": (_c.c_int32, [_c.POINTER(Dims)]),
    "ress_num_query_blocks": (_c.c_int32, [_c.POINTER(Dims)]),
    "ress_num_query_candidates": (_c.c_int32, [_c.POINTER(Dims)]),
    "ress_workspace_bytes": (_c.c_size_t, [_c.POINTER(Dims)]),
    "ress_workspace_layout": (_c.c_int, [_c.POINTER(Dims), _c.POINTER(WsLayout)]),
    "ress_csr_capacity": (_c.c_int64, [_c.POINTER(Dims), _P]),
    "ress_csr_capacity_variant": (_c.c_int64, [_c.POINTER(Dims), _P, _c.POINTER(Variant)]),
    "ress_prepare_wo": (_c.c_int, [_c.POINTER(Dims), _P, _P, _P]),
    "ress_score": (_c.c_int, [_c.POINTER(Dims), _P, _P, _P, _P, _P, _P, _c.c_size_t, _P]),
    "ress_restore": (_c.c_int, [_c.POINTER(Dims), _P, _c.c_int32, _c.c_float, _P, _c.c_size_t,
                                _P, _P, _c.c_int64, _P, _P, _P]),
    "ress_sparse_attn": (_c.c_int, [_c.POINTER(Dims), _P, _P, _P, _P, _P, _c.c_int64, _P, _P,
                                    _c.c_size_t, _P]),
    "ress_sparse_attn_f32": (_c.c_int, [_c.POINTER(Dims), _P, _P, _P, _P, _P, _c.c_int64, _P, _P,
                                        _c.c_size_t, _P]),
    "ress_forward": (_c.c_int, [_c.POINTER(Dims), _P, _P, _P, _P, _P, _c.c_int32, _c.c_float, _P,
                                _c.c_size_t, _P, _P, _c.c_int64, _P, _P, _P]),
    "ress_forward_host": (_c.c_int, [_c.POINTER(Dims), _P, _P, _P, _P, _P, _P, _P, _P, _P, _P,
                                     _c.c_int32, _c.c_float, _P, _c.c_size_t, _P, _P, _c.c_int64,
                                     _P, _P]),
    "ress_status": (_c.c_int, [_P, _P]),
    "ress_wait_selftest": (_c.c_int, [_P, _c.c_size_t, _c.c_uint32, _P]),
    "ress_score_variant": (_c.c_int, [_c.POINTER(Dims), _P, _P, _P, _P, _P, _c.POINTER(Variant), _P,
                                      _c.c_size_t, _P]),
    "ress_restore_variant": (_c.c_int, [_c.POINTER(Dims), _P, _c.c_int32, _c.c_float,
                                        _c.POINTER(Variant), _P, _c.c_size_t, _P, _P, _c.c_int64,
                                        _P, _P, _P]),
    "ress_out_proj": (_c.c_int, [_c.POINTER(Dims), _P, _P, _P, _P, _P, _c.c_size_t, _P]),
    "ress_token_drift": (_c.c_int, [_c.POINTER(Dims), _P, _P, _P, _P, _P, _c.c_size_t, _P]),
    "ress_sparse_attn_noalloc": (_c.c_int, [_c.POINTER(Dims), _P, _P, _P, _P, _P, _c.c_int64, _P,
                                            _c.c_int32, _P]),
}
for _name, (_res, _args) in _SIGS.items():
    _f = getattr(_lib, _name)
    _f.restype = _res
    _f.argtypes = _args


def exported_names_in_header(path: str = HEADER) -> list[str]:
    """Function names declared in include/ress.h."""
    text = open(path).read()
    return sorted(set(re.findall(r"\b(ress_[a-z_]+)\s*\(", text)))


def _check(rc: int):
    if rc != 0:
        raise RessError(rc, _lib.ress_last_error().decode())


def dims(n_tokens: int, n_heads: int, n_special: int, d_model: int, q_block: int = 64) -> Dims:
    """ress_dims; q_block 128 selects the paper's grid of 128-token query blocks."""
    return Dims(n_tokens, n_heads, HEAD_DIM, BLOCK, n_special, d_model, q_block)


def kernel_launches() -> int:
    """ress_kernel_launches: kernels this library has enqueued so far in the process."""
    return int(_lib.ress_kernel_launches())


def num_blocks(d: Dims) -> int:
    return _lib.ress_num_blocks(_c.byref(d))


def num_candidates(d: Dims) -> int:
    return _lib.ress_num_candidates(_c.byref(d))


def num_query_blocks(d: Dims) -> int:
    return _lib.ress_num_query_blocks(_c.byref(d))


def num_query_candidates(d: Dims) -> int:
    return _lib.ress_num_query_candidates(_c.byref(d))


def workspace_bytes(d: Dims) -> int:
    n = _lib.ress_workspace_bytes(_c.byref(d))
    if n == 0:
        raise RessError(-1, _lib.ress_last_error().decode())
    return n


def workspace_layout(d: Dims) -> WsLayout:
    L = WsLayout()
    _check(_lib.ress_workspace_layout(_c.byref(d), _c.byref(L)))
    return L


def _budget_array(c_h):
    arr = (_c.c_int32 * len(c_h))(*[int(c) for c in c_h])
    return arr


def csr_capacity(d: Dims, c_h, variant: Variant = None) -> int:
    """col_idx entries the restore may write (every row kept whole under a CDF threshold)."""
    if variant is None:
        n = _lib.ress_csr_capacity(_c.byref(d), _c.cast(_budget_array(c_h), _P))
    else:
        n = _lib.ress_csr_capacity_variant(_c.byref(d), _c.cast(_budget_array(c_h), _P),
                                           _c.byref(variant))
    if n < 0:
        raise RessError(-1, _lib.ress_last_error().decode())
    return n


# ---- tensors -> pointers -------------------------------------------------------------
def _torch():
    import torch
    return torch


def _dev(t, dtypes, name):
    """Device pointer of a contiguous CUDA tensor (None -> NULL)."""
    if t is None:
        return None
    torch = _torch()
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor")
    if t.device.type != "cuda":
        raise ValueError(f"{name} must live on a CUDA device")
    if dtypes and t.dtype not in dtypes:
        raise TypeError(f"{name} has dtype {t.dtype}, expected one of {dtypes}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return _c.c_void_p(t.data_ptr())


def _host(t, dtypes, name):
    """Host pointer of a contiguous CPU tensor (page-locked for asynchronous copies)."""
    torch = _torch()
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor")
    if t.device.type != "cpu":
        raise ValueError(f"{name} must live in host memory")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if dtypes is not None and t.dtype not in dtypes:
        raise TypeError(f"{name} has dtype {t.dtype}, expected one of {dtypes}")
    return _c.c_void_p(t.data_ptr())


def _stream(stream):
    torch = _torch()
    s = torch.cuda.current_stream() if stream is None else stream
    return _c.c_void_p(s.cuda_stream)


def _bf16():
    torch = _torch()
    return (torch.bfloat16, torch.uint16, torch.int16)


def prepare_wo(d: Dims, W_o, F, stream=None):
    torch = _torch()
    _check(_lib.ress_prepare_wo(_c.byref(d), _dev(W_o, _bf16(), "W_o"), _dev(F, (torch.float32,), "F"),
                                _stream(stream)))


def score(d: Dims, Q, K, V, F, c_h, ws, stream=None, variant: Variant = None):
    """ress_score, or ress_score_variant when a Variant is given."""
    torch = _torch()
    args = (_dev(Q, _bf16(), "Q"), _dev(K, _bf16(), "K"), _dev(V, _bf16(), "V"),
            _dev(F, (torch.float32,), "F"), _c.cast(_budget_array(c_h), _P))
    tail = (_dev(ws, None, "ws"), ws.numel() * ws.element_size(), _stream(stream))
    if variant is None:
        _check(_lib.ress_score(_c.byref(d), *args, *tail))
    else:
        _check(_lib.ress_score_variant(_c.byref(d), *args, _c.byref(variant), *tail))


def restore(d: Dims, c_h, rounds: int, rho: float, ws, row_ptr, col_idx, J_best=None,
            drop_mask=None, stream=None, variant: Variant = None):
    """ress_restore, or ress_restore_variant when a Variant is given."""
    torch = _torch()
    head = (_c.cast(_budget_array(c_h), _P), int(rounds), float(rho))
    tail = (_dev(ws, None, "ws"), ws.numel() * ws.element_size(),
            _dev(row_ptr, (torch.int32,), "row_ptr"), _dev(col_idx, (torch.int32,), "col_idx"),
            col_idx.numel(), _dev(J_best, (torch.float32,), "J_best"),
            _dev(drop_mask, (torch.int32, torch.uint32), "drop_mask"), _stream(stream))
    if variant is None:
        _check(_lib.ress_restore(_c.byref(d), *head, *tail))
    else:
        _check(_lib.ress_restore_variant(_c.byref(d), *head, _c.byref(variant), *tail))


def sparse_attn(d: Dims, Q, K, V, row_ptr, col_idx, O, ws, stream=None):
    torch = _torch()
    _check(_lib.ress_sparse_attn(_c.byref(d), _dev(Q, _bf16(), "Q"), _dev(K, _bf16(), "K"),
                                 _dev(V, _bf16(), "V"), _dev(row_ptr, (torch.int32,), "row_ptr"),
                                 _dev(col_idx, (torch.int32,), "col_idx"), col_idx.numel(),
                                 _dev(O, _bf16(), "O"), _dev(ws, None, "ws"),
                                 ws.numel() * ws.element_size(), _stream(stream)))


def out_proj(d: Dims, O, W_o, x, y, ws, stream=None):
    """ress_out_proj: y = x + O W_o^T (x None: y = O W_o^T); bf16 tensors."""
    _check(_lib.ress_out_proj(_c.byref(d), _dev(O, _bf16(), "O"), _dev(W_o, _bf16(), "W_o"),
                              _dev(x, _bf16(), "x"), _dev(y, _bf16(), "y"), _dev(ws, None, "ws"),
                              ws.numel() * ws.element_size(), _stream(stream)))


def token_drift(d: Dims, O_a, O_b, W_o, drift, ws, stream=None):
    """ress_token_drift: drift[b] = sum over block b's tokens of ||W_o (O_a - O_b)||^2."""
    torch = _torch()
    _check(_lib.ress_token_drift(_c.byref(d), _dev(O_a, _bf16(), "O_a"), _dev(O_b, _bf16(), "O_b"),
                                 _dev(W_o, _bf16(), "W_o"), _dev(drift, (torch.float32,), "drift"),
                                 _dev(ws, None, "ws"), ws.numel() * ws.element_size(),
                                 _stream(stream)))


def sparse_attn_f32(d: Dims, Q, K, V, row_ptr, col_idx, O, ws, stream=None):
    """ress_sparse_attn with a float32 output tensor O [N, H, 64]."""
    torch = _torch()
    _check(_lib.ress_sparse_attn_f32(_c.byref(d), _dev(Q, _bf16(), "Q"), _dev(K, _bf16(), "K"),
                                     _dev(V, _bf16(), "V"), _dev(row_ptr, (torch.int32,), "row_ptr"),
                                     _dev(col_idx, (torch.int32,), "col_idx"), col_idx.numel(),
                                     _dev(O, (torch.float32,), "O"), _dev(ws, None, "ws"),
                                     ws.numel() * ws.element_size(), _stream(stream)))


def forward(d: Dims, Q, K, V, F, c_h, rounds: int, rho: float, ws, row_ptr, col_idx, O,
            J_best=None, stream=None):
    torch = _torch()
    _check(_lib.ress_forward(_c.byref(d), _dev(Q, _bf16(), "Q"), _dev(K, _bf16(), "K"),
                             _dev(V, _bf16(), "V"), _dev(F, (torch.float32,), "F"),
                             _c.cast(_budget_array(c_h), _P), int(rounds), float(rho),
                             _dev(ws, None, "ws"), ws.numel() * ws.element_size(),
                             _dev(row_ptr, (torch.int32,), "row_ptr"),
                             _dev(col_idx, (torch.int32,), "col_idx"), col_idx.numel(),
                             _dev(O, _bf16(), "O"), _dev(J_best, (torch.float32,), "J_best"),
                             _stream(stream)))


def forward_host(d: Dims, Q_host, K_host, V_host, O_host, Q_dev, K_dev, V_dev, O_dev, F, c_h,
                 rounds: int, rho: float, ws, row_ptr, col_idx, J_best=None, stream=None):
    """ress_forward_host: copies of Q, K, V in, the forward, the copy of O out, all enqueued
    on `stream` (host tensors should be pinned)."""
    torch = _torch()
    b = _bf16()
    _check(_lib.ress_forward_host(_c.byref(d), _host(Q_host, b, "Q_host"), _host(K_host, b, "K_host"),
                                  _host(V_host, b, "V_host"), _host(O_host, b, "O_host"),
                                  _dev(Q_dev, b, "Q_dev"), _dev(K_dev, b, "K_dev"),
                                  _dev(V_dev, b, "V_dev"), _dev(O_dev, b, "O_dev"),
                                  _dev(F, (torch.float32,), "F"), _c.cast(_budget_array(c_h), _P),
                                  int(rounds), float(rho), _dev(ws, None, "ws"),
                                  ws.numel() * ws.element_size(),
                                  _dev(row_ptr, (torch.int32,), "row_ptr"),
                                  _dev(col_idx, (torch.int32,), "col_idx"), col_idx.numel(),
                                  _dev(J_best, (torch.float32,), "J_best"), _stream(stream)))


def sparse_attn_noalloc(d: Dims, Q, K, V, row_ptr, col_idx, O, wait: bool = True, stream=None):
    """ress_sparse_attn without a workspace: scratch is the library's built-in device array
    (see include/ress.h for its size limit and the sharing rules)."""
    torch = _torch()
    _check(_lib.ress_sparse_attn_noalloc(_c.byref(d), _dev(Q, _bf16(), "Q"), _dev(K, _bf16(), "K"),
                                         _dev(V, _bf16(), "V"), _dev(row_ptr, (torch.int32,), "row_ptr"),
                                         _dev(col_idx, (torch.int32,), "col_idx"), col_idx.numel(),
                                         _dev(O, _bf16(), "O"), 1 if wait else 0, _stream(stream)))


def wait_selftest(ws, limit_us: int = 20000, stream=None):
    """ress_wait_selftest: a bounded wait that nothing completes, recorded as RESS_ETIMEOUT in
    the workspace status word (read it with status())."""
    _check(_lib.ress_wait_selftest(_dev(ws, None, "ws"), ws.numel() * ws.element_size(),
                                   int(limit_us), _stream(stream)))


def status(ws, stream=None):
    """Synchronise, read and clear the device status word; raise on a device-side error."""
    _check(_lib.ress_status(_dev(ws, None, "ws"), _stream(stream)))


class Buffers:
    """Device buffers of one layer shape (workspace, F, CSR, output), allocated by torch."""

    def __init__(self, d: Dims, c_h, device="cuda", variant: Variant = None):
        torch = _torch()
        self.d = d
        self.c_h = [int(c) for c in c_h]
        self.nb = num_blocks(d)
        self.nq = num_query_blocks(d)
        H = d.n_heads
        self.ws = torch.zeros(workspace_bytes(d), dtype=torch.uint8, device=device)
        self.F = torch.zeros(H, 64, 64, dtype=torch.float32, device=device)
        self.row_ptr = torch.zeros(H * self.nq + 1, dtype=torch.int32, device=device)
        self.col_idx = torch.zeros(csr_capacity(d, c_h, variant), dtype=torch.int32, device=device)
        self.O = torch.zeros(d.n_tokens, H, 64, dtype=torch.bfloat16, device=device)
        self.J_best = torch.zeros(H * self.nq, dtype=torch.float32, device=device)
        self.layout = workspace_layout(d)

    def ws_view(self, name: str, dtype=None, shape=None):
        """A typed view of one workspace array (see WsLayout)."""
        torch = _torch()
        L = self.layout
        names = [f[0] for f in WsLayout._fields_]
        off = getattr(L, name)
        order = sorted(getattr(L, n) for n in names[:names.index("ld")])
        nxt = min([o for o in order if o > off] + [L.total])
        dtype = dtype or torch.float32
        raw = self.ws[off:nxt]
        t = raw.view(dtype)
        if shape is not None:
            n = 1
            for s in shape:
                n *= s
            t = t[:n].view(*shape)
        return t
