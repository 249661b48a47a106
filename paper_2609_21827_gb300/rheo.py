"""ctypes binding of ``librheo.so`` (include/rheo.h): argument marshalling only.

Every step of the path runs in the library's CUDA kernels.  PyTorch provides
device memory and the current stream.  There is no CPU fallback: importing
works anywhere, but the first call raises if the library has not been built.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass

import torch

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "librheo.so")

RHEO_F32, RHEO_BF16 = 0, 1
RHEO_OK, RHEO_EINVAL, RHEO_ELAUNCH, RHEO_ETOOLARGE = 0, -1, -2, -3
VERIFY_RHEO, VERIFY_RRSW, VERIFY_ONEHOT = 0, 1, 2
STATUS_BAD_LOGIT, STATUS_EMPTY_ROW, STATUS_BAD_TEMPERATURE, STATUS_INTERNAL = 1, 2, 4, 8
SLOT_ROOT, SLOT_LEAD, SLOT_SAMPLED, SLOT_FILL = 0, 1, 2, 3

EXPORTS = ("rheo_sizes", "rheo_workspace_init", "rheo_expand", "rheo_prune", "rheo_verify", "rheo_verify_static",
           "rheo_tree_attention", "rheo_verify_variant", "rheo_verify_full",
           "rheo_get_status")


class RheoError(RuntimeError):
    pass


class _Config(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int32), ("vocab", ctypes.c_int32), ("K", ctypes.c_int32),
                ("m", ctypes.c_int32), ("support", ctypes.c_int32), ("depth", ctypes.c_int32),
                ("budget", ctypes.c_int32), ("eps", ctypes.c_float), ("dtype", ctypes.c_int32)]


_VP = ctypes.c_void_p


class _Tree(ctypes.Structure):
    _fields_ = [(n, _VP) for n in ("token", "parent", "log_proxy", "score", "qtilde", "slot", "frontier",
                                   "tail_ids", "tail_q", "lse1", "lse_tail")]


class _Pruned(ctypes.Structure):
    _fields_ = [(n, _VP) for n in ("gen_id", "token", "parent", "depth", "first_child", "n_child",
                                   "sampled_child")]


class _VerifyOut(ctypes.Structure):
    _fields_ = [(n, _VP) for n in ("accepted_len", "accepted_tokens", "accepted_nodes", "bonus_token",
                                   "row_lse")]


class _TreeAttn(ctypes.Structure):
    _fields_ = [(n, _VP) for n in ("mask", "position", "retrieve", "n_leaves")]


_lib = None


def library_path() -> str:
    return _LIB_PATH


def lib():
    """Load librheo.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(_LIB_PATH):
            raise RheoError(f"{_LIB_PATH} not found: build it with paper_2609_21827_gb300.build.build()")
        L = ctypes.CDLL(_LIB_PATH)
        C = ctypes.POINTER(_Config)
        L.rheo_sizes.argtypes = [C, ctypes.POINTER(ctypes.c_int64), ctypes.POINTER(ctypes.c_int64),
                                 ctypes.POINTER(ctypes.c_size_t)]
        L.rheo_workspace_init.argtypes = [C, _VP, ctypes.c_size_t, _VP]
        L.rheo_expand.argtypes = [C, ctypes.c_int32, _VP, ctypes.c_int64, _VP, _VP, _VP, ctypes.POINTER(_Tree),
                                  _VP, _VP]
        L.rheo_prune.argtypes = [C, ctypes.POINTER(_Tree), ctypes.POINTER(_Pruned), _VP, _VP]
        L.rheo_verify.argtypes = [C, _VP, ctypes.c_int64, _VP, _VP, _VP, ctypes.POINTER(_Tree),
                                  ctypes.POINTER(_Pruned), ctypes.POINTER(_VerifyOut), _VP, _VP]
        L.rheo_verify_static.argtypes = [C, _VP, ctypes.c_int64, _VP, _VP, _VP, ctypes.POINTER(_Tree),
                                         ctypes.POINTER(_Pruned), ctypes.POINTER(_VerifyOut), _VP, _VP]
        L.rheo_get_status.argtypes = [C, _VP, _VP, ctypes.POINTER(ctypes.c_int32)]
        L.rheo_verify_variant.argtypes = [C, ctypes.c_int32, _VP, ctypes.c_int64, _VP, _VP, _VP,
                                          ctypes.POINTER(_Tree), ctypes.POINTER(_Pruned), ctypes.POINTER(_VerifyOut),
                                          _VP, _VP]
        L.rheo_verify_full.argtypes = [C, _VP, ctypes.c_int64, _VP, ctypes.c_int64, _VP, _VP, _VP,
                                       ctypes.POINTER(_Tree), ctypes.POINTER(_Pruned), ctypes.POINTER(_VerifyOut),
                                       _VP, _VP]
        L.rheo_tree_attention.argtypes = [C, ctypes.POINTER(_Pruned), ctypes.POINTER(_TreeAttn), _VP, _VP]
        for name in EXPORTS:
            getattr(L, name).restype = ctypes.c_int
        _lib = L
    return _lib


def _stream(stream) -> int:
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream


def _check(rc: int, what: str):
    if rc != RHEO_OK:
        raise RheoError(f"{what} failed with code {rc}")


@dataclass
class Config:
    batch: int
    vocab: int
    K: int
    depth: int
    budget: int
    m: int = 1
    support: int | None = None
    eps: float = 1e-6
    dtype: str = "bf16"

    def __post_init__(self):
        if self.support is None:
            self.support = min(128, self.vocab)

    @property
    def dtype_code(self) -> int:
        return RHEO_BF16 if self.dtype == "bf16" else RHEO_F32

    @property
    def torch_dtype(self):
        return torch.bfloat16 if self.dtype == "bf16" else torch.float32

    def c(self) -> _Config:
        return _Config(self.batch, self.vocab, self.K, self.m, self.support, self.depth, self.budget,
                       self.eps, self.dtype_code)

    def sizes(self):
        g1, e, ws = ctypes.c_int64(), ctypes.c_int64(), ctypes.c_size_t()
        _check(lib().rheo_sizes(ctypes.byref(self.c()), ctypes.byref(g1), ctypes.byref(e), ctypes.byref(ws)),
               "rheo_sizes")
        return g1.value, e.value, ws.value

    def rows_at(self, d: int) -> int:
        return 1 if d == 1 else self.K


class Tree:
    """Device buffers of the unpruned tree (include/rheo.h rheo_tree)."""

    def __init__(self, cfg: Config, device="cuda"):
        G1, E, _ = cfg.sizes()
        B, TL = cfg.batch, (0 if cfg.support == 0 else cfg.support - cfg.m)
        i32, f32 = torch.int32, torch.float32
        self.token = torch.full((B, G1), -1, dtype=i32, device=device)
        self.parent = torch.full((B, G1), -1, dtype=i32, device=device)
        self.log_proxy = torch.zeros((B, G1), dtype=f32, device=device)
        self.score = torch.zeros((B, G1), dtype=f32, device=device)
        self.qtilde = torch.zeros((B, G1), dtype=f32, device=device)
        self.slot = torch.zeros((B, G1), dtype=torch.uint8, device=device)
        self.frontier = torch.zeros((B, max(cfg.K, 1)), dtype=i32, device=device)
        self.tail_ids = torch.zeros((B, E, TL), dtype=i32, device=device)
        self.tail_q = torch.zeros((B, E, TL), dtype=f32, device=device)
        self.lse1 = torch.zeros((B, E), dtype=f32, device=device)
        self.lse_tail = torch.zeros((B, E), dtype=f32, device=device)

    def c(self) -> _Tree:
        return _Tree(*[getattr(self, n).data_ptr() for n, _ in _Tree._fields_])


class Pruned:
    def __init__(self, cfg: Config, device="cuda"):
        shape = (cfg.batch, cfg.budget + 1)
        for n, _ in _Pruned._fields_:
            setattr(self, n, torch.zeros(shape, dtype=torch.int32, device=device))

    def c(self) -> _Pruned:
        return _Pruned(*[getattr(self, n).data_ptr() for n, _ in _Pruned._fields_])


class VerifyOut:
    def __init__(self, cfg: Config, device="cuda", row_lse: bool = True):
        B, D = cfg.batch, cfg.depth
        self.accepted_len = torch.zeros(B, dtype=torch.int32, device=device)
        self.accepted_tokens = torch.zeros((B, D), dtype=torch.int32, device=device)
        self.accepted_nodes = torch.zeros((B, D), dtype=torch.int32, device=device)
        self.bonus_token = torch.zeros(B, dtype=torch.int32, device=device)
        self.row_lse = torch.zeros((B, cfg.budget + 1), dtype=torch.float32, device=device) if row_lse else None

    def c(self) -> _VerifyOut:
        return _VerifyOut(self.accepted_len.data_ptr(), self.accepted_tokens.data_ptr(),
                          self.accepted_nodes.data_ptr(), self.bonus_token.data_ptr(),
                          self.row_lse.data_ptr() if self.row_lse is not None else None)


class Workspace:
    def __init__(self, cfg: Config, device="cuda", stream=None):
        _, _, nbytes = cfg.sizes()
        self.nbytes = nbytes
        self.buf = torch.empty(max(nbytes, 1), dtype=torch.uint8, device=device)
        self.init(cfg, stream)

    def init(self, cfg: Config, stream=None):
        _check(lib().rheo_workspace_init(ctypes.byref(cfg.c()), self.buf.data_ptr(), self.nbytes, _stream(stream)),
               "rheo_workspace_init")

    def ptr(self) -> int:
        return self.buf.data_ptr()


def _rows(cfg: Config, logits: torch.Tensor, n_rows: int):
    """Validate a [.., V] logits tensor whose rows are uniformly strided; returns the row stride."""
    if logits.dtype != cfg.torch_dtype:
        raise RheoError(f"logits dtype {logits.dtype} does not match config dtype {cfg.dtype}")
    if not logits.is_cuda:
        raise RheoError("logits must be a CUDA tensor")
    if logits.shape[-1] != cfg.vocab or logits.stride(-1) != 1:
        raise RheoError("the last dimension must be the vocabulary, unit stride")
    rows = logits.reshape(-1, cfg.vocab) if logits.dim() != 2 else logits
    if rows.shape[0] != n_rows:
        raise RheoError(f"expected {n_rows} rows, got {rows.shape[0]}")
    if rows.data_ptr() != logits.data_ptr():
        raise RheoError("rows must be addressable with a single row stride")
    return rows.stride(0)


def _i64(x: torch.Tensor) -> torch.Tensor:
    if x.dtype not in (torch.int64, torch.uint64) or not x.is_cuda or not x.is_contiguous():
        raise RheoError("seed/offset must be contiguous 64-bit CUDA tensors")
    return x


def _f32(x: torch.Tensor) -> torch.Tensor:
    if x.dtype != torch.float32 or not x.is_cuda or not x.is_contiguous():
        raise RheoError("temperature must be a contiguous float32 CUDA tensor")
    return x


def expand(cfg: Config, d: int, logits: torch.Tensor, temperature: torch.Tensor, seed: torch.Tensor,
           offset: torch.Tensor, tree: Tree, ws: Workspace, stream=None) -> None:
    """rheo_expand: logits [B, F_d, V] (or [B*F_d, V]) of the frontier rows in frontier order."""
    stride = _rows(cfg, logits, cfg.batch * cfg.rows_at(d))
    _check(lib().rheo_expand(ctypes.byref(cfg.c()), d, logits.data_ptr(), stride, _f32(temperature).data_ptr(),
                             _i64(seed).data_ptr(), _i64(offset).data_ptr(), ctypes.byref(tree.c()), ws.ptr(),
                             _stream(stream)), "rheo_expand")


def prune(cfg: Config, tree: Tree, pruned: Pruned, ws: Workspace, stream=None) -> None:
    _check(lib().rheo_prune(ctypes.byref(cfg.c()), ctypes.byref(tree.c()), ctypes.byref(pruned.c()), ws.ptr(),
                            _stream(stream)), "rheo_prune")


class TreeAttn:
    """Outputs of rheo_tree_attention (ancestor mask, positions, root-to-leaf paths)."""

    def __init__(self, cfg: Config, device="cuda"):
        B, NP, W = cfg.batch, cfg.budget + 1, cfg.depth + 1
        self.mask = torch.zeros((B, NP, NP), dtype=torch.uint8, device=device)
        self.position = torch.zeros((B, NP), dtype=torch.int32, device=device)
        self.retrieve = torch.zeros((B, NP, W), dtype=torch.int32, device=device)
        self.n_leaves = torch.zeros((B,), dtype=torch.int32, device=device)

    def c(self) -> _TreeAttn:
        return _TreeAttn(*[getattr(self, n).data_ptr() for n, _ in _TreeAttn._fields_])


def tree_attention(cfg: Config, pruned: Pruned, out: TreeAttn, ws: Workspace, stream=None) -> None:
    _check(lib().rheo_tree_attention(ctypes.byref(cfg.c()), ctypes.byref(pruned.c()), ctypes.byref(out.c()),
                                     ws.ptr(), _stream(stream)), "rheo_tree_attention")


def verify(cfg: Config, logits: torch.Tensor, temperature: torch.Tensor, seed: torch.Tensor,
           offset: torch.Tensor, tree: Tree, pruned: Pruned, out: VerifyOut, ws: Workspace, stream=None) -> None:
    """rheo_verify: logits [B, N+1, V] of the pruned nodes in pruned order."""
    stride = _rows(cfg, logits, cfg.batch * (cfg.budget + 1))
    _check(lib().rheo_verify(ctypes.byref(cfg.c()), logits.data_ptr(), stride, _f32(temperature).data_ptr(),
                             _i64(seed).data_ptr(), _i64(offset).data_ptr(), ctypes.byref(tree.c()),
                             ctypes.byref(pruned.c()), ctypes.byref(out.c()), ws.ptr(), _stream(stream)),
           "rheo_verify")


def verify_variant(cfg: Config, variant: int, logits: torch.Tensor, temperature: torch.Tensor, seed: torch.Tensor,
                   offset: torch.Tensor, tree: Tree, pruned: Pruned, out: VerifyOut, ws: Workspace,
                   stream=None) -> None:
    """rheo_verify_variant: VERIFY_RHEO (Algorithm 1), VERIFY_RRSW or VERIFY_ONEHOT."""
    stride = _rows(cfg, logits, cfg.batch * (cfg.budget + 1))
    _check(lib().rheo_verify_variant(ctypes.byref(cfg.c()), int(variant), logits.data_ptr(), stride,
                                     _f32(temperature).data_ptr(), _i64(seed).data_ptr(), _i64(offset).data_ptr(),
                                     ctypes.byref(tree.c()), ctypes.byref(pruned.c()), ctypes.byref(out.c()),
                                     ws.ptr(), _stream(stream)),
           "rheo_verify_variant")


def verify_full(cfg: Config, logits: torch.Tensor, draft_rows: list, temperature: torch.Tensor, seed: torch.Tensor,
                offset: torch.Tensor, tree: Tree, pruned: Pruned, out: VerifyOut, ws: Workspace, stream=None) -> None:
    """rheo_verify_full: draft_rows[d-1] = the [B, F_d, V] rows given to expand at depth d."""
    stride = _rows(cfg, logits, cfg.batch * (cfg.budget + 1))
    dstride = None
    ptrs = (ctypes.c_void_p * cfg.depth)()
    for d, x in enumerate(draft_rows):
        st = _rows(cfg, x, x.shape[0] * x.shape[1])
        if dstride is None:
            dstride = st
        elif st != dstride:
            raise RheoError("draft rows of every depth need the same row stride")
        ptrs[d] = x.data_ptr()
    _check(lib().rheo_verify_full(ctypes.byref(cfg.c()), logits.data_ptr(), stride, ptrs, dstride,
                                  _f32(temperature).data_ptr(), _i64(seed).data_ptr(), _i64(offset).data_ptr(),
                                  ctypes.byref(tree.c()), ctypes.byref(pruned.c()), ctypes.byref(out.c()), ws.ptr(),
                                  _stream(stream)),
           "rheo_verify_full")


def verify_static(cfg: Config, logits: torch.Tensor, temperature: torch.Tensor, seed: torch.Tensor,
                  offset: torch.Tensor, tree: Tree, pruned: Pruned, out: VerifyOut,
                  status: torch.Tensor = None, stream=None) -> None:
    """rheo_verify_static: rheo_verify without a workspace, for callers that may
    not allocate device memory when they verify.  Its scratch is a fixed static
    array inside the library (calls must not overlap on the GPU); configurations
    that need more than it holds raise RheoError with code RHEO_ETOOLARGE.
    status: optional int32 device tensor of one element that receives the
    call's status word."""
    stride = _rows(cfg, logits, cfg.batch * (cfg.budget + 1))
    st = 0
    if status is not None:
        if status.dtype != torch.int32 or status.numel() < 1 or not status.is_cuda:
            raise RheoError("status must be an int32 device tensor")
        st = status.data_ptr()
    _check(lib().rheo_verify_static(ctypes.byref(cfg.c()), logits.data_ptr(), stride, _f32(temperature).data_ptr(),
                                    _i64(seed).data_ptr(), _i64(offset).data_ptr(), ctypes.byref(tree.c()),
                                    ctypes.byref(pruned.c()), ctypes.byref(out.c()), st,
                                    _stream(stream)),
           "rheo_verify_static")


def status(cfg: Config, ws: Workspace, stream=None) -> int:
    """Synchronise the stream, return and clear the device status word."""
    st = ctypes.c_int32()
    _check(lib().rheo_get_status(ctypes.byref(cfg.c()), ws.ptr(), _stream(stream), ctypes.byref(st)),
           "rheo_get_status")
    return st.value
