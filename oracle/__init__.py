"""CPU oracle of the RheoSampling draft-tree hot path.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import this
package.  The product path (``paper_2609_21827_gb300``) never imports it and
shares no code with it.

The arithmetic lives in ``rheo_oracle.c`` (plain C, fp64 sums, full sorts);
this module compiles it with gcc and marshals numpy arrays through ctypes.
See ``rheo_oracle.c`` for the conventions the paper leaves open.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from dataclasses import dataclass, field

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "rheo_oracle.c")
_HDR = os.path.join(_HERE, "rheo_oracle.h")
_SO = os.path.join(_HERE, "librheo_oracle.so")

SLOT_ROOT, SLOT_LEAD, SLOT_SAMPLED, SLOT_FILL = 0, 1, 2, 3
TAG_CONTINUE, TAG_SAMPLE, TAG_VERIFY, TAG_RESIDUAL = 0, 1, 2, 3


def build(force: bool = False) -> str:
    """Compile the oracle into ``oracle/librheo_oracle.so`` (gcc, no fast-math)."""
    newest = max(os.path.getmtime(_SRC), os.path.getmtime(_HDR))
    if not force and os.path.exists(_SO) and os.path.getmtime(_SO) >= newest:
        return _SO
    base = ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared"]
    tmp = _SO + f".tmp{os.getpid()}"
    try:
        subprocess.check_call(base + ["-fopenmp", "-o", tmp, _SRC, "-lm"])
    except subprocess.CalledProcessError:
        subprocess.check_call(base + ["-o", tmp, _SRC, "-lm"])
    os.replace(tmp, _SO)
    return _SO


VERIFY_RHEO, VERIFY_RRSW, VERIFY_ONEHOT = 0, 1, 2
# mistakes planted on purpose (tests that must reject them); see rheo_oracle.h
PLANT_NONE, PLANT_RESIDUAL_ON_SUPPORT, PLANT_MASS_ON_SUPPORT, PLANT_BLOCK_UNWEIGHTED = 0, 1, 2, 3


class _Cfg(ctypes.Structure):
    _fields_ = [
        ("B", ctypes.c_int32), ("V", ctypes.c_int32), ("K", ctypes.c_int32),
        ("m", ctypes.c_int32), ("S", ctypes.c_int32), ("D", ctypes.c_int32),
        ("N", ctypes.c_int32), ("eps", ctypes.c_double),
        ("proxy_mode", ctypes.c_int32), ("fixed_log_proxy", ctypes.c_double),
        ("verify_mode", ctypes.c_int32), ("plant_mode", ctypes.c_int32),
    ]


_P = ctypes.c_void_p


class _Tree(ctypes.Structure):
    _fields_ = [(n, _P) for n in (
        "token", "parent", "log_proxy", "score", "qtilde", "slot", "frontier",
        "tail_ids", "tail_q", "lse1", "gap_sample", "gap_frontier", "lse_tail")]


class _Pruned(ctypes.Structure):
    _fields_ = [(n, _P) for n in (
        "gen_id", "token", "parent", "depth", "first_child", "n_child", "sampled_child",
        "gap_prune")]


class _VerifyOut(ctypes.Structure):
    _fields_ = [(n, _P) for n in (
        "accepted_len", "accepted_tokens", "accepted_nodes", "bonus_token", "row_lse",
        "gap_level", "stop_mass")]


_lib = None


def lib():
    global _lib
    if _lib is None:
        _lib = ctypes.CDLL(build())
        L = _lib
        L.orc_check_cfg.argtypes = [ctypes.POINTER(_Cfg)]
        L.orc_nodes_per_request.argtypes = [ctypes.POINTER(_Cfg)]
        L.orc_nodes_per_request.restype = ctypes.c_int64
        L.orc_expansions_per_request.argtypes = [ctypes.POINTER(_Cfg)]
        L.orc_expansions_per_request.restype = ctypes.c_int64
        L.orc_philox4x32_10.argtypes = [_P, _P, _P]
        L.orc_uniform.argtypes = [ctypes.c_uint64, ctypes.c_uint64, ctypes.c_int32,
                                  ctypes.c_int32, ctypes.c_uint64]
        L.orc_uniform.restype = ctypes.c_float
        L.orc_topk_row.argtypes = [_P, ctypes.c_int32, ctypes.c_int32, _P]
        L.orc_expand.argtypes = [ctypes.POINTER(_Cfg), ctypes.c_int32, _P, _P, _P, _P,
                                 ctypes.POINTER(_Tree)]
        L.orc_prune.argtypes = [ctypes.POINTER(_Cfg), ctypes.POINTER(_Tree),
                                ctypes.POINTER(_Pruned)]
        L.orc_verify.argtypes = [ctypes.POINTER(_Cfg), _P, _P, _P, _P, ctypes.POINTER(_Tree),
                                 ctypes.POINTER(_Pruned), ctypes.POINTER(_VerifyOut)]
        L.orc_run_prefix_lm.argtypes = [ctypes.POINTER(_Cfg), _P, _P, ctypes.c_int32,
                                        ctypes.c_int64, ctypes.c_float, ctypes.c_uint64,
                                        ctypes.c_int32, _P, _P]
        L.orc_tree_attention.argtypes = [ctypes.POINTER(_Cfg), ctypes.POINTER(_Pruned), _P, _P, _P, _P]
        L.orc_threads_used.argtypes = [ctypes.c_int32]
        L.orc_set_threads.argtypes = [ctypes.c_int32]
        L.orc_set_threads.restype = None
    return _lib


def _ptr(a: np.ndarray) -> int:
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data


@dataclass
class Config:
    """Problem size; K counts the deterministic slots (pool = K + 1)."""

    B: int
    V: int
    K: int
    m: int = 1
    S: int | None = None
    D: int = 1
    N: int = 1
    eps: float = 1e-6
    proxy_mode: int = 0
    fixed_log_proxy: float = 0.0
    verify_mode: int = 0  # VERIFY_RHEO, VERIFY_RRSW or VERIFY_ONEHOT
    plant_mode: int = 0   # PLANT_*: tests only

    def __post_init__(self):
        if self.S is None:
            self.S = min(128, self.V)

    def c(self) -> _Cfg:
        return _Cfg(self.B, self.V, self.K, self.m, self.S, self.D, self.N, self.eps,
                    self.proxy_mode, self.fixed_log_proxy, self.verify_mode, self.plant_mode)

    @property
    def G1(self) -> int:
        return 1 + (self.K + 1) + (self.D - 1) * self.K * (self.K + 1)

    @property
    def E(self) -> int:
        return 1 + (self.D - 1) * self.K

    @property
    def TL(self) -> int:
        return (self.V if self.S == 0 else self.S) - self.m

    def rows_at(self, d: int) -> int:
        return 1 if d == 1 else self.K

    def valid(self) -> bool:
        return lib().orc_check_cfg(ctypes.byref(self.c())) == 0


@dataclass
class Tree:
    cfg: Config
    token: np.ndarray = field(init=False)
    parent: np.ndarray = field(init=False)
    log_proxy: np.ndarray = field(init=False)
    score: np.ndarray = field(init=False)
    qtilde: np.ndarray = field(init=False)
    slot: np.ndarray = field(init=False)
    frontier: np.ndarray = field(init=False)
    tail_ids: np.ndarray = field(init=False)
    tail_q: np.ndarray = field(init=False)
    lse1: np.ndarray = field(init=False)
    gap_sample: np.ndarray = field(init=False)
    gap_frontier: np.ndarray = field(init=False)
    lse_tail: np.ndarray = field(init=False)

    def __post_init__(self):
        c = self.cfg
        B, G1, E, TL = c.B, c.G1, c.E, c.TL
        self.token = np.full((B, G1), -1, np.int32)
        self.parent = np.full((B, G1), -1, np.int32)
        self.log_proxy = np.zeros((B, G1), np.float32)
        self.score = np.zeros((B, G1), np.float32)
        self.qtilde = np.zeros((B, G1), np.float32)
        self.slot = np.zeros((B, G1), np.uint8)
        self.frontier = np.zeros((B, max(c.K, 1)), np.int32)
        self.tail_ids = np.zeros((B, E, TL), np.int32)
        self.tail_q = np.zeros((B, E, TL), np.float32)
        self.lse1 = np.zeros((B, E), np.float32)
        self.gap_sample = np.full((B, E), np.inf)
        self.gap_frontier = np.full((B, c.D), np.inf)
        self.lse_tail = np.zeros((B, E), np.float32)

    def c(self) -> _Tree:
        return _Tree(*[_ptr(getattr(self, n)) for n, _ in _Tree._fields_])


@dataclass
class Pruned:
    cfg: Config

    def __post_init__(self):
        B, n = self.cfg.B, self.cfg.N + 1
        for name in ("gen_id", "token", "parent", "depth", "first_child", "n_child",
                     "sampled_child"):
            setattr(self, name, np.zeros((B, n), np.int32))
        self.gap_prune = np.full(B, np.inf)

    def c(self) -> _Pruned:
        return _Pruned(*[_ptr(getattr(self, n)) for n, _ in _Pruned._fields_])


@dataclass
class VerifyOut:
    cfg: Config

    def __post_init__(self):
        c = self.cfg
        self.accepted_len = np.zeros(c.B, np.int32)
        self.accepted_tokens = np.full((c.B, c.D), -1, np.int32)
        self.accepted_nodes = np.full((c.B, c.D), -1, np.int32)
        self.bonus_token = np.zeros(c.B, np.int32)
        self.row_lse = np.zeros((c.B, c.N + 1), np.float32)
        self.gap_level = np.full((c.B, c.D + 1), np.inf)
        self.stop_mass = np.zeros(c.B, np.float32)

    def c(self) -> _VerifyOut:
        return _VerifyOut(*[_ptr(getattr(self, n)) for n, _ in _VerifyOut._fields_])


def _vec(x, n, dtype):
    a = np.asarray(x, dtype=dtype)
    if a.ndim == 0:
        a = np.full(n, a, dtype=dtype)
    return np.ascontiguousarray(a)


class OracleError(RuntimeError):
    pass


def expand(cfg: Config, d: int, rows: np.ndarray, T, seed, offset, tree: Tree) -> None:
    """One expansion call at depth d; rows [B, F_d, V] float32 in frontier order."""
    rows = np.ascontiguousarray(rows, dtype=np.float32)
    assert rows.shape == (cfg.B, cfg.rows_at(d), cfg.V), rows.shape
    T = _vec(T, cfg.B, np.float32)
    seed = _vec(seed, cfg.B, np.uint64)
    offset = _vec(offset, cfg.B, np.uint64)
    rc = lib().orc_expand(ctypes.byref(cfg.c()), d, _ptr(rows), _ptr(T), _ptr(seed),
                          _ptr(offset), ctypes.byref(tree.c()))
    if rc:
        raise OracleError(f"orc_expand returned {rc}")


def prune(cfg: Config, tree: Tree) -> Pruned:
    p = Pruned(cfg)
    rc = lib().orc_prune(ctypes.byref(cfg.c()), ctypes.byref(tree.c()), ctypes.byref(p.c()))
    if rc:
        raise OracleError(f"orc_prune returned {rc}")
    return p


def verify(cfg: Config, target: np.ndarray, T, seed, offset, tree: Tree, pruned: Pruned) -> VerifyOut:
    """Algorithm 1 layer by layer; target [B, N+1, V] float32 in pruned order."""
    target = np.ascontiguousarray(target, dtype=np.float32)
    assert target.shape == (cfg.B, cfg.N + 1, cfg.V), target.shape
    T = _vec(T, cfg.B, np.float32)
    seed = _vec(seed, cfg.B, np.uint64)
    offset = _vec(offset, cfg.B, np.uint64)
    o = VerifyOut(cfg)
    rc = lib().orc_verify(ctypes.byref(cfg.c()), _ptr(target), _ptr(T), _ptr(seed), _ptr(offset),
                          ctypes.byref(tree.c()), ctypes.byref(pruned.c()), ctypes.byref(o.c()))
    if rc:
        raise OracleError(f"orc_verify returned {rc}")
    return o


@dataclass
class TreeAttention:
    mask: np.ndarray       # [B, N+1, N+1] uint8
    position: np.ndarray   # [B, N+1] int32
    retrieve: np.ndarray   # [B, N+1, D+1] int32
    n_leaves: np.ndarray   # [B] int32


def tree_attention(cfg: Config, pruned: Pruned) -> TreeAttention:
    """Tree attention inputs of the pruned tree (mask, positions, root-to-leaf paths)."""
    B, NP, W = cfg.B, cfg.N + 1, cfg.D + 1
    ta = TreeAttention(np.zeros((B, NP, NP), np.uint8), np.zeros((B, NP), np.int32),
                       np.zeros((B, NP, W), np.int32), np.zeros(B, np.int32))
    rc = lib().orc_tree_attention(ctypes.byref(cfg.c()), ctypes.byref(pruned.c()), _ptr(ta.mask),
                                  _ptr(ta.position), _ptr(ta.retrieve), _ptr(ta.n_leaves))
    if rc:
        raise OracleError(f"orc_tree_attention returned {rc}")
    return ta


def philox(ctr, key) -> np.ndarray:
    c = np.ascontiguousarray(ctr, dtype=np.uint32)
    k = np.ascontiguousarray(key, dtype=np.uint32)
    out = np.zeros(4, np.uint32)
    lib().orc_philox4x32_10(_ptr(c), _ptr(k), _ptr(out))
    return out


def uniform(seed: int, offset: int, tag: int, node: int, draw: int) -> float:
    return float(lib().orc_uniform(seed, offset, tag, node, draw))


def topk_row(row: np.ndarray, S: int) -> np.ndarray:
    row = np.ascontiguousarray(row, dtype=np.float32)
    out = np.zeros(S, np.int32)
    if lib().orc_topk_row(_ptr(row), row.shape[0], S, _ptr(out)):
        raise OracleError("orc_topk_row failed")
    return out


def run_prefix_lm(cfg: Config, draft_table: np.ndarray, target_table: np.ndarray, table_depth: int,
                  n_trials: int, T: float, seed0: int, L: int):
    """Whole cycles against prefix-indexed tables; returns (streams [n, L], accepted_len [n])."""
    draft_table = np.ascontiguousarray(draft_table, dtype=np.float32)
    target_table = np.ascontiguousarray(target_table, dtype=np.float32)
    streams = np.zeros((n_trials, L), np.int32)
    acc = np.zeros(n_trials, np.int32)
    rc = lib().orc_run_prefix_lm(ctypes.byref(cfg.c()), _ptr(draft_table), _ptr(target_table),
                                 table_depth, n_trials, T, seed0, L, _ptr(streams), _ptr(acc))
    if rc:
        raise OracleError(f"orc_run_prefix_lm returned {rc}")
    return streams, acc


def run_step(cfg: Config, draft_rows, target_rows, T, seed, offset):
    """Expand at every depth, prune, verify.  draft_rows[d-1] is [B, F_d, V];
    target_rows is an array [B, N+1, V] or a callable (tree, pruned) -> array."""
    tree = Tree(cfg)
    for d in range(1, cfg.D + 1):
        expand(cfg, d, draft_rows[d - 1], T, seed, offset, tree)
    pr = prune(cfg, tree)
    tgt = target_rows(tree, pr) if callable(target_rows) else target_rows
    out = verify(cfg, tgt, T, seed, offset, tree, pr)
    return tree, pr, out


def threads_used(reset: bool = True) -> int:
    """OpenMP threads that ran part of the oracle's parallel loops since the last reset."""
    return int(lib().orc_threads_used(1 if reset else 0))


def set_threads(n: int) -> None:
    """Team size of the oracle's parallel loops from now on."""
    lib().orc_set_threads(int(n))


def max_threads() -> int:
    return int(lib().orc_max_threads())
