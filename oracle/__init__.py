"""ctypes wrapper of the fp64 CPU oracle (``kvec_oracle.c``).

TEST INFRASTRUCTURE ONLY: imported by ``tests/``, ``__graft_entry__.smoke()``
and the CPU-baseline leg of ``bench.py``.  The CUDA product path never
imports this package.  The oracle follows Algorithm 1 and Sections 4.1-4.2
of the K-VEC paper; see ``kvec_oracle.c`` for the readings it takes.
"""
from __future__ import annotations

import ctypes
import dataclasses
import os
import subprocess
import threading
from typing import Dict, Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIB_PATH = os.path.join(_HERE, "_build", "libkvec_oracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (-O2, OpenMP) into oracle/_build/."""
    src = os.path.join(_HERE, "kvec_oracle.c")
    os.makedirs(os.path.dirname(_LIB_PATH), exist_ok=True)
    fresh = os.path.exists(_LIB_PATH) and os.path.getmtime(_LIB_PATH) >= max(
        os.path.getmtime(src), os.path.getmtime(os.path.join(_HERE, "kvec_oracle.h")))
    if fresh and not force:
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    compile_source(src, tmp)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def compile_source(src: str, out: str) -> None:
    """gcc -O2 (OpenMP, no FMA contraction) of an oracle source into a shared library."""
    cmd = ["gcc", "-O2", "-std=c99", "-fPIC", "-shared", "-fopenmp", "-ffp-contract=off",
           "-I", _HERE, "-o", out, src, "-lm"]
    subprocess.run(cmd, check=True)


class _Params(ctypes.Structure):
    _fields_ = [
        ("num_q_heads", ctypes.c_int), ("num_kv_heads", ctypes.c_int), ("head_dim", ctypes.c_int),
        ("window", ctypes.c_int), ("obs_window", ctypes.c_int), ("ext_window", ctypes.c_int),
        ("pool_kernel", ctypes.c_int), ("num_ext_heads", ctypes.c_int),
        ("lam", ctypes.c_double), ("beta", ctypes.c_double), ("softmax_scale", ctypes.c_double),
        ("pool_mode", ctypes.c_int), ("head_criterion", ctypes.c_int), ("all_positions", ctypes.c_int),
        ("head_budget", ctypes.c_int), ("ada_floor", ctypes.c_double),
    ]


_dp = ctypes.POINTER(ctypes.c_double)


class _Debug(ctypes.Structure):
    _fields_ = [
        ("P_O_raw", _dp), ("P_Oext_raw", _dp), ("I_raw", _dp),
        ("P_O", _dp), ("P_Oext", _dp), ("I", _dp), ("sigma", _dp),
        ("htop", ctypes.POINTER(ctypes.c_int32)), ("P", _dp),
        ("pres", ctypes.POINTER(ctypes.c_uint8)), ("Pprime", _dp), ("row_sums", _dp),
        ("coverage", ctypes.POINTER(ctypes.c_int64)), ("literal_override_differs", ctypes.c_int64),
    ]


def _load():
    global _lib
    with _lock:
        if _lib is None:
            # KVEC_ORACLE_LIB: another build of kvec_oracle.c to load instead (the
            # test that plants mistakes in copies of the oracle runs the pins on them).
            path = os.environ.get("KVEC_ORACLE_LIB") or build()
            lib = ctypes.CDLL(path)
            lib.kvo_state_bytes.restype = ctypes.c_size_t
            lib.kvo_state_bytes.argtypes = [ctypes.c_int]
            lib.kvo_num_threads.restype = ctypes.c_int
            lib.kvo_head_capacity.restype = ctypes.c_int
            lib.kvo_head_capacity.argtypes = [ctypes.POINTER(_Params), ctypes.c_int]
            lib.kvo_select_layer.restype = ctypes.c_int
            lib.kvo_select_layer.argtypes = [
                ctypes.POINTER(_Params), ctypes.c_int, ctypes.c_void_p, ctypes.c_int,
                ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int,
                ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.POINTER(_Debug)]
            _lib = lib
    return _lib


@dataclasses.dataclass
class OracleParams:
    num_q_heads: int
    num_kv_heads: int
    head_dim: int = 128
    window: int = 32
    obs_window: int = 16
    ext_window: int = 32
    pool_kernel: int = 7
    num_ext_heads: int = 3
    lam: float = 1.0
    beta: float = 0.25
    softmax_scale: float = 0.0
    pool_mode: int = 0        # 0 max-pool, 1 average pool
    head_criterion: int = 0   # 0 standard deviation, 1 entropy
    all_positions: int = 0    # 0 keep the window tail, 1 every position is a candidate
    head_budget: int = 0      # 0 uniform fill, 1 head-wise adaptive fill
    ada_floor: float = 1.0    # share of a head's fill it keeps by its own ranking (adaptive fill)

    @classmethod
    def from_workload(cls, wl, **over) -> "OracleParams":
        kw = dict(num_q_heads=wl.num_q_heads, num_kv_heads=wl.num_kv_heads, head_dim=wl.head_dim,
                  window=wl.window, obs_window=wl.obs_window, ext_window=wl.ext_window,
                  pool_kernel=wl.pool_kernel, num_ext_heads=wl.num_ext_heads,
                  lam=float(np.float32(wl.lam)), beta=float(np.float32(wl.beta)),
                  pool_mode=getattr(wl, "pool_mode", 0), head_criterion=getattr(wl, "head_criterion", 0),
                  all_positions=getattr(wl, "all_positions", 0), head_budget=getattr(wl, "head_budget", 0),
                  ada_floor=float(np.float32(getattr(wl, "ada_floor", 1.0))))
        kw.update(over)
        return cls(**kw)

    def _c(self) -> _Params:
        return _Params(self.num_q_heads, self.num_kv_heads, self.head_dim, self.window,
                       self.obs_window, self.ext_window, self.pool_kernel, self.num_ext_heads,
                       float(self.lam), float(self.beta), float(self.softmax_scale), int(self.pool_mode),
                       int(self.head_criterion), int(self.all_positions), int(self.head_budget),
                       float(self.ada_floor))


def head_capacity(params: OracleParams, budget: int) -> int:
    """Rows per KV head of the outputs (budget for the uniform fill)."""
    cap = int(_load().kvo_head_capacity(ctypes.byref(params._c()), int(budget)))
    if cap < 1:
        raise ValueError("invalid parameters for the output capacity")
    return cap


def state_bytes(max_seqlen: int) -> int:
    return int(_load().kvo_state_bytes(int(max_seqlen)))


def num_threads() -> int:
    return int(_load().kvo_num_threads())


def new_state(batch: int, max_seqlen: int) -> np.ndarray:
    return np.zeros((batch, state_bytes(max_seqlen)), np.uint8)


def state_fields(state: np.ndarray, max_seqlen: int) -> Dict[str, np.ndarray]:
    """Views of the per-sequence state: layers_done, seqlen, n[max_seqlen], last_union words."""
    ns = (max_seqlen + 15) // 16 * 16
    words = (max_seqlen + 31) // 32
    hdr = state[:, :16].copy().view(np.uint32)
    return {
        "layers_done": hdr[:, 0], "seqlen": hdr[:, 1],
        "n": state[:, 16:16 + max_seqlen],
        "last_union": state[:, 16 + ns:16 + ns + 4 * words].copy().view(np.uint32),
    }


def _as_u16(x) -> np.ndarray:
    """bf16 tensor / uint16 array -> contiguous uint16 bit patterns."""
    try:
        import torch
        if isinstance(x, torch.Tensor):
            return np.ascontiguousarray(x.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16))
    except ImportError:  # pragma: no cover
        pass
    a = np.ascontiguousarray(x)
    assert a.dtype == np.uint16
    return a


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def select_layer(params: OracleParams, cu_seqlens, q_obs, k, v, state: np.ndarray, budget: int,
                 max_seqlen: Optional[int] = None, debug: bool = True) -> Dict[str, np.ndarray]:
    """Runs one layer of the oracle.  ``state`` (uint8 [batch][state_bytes]) is updated in place.

    Returns out_idx [batch][Hkv][cap] int32, out_k / out_v [batch][Hkv][cap][d] uint16 (bf16 bits),
    cap = head_capacity(params, budget) (= budget for the uniform fill),
    and, with ``debug``, every intermediate listed in ``kvo_debug``.
    """
    lib = _load()
    cu = np.ascontiguousarray(np.asarray(cu_seqlens, dtype=np.int32))
    batch = cu.size - 1
    lens = np.diff(cu)
    ML = int(max_seqlen if max_seqlen is not None else lens.max())
    Hq, Hkv, d, w = params.num_q_heads, params.num_kv_heads, params.head_dim, params.window
    qa, ka, va = _as_u16(q_obs), _as_u16(k), _as_u16(v)
    assert state.dtype == np.uint8 and state.shape == (batch, state_bytes(ML)) and state.flags.c_contiguous
    cap = head_capacity(params, budget)
    out_idx = np.empty((batch, Hkv, cap), np.int32)
    out_k = np.empty((batch, Hkv, cap, d), np.uint16)
    out_v = np.empty((batch, Hkv, cap, d), np.uint16)
    res: Dict[str, np.ndarray] = {}
    dbg = None
    if debug:
        res = {
            "P_O_raw": np.zeros((batch, Hkv, ML)), "P_Oext_raw": np.zeros((batch, Hkv, ML)),
            "I_raw": np.zeros((batch, ML)), "P_O": np.zeros((batch, Hkv, ML)),
            "P_Oext": np.zeros((batch, Hkv, ML)), "I": np.zeros((batch, ML)),
            "sigma": np.zeros((batch, Hkv)), "htop": np.zeros((batch, Hkv), np.int32),
            "P": np.zeros((batch, Hkv, ML)), "pres": np.zeros((batch, Hkv, ML), np.uint8),
            "Pprime": np.zeros((batch, Hkv, ML)), "row_sums": np.zeros((batch, Hq, w)),
            "coverage": np.zeros(batch, np.int64),
        }
        dbg = _Debug()
        ctype_of = dict(_Debug._fields_)
        for name, arr in res.items():
            setattr(dbg, name, arr.ctypes.data_as(ctype_of[name]))
    rc = lib.kvo_select_layer(ctypes.byref(params._c()), batch, _ptr(cu), ML, _ptr(qa), _ptr(ka), _ptr(va),
                              _ptr(state), int(budget), _ptr(out_idx), _ptr(out_k), _ptr(out_v),
                              ctypes.byref(dbg) if dbg is not None else None)
    if rc != 0:
        raise ValueError(f"oracle rejected the arguments (code {rc})")
    res.update(out_idx=out_idx, out_k=out_k, out_v=out_v)
    if dbg is not None:
        res["literal_override_differs"] = int(dbg.literal_override_differs)
    return res
