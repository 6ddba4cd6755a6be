"""Python binding of libkvec (include/kvec.h): ctypes marshalling only.

Every function here forwards to the C ABI entry point of the same name.  All
computation happens in the CUDA kernels of libkvec; there is no Python or CPU
fallback.  If the library is missing, importing this module still works but the
first call raises ``KvecUnavailable`` (build it with ``build.build()``).
"""
from __future__ import annotations

import ctypes
import os
import threading
from typing import Optional, Sequence

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_build", "libkvec.so")

KVEC_OK = 0
KVEC_ERR_INVALID_ARG = 1
KVEC_ERR_UNSUPPORTED = 2
KVEC_ERR_CUDA = 3
KVEC_ERR_DEVICE_TIMEOUT = 4
KVEC_ERR_OOM = 5

# kernel ids of kvec_kernel_time
KERNEL_NAMES = ("score", "window", "heads", "select", "gather")

EXPORTED = ("kvec_create", "kvec_destroy", "kvec_state_bytes", "kvec_reset", "kvec_select_layer",
            "kvec_select_layers", "kvec_debug_scores", "kvec_sync_status", "kvec_set_profiling",
            "kvec_kernel_time", "kvec_status_string", "kvec_last_error", "kvec_select_layer_noalloc",
            "kvec_select_layer_lse", "kvec_select_layers_lse", "kvec_decode_attention",
            "kvec_noalloc_sync_status", "kvec_set_test_fault", "kvec_output_capacity")


class KvecUnavailable(ImportError):
    pass


class KvecError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"kvec status {status}: {message}")
        self.status = status


class kvec_params(ctypes.Structure):
    _fields_ = [
        ("num_q_heads", ctypes.c_int), ("num_kv_heads", ctypes.c_int), ("head_dim", ctypes.c_int),
        ("window", ctypes.c_int), ("obs_window", ctypes.c_int), ("ext_window", ctypes.c_int),
        ("pool_kernel", ctypes.c_int), ("num_ext_heads", ctypes.c_int),
        ("lam", ctypes.c_float), ("beta", ctypes.c_float), ("softmax_scale", ctypes.c_float),
        ("max_batch", ctypes.c_int), ("max_seqlen", ctypes.c_int), ("max_layers", ctypes.c_int),
        ("pool_mode", ctypes.c_int), ("head_criterion", ctypes.c_int), ("all_positions", ctypes.c_int),
        ("head_budget", ctypes.c_int), ("ada_floor", ctypes.c_float),
    ]


class kvec_debug_view(ctypes.Structure):
    _fields_ = [
        ("P_O", ctypes.c_void_p), ("P_Oext", ctypes.c_void_p), ("I", ctypes.c_void_p),
        ("sigma", ctypes.c_void_p), ("htop", ctypes.c_void_p), ("pres_bits", ctypes.c_void_p),
        ("Pprime", ctypes.c_void_p), ("row_stats", ctypes.c_void_p),
        ("max_seqlen", ctypes.c_int), ("words_per_row", ctypes.c_int),
    ]


_lib = None
_lock = threading.Lock()
_vp = ctypes.c_void_p
_pp = ctypes.POINTER(ctypes.c_void_p)


def load() -> ctypes.CDLL:
    """Loads libkvec.so once; raises KvecUnavailable when it has not been built."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        if not os.path.exists(LIB_PATH):
            raise KvecUnavailable(f"{LIB_PATH} is missing: build the CUDA library first "
                                  "(python -c 'import __graft_entry__ as g; g.build()')")
        lib = ctypes.CDLL(LIB_PATH)
        i, st = ctypes.c_int, ctypes.c_int
        sig = {
            "kvec_create": ([ctypes.POINTER(kvec_params), ctypes.POINTER(_vp)], st),
            "kvec_destroy": ([_vp], st),
            "kvec_state_bytes": ([i], ctypes.c_size_t),
            "kvec_reset": ([_vp, _vp, i, _vp], st),
            "kvec_select_layer": ([_vp, i, _vp, _vp, _vp, _vp, _vp, _vp, i, _vp, _vp, _vp, _vp], st),
            "kvec_select_layers": ([_vp, i, i, _vp, _vp, _pp, _pp, _pp, _vp, i, _pp, _pp, _pp, _vp], st),
            "kvec_debug_scores": ([_vp, ctypes.POINTER(kvec_debug_view)], st),
            "kvec_sync_status": ([_vp], st),
            "kvec_set_profiling": ([_vp, i], st),
            "kvec_kernel_time": ([_vp, i, ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_int)], st),
            "kvec_status_string": ([i], ctypes.c_char_p),
            "kvec_last_error": ([], ctypes.c_char_p),
            "kvec_select_layer_noalloc": ([ctypes.POINTER(kvec_params), i, _vp, _vp, _vp, _vp, _vp, _vp, i, _vp,
                                           _vp, _vp, _vp], st),
            "kvec_select_layer_lse": ([_vp, i, _vp, _vp, _vp, _vp, _vp, _vp, _vp, i, _vp, _vp, _vp, _vp], st),
            "kvec_select_layers_lse": ([_vp, i, i, _vp, _vp, _pp, _pp, _pp, _pp, _vp, i, _pp, _pp, _pp, _vp], st),
            "kvec_decode_attention": ([_vp, i, _vp, _vp, _vp, _vp, i, _vp, _vp], st),
            "kvec_noalloc_sync_status": ([_vp], st),
            "kvec_set_test_fault": ([i], None),
            "kvec_output_capacity": ([ctypes.POINTER(kvec_params), i], i),
        }
        for name, (args, res) in sig.items():
            fn = getattr(lib, name)
            fn.argtypes = args
            fn.restype = res
        _lib = lib
        return lib


def _check(status: int) -> None:
    if status != KVEC_OK:
        msg = load().kvec_last_error().decode(errors="replace")
        raise KvecError(status, msg)


def _arr(ptrs: Sequence[int]):
    return (ctypes.c_void_p * len(ptrs))(*[ctypes.c_void_p(int(p)) for p in ptrs])


def kvec_create(params: kvec_params) -> int:
    h = ctypes.c_void_p()
    _check(load().kvec_create(ctypes.byref(params), ctypes.byref(h)))
    return h.value


def kvec_destroy(handle: int) -> None:
    _check(load().kvec_destroy(handle))


def kvec_state_bytes(max_seqlen: int) -> int:
    return int(load().kvec_state_bytes(int(max_seqlen)))


def kvec_reset(handle: int, state_ptr: int, batch: int, stream: int = 0) -> None:
    _check(load().kvec_reset(handle, state_ptr, int(batch), stream))


def kvec_select_layer(handle: int, batch: int, cu_host_ptr: int, cu_dev_ptr: int, q_obs: int, k: int, v: int,
                      state: int, budget: int, out_idx: int, out_k: int, out_v: int, stream: int = 0) -> None:
    _check(load().kvec_select_layer(handle, int(batch), cu_host_ptr, cu_dev_ptr, q_obs, k, v, state, int(budget),
                                    out_idx, out_k, out_v, stream))


def kvec_select_layers(handle: int, batch: int, cu_host_ptr: int, cu_dev_ptr: int, q_obs: Sequence[int],
                       k: Sequence[int], v: Sequence[int], state: int, budget: int, out_idx: Sequence[int],
                       out_k: Sequence[int], out_v: Sequence[int], stream: int = 0) -> None:
    n = len(q_obs)
    _check(load().kvec_select_layers(handle, n, int(batch), cu_host_ptr, cu_dev_ptr, _arr(q_obs), _arr(k), _arr(v),
                                     state, int(budget), _arr(out_idx), _arr(out_k), _arr(out_v), stream))


def kvec_select_layer_lse(handle: int, batch: int, cu_host_ptr: int, cu_dev_ptr: int, q_obs: int, k: int, v: int,
                          lse: int, state: int, budget: int, out_idx: int, out_k: int, out_v: int,
                          stream: int = 0) -> None:
    _check(load().kvec_select_layer_lse(handle, int(batch), cu_host_ptr, cu_dev_ptr, q_obs, k, v, lse, state,
                                        int(budget), out_idx, out_k, out_v, stream))


def kvec_select_layers_lse(handle: int, batch: int, cu_host_ptr: int, cu_dev_ptr: int, q_obs: Sequence[int],
                           k: Sequence[int], v: Sequence[int], lse: Sequence[int], state: int, budget: int,
                           out_idx: Sequence[int], out_k: Sequence[int], out_v: Sequence[int],
                           stream: int = 0) -> None:
    n = len(q_obs)
    _check(load().kvec_select_layers_lse(handle, n, int(batch), cu_host_ptr, cu_dev_ptr, _arr(q_obs), _arr(k),
                                         _arr(v), _arr(lse), state, int(budget), _arr(out_idx), _arr(out_k),
                                         _arr(out_v), stream))


def kvec_select_layer_noalloc(params: kvec_params, batch: int, cu_host_ptr: int, cu_dev_ptr: int, q_obs: int,
                              k: int, v: int, state: int, budget: int, out_idx: int, out_k: int, out_v: int,
                              stream: int = 0) -> None:
    """kvec_select_layer without a handle; scratch comes from the library's static device array."""
    _check(load().kvec_select_layer_noalloc(ctypes.byref(params), int(batch), cu_host_ptr, cu_dev_ptr, q_obs, k, v,
                                            state, int(budget), out_idx, out_k, out_v, stream))


def kvec_noalloc_sync_status(stream: int = 0) -> None:
    """Raises KvecError for a device-side error recorded by kvec_select_layer_noalloc calls."""
    _check(load().kvec_noalloc_sync_status(stream))


def kvec_output_capacity(params: kvec_params, budget: int) -> int:
    """Rows per KV head of the selection outputs (the budget for the uniform fill)."""
    cap = int(load().kvec_output_capacity(ctypes.byref(params), int(budget)))
    if cap < 1:
        raise KvecError(KVEC_ERR_INVALID_ARG, "invalid parameters or budget for the output capacity")
    return cap


def kvec_set_test_fault(fault: int) -> None:
    """Test hook of the error path (1: window kernels give up on a withheld accumulator; 0: off)."""
    load().kvec_set_test_fault(int(fault))


def kvec_decode_attention(handle: int, batch: int, q: int, k_cache: int, v_cache: int, lens: int, cap: int,
                          out: int, stream: int = 0) -> None:
    _check(load().kvec_decode_attention(handle, int(batch), q, k_cache, v_cache, lens, int(cap), out, stream))


def kvec_debug_scores(handle: int) -> kvec_debug_view:
    view = kvec_debug_view()
    _check(load().kvec_debug_scores(handle, ctypes.byref(view)))
    return view


def kvec_sync_status(handle: int) -> None:
    _check(load().kvec_sync_status(handle))


def kvec_set_profiling(handle: int, enable: bool) -> None:
    _check(load().kvec_set_profiling(handle, 1 if enable else 0))


def kvec_kernel_time(handle: int, kernel: int):
    ms, n = ctypes.c_double(), ctypes.c_int()
    _check(load().kvec_kernel_time(handle, int(kernel), ctypes.byref(ms), ctypes.byref(n)))
    return ms.value, n.value


def kvec_status_string(status: int) -> str:
    return load().kvec_status_string(int(status)).decode()


def make_params(num_q_heads: int, num_kv_heads: int, head_dim: int = 128, window: int = 32, obs_window: int = 16,
                ext_window: int = 32, pool_kernel: int = 7, num_ext_heads: int = 3, lam: float = 1.0,
                beta: float = 0.25, softmax_scale: float = 0.0, max_batch: int = 1, max_seqlen: int = 8192,
                max_layers: int = 32, pool_mode: int = 0, head_criterion: int = 0,
                all_positions: int = 0, head_budget: int = 0, ada_floor: float = 1.0) -> kvec_params:
    return kvec_params(num_q_heads, num_kv_heads, head_dim, window, obs_window, ext_window, pool_kernel,
                       num_ext_heads, lam, beta, softmax_scale, max_batch, max_seqlen, max_layers, pool_mode,
                       head_criterion, all_positions, head_budget, ada_floor)


def params_from_workload(wl, max_batch: Optional[int] = None, max_seqlen: Optional[int] = None,
                         max_layers: Optional[int] = None) -> kvec_params:
    return make_params(wl.num_q_heads, wl.num_kv_heads, wl.head_dim, wl.window, wl.obs_window, wl.ext_window,
                       wl.pool_kernel, wl.num_ext_heads, wl.lam, wl.beta, 0.0,
                       max_batch or wl.batch, max_seqlen or wl.max_seqlen, max_layers or max(wl.layers, 1),
                       getattr(wl, "pool_mode", 0), getattr(wl, "head_criterion", 0),
                       getattr(wl, "all_positions", 0), getattr(wl, "head_budget", 0),
                       getattr(wl, "ada_floor", 1.0))


class _DeviceArray:
    """Exposes a raw device pointer through __cuda_array_interface__ (zero copy)."""

    def __init__(self, ptr: int, shape, typestr: str):
        self.__cuda_array_interface__ = {"shape": tuple(shape), "typestr": typestr, "data": (int(ptr), False),
                                         "version": 3, "strides": None}


class KvecSelector:
    """Owns a kvec handle; torch tensors in, torch tensors out.  Marshalling only.

    torch provides device memory and streams; every step runs in libkvec.
    """

    def __init__(self, params: kvec_params):
        import torch
        self._torch = torch
        self.params = params
        self.handle = kvec_create(params)
        self.state_bytes = kvec_state_bytes(params.max_seqlen)

    def close(self) -> None:
        if self.handle:
            kvec_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def new_state(self, batch: int, device="cuda"):
        t = self._torch
        st = t.empty((batch, self.state_bytes), dtype=t.uint8, device=device)
        kvec_reset(self.handle, st.data_ptr(), batch, t.cuda.current_stream(st.device).cuda_stream)
        return st

    def alloc_outputs(self, batch: int, budget: int, device="cuda"):
        """out_idx, out_k, out_v with kvec_output_capacity rows per head."""
        t = self._torch
        p = self.params
        cap = kvec_output_capacity(p, budget)
        return (t.empty((batch, p.num_kv_heads, cap), dtype=t.int32, device=device),
                t.empty((batch, p.num_kv_heads, cap, p.head_dim), dtype=t.bfloat16, device=device),
                t.empty((batch, p.num_kv_heads, cap, p.head_dim), dtype=t.bfloat16, device=device))

    def select_layer(self, cu_host, cu_dev, q_obs, k, v, state, budget: int, outs=None, stream=None, lse=None):
        """lse: optional fp32 [batch][w][H_q] window-row log-sum-exp (kvec_select_layer_lse)."""
        t = self._torch
        batch = cu_host.numel() - 1
        if outs is None:
            outs = self.alloc_outputs(batch, budget, q_obs.device)
        s = stream if stream is not None else t.cuda.current_stream(q_obs.device)
        if lse is None:
            kvec_select_layer(self.handle, batch, cu_host.data_ptr(), cu_dev.data_ptr(), q_obs.data_ptr(),
                              k.data_ptr(), v.data_ptr(), state.data_ptr(), budget, outs[0].data_ptr(),
                              outs[1].data_ptr(), outs[2].data_ptr(), s.cuda_stream)
        else:
            kvec_select_layer_lse(self.handle, batch, cu_host.data_ptr(), cu_dev.data_ptr(), q_obs.data_ptr(),
                                  k.data_ptr(), v.data_ptr(), lse.data_ptr(), state.data_ptr(), budget,
                                  outs[0].data_ptr(), outs[1].data_ptr(), outs[2].data_ptr(), s.cuda_stream)
        return outs

    def select_layers(self, cu_host, cu_dev, qs, ks, vs, state, budget: int, outs, stream=None, lses=None):
        """lses: optional per-layer fp32 [batch][w][H_q] window-row log-sum-exp (kvec_select_layers_lse)."""
        t = self._torch
        batch = cu_host.numel() - 1
        s = stream if stream is not None else t.cuda.current_stream(qs[0].device)
        common = ([x.data_ptr() for x in qs], [x.data_ptr() for x in ks], [x.data_ptr() for x in vs])
        tail = ([o[0].data_ptr() for o in outs], [o[1].data_ptr() for o in outs], [o[2].data_ptr() for o in outs],
                s.cuda_stream)
        if lses is None:
            kvec_select_layers(self.handle, batch, cu_host.data_ptr(), cu_dev.data_ptr(), *common, state.data_ptr(),
                               budget, *tail)
        else:
            kvec_select_layers_lse(self.handle, batch, cu_host.data_ptr(), cu_dev.data_ptr(), *common,
                                   [x.data_ptr() for x in lses], state.data_ptr(), budget, *tail)
        return outs

    def decode_attention(self, q, k_cache, v_cache, lens, out=None, stream=None):
        """One decoding step over a compacted cache (kvec_decode_attention).

        q bf16 [batch][H_q][d]; k_cache, v_cache bf16 [batch][H_kv][cap][d];
        lens int32 [batch] on the device.  Returns fp32 [batch][H_q][d]."""
        t = self._torch
        batch, cap = q.shape[0], k_cache.shape[2]
        if out is None:
            out = t.empty((batch, q.shape[1], q.shape[2]), dtype=t.float32, device=q.device)
        s = stream if stream is not None else t.cuda.current_stream(q.device)
        kvec_decode_attention(self.handle, batch, q.data_ptr(), k_cache.data_ptr(), v_cache.data_ptr(),
                              lens.data_ptr(), cap, out.data_ptr(), s.cuda_stream)
        return out

    def debug(self, device="cuda"):
        """Copies of the last layer's intermediates (see kvec_debug_view)."""
        t = self._torch
        p = self.params
        v = kvec_debug_scores(self.handle)
        MB, H, ML, W = p.max_batch, p.num_kv_heads, v.max_seqlen, v.words_per_row
        R = (p.num_q_heads // p.num_kv_heads) * p.window

        def grab(ptr, shape, typestr):
            return t.as_tensor(_DeviceArray(ptr, shape, typestr), device=device).clone()

        return {
            "P_O": grab(v.P_O, (MB, H, ML), "<f4"), "P_Oext": grab(v.P_Oext, (MB, H, ML), "<f4"),
            "I": grab(v.I, (MB, ML), "<f4"), "sigma": grab(v.sigma, (MB, H), "<f4"),
            "htop": grab(v.htop, (MB, H), "<i4"), "pres_bits": grab(v.pres_bits, (MB, H, W), "<u4"),
            "Pprime": grab(v.Pprime, (MB, H, ML), "<f4"), "row_stats": grab(v.row_stats, (MB, H, R, 2), "<f4"),
        }
