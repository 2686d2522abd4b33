"""Python binding of libkvevict.so (include/kv_evict.h): argument marshalling only.

Every step runs in the library's CUDA kernels; tensors are torch tensors used as
device buffers and passed by pointer. Loading fails loudly when the library has
not been built (``python -c "import __graft_entry__ as g; g.build()"``).
"""

from __future__ import annotations

import ctypes
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libkvevict.so")

KVE_OK, KVE_EINVAL, KVE_ECUDA, KVE_ETIMEOUT, KVE_ENOMEM = range(5)

# Names declared in include/kv_evict.h.
EXPORTS = ("kv_evict_plan", "kv_evict_plan_layered", "kv_evict_plan_ex", "kv_evict_plan_destroy",
           "kv_evict_plan_set_debug", "kv_evict_plan_set_kv_strides",
           "kv_evict_score", "kv_evict_score_lse", "kv_evict_score_attn", "kv_evict_score_attn_workspace",
           "kv_evict_select", "kv_evict_select_noalloc", "kv_evict_select_profiles",
           "kv_evict_select_profiles_workspace", "kv_evict_gather", "kv_evict_select_gather",
           "kv_evict_status", "kv_evict_profile", "kv_evict_budget_pyramid", "kv_evict_strerror")


class KvEvictError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        super().__init__(f"{what}: {_lib().kv_evict_strerror(status).decode()} (status {status})")


class Config(ctypes.Structure):
    _fields_ = [("num_layers", ctypes.c_int32), ("num_q_heads", ctypes.c_int32),
                ("num_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("window", ctypes.c_int32), ("budget", ctypes.c_int32),
                ("pool_kernel", ctypes.c_int32), ("candidate_factor", ctypes.c_int32),
                ("norm_eps", ctypes.c_float)]


_LIB = None


def _lib():
    global _LIB
    if _LIB is None:
        if not os.path.exists(LIB_PATH):
            raise ImportError(f"{LIB_PATH} is missing: build the CUDA library first "
                              "(python -c 'import __graft_entry__ as g; g.build()')")
        lib = ctypes.CDLL(LIB_PATH)
        vp, i32, i64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
        lib.kv_evict_plan.argtypes = [ctypes.POINTER(Config), ctypes.POINTER(i64), i32,
                                      ctypes.POINTER(vp), ctypes.POINTER(ctypes.c_size_t)]
        lib.kv_evict_plan_layered.argtypes = [ctypes.POINTER(Config), ctypes.POINTER(i64), i32, vp,
                                              ctypes.POINTER(vp), ctypes.POINTER(ctypes.c_size_t)]
        lib.kv_evict_plan_ex.argtypes = [ctypes.POINTER(Config), ctypes.POINTER(i64), i32, vp, i32,
                                         vp, vp]
        lib.kv_evict_budget_pyramid.argtypes = [i32, i32, ctypes.c_float, vp]
        lib.kv_evict_plan_destroy.argtypes = [vp]
        lib.kv_evict_plan_destroy.restype = None
        lib.kv_evict_plan_set_debug.argtypes = [vp, ctypes.c_uint64, i32]
        lib.kv_evict_plan_set_kv_strides.argtypes = [vp, vp, vp]
        lib.kv_evict_score.argtypes = [vp] * 7
        lib.kv_evict_score_lse.argtypes = [vp] * 8
        lib.kv_evict_score_attn.argtypes = [vp] * 10
        lib.kv_evict_score_attn_workspace.argtypes = [vp, vp]
        lib.kv_evict_select.argtypes = [vp] * 11
        lib.kv_evict_select_noalloc.argtypes = [vp] * 10
        lib.kv_evict_select_profiles.argtypes = [vp, i32] + [vp] * 10
        lib.kv_evict_select_profiles_workspace.argtypes = [vp, i32, vp]
        lib.kv_evict_gather.argtypes = [vp] * 7
        lib.kv_evict_select_gather.argtypes = [vp] * 14
        lib.kv_evict_status.argtypes = [vp, vp, vp]
        lib.kv_evict_profile.argtypes = [i32, vp, i32, vp, vp]
        lib.kv_evict_strerror.argtypes = [ctypes.c_int]
        lib.kv_evict_strerror.restype = ctypes.c_char_p
        for name in ("kv_evict_plan", "kv_evict_plan_layered", "kv_evict_plan_ex", "kv_evict_plan_set_debug",
                     "kv_evict_plan_set_kv_strides",
                     "kv_evict_score", "kv_evict_score_lse", "kv_evict_score_attn", "kv_evict_score_attn_workspace",
                     "kv_evict_select", "kv_evict_select_noalloc",
                     "kv_evict_select_profiles", "kv_evict_select_profiles_workspace", "kv_evict_gather",
                     "kv_evict_select_gather", "kv_evict_status", "kv_evict_profile",
                     "kv_evict_budget_pyramid"):
            getattr(lib, name).restype = ctypes.c_int
        _LIB = lib
    return _LIB


def library():
    """The loaded ctypes library (loads it on first use)."""
    return _lib()


def _ptr(t):
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _check(status: int, what: str):
    if status != KVE_OK:
        raise KvEvictError(status, what)


def _stream_ptr(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def make_config(spec: dict) -> Config:
    return Config(spec["num_layers"], spec["num_q_heads"], spec["num_kv_heads"], spec["head_dim"],
                  spec["window"], spec["budget"], spec.get("pool_kernel", 7),
                  spec.get("candidate_factor", 4), spec.get("norm_eps", 1e-12))


KVE_PLAN_PER_QUERY_HEAD = 1


class Plan:
    """kv_evict_plan (kv_evict_plan_layered when layer_budgets is given,
    kv_evict_plan_ex with KVE_PLAN_PER_QUERY_HEAD when per_query_head) for a
    configuration and the prefix lengths of the requests."""

    def __init__(self, spec: dict, seq_lens, layer_budgets=None, per_query_head: bool = False,
                 k_strides=None, v_strides=None):
        lib = _lib()
        self.spec = dict(spec)
        self.seq_lens = [int(x) for x in seq_lens]
        self._cfg = make_config(spec)
        lens = (ctypes.c_int64 * len(self.seq_lens))(*self.seq_lens)
        handle = ctypes.c_void_p()
        ws = ctypes.c_size_t()
        self.per_query_head = bool(per_query_head)
        if self.per_query_head:
            self.layer_budgets = ([int(spec["budget"])] * int(spec["num_layers"]) if layer_budgets is None
                                  else [int(b) for b in layer_budgets])
            lb = np.ascontiguousarray(self.layer_budgets, dtype=np.int32)
            _check(lib.kv_evict_plan_ex(ctypes.byref(self._cfg), lens, len(self.seq_lens), lb.ctypes.data,
                                        KVE_PLAN_PER_QUERY_HEAD, ctypes.byref(handle), ctypes.byref(ws)),
                   "kv_evict_plan_ex")
        elif layer_budgets is None:
            self.layer_budgets = [int(spec["budget"])] * int(spec["num_layers"])
            _check(lib.kv_evict_plan(ctypes.byref(self._cfg), lens, len(self.seq_lens),
                                     ctypes.byref(handle), ctypes.byref(ws)), "kv_evict_plan")
        else:
            self.layer_budgets = [int(b) for b in layer_budgets]
            lb = np.ascontiguousarray(self.layer_budgets, dtype=np.int32)
            _check(lib.kv_evict_plan_layered(ctypes.byref(self._cfg), lens, len(self.seq_lens),
                                             lb.ctypes.data, ctypes.byref(handle), ctypes.byref(ws)),
                   "kv_evict_plan_layered")
        self._h = handle
        self.workspace_bytes = ws.value
        if k_strides is not None or v_strides is not None:
            self.set_kv_strides(k_strides, v_strides)

    def __del__(self):
        h = getattr(self, "_h", None)
        if h is not None and h.value and _LIB is not None:
            _LIB.kv_evict_plan_destroy(h)
            self._h = None

    # -- sizes of the documented layouts
    @property
    def unit_heads(self) -> int:
        """Heads per layer that own a unit: KV heads, or query heads per_query_head."""
        return self.spec["num_q_heads"] if self.per_query_head else self.spec["num_kv_heads"]

    @property
    def n_units(self) -> int:
        return len(self.seq_lens) * self.spec["num_layers"] * self.unit_heads

    @property
    def score_elems(self) -> int:
        return self.spec["num_layers"] * self.unit_heads * sum(self.seq_lens)

    def set_kv_strides(self, k_strides=None, v_strides=None):
        """kv_evict_plan_set_kv_strides: element strides (layer, KV head, token) of k
        and v, None for the dense default. For a torch tensor viewed as
        [N_L][Hkv][SL][d], pass t.stride()[:3]."""
        ks = None if k_strides is None else np.ascontiguousarray(k_strides, dtype=np.int64)
        vs = None if v_strides is None else np.ascontiguousarray(v_strides, dtype=np.int64)
        _check(_lib().kv_evict_plan_set_kv_strides(self._h, None if ks is None else ks.ctypes.data,
                                                    None if vs is None else vs.ctypes.data),
               "kv_evict_plan_set_kv_strides")

    def set_debug(self, wait_limit_ns: int, fault: int = 0):
        _check(_lib().kv_evict_plan_set_debug(self._h, int(wait_limit_ns), int(fault)),
               "kv_evict_plan_set_debug")

    def score(self, q_win, k, mu, sigma, ws, stream=None):
        _check(_lib().kv_evict_score(self._h, _ptr(q_win), _ptr(k), _ptr(mu), _ptr(sigma), _ptr(ws),
                                     _stream_ptr(stream)), "kv_evict_score")

    def score_lse(self, q_win, k, lse, mu, sigma, ws, stream=None):
        """kv_evict_score_lse: the column pass only, given every window row's natural-log
        softmax normaliser lse (fp32, q_win's row order)."""
        _check(_lib().kv_evict_score_lse(self._h, _ptr(q_win), _ptr(k), _ptr(lse), _ptr(mu), _ptr(sigma),
                                         _ptr(ws), _stream_ptr(stream)), "kv_evict_score_lse")

    def score_attn_workspace(self) -> int:
        """Bytes of the second scratch buffer of score_attn."""
        out = ctypes.c_size_t(0)
        _check(_lib().kv_evict_score_attn_workspace(self._h, ctypes.byref(out)),
               "kv_evict_score_attn_workspace")
        return out.value

    def score_attn(self, q_win, k, v, mu, sigma, o_win, ws, attn_ws, stream=None):
        """kv_evict_score_attn: score plus the window rows' attention output o_win
        (q_win's layout, bf16)."""
        _check(_lib().kv_evict_score_attn(self._h, _ptr(q_win), _ptr(k), _ptr(v), _ptr(mu), _ptr(sigma),
                                          _ptr(o_win), _ptr(ws), _ptr(attn_ws), _stream_ptr(stream)),
               "kv_evict_score_attn")

    def select(self, mu, sigma, k, lambda1, lambda2, indices, ws, order=None, margins=None,
               stream=None):
        l1 = np.ascontiguousarray(lambda1, dtype=np.float32)
        l2 = np.ascontiguousarray(lambda2, dtype=np.float32)
        assert l1.shape == (self.spec["num_layers"],) and l2.shape == l1.shape
        _check(_lib().kv_evict_select(self._h, _ptr(mu), _ptr(sigma), _ptr(k),
                                      l1.ctypes.data, l2.ctypes.data, _ptr(indices), _ptr(order),
                                      _ptr(margins), _ptr(ws), _stream_ptr(stream)),
               "kv_evict_select")

    def select_noalloc(self, mu, sigma, k, lambda1, lambda2, indices, order=None, margins=None,
                       stream=None):
        """kv_evict_select without a workspace, for callers that cannot allocate
        device memory while they evict; its scratch is a fixed 16 MiB array inside
        the library (at most N_L * units per layer * SL = 4194304 tokens per call).
        status(None) reads its error word."""
        l1 = np.ascontiguousarray(lambda1, dtype=np.float32)
        l2 = np.ascontiguousarray(lambda2, dtype=np.float32)
        assert l1.shape == (self.spec["num_layers"],) and l2.shape == l1.shape
        _check(_lib().kv_evict_select_noalloc(self._h, _ptr(mu), _ptr(sigma), _ptr(k),
                                              l1.ctypes.data, l2.ctypes.data, _ptr(indices),
                                              _ptr(order), _ptr(margins), _stream_ptr(stream)),
               "kv_evict_select_noalloc")

    def select_profiles_workspace(self, n_profiles: int) -> int:
        """Bytes of scratch that select_profiles needs for n_profiles profiles."""
        out = ctypes.c_size_t(0)
        _check(_lib().kv_evict_select_profiles_workspace(self._h, int(n_profiles), ctypes.byref(out)),
               "kv_evict_select_profiles_workspace")
        return out.value

    def select_profiles(self, mu, sigma, k, lambda1, lambda2, indices, ws, order=None, margins=None,
                        stream=None):
        """Selection for P coefficient profiles at once: lambda1 / lambda2 are
        [P, N_L]; indices (and order / margins) are [P, n_units, B]; ws holds
        select_profiles_workspace(P) bytes."""
        l1 = np.ascontiguousarray(lambda1, dtype=np.float32)
        l2 = np.ascontiguousarray(lambda2, dtype=np.float32)
        assert l1.ndim == 2 and l1.shape[1] == self.spec["num_layers"] and l2.shape == l1.shape
        _check(_lib().kv_evict_select_profiles(self._h, int(l1.shape[0]), _ptr(mu), _ptr(sigma), _ptr(k),
                                               l1.ctypes.data, l2.ctypes.data, _ptr(indices),
                                               _ptr(order), _ptr(margins), _ptr(ws),
                                               _stream_ptr(stream)),
               "kv_evict_select_profiles")

    def gather(self, k, v, indices, k_out, v_out, stream=None):
        """kv_evict_gather. k and v may be pinned CPU tensors (read in place by the
        kernel; only the kept rows cross the host link); pageable CPU tensors are
        refused."""
        for name, t in (("k", k), ("v", v)):
            dev = getattr(t, "device", None)
            if dev is not None and getattr(dev, "type", None) == "cpu" and not t.is_pinned():
                raise ValueError(f"gather: {name} is a pageable CPU tensor; pin it or move it to the GPU")
        _check(_lib().kv_evict_gather(self._h, _ptr(k), _ptr(v), _ptr(indices), _ptr(k_out),
                                      _ptr(v_out), _stream_ptr(stream)), "kv_evict_gather")

    def select_gather(self, mu, sigma, k, v, lambda1, lambda2, indices, k_out, v_out, ws, order=None,
                      margins=None, stream=None):
        """kv_evict_select_gather: select, then the compact cache, in one launch (the
        outputs of select followed by gather). v (and k) may be pinned CPU tensors."""
        for name, t in (("k", k), ("v", v)):
            dev = getattr(t, "device", None)
            if dev is not None and getattr(dev, "type", None) == "cpu" and not t.is_pinned():
                raise ValueError(f"select_gather: {name} is a pageable CPU tensor; pin it or move it to the GPU")
        l1 = np.ascontiguousarray(lambda1, dtype=np.float32)
        l2 = np.ascontiguousarray(lambda2, dtype=np.float32)
        assert l1.shape == (self.spec["num_layers"],) and l2.shape == l1.shape
        _check(_lib().kv_evict_select_gather(self._h, _ptr(mu), _ptr(sigma), _ptr(k), _ptr(v),
                                             l1.ctypes.data, l2.ctypes.data, _ptr(indices), _ptr(order),
                                             _ptr(margins), _ptr(k_out), _ptr(v_out), _ptr(ws),
                                             _stream_ptr(stream)), "kv_evict_select_gather")

    def status(self, ws, stream=None) -> int:
        """Synchronise, return the device status (KVE_OK, KVE_ETIMEOUT or KVE_ECUDA) of
        ws and clear it; ws = None reads the error word of select_noalloc."""
        return int(_lib().kv_evict_status(self._h, _ptr(ws), _stream_ptr(stream)))


def profile(kind: str, c, num_layers: int, seg_bounds=None) -> np.ndarray:
    """Eq. 6 depth profile computed by the library (kind: global/segments/curve)."""
    k = {"global": 0, "segments": 1, "curve": 2}[kind]
    cc = np.zeros(3, dtype=np.float32)
    cc[: len(np.atleast_1d(c))] = np.atleast_1d(c)
    out = np.zeros(num_layers, dtype=np.float32)
    sb = None if seg_bounds is None else np.ascontiguousarray(seg_bounds, dtype=np.int32)
    _check(_lib().kv_evict_profile(k, cc.ctypes.data, num_layers,
                                   None if sb is None else sb.ctypes.data, out.ctypes.data),
           "kv_evict_profile")
    return out


def budget_pyramid(budget: int, num_layers: int, last_ratio: float) -> np.ndarray:
    """kv_evict_budget_pyramid: a depth-decreasing schedule with the uniform total."""
    out = np.zeros(num_layers, dtype=np.int32)
    _check(_lib().kv_evict_budget_pyramid(int(budget), int(num_layers), float(last_ratio),
                                          out.ctypes.data), "kv_evict_budget_pyramid")
    return out


class Buffers:
    """Device outputs and workspace of one call, allocated with torch."""

    def __init__(self, plan: Plan, device="cuda", with_trace: bool = True):
        import torch
        B, W, d = plan.spec["budget"], plan.spec["window"], plan.spec["head_dim"]
        n = plan.n_units
        self.mu = torch.empty(plan.score_elems, dtype=torch.float32, device=device)
        self.sigma = torch.empty_like(self.mu)
        self.indices = torch.empty((n, B), dtype=torch.int32, device=device)
        self.order = torch.empty((n, B), dtype=torch.int32, device=device) if with_trace else None
        self.margins = torch.empty((n, B), dtype=torch.float32, device=device) if with_trace else None
        self.k_out = torch.empty((n, B + W, d), dtype=torch.bfloat16, device=device)
        self.v_out = torch.empty_like(self.k_out)
        self.ws = torch.empty(plan.workspace_bytes, dtype=torch.uint8, device=device)


def run_step(plan: Plan, bufs: Buffers, q_win, k, v, lambda1, lambda2, stream=None, fused=True):
    """The whole eviction step: score, then select with the compact cache in one call
    (fused), or select and gather as two calls."""
    plan.score(q_win, k, bufs.mu, bufs.sigma, bufs.ws, stream)
    if fused:
        plan.select_gather(bufs.mu, bufs.sigma, k, v, lambda1, lambda2, bufs.indices, bufs.k_out,
                           bufs.v_out, bufs.ws, bufs.order, bufs.margins, stream)
        return
    plan.select(bufs.mu, bufs.sigma, k, lambda1, lambda2, bufs.indices, bufs.ws, bufs.order,
                bufs.margins, stream)
    plan.gather(k, v, bufs.indices, bufs.k_out, bufs.v_out, stream)
