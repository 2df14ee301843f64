"""Python binding of the BACON C ABI (``include/bacon.h``).

Argument marshalling only: every step of the compression runs in the CUDA
kernels of ``libbacon.so``.  torch tensors provide device memory and streams;
their raw pointers cross the ABI.  There is no CPU fallback: if the library
is missing, loading it raises.
"""

from __future__ import annotations

import ctypes
import os

import torch

LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libbacon.so")

BACON_OK, BACON_EINVAL, BACON_ENOMEM, BACON_ECUDA, BACON_ESTATE, BACON_ETIMEOUT, \
    BACON_EUNSUPPORTED = range(7)
STATUS_NAMES = {0: "BACON_OK", 1: "BACON_EINVAL", 2: "BACON_ENOMEM", 3: "BACON_ECUDA",
                4: "BACON_ESTATE", 5: "BACON_ETIMEOUT", 6: "BACON_EUNSUPPORTED"}
SCORE_KINDS = {"B": 0, "Q": 1, "E": 2, "V": 3, "Bpool": 4, "S": 5, "lambda": 6}

# every symbol include/bacon.h declares
EXPORTS = ("bacon_default_params", "bacon_init", "bacon_destroy", "bacon_last_error",
           "bacon_state_create", "bacon_state_reset", "bacon_state_destroy",
           "bacon_score_layer", "bacon_select", "bacon_compact",
           "bacon_compress_all_layers", "bacon_compress_host", "bacon_get_scores",
           "bacon_profile_enable", "bacon_profile_read", "bacon_window_scores_noalloc",
           "bacon_compress_layer_budgets", "bacon_pyramid_budgets",
           "bacon_compress_adaptive", "bacon_compress_with_lse", "bacon_sweep",
           "bacon_sync")
MAX_VARIANTS = 32
PROFILE_STAGES = ("window_stats", "window_combine", "window_scores", "calibrate_select",
                  "gather")


class BaconError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {message}")
        self.status = status


class Params(ctypes.Structure):
    """Mirror of ``bacon_params``."""
    _fields_ = [("r", ctypes.c_int), ("m", ctypes.c_int), ("rho", ctypes.c_int),
                ("gamma", ctypes.c_float), ("eps", ctypes.c_float),
                ("use_E", ctypes.c_int), ("use_L", ctypes.c_int), ("use_T", ctypes.c_int),
                ("keep_window", ctypes.c_int), ("max_seq_len", ctypes.c_int),
                ("max_requests", ctypes.c_int), ("keep_scores", ctypes.c_int)]


class Variant(ctypes.Structure):
    """Mirror of ``bacon_variant``."""
    _fields_ = [("r", ctypes.c_int), ("m", ctypes.c_int), ("rho", ctypes.c_int),
                ("gamma", ctypes.c_float), ("use_E", ctypes.c_int), ("use_L", ctypes.c_int),
                ("use_T", ctypes.c_int)]


_lib = None
_vp = ctypes.c_void_p
_int = ctypes.c_int


def load() -> ctypes.CDLL:
    """Load libbacon.so (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is missing: build it with "
                           "`python -m paper_2606_14782_gb300.build` (needs nvcc)")
    lib = ctypes.CDLL(LIB_PATH)
    lib.bacon_default_params.argtypes = [ctypes.POINTER(Params)]
    lib.bacon_default_params.restype = None
    lib.bacon_init.argtypes = [ctypes.POINTER(_vp), _int, _int, _int, _int, _int, _int, _int,
                               ctypes.POINTER(Params)]
    lib.bacon_destroy.argtypes = [_vp]
    lib.bacon_destroy.restype = None
    lib.bacon_last_error.argtypes = []
    lib.bacon_last_error.restype = ctypes.c_char_p
    lib.bacon_state_create.argtypes = [_vp, ctypes.POINTER(_vp)]
    lib.bacon_state_reset.argtypes = [_vp]
    lib.bacon_state_destroy.argtypes = [_vp]
    lib.bacon_state_destroy.restype = None
    lib.bacon_score_layer.argtypes = [_vp, _vp, _int, _vp, _vp, _int, _vp, _vp]
    lib.bacon_select.argtypes = [_vp, _vp, _int, _vp, _vp]
    lib.bacon_compact.argtypes = [_vp, _vp, _vp, _vp, _int, _int, _vp, _vp, _vp]
    lib.bacon_compress_all_layers.argtypes = [_vp, _int, ctypes.POINTER(_vp), ctypes.POINTER(_vp),
                                              ctypes.POINTER(_vp), _int, _int, ctypes.POINTER(_vp),
                                              ctypes.POINTER(_vp), _vp, _vp]
    lib.bacon_compress_host.argtypes = [_vp, _int, _vp, _vp, _vp, _int, _int, _vp, _vp, _vp, _vp]
    lib.bacon_get_scores.argtypes = [_vp, _int, _vp, ctypes.c_size_t, _vp]
    lib.bacon_sync.argtypes = [_vp, _vp]
    lib.bacon_compress_layer_budgets.argtypes = [_vp, _int, ctypes.POINTER(_vp),
                                                 ctypes.POINTER(_vp), ctypes.POINTER(_vp), _int,
                                                 ctypes.POINTER(_int), ctypes.POINTER(_vp),
                                                 ctypes.POINTER(_vp), ctypes.POINTER(_vp), _vp]
    lib.bacon_pyramid_budgets.argtypes = [_int, _int, _int, _int, ctypes.POINTER(_int)]
    lib.bacon_compress_with_lse.argtypes = [_vp, _int, ctypes.POINTER(_vp), ctypes.POINTER(_vp),
                                            ctypes.POINTER(_vp), ctypes.POINTER(_vp), _int, _int,
                                            ctypes.POINTER(_vp), ctypes.POINTER(_vp), _vp, _vp]
    lib.bacon_compress_adaptive.argtypes = [_vp, _int, ctypes.POINTER(_vp), ctypes.POINTER(_vp),
                                            ctypes.POINTER(_vp), _int, _int, ctypes.c_float,
                                            ctypes.POINTER(_vp), ctypes.POINTER(_vp),
                                            ctypes.POINTER(_vp), _vp, _vp]
    lib.bacon_sweep.argtypes = [_vp, _int, ctypes.POINTER(_vp), ctypes.POINTER(_vp), _int, _int,
                                _int, ctypes.POINTER(Variant), _vp, _vp, _vp]
    lib.bacon_pyramid_budgets.restype = None
    lib.bacon_window_scores_noalloc.argtypes = [_int, _int, _int, _int, _vp, _vp, _int, _vp,
                                                _vp, _vp, _vp]
    lib.bacon_profile_enable.argtypes = [_vp, _int]
    lib.bacon_profile_read.argtypes = [_vp, ctypes.POINTER(ctypes.c_double),
                                       ctypes.POINTER(_int), _int]
    for name in ("bacon_sweep", "bacon_compress_with_lse", "bacon_compress_adaptive",
                 "bacon_compress_layer_budgets",
                 "bacon_window_scores_noalloc",
                 "bacon_profile_enable", "bacon_profile_read",
                 "bacon_init", "bacon_state_create", "bacon_state_reset", "bacon_score_layer",
                 "bacon_select", "bacon_compact", "bacon_compress_all_layers",
                 "bacon_compress_host", "bacon_get_scores", "bacon_sync"):
        getattr(lib, name).restype = _int
    _lib = lib
    return lib


def _check(status: int):
    if status != BACON_OK:
        msg = load().bacon_last_error().decode(errors="replace")
        raise BaconError(status, msg)


def default_params(**overrides) -> Params:
    p = Params()
    load().bacon_default_params(ctypes.byref(p))
    for k, v in overrides.items():
        setattr(p, k, v)
    return p


def _stream_ptr(stream) -> int:
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream


def _ptr(t) -> int | None:
    return None if t is None else t.data_ptr()


def _ptr_array(ptrs):
    arr = (_vp * len(ptrs))()
    for i, p in enumerate(ptrs):
        arr[i] = p
    return arr


def _pair_table(t, pairs):
    """Pointers of t[r, l] for pair i = r * layers + l of a contiguous
    [R, layers, ...] tensor."""
    if not t.is_contiguous():
        raise ValueError("tensors must be contiguous")
    base, stride = t.data_ptr(), t[0, 0].numel() * t.element_size()
    return _ptr_array([base + stride * i for i in range(pairs)])


class Context:
    """Owns a ``bacon_ctx`` (one model shape)."""

    def __init__(self, layers, kv_heads, q_heads, head_dim, window, pool=7, budget=None,
                 params: Params | None = None, **param_overrides):
        lib = load()
        if params is None:
            params = default_params(**param_overrides)
        self.params = params
        self.layers, self.kv_heads, self.q_heads = layers, kv_heads, q_heads
        self.head_dim, self.window, self.pool = head_dim, window, pool
        self.budget = budget if budget is not None else window
        h = _vp()
        _check(lib.bacon_init(ctypes.byref(h), layers, kv_heads, q_heads, head_dim, window,
                              pool, self.budget, ctypes.byref(params)))
        self.handle = h

    def close(self):
        if getattr(self, "handle", None):
            load().bacon_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    # -------------------------------------------------------- whole step
    def compress_all_layers(self, qwin, k, v, budget, k_out=None, v_out=None, idx_out=None,
                            stream=None):
        """qwin [R, layers, Hq, W, d], k/v [R, layers, Hkv, N, d] (bf16, cuda,
        contiguous).  Returns (k_out, v_out, idx) with shapes
        [R, layers, Hkv, kept, d] and [R, layers, Hkv, kept]."""
        R, Ly, Hq, W, d = qwin.shape
        N = k.shape[3]
        kept = min(budget, N)
        shape_o = (R, Ly, self.kv_heads, kept, d)
        if k_out is None:
            k_out = torch.empty(shape_o, dtype=k.dtype, device=k.device)
        if v_out is None:
            v_out = torch.empty(shape_o, dtype=v.dtype, device=v.device)
        if idx_out is None:
            idx_out = torch.empty(shape_o[:-1], dtype=torch.int32, device=k.device)
        for t in (qwin, k, v, k_out, v_out, idx_out):
            if not t.is_contiguous():
                raise ValueError("tensors must be contiguous")
        tq, tk, tv, tko, tvo = (_pair_table(t, R * Ly) for t in (qwin, k, v, k_out, v_out))
        _check(load().bacon_compress_all_layers(self.handle, R, tq, tk, tv, N, budget, tko, tvo,
                                                idx_out.data_ptr(), _stream_ptr(stream)))
        self._last_units, self._last_N = R * Ly * self.kv_heads, N
        return k_out, v_out, idx_out

    def compress_layer_budgets(self, qwin, k, v, layer_budgets, stream=None):
        """Per-layer budgets (window included).  Returns lists indexed
        [request][layer] of k_out [Hkv, kept_l, d], v_out and idx [Hkv, kept_l]."""
        R, Ly, Hq, W, d = qwin.shape
        N = k.shape[3]
        assert len(layer_budgets) == Ly
        kept = [min(int(b), N) for b in layer_budgets]
        ko = [[torch.empty((self.kv_heads, kept[l], d), dtype=k.dtype, device=k.device)
               for l in range(Ly)] for _ in range(R)]
        vo = [[torch.empty_like(ko[r][l]) for l in range(Ly)] for r in range(R)]
        ix = [[torch.empty((self.kv_heads, kept[l]), dtype=torch.int32, device=k.device)
               for l in range(Ly)] for _ in range(R)]
        pairs = [(r, l) for r in range(R) for l in range(Ly)]
        tq = _ptr_array([qwin[r, l].data_ptr() for r, l in pairs])
        tk = _ptr_array([k[r, l].data_ptr() for r, l in pairs])
        tv = _ptr_array([v[r, l].data_ptr() for r, l in pairs])
        tko = _ptr_array([ko[r][l].data_ptr() for r, l in pairs])
        tvo = _ptr_array([vo[r][l].data_ptr() for r, l in pairs])
        tix = _ptr_array([ix[r][l].data_ptr() for r, l in pairs])
        b = (_int * Ly)(*[int(x) for x in layer_budgets])
        _check(load().bacon_compress_layer_budgets(self.handle, R, tq, tk, tv, N, b, tko, tvo,
                                                   tix, _stream_ptr(stream)))
        self._last_units, self._last_N = R * Ly * self.kv_heads, N
        return ko, vo, ix

    def compress_with_lse(self, qwin, k, v, lse, budget, k_out=None, v_out=None, idx_out=None,
                          stream=None):
        """As compress_all_layers, with the window rows' natural-log softmax
        normalisers lse [R, layers, Hq, W] (fp32, cuda) from the prefill."""
        R, Ly, Hq, W, d = qwin.shape
        N = k.shape[3]
        kept = min(budget, N)
        shape_o = (R, Ly, self.kv_heads, kept, d)
        k_out = torch.empty(shape_o, dtype=k.dtype, device=k.device) if k_out is None else k_out
        v_out = torch.empty(shape_o, dtype=v.dtype, device=v.device) if v_out is None else v_out
        if idx_out is None:
            idx_out = torch.empty(shape_o[:-1], dtype=torch.int32, device=k.device)
        tq, tk, tv, tl, tko, tvo = (_pair_table(t, R * Ly) for t in (qwin, k, v, lse, k_out, v_out))
        _check(load().bacon_compress_with_lse(self.handle, R, tq, tk, tv, tl, N, budget, tko, tvo,
                                              idx_out.data_ptr(), _stream_ptr(stream)))
        self._last_units, self._last_N = R * Ly * self.kv_heads, N
        return k_out, v_out, idx_out

    def compress_adaptive(self, qwin, k, v, budget, alpha=0.2, stream=None):
        """AdaKV-style head budgets.  Returns (k_out, v_out, idx, counts):
        k_out/v_out [R, layers, Hkv * kept, d] and idx [R, layers, Hkv * kept]
        flat per layer (heads in order), counts [R, layers, Hkv]."""
        R, Ly, Hq, W, d = qwin.shape
        N = k.shape[3]
        kept = min(budget, N)
        ko = torch.empty((R, Ly, self.kv_heads * kept, d), dtype=k.dtype, device=k.device)
        vo = torch.empty_like(ko)
        ix = torch.empty((R, Ly, self.kv_heads * kept), dtype=torch.int32, device=k.device)
        counts = torch.empty((R, Ly, self.kv_heads), dtype=torch.int32, device=k.device)
        tq, tk, tv, tko, tvo, tix = (_pair_table(t, R * Ly) for t in (qwin, k, v, ko, vo, ix))
        _check(load().bacon_compress_adaptive(self.handle, R, tq, tk, tv, N, budget,
                                              float(alpha), tko, tvo, tix, counts.data_ptr(),
                                              _stream_ptr(stream)))
        self._last_units, self._last_N = R * Ly * self.kv_heads, N
        return ko, vo, ix, counts

    def sweep(self, qwin, k, budget, variants, idx_out=None, lambda_out=None, stream=None):
        """Selections under several hyper-parameter sets from one set of
        window passes.  variants: sequence of dicts with any of r, m, rho,
        gamma, use_E, use_L, use_T (the rest from the context's parameters).
        Returns (idx [V, R, layers, Hkv, kept] int32, lambda [V, R, layers,
        Hkv] fp32)."""
        R, Ly, Hq, W, d = qwin.shape
        N = k.shape[3]
        kept = min(budget, N)
        nv = len(variants)
        arr = (Variant * max(nv, 1))()
        for j, x in enumerate(variants):
            for f, _ in Variant._fields_:
                setattr(arr[j], f, x.get(f, getattr(self.params, f)))
        if idx_out is None:
            idx_out = torch.empty((nv, R, Ly, self.kv_heads, kept), dtype=torch.int32,
                                  device=k.device)
        if lambda_out is None:
            lambda_out = torch.empty((nv, R, Ly, self.kv_heads), dtype=torch.float32,
                                     device=k.device)
        tq, tk = (_pair_table(t, R * Ly) for t in (qwin, k))
        _check(load().bacon_sweep(self.handle, R, tq, tk, N, budget, nv, arr,
                                  idx_out.data_ptr(), lambda_out.data_ptr(),
                                  _stream_ptr(stream)))
        return idx_out, lambda_out

    def compress_host(self, qwin, k, v, budget, k_out=None, v_out=None, idx_out=None,
                      stream=None):
        """The same step on host (CPU, ideally pinned) tensors; blocks until
        the outputs are on the host."""
        R, Ly, Hq, W, d = qwin.shape
        N = k.shape[3]
        kept = min(budget, N)
        shape_o = (R, Ly, self.kv_heads, kept, d)
        pin = k.is_pinned()
        if k_out is None:
            k_out = torch.empty(shape_o, dtype=k.dtype, pin_memory=pin)
        if v_out is None:
            v_out = torch.empty(shape_o, dtype=v.dtype, pin_memory=pin)
        if idx_out is None:
            idx_out = torch.empty(shape_o[:-1], dtype=torch.int32, pin_memory=pin)
        _check(load().bacon_compress_host(self.handle, R, qwin.data_ptr(), k.data_ptr(),
                                          v.data_ptr(), N, budget, k_out.data_ptr(),
                                          v_out.data_ptr(), idx_out.data_ptr(),
                                          _stream_ptr(stream)))
        self._last_units, self._last_N = R * Ly * self.kv_heads, N
        return k_out, v_out, idx_out

    def scores(self, kind: str, out=None, stream=None):
        """Intermediate per-token arrays of the last whole-step call (fp32)."""
        n = self._last_count(kind)
        if out is None:
            out = torch.empty(n, dtype=torch.float32, device="cuda")
        _check(load().bacon_get_scores(self.handle, SCORE_KINDS[kind], out.data_ptr(),
                                       out.numel(), _stream_ptr(stream)))
        return out

    def _last_count(self, kind):
        return self._last_units * (1 if kind == "lambda" else self._last_N)

    def sync(self, stream=None):
        _check(load().bacon_sync(self.handle, _stream_ptr(stream)))

    def profile(self, enable: bool):
        _check(load().bacon_profile_enable(self.handle, int(enable)))

    def profile_read(self):
        """{stage: (total ms, launches)} since the previous read."""
        n = len(PROFILE_STAGES)
        ms = (ctypes.c_double * n)()
        cnt = (_int * n)()
        _check(load().bacon_profile_read(self.handle, ms, cnt, n))
        return {name: (ms[i], cnt[i]) for i, name in enumerate(PROFILE_STAGES)}

    # ----------------------------------------------- layer by layer
    def compact(self, k, v, idx, k_out=None, v_out=None, stream=None):
        """k/v [Hkv, N, d], idx [Hkv, count] int32 (cuda)."""
        Hkv, N, d = k.shape
        count = idx.shape[-1]
        if k_out is None:
            k_out = torch.empty((Hkv, count, d), dtype=k.dtype, device=k.device)
        if v_out is None:
            v_out = torch.empty((Hkv, count, d), dtype=v.dtype, device=v.device)
        _check(load().bacon_compact(self.handle, k.data_ptr(), v.data_ptr(), idx.data_ptr(), N,
                                    count, k_out.data_ptr(), v_out.data_ptr(),
                                    _stream_ptr(stream)))
        return k_out, v_out


def pyramid_budgets(layers, window, budget, beta=20):
    """The library's pyramid budget schedule (bacon_pyramid_budgets)."""
    out = (_int * layers)()
    load().bacon_pyramid_budgets(layers, window, budget, beta, out)
    return list(out)


class State:
    """Per-request persistence state for layer-by-layer scoring."""

    def __init__(self, ctx: Context):
        self.ctx = ctx
        h = _vp()
        _check(load().bacon_state_create(ctx.handle, ctypes.byref(h)))
        self.handle = h

    def close(self):
        if getattr(self, "handle", None):
            load().bacon_state_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def reset(self):
        _check(load().bacon_state_reset(self.handle))

    def score_layer(self, layer, qwin, k, scores_out=None, stream=None):
        """qwin [Hq, W, d], k [Hkv, N, d] of one layer; returns S [Hkv, N]
        when scores_out is given or requested (pass True)."""
        N = k.shape[1]
        if scores_out is True:
            scores_out = torch.empty((self.ctx.kv_heads, N), dtype=torch.float32,
                                     device=k.device)
        _check(load().bacon_score_layer(self.ctx.handle, self.handle, layer, qwin.data_ptr(),
                                        k.data_ptr(), N, _ptr(scores_out), _stream_ptr(stream)))
        return scores_out

    def select(self, budget, N, idx_out=None, stream=None, device="cuda"):
        kept = min(budget, N)
        if idx_out is None:
            idx_out = torch.empty((self.ctx.kv_heads, kept), dtype=torch.int32, device=device)
        _check(load().bacon_select(self.ctx.handle, self.handle, budget, idx_out.data_ptr(),
                                   _stream_ptr(stream)))
        return idx_out
