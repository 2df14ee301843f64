"""BACON CPU oracle -- TEST INFRASTRUCTURE ONLY.

A plain, slow, double-precision restatement of the BACON scoring method
(Sections 4.1-4.4, Eqs. 1-17), used to check the CUDA library.  Only the
tests, ``__graft_entry__.smoke()`` and the benchmark's ``cpu_baseline`` /
``--impl reference`` legs may import it.  The arithmetic lives in
``bacon_oracle.c``; this module only marshals numpy arrays and runs
independent (request, kv-head) chains on host threads.  It imports nothing
from the CUDA package, and the CUDA package never imports it.

Readings of the paper where it is silent (all shared with the CUDA path's
specification, not with its code):

* GQA: the G query heads of a kv-head are averaged into one window score and
  one last-query score before the residual (Eq. 4).
* The backbone score used from Eq. 12 on is the 1-D max pool (width 7) of
  Eq. 1's score over the candidates; Eq. 4 uses the unpooled score.
* Candidates are [0, N-W); the W window tokens are always kept and count
  against the budget, so K_{l,h} = budget - W.
* gamma = 1, eps = 1e-8, population standard deviation, ties broken towards
  the lower position, 0-based positions.
"""

from __future__ import annotations

import ctypes
import dataclasses
import os
import subprocess
import threading
from concurrent.futures import ThreadPoolExecutor

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "bacon_oracle.c")
_HDR = os.path.join(_HERE, "bacon_oracle.h")
_LIB_PATH = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with plain gcc (no fast-math) into liboracle.so."""
    stale = (not os.path.exists(_LIB_PATH)) or any(
        os.path.getmtime(s) > os.path.getmtime(_LIB_PATH) for s in (_SRC, _HDR))
    if force or stale:
        tmp = _LIB_PATH + f".{os.getpid()}.tmp"
        subprocess.check_call(["gcc", "-std=c11", "-O2", "-fPIC", "-shared",
                               "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


class _Params(ctypes.Structure):
    _fields_ = [("r", ctypes.c_int), ("m", ctypes.c_int), ("rho", ctypes.c_int),
                ("gamma", ctypes.c_double), ("eps", ctypes.c_double),
                ("use_E", ctypes.c_int), ("use_L", ctypes.c_int),
                ("use_T", ctypes.c_int), ("pool_kernel", ctypes.c_int),
                ("keep_window", ctypes.c_int)]


@dataclasses.dataclass
class Params:
    """Hyper-parameters of Sections 4.3-4.4 (defaults as the paper states,
    gamma/eps/pool as read where it is silent)."""
    r: int = 5
    m: int = 4
    rho: int = 2
    gamma: float = 1.0
    eps: float = 1e-8
    use_E: bool = True
    use_L: bool = True
    use_T: bool = True
    pool_kernel: int = 7
    keep_window: bool = True

    def _c(self) -> _Params:
        return _Params(int(self.r), int(self.m), int(self.rho), float(self.gamma),
                       float(self.eps), int(self.use_E), int(self.use_L),
                       int(self.use_T), int(self.pool_kernel), int(self.keep_window))


_D = ctypes.POINTER(ctypes.c_double)
_I32 = ctypes.POINTER(ctypes.c_int32)
_U16 = ctypes.POINTER(ctypes.c_uint16)


def _lib_handle():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            c_int, c_double = ctypes.c_int, ctypes.c_double
            lib.bo_window_scores.argtypes = [_D, _D, c_int, c_int, c_int, c_int, _D, _D]
            lib.bo_residual.argtypes = [_D, _D, c_int, _D]
            lib.bo_coherence.argtypes = [_D, c_int, c_int, _D]
            lib.bo_persistence.argtypes = [ctypes.POINTER(_D), c_int, c_int, _D]
            lib.bo_evidence.argtypes = [_D, _D, _D, c_int, c_int, c_int, c_int, _D]
            lib.bo_maxpool.argtypes = [_D, c_int, c_int, _D]
            lib.bo_rank_topk.argtypes = [_D, c_int, c_int, _I32]
            lib.bo_lambda.argtypes = [_D, _D, c_int, c_int, c_int, c_double, c_double,
                                      ctypes.POINTER(c_int)]
            lib.bo_lambda.restype = c_double
            lib.bo_score_unit.argtypes = [_D, _D, c_int, c_int, c_int, c_int,
                                          ctypes.POINTER(_D), c_int,
                                          ctypes.POINTER(_Params), c_int,
                                          _D, _D, _D, _D, _D, _D, _D, _D, _D]
            lib.bo_score_unit.restype = c_int
            lib.bo_select.argtypes = [_D, c_int, c_int, c_int, ctypes.POINTER(_Params),
                                      _I32, _D]
            lib.bo_select.restype = c_int
            lib.bo_gather.argtypes = [_U16, c_int, c_int, _I32, c_int, _U16]
            lib.bo_bf16_to_double.argtypes = [_U16, ctypes.c_long, _D]
            lib.bo_pyramid_budgets.argtypes = [c_int, c_int, c_int, c_int, _I32]
            lib.bo_select_adaptive.argtypes = [_D, c_int, c_int, c_int, c_int, c_double,
                                               ctypes.POINTER(_Params), _I32, _I32]
            lib.bo_select_adaptive.restype = c_int
            _lib = lib
    return _lib


def _f64(x) -> np.ndarray:
    return np.ascontiguousarray(x, dtype=np.float64)


def _p(a: np.ndarray, typ=_D):
    return a.ctypes.data_as(typ)


# --------------------------------------------------------------------------
# one equation at a time
# --------------------------------------------------------------------------

def bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns (uint16) to float64."""
    b = np.ascontiguousarray(bits, dtype=np.uint16)
    out = np.empty(b.shape, dtype=np.float64)
    _lib_handle().bo_bf16_to_double(_p(b, _U16), b.size, _p(out))
    return out


def window_scores(qwin, k):
    """Eqs. 1-2.  qwin [G, W, d] (query w at position N-W+w), k [N, d]."""
    qwin, k = _f64(qwin), _f64(k)
    G, W, d = qwin.shape
    N = k.shape[0]
    assert k.shape[1] == d and W <= N
    B = np.empty(N)
    Q = np.empty(N)
    _lib_handle().bo_window_scores(_p(qwin), _p(k), G, W, N, d, _p(B), _p(Q))
    return B, Q


def residual(Q, B):
    """Eq. 4."""
    Q, B = _f64(Q), _f64(B)
    E = np.empty_like(Q)
    _lib_handle().bo_residual(_p(Q), _p(B), Q.size, _p(E))
    return E


def coherence(E, r):
    """Eqs. 5-7."""
    E = _f64(E)
    L = np.empty_like(E)
    _lib_handle().bo_coherence(_p(E), E.size, int(r), _p(L))
    return L


def persistence(E_prev, N):
    """Eqs. 8-9.  E_prev: residuals of the layers in P_m(l)."""
    arrs = [_f64(e) for e in E_prev]
    ptrs = (_D * max(1, len(arrs)))(*[_p(a) for a in arrs])
    T = np.empty(N)
    _lib_handle().bo_persistence(ptrs, len(arrs), N, _p(T))
    return T


def evidence(E, L, T, use_E=True, use_L=True, use_T=True):
    """Eq. 10."""
    E, L, T = _f64(E), _f64(L), _f64(T)
    V = np.empty_like(E)
    _lib_handle().bo_evidence(_p(E), _p(L), _p(T), E.size, int(use_E),
                              int(use_L), int(use_T), _p(V))
    return V


def maxpool(x, kernel):
    x = _f64(x)
    y = np.empty_like(x)
    _lib_handle().bo_maxpool(_p(x), x.size, int(kernel), _p(y))
    return y


def rank_topk(x, k):
    """Best k positions of x, best first (value desc, index asc)."""
    x = _f64(x)
    out = np.empty(k, dtype=np.int32)
    _lib_handle().bo_rank_topk(_p(x), x.size, int(k), _p(out, _I32))
    return out


def calibration_lambda(Bt, V, keep, rho=2, gamma=1.0, eps=1e-8):
    """Eqs. 12-15 over the candidate arrays Bt, V.  Returns (lambda, M)."""
    Bt, V = _f64(Bt), _f64(V)
    M = ctypes.c_int(0)
    lam = _lib_handle().bo_lambda(_p(Bt), _p(V), Bt.size, int(keep), int(rho),
                                  float(gamma), float(eps), ctypes.byref(M))
    return lam, M.value


def score_unit(qwin, k, E_prev, params: Params, budget: int):
    """Eqs. 1-16 for one (layer, kv-head).  Returns a dict of float64 arrays
    (B, Q, E, L, T, V, Bt, S) and the scalar 'lambda'."""
    qwin, k = _f64(qwin), _f64(k)
    G, W, d = qwin.shape
    N = k.shape[0]
    arrs = [_f64(e) for e in E_prev]
    ptrs = (_D * max(1, len(arrs)))(*[_p(a) for a in arrs])
    out = {name: np.empty(N) for name in ("B", "Q", "E", "L", "T", "V", "Bt", "S")}
    lam = ctypes.c_double(0.0)
    cp = params._c()
    rc = _lib_handle().bo_score_unit(
        _p(qwin), _p(k), G, W, N, d, ptrs, len(arrs), ctypes.byref(cp), int(budget),
        *[_p(out[n]) for n in ("B", "Q", "E", "L", "T", "V", "Bt", "S")],
        ctypes.cast(ctypes.byref(lam), _D))
    if rc != 0:
        raise ValueError("oracle: invalid unit arguments")
    out["lambda"] = lam.value
    return out


def select(S, N, W, budget, params: Params):
    """Eq. 17 + cache layout.  Returns (ascending kept positions, gap)."""
    S = _f64(S)
    assert S.size == N
    idx = np.empty(max(1, min(budget, N)), dtype=np.int32)
    gap = ctypes.c_double(0.0)
    cp = params._c()
    n = _lib_handle().bo_select(_p(S), N, W, int(budget), ctypes.byref(cp),
                                _p(idx, _I32), ctypes.cast(ctypes.byref(gap), _D))
    if n < 0:
        raise ValueError("oracle: invalid selection arguments")
    return idx[:n].copy(), gap.value


def pyramid_budgets(layers, window, budget, beta=20):
    """Per-layer budgets of the PyramidKV-style schedule (window included)."""
    out = np.empty(max(1, layers), dtype=np.int32)
    _lib_handle().bo_pyramid_budgets(int(layers), int(window), int(budget), int(beta),
                                     _p(out, _I32))
    return out[:layers].copy()


def select_adaptive(S_heads, W, budget, alpha, params: Params):
    """AdaKV-style selection over the heads of one (request, layer).
    S_heads [H, N].  Returns a list of per-head ascending kept positions."""
    S = _f64(S_heads)
    H, N = S.shape
    idx = np.empty((H, N), dtype=np.int32)
    counts = np.empty(H, dtype=np.int32)
    cp = params._c()
    rc = _lib_handle().bo_select_adaptive(_p(S), H, N, int(W), int(budget), float(alpha),
                                          ctypes.byref(cp), _p(idx, _I32), _p(counts, _I32))
    if rc != 0:
        raise ValueError("oracle: invalid adaptive selection arguments")
    return [idx[h, :counts[h]].copy() for h in range(H)]


def gather(x_bits, idx):
    """Compacted cache rows x[idx] (bf16 bit patterns, bitwise copy)."""
    x = np.ascontiguousarray(x_bits, dtype=np.uint16)
    idx = np.ascontiguousarray(idx, dtype=np.int32)
    N, d = x.shape
    out = np.empty((idx.size, d), dtype=np.uint16)
    _lib_handle().bo_gather(_p(x, _U16), N, d, _p(idx, _I32), idx.size, _p(out, _U16))
    return out


# --------------------------------------------------------------------------
# whole step over requests x layers x kv-heads
# --------------------------------------------------------------------------

def persistence_layers(layer: int, m: int):
    """P_m(l) in 0-based layer numbers: max(0, l-m) .. l-1 (Eq. 8)."""
    return list(range(max(0, layer - m), layer))


def compress(qwin_bits, k_bits, v_bits, budget, params: Params | None = None,
             threads: int | None = None, units=None, keep_scores=False, adaptive_alpha=None):
    """The whole compression step on the host.

    qwin_bits [R, Ly, Hq, W, d], k_bits / v_bits [R, Ly, Hkv, N, d] are bf16
    bit patterns (uint16).  ``units`` optionally restricts the work to a list
    of (request, layer, kv_head); the residuals of the preceding layers that
    the persistence term needs are then computed as well.

    ``budget`` is one budget for every layer or a sequence of per-layer
    budgets (window included).  With ``adaptive_alpha`` the kept sets of a
    (request, layer) are chosen jointly over its heads (select_adaptive);
    ``units`` must then list whole layers (every head).

    Returns a dict keyed by (r, l, h) with 'idx', 'gap', 'lambda', 'Kc', 'Vc'
    and, when keep_scores, the score arrays of ``score_unit``.
    """
    params = params or Params()
    layer_budget = (lambda l: int(budget[l])) if hasattr(budget, "__len__") else (lambda l: int(budget))
    R, Ly, Hq, W, d = qwin_bits.shape
    _, _, Hkv, N, _ = k_bits.shape
    G = Hq // Hkv
    if units is None:
        units = [(r, l, h) for r in range(R) for l in range(Ly) for h in range(Hkv)]
    chains = {}
    for (r, l, h) in units:
        chains.setdefault((r, h), set()).add(l)

    def run_chain(key):
        r, h = key
        wanted = chains[key]
        need = set(wanted)
        for l in wanted:
            need.update(persistence_layers(l, params.m))
        E_of = {}
        res = {}
        for l in sorted(need):
            q = bf16_bits_to_f64(qwin_bits[r, l, h * G:(h + 1) * G])
            kk = bf16_bits_to_f64(k_bits[r, l, h])
            if l not in wanted:
                B, Q = window_scores(q, kk)
                E_of[l] = residual(Q, B)
                continue
            prev = [E_of[j] for j in persistence_layers(l, params.m)]
            sc = score_unit(q, kk, prev, params, layer_budget(l))
            E_of[l] = sc["E"]
            idx, gap = select(sc["S"], N, W, layer_budget(l), params)
            entry = {"idx": idx, "gap": gap, "lambda": sc["lambda"],
                     "Kc": gather(k_bits[r, l, h], idx),
                     "Vc": gather(v_bits[r, l, h], idx)}
            if keep_scores or adaptive_alpha is not None:
                entry.update(sc)
            res[(r, l, h)] = entry
        return res

    threads = threads or os.cpu_count() or 1
    out = {}
    with ThreadPoolExecutor(max_workers=threads) as ex:
        for part in ex.map(run_chain, list(chains)):
            out.update(part)
    if adaptive_alpha is not None:
        layers_seen = sorted({(r, l) for (r, l, h) in out})
        for (r, l) in layers_seen:
            S = np.stack([out[(r, l, h)]["S"] for h in range(Hkv)])
            kept = select_adaptive(S, W, layer_budget(l), adaptive_alpha, params)
            for h in range(Hkv):
                e = out[(r, l, h)]
                e["idx"] = kept[h]
                e["Kc"] = gather(k_bits[r, l, h], kept[h])
                e["Vc"] = gather(v_bits[r, l, h], kept[h])
    return out


def sweep(qwin_bits, k_bits, v_bits, budget, variants, params: Params | None = None,
          threads: int | None = None, units=None, keep_scores=False):
    """Ablation / sensitivity sweep (Sec. 5.3): the whole step once per
    variant, a dict of Params fields that override ``params``.  Returns the
    ``compress`` results in variant order."""
    params = params or Params()
    out = []
    for var in variants:
        fields = {f: (bool(x) if f.startswith("use_") else x) for f, x in var.items()}
        out.append(compress(qwin_bits, k_bits, v_bits, budget,
                            dataclasses.replace(params, **fields), threads, units,
                            keep_scores=keep_scores))
    return out

