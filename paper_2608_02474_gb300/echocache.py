"""ctypes binding of libechocache.so (include/echocache.h), same names as the C entry points.

Argument marshalling only: every step of the cached DiT step runs in the
library's CUDA kernels.  Tensors are torch CUDA tensors (device memory and
streams come from PyTorch); outputs are allocated here when not given.  There
is no fallback: a missing library or a non-sm_103 device raises.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass

import numpy as np
import torch

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libechocache.so")

ECHO_OK = 0
ECHO_BF16, ECHO_F32 = 0, 1
MODE_ENERGY_DRIFT, MODE_SEGMENT, MODE_DRIFT_ONLY = 0, 1, 2

_c = ctypes
_vp, _i32, _i64, _sz, _f32 = _c.c_void_p, _c.c_int32, _c.c_int64, _c.c_size_t, _c.c_float
_f64 = _c.c_double


class EchoError(RuntimeError):
    def __init__(self, fn: str, status: int):
        self.status = status
        super().__init__(f"{fn} failed: {status_str(status)} ({status})")


class SelectParams(_c.Structure):
    _fields_ = [("lambda_", _f32), ("xi", _f32), ("mode", _i32)]


class RateParams(_c.Structure):
    _fields_ = [("r_min", _f64), ("r_max", _f64), ("alpha", _f64)]


CACHE_INT8, CACHE_BF16, CACHE_REF = 0, 1, 2


class CacheC(_c.Structure):
    _fields_ = [("kind", _i32), ("NT", _i32), ("D", _i32), ("q", _vp), ("scale", _vp),
                ("full", _vp), ("ref", _vp), ("pool", _vp), ("refcount", _vp), ("R_cap", _i32),
                ("seg_len", _i32), ("tau", _f32)]


class BlockDims(_c.Structure):
    _fields_ = [("T", _i32), ("N", _i32), ("D", _i32), ("H", _i32), ("d", _i32), ("F", _i32),
                ("Lc", _i32)]


class BlockWeightsC(_c.Structure):
    _fields_ = [(n, _vp) for n in ("Wq", "bq", "Wkv", "bkv", "Wo", "bo", "Wqc", "bqc", "Woc",
                                   "boc", "W1", "b1", "W2", "b2", "KVc")]


_SIGS = {
    "echo_status_str": (_c.c_char_p, [_i32]),
    "echo_get_device_error": (_i32, [_vp]),
    "echo_audio_energy": (_i32, [_vp, _i64, _i32, _i32, _i32, _i32, _vp, _vp, _vp]),
    "echo_select_workspace_size": (_sz, [_i32, _i32]),
    "echo_select": (_i32, [_vp, _i32, _vp, _vp, _vp, _i32, _i32, _i32, _i32, _i32,
                           _c.POINTER(SelectParams), _vp, _c.POINTER(_i32), _vp, _vp, _sz, _vp]),
    "echo_select_static": (_i32, [_vp, _i32, _vp, _vp, _vp, _i32, _i32, _i32, _i32, _i32,
                                  _c.POINTER(SelectParams), _vp, _c.POINTER(_i32), _vp]),
    "echo_cache_reset": (_i32, [_c.POINTER(CacheC), _vp]),
    "echo_cache_write_workspace_size": (_sz, [_c.POINTER(CacheC), _i32]),
    "echo_cache_write": (_i32, [_c.POINTER(CacheC), _vp, _vp, _i32, _vp, _sz, _vp]),
    "echo_cache_read": (_i32, [_c.POINTER(CacheC), _vp, _i32, _vp, _vp]),
    "echo_cache_stats": (_i32, [_c.POINTER(CacheC), _vp, _vp]),
    "echo_select_cache": (_i32, [_vp, _i32, _c.POINTER(CacheC), _vp, _i32, _i32, _i32, _i32,
                                 _c.POINTER(SelectParams), _vp, _c.POINTER(_i32), _vp, _vp, _sz,
                                 _vp]),
    "echo_block_step_cache_workspace_size": (_sz, [_c.POINTER(BlockDims), _i32,
                                                   _c.POINTER(CacheC)]),
    "echo_block_step_cache": (_i32, [_c.POINTER(BlockWeightsC), _c.POINTER(BlockDims), _vp, _vp,
                                     _i32, _c.POINTER(CacheC), _vp, _vp, _sz, _vp]),
    "echo_select_uniform": (_i32, [_i32, _i32, _i32, _i32, _vp, _c.POINTER(_i32), _vp]),
    "echo_select_random": (_i32, [_vp, _i32, _i32, _i32, _i32, _vp, _c.POINTER(_i32), _vp]),
    "echo_step_delta_workspace_size": (_sz, [_i64]),
    "echo_step_delta": (_i32, [_vp, _vp, _i32, _i64, _f64, _vp, _vp, _sz, _vp]),
    "echo_update_rate": (_i32, [_f64, _f64, _c.POINTER(RateParams), _i32, _c.POINTER(_f64),
                                _c.POINTER(_i32)]),
    "echo_workspace_size": (_sz, [_c.POINTER(BlockDims), _i32]),
    "echo_precompute_cross_kv": (_i32, [_vp, _vp, _vp, _i32, _i32, _vp, _vp]),
    "echo_block_step": (_i32, [_c.POINTER(BlockWeightsC), _c.POINTER(BlockDims), _vp, _vp, _i32,
                               _vp, _vp, _vp, _vp, _sz, _vp]),
    "echo_workspace_size_kv": (_sz, [_c.POINTER(BlockDims), _i32, _i32]),
    "echo_block_step_kv": (_i32, [_c.POINTER(BlockWeightsC), _c.POINTER(BlockDims), _vp, _vp, _i32,
                                  _vp, _i32, _vp, _i32, _vp, _i32, _vp, _vp, _vp, _vp, _sz, _vp]),
    "echo_cache_quant": (_i32, [_vp, _i32, _vp, _i32, _i32, _vp, _vp, _vp]),
    "echo_cache_dequant": (_i32, [_vp, _vp, _vp, _i32, _i32, _vp, _i32, _vp]),
    "echo_linear": (_i32, [_vp, _i64, _i32, _i32, _vp, _vp, _i32, _i32, _vp, _i32, _vp, _vp, _i64,
                           _i32, _vp]),
    "echo_attention": (_i32, [_vp, _i64, _vp, _vp, _i64, _i32, _i32, _i32, _i32, _vp, _i64, _vp]),
    "echo_layernorm": (_i32, [_vp, _i32, _vp, _i32, _i32, _vp, _vp]),
    "echo_check_timeout_path": (_i32, [_i64, _vp]),
    "echo_launch_count": (_c.c_uint64, []),
    "echo_profile_enable": (_i32, [_i32]),
    "echo_profile_read": (_i32, [_i32, _vp, _vp, _vp, _vp, _vp]),
    "echo_kernel_name": (_c.c_char_p, [_i32]),
}

_LIB = None


def lib():
    """Load the in-tree library (built by __graft_entry__.build() or build.py)."""
    global _LIB
    if _LIB is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it first (python -c "
                               "'import __graft_entry__ as g; g.build()')")
        L = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in _SIGS.items():
            f = getattr(L, name)
            f.restype, f.argtypes = res, args
        _LIB = L
    return _LIB


def status_str(s: int) -> str:
    return lib().echo_status_str(int(s)).decode()


def _check(fn: str, s: int):
    if s != ECHO_OK:
        raise EchoError(fn, s)


def _p(t):
    return None if t is None else _vp(t.data_ptr())


def _stream(stream=None):
    s = stream if stream is not None else torch.cuda.current_stream()
    return _vp(s.cuda_stream)


def _dtype(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return ECHO_BF16
    if t.dtype == torch.float32:
        return ECHO_F32
    raise TypeError(f"unsupported dtype {t.dtype}")


def _dev(t: torch.Tensor, name: str):
    if not (t.is_cuda and t.is_contiguous()):
        raise ValueError(f"{name} must be a contiguous CUDA tensor")


# ---------------------------------------------------------------------------
def echo_get_device_error(stream=None) -> int:
    return lib().echo_get_device_error(_stream(stream))


def echo_audio_energy(audio: torch.Tensor, T: int, n_fft: int = 512, hop: int = 160,
                      n_bands: int = 8, band=None, seg=None, stream=None):
    _dev(audio, "audio")
    band = band if band is not None else torch.empty(T, n_bands, dtype=torch.float32,
                                                     device=audio.device)
    seg = seg if seg is not None else torch.empty(T, dtype=torch.float32, device=audio.device)
    _check("echo_audio_energy", lib().echo_audio_energy(
        _p(audio), audio.numel(), T, n_fft, hop, n_bands, _p(band), _p(seg), _stream(stream)))
    return band, seg


def echo_select_workspace_size(T: int, N: int) -> int:
    return lib().echo_select_workspace_size(T, N)


def echo_select(x, cache_q, cache_scale, seg_energy, T: int, N: int, ratio_num: int,
                ratio_den: int, lam: float = 0.1, xi: float = 1e-6, mode: int = MODE_ENERGY_DRIFT,
                idx=None, scores=None, workspace=None, stream=None):
    """Returns (idx[:K] int32, K, scores or None)."""
    for t, n in ((x, "x"), (cache_q, "cache_q"), (cache_scale, "cache_scale"),
                 (seg_energy, "seg_energy")):
        _dev(t, n)
    NT, D = x.shape
    idx = idx if idx is not None else torch.empty(NT, dtype=torch.int32, device=x.device)
    if scores is None and workspace is None:
        workspace = torch.empty(echo_select_workspace_size(T, N), dtype=torch.uint8, device=x.device)
    prm = SelectParams(lam, xi, mode)
    K = _i32(0)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    _check("echo_select", lib().echo_select(
        _p(x), _dtype(x), _p(cache_q), _p(cache_scale), _p(seg_energy), T, N, D, ratio_num,
        ratio_den, _c.byref(prm), _p(idx), _c.byref(K), _p(scores), _p(workspace), ws_bytes,
        _stream(stream)))
    return idx[:K.value], K.value, scores


def echo_select_uniform(T: int, N: int, ratio_num: int, ratio_den: int, idx=None, device=None,
                        stream=None):
    """Uniform ablation selection; returns (idx[:K], K)."""
    dev = idx.device if idx is not None else (device or torch.device("cuda"))
    idx = idx if idx is not None else torch.empty(T * N, dtype=torch.int32, device=dev)
    K = _i32(0)
    _check("echo_select_uniform", lib().echo_select_uniform(T, N, ratio_num, ratio_den, _p(idx),
                                                            _c.byref(K), _stream(stream)))
    return idx[:K.value], K.value


def echo_select_random(keys, T: int, N: int, ratio_num: int, ratio_den: int, idx=None,
                       stream=None):
    """Random ablation selection over caller-drawn keys; returns (idx[:K], K)."""
    _dev(keys, "keys")
    idx = idx if idx is not None else torch.empty(T * N, dtype=torch.int32, device=keys.device)
    K = _i32(0)
    _check("echo_select_random", lib().echo_select_random(_p(keys), T, N, ratio_num, ratio_den,
                                                          _p(idx), _c.byref(K), _stream(stream)))
    return idx[:K.value], K.value


def echo_step_delta_workspace_size(n: int) -> int:
    return lib().echo_step_delta_workspace_size(n)


def echo_step_delta(h_prev, h_cur, xi: float = 1e-6, out=None, workspace=None, stream=None):
    """Eq. 1 between two step outputs; returns the device double[3]
    {Delta, sum|h_prev - h_cur|, sum|h_cur|} (no host synchronisation)."""
    _dev(h_prev, "h_prev")
    _dev(h_cur, "h_cur")
    if h_prev.dtype != h_cur.dtype or h_prev.numel() != h_cur.numel():
        raise ValueError("h_prev and h_cur must have the same dtype and size")
    n = h_cur.numel()
    out = out if out is not None else torch.empty(3, dtype=torch.float64, device=h_cur.device)
    ws_n = echo_step_delta_workspace_size(n)
    ws = workspace if workspace is not None else torch.empty(ws_n, dtype=torch.uint8,
                                                             device=h_cur.device)
    _check("echo_step_delta", lib().echo_step_delta(
        _p(h_prev), _p(h_cur), _dtype(h_cur), n, float(xi), _p(out), _p(ws), ws.numel(),
        _stream(stream)))
    return out


def echo_update_rate(delta: float, delta_ref: float, NT: int, r_min: float = 0.1,
                     r_max: float = 0.5, alpha: float = 0.2) -> tuple[float, int]:
    """Host rule of the adaptive update rate: returns (r_t, K)."""
    prm = RateParams(r_min, r_max, alpha)
    rate, K = _f64(0.0), _i32(0)
    _check("echo_update_rate", lib().echo_update_rate(float(delta), float(delta_ref),
                                                      _c.byref(prm), NT, _c.byref(rate),
                                                      _c.byref(K)))
    return rate.value, K.value


def echo_workspace_size(dims: BlockDims, K_max: int) -> int:
    return lib().echo_workspace_size(_c.byref(dims), K_max)


def echo_precompute_cross_kv(cond, Wkvc, bkvc, KVc=None, stream=None):
    Lc, D = cond.shape
    KVc = KVc if KVc is not None else torch.empty(Lc, 2 * D, dtype=torch.bfloat16, device=cond.device)
    _check("echo_precompute_cross_kv", lib().echo_precompute_cross_kv(
        _p(cond), _p(Wkvc), _p(bkvc), Lc, D, _p(KVc), _stream(stream)))
    return KVc


def echo_block_step(weights: "DeviceBlock", dims: BlockDims, x, idx, K: int, cache_q, cache_scale,
                    y=None, workspace=None, stream=None):
    y = y if y is not None else torch.empty_like(x)
    if workspace is None:
        workspace = torch.empty(echo_workspace_size(dims, K), dtype=torch.uint8, device=x.device)
    _check("echo_block_step", lib().echo_block_step(
        _c.byref(weights.cstruct), _c.byref(dims), _p(x), _p(idx) if K > 0 else None, K,
        _p(cache_q), _p(cache_scale), _p(y), _p(workspace),
        workspace.numel() * workspace.element_size(), _stream(stream)))
    return y


def echo_workspace_size_kv(dims: BlockDims, K_max: int, n_rows_max: int) -> int:
    return int(lib().echo_workspace_size_kv(_c.byref(dims), int(K_max), int(n_rows_max)))


def echo_block_step_kv(weights: "DeviceBlock", dims: BlockDims, x, idx, K: int, kv,
                       kv_valid: bool, cache_q, cache_scale, rows_a=None, n_a: int = 0,
                       rows_b=None, n_b: int = 0, y=None, workspace=None, stream=None):
    """echo_block_step with K/V of every token kept in `kv` (bf16 [NT, 2D])
    across calls; with kv_valid only the rows rows_a[:n_a] and rows_b[:n_b]
    are recomputed (the rows whose layer input changed)."""
    y = y if y is not None else torch.empty_like(x)
    if workspace is None:
        workspace = torch.empty(echo_workspace_size_kv(dims, K, n_a + n_b), dtype=torch.uint8,
                                device=x.device)
    _check("echo_block_step_kv", lib().echo_block_step_kv(
        _c.byref(weights.cstruct), _c.byref(dims), _p(x), _p(idx) if K > 0 else None, K,
        _p(kv), 1 if kv_valid else 0, _p(rows_a) if n_a > 0 else None, n_a,
        _p(rows_b) if n_b > 0 else None, n_b, _p(cache_q), _p(cache_scale), _p(y),
        _p(workspace), workspace.numel() * workspace.element_size(), _stream(stream)))
    return y


def echo_cache_quant(src, rows, q, scale, stream=None):
    n, D = src.shape
    _check("echo_cache_quant", lib().echo_cache_quant(
        _p(src), _dtype(src), _p(rows), n, D, _p(q), _p(scale), _stream(stream)))


def echo_cache_dequant(q, scale, rows=None, dtype=torch.bfloat16, out=None, stream=None):
    n = q.shape[0] if rows is None else rows.numel()
    D = q.shape[1]
    out = out if out is not None else torch.empty(n, D, dtype=dtype, device=q.device)
    _check("echo_cache_dequant", lib().echo_cache_dequant(
        _p(q), _p(scale), _p(rows), n, D, _p(out), _dtype(out), _stream(stream)))
    return out


def echo_linear(A, W, bias=None, act: int = 0, resid=None, resid_rows=None,
                out_dtype=torch.bfloat16, out=None, stream=None):
    M, Kd = A.shape
    N = W.shape[0]
    out = out if out is not None else torch.empty(M, N, dtype=out_dtype, device=A.device)
    rt = _dtype(resid) if resid is not None else ECHO_BF16
    _check("echo_linear", lib().echo_linear(
        _p(A), A.stride(0), M, Kd, _p(W), _p(bias), N, act, _p(resid), rt, _p(resid_rows),
        _p(out), out.stride(0), _dtype(out), _stream(stream)))
    return out


def echo_attention(Q, K, V, H: int, d: int, out=None, stream=None):
    """Q [M, >=H d] (row stride Q.stride(0)), K and V [L, *] sharing one row stride."""
    M, L = Q.shape[0], K.shape[0]
    if K.stride(0) != V.stride(0):
        raise ValueError("K and V must share a row stride")
    out = out if out is not None else torch.empty(M, H * d, dtype=torch.bfloat16, device=Q.device)
    _check("echo_attention", lib().echo_attention(
        _p(Q), Q.stride(0), _p(K), _p(V), K.stride(0), M, L, H, d, _p(out), out.stride(0),
        _stream(stream)))
    return out


def echo_layernorm(inp, rows=None, out=None, stream=None):
    n = inp.shape[0] if rows is None else rows.numel()
    D = inp.shape[1]
    out = out if out is not None else torch.empty(n, D, dtype=torch.bfloat16, device=inp.device)
    _check("echo_layernorm", lib().echo_layernorm(
        _p(inp), _dtype(inp), _p(rows), n, D, _p(out), _stream(stream)))
    return out


def echo_check_timeout_path(limit_ns: int = 1_000_000, stream=None):
    _check("echo_check_timeout_path", lib().echo_check_timeout_path(int(limit_ns), _stream(stream)))


def echo_launch_count() -> int:
    return int(lib().echo_launch_count())


def echo_profile_enable(on: bool = True):
    _check("echo_profile_enable", lib().echo_profile_enable(1 if on else 0))


def echo_kernel_name(kind: int) -> str:
    return lib().echo_kernel_name(int(kind)).decode()


def echo_profile_read(max_records: int = 65536):
    """List of (kernel name, m, n, k, ms) for every launch recorded since the last read."""
    import numpy as np
    kinds = np.zeros(max_records, np.int32)
    m, n, k = (np.zeros(max_records, np.int64) for _ in range(3))
    ms = np.zeros(max_records, np.float32)
    cnt = lib().echo_profile_read(max_records, kinds.ctypes.data, m.ctypes.data, n.ctypes.data,
                                  k.ctypes.data, ms.ctypes.data)
    if cnt < 0:
        raise EchoError("echo_profile_read", 4)
    return [(echo_kernel_name(kinds[i]), int(m[i]), int(n[i]), int(k[i]), float(ms[i]))
            for i in range(cnt)]


# ---------------------------------------------------------------------------
@dataclass
class DeviceBlock:
    """One block's parameters resident on the device, in the layout the C ABI takes."""
    tensors: dict
    cstruct: BlockWeightsC

    @staticmethod
    def from_host(W: dict, cond, device="cuda", stream=None) -> "DeviceBlock":
        """W: nn.Linear-convention arrays (numpy or torch, bf16 values); cond [Lc, D]."""
        bf = lambda a: torch.as_tensor(a).to(device=device, dtype=torch.bfloat16).contiguous()
        t = {
            "Wq": bf(W["Wq"]), "bq": bf(W["bq"]),
            "Wkv": torch.cat([bf(W["Wk"]), bf(W["Wv"])]).contiguous(),
            "bkv": torch.cat([bf(W["bk"]), bf(W["bv"])]).contiguous(),
            "Wo": bf(W["Wo"]), "bo": bf(W["bo"]),
            "Wqc": bf(W["Wqc"]), "bqc": bf(W["bqc"]),
            "Woc": bf(W["Woc"]), "boc": bf(W["boc"]),
            "W1": bf(W["W1"]), "b1": bf(W["b1"]),
            "W2": bf(W["W2"]), "b2": bf(W["b2"]),
        }
        Wkvc = torch.cat([bf(W["Wkc"]), bf(W["Wvc"])]).contiguous()
        bkvc = torch.cat([bf(W["bkc"]), bf(W["bvc"])]).contiguous()
        t["KVc"] = echo_precompute_cross_kv(bf(cond), Wkvc, bkvc, stream=stream)
        c = BlockWeightsC(*[_p(t[n]) for n, _ in BlockWeightsC._fields_])
        return DeviceBlock(t, c)


class DeviceCache:
    """One layer's cache in one of the forms of echo_cache, with its device
    tensors owned here.  kind CACHE_INT8: q, scale; CACHE_BF16: full;
    CACHE_REF: q, scale, ref, pool [R_cap, D], refcount (R_cap defaults to NT,
    the most references a cache can hold; seg_len, tau as echo_cache).
    Starts empty (echo_cache_reset)."""

    def __init__(self, kind: int, NT: int, D: int, R_cap: int | None = None, seg_len: int = 1,
                 tau: float = 0.9, device="cuda", stream=None):
        dev = torch.device(device)
        self.kind, self.NT, self.D = kind, NT, D
        self.t = {}
        if kind in (CACHE_INT8, CACHE_REF):
            self.t["q"] = torch.empty(NT, D, dtype=torch.int8, device=dev)
            self.t["scale"] = torch.empty(NT, dtype=torch.float32, device=dev)
        if kind == CACHE_BF16:
            self.t["full"] = torch.empty(NT, D, dtype=torch.bfloat16, device=dev)
        R_cap = (NT if R_cap is None else R_cap) if kind == CACHE_REF else 0
        if kind == CACHE_REF:
            self.t["ref"] = torch.empty(NT, dtype=torch.int32, device=dev)
            self.t["pool"] = torch.empty(max(R_cap, 1), D, dtype=torch.bfloat16, device=dev)
            self.t["refcount"] = torch.empty(max(R_cap, 1), dtype=torch.int32, device=dev)
        self.R_cap, self.seg_len, self.tau = R_cap, seg_len, tau
        self.cstruct = CacheC(kind, NT, D, *[_p(self.t.get(n)) for n in
                                             ("q", "scale", "full", "ref", "pool", "refcount")],
                              R_cap, seg_len, tau)
        self.reset(stream)

    def reset(self, stream=None):
        _check("echo_cache_reset", lib().echo_cache_reset(_c.byref(self.cstruct), _stream(stream)))

    def load(self, **arrays):
        """Overwrite state tensors (q, scale, full, ref, pool, refcount) from
        host arrays of the same shapes (pool and full as bf16 values)."""
        for n, a in arrays.items():
            t = self.t[n]
            src = torch.as_tensor(np.ascontiguousarray(a)).to(t.dtype)
            t[:src.shape[0]].copy_(src.to(t.device))

    def clone(self) -> "DeviceCache":
        c = DeviceCache.__new__(DeviceCache)
        c.kind, c.NT, c.D = self.kind, self.NT, self.D
        c.R_cap, c.seg_len, c.tau = self.R_cap, self.seg_len, self.tau
        c.t = {n: t.clone() for n, t in self.t.items()}
        c.cstruct = CacheC(c.kind, c.NT, c.D, *[_p(c.t.get(n)) for n in
                                               ("q", "scale", "full", "ref", "pool", "refcount")],
                           c.R_cap, c.seg_len, c.tau)
        return c

    def write_workspace_size(self, n_rows: int) -> int:
        return lib().echo_cache_write_workspace_size(_c.byref(self.cstruct), n_rows)

    def write(self, src, rows, workspace=None, stream=None):
        _dev(src, "src")
        _dev(rows, "rows")
        n = rows.numel()
        need = self.write_workspace_size(n)
        if workspace is None and need:
            workspace = torch.empty(need, dtype=torch.uint8, device=src.device)
        wsb = 0 if workspace is None else workspace.numel()
        _check("echo_cache_write", lib().echo_cache_write(
            _c.byref(self.cstruct), _p(src), _p(rows), n, _p(workspace), wsb, _stream(stream)))

    def read(self, rows=None, out=None, stream=None):
        n = self.NT if rows is None else rows.numel()
        dev = self.t["q" if "q" in self.t else "full"].device
        out = out if out is not None else torch.empty(n, self.D, dtype=torch.bfloat16, device=dev)
        _check("echo_cache_read", lib().echo_cache_read(_c.byref(self.cstruct), _p(rows), n,
                                                        _p(out), _stream(stream)))
        return out

    def stats(self, stream=None) -> tuple[int, int]:
        """(live references, high-water mark); synchronises the stream."""
        out = torch.zeros(2, dtype=torch.int32, device=self.t["ref"].device)
        _check("echo_cache_stats", lib().echo_cache_stats(_c.byref(self.cstruct), _p(out),
                                                          _stream(stream)))
        a, b = out.cpu().tolist()
        return a, b

    def nbytes(self, pool_rows: int | None = None) -> int:
        """Device bytes of this cache; for CACHE_REF with `pool_rows`, the bytes
        of a pool sized to that many rows instead of R_cap."""
        total = 0
        for n, t in self.t.items():
            if n in ("pool", "refcount") and pool_rows is not None:
                total += pool_rows * t[0].numel() * t.element_size()
            else:
                total += t.numel() * t.element_size()
        return total


def echo_select_cache(x, cache: DeviceCache, seg_energy, T: int, N: int, ratio_num: int,
                      ratio_den: int, lam: float = 0.1, xi: float = 1e-6,
                      mode: int = MODE_ENERGY_DRIFT, idx=None, scores=None, workspace=None,
                      stream=None):
    """echo_select against any cache form; returns (idx[:K] int32, K, scores or None)."""
    _dev(x, "x")
    _dev(seg_energy, "seg_energy")
    NT = x.shape[0]
    idx = idx if idx is not None else torch.empty(NT, dtype=torch.int32, device=x.device)
    if scores is None and workspace is None:
        workspace = torch.empty(echo_select_workspace_size(T, N), dtype=torch.uint8, device=x.device)
    prm = SelectParams(lam, xi, mode)
    K = _i32(0)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    _check("echo_select_cache", lib().echo_select_cache(
        _p(x), _dtype(x), _c.byref(cache.cstruct), _p(seg_energy), T, N, ratio_num, ratio_den,
        _c.byref(prm), _p(idx), _c.byref(K), _p(scores), _p(workspace), ws_bytes,
        _stream(stream)))
    return idx[:K.value], K.value, scores


def echo_block_step_cache_workspace_size(dims: BlockDims, K_max: int, cache: DeviceCache) -> int:
    return lib().echo_block_step_cache_workspace_size(_c.byref(dims), K_max,
                                                      _c.byref(cache.cstruct))


def echo_block_step_cache(weights: DeviceBlock, dims: BlockDims, x, idx, K: int,
                          cache: DeviceCache, y=None, workspace=None, stream=None):
    y = y if y is not None else torch.empty_like(x)
    if workspace is None:
        workspace = torch.empty(echo_block_step_cache_workspace_size(dims, K, cache),
                                dtype=torch.uint8, device=x.device)
    _check("echo_block_step_cache", lib().echo_block_step_cache(
        _c.byref(weights.cstruct), _c.byref(dims), _p(x), _p(idx) if K > 0 else None, K,
        _c.byref(cache.cstruct), _p(y), _p(workspace),
        workspace.numel() * workspace.element_size(), _stream(stream)))
    return y
