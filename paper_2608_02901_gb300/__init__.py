"""Python binding of the AnchorKV decode-attention library (``libakv.so``).

Argument marshalling only: every function below converts its arguments to
plain pointers and sizes and calls the C entry point of the same name
declared in ``include/akv.h``.  Device buffers are torch CUDA tensors; host
buffers are numpy arrays.  If ``libakv.so`` has not been built, importing the
library fails loudly -- there is no fallback implementation.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libakv.so")

AKV_OK, AKV_ERR_INVALID, AKV_ERR_UNSUPPORTED, AKV_ERR_TOO_SMALL, AKV_ERR_CUDA = range(5)
AKV_FLAG_ROTATE = 1
AKV_FLAG_LLOYD = 2
AKV_FLAG_ROPE = 4
HEAD_DIM = 128

EXPORTED = (
    "akv_status_string", "akv_last_error", "akv_unit_shapes", "akv_cache_size", "akv_cache_header_host",
    "akv_encode", "akv_encode_noalloc", "akv_cache_pack_host", "akv_decode_workspace_size", "akv_decode_attn",
    "akv_decode_set_debug", "akv_decode_set_events", "akv_cache_size_select", "akv_encode_select",
    "akv_decode_workspace_size_suffix", "akv_decode_attn_suffix", "akv_suffix_append", "akv_table1_bytes",
    "akv_pack_table1_host",
)
AKV_MAX_SUFFIX = 1 << 20
NOALLOC_SCRATCH_BYTES = 16 << 20


class AkvError(RuntimeError):
    def __init__(self, status: int, where: str, detail: str):
        super().__init__(f"{where}: status {status} ({_status_name(status)}): {detail}")
        self.status = status


class _Params(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int32), ("n_kv_heads", ctypes.c_int32), ("n_q_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("anchor_frac", ctypes.c_float), ("res_frac_k", ctypes.c_float),
                ("res_frac_v", ctypes.c_float), ("window", ctypes.c_int32), ("seed", ctypes.c_uint64),
                ("rot_seed", ctypes.c_uint64), ("flags", ctypes.c_uint32), ("rope_theta", ctypes.c_float)]


class _SelectParams(ctypes.Structure):
    _fields_ = [("theta", ctypes.c_float), ("rho", ctypes.c_float), ("kappa", ctypes.c_int32),
                ("reserved", ctypes.c_int32)]


@dataclass
class SelectParams:
    """The paper's full selection (see akv_select_params in include/akv.h)."""
    theta: float = 0.05
    rho: float = 0.7
    kappa: int = 7

    def c(self) -> _SelectParams:
        return _SelectParams(self.theta, self.rho, self.kappa, 0)


class _Suffix(ctypes.Structure):
    _fields_ = [("K", ctypes.c_void_p), ("V", ctypes.c_void_p), ("len", ctypes.c_void_p), ("cap", ctypes.c_int32)]


class _UnitHost(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in (
        "anchor_k", "anchor_v", "anchor_pos", "idx_k", "gamma_k", "idx_v", "gamma_v", "res_pos_k", "codes_k",
        "scale_k", "min_k", "res_pos_v", "codes_v", "scale_v", "min_v")]


@dataclass
class Params:
    """Compression parameters of one layer (see akv_params in include/akv.h)."""
    batch: int
    n_kv_heads: int
    n_q_heads: int
    anchor_frac: float = 0.02
    res_frac_k: float = 0.10
    res_frac_v: float = 0.10
    window: int = 32
    seed: int = 0
    rot_seed: int = 0x5EED
    rotate: bool = True
    head_dim: int = HEAD_DIM
    lloyd: bool = False  # the Lloyd-Max residual codec (AKV_FLAG_LLOYD) instead of the uniform one
    rope: bool = False  # pre-RoPE keys, RoPE applied at decode (AKV_FLAG_ROPE)
    rope_theta: float = 500000.0

    @property
    def G(self) -> int:
        return self.n_q_heads // self.n_kv_heads

    @property
    def n_units(self) -> int:
        return self.batch * self.n_kv_heads

    def c(self) -> _Params:
        return _Params(self.batch, self.n_kv_heads, self.n_q_heads, self.head_dim, self.anchor_frac,
                       self.res_frac_k, self.res_frac_v, self.window, self.seed & (2**64 - 1),
                       self.rot_seed & (2**64 - 1),
                       (AKV_FLAG_ROTATE if self.rotate else 0) | (AKV_FLAG_LLOYD if self.lloyd else 0) |
                       (AKV_FLAG_ROPE if self.rope else 0), float(self.rope_theta) if self.rope else 0.0)


_lib = None


def lib():
    """Load libakv.so; raises if it has not been built (no fallback path exists)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise ImportError(f"libakv.so not built at {LIB_PATH}: run `python -c 'import __graft_entry__ as g; g.build()'`")
        L = ctypes.CDLL(LIB_PATH)
        vp, i32p, st = ctypes.c_void_p, ctypes.POINTER(ctypes.c_int32), ctypes.c_int
        P = ctypes.POINTER(_Params)
        sz = ctypes.POINTER(ctypes.c_size_t)
        L.akv_status_string.restype = ctypes.c_char_p
        L.akv_status_string.argtypes = [st]
        L.akv_last_error.restype = ctypes.c_char_p
        L.akv_last_error.argtypes = []
        L.akv_unit_shapes.restype = st
        L.akv_unit_shapes.argtypes = [P, i32p, i32p]
        L.akv_cache_size.restype = st
        L.akv_cache_size.argtypes = [P, i32p, sz, sz]
        L.akv_cache_header_host.restype = st
        L.akv_cache_header_host.argtypes = [P, i32p, vp, ctypes.c_size_t]
        L.akv_encode.restype = st
        L.akv_encode.argtypes = [P, i32p, vp, vp, ctypes.c_int32, vp, ctypes.c_size_t, vp, ctypes.c_size_t, vp]
        L.akv_encode_noalloc.restype = st
        L.akv_encode_noalloc.argtypes = [P, i32p, vp, vp, ctypes.c_int32, vp, ctypes.c_size_t, vp]
        L.akv_cache_pack_host.restype = st
        L.akv_cache_pack_host.argtypes = [P, i32p, ctypes.POINTER(_UnitHost), vp, ctypes.c_size_t]
        L.akv_decode_workspace_size.restype = st
        L.akv_decode_workspace_size.argtypes = [P, i32p, sz]
        L.akv_decode_attn.restype = st
        L.akv_decode_attn.argtypes = [P, i32p, vp, ctypes.c_size_t, vp, vp, vp, ctypes.c_float, vp,
                                      ctypes.c_size_t, vp]
        SP = ctypes.POINTER(_SelectParams)
        L.akv_cache_size_select.restype = st
        L.akv_cache_size_select.argtypes = [P, SP, i32p, sz, sz]
        L.akv_encode_select.restype = st
        L.akv_encode_select.argtypes = [P, SP, i32p, vp, vp, vp, ctypes.c_int32, vp, ctypes.c_size_t, vp,
                                        ctypes.c_size_t, vp]
        L.akv_decode_set_debug.restype = st
        L.akv_decode_set_debug.argtypes = [ctypes.c_int32, ctypes.c_int32]
        L.akv_decode_set_events.restype = st
        L.akv_decode_set_events.argtypes = [ctypes.c_void_p, ctypes.c_void_p]
        L.akv_decode_workspace_size_suffix.restype = st
        L.akv_decode_workspace_size_suffix.argtypes = [P, i32p, ctypes.c_int32, sz]
        L.akv_decode_attn_suffix.restype = st
        L.akv_decode_attn_suffix.argtypes = [P, i32p, vp, ctypes.c_size_t, vp, vp, vp, ctypes.c_float,
                                             ctypes.POINTER(_Suffix), vp, ctypes.c_size_t, vp]
        L.akv_suffix_append.restype = st
        L.akv_suffix_append.argtypes = [P, vp, vp, vp, vp, vp, ctypes.c_int32, vp]
        L.akv_table1_bytes.restype = st
        L.akv_table1_bytes.argtypes = [P, i32p, ctypes.POINTER(ctypes.c_size_t)]
        L.akv_pack_table1_host.restype = st
        L.akv_pack_table1_host.argtypes = [P, i32p, ctypes.POINTER(_UnitHost), vp, ctypes.c_size_t]
        _lib = L
    return _lib


def _status_name(s: int) -> str:
    try:
        return lib().akv_status_string(s).decode()
    except Exception:  # noqa: BLE001 - only used to format an error text
        return str(s)


def _check(status: int, where: str):
    if status != AKV_OK:
        raise AkvError(status, where, lib().akv_last_error().decode())


def _lens(ctx_lens) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(ctx_lens, dtype=np.int32))


def _i32p(a: np.ndarray):
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_int32))


def _dev_ptr(t) -> int | None:
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("expected a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError("expected a contiguous tensor")
    return t.data_ptr()


def _stream_ptr(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    return getattr(stream, "cuda_stream", stream)


# ---- entry points (same names as the C ABI) --------------------------------------

def akv_status_string(s: int) -> str:
    return lib().akv_status_string(s).decode()


def akv_last_error() -> str:
    return lib().akv_last_error().decode()


def akv_unit_shapes(p: Params, ctx_lens) -> np.ndarray:
    lens = _lens(ctx_lens)
    out = np.zeros((p.n_units, 4), np.int32)
    _check(lib().akv_unit_shapes(ctypes.byref(p.c()), _i32p(lens), _i32p(out)), "akv_unit_shapes")
    return out


def akv_cache_size(p: Params, ctx_lens):
    lens = _lens(ctx_lens)
    a, w = ctypes.c_size_t(), ctypes.c_size_t()
    _check(lib().akv_cache_size(ctypes.byref(p.c()), _i32p(lens), ctypes.byref(a), ctypes.byref(w)),
           "akv_cache_size")
    return a.value, w.value


def akv_cache_header_host(p: Params, ctx_lens) -> np.ndarray:
    lens = _lens(ctx_lens)
    buf = np.zeros(256 * (1 + p.n_units), np.uint8)
    _check(lib().akv_cache_header_host(ctypes.byref(p.c()), _i32p(lens), buf.ctypes.data, buf.size),
           "akv_cache_header_host")
    return buf


def akv_encode(p: Params, ctx_lens, K, V, arena, ws, stream=None):
    """K, V: CUDA bf16 [B][H][s_max][128]; arena, ws: CUDA uint8 buffers."""
    lens = _lens(ctx_lens)
    s_max = int(K.shape[2])
    _check(lib().akv_encode(ctypes.byref(p.c()), _i32p(lens), _dev_ptr(K), _dev_ptr(V), s_max, _dev_ptr(arena),
                            arena.numel() * arena.element_size(), _dev_ptr(ws), ws.numel() * ws.element_size(),
                            _stream_ptr(stream)), "akv_encode")


def akv_encode_noalloc(p: Params, ctx_lens, K, V, arena, stream=None):
    """akv_encode without a workspace argument: for callers that cannot obtain
    device memory for scratch.  The library's own static scratch array (16 MiB
    per device) is used instead; calls that overlap on the GPU race on it."""
    lens = _lens(ctx_lens)
    s_max = int(K.shape[2])
    _check(lib().akv_encode_noalloc(ctypes.byref(p.c()), _i32p(lens), _dev_ptr(K), _dev_ptr(V), s_max,
                                    _dev_ptr(arena), arena.numel() * arena.element_size(), _stream_ptr(stream)),
           "akv_encode_noalloc")


def akv_cache_size_select(p: Params, sel: SelectParams, ctx_lens):
    lens = _lens(ctx_lens)
    a, w = ctypes.c_size_t(), ctypes.c_size_t()
    _check(lib().akv_cache_size_select(ctypes.byref(p.c()), ctypes.byref(sel.c()), _i32p(lens), ctypes.byref(a),
                                       ctypes.byref(w)), "akv_cache_size_select")
    return a.value, w.value


def akv_encode_select(p: Params, sel: SelectParams, ctx_lens, K, V, Q, arena, ws, stream=None):
    """K, V: CUDA bf16 [B][H][s_max][128]; Q: CUDA bf16 [B][H][W*G][128] observation rows."""
    lens = _lens(ctx_lens)
    s_max = int(K.shape[2])
    _check(lib().akv_encode_select(ctypes.byref(p.c()), ctypes.byref(sel.c()), _i32p(lens), _dev_ptr(K), _dev_ptr(V),
                                   _dev_ptr(Q), s_max, _dev_ptr(arena), arena.numel() * arena.element_size(),
                                   _dev_ptr(ws), ws.numel() * ws.element_size(), _stream_ptr(stream)),
           "akv_encode_select")


_UNIT_FIELDS = (("anchor_k", np.uint16), ("anchor_v", np.uint16), ("anchor_pos", np.int32), ("idx_k", np.uint16),
                ("gamma_k", np.uint16), ("idx_v", np.uint16), ("gamma_v", np.uint16), ("res_pos_k", np.int32),
                ("codes_k", np.uint8), ("scale_k", np.uint16), ("min_k", np.uint16), ("res_pos_v", np.int32),
                ("codes_v", np.uint8), ("scale_v", np.uint16), ("min_v", np.uint16))


def akv_cache_pack_host(p: Params, ctx_lens, units) -> np.ndarray:
    """units: sequence of B*H mappings with the akv_unit_host array names; returns the arena image."""
    lens = _lens(ctx_lens)
    arena_bytes, _ = akv_cache_size(p, lens)
    keep = []
    arr = (_UnitHost * len(units))()
    for i, u in enumerate(units):
        for name, dt in _UNIT_FIELDS:
            a = np.ascontiguousarray(u[name], dtype=dt)
            keep.append(a)
            setattr(arr[i], name, a.ctypes.data if a.size else None)
    out = np.zeros(arena_bytes, np.uint8)
    _check(lib().akv_cache_pack_host(ctypes.byref(p.c()), _i32p(lens), arr, out.ctypes.data, out.size),
           "akv_cache_pack_host")
    return out


def akv_table1_bytes(p: Params, ctx_lens) -> np.ndarray:
    """Bytes of each request's layer in the paper's Table 1 layout (Lloyd-Max codec)."""
    lens = _lens(ctx_lens)
    out = np.zeros(p.batch, np.uint64)
    _check(lib().akv_table1_bytes(ctypes.byref(p.c()), _i32p(lens),
                                  out.ctypes.data_as(ctypes.POINTER(ctypes.c_size_t))), "akv_table1_bytes")
    return out


def akv_pack_table1_host(p: Params, ctx_lens, units) -> np.ndarray:
    """units as for akv_cache_pack_host (minima 0); returns the requests' Table 1 layers, concatenated."""
    lens = _lens(ctx_lens)
    total = int(akv_table1_bytes(p, lens).sum())
    keep = []
    arr = (_UnitHost * len(units))()
    for i, u in enumerate(units):
        for name, dt in _UNIT_FIELDS:
            a = np.ascontiguousarray(u[name], dtype=dt)
            keep.append(a)
            setattr(arr[i], name, a.ctypes.data if a.size else None)
    out = np.zeros(total, np.uint8)
    _check(lib().akv_pack_table1_host(ctypes.byref(p.c()), _i32p(lens), arr, out.ctypes.data, out.size),
           "akv_pack_table1_host")
    return out


def akv_decode_workspace_size(p: Params, ctx_lens, suffix_cap: int = 0) -> int:
    """Decode workspace bytes; with suffix_cap > 0, for akv_decode_attn with a dense suffix of at
    most that many tokens per request."""
    lens = _lens(ctx_lens)
    w = ctypes.c_size_t()
    _check(lib().akv_decode_workspace_size_suffix(ctypes.byref(p.c()), _i32p(lens), int(suffix_cap), ctypes.byref(w)),
           "akv_decode_workspace_size_suffix")
    return w.value


# The marshalled (params, lengths) of recent decode calls: a decode loop repeats them, and
# building the ctypes structures dominates the binding's share of a call.
_DECODE_ARGS: dict = {}


def _decode_args(p: Params, ctx_lens):
    key = (p.batch, p.n_kv_heads, p.n_q_heads, p.head_dim, p.anchor_frac, p.res_frac_k, p.res_frac_v, p.window,
           p.seed, p.rot_seed, p.rotate, p.lloyd, p.rope, p.rope_theta, tuple(int(x) for x in ctx_lens))
    ent = _DECODE_ARGS.get(key)
    if ent is None:
        if len(_DECODE_ARGS) >= 64:
            _DECODE_ARGS.clear()
        pc = p.c()
        lens = _lens(ctx_lens)
        ent = (pc, lens, ctypes.byref(pc), _i32p(lens))
        _DECODE_ARGS[key] = ent
    return ent[2], ent[3]


def akv_decode_attn(p: Params, ctx_lens, arena, q, out, out_f32=None, sm_scale: float = 1.0, ws=None, stream=None,
                    suffix=None):
    """q, out: CUDA bf16 [B][H_q][128]; out_f32 optional fp32 of the same shape.
    suffix: optional Suffix (the exact dense suffix attended in the same softmax).
    ws: CUDA uint8 workspace of akv_decode_workspace_size(p, ctx_lens, suffix.cap) bytes; when
    None, one is taken from torch's allocator on out's device for this call."""
    pref, lref = _decode_args(p, ctx_lens)
    if ws is None:
        import torch
        ws = torch.empty(akv_decode_workspace_size(p, ctx_lens, suffix.cap if suffix is not None else 0),
                         dtype=torch.uint8, device=out.device)
    ws_bytes = ws.numel() * ws.element_size()
    args = (pref, lref, _dev_ptr(arena), arena.numel() * arena.element_size(), _dev_ptr(q), _dev_ptr(out),
            _dev_ptr(out_f32), float(sm_scale))
    if suffix is None:
        _check(lib().akv_decode_attn(*args, _dev_ptr(ws), ws_bytes, _stream_ptr(stream)), "akv_decode_attn")
    else:
        _check(lib().akv_decode_attn_suffix(*args, ctypes.byref(suffix.c()), _dev_ptr(ws), ws_bytes,
                                            _stream_ptr(stream)), "akv_decode_attn_suffix")


class Suffix:
    """The exact dense suffix of a batch (generated tokens): CUDA bf16 K and V [B][H_kv][cap][128]
    and CUDA int32 lengths [B] (tokens held per request), all owned by the caller."""

    def __init__(self, K, V, lens):
        if K.dim() != 4 or tuple(K.shape) != tuple(V.shape) or K.shape[3] != HEAD_DIM:
            raise ValueError("suffix K and V must be [B][H_kv][cap][128] of the same shape")
        if str(K.dtype) != "torch.bfloat16" or str(V.dtype) != "torch.bfloat16" or str(lens.dtype) != "torch.int32":
            raise ValueError("suffix K, V must be bf16 and lens int32")
        if lens.numel() != K.shape[0]:
            raise ValueError("suffix lens must hold one length per request")
        self.K, self.V, self.lens = K, V, lens
        self.cap = int(K.shape[2])
        self._c = _Suffix(_dev_ptr(K), _dev_ptr(V), _dev_ptr(lens), self.cap)

    def c(self):
        return self._c


def akv_suffix_append(p: Params, K_new, V_new, suffix: "Suffix", stream=None):
    """Appends one token per request (K_new, V_new: CUDA bf16 [B][H_kv][128]) at each request's
    length, on the device; requests whose suffix is full are left unchanged."""
    _check(lib().akv_suffix_append(ctypes.byref(p.c()), _dev_ptr(K_new), _dev_ptr(V_new), _dev_ptr(suffix.K),
                                   _dev_ptr(suffix.V), _dev_ptr(suffix.lens), suffix.cap, _stream_ptr(stream)),
           "akv_suffix_append")


def akv_decode_set_debug(ctas: int = 0, withhold_last: int = 0):
    """Testing controls of the decode launch (0, 0 = normal operation): the number of decode
    CTAs (0 = one per SM), and withholding each CTA's last tile block."""
    _check(lib().akv_decode_set_debug(int(ctas), int(withhold_last)), "akv_decode_set_debug")


def akv_decode_set_events(after_scores=None, after_decode=None):
    """Timing aid: torch.cuda.Event objects (already recorded once, so that their CUDA events
    exist) that every later decode call records after its score launch and after its decode
    launch; call with no arguments to clear."""
    a = ctypes.c_void_p(after_scores.cuda_event) if after_scores is not None else None
    b = ctypes.c_void_p(after_decode.cuda_event) if after_decode is not None else None
    _check(lib().akv_decode_set_events(a, b), "akv_decode_set_events")


def unit_host_from_logical(u: dict) -> dict:
    """Map a logical-array dict (gen.seeded_cache naming) to akv_unit_host names."""
    return dict(anchor_k=u["anchor_k"], anchor_v=u["anchor_v"], anchor_pos=u["anchor_pos"], idx_k=u["idx_k"],
                gamma_k=u["gam_k"], idx_v=u["idx_v"], gamma_v=u["gam_v"], res_pos_k=u["res_k"],
                codes_k=u["codes_k"], scale_k=u["scale_k"], min_k=u["min_k"], res_pos_v=u["res_v"],
                codes_v=u["codes_v"], scale_v=u["scale_v"], min_v=u["min_v"])
