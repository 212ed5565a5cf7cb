"""fp64 CPU oracle of AnchorKV (arXiv 2608.02901) -- test infrastructure only.

Only the tests, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  The product library never calls it and
shares no code with it: ``akv_oracle.c`` is written from the paper's
equations (Section 3.1 Eq. 1-3, Section 3.3 Eq. 4, Appendix A.1 Eq. 12-14,
Section 3.2 anchor selection) and the readings R1-R16 where the paper is
silent or ambiguous (GQA mapping, anchor sampling, tie rules, rounding, the
quantizer's scale and min, the stored token order).

Every function here is marshalling around the C file; the arithmetic lives
there.  Parity status: every function is pinned by ``tests/test_oracle_*.py``
against brute force, closed forms and the paper's worked example.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from dataclasses import dataclass

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "akv_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None

D = 128


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (IEEE semantics: no contraction, no fast-math)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp", "-ffp-contract=off",
               "-fno-fast-math", "-o", tmp, _SRC, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB)
    return _LIB


class _OrUnit(ctypes.Structure):
    _fields_ = [("S", ctypes.c_int32), ("k", ctypes.c_int32), ("nk", ctypes.c_int32), ("nv", ctypes.c_int32)] + [
        (name, ctypes.c_void_p)
        for name in ("anchor_k", "anchor_v", "anchor_pos", "idx_k", "gam_k", "idx_v", "gam_v", "res_k", "codes_k",
                     "scale_k", "min_k", "res_v", "codes_v", "scale_v", "min_v", "pos")
    ]


def lib():
    global _lib
    with _lock:
        if _lib is None:
            path = build()
            L = ctypes.CDLL(path)
            u64, i32, vp, dbl = ctypes.c_uint64, ctypes.c_int32, ctypes.c_void_p, ctypes.c_double
            L.or_splitmix64.restype = u64
            L.or_splitmix64.argtypes = [u64]
            L.or_fp16_from_double.restype = ctypes.c_uint16
            L.or_fp16_from_double.argtypes = [dbl]
            L.or_fp16_to_double.restype = dbl
            L.or_fp16_to_double.argtypes = [ctypes.c_uint16]
            L.or_bf16_to_double.restype = dbl
            L.or_bf16_to_double.argtypes = [ctypes.c_uint16]
            L.or_signs.argtypes = [u64, vp]
            L.or_wht128.argtypes = [vp]
            L.or_unit_shape.argtypes = [i32, ctypes.c_float, ctypes.c_float, ctypes.c_float, i32, vp, vp, vp]
            L.or_encode_unit.restype = ctypes.c_int
            L.or_encode_unit.argtypes = [vp, vp, i32, i32, i32, u64, u64, ctypes.c_int, ctypes.POINTER(_OrUnit)]
            L.or_encode_batch.restype = ctypes.c_int
            L.or_encode_batch.argtypes = [vp, vp, i32, i32, i32, i32, u64, u64, ctypes.c_int, vp]
            L.or_attend_unit.argtypes = [ctypes.POINTER(_OrUnit), vp, i32, dbl, u64, ctypes.c_int, vp]
            L.or_attend_batch.argtypes = [vp, i32, vp, i32, dbl, u64, ctypes.c_int, dbl, vp, vp]
            L.or_attend_batch_suffix.argtypes = [vp, i32, i32, vp, i32, dbl, u64, ctypes.c_int, dbl, vp, vp, vp, i32,
                                                 vp]
            L.or_rope.argtypes = [vp, ctypes.c_int64, dbl]
            L.or_attend_factorized.argtypes = [ctypes.POINTER(_OrUnit), vp, i32, dbl, u64, ctypes.c_int, vp]
            L.or_reconstruct_side.argtypes = [i32, vp, vp, vp, i32, vp, vp, vp, vp, u64, ctypes.c_int, vp]
            L.or_quantize_residual.argtypes = [vp, u64, ctypes.c_int, vp, vp, vp]
            L.or_dequantize_residual.argtypes = [vp, ctypes.c_uint16, ctypes.c_uint16, u64, ctypes.c_int, vp]
            L.or_arena_shape.restype = ctypes.c_int
            L.or_arena_shape.argtypes = [vp, u64, i32, vp]
            L.or_exp_neg.restype = dbl
            L.or_exp_neg.argtypes = [dbl]
            L.or_selector_scores_unit.argtypes = [i32, i32, i32, i32, vp, vp, vp]
            L.or_budget_n.restype = ctypes.c_int64
            L.or_budget_n.argtypes = [dbl, i32, i32, i32, i32]
            L.or_utilities_unit.argtypes = [ctypes.POINTER(_OrUnit), vp, vp, vp, i32, vp, vp]
            L.or_encode_select_batch.restype = ctypes.c_int
            L.or_encode_select_batch.argtypes = [vp, vp, vp, i32, i32, i32, i32, i32, ctypes.c_float, ctypes.c_float,
                                                 i32, u64, u64, ctypes.c_int, vp]
            L.or_arena_unpack.restype = ctypes.c_int
            L.or_arena_unpack.argtypes = [vp, u64, i32, ctypes.POINTER(_OrUnit)]
            _lib = L
    return _lib


def _p(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


@dataclass
class Unit:
    """Logical compressed cache of one (request, KV head): the arrays of Table 1."""
    S: int
    k: int
    nk: int
    nv: int
    anchor_k: np.ndarray
    anchor_v: np.ndarray
    anchor_pos: np.ndarray
    idx_k: np.ndarray
    gam_k: np.ndarray
    idx_v: np.ndarray
    gam_v: np.ndarray
    res_k: np.ndarray
    codes_k: np.ndarray
    scale_k: np.ndarray
    min_k: np.ndarray
    res_v: np.ndarray
    codes_v: np.ndarray
    scale_v: np.ndarray
    min_v: np.ndarray
    pos: np.ndarray = None  # [S] int32 position of index i (RoPE at decode); None: position i

    def c_struct(self) -> _OrUnit:
        s = _OrUnit(self.S, self.k, self.nk, self.nv)
        for name in ("anchor_k", "anchor_v", "anchor_pos", "idx_k", "gam_k", "idx_v", "gam_v", "res_k", "codes_k",
                     "scale_k", "min_k", "res_v", "codes_v", "scale_v", "min_v", "pos"):
            arr = getattr(self, name)
            if arr is None:
                continue
            assert arr.flags.c_contiguous
            setattr(s, name, arr.ctypes.data if arr.size else None)
        return s


def alloc_unit(S: int, k: int, nk: int, nv: int) -> Unit:
    z = np.zeros
    return Unit(S, k, nk, nv,
                z((k, D), np.uint16), z((k, D), np.uint16), z(k, np.int32),
                z(S, np.uint16), z(S, np.uint16), z(S, np.uint16), z(S, np.uint16),
                z(nk, np.int32), z((nk, 32), np.uint8), z(nk, np.uint16), z(nk, np.uint16),
                z(nv, np.int32), z((nv, 32), np.uint8), z(nv, np.uint16), z(nv, np.uint16), np.arange(S, dtype=np.int32))


# ---- scalar helpers -------------------------------------------------------

def _flags(rotate: bool, lloyd: bool) -> int:
    """Codec flags of the C oracle: bit 0 the Hadamard rotation, bit 1 the Lloyd-Max codebook."""
    return (1 if rotate else 0) | (2 if lloyd else 0)


def splitmix64(x: int) -> int:
    return int(lib().or_splitmix64(ctypes.c_uint64(x & 0xFFFFFFFFFFFFFFFF)))


def fp16_from_double(x: float) -> int:
    return int(lib().or_fp16_from_double(float(x)))


def fp16_to_double(h: int) -> float:
    return float(lib().or_fp16_to_double(int(h) & 0xFFFF))


def bf16_to_double(b: int) -> float:
    return float(lib().or_bf16_to_double(int(b) & 0xFFFF))


def signs(rot_seed: int) -> np.ndarray:
    s = np.zeros(D, np.float64)
    lib().or_signs(ctypes.c_uint64(rot_seed), _p(s))
    return s


def wht128(v: np.ndarray) -> np.ndarray:
    out = np.ascontiguousarray(v, dtype=np.float64).copy()
    assert out.shape == (D,)
    lib().or_wht128(_p(out))
    return out


def rope(x: np.ndarray, p: int, base: float) -> np.ndarray:
    """The oracle's RoPE turn of one 128-vector to position p (rotate-half pairs (j, j + 64))."""
    out = np.ascontiguousarray(x, dtype=np.float64).copy()
    assert out.shape == (D,)
    lib().or_rope(_p(out), int(p), float(base))
    return out


def quantize_residual(r: np.ndarray, rot_seed: int, rotate: bool = True, lloyd: bool = False):
    """Rotate and quantize one residual; returns (codes[32] uint8, scale fp16 bits, min fp16 bits)."""
    r = np.ascontiguousarray(r, dtype=np.float64)
    assert r.shape == (D,)
    codes = np.zeros(32, np.uint8)
    sc = np.zeros(1, np.uint16)
    mn = np.zeros(1, np.uint16)
    lib().or_quantize_residual(_p(r), ctypes.c_uint64(rot_seed), _flags(rotate, lloyd), _p(codes), _p(sc), _p(mn))
    return codes, int(sc[0]), int(mn[0])


def dequantize_residual(codes: np.ndarray, sc: int, mn: int, rot_seed: int, rotate: bool = True,
                        lloyd: bool = False) -> np.ndarray:
    """r~ = U^T C^-1(q) of one record (Eq. 14): fp64 [128]."""
    codes = np.ascontiguousarray(codes, dtype=np.uint8)
    out = np.zeros(D, np.float64)
    lib().or_dequantize_residual(_p(codes), int(sc), int(mn), ctypes.c_uint64(rot_seed), _flags(rotate, lloyd),
                                 _p(out))
    return out


def eta(residuals: np.ndarray, rot_seed: int, rotate: bool = True, lloyd: bool = False) -> float:
    """Eq. 13: the relative squared distortion E||r - r~||^2 / ||r||^2 the codec leaves, as the mean
    over the given residuals (fp64 [n][128], zero rows skipped) of ||r - r~||^2 / ||r||^2."""
    vals = []
    for r in np.asarray(residuals, np.float64):
        nr = float(r @ r)
        if nr == 0.0:
            continue
        codes, sc, mn = quantize_residual(r, rot_seed, rotate, lloyd)
        e = r - dequantize_residual(codes, sc, mn, rot_seed, rotate, lloyd)
        vals.append(float(e @ e) / nr)
    return float(np.mean(vals))


def unit_shape(S: int, f_a: float, f_rk: float, f_rv: float, W: int):
    k, nk, nv = ctypes.c_int32(), ctypes.c_int32(), ctypes.c_int32()
    lib().or_unit_shape(S, f_a, f_rk, f_rv, W, ctypes.byref(k), ctypes.byref(nk), ctypes.byref(nv))
    return k.value, nk.value, nv.value


# ---- encode / attend --------------------------------------------------------

def encode(K: np.ndarray, V: np.ndarray, ctx_lens, n_kv_heads: int, f_a: float, f_rk: float, f_rv: float, W: int,
           seed: int, rot_seed: int, rotate: bool = True, lloyd: bool = False) -> list:
    """K, V: uint16 bf16 bits [B][H][s_max][128].  Returns B*H Units (u = b*H + h)."""
    K = np.ascontiguousarray(K, dtype=np.uint16)
    V = np.ascontiguousarray(V, dtype=np.uint16)
    B, H, s_max, d = K.shape
    assert H == n_kv_heads and d == D and V.shape == K.shape and len(ctx_lens) == B
    units = []
    for b in range(B):
        for h in range(H):
            S = int(ctx_lens[b])
            assert 1 <= S <= s_max
            units.append(alloc_unit(S, *unit_shape(S, f_a, f_rk, f_rv, W)))
    structs = (_OrUnit * len(units))(*[u.c_struct() for u in units])
    rc = lib().or_encode_batch(_p(K), _p(V), s_max, len(units), H, W, ctypes.c_uint64(seed),
                               ctypes.c_uint64(rot_seed), _flags(rotate, lloyd), ctypes.cast(structs, ctypes.c_void_p))
    if rc != 0:
        raise RuntimeError("oracle encode failed")
    return units


# ---- the paper's full selection (Algorithm 1; Section 3.2-3.4, Appendix A.2) ----------

def exp_neg(x: float) -> float:
    """e^x for x <= 0 by the oracle's Cody-Waite + Taylor evaluation."""
    return float(lib().or_exp_neg(float(x)))


def selector_scores(K: np.ndarray, Q: np.ndarray, W: int, kappa: int) -> np.ndarray:
    """Appendix A.2 selector scores of positions [0, S - min(W, S)) of one unit:
    K bf16 bits [S][128], Q bf16 bits [m][128] (the observation rows)."""
    K = np.ascontiguousarray(K, dtype=np.uint16)
    Q = np.ascontiguousarray(Q, dtype=np.uint16)
    S, m = K.shape[0], Q.shape[0]
    out = np.zeros(max(0, S - min(W, S)), np.float64)
    lib().or_selector_scores_unit(S, W, m, kappa, _p(K), _p(Q), _p(out) if out.size else None)
    return out


def budget_n(theta: float, S: int, H: int, W: int, k: int) -> int:
    """Eq. 9 residual count of one layer with the Appendix A.1 accounting."""
    return int(lib().or_budget_n(float(theta), S, H, W, k))


def utilities(unit: "Unit", K: np.ndarray, V: np.ndarray, Q: np.ndarray):
    """Eq. 6 utilities (u^K, u^V) of every position of a unit given its anchors and
    coefficients; anchors get -1."""
    K = np.ascontiguousarray(K, dtype=np.uint16)
    V = np.ascontiguousarray(V, dtype=np.uint16)
    Q = np.ascontiguousarray(Q, dtype=np.uint16)
    uk = np.zeros(unit.S, np.float64)
    uv = np.zeros(unit.S, np.float64)
    s = unit.c_struct()
    lib().or_utilities_unit(ctypes.byref(s), _p(K), _p(V), _p(Q), Q.shape[0], _p(uk), _p(uv))
    return uk, uv


def encode_select(K: np.ndarray, V: np.ndarray, Q: np.ndarray, ctx_lens, n_kv_heads: int, f_a: float, W: int,
                  theta: float, rho: float, kappa: int, seed: int, rot_seed: int, rotate: bool = True, lloyd: bool = False) -> list:
    """Algorithm 1 with the paper's selection.  K, V bf16 bits [B][H][s_max][128];
    Q bf16 bits [B][H][m][128], m = W G.  Returns B*H Units with per-unit residual counts."""
    K = np.ascontiguousarray(K, dtype=np.uint16)
    V = np.ascontiguousarray(V, dtype=np.uint16)
    Q = np.ascontiguousarray(Q, dtype=np.uint16)
    B, H, s_max, d = K.shape
    m = Q.shape[2]
    assert H == n_kv_heads and d == D and Q.shape[:2] == (B, H) and len(ctx_lens) == B
    f32 = ctypes.c_float
    units = []
    for b in range(B):
        S = int(ctx_lens[b])
        k, _, _ = unit_shape(S, f_a, 0.0, 0.0, W)
        N = budget_n(float(f32(theta).value), S, H, W, k)
        cap_k, cap_v = min(N // 2, S - k), min(N - N // 2, S - k)
        for h in range(H):
            units.append(alloc_unit(S, k, cap_k, cap_v))
    structs = (_OrUnit * len(units))(*[u.c_struct() for u in units])
    rc = lib().or_encode_select_batch(_p(K), _p(V), _p(Q), s_max, B, H, m, W, theta, rho, kappa,
                                      ctypes.c_uint64(seed), ctypes.c_uint64(rot_seed), _flags(rotate, lloyd),
                                      ctypes.cast(structs, ctypes.c_void_p))
    if rc != 0:
        raise RuntimeError("oracle select encode failed")
    out = []
    for u, s in zip(units, structs):
        nk, nv = int(s.nk), int(s.nv)
        out.append(Unit(u.S, u.k, nk, nv, u.anchor_k, u.anchor_v, u.anchor_pos, u.idx_k, u.gam_k, u.idx_v, u.gam_v,
                        u.res_k[:nk].copy(), u.codes_k[:nk].copy(), u.scale_k[:nk].copy(), u.min_k[:nk].copy(),
                        u.res_v[:nv].copy(), u.codes_v[:nv].copy(), u.scale_v[:nv].copy(), u.min_v[:nv].copy()))
    return out


def attend(units, q: np.ndarray, G: int, sm_scale: float, rot_seed: int, rotate: bool = True, lloyd: bool = False,
           sel=None, rope_theta: float = 0.0) -> np.ndarray:
    """q: uint16 bf16 bits [n_units][G][128] (or [B][H_q][128]); returns fp64 of the same shape.
    rope_theta > 0: keys are pre-RoPE and each is turned to its position (unit.pos) first."""
    n = len(units)
    q = np.ascontiguousarray(q, dtype=np.uint16).reshape(n, G, D)
    out = np.zeros((n, G, D), np.float64)
    structs = (_OrUnit * n)(*[u.c_struct() for u in units])
    selp = None
    if sel is not None:
        sel_arr = np.ascontiguousarray(sel, dtype=np.uint8)
        assert sel_arr.shape == (n,)
        selp = _p(sel_arr)
    lib().or_attend_batch(ctypes.cast(structs, ctypes.c_void_p), n, _p(q), G, float(sm_scale),
                          ctypes.c_uint64(rot_seed), _flags(rotate, lloyd) | (4 if rope_theta > 0 else 0),
                          float(rope_theta), selp, _p(out))
    return out


def attend_suffix(units, q: np.ndarray, G: int, H: int, sm_scale: float, rot_seed: int, ksuf: np.ndarray,
                  vsuf: np.ndarray, suf_len, rotate: bool = True, lloyd: bool = False,
                  rope_theta: float = 0.0) -> np.ndarray:
    """Attention over each unit's compressed positions and the first suf_len[b] rows of its exact
    dense suffix, in one softmax (Appendix E.1, E.2).  ksuf, vsuf: uint16 bf16 bits
    [n_units][cap][128] (unit u = b*H + h); suf_len: int [B].  Returns fp64 [n_units][G][128]."""
    n = len(units)
    q = np.ascontiguousarray(q, dtype=np.uint16).reshape(n, G, D)
    ksuf = np.ascontiguousarray(ksuf, dtype=np.uint16)
    vsuf = np.ascontiguousarray(vsuf, dtype=np.uint16)
    assert ksuf.shape == vsuf.shape and ksuf.shape[0] == n and ksuf.shape[2] == D
    lens = np.ascontiguousarray(np.minimum(np.asarray(suf_len, dtype=np.int32), ksuf.shape[1]), dtype=np.int32)
    assert lens.shape == (n // H,)
    out = np.zeros((n, G, D), np.float64)
    structs = (_OrUnit * n)(*[u.c_struct() for u in units])
    lib().or_attend_batch_suffix(ctypes.cast(structs, ctypes.c_void_p), n, H, _p(q), G, float(sm_scale),
                                 ctypes.c_uint64(rot_seed), _flags(rotate, lloyd) | (4 if rope_theta > 0 else 0),
                                 float(rope_theta), _p(ksuf), _p(vsuf), _p(lens),
                                 int(ksuf.shape[1]), _p(out))
    return out


def attend_factorized(unit: Unit, q: np.ndarray, G: int, sm_scale: float, rot_seed: int, rotate: bool = True, lloyd: bool = False):
    q = np.ascontiguousarray(q, dtype=np.uint16).reshape(G, D)
    out = np.zeros((G, D), np.float64)
    s = unit.c_struct()
    lib().or_attend_factorized(ctypes.byref(s), _p(q), G, float(sm_scale), ctypes.c_uint64(rot_seed),
                               _flags(rotate, lloyd), _p(out))
    return out


def reconstruct(unit: Unit, side: str, rot_seed: int, rotate: bool = True, lloyd: bool = False) -> np.ndarray:
    """x^ of Eq. 3 for every position of one side ('k' or 'v'): fp64 [S][128]."""
    out = np.zeros((unit.S, D), np.float64)
    if side == "k":
        arrs = (unit.anchor_k, unit.idx_k, unit.gam_k, unit.nk, unit.res_k, unit.codes_k, unit.scale_k, unit.min_k)
    else:
        arrs = (unit.anchor_v, unit.idx_v, unit.gam_v, unit.nv, unit.res_v, unit.codes_v, unit.scale_v, unit.min_v)
    anc, idx, gam, n, res, codes, sc, mn = arrs
    lib().or_reconstruct_side(unit.S, _p(anc), _p(idx), _p(gam), n, _p(res), _p(codes), _p(sc), _p(mn),
                              ctypes.c_uint64(rot_seed), _flags(rotate, lloyd), _p(out))
    return out


def unpack_arena(arena) -> list:
    """Independent reader of the packed arena bytes; returns the Units."""
    buf = np.frombuffer(arena, dtype=np.uint8) if not isinstance(arena, np.ndarray) else arena.view(np.uint8)
    buf = np.ascontiguousarray(buf)
    n_units = int(buf[72:76].view(np.int32)[0])
    units = []
    for u in range(n_units):
        sh = np.zeros(4, np.int32)
        if lib().or_arena_shape(_p(buf), buf.size, u, _p(sh)) != 0:
            raise ValueError(f"malformed arena header/descriptor for unit {u}")
        unit = alloc_unit(*[int(x) for x in sh])
        s = unit.c_struct()
        if lib().or_arena_unpack(_p(buf), buf.size, u, ctypes.byref(s)) != 0:
            raise ValueError(f"inconsistent arena contents for unit {u}")
        units.append(unit)
    return units
