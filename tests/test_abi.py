"""C-ABI checks that need no GPU: exports, shapes, layout, host packer, validation."""
import ctypes
import os
import re

import numpy as np
import pytest

import gen
import oracle
from oracle import accounting as acc
import paper_2608_02901_gb300 as akv

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2608_02901_gb300 import build
    build.build()
    akv.lib()


def _declared_functions():
    txt = open(os.path.join(ROOT, "include", "akv.h")).read()
    txt = re.sub(r"/\*.*?\*/", "", txt, flags=re.S)
    return sorted(set(re.findall(r"\b(akv_[a-z0-9_]+)\s*\(", txt)))


def test_every_declared_symbol_is_exported():
    names = _declared_functions()
    assert len(names) >= 9
    L = ctypes.CDLL(akv.LIB_PATH)
    for n in names:
        assert hasattr(L, n), n
    assert set(names) == set(akv.EXPORTED)


def test_status_strings():
    assert akv.akv_status_string(0) == "AKV_OK"
    assert akv.akv_status_string(4) == "AKV_ERR_CUDA"
    assert akv.akv_status_string(99) == "AKV_ERR_UNKNOWN"


@pytest.mark.parametrize("S", [1, 7, 31, 32, 33, 100, 4096, 32768, 131072, 99991])
@pytest.mark.parametrize("fr", [(0.02, 0.1, 0.1), (0.01, 0.0, 0.2), (0.04, 1.0, 0.05)])
def test_unit_shapes_match_oracle(S, fr):
    p = akv.Params(batch=1, n_kv_heads=1, n_q_heads=1, anchor_frac=fr[0], res_frac_k=fr[1], res_frac_v=fr[2])
    got = akv.akv_unit_shapes(p, [S])[0]
    assert tuple(got) == (S, *oracle.unit_shape(S, *fr, 32))


def test_layout_header_and_sections():
    lens = [4096, 1000, 33]
    p = akv.Params(batch=3, n_kv_heads=2, n_q_heads=8, seed=3, rot_seed=9)
    arena_bytes, ws_bytes = akv.akv_cache_size(p, lens)
    hdr = akv.akv_cache_header_host(p, lens)
    assert hdr[:4].view(np.uint32)[0] == 0x31564B41 and hdr[4:8].view(np.uint32)[0] == 1
    assert hdr[8:16].view(np.uint64)[0] == arena_bytes
    assert hdr[72:76].view(np.int32)[0] == 6 and hdr[76:80].view(np.int32)[0] == 4096
    # sign bits: s_j = -1 iff bit j set, the same pattern the oracle derives from rot_seed
    bits = hdr[88:104].view(np.uint64)
    s = np.array([-1.0 if (int(bits[j // 64]) >> (j % 64)) & 1 else 1.0 for j in range(128)])
    assert np.array_equal(s, oracle.signs(9))
    prev_end = 256 * 7
    for u in range(6):
        d = hdr[256 * (u + 1): 256 * (u + 2)]
        S, k, nk, nv, nw, b, h = d[:28].view(np.int32)
        assert (b, h) == (u // 2, u % 2) and S == lens[b] and nw == (S + 63) // 64
        offs = d[32:136].view(np.uint64)
        sizes = [k * 256, k * 256, 4 * k, 4 * S, 4 * S, 8 * nw, 4 * nw, 8 * nw, 4 * nw, 32 * nk, 4 * nk, 32 * nv, 4 * nv]
        assert offs[0] % 256 == 0
        for o, sz in zip(offs, sizes):
            assert o % 128 == 0 and o >= prev_end
            prev_end = o + sz
        data = int(d[136:144].view(np.uint64)[0])
        assert data == acc.decode_read_bytes(S, k, nk, nv, G=0)
    assert prev_end <= arena_bytes
    assert ws_bytes > 0


def _seeded_units(p, lens, seed=5):
    shapes = akv.akv_unit_shapes(p, lens)
    return [gen.seeded_cache(int(S), int(k), int(nk), int(nv), p.window, seed, u)
            for u, (S, k, nk, nv) in enumerate(shapes)]


def test_pack_roundtrip_through_independent_unpacker():
    lens = [5000, 37, 129]
    p = akv.Params(batch=3, n_kv_heads=2, n_q_heads=4, res_frac_k=0.3, res_frac_v=0.05)
    units = _seeded_units(p, lens)
    arena = akv.akv_cache_pack_host(p, lens, [akv.unit_host_from_logical(u) for u in units])
    back = oracle.unpack_arena(arena)
    assert len(back) == len(units)
    for u, b in zip(units, back):
        for name in ("anchor_k", "anchor_v", "anchor_pos", "idx_k", "gam_k", "idx_v", "gam_v", "res_k", "codes_k",
                     "scale_k", "min_k", "res_v", "codes_v", "scale_v", "min_v"):
            assert np.array_equal(np.asarray(u[name]), getattr(b, name)), name


def _err(fn, *a):
    with pytest.raises(akv.AkvError) as e:
        fn(*a)
    return e.value.status


def test_parameter_validation():
    base = dict(batch=1, n_kv_heads=1, n_q_heads=1)
    assert _err(akv.akv_cache_size, akv.Params(**base, head_dim=64), [100]) == akv.AKV_ERR_UNSUPPORTED
    assert _err(akv.akv_cache_size, akv.Params(batch=1, n_kv_heads=2, n_q_heads=6), [100]) == akv.AKV_ERR_UNSUPPORTED
    assert _err(akv.akv_cache_size, akv.Params(batch=1, n_kv_heads=2, n_q_heads=3), [100]) == akv.AKV_ERR_INVALID
    assert _err(akv.akv_cache_size, akv.Params(**base, anchor_frac=1.5), [100]) == akv.AKV_ERR_INVALID
    assert _err(akv.akv_cache_size, akv.Params(**base, res_frac_k=float("nan")), [100]) == akv.AKV_ERR_INVALID
    assert _err(akv.akv_cache_size, akv.Params(**base, window=-1), [100]) == akv.AKV_ERR_INVALID
    assert _err(akv.akv_cache_size, akv.Params(**base), [0]) == akv.AKV_ERR_INVALID
    assert _err(akv.akv_cache_size, akv.Params(**base, window=0, anchor_frac=0.0), [100]) == akv.AKV_ERR_INVALID
    assert _err(akv.akv_cache_size, akv.Params(**base, anchor_frac=0.02), [4_000_000]) == akv.AKV_ERR_UNSUPPORTED
    assert akv.akv_decode_workspace_size(akv.Params(**base), [100]) == 0


def test_pack_rejects_bad_arrays():
    lens = [300]
    p = akv.Params(batch=1, n_kv_heads=1, n_q_heads=1)
    u = akv.unit_host_from_logical(_seeded_units(p, lens)[0])
    bad = dict(u)
    bad["idx_k"] = u["idx_k"].copy()
    bad["idx_k"][3] = 60000
    assert _err(akv.akv_cache_pack_host, p, lens, [bad]) == akv.AKV_ERR_INVALID
    bad = dict(u)
    bad["res_pos_v"] = u["res_pos_v"][::-1].copy()
    assert _err(akv.akv_cache_pack_host, p, lens, [bad]) == akv.AKV_ERR_INVALID


def test_entry_points_validate_before_any_launch():
    """Null or misaligned device pointers are rejected on the host (no CUDA call is made)."""
    L = akv.lib()
    p = akv.Params(batch=1, n_kv_heads=1, n_q_heads=1).c()
    lens = np.array([100], np.int32)
    lp = lens.ctypes.data_as(ctypes.POINTER(ctypes.c_int32))
    nbytes, _ = akv.akv_cache_size(akv.Params(batch=1, n_kv_heads=1, n_q_heads=1), lens)
    st = L.akv_decode_attn(ctypes.byref(p), lp, None, nbytes, 256, 256, None, 1.0, None, 0, None)
    assert st == akv.AKV_ERR_INVALID
    st = L.akv_decode_attn(ctypes.byref(p), lp, 0x1000 + 8, nbytes, 256, 256, None, 1.0, None, 0, None)
    assert st == akv.AKV_ERR_INVALID and "aligned" in akv.akv_last_error()
    st = L.akv_decode_attn(ctypes.byref(p), lp, 0x1000, nbytes - 1, 256, 256, None, 1.0, None, 0, None)
    assert st == akv.AKV_ERR_TOO_SMALL
    st = L.akv_decode_attn(ctypes.byref(p), lp, 0x1000, nbytes, 256, 256, None, float("inf"), None, 0, None)
    assert st == akv.AKV_ERR_INVALID
    st = L.akv_encode(ctypes.byref(p), lp, None, 256, 128, 0x1000, nbytes, 0x2000, 1 << 20, None)
    assert st == akv.AKV_ERR_INVALID
    st = L.akv_encode(ctypes.byref(p), lp, 256, 256, 50, 0x1000, nbytes, 0x2000, 1 << 20, None)
    assert st == akv.AKV_ERR_INVALID  # s_max < S
    st = L.akv_encode(ctypes.byref(p), lp, 256, 256, 128, 0x1000, nbytes, 0x2000, 16, None)
    assert st == akv.AKV_ERR_TOO_SMALL
