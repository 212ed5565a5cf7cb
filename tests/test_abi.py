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
from helpers import assert_same_unit, stored_order

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
    lens = [4096, 1000, 33, 5000]
    p = akv.Params(batch=4, n_kv_heads=2, n_q_heads=8, seed=3, rot_seed=9)
    arena_bytes, ws_bytes = akv.akv_cache_size(p, lens)
    hdr = akv.akv_cache_header_host(p, lens)
    assert hdr[:4].view(np.uint32)[0] == 0x32564B41 and hdr[4:8].view(np.uint32)[0] == 4
    assert hdr[8:16].view(np.uint64)[0] == arena_bytes
    assert hdr[72:76].view(np.int32)[0] == 8 and hdr[76:80].view(np.int32)[0] == 5000
    assert hdr[104:108].view(np.int32)[0] == 1024
    # sign bits: s_j = -1 iff bit j set, the same pattern the oracle derives from rot_seed
    bits = hdr[88:104].view(np.uint64)
    s = np.array([-1.0 if (int(bits[j // 64]) >> (j % 64)) & 1 else 1.0 for j in range(128)])
    assert np.array_equal(s, oracle.signs(9))
    prev_end = 256 * 9
    for u in range(8):
        d = hdr[256 * (u + 1): 256 * (u + 2)]
        S, k, nk, nv, nt, b, h = d[:28].view(np.int32)
        assert (b, h) == (u // 2, u % 2) and S == lens[b] and nt == (S + 1023) // 1024
        offs = d[32:72].view(np.uint64)
        cap, data = (int(x) for x in d[72:88].view(np.uint64))
        # fixed part of every tile (streams, bitmaps, rank words), records, <= 24 B of scale
        # padding and <= 480 B of value-code group padding per tile
        fixed = 0
        for j in range(nt):
            nw = (min(1024, S - 1024 * j) + 63) // 64
            fixed += 512 * nw + 16 * nw + 2 * ((2 * nw + 15) // 16 * 16)
        assert cap == fixed + 36 * (nk + nv) + 504 * nt
        # tile table: nt + 1 block offsets and one value-slot range word per tile
        sizes = [k * 256, k * 256, 4 * k, 4 * (2 * nt + 1), cap]
        assert offs[0] % 256 == 0
        for o, sz in zip(offs, sizes):
            assert o % 128 == 0 and o >= prev_end
            prev_end = o + sz
        assert data == 512 * k + 4 * (2 * nt + 1) + cap
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
    for i, (u, b) in enumerate(zip(units, back)):
        assert_same_unit(b, stored_order(u), f"unit {i}")
    # attention does not depend on the token order: the unpacked (stored-order) units
    # attend exactly like the position-ordered ones
    q = gen.queries(p.n_units * p.G, seed=3).reshape(p.n_units, p.G, 128)
    pos_units = [oracle.alloc_unit(d["S"], d["k"], d["nk"], d["nv"]) for d in units]
    for pu, d in zip(pos_units, units):
        for name in ("anchor_k", "anchor_v", "anchor_pos", "idx_k", "gam_k", "idx_v", "gam_v", "res_k", "codes_k",
                     "scale_k", "min_k", "res_v", "codes_v", "scale_v", "min_v"):
            getattr(pu, name)[...] = d[name]
    a = oracle.attend(pos_units, q, p.G, 1.0, p.rot_seed, p.rotate)
    b = oracle.attend(back, q, p.G, 1.0, p.rot_seed, p.rotate)
    assert np.max(np.abs(a - b)) <= 1e-12 * max(1.0, np.max(np.abs(a)))


def test_stored_order_is_sorted_by_value_anchor_and_tiles_are_consistent():
    lens = [3000]
    p = akv.Params(batch=1, n_kv_heads=1, n_q_heads=1, anchor_frac=0.01, res_frac_k=0.2, res_frac_v=0.1)
    units = _seeded_units(p, lens, seed=9)
    arena = akv.akv_cache_pack_host(p, lens, [akv.unit_host_from_logical(u) for u in units])
    back = oracle.unpack_arena(arena)[0]
    assert np.all(np.diff(back.idx_v.astype(np.int64)) >= 0)
    hdr = akv.akv_cache_header_host(p, lens)
    d = hdr[256:512]
    o_tt = int(d[56:64].view(np.uint64)[0])
    nt = int(d[16:20].view(np.int32)[0])
    table = arena[o_tt:o_tt + 4 * (nt + 1)].view(np.uint32)
    assert table[0] == 0 and np.all(np.diff(table.astype(np.int64)) > 0) and np.all(table % 16 == 0)
    # a damaged table is refused by the independent reader
    bad = arena.copy()
    bad[o_tt + 4:o_tt + 8] = np.frombuffer(np.uint32(table[1] + 16).tobytes(), np.uint8)
    with pytest.raises(ValueError):
        oracle.unpack_arena(bad)


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
    assert akv.akv_decode_workspace_size(akv.Params(**base), [100]) > 0


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
    wbytes = akv.akv_decode_workspace_size(akv.Params(batch=1, n_kv_heads=1, n_q_heads=1), lens)
    st = L.akv_decode_attn(ctypes.byref(p), lp, 0x1000, nbytes, 256, 256, None, 1.0, None, wbytes, None)
    assert st == akv.AKV_ERR_INVALID and "workspace" in akv.akv_last_error()
    st = L.akv_decode_attn(ctypes.byref(p), lp, 0x1000, nbytes, 256, 256, None, 1.0, 0x3000 + 16, wbytes, None)
    assert st == akv.AKV_ERR_INVALID
    st = L.akv_decode_attn(ctypes.byref(p), lp, 0x1000, nbytes, 256, 256, None, 1.0, 0x3000, wbytes - 1, None)
    assert st == akv.AKV_ERR_TOO_SMALL
    st = L.akv_encode(ctypes.byref(p), lp, None, 256, 128, 0x1000, nbytes, 0x2000, 1 << 20, None)
    assert st == akv.AKV_ERR_INVALID
    st = L.akv_encode(ctypes.byref(p), lp, 256, 256, 50, 0x1000, nbytes, 0x2000, 1 << 20, None)
    assert st == akv.AKV_ERR_INVALID  # s_max < S
    st = L.akv_encode(ctypes.byref(p), lp, 256, 256, 128, 0x1000, nbytes, 0x2000, 16, None)
    assert st == akv.AKV_ERR_TOO_SMALL
    # the dense suffix: pointers, capacity, and a workspace sized for the suffix's chunks
    sp = ctypes.byref
    S = akv._Suffix
    wb = akv.akv_decode_workspace_size(akv.Params(batch=1, n_kv_heads=1, n_q_heads=1), lens)
    ws_s = akv.akv_decode_workspace_size(akv.Params(batch=1, n_kv_heads=1, n_q_heads=1), lens, 1000)
    assert ws_s > wb
    for bad_sfx in (S(None, 0x5000, 0x6000, 10), S(0x4000, 0x5000, None, 10), S(0x4008, 0x5000, 0x6000, 10),
                    S(0x4000, 0x5000, 0x6002, 10), S(0x4000, 0x5000, 0x6000, 0),
                    S(0x4000, 0x5000, 0x6000, akv.AKV_MAX_SUFFIX + 1)):
        st = L.akv_decode_attn_suffix(sp(p), lp, 0x1000, nbytes, 256, 256, None, 1.0, sp(bad_sfx), 0x3000, ws_s, None)
        assert st == akv.AKV_ERR_INVALID, akv.akv_last_error()
    st = L.akv_decode_attn_suffix(sp(p), lp, 0x1000, nbytes, 256, 256, None, 1.0, sp(S(0x4000, 0x5000, 0x6000, 1000)),
                                  0x3000, ws_s - 1, None)
    assert st == akv.AKV_ERR_TOO_SMALL
    w = ctypes.c_size_t()
    assert L.akv_decode_workspace_size_suffix(sp(p), lp, -1, sp(w)) == akv.AKV_ERR_INVALID
    assert L.akv_suffix_append(sp(p), None, 0x2000, 0x3000, 0x4000, 0x5000, 8, None) == akv.AKV_ERR_INVALID
    assert L.akv_suffix_append(sp(p), 0x1000, 0x2000, 0x3000, 0x4000, 0x5002, 8, None) == akv.AKV_ERR_INVALID
    assert L.akv_suffix_append(sp(p), 0x1000, 0x2000, 0x3000, 0x4000, 0x5000, 0, None) == akv.AKV_ERR_INVALID
    # RoPE at decode: the base must be given with the flag (and only with it); no suffix with it
    pr = akv.Params(batch=1, n_kv_heads=1, n_q_heads=1, rope=True).c()
    sz = ctypes.c_size_t()
    assert L.akv_cache_size(sp(pr), lp, sp(sz), None) == akv.AKV_OK and sz.value > nbytes  # + positions
    for theta in (0.0, 1.0, float("inf"), float("nan")):
        bad = akv.Params(batch=1, n_kv_heads=1, n_q_heads=1, rope=True).c()
        bad.rope_theta = theta
        assert L.akv_cache_size(sp(bad), lp, sp(sz), None) == akv.AKV_ERR_INVALID
    bad = akv.Params(batch=1, n_kv_heads=1, n_q_heads=1).c()
    bad.rope_theta = 10000.0
    assert L.akv_cache_size(sp(bad), lp, sp(sz), None) == akv.AKV_ERR_INVALID
    # a suffix with RoPE: validated like any other (a short workspace is refused before any launch)
    ws_r = akv.akv_decode_workspace_size(akv.Params(batch=1, n_kv_heads=1, n_q_heads=1, rope=True), lens, 1000)
    st = L.akv_decode_attn_suffix(sp(pr), lp, 0x1000, sz.value, 256, 256, None, 1.0,
                                  sp(S(0x4000, 0x5000, 0x6000, 1000)), 0x3000, ws_r - 1, None)
    assert st == akv.AKV_ERR_TOO_SMALL


def test_decode_debug_controls_validate():
    assert _err(akv.akv_decode_set_debug, 257, 0) == akv.AKV_ERR_INVALID
    assert _err(akv.akv_decode_set_debug, -1, 0) == akv.AKV_ERR_INVALID
    assert _err(akv.akv_decode_set_debug, 0, 2) == akv.AKV_ERR_INVALID
    akv.akv_decode_set_debug(0, 0)
    assert akv.lib().akv_decode_set_events(ctypes.c_void_p(16), None) == akv.AKV_ERR_INVALID
    assert akv.lib().akv_decode_set_events(None, None) == akv.AKV_OK


def test_select_parameters_validate_and_size_the_pooled_capacity():
    p = akv.Params(batch=2, n_kv_heads=4, n_q_heads=16, anchor_frac=0.02, res_frac_k=0.0, res_frac_v=0.0)
    lens = [4096, 1000]
    for bad in (akv.SelectParams(theta=0.0), akv.SelectParams(theta=1.5), akv.SelectParams(rho=-0.1),
                akv.SelectParams(kappa=4), akv.SelectParams(kappa=0)):
        assert _err(akv.akv_cache_size_select, p, bad, lens) == akv.AKV_ERR_INVALID
    p0 = akv.Params(batch=2, n_kv_heads=4, n_q_heads=16, window=0, anchor_frac=0.02)
    assert _err(akv.akv_cache_size_select, p0, akv.SelectParams(), lens) == akv.AKV_ERR_INVALID
    sel = akv.SelectParams(theta=0.05)
    a_sel, w_sel = akv.akv_cache_size_select(p, sel, lens)
    a_plain, w_plain = akv.akv_cache_size(p, lens)
    assert a_sel > a_plain and w_sel > w_plain  # residual room for the pooled budget; attention scratch
    # each unit may hold up to its request's whole side budget (Eq. 9), capped by its non-anchors
    hdr = akv.akv_cache_header_host(p, lens)  # plain layout: no residuals at fractions 0
    assert int(hdr[256 + 8:256 + 12].view(np.int32)[0]) == 0


def _lloyd_units(p, lens, seed):
    units = []
    for u in helpers_seeded(p, lens, seed):
        u["min_k"] = np.zeros_like(u["min_k"])
        u["min_v"] = np.zeros_like(u["min_v"])
        units.append(u)
    return units


def helpers_seeded(p, lens, seed):
    from helpers import seeded_units
    return seeded_units(p, lens, seed=seed)


def test_table1_layout_has_the_paper_bytes_and_round_trips():
    """Appendix A.1 Table 1: the packed layer has exactly M_base (Eq. 11) + N_K (D/4 + 4) + N_V (D/4 + 5)
    bytes, and an independent reader gets every logical array back (value slot positions = p mod 64)."""
    lens = [3000, 700]
    p = akv.Params(batch=2, n_kv_heads=2, n_q_heads=4, seed=3, lloyd=True)
    units = _lloyd_units(p, lens, 5)
    shapes = akv.akv_unit_shapes(p, lens)
    per_req = akv.akv_table1_bytes(p, lens)
    blob = akv.akv_pack_table1_host(p, lens, [akv.unit_host_from_logical(u) for u in units])
    at = 0
    for b, S in enumerate(lens):
        k = int(shapes[2 * b][1])
        nk = [int(shapes[2 * b + h][2]) for h in range(2)]
        nv = [int(shapes[2 * b + h][3]) for h in range(2)]
        want = acc.paper_m_base(S, 2, 128, p.window, k) + sum(nk) * acc.paper_c_k(128) + sum(nv) * acc.paper_c_v(128)
        assert int(per_req[b]) == want
        heads = acc.read_table1(blob[at:at + want], S, 2, p.window, k, nk, nv)
        at += want
        P = S - p.window
        for h, got in enumerate(heads):
            u = units[2 * b + h]
            assert np.array_equal(got["anchor_k"], u["anchor_k"]) and np.array_equal(got["anchor_v"], u["anchor_v"])
            assert np.array_equal(got["anchor_pos"], u["anchor_pos"][:k - p.window])
            for n in ("idx_k", "gam_k", "idx_v", "gam_v"):
                assert np.array_equal(got[n], u[n][:P])
            for side in ("k", "v"):
                assert np.array_equal(got["res_" + side], u["res_" + side])
                assert np.array_equal(got["codes_" + side], u["codes_" + side])
                assert np.array_equal(got["scale_" + side], u["scale_" + side].view(np.float16).astype(np.float32))
            assert np.array_equal(got["vslot"], u["res_v"] % 64)
            # the window positions the layout leaves out are anchors of their own slot, gamma 1
            assert np.array_equal(u["idx_k"][P:], np.arange(k - p.window, k)) and np.all(u["gam_k"][P:] == 0x3C00)
    assert at == blob.size


def test_table1_layout_of_the_worked_example_layer():
    """The paper's worked example (S = 32K, H = 8, W = 32, k = 256, theta = 0.05: N = 91,056 residual
    slots, 45,528 per side): the packed layer holds M_base (3.39 MB) + the residual bytes, within one
    residual's bytes of theta M_full (6.71 MB)."""
    S, H = 32768, 8
    f = 5691 / 32768  # 45,528 / 8 records per head and side, exactly floor(f S)
    p = akv.Params(batch=1, n_kv_heads=H, n_q_heads=H, anchor_frac=256 / 32768, res_frac_k=f, res_frac_v=f,
                   lloyd=True)
    shapes = akv.akv_unit_shapes(p, [S])
    assert shapes[:, 1].tolist() == [256] * H and shapes[:, 2].sum() == 45528 and shapes[:, 3].sum() == 45528
    n = int(akv.akv_table1_bytes(p, [S])[0])
    m_full = acc.paper_m_full(S, H, 128)
    assert n == acc.paper_m_base(S, H, 128, 32, 256) + 45528 * 36 + 45528 * 37
    assert 0 <= 0.05 * m_full - n < 37
    units = _lloyd_units(p, [S], 7)
    assert akv.akv_pack_table1_host(p, [S], [akv.unit_host_from_logical(u) for u in units]).size == n


def test_table1_layout_needs_the_lloyd_codec():
    p = akv.Params(batch=1, n_kv_heads=1, n_q_heads=1)
    assert _err(akv.akv_table1_bytes, p, [1000]) == akv.AKV_ERR_UNSUPPORTED
