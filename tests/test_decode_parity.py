"""Decode parity: the CUDA path through the C ABI against the fp64 oracle (GPU)."""
import math

import numpy as np
import pytest

import gen
import oracle
import paper_2608_02901_gb300 as akv
from helpers import check_outputs, decode_on_gpu, oracle_decode, oracle_unit, seeded_units, to_dev_u16

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    akv.lib()
    return torch.device("cuda:0")


@pytest.fixture
def debug_controls():
    """The decode testing controls, put back to normal operation after the test."""
    yield
    akv.akv_decode_set_debug(0, 0)


def _run_seeded(dev, p, lens, sm_scale=1.0, seed=5, mutate=None, qseed=17):
    units = seeded_units(p, lens, seed=seed, mutate=mutate)
    arena = akv.akv_cache_pack_host(p, lens, [akv.unit_host_from_logical(u) for u in units])
    arena_dev = torch.from_numpy(arena).to(dev)
    q = gen.queries(p.batch * p.n_q_heads, seed=qseed)
    out, out32 = decode_on_gpu(torch, p, lens, arena_dev, q, sm_scale)
    ref = oracle_decode(p, [oracle_unit(u) for u in units], q, sm_scale)
    return check_outputs(out, out32, ref, where=f"lens={lens} G={p.G}")


@pytest.mark.parametrize("G", [1, 2, 4, 8])
@pytest.mark.parametrize("lens", [[1], [5, 31], [32, 33, 64], [511, 512, 513], [1000, 4173]])
def test_seeded_small_and_ragged(dev, G, lens):
    p = akv.Params(batch=len(lens), n_kv_heads=2, n_q_heads=2 * G, seed=3, rot_seed=77)
    _run_seeded(dev, p, lens)


@pytest.mark.parametrize("fr", [(0.02, 0.0, 0.0), (0.02, 1.0, 1.0), (0.5, 0.3, 0.0), (0.01, 0.2, 0.05)])
@pytest.mark.parametrize("sm_scale", [1.0, 1.0 / math.sqrt(128)])
def test_budgets_and_scales(dev, fr, sm_scale):
    p = akv.Params(batch=2, n_kv_heads=2, n_q_heads=8, anchor_frac=fr[0], res_frac_k=fr[1], res_frac_v=fr[2],
                   seed=9, rot_seed=5)
    _run_seeded(dev, p, [3000, 2047], sm_scale=sm_scale)


def test_rotation_off(dev):
    p = akv.Params(batch=1, n_kv_heads=2, n_q_heads=4, rotate=False, res_frac_k=0.3, res_frac_v=0.3)
    _run_seeded(dev, p, [2500])


def test_negative_and_saturated_gamma_and_zero_anchor(dev):
    def mutate(u, d):
        d["gam_k"] = d["gam_k"].copy()
        d["gam_v"] = d["gam_v"].copy()
        non = np.setdiff1d(np.arange(d["S"]), d["anchor_pos"])
        d["gam_k"][non[::3]] ^= 0x8000  # negative gamma
        d["gam_v"][non[1::5]] ^= 0x8000
        if u == 0:
            d["gam_v"][non[7]] = 0x7BFF  # fp16 maximum on a value coefficient
        d["anchor_k"] = d["anchor_k"].copy()
        d["anchor_k"][1] = 0  # an all-zero anchor key
    p = akv.Params(batch=2, n_kv_heads=1, n_q_heads=4)
    _run_seeded(dev, p, [1500, 900], mutate=mutate)


def test_many_units_cta_counts(dev, debug_controls):
    """The tile blocks of 16 units (ragged) split over 1 .. 37 CTAs: ranges that start and end
    inside units, CTAs that cross several units, units shared by several CTAs."""
    p = akv.Params(batch=4, n_kv_heads=4, n_q_heads=16)
    for c in (1, 2, 3, 8, 16, 37):
        akv.akv_decode_set_debug(ctas=c)
        _run_seeded(dev, p, [8192, 3000, 6001, 700], qseed=c)


@pytest.mark.parametrize("H,G", [(1, 1), (2, 4)])
def test_tiny_encoded_config(dev, H, G):
    """The tiny workload's shape (S = 4096, one KV head, G = 1) and a 2-head G = 4 variant, encoded on
    the GPU: clustered keys and values with real residual structure, where the key-residual
    products need every bit of their fp32 accumulation at sm_scale = 1."""
    S = 4096
    p = akv.Params(batch=1, n_kv_heads=H, n_q_heads=H * G, seed=7, rot_seed=11)
    K, V = gen.clustered_batch(1, H, [S], seed=42)
    a_bytes, w_bytes = akv.akv_cache_size(p, [S])
    arena = torch.empty(a_bytes, dtype=torch.uint8, device=dev)
    ws = torch.empty(w_bytes, dtype=torch.uint8, device=dev)
    akv.akv_encode(p, [S], to_dev_u16(K, torch, dev), to_dev_u16(V, torch, dev), arena, ws)
    units = oracle.unpack_arena(arena.cpu().numpy())
    for qseed in (1, 100, 101, 102, 103):
        for sm in (1.0, 1 / math.sqrt(128)):
            q = gen.queries(H * G, seed=qseed)
            out, out32 = decode_on_gpu(torch, p, [S], arena, q, sm)
            ref = oracle_decode(p, units, q, sm)
            check_outputs(out, out32, ref, f"tiny H={H} G={G} q={qseed} sm={sm:.3f}")


def test_8b_32k_encoded(dev):
    """Llama-3.1-8B layer shape, 32K context, GPU encode, several fresh queries."""
    S, H, Hq = 32768, 8, 32
    p = akv.Params(batch=1, n_kv_heads=H, n_q_heads=Hq, seed=1, rot_seed=2)
    K, V = gen.clustered_batch(1, H, [S], seed=42)
    a_bytes, w_bytes = akv.akv_cache_size(p, [S])
    arena = torch.empty(a_bytes, dtype=torch.uint8, device=dev)
    ws = torch.empty(w_bytes, dtype=torch.uint8, device=dev)
    akv.akv_encode(p, [S], to_dev_u16(K, torch, dev), to_dev_u16(V, torch, dev), arena, ws)
    units = oracle.unpack_arena(arena.cpu().numpy())
    for t in range(3):
        q = gen.queries(Hq, seed=200 + t)
        out, out32 = decode_on_gpu(torch, p, [S], arena, q, 1.0)
        check_outputs(out, out32, oracle_decode(p, units, q, 1.0), "8b-32k")


@pytest.mark.parametrize("shape", [("8b-128k", 4, 8, 32), ("70b-128k", 8, 8, 64)])
def test_128k_seeded(dev, shape):
    name, B, H, Hq = shape
    S = 131072
    p = akv.Params(batch=B, n_kv_heads=H, n_q_heads=Hq, seed=4, rot_seed=8)
    _run_seeded(dev, p, [S] * B, seed=11)


def test_ragged_sweep_points(dev):
    lens = gen.ragged_lens(16, 8192, 131072, seed=3)
    for fa, fr in ((0.01, 0.0), (0.04, 0.2), (0.02, 0.1)):
        p = akv.Params(batch=16, n_kv_heads=8, n_q_heads=32, anchor_frac=fa, res_frac_k=fr, res_frac_v=fr)
        _run_seeded(dev, p, lens, seed=int(fa * 1000 + fr * 100))


def _stored_non_anchor(d):
    """Non-anchor positions in stored order: tokens are stored sorted by value-anchor slot
    (stable, so by position within a slot), and tiles are runs of 1024 stored tokens."""
    order = np.argsort(d["idx_v"], kind="stable")
    is_anchor = np.zeros(d["S"], bool)
    is_anchor[d["anchor_pos"]] = True
    return order[~is_anchor[order]]


def test_locally_dense_residuals_exceed_staging(dev):
    """Key residuals on the first non-anchor tokens in stored order, value residuals on the
    last: the first tile holds about 600 key records and the last about 600 value records, far
    more than the kernel stages per tile (sized from the mean density), so the key records
    whose codes fall beyond the staged bytes and the value records beyond the staged count
    take the CUDA-core paths."""
    def mutate(u, d):
        non = _stored_non_anchor(d)
        d["res_k"] = np.sort(non[: d["nk"]]).astype(np.int32)
        d["res_v"] = np.sort(non[len(non) - d["nv"]:]).astype(np.int32)
    for G in (1, 4, 8):
        p = akv.Params(batch=2, n_kv_heads=2, n_q_heads=2 * G, seed=31)
        _run_seeded(dev, p, [6000, 3000], mutate=mutate)


def test_value_records_a_little_beyond_the_staged_count(dev):
    """Value residuals on every fifth non-anchor token in stored order (about 205 a tile, R = 176
    staged): each tile's few dozen extra records go through the group's overflow list."""
    def mutate(u, d):
        non = _stored_non_anchor(d)
        d["res_v"] = np.sort(non[::5][: d["nv"]]).astype(np.int32)
    for G in (1, 4, 8):
        p = akv.Params(batch=2, n_kv_heads=2, n_q_heads=2 * G, seed=43)
        _run_seeded(dev, p, [6000, 9000], mutate=mutate, qseed=G)


def test_key_records_beyond_the_value_staging_count(dev):
    """Key residuals on every fourth non-anchor token in stored order (about 250 a tile, 2.5x
    the mean): more key records than the value records a tile stages, yet their codes fit the
    tile's staging, so they stay on the tensor-core path; the value residuals sit in the last
    tiles, beyond their staged count."""
    def mutate(u, d):
        non = _stored_non_anchor(d)
        d["res_k"] = np.sort(non[::4][: d["nk"]]).astype(np.int32)
        d["res_v"] = np.sort(non[len(non) - d["nv"]:]).astype(np.int32)
    for G in (4, 8):
        p = akv.Params(batch=2, n_kv_heads=2, n_q_heads=2 * G, seed=37)
        _run_seeded(dev, p, [6000, 9000], mutate=mutate, qseed=G)


def test_tiles_covering_more_value_slots_than_the_weight_table(dev, debug_controls):
    """Every non-anchor token on the last value anchor: stored in value-slot order, the first
    tile then holds one token of each of about a thousand anchors, more value slots than the
    anchor-value rows staged with a tile, so most of its runs take the path that adds their
    anchor-value products on CUDA cores; the tiles (and CTAs) that hold the long last run share
    that slot, each with its own tokens' weights."""
    def mutate(u, d):
        non = np.setdiff1d(np.arange(d["S"]), d["anchor_pos"])
        d["idx_v"] = d["idx_v"].copy()
        d["idx_v"][non] = d["k"] - 1
    for c in (4, 8):
        akv.akv_decode_set_debug(ctas=c)
        for G in (1, 4):
            p = akv.Params(batch=1, n_kv_heads=2, n_q_heads=2 * G, anchor_frac=0.2, seed=41)
            _run_seeded(dev, p, [6000], mutate=mutate, qseed=c + G)


def test_back_to_back_launches_follow_stream_order(dev):
    """Consecutive decode calls in one stream see stream order: a call whose query is the
    previous call's output, and a call that overwrites a buffer an earlier one read."""
    p = akv.Params(batch=2, n_kv_heads=2, n_q_heads=8, seed=3, rot_seed=77)
    lens = [6001, 3000]
    ua = seeded_units(p, lens, seed=5)
    ub = seeded_units(p, lens, seed=6)
    arena_a = torch.from_numpy(akv.akv_cache_pack_host(p, lens, [akv.unit_host_from_logical(u) for u in ua])).to(dev)
    arena_b = torch.from_numpy(akv.akv_cache_pack_host(p, lens, [akv.unit_host_from_logical(u) for u in ub])).to(dev)
    q0 = gen.queries(p.batch * p.n_q_heads, seed=17)
    shape = (p.batch, p.n_q_heads, 128)
    q0_dev = to_dev_u16(q0.reshape(shape), torch, dev)
    x = torch.empty(shape, dtype=torch.bfloat16, device=dev)
    y = torch.empty_like(x)
    z = torch.empty_like(x)
    y32 = torch.empty(shape, dtype=torch.float32, device=dev)
    z32 = torch.empty_like(y32)
    x32 = torch.empty_like(y32)
    akv.akv_decode_attn(p, lens, arena_a, q0_dev, x)            # x = attn(A, q0)
    akv.akv_decode_attn(p, lens, arena_b, x, y, y32)            # reads x as its query
    akv.akv_decode_attn(p, lens, arena_a, y, z, z32)            # reads y as its query
    akv.akv_decode_attn(p, lens, arena_b, q0_dev, x, x32)       # overwrites x after y's launch read it
    torch.cuda.synchronize()
    oa = [oracle_unit(u) for u in ua]
    ob = [oracle_unit(u) for u in ub]
    # z from the y this chain produced (exact input), and the final x from q0
    y_bits = y.view(torch.int16).cpu().numpy().astype(np.uint16).reshape(-1, 128)
    check_outputs(z.float().cpu().numpy(), z32.cpu().numpy(), oracle_decode(p, oa, y_bits, 1.0), where="z = attn(A, y)")
    check_outputs(x.float().cpu().numpy(), x32.cpu().numpy(), oracle_decode(p, ob, q0, 1.0), where="x = attn(B, q0)")
    # y from the bf16 rounding of the oracle's attn(A, q0): a launch that read x before the first
    # one finished would be far off; a last-place difference in x moves y well within 5e-3
    x1 = gen.bf16_bits(oracle_decode(p, oa, q0, 1.0)).reshape(-1, 128)
    y_ref = oracle_decode(p, ob, x1, 1.0)
    assert np.all(np.isfinite(y32.cpu().numpy()))
    assert np.abs(y32.cpu().numpy().astype(np.float64) - y_ref).max() <= 5e-3


@pytest.mark.parametrize("G", [4, 8])
def test_large_anchor_tables(dev, G):
    """80 units with 5243 anchors each: 84 KB of anchor scores per unit at G = 4 (staged in shared
    memory next to the pipeline), 168 KB at G = 8 (beyond it: the token gathers read the
    workspace table).  Checked against the oracle on a sample of units; all outputs finite."""
    p = akv.Params(batch=40, n_kv_heads=2, n_q_heads=2 * G, anchor_frac=0.16, res_frac_k=0.1, res_frac_v=0.1, seed=4,
                   rot_seed=9)
    lens = [32768] * p.batch
    units = seeded_units(p, lens, seed=12)
    arena = torch.from_numpy(akv.akv_cache_pack_host(p, lens, [akv.unit_host_from_logical(u) for u in units])).to(dev)
    q = gen.queries(p.batch * p.n_q_heads, seed=23)
    out, out32 = decode_on_gpu(torch, p, lens, arena, q, 1.0)
    assert np.all(np.isfinite(out32))
    sel = np.zeros(p.n_units, np.uint8)
    sel[[0, 37, 79]] = 1
    ref = oracle_decode(p, [oracle_unit(u) for u in units], q, 1.0, sel=sel)
    rows = np.repeat(sel.astype(bool), p.G).reshape(p.batch, p.n_q_heads)
    check_outputs(out[rows], out32[rows], ref[rows], where=f"large anchor tables G={G}")


def test_withheld_item_times_out_to_nan_and_context_survives(dev, debug_controls):
    """Failure detection without a GPU fault: with the test hook every CTA withholds the last
    tile of its range (here every CTA has one tile), so the waits on it run out after their
    bound (about 2 s).  The call returns, the outputs are NaN, and the next call on the same
    context is correct."""
    import time
    p = akv.Params(batch=1, n_kv_heads=2, n_q_heads=8, seed=3, rot_seed=77)
    lens = [5000]
    units = seeded_units(p, lens, seed=5)
    arena = torch.from_numpy(akv.akv_cache_pack_host(p, lens, [akv.unit_host_from_logical(u) for u in units])).to(dev)
    q = gen.queries(p.batch * p.n_q_heads, seed=17)
    akv.akv_decode_set_debug(withhold_last=1)
    t0 = time.perf_counter()
    out, out32 = decode_on_gpu(torch, p, lens, arena, q, 1.0)
    waited = time.perf_counter() - t0
    akv.akv_decode_set_debug(withhold_last=0)
    assert np.all(np.isnan(out32)) and np.all(np.isnan(out))
    assert waited > 1.0, waited
    out, out32 = decode_on_gpu(torch, p, lens, arena, q, 1.0)
    check_outputs(out, out32, oracle_decode(p, [oracle_unit(u) for u in units], q, 1.0), where="after the timed-out call")


@pytest.mark.parametrize("G", [1, 4, 8])
@pytest.mark.parametrize("fr", [(0.02, 0.1, 0.1), (0.02, 1.0, 1.0)])
def test_lloyd_max_codec_seeded(dev, G, fr):
    """The Lloyd-Max codec's levels on both tensor-core paths (key and value residuals) and, with
    every token a residual, on the CUDA-core paths for records beyond the staged ones."""
    p = akv.Params(batch=2, n_kv_heads=2, n_q_heads=2 * G, anchor_frac=fr[0], res_frac_k=fr[1], res_frac_v=fr[2],
                   seed=12, rot_seed=13, lloyd=True)
    _run_seeded(dev, p, [3000, 1100], qseed=G)


@pytest.mark.parametrize("G", [4, 8])
def test_lloyd_max_codec_encoded(dev, G):
    """GPU encode with the Lloyd-Max codec, then decode, against the oracle reading the arena."""
    S, H = 8192, 2
    p = akv.Params(batch=1, n_kv_heads=H, n_q_heads=H * G, seed=7, rot_seed=11, lloyd=True)
    K, V = gen.clustered_batch(1, H, [S], seed=44)
    a_bytes, w_bytes = akv.akv_cache_size(p, [S])
    arena = torch.empty(a_bytes, dtype=torch.uint8, device=dev)
    ws = torch.empty(w_bytes, dtype=torch.uint8, device=dev)
    akv.akv_encode(p, [S], to_dev_u16(K, torch, dev), to_dev_u16(V, torch, dev), arena, ws)
    units = oracle.unpack_arena(arena.cpu().numpy())
    for qseed in (1, 2):
        q = gen.queries(H * G, seed=qseed)
        out, out32 = decode_on_gpu(torch, p, [S], arena, q, 1.0)
        check_outputs(out, out32, oracle_decode(p, units, q, 1.0), f"lloyd encoded G={G} q={qseed}")


# ---- RoPE at decode (pre-RoPE keys, each token turned to its stored position) ----

@pytest.mark.parametrize("G", [1, 2, 4, 8])
def test_rope_seeded_ragged(dev, G):
    """Seeded caches packed with their positions (the stored order's permutation), ragged lengths
    (one token, partial chunks and tiles), both codecs."""
    for lloyd, base in ((False, 10000.0), (True, 500000.0)):
        p = akv.Params(batch=3, n_kv_heads=2, n_q_heads=2 * G, seed=21, rot_seed=22, rope=True, rope_theta=base,
                       lloyd=lloyd)
        _run_seeded(dev, p, [1, 777, 3000], qseed=G + int(lloyd))


def test_rope_dense_residuals_and_cta_splits(dev, debug_controls):
    """Every token a residual (the CUDA-core token path) and tile ranges split over few CTAs."""
    p = akv.Params(batch=2, n_kv_heads=2, n_q_heads=8, anchor_frac=0.05, res_frac_k=1.0, res_frac_v=1.0, seed=23,
                   rope=True)
    _run_seeded(dev, p, [2500, 1200])
    for c in (1, 3):
        akv.akv_decode_set_debug(ctas=c)
        _run_seeded(dev, p, [2500, 1200], qseed=c)


def test_rope_long_context_positions(dev):
    """128K positions: the angles of the fast pairs reach 1e5 radians; the integer turn keeps the
    sine and cosine accurate at every position."""
    S = 131072
    p = akv.Params(batch=1, n_kv_heads=1, n_q_heads=4, seed=24, rope=True, rope_theta=500000.0)
    _run_seeded(dev, p, [S], seed=9)


def test_rope_encoded(dev):
    """GPU encode of pre-RoPE clustered keys: the arena's positions (read back by the oracle's
    reader) drive the rotation."""
    S, H, G = 8192, 2, 4
    p = akv.Params(batch=1, n_kv_heads=H, n_q_heads=H * G, seed=7, rot_seed=11, rope=True, rope_theta=500000.0)
    K, V = gen.clustered_batch(1, H, [S], seed=45)
    a_bytes, w_bytes = akv.akv_cache_size(p, [S])
    arena = torch.empty(a_bytes, dtype=torch.uint8, device=dev)
    ws = torch.empty(w_bytes, dtype=torch.uint8, device=dev)
    akv.akv_encode(p, [S], to_dev_u16(K, torch, dev), to_dev_u16(V, torch, dev), arena, ws)
    units = oracle.unpack_arena(arena.cpu().numpy())
    want = oracle.encode(K, V, [S], H, p.anchor_frac, p.res_frac_k, p.res_frac_v, p.window, p.seed, p.rot_seed)
    for g, w in zip(units, want):  # the stored tokens' positions: the stable sort of positions by value slot
        assert np.array_equal(g.pos, np.argsort(w.idx_v, kind="stable"))
    for qseed in (1, 2):
        q = gen.queries(H * G, seed=qseed)
        out, out32 = decode_on_gpu(torch, p, [S], arena, q, 1.0)
        check_outputs(out, out32, oracle_decode(p, units, q, 1.0), f"rope encoded q={qseed}")
