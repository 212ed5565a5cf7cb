"""Encode parity: the GPU encoder's packed cache, bit for bit, against the fp64 oracle (GPU)."""
import pytest

import gen
import oracle
import paper_2608_02901_gb300 as akv
from helpers import assert_same_unit, stored_order, to_dev_u16

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

@pytest.fixture(scope="module")
def dev():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    akv.lib()
    return torch.device("cuda:0")


def _encode_both(dev, p, lens, K, V):
    a_bytes, w_bytes = akv.akv_cache_size(p, lens)
    arena = torch.empty(a_bytes, dtype=torch.uint8, device=dev)
    ws = torch.full((w_bytes,), 0xAB, dtype=torch.uint8, device=dev)  # scratch contents must not matter
    akv.akv_encode(p, lens, to_dev_u16(K, torch, dev), to_dev_u16(V, torch, dev), arena, ws)
    torch.cuda.synchronize()
    got = oracle.unpack_arena(arena.cpu().numpy())
    want = oracle.encode(K, V, lens, p.n_kv_heads, p.anchor_frac, p.res_frac_k, p.res_frac_v, p.window, p.seed,
                         p.rot_seed, p.rotate, lloyd=p.lloyd)
    assert len(got) == len(want)
    for u, (g, w) in enumerate(zip(got, want)):
        assert (g.S, g.k, g.nk, g.nv) == (w.S, w.k, w.nk, w.nv)
        # the arena keeps tokens sorted by value anchor slot: compare in that order
        assert_same_unit(g, stored_order(w), f"unit {u}")
    return got


def test_tiny_bit_exact(dev):
    S = 4096
    p = akv.Params(batch=1, n_kv_heads=1, n_q_heads=1, seed=7, rot_seed=11)
    K, V = gen.clustered_batch(1, 1, [S], seed=42)
    _encode_both(dev, p, [S], K, V)


def test_8b_32k_bit_exact(dev):
    S = 32768
    p = akv.Params(batch=1, n_kv_heads=8, n_q_heads=32, seed=1, rot_seed=2)
    K, V = gen.clustered_batch(1, 8, [S], seed=42)
    _encode_both(dev, p, [S], K, V)


@pytest.mark.parametrize("lens", [[1, 20], [33, 64, 65], [127, 1000, 2049]])
@pytest.mark.parametrize("rotate", [True, False])
def test_edge_lengths(dev, lens, rotate):
    p = akv.Params(batch=len(lens), n_kv_heads=2, n_q_heads=4, res_frac_k=0.5, res_frac_v=1.0, seed=3, rot_seed=4,
                   rotate=rotate)
    K, V = gen.clustered_batch(len(lens), 2, lens, seed=sum(lens))
    _encode_both(dev, p, lens, K, V)


def test_zero_rows_duplicates_and_ties(dev):
    lens = [600]
    p = akv.Params(batch=1, n_kv_heads=1, n_q_heads=1, res_frac_k=0.2, res_frac_v=0.2, seed=5, rot_seed=6)
    K, V = gen.clustered_batch(1, 1, lens, seed=8)
    K, V = K.copy(), V.copy()
    K[0, 0, 10:20] = 0  # zero keys
    V[0, 0, 30] = 0
    K[0, 0, 100:140] = K[0, 0, 50]  # duplicated rows: equal cosines and equal residual energies
    V[0, 0, 200:260] = V[0, 0, 599]  # copies of a window anchor
    _encode_both(dev, p, lens, K, V)


def test_all_anchor_rows_zero(dev):
    lens = [64]
    p = akv.Params(batch=1, n_kv_heads=1, n_q_heads=1, window=32, anchor_frac=0.0, res_frac_k=0.5, res_frac_v=0.5)
    K, V = gen.clustered_batch(1, 1, lens, seed=9)
    K, V = K.copy(), V.copy()
    K[0, 0, 32:] = 0  # every anchor key is zero: no usable direction on the key side
    _encode_both(dev, p, lens, K, V)


@pytest.mark.parametrize("rotate", [True, False])
def test_lloyd_max_codec_bit_exact(dev, rotate):
    """The Lloyd-Max codec (per-token RMS scale, min 0, decision-region codes), every residual
    stored (res_frac 1), on clustered rows and ragged lengths."""
    lens = [1, 700, 3000]
    p = akv.Params(batch=3, n_kv_heads=2, n_q_heads=4, res_frac_k=1.0, res_frac_v=0.6, seed=5, rot_seed=9,
                   rotate=rotate, lloyd=True)
    K, V = gen.clustered_batch(3, 2, lens, seed=123)
    got = _encode_both(dev, p, lens, K, V)
    assert any(u.nk and not u.min_k.any() and u.scale_k.any() for u in got)  # min 0, scales stored


def test_lloyd_max_codec_8b_32k_bit_exact(dev):
    S = 32768
    p = akv.Params(batch=1, n_kv_heads=8, n_q_heads=32, seed=1, rot_seed=2, lloyd=True)
    K, V = gen.clustered_batch(1, 8, [S], seed=42)
    _encode_both(dev, p, [S], K, V)
