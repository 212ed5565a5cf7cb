"""The paper's full selection on the GPU (akv_encode_select) against the fp64 oracle (GPU).

Encode: every byte of the packed cache -- the scored and sampled anchors, indices,
coefficients, each head's pooled residual slots, codes, scales -- equals the oracle's
(oracle.encode_select), after the oracle's independent reader unpacks the GPU arena.
Decode: akv_decode_attn over the select-encoded cache against the oracle's attention over
the same cache, at the decode parity bar."""
import numpy as np
import pytest

import gen
import oracle
import paper_2608_02901_gb300 as akv
from helpers import (assert_same_unit, check_outputs, decode_on_gpu, oracle_decode, stored_order, to_dev_u16)

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    akv.lib()
    return torch.device("cuda:0")


def _case(dev, lens, H, G, sel, anchor_frac=0.02, W=32, rotate=True, seed=3, check_decode=True, extra=None):
    B = len(lens)
    extra = extra or {}  # further Params flags (codec, RoPE at decode)
    p = akv.Params(batch=B, n_kv_heads=H, n_q_heads=H * G, anchor_frac=anchor_frac, res_frac_k=0.0,
                   res_frac_v=0.0, window=W, seed=seed, rot_seed=seed + 1, rotate=rotate, **extra)
    K, V = gen.clustered_batch(B, H, lens, seed=seed)
    Q = gen.observation_queries(K, lens, W * G, seed=seed + 2)
    a_bytes, w_bytes = akv.akv_cache_size_select(p, sel, lens)
    arena = torch.empty(a_bytes, dtype=torch.uint8, device=dev)
    ws = torch.full((w_bytes,), 0xAB, dtype=torch.uint8, device=dev)  # scratch contents must not matter
    akv.akv_encode_select(p, sel, lens, to_dev_u16(K, torch, dev), to_dev_u16(V, torch, dev),
                          to_dev_u16(Q, torch, dev), arena, ws)
    torch.cuda.synchronize()
    got = oracle.unpack_arena(arena.cpu().numpy())
    want = oracle.encode_select(K, V, Q, lens, H, anchor_frac, W, sel.theta, sel.rho, sel.kappa, p.seed, p.rot_seed,
                                rotate, lloyd=p.lloyd)
    assert len(got) == len(want)
    for u, (g, w) in enumerate(zip(got, want)):
        assert (g.S, g.k, g.nk, g.nv) == (w.S, w.k, w.nk, w.nv), u
        assert_same_unit(g, stored_order(w), f"unit {u}")
    # the pooled budget is spent in full (up to the candidates), and heads differ
    for b, S in enumerate(lens):
        k = want[b * H].k
        N = oracle.budget_n(np.float32(sel.theta).item(), S, H, W, k)
        nk = sum(w.nk for w in want[b * H:(b + 1) * H])
        nv = sum(w.nv for w in want[b * H:(b + 1) * H])
        assert nk == min(N // 2, H * (S - k)) and nv == min(N - N // 2, H * (S - k))
    if check_decode:
        q = gen.queries(B * H * G, seed=seed + 5)
        # the decode planner stages records per tile from the fractions it is given: once with
        # the chosen densities, once with 0 (every record then read from global memory)
        dk = min(0.999, sum(w.nk for w in want) / sum(w.S for w in want))
        dv = min(0.999, sum(w.nv for w in want) / sum(w.S for w in want))
        p_dens = akv.Params(batch=B, n_kv_heads=H, n_q_heads=H * G, anchor_frac=anchor_frac, res_frac_k=dk,
                            res_frac_v=dv, window=W, seed=seed, rot_seed=seed + 1, rotate=rotate, **extra)
        for pd, sm in ((p_dens, 1.0), (p, 1.0 / np.sqrt(128.0))):
            out, out32 = decode_on_gpu(torch, pd, lens, arena, q, sm)
            check_outputs(out, out32, oracle_decode(pd, got, q, sm), where=f"select lens={lens} G={G} sm={sm:.3f}")
    return want


def test_select_tiny_config(dev):
    """The tiny workload's shape (S = 4096, one KV head, G = 1) with the paper's defaults."""
    _case(dev, [4096], 1, 1, akv.SelectParams(theta=0.05, rho=0.7, kappa=7))


def test_select_pooled_over_heads_ragged(dev):
    want = _case(dev, [4096, 2500], 4, 4, akv.SelectParams(theta=0.08, rho=0.7, kappa=7))
    counts = [w.nk for w in want[:4]]
    assert len(set(counts)) > 1, counts  # the pooled budget is shared unevenly


@pytest.mark.parametrize("G", [2, 8])
def test_select_group_sizes(dev, G):
    _case(dev, [3000], 2, G, akv.SelectParams(theta=0.1, rho=0.7, kappa=7), seed=G)


@pytest.mark.parametrize("rho,kappa", [(0.0, 7), (1.0, 1), (0.5, 3)])
def test_select_anchor_shares_and_pooling_widths(dev, rho, kappa):
    _case(dev, [2047, 1100], 2, 4, akv.SelectParams(theta=0.06, rho=rho, kappa=kappa), anchor_frac=0.05)


def test_select_edge_lengths_and_no_rotation(dev):
    _case(dev, [33, 64, 513], 2, 2, akv.SelectParams(theta=0.3, rho=0.7, kappa=5), W=16, rotate=False)


def test_select_budget_beyond_every_candidate(dev):
    """theta = 1: more residual budget than non-anchor positions -- every one gets both."""
    want = _case(dev, [700], 2, 2, akv.SelectParams(theta=1.0, rho=0.7, kappa=7), anchor_frac=0.1)
    for w in want:
        assert w.nk == w.nv == w.S - w.k


def test_select_8b_32k_shape(dev):
    """One request at the 8B layer shape (32 query / 8 KV heads, 32K context), theta = 0.05:
    the pooled budget over eight heads at full context (encode bytes only; the decode of such
    caches is covered by the smaller cases)."""
    _case(dev, [32768], 8, 4, akv.SelectParams(theta=0.05, rho=0.7, kappa=7), check_decode=False)


def test_select_with_rope_positions_and_the_lloyd_max_codec(dev):
    """The full selection writing a RoPE arena (the stored tokens' positions) with the Lloyd-Max
    codec: bit-exact encode, then the RoPE decode against the oracle over the read-back units."""
    _case(dev, [3000, 1500], 2, 4, akv.SelectParams(theta=0.06, rho=0.7, kappa=7), seed=11,
          extra=dict(rope=True, lloyd=True))
