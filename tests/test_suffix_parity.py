"""Exact dense suffix (generated tokens kept in bf16, Appendix E.1 and E.2): the decode over the
compressed prefix and the suffix in one softmax, and the append path, through the C ABI against the
fp64 oracle (GPU)."""
import math

import numpy as np
import pytest

import gen
import oracle
import paper_2608_02901_gb300 as akv
from helpers import check_outputs, oracle_unit, seeded_units, to_dev_u16

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    akv.lib()
    return torch.device("cuda:0")


def _suffix_rows(n_units, cap, seed, key_scale=1.0):
    """bf16 bits [n_units][cap][128] of clustered rows for the suffix keys and values."""
    K, V = gen.clustered_batch(1, n_units, [cap], seed=seed)
    K, V = K[0], V[0]
    if key_scale != 1.0:
        K = gen.bf16_bits(gen.bf16_to_f64(K) * key_scale)
    return np.ascontiguousarray(K), np.ascontiguousarray(V)


def _run(dev, p, lens, suf_lens, cap, sm_scale=1.0, seed=5, qseed=17, key_scale=1.0, where=""):
    units = seeded_units(p, lens, seed=seed)
    arena = torch.from_numpy(akv.akv_cache_pack_host(p, lens, [akv.unit_host_from_logical(u) for u in units])).to(dev)
    ks, vs = _suffix_rows(p.n_units, cap, seed + 1000, key_scale)
    H = p.n_kv_heads
    sfx = akv.Suffix(to_dev_u16(ks.reshape(p.batch, H, cap, 128), torch, dev),
                     to_dev_u16(vs.reshape(p.batch, H, cap, 128), torch, dev),
                     torch.tensor(suf_lens, dtype=torch.int32, device=dev))
    q = gen.queries(p.batch * p.n_q_heads, seed=qseed)
    qt = to_dev_u16(q.reshape(p.batch, p.n_q_heads, 128), torch, dev)
    out = torch.empty((p.batch, p.n_q_heads, 128), dtype=torch.bfloat16, device=dev)
    out32 = torch.empty((p.batch, p.n_q_heads, 128), dtype=torch.float32, device=dev)
    akv.akv_decode_attn(p, lens, arena, qt, out, out32, sm_scale=sm_scale, suffix=sfx)
    torch.cuda.synchronize()
    ref = oracle.attend_suffix([oracle_unit(u) for u in units], q.reshape(p.n_units, p.G, 128), p.G, H, sm_scale,
                               p.rot_seed, ks, vs, suf_lens, p.rotate, lloyd=p.lloyd,
                               rope_theta=p.rope_theta if p.rope else 0.0).reshape(p.batch, p.n_q_heads, 128)
    return check_outputs(out.float().cpu().numpy(), out32.cpu().numpy(), ref, where=where)


@pytest.mark.parametrize("G", [1, 2, 4, 8])
def test_suffix_decode_ragged_lengths(dev, G):
    """Ragged prefixes and suffixes (0, 1, one chunk, one chunk and one, several chunks)."""
    p = akv.Params(batch=5, n_kv_heads=2, n_q_heads=2 * G, seed=3, rot_seed=77)
    _run(dev, p, [3000, 700, 5000, 1, 2048], [0, 1, 64, 65, 200], 200, where=f"suffix G={G}")


@pytest.mark.parametrize("sm_scale", [1.0, 1.0 / math.sqrt(128)])
def test_suffix_decode_scales_and_full_capacity(dev, sm_scale):
    p = akv.Params(batch=2, n_kv_heads=2, n_q_heads=8, seed=9, rot_seed=5)
    _run(dev, p, [4096, 1500], [128, 127], 128, sm_scale=sm_scale, where=f"suffix sm={sm_scale:.3f}")


def test_suffix_with_the_lloyd_max_codec(dev):
    p = akv.Params(batch=3, n_kv_heads=2, n_q_heads=16, seed=19, lloyd=True)
    _run(dev, p, [2000, 4500, 700], [17, 64, 130], 160, where="suffix lloyd")


@pytest.mark.parametrize("G", [1, 4, 8])
def test_suffix_with_rope_at_decode(dev, G):
    """Pre-RoPE suffix keys turned to positions S_b + t (after the request's compressed tokens),
    in the same softmax as the RoPE-decoded prefix; ragged lengths, several chunks."""
    p = akv.Params(batch=3, n_kv_heads=2, n_q_heads=2 * G, seed=23, rope=True, rope_theta=10000.0)
    _run(dev, p, [2500, 700, 5000], [0, 65, 150], 150, where=f"suffix rope G={G}")


def test_suffix_logits_far_above_the_anchor_reference(dev):
    """Suffix keys scaled up so their logits exceed every anchor score by far: the compressed part
    is rescaled to the suffix's maximum in the combine (and carries almost no weight)."""
    p = akv.Params(batch=2, n_kv_heads=2, n_q_heads=8, seed=11)
    _run(dev, p, [3000, 3000], [40, 3], 64, key_scale=6.0, where="suffix dominant")


def test_suffix_lengths_above_capacity_are_taken_as_capacity(dev):
    """Lengths past the capacity read as the capacity.  The decode launch's shared-memory float
    reductions make its fp32 output depend on the order warps arrive in, at the last bit: the two
    calls agree to 1e-6 (a length taken past 70 rows would move the output by far more)."""
    p = akv.Params(batch=2, n_kv_heads=1, n_q_heads=4, seed=13)
    lens = [2000, 900]
    units = seeded_units(p, lens, seed=5)
    arena = torch.from_numpy(akv.akv_cache_pack_host(p, lens, [akv.unit_host_from_logical(u) for u in units])).to(dev)
    ks, vs = _suffix_rows(p.n_units, 70, 21)
    kt = to_dev_u16(ks.reshape(2, 1, 70, 128), torch, dev)
    vt = to_dev_u16(vs.reshape(2, 1, 70, 128), torch, dev)
    q = gen.queries(8, seed=4)
    qt = to_dev_u16(q.reshape(2, 4, 128), torch, dev)
    outs = []
    for ln in ([70, 70], [500, 1 << 30]):
        out = torch.empty((2, 4, 128), dtype=torch.float32, device=dev)
        o16 = torch.empty((2, 4, 128), dtype=torch.bfloat16, device=dev)
        akv.akv_decode_attn(p, lens, arena, qt, o16, out,
                            suffix=akv.Suffix(kt, vt, torch.tensor(ln, dtype=torch.int32, device=dev)))
        outs.append(out.cpu().numpy())
    assert np.allclose(outs[0], outs[1], rtol=1e-6, atol=1e-7)


def test_suffix_append_writes_rows_and_counts_them(dev):
    """Appends write row len[b] of each (request, KV head) and count it in; a full suffix is left as
    it is (bit-exact copies)."""
    p = akv.Params(batch=3, n_kv_heads=2, n_q_heads=4)
    cap = 5
    K = torch.zeros((3, 2, cap, 128), dtype=torch.bfloat16, device=dev)
    V = torch.zeros_like(K)
    lens = torch.tensor([0, 3, 5], dtype=torch.int32, device=dev)
    sfx = akv.Suffix(K, V, lens)
    expect_k = np.zeros((3, 2, cap, 128), np.uint16)
    expect_v = np.zeros_like(expect_k)
    n = [0, 3, 5]
    for step in range(4):
        kn, vn = _suffix_rows(6, 1, 300 + step)
        kn, vn = kn.reshape(3, 2, 128), vn.reshape(3, 2, 128)
        akv.akv_suffix_append(p, to_dev_u16(kn, torch, dev), to_dev_u16(vn, torch, dev), sfx)
        for b in range(3):
            if n[b] < cap:
                expect_k[b, :, n[b]] = kn[b]
                expect_v[b, :, n[b]] = vn[b]
                n[b] += 1
    torch.cuda.synchronize()
    assert lens.cpu().tolist() == n == [4, 5, 5]
    assert np.array_equal(K.view(torch.int16).cpu().numpy().view(np.uint16), expect_k)
    assert np.array_equal(V.view(torch.int16).cpu().numpy().view(np.uint16), expect_v)


def test_append_then_decode_replayed_from_one_graph(dev):
    """A serving step (append the new token, decode over prefix and suffix) captured once as a
    CUDA graph and replayed: each replay sees the lengths the previous one left on the device."""
    p = akv.Params(batch=2, n_kv_heads=2, n_q_heads=8, seed=17)
    lens = [2500, 4000]
    cap = 80
    units = seeded_units(p, lens, seed=6)
    arena = torch.from_numpy(akv.akv_cache_pack_host(p, lens, [akv.unit_host_from_logical(u) for u in units])).to(dev)
    K = torch.zeros((2, 2, cap, 128), dtype=torch.bfloat16, device=dev)
    V = torch.zeros_like(K)
    sl = torch.tensor([62, 0], dtype=torch.int32, device=dev)
    sfx = akv.Suffix(K, V, sl)
    ks, vs = _suffix_rows(4, cap, 33)
    K.view(torch.int16).copy_(torch.from_numpy(ks.reshape(2, 2, cap, 128).view(np.int16)))
    V.view(torch.int16).copy_(torch.from_numpy(vs.reshape(2, 2, cap, 128).view(np.int16)))
    kn = torch.empty((2, 2, 128), dtype=torch.bfloat16, device=dev)
    vn = torch.empty_like(kn)
    q = gen.queries(16, seed=8)
    qt = to_dev_u16(q.reshape(2, 8, 128), torch, dev)
    out = torch.empty((2, 8, 128), dtype=torch.bfloat16, device=dev)
    out32 = torch.empty((2, 8, 128), dtype=torch.float32, device=dev)
    ws = torch.empty(akv.akv_decode_workspace_size(p, lens, cap), dtype=torch.uint8, device=dev)
    akv.akv_decode_attn(p, lens, arena, qt, out, out32, ws=ws, suffix=sfx)  # sets kernel attributes
    torch.cuda.synchronize()
    sl.copy_(torch.tensor([62, 0], dtype=torch.int32))
    stream = torch.cuda.Stream(device=dev)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        s = torch.cuda.current_stream()
        akv.akv_suffix_append(p, kn, vn, sfx, stream=s)
        akv.akv_decode_attn(p, lens, arena, qt, out, out32, ws=ws, stream=s, suffix=sfx)
    n = [62, 0]
    ounits = [oracle_unit(u) for u in units]
    for step in range(3):
        # the new token's rows are the ones already in place at row len[b] (so the oracle's rows hold)
        for b in range(2):
            kn[b].view(torch.int16).copy_(torch.from_numpy(ks.reshape(2, 2, cap, 128)[b, :, n[b]].view(np.int16)))
            vn[b].view(torch.int16).copy_(torch.from_numpy(vs.reshape(2, 2, cap, 128)[b, :, n[b]].view(np.int16)))
        with torch.cuda.stream(stream):
            g.replay()
        stream.synchronize()
        n = [x + 1 for x in n]
        assert sl.cpu().tolist() == n
        ref = oracle.attend_suffix(ounits, q.reshape(4, 4, 128), 4, 2, 1.0, p.rot_seed, ks, vs, n, p.rotate)
        check_outputs(out.float().cpu().numpy(), out32.cpu().numpy(), ref.reshape(2, 8, 128), f"graph step {step}")
