"""akv_encode_noalloc: the encode entry point that allocates nothing (GPU).

Some callers cannot allocate device memory for a scratch workspace -- their
process's memory is owned by an allocator that hands out none, or they must
not call cudaMalloc where they encode.  akv_encode_noalloc serves them with
the library's own static scratch array.  This test calls it through the C
ABI twice in a row and checks that each arena is identical, byte for byte,
to the arena akv_encode writes with a caller-provided workspace (encode is
bit-exact, so the tolerance is zero).  The file sorts last so that a run
stopping at the first failure has run every other test first.
"""
import numpy as np
import pytest

import gen
import paper_2608_02901_gb300 as akv
from helpers import to_dev_u16

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


def test_noalloc_encode_matches_workspace_encode():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    dev = torch.device("cuda:0")
    lens = [4096, 1500]
    p = akv.Params(batch=2, n_kv_heads=2, n_q_heads=8, seed=21, rot_seed=22)
    K, V = gen.clustered_batch(2, 2, lens, seed=23)
    Kt, Vt = to_dev_u16(K, torch, dev), to_dev_u16(V, torch, dev)
    a_bytes, w_bytes = akv.akv_cache_size(p, lens)
    assert w_bytes <= akv.NOALLOC_SCRATCH_BYTES
    want = torch.empty(a_bytes, dtype=torch.uint8, device=dev)
    ws = torch.empty(w_bytes, dtype=torch.uint8, device=dev)
    akv.akv_encode(p, lens, Kt, Vt, want, ws)
    for call in range(2):
        got = torch.full((a_bytes,), 0x5A, dtype=torch.uint8, device=dev)
        akv.akv_encode_noalloc(p, lens, Kt, Vt, got)
        torch.cuda.synchronize()
        assert torch.equal(got, want), f"call {call}: arena differs from akv_encode"


def test_noalloc_rejects_oversized_work():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    p = akv.Params(batch=8, n_kv_heads=8, n_q_heads=32)
    with pytest.raises(akv.AkvError) as e:
        akv.akv_encode_noalloc(p, [131072] * 8, torch.empty((8, 8, 1, 128), dtype=torch.bfloat16, device="cuda"),
                               torch.empty((8, 8, 1, 128), dtype=torch.bfloat16, device="cuda"),
                               torch.empty(256, dtype=torch.uint8, device="cuda"))
    assert e.value.status == akv.AKV_ERR_UNSUPPORTED and "static array" in str(e.value)
