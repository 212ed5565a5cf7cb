"""Seeded synthetic inputs shared by the tests, the smoke check and the benchmark.

This module draws random numbers and rounds them to the storage types; it
holds none of AnchorKV's arithmetic (no assignment, projection, ranking,
rotation, quantization or attention).  Everything is numpy PCG64 with
explicit seeds, so the oracle and the CUDA path see identical inputs.

Recipes (the synthetic stand-ins for the paper's Llama-3.1 workloads,
Section 4.1: head_dim 128, 8 KV heads, GQA 4 or 8, 32K-128K context):

clustered_kv  Keys and values of one (request, KV head): 64 centres
              ~ N(0, I_128) per side; each token picks one centre id
              uniformly (shared by K and V); x = (1 + 0.2 n) (c + 0.3 e)
              with n ~ N(0, 1) and e ~ N(0, I); keys scale 4 seed-chosen
              channels by 8 (outlier channels).  Drawn in fp64, rounded to
              bf16 (round-to-nearest-even, direct from fp64).
queries       q ~ N(0, I) / sqrt(128), rounded to bf16.
observation_queries  the observation rows of the full selection (the queries of the last
              W positions of the G query heads of each KV head; Section 3.2): each row
              is 0.25 x one of the unit's keys, picked uniformly, plus N(0, I) noise, so
              that its attention concentrates on that key's cluster, rounded to bf16.
seeded_cache  A compressed cache drawn directly: the last W positions plus a
              uniform sample are anchors, anchor rows from clustered_kv,
              non-anchor indices uniform over the anchors, gamma ~ N(1, 0.1)
              in fp16, residual positions a uniform subset of non-anchors,
              codes uniform in {0..3}, scale ~ U(0.01, 0.1) in fp16 and
              min = fp16(-1.5 scale).
"""
from __future__ import annotations

import numpy as np

D = 128


def _rng(*key) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([int(x) & 0xFFFFFFFF for x in key])))


def bf16_bits(x: np.ndarray) -> np.ndarray:
    """fp64 -> bf16 bit patterns, round to nearest even, direct from fp64.

    Inputs are finite and well inside the bf16 normal range."""
    x = np.asarray(x, dtype=np.float64)
    m, e = np.frexp(x)  # x = m 2^e, |m| in [0.5, 1)
    r = np.rint(m * 256.0)  # 8 significant bits, ties to even
    y = np.ldexp(r, e - 8).astype(np.float32)  # exact: 8-bit significand
    return (y.view(np.uint32) >> 16).astype(np.uint16)


def bf16_to_f64(b: np.ndarray) -> np.ndarray:
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def fp16_bits(x: np.ndarray) -> np.ndarray:
    """fp64 -> fp16 bit patterns (numpy's conversion, round to nearest even)."""
    return np.asarray(x, dtype=np.float64).astype(np.float16).view(np.uint16)


def outlier_channels(seed: int, n: int = 4) -> np.ndarray:
    return np.sort(_rng(seed, 0xC4A7).choice(D, size=n, replace=False))


def clustered_kv(S: int, seed: int, unit: int, n_centres: int = 64, n_outliers: int = 4,
                 outlier_scale: float = 8.0):
    """One unit's keys and values: uint16 bf16 bits, each [S][128]."""
    rng = _rng(seed, unit, 0x4B56)
    ck = rng.standard_normal((n_centres, D))
    cv = rng.standard_normal((n_centres, D))
    cid = rng.integers(0, n_centres, size=S)
    nk = rng.standard_normal(S)
    nv = rng.standard_normal(S)
    ek = rng.standard_normal((S, D))
    ev = rng.standard_normal((S, D))
    K = (1.0 + 0.2 * nk)[:, None] * (ck[cid] + 0.3 * ek)
    V = (1.0 + 0.2 * nv)[:, None] * (cv[cid] + 0.3 * ev)
    K[:, outlier_channels(seed, n_outliers)] *= outlier_scale
    return bf16_bits(K), bf16_bits(V)


def clustered_batch(B: int, H: int, ctx_lens, seed: int, s_max: int | None = None):
    """K, V uint16 [B][H][s_max][128]; rows past S_b are zero."""
    ctx_lens = [int(s) for s in ctx_lens]
    s_max = s_max or max(ctx_lens)
    K = np.zeros((B, H, s_max, D), np.uint16)
    V = np.zeros((B, H, s_max, D), np.uint16)
    for b in range(B):
        for h in range(H):
            k, v = clustered_kv(ctx_lens[b], seed, b * H + h)
            K[b, h, :ctx_lens[b]] = k
            V[b, h, :ctx_lens[b]] = v
    return K, V


def queries(n_rows: int, seed: int, step: int = 0) -> np.ndarray:
    """n_rows query vectors, uint16 bf16 bits [n_rows][128]."""
    rng = _rng(seed, step, 0x5159)
    return bf16_bits(rng.standard_normal((n_rows, D)) / np.sqrt(D))


def observation_queries(K: np.ndarray, ctx_lens, m: int, seed: int) -> np.ndarray:
    """m observation rows per (request, KV head): uint16 bf16 bits [B][H][m][128]; K is the
    uint16 [B][H][s_max][128] of clustered_batch."""
    B, H = K.shape[:2]
    out = np.zeros((B, H, m, D), np.uint16)
    for b in range(B):
        for h in range(H):
            rng = _rng(seed, b * H + h, 0x0B5E)
            t = rng.integers(0, int(ctx_lens[b]), size=m)
            out[b, h] = bf16_bits(0.25 * bf16_to_f64(K[b, h, t]) + rng.standard_normal((m, D)))
    return out


def ragged_lens(B: int, lo: int, hi: int, seed: int) -> np.ndarray:
    """Per-request context lengths uniform in [lo, hi] (integers)."""
    return _rng(seed, 0x4C45).integers(lo, hi + 1, size=B).astype(np.int32)


def seeded_cache(S: int, k: int, nk: int, nv: int, W: int, seed: int, unit: int) -> dict:
    """Logical arrays of one unit's compressed cache, drawn directly (no encode)."""
    rng = _rng(seed, unit, 0x5345)
    w = min(W, S)
    rest = k - w
    head = rng.choice(S - w, size=rest, replace=False) if rest > 0 else np.zeros(0, np.int64)
    anchor_pos = np.sort(np.concatenate([head, np.arange(S - w, S)])).astype(np.int32)
    ak, av = clustered_kv(k, seed ^ 0x5EED, unit)
    slot_of = np.full(S, -1, np.int64)
    slot_of[anchor_pos] = np.arange(k)
    non_anchor = np.flatnonzero(slot_of < 0)

    def side():
        idx = rng.integers(0, k, size=S).astype(np.uint16)
        gam = fp16_bits(rng.normal(1.0, 0.1, size=S))
        idx[anchor_pos] = np.arange(k, dtype=np.uint16)
        gam[anchor_pos] = 0x3C00
        return idx, gam

    def residuals(n):
        pos = np.sort(rng.choice(non_anchor, size=n, replace=False)).astype(np.int32) if n else np.zeros(0, np.int32)
        codes = rng.integers(0, 256, size=(n, 32), dtype=np.uint8)
        sc = fp16_bits(rng.uniform(0.01, 0.1, size=n))
        sc_f = sc.view(np.float16).astype(np.float64)
        mn = fp16_bits(-1.5 * sc_f)
        return pos, codes, sc, mn

    idx_k, gam_k = side()
    idx_v, gam_v = side()
    res_k, codes_k, scale_k, min_k = residuals(nk)
    res_v, codes_v, scale_v, min_v = residuals(nv)
    return dict(S=S, k=k, nk=nk, nv=nv, anchor_k=ak, anchor_v=av, anchor_pos=anchor_pos,
                idx_k=idx_k, gam_k=gam_k, idx_v=idx_v, gam_v=gam_v,
                res_k=res_k, codes_k=codes_k, scale_k=scale_k, min_k=min_k,
                res_v=res_v, codes_v=codes_v, scale_v=scale_v, min_v=min_v)


# ---- device-side variants of the same recipes (benchmark inputs only) --------

def clustered_batch_torch(B: int, H: int, S: int, seed: int, device, n_centres: int = 64, n_outliers: int = 4,
                          outlier_scale: float = 8.0):
    """clustered_kv drawn with torch's generator on the device: bf16 [B][H][S][128] K and V."""
    import torch
    g = torch.Generator(device=device)
    g.manual_seed(int(seed) & 0x7FFFFFFFFFFFFFFF)
    K = torch.empty((B, H, S, D), dtype=torch.bfloat16, device=device)
    V = torch.empty((B, H, S, D), dtype=torch.bfloat16, device=device)
    ch = torch.as_tensor(outlier_channels(seed, n_outliers), device=device)
    for b in range(B):
        for h in range(H):
            ck = torch.randn((n_centres, D), generator=g, device=device)
            cv = torch.randn((n_centres, D), generator=g, device=device)
            cid = torch.randint(0, n_centres, (S,), generator=g, device=device)
            nk = torch.randn((S, 1), generator=g, device=device)
            nv = torch.randn((S, 1), generator=g, device=device)
            k = (1.0 + 0.2 * nk) * (ck[cid] + 0.3 * torch.randn((S, D), generator=g, device=device))
            v = (1.0 + 0.2 * nv) * (cv[cid] + 0.3 * torch.randn((S, D), generator=g, device=device))
            k[:, ch] *= outlier_scale
            K[b, h] = k.to(torch.bfloat16)
            V[b, h] = v.to(torch.bfloat16)
    return K, V


def queries_torch(n_rows: int, seed: int, device):
    """queries drawn with torch's generator on the device: bf16 [n_rows][128]."""
    import torch
    g = torch.Generator(device=device)
    g.manual_seed(int(seed) & 0x7FFFFFFFFFFFFFFF)
    return (torch.randn((n_rows, D), generator=g, device=device) / np.sqrt(D)).to(torch.bfloat16)
