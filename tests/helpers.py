"""Shared helpers of the GPU parity tests (inputs, device copies, tolerances)."""
from __future__ import annotations

import numpy as np

import gen
import oracle
import paper_2608_02901_gb300 as akv

# Parity bar (derived from the arithmetic of the kernel):
#  * fp32 output vs the fp64 oracle: max-abs <= 1e-4 * max(1, |y|).  The kernel
#    accumulates in fp32 over <= 2^17 terms of magnitude <= 1 with hardware exp2;
#    1e-4 is ~100x the expected error and 50x tighter than the 5e-3 target.
#  * bf16 output: exactly the round-to-nearest-even of the kernel's fp32 result,
#    and within one bf16 ulp of the oracle rounded to bf16 the same way.
#  * the target bar (max-abs 5e-3, mean-abs 5e-4) on the bf16 output, widened only
#    where bf16 rounding alone exceeds it: an element may differ by its half-ulp
#    (7.8e-3 for |y| in [2, 4)), and the mean may reach the mean half-ulp.
F32_MAX_ABS = 1e-4
BF16_MAX_ABS = 5e-3
BF16_MEAN_ABS = 5e-4
# (case, bf16 max-abs, bf16 mean-abs, fp32 max-abs, widened bar needed) of every parity check
# this session, printed in pytest's terminal summary (tests/conftest.py)
PARITY_LOG: list = []


def bf16_half_ulp(y: np.ndarray) -> np.ndarray:
    a = np.maximum(np.abs(y), 2.0**-126)
    e = np.floor(np.log2(a))
    return 0.5 * 2.0 ** (e - 7)


def f32_to_bf16_rne(x: np.ndarray) -> np.ndarray:
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    r = ((u + 0x7FFF + ((u >> 16) & 1)) >> 16).astype(np.uint32) << 16
    return r.astype(np.uint32).view(np.float32).astype(np.float64)


def check_outputs(out_bf16: np.ndarray, out_f32: np.ndarray, ref: np.ndarray, where: str = ""):
    assert np.all(np.isfinite(out_f32)), where
    e32 = np.abs(out_f32.astype(np.float64) - ref)
    tol32 = F32_MAX_ABS * np.maximum(1.0, np.abs(ref))
    assert np.all(e32 <= tol32), f"{where}: fp32 max err {e32.max():.3e}"
    assert np.array_equal(out_bf16.astype(np.float64), f32_to_bf16_rne(out_f32)), f"{where}: bf16 != RNE(fp32)"
    # both sides rounded to bf16 the same way differ by at most their fp32 gap plus two half-ulps
    ref16 = gen.bf16_to_f64(gen.bf16_bits(ref))
    gap = np.abs(out_bf16 - ref16)
    assert np.all(gap <= (e32 + bf16_half_ulp(out_f32) + bf16_half_ulp(ref)) * (1 + 1e-9)), f"{where}: bf16 rounding"
    e16 = np.abs(out_bf16.astype(np.float64) - ref)
    hu = bf16_half_ulp(ref)
    assert np.all(e16 <= np.maximum(BF16_MAX_ABS, hu + tol32)), f"{where}: bf16 max err {e16.max():.3e}"
    assert e16.mean() <= max(BF16_MEAN_ABS, hu.mean()), f"{where}: bf16 mean err {e16.mean():.3e}"
    widened = bool(e16.max() > BF16_MAX_ABS or e16.mean() > BF16_MEAN_ABS)
    PARITY_LOG.append((where or "?", float(e16.max()), float(e16.mean()), float(e32.max()), widened))
    return e16.max(), e16.mean(), e32.max()


UNIT_FIELDS = ("anchor_k", "anchor_v", "anchor_pos", "idx_k", "gam_k", "idx_v", "gam_v", "res_k", "codes_k",
               "scale_k", "min_k", "res_v", "codes_v", "scale_v", "min_v")


def stored_order(u) -> dict:
    """A unit's logical arrays (a dict or an oracle.Unit, indexed by position) rearranged
    into the arena's stored order: tokens sorted by value anchor slot, ties by position.
    Residual lists become the sorted stored indices, their records moved along."""
    get = (lambda n: np.asarray(u[n])) if isinstance(u, dict) else (lambda n: np.asarray(getattr(u, n)))
    idx_v = get("idx_v")
    perm = np.argsort(idx_v, kind="stable")
    inv = np.empty_like(perm)
    inv[perm] = np.arange(perm.size)
    out = {n: get(n) for n in ("anchor_k", "anchor_v", "anchor_pos")}
    for n in ("idx_k", "gam_k", "idx_v", "gam_v"):
        out[n] = get(n)[perm]
    for side in ("k", "v"):
        st = inv[get("res_" + side)]
        order = np.argsort(st, kind="stable")
        out["res_" + side] = st[order].astype(np.int32)
        for n in ("codes_", "scale_", "min_"):
            out[n + side] = get(n + side)[order]
    return out


def assert_same_unit(got, want: dict, where: str = ""):
    for f in UNIT_FIELDS:
        a, b = np.asarray(getattr(got, f)), np.asarray(want[f])
        if not np.array_equal(a, b):
            bad = np.flatnonzero((a != b).reshape(a.shape[0], -1).any(axis=1)) if a.ndim and a.shape == b.shape else []
            raise AssertionError(f"{where} field {f}: shapes {a.shape}/{b.shape}, {len(bad)} mismatching rows, "
                                 f"first {bad[:5]}")


def to_dev_u16(a: np.ndarray, torch, dev, dtype=None):
    t = torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).to(dev)
    return t.view(dtype or torch.bfloat16)


def seeded_units(p: akv.Params, lens, seed=5, mutate=None):
    shapes = akv.akv_unit_shapes(p, lens)
    units = []
    for u, (S, k, nk, nv) in enumerate(shapes):
        d = gen.seeded_cache(int(S), int(k), int(nk), int(nv), p.window, seed, u)
        if mutate:
            mutate(u, d)
        units.append(d)
    return units


def oracle_unit(d: dict) -> oracle.Unit:
    u = oracle.alloc_unit(d["S"], d["k"], d["nk"], d["nv"])
    for name in ("anchor_k", "anchor_v", "anchor_pos", "idx_k", "gam_k", "idx_v", "gam_v", "res_k", "codes_k",
                 "scale_k", "min_k", "res_v", "codes_v", "scale_v", "min_v"):
        getattr(u, name)[...] = d[name]
    return u


def decode_on_gpu(torch, p: akv.Params, lens, arena_dev, q: np.ndarray, sm_scale: float):
    dev = arena_dev.device
    B, Hq = p.batch, p.n_q_heads
    qt = to_dev_u16(q.reshape(B, Hq, 128), torch, dev)
    out = torch.empty((B, Hq, 128), dtype=torch.bfloat16, device=dev)
    out32 = torch.empty((B, Hq, 128), dtype=torch.float32, device=dev)
    akv.akv_decode_attn(p, lens, arena_dev, qt, out, out32, sm_scale=sm_scale)
    torch.cuda.synchronize()
    return out.float().cpu().numpy(), out32.cpu().numpy()


def oracle_decode(p: akv.Params, units, q: np.ndarray, sm_scale: float, sel=None):
    G = p.G
    ref = oracle.attend(units, q.reshape(p.n_units, G, 128), G, sm_scale, p.rot_seed, p.rotate, lloyd=p.lloyd, sel=sel,
                        rope_theta=p.rope_theta if p.rope else 0.0)
    return ref.reshape(p.batch, p.n_q_heads, 128)
