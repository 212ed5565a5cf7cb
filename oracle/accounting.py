"""Byte accounting of AnchorKV, written out from the paper (test infrastructure only).

paper_* functions follow Appendix A.1 "Layout" (Eq. 11 and Table 1) and
Section 3.4 (Eq. 9).  format_unit_bytes is the data-byte count of this
build's packed format (the sections a decode step reads for one unit).
"""
from __future__ import annotations

import math


def paper_m_full(S: int, H: int, D: int) -> int:
    """Uncompressed bf16 K and V of one layer: 4 S H D bytes (Appendix A.1 worked example)."""
    return 4 * S * H * D


def paper_m_base(S: int, H: int, D: int, W: int, k: int, b_a: int = 2, b_gamma: int = 2) -> int:
    """Eq. 11: anchors, anchor positions, per-side index and coefficient over
    the P = S - W non-window positions, residual mask and prefix words,
    head offsets and shared position ids."""
    P = S - W
    words = math.ceil(P / 64)
    return H * (4 * k * D + 8 * (k - W) + 2 * P * (b_a + b_gamma)) + 24 * H * words + 8 * (H + 1) + 4 * P


def paper_c_k(D: int) -> int:
    """Bytes of one key residual: D/4 code bytes + an fp32 scale (Table 1)."""
    return D // 4 + 4


def paper_c_v(D: int) -> int:
    """Bytes of one value residual: adds a one-byte chunk-local position (Table 1)."""
    return D // 4 + 5


def paper_n_residuals(theta: float, m_full: int, m_base: int, b_res: float) -> int:
    """Eq. 9: N = max(0, floor((theta M_full - M_base) / b_res))."""
    return max(0, math.floor((theta * m_full - m_base) / b_res))


def paper_split(N: int):
    """Keys receive floor(N/2) slots and values the rest (Section 3.4)."""
    return N // 2, N - N // 2


def format_unit_bytes(S: int, k: int, nk: int, nv: int, D: int = 128) -> int:
    """Data bytes of one unit in this build's layout: two bf16 anchor tiles,
    int32 anchor positions, two u32 (index, fp16 gamma) streams, two u64
    bitmaps with u32 prefix words, and 32-byte code records with a 4-byte
    (scale, min) pair per residual slot."""
    words = math.ceil(S / 64)
    return 2 * k * D * 2 + 4 * k + 2 * 4 * S + 2 * 12 * words + (nk + nv) * (D // 4 + 4)


def decode_read_bytes(S: int, k: int, nk: int, nv: int, G: int, D: int = 128) -> int:
    """Bytes one decode step reads and writes for one unit: everything of
    format_unit_bytes except the anchor positions, plus G bf16 query rows in
    and G bf16 output rows out."""
    return format_unit_bytes(S, k, nk, nv, D) - 4 * k + 2 * G * D * 2


def read_table1(buf, S: int, H: int, W: int, k: int, nk, nv, D: int = 128) -> list:
    """Independent reader of one request's layer in the paper's Table 1 layout (Appendix A.1):
    returns per KV head a dict of the logical arrays (positions 0 .. P-1 for the per-position ones,
    P = S - W), checking the prefix counts and head offsets against the masks."""
    import numpy as np
    b = np.frombuffer(bytes(buf), np.uint8)
    P, nw = S - W, -(-(S - W) // 64)
    at = 0

    def take(n, dt, shape):
        nonlocal at
        a = b[at:at + n * np.dtype(dt).itemsize].view(dt).reshape(shape)
        at += n * np.dtype(dt).itemsize
        return a
    ak = take(H * k * D, np.uint16, (H, k, D))
    av = take(H * k * D, np.uint16, (H, k, D))
    apos = take(H * (k - W), np.int64, (H, k - W))
    idx = take(2 * H * P, np.uint16, (2, H, P))
    gam = take(2 * H * P, np.uint16, (2, H, P))
    mask = take(2 * H * nw, np.uint64, (2, H, nw))
    pref = take(2 * H * nw, np.int32, (2, H, nw))
    hoff = take(2 * (H + 1), np.int32, (2, H + 1))
    ids = take(P, np.int32, (P,))
    NK, NV = int(sum(nk)), int(sum(nv))
    codes = take((NK + NV) * (D // 4), np.uint8, (NK + NV, D // 4))
    scales = take(NK + NV, np.float32, (NK + NV,))
    vslot = take(NV, np.uint8, (NV,))
    assert at == b.size, "trailing or missing bytes"
    assert np.array_equal(ids, np.arange(P))
    out = []
    for h in range(H):
        u = dict(anchor_k=ak[h], anchor_v=av[h], anchor_pos=apos[h], idx_k=idx[0, h], gam_k=gam[0, h],
                 idx_v=idx[1, h], gam_v=gam[1, h])
        for side, name in ((0, "k"), (1, "v")):
            bits = [(int(mask[side, h, w]) >> j) & 1 for w in range(nw) for j in range(64)]
            pos = np.flatnonzero(np.array(bits[:P], bool)).astype(np.int32)
            cnt = np.array([bin(int(m)).count("1") for m in mask[side, h]])
            assert np.array_equal(pref[side, h], np.concatenate([[0], np.cumsum(cnt)[:-1]])), "prefix counts"
            assert hoff[side, h + 1] - hoff[side, h] == pos.size, "head offsets"
            first = (0 if side == 0 else NK) + int(hoff[side, h])
            u["res_" + name] = pos
            u["codes_" + name] = codes[first:first + pos.size]
            u["scale_" + name] = scales[first:first + pos.size]
            if side == 1:
                u["vslot"] = vslot[int(hoff[1, h]):int(hoff[1, h]) + pos.size]
        out.append(u)
    return out
