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
