// Decode attention read directly from the AnchorKV compressed cache (Eq. 3 folded into
// Eq. 4: no key or value row is ever rebuilt in memory).  Two launches per call:
//
// 1. akv_scores_kernel.  The anchor scores S_A[a][g] = q_g . k_a of every anchor of every
//    unit, once per anchor (Eq. 2-3), bf16 tensor cores, in log2 units with sm_scale
//    folded in, into the workspace; with the largest score per query head of each chunk of
//    64 anchors.  It streams the anchor keys, a fifth of the compressed bytes, at full width.
//
// 2. akv_decode_kernel.  Persistent: one CTA per SM.  The tile blocks of all units, in unit
//    order, are split into equal contiguous ranges, one per CTA (stream-K): a unit's tiles may
//    lie in several CTAs and a CTA's range may cross units (its segments).  Per CTA:
//      producer warp   one lane streams each tile block, followed by the anchor-value rows of
//                      the value slots the tile covers (the tile table records the range),
//                      into a byte ring of shared memory with one bulk asynchronous copy
//                      each, completing a transaction-counted mbarrier; per segment it also
//                      copies the unit's anchor-score table and flushes the CTA's overflow sums;
//      2 groups of 4 warps  each group takes every other tile of the range, end to end:
//        key residuals  q' . c of the staged key records on tensor cores (q' = H(s o q)/128,
//                       Appendix A.1 Eq. 12), written over the records' codes;
//        tokens         each lane 8 consecutive stored tokens, every head: logits
//                       gamma_i S_A[a(i)] + residual term, p = 2^(l - m), the normaliser,
//                       p rows of the value records, and the value weights
//                       w[a] = sum_i p_i gamma_i (Eq. 3): tokens are stored sorted by value
//                       anchor, so a lane sums a run in registers and adds it into the
//                       tile's weight table when the anchor changes;
//        value side     the value-residual sum (p scale) c over the records and the
//                       anchor-value product w^T V_A over the tile's slots, both on tensor
//                       cores (weights and p scale as bf16 high + low parts, codes exact),
//                       accumulated in registers across the segment's tiles.
//    At the end of a segment every group (and the producer, for the overflow sums) stores its
//    partial numerator and normaliser into its own workspace slot and counts itself in on the
//    unit's counter; the one that completes the count sums the unit's slots in a fixed order,
//    applies the inverse rotation once (Appendix E.1) and writes the output.
//
// The exponent reference m is the largest anchor score of each query row.  Anchors are
// tokens of the unit, so it is a lower bound of the largest logit (sums cannot overflow unless
// a logit exceeds m by more than 2^120, which is flagged); every CTA of a unit takes the same
// m, so partial sums combine by plain addition.  Every wait on an mbarrier is bounded; a wait
// that runs out marks the CTA failed and the outputs of its units NaN.
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <cstdio>
#include <cstdlib>
#include <map>
#include <mutex>
#include <string>
#include <tuple>
#include <type_traits>
#include <vector>

#include "akv_internal.h"

namespace akv {
namespace {

constexpr int NG = 2;               // tile groups per CTA: tiles in processing at once
constexpr int WPG = 4;              // warps per group
constexpr int NCW = NG * WPG;       // compute warps 0 .. 7
constexpr int W_PROD = NCW;         // producer warp
constexpr int NT = (NCW + 1) * 32;  // 288 threads
constexpr int T = kTile;            // tokens per tile block
constexpr int LCH = T / (WPG * 32); // consecutive stored tokens per lane
static_assert(LCH == 8, "a lane's tokens are one byte of a bitmap word");
constexpr int NSLOT = 8;            // stage descriptors; a multiple of NG, so a slot always serves one group
static_assert(NSLOT % NG == 0, "slot reuse must stay within one group");
constexpr int kMaxGrid = 256;       // CTAs of the decode launch at most
constexpr int CHA = 64;             // anchors per score-kernel CTA (4 warps x 16 rows)
constexpr int kRingSlack = 4096;    // shared memory after the ring: the masked rows of the last
                                    // 16-row block of staged anchor values are read from here
constexpr unsigned long long kWaitNs = 2000000000ull;  // an mbarrier wait gives up after 2 s
constexpr float kLog2e = 1.4426950408889634f;
constexpr uint32_t F_MAX = tile_fixed_bytes(T);  // streams, bitmaps, rank words of a full tile

// floats of one partial slot: A [GS][128], R [GS][128], l [WPG][GS], pm [WPG][GS], flag, pad
__host__ __device__ constexpr int part_floats(int GS) { return 256 * GS + 2 * WPG * GS + 4; }
__host__ __device__ constexpr int part_flag(int GS) { return 256 * GS + 2 * WPG * GS; }

struct ScoreParams {
  const uint8_t* arena;
  const __nv_bfloat16* q;
  float* sa;      // [units][ka_stride][G] anchor scores (log2 units)
  float* cmax;    // [units][n_ch][G] largest score of each chunk of CHA anchors
  unsigned* cnt;  // [units] arrival counters of the decode launch, zeroed here
  int n_kv_heads, n_q_heads, G, ka_stride, n_ch;
  float scale_log2;
};

struct Meta {  // a staged tile, as the producer recorded it
  uint32_t ring_off, blk_off, blk_bytes, staged, lo, nrows, j, pad;
};

struct DecodeParams {
  const uint8_t* arena;
  const __nv_bfloat16* q;
  __nv_bfloat16* out;
  float* out_f32;
  const float* sa;
  const float* cmax;
  float* part;
  unsigned* cnt;
  long long ttot;  // tiles of all units
  int grid, n_kv_heads, n_q_heads, rotate, ka_stride, n_ch;
  float scale_log2;
  unsigned long long sign_lo, sign_hi;
  int R;           // records per side and tile that are staged and handled on tensor cores
  int X;           // anchor-value rows per tile that are staged (the weight table's rows)
  int cap;         // staged bytes of a tile block at most
  int ring_bytes, drop_last, smem_sa;
  int o_bar, o_meta, o_misc, o_sa, o_ovf, o_grp, grp_bytes, o_ring;
  int g_qp, g_rows, g_red, g_wb, g_pv, g_qf;  // offsets inside a group's block
  int cta_unit[kMaxGrid];  // first unit of each CTA's range
  int cta_tile[kMaxGrid];  // its first tile inside that unit
};

// ---- device helpers ---------------------------------------------------------------

__device__ __forceinline__ uint32_t smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
// One arrival that also announces `bytes` of transactions the bulk copies will complete.
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}
// Test for completion of the phase with the given parity.
__device__ __forceinline__ uint32_t mbar_try(uint32_t bar, uint32_t parity) {
  uint32_t done;
  asm volatile(
      "{ .reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2; selp.u32 %0, 1, 0, p; }"
      : "=r"(done)
      : "r"(bar), "r"(parity)
      : "memory");
  return done;
}
__device__ __forceinline__ unsigned long long global_ns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
// Bounded wait of one thread; false if kWaitNs passed first (the clock is read every 64 tries).
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity) {
  if (mbar_try(bar, parity)) return true;
  const unsigned long long t0 = global_ns();
  for (unsigned i = 1;; ++i) {
    if (mbar_try(bar, parity)) return true;
    if ((i & 63u) == 0 && global_ns() - t0 >= kWaitNs) return false;
  }
}
// The same by a whole warp: every lane observes the completion itself, and all lanes return
// together with the same result (the clock is lane 0's).
__device__ __forceinline__ bool mbar_wait_w(uint32_t bar, uint32_t parity) {
  uint32_t done = mbar_try(bar, parity);
  if (__all_sync(0xffffffffu, done)) return true;
  const unsigned long long t0 = global_ns();
  for (unsigned i = 1;; ++i) {
    if (!done) done = mbar_try(bar, parity);
    if (__all_sync(0xffffffffu, done)) return true;
    if ((i & 63u) == 0 && __shfl_sync(0xffffffffu, global_ns() - t0 >= kWaitNs ? 1 : 0, 0)) return false;
  }
}
// The CTA's failure flag as lane 0 reads it, the same for every lane of the warp.
__device__ __forceinline__ bool warp_failed(const volatile int* failed) {
  return __shfl_sync(0xffffffffu, *failed, 0) != 0;
}
// Bulk copy global -> this CTA's shared memory (16-byte aligned, a multiple of 16 bytes),
// completing `bytes` transactions on the mbarrier.
__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
               ::"r"(dst), "l"(src), "r"(bytes), "r"(bar)
               : "memory");
}
__device__ __forceinline__ void named_sync(int id, int n) { asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(n) : "memory"); }
// Programmatic dependent launch: the next launch in the stream may be scheduled while this
// one runs; before it reads inputs or writes outputs, a launch waits for the preceding work.
__device__ __forceinline__ void pdl_allow_next() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void pdl_wait_prev() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
// Reduction (no return value) into this CTA's shared memory.
__device__ __forceinline__ void red_local(float* p, float v) {
  asm volatile("red.shared.add.f32 [%0], %1;" ::"r"(smem_u32(p)), "f"(v) : "memory");
}
__device__ __forceinline__ void mma_f16(float (&d)[4], const uint4& a, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a.x), "r"(a.y), "r"(a.z), "r"(a.w), "r"(b0), "r"(b1));
}
__device__ __forceinline__ void mma_bf16(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3, uint32_t b0,
                                         uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}
__device__ __forceinline__ void ldsm_x4_trans(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
// 16 bytes of read-only global data, not kept in L1 (streamed once)
__device__ __forceinline__ uint4 ldg_stream(const void* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

// Two 2-bit codes, at bits 0-1 and 16-17 of x, as an fp16 pair of exact small integers: OR
// them into the mantissa of 1024.0 (0x6400, unit spacing), then subtract 1024.
__device__ __forceinline__ uint32_t codes2_to_h2(uint32_t x) {
  uint32_t t, r;
  asm("lop3.b32 %0, %1, %2, %3, 0xEA;" : "=r"(t) : "r"(x), "r"(0x00030003u), "r"(0x64006400u));
  asm("sub.f16x2 %0, %1, %2;" : "=r"(r) : "r"(t), "r"(0x64006400u));
  return r;
}
// Two 2-bit codes as the exact bf16 pair c: OR into the mantissa of 128.0 (0x4300, unit
// spacing), then t * 1 - 128.
__device__ __forceinline__ uint32_t codes2_to_b2(uint32_t x) {
  uint32_t t, r;
  asm("lop3.b32 %0, %1, %2, %3, 0xEA;" : "=r"(t) : "r"(x), "r"(0x00030003u), "r"(0x43004300u));
  asm("fma.rn.bf16x2 %0, %1, %2, %3;" : "=r"(r) : "r"(t), "r"(0x3F803F80u), "r"(0xC300C300u));
  return r;
}
__device__ __forceinline__ uint32_t pack_h2(__half lo, __half hi) {
  return (uint32_t)__half_as_ushort(lo) | ((uint32_t)__half_as_ushort(hi) << 16);
}
__device__ __forceinline__ uint32_t pack_b2(__nv_bfloat16 lo, __nv_bfloat16 hi) {
  return (uint32_t)__bfloat16_as_ushort(lo) | ((uint32_t)__bfloat16_as_ushort(hi) << 16);
}
// bf16 high part of x and the bf16 of what is left: x ~= hi + lo to about 2^-17 relative
__device__ __forceinline__ void split_b(float x, __nv_bfloat16& hi, __nv_bfloat16& lo) {
  hi = __float2bfloat16_rn(x);
  lo = __float2bfloat16_rn(x - __bfloat162float(hi));
}
__device__ __forceinline__ float half_lo(uint32_t w) {
  return __half2float(__ushort_as_half((unsigned short)(w & 0xFFFFu)));
}
__device__ __forceinline__ float half_hi(uint32_t w) { return __half2float(__ushort_as_half((unsigned short)(w >> 16))); }

// Packed pairs of fp32 (one instruction for both lanes of the pair).
__device__ __forceinline__ float2 f2fma(float2 a, float2 b, float2 c) {
  unsigned long long ra, rb, rc, rd;
  asm("mov.b64 %0, {%1, %2};" : "=l"(ra) : "f"(a.x), "f"(a.y));
  asm("mov.b64 %0, {%1, %2};" : "=l"(rb) : "f"(b.x), "f"(b.y));
  asm("mov.b64 %0, {%1, %2};" : "=l"(rc) : "f"(c.x), "f"(c.y));
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(rd) : "l"(ra), "l"(rb), "l"(rc));
  float2 d;
  asm("mov.b64 {%0, %1}, %2;" : "=f"(d.x), "=f"(d.y) : "l"(rd));
  return d;
}
__device__ __forceinline__ float2 f2add(float2 a, float2 b) {
  unsigned long long ra, rb, rd;
  asm("mov.b64 %0, {%1, %2};" : "=l"(ra) : "f"(a.x), "f"(a.y));
  asm("mov.b64 %0, {%1, %2};" : "=l"(rb) : "f"(b.x), "f"(b.y));
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(rd) : "l"(ra), "l"(rb));
  float2 d;
  asm("mov.b64 {%0, %1}, %2;" : "=f"(d.x), "=f"(d.y) : "l"(rd));
  return d;
}

// 2^x with the hardware approximation (relative error near 2^-22; results below the
// smallest normal flush to 0, which only drops weights under 2^-126 of the reference).
__device__ __forceinline__ float exp2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// Unnormalised 128-point Walsh-Hadamard transform of one row held by a warp, lane l holding
// elements 4 l .. 4 l + 3: two butterfly stages inside the lane, five across lanes.
__device__ __forceinline__ void warp_wht128(float (&x)[4], int lane) {
  const float a0 = x[0] + x[1], a1 = x[0] - x[1], a2 = x[2] + x[3], a3 = x[2] - x[3];
  x[0] = a0 + a2;
  x[1] = a1 + a3;
  x[2] = a0 - a2;
  x[3] = a1 - a3;
#pragma unroll
  for (int m = 1; m < 32; m <<= 1) {  // stage of distance 4 m: partner lane l ^ m
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float v = __shfl_xor_sync(0xffffffffu, x[j], m);
      x[j] = (lane & m) ? v - x[j] : x[j] + v;
    }
  }
}
// The rotation's signs s_j of dims 4 l .. 4 l + 3 applied to x.
__device__ __forceinline__ void apply_signs(float (&x)[4], int lane, unsigned long long lo, unsigned long long hi) {
  const unsigned long long sb = lane < 16 ? lo : hi;
#pragma unroll
  for (int j = 0; j < 4; ++j)
    if ((sb >> ((4 * lane + j) & 63)) & 1ull) x[j] = -x[j];
}

__device__ __forceinline__ const akv_unit_desc* unit_desc(const uint8_t* A, int u) {
  return reinterpret_cast<const akv_unit_desc*>(A + 256) + u;
}
// first element of unit u's query (and output) rows
__device__ __forceinline__ size_t qrow_base(int u, int n_kv_heads, int n_q_heads) {
  const int b = u / n_kv_heads, h = u % n_kv_heads;
  const int G = n_q_heads / n_kv_heads;
  return ((size_t)b * n_q_heads + (size_t)h * G) * 128;
}

// Sections of one unit.
struct UnitView {
  int S, k, nt;
  const uint8_t* AV;
  const uint32_t* table;  // [nt + 1] block offsets, then [nt] value-slot ranges
  const uint8_t* tiles;
};
__device__ __forceinline__ UnitView unit_view(const uint8_t* A, int u) {
  const akv_unit_desc* d = unit_desc(A, u);
  UnitView v;
  v.S = d->len;
  v.k = d->n_anchors;
  v.nt = d->n_tiles;
  v.AV = A + d->off_anchor_v;
  v.table = reinterpret_cast<const uint32_t*>(A + d->off_tile_table);
  v.tiles = A + d->off_tiles;
  return v;
}

// Geometry of one staged tile block: the first `staged` bytes are in shared memory, the
// rest is read from global memory (a tile with more records than the stage holds).
struct TileView {
  const uint8_t* st;   // stage
  const uint8_t* gb;   // the block in global memory
  uint32_t staged;
  int n, nw, n64, nk, nv;
  uint32_t sm_k, sm_v, cd_k, cd_v;  // byte offsets of scales and codes in the block
  __device__ __forceinline__ const uint8_t* at(uint32_t off) const { return off < staged ? st + off : gb + off; }
  __device__ __forceinline__ uint64_t bm(int side, int w) const {
    return reinterpret_cast<const uint64_t*>(st + 8 * n64)[side * nw + w];
  }
  __device__ __forceinline__ int rk(int side, int w) const {
    return reinterpret_cast<const uint16_t*>(st + 8 * n64 + 16 * nw + side * round16(2u * nw))[w];
  }
};
__device__ __forceinline__ TileView tile_view(const uint8_t* st, const Meta& mt, const UnitView& U) {
  TileView v;
  v.st = st;
  v.gb = U.tiles + mt.blk_off;
  v.staged = mt.staged;
  v.n = min(T, U.S - (int)mt.j * T);
  v.nw = (int)tile_words(v.n);
  v.n64 = 64 * v.nw;
  v.nk = v.rk(0, v.nw - 1) + __popcll(v.bm(0, v.nw - 1));
  v.nv = v.rk(1, v.nw - 1) + __popcll(v.bm(1, v.nw - 1));
  const uint32_t F = tile_fixed_bytes(v.n);
  v.sm_k = F;
  v.sm_v = F + round16(4u * (uint32_t)v.nk);
  v.cd_k = v.sm_v + round16(4u * (uint32_t)v.nv);
  v.cd_v = v.cd_k + 32u * (uint32_t)v.nk;
  return v;
}

// Records beyond the staged ones (a locally dense tile) take these rare paths on CUDA
// cores, kept out of line so that the token loop stays small.
// Key residual term scale (q'_g . c) + min sum(q'_g) of key record r.
__device__ __noinline__ float key_record_term(const TileView& tv, int r, const float* qpg, float sqg) {
  const uint32_t smn = *reinterpret_cast<const uint32_t*>(tv.at(tv.sm_k + 4u * (uint32_t)r));
  float dot = 0.f;
  for (int bb = 0; bb < 32; ++bb) {
    const uint32_t byte = *tv.at(tv.cd_k + 32u * (uint32_t)r + (uint32_t)bb);
#pragma unroll
    for (int c = 0; c < 4; ++c) dot += qpg[4 * bb + c] * (float)((byte >> (2 * c)) & 3u);
  }
  return half_hi(smn) * sqg + half_lo(smn) * dot;
}
// accg += p (min + scale c) of value record r, in the rotated domain (value codes are
// dimension-major groups of 16 records).
__device__ __noinline__ void value_record_add(const TileView& tv, int r, float p, float* accg) {
  const uint32_t smn = *reinterpret_cast<const uint32_t*>(tv.at(tv.sm_v + 4u * (uint32_t)r));
  const float ps = p * half_lo(smn), pm = p * half_hi(smn);
  const uint32_t base = tv.cd_v + 512u * (uint32_t)(r / 16);
  for (int d = 0; d < 128; ++d) {
    const uint32_t w = *reinterpret_cast<const uint32_t*>(tv.at(base + 4u * value_code_word(d)));
    atomicAdd(&accg[d], fmaf(ps, (float)((w >> value_code_bit(r % 16)) & 3u), pm));
  }
}
// acc[g] x the anchor's value row (global memory, swizzled by the slot), added into ov[g][:]:
// a run whose value slot lies beyond the tile's staged anchor-value rows (rare).
template <int GS>
__device__ __noinline__ void anchor_value_add(const uint8_t* AV, int anchor, const float* acc, float* ov) {
  const uint8_t* row = AV + (size_t)anchor * 256;
  for (int d = 0; d < 128; ++d) {  // dim d: element d % 8 of chunk d / 8, stored at (d / 8) ^ (row % 8)
    const float x = __bfloat162float(*reinterpret_cast<const __nv_bfloat16*>(row + 16 * ((d >> 3) ^ (anchor & 7)) + 2 * (d & 7)));
#pragma unroll
    for (int g = 0; g < GS; ++g) atomicAdd(&ov[g * 128 + d], acc[g] * x);
  }
}

// A row of GS floats (16-byte aligned for GS >= 4, else 8 or 4) as GS probabilities (pairs).
template <int GS, int NP>
__device__ __forceinline__ void store_row(float* p, const float2 (&v)[NP]) {
  if constexpr (GS == 8) {
    *reinterpret_cast<float4*>(p) = make_float4(v[0].x, v[0].y, v[1].x, v[1].y);
    *reinterpret_cast<float4*>(p + 4) = make_float4(v[2].x, v[2].y, v[3].x, v[3].y);
  } else if constexpr (GS == 4) {
    *reinterpret_cast<float4*>(p) = make_float4(v[0].x, v[0].y, v[1].x, v[1].y);
  } else if constexpr (GS == 2) {
    *reinterpret_cast<float2*>(p) = v[0];
  } else {
    p[0] = v[0].x;
  }
}
// A row of GS consecutive floats (16-byte aligned for GS >= 4, else 8 or 4) into registers.
template <int GS>
__device__ __forceinline__ void load_row(const float* p, float (&out)[GS]) {
  if constexpr (GS == 8) {
    const float4 v = *reinterpret_cast<const float4*>(p), w = *reinterpret_cast<const float4*>(p + 4);
    out[0] = v.x; out[1] = v.y; out[2] = v.z; out[3] = v.w;
    out[4] = w.x; out[5] = w.y; out[6] = w.z; out[7] = w.w;
  } else if constexpr (GS == 4) {
    const float4 v = *reinterpret_cast<const float4*>(p);
    out[0] = v.x; out[1] = v.y; out[2] = v.z; out[3] = v.w;
  } else if constexpr (GS == 2) {
    const float2 v = *reinterpret_cast<const float2*>(p);
    out[0] = v.x; out[1] = v.y;
  } else {
    out[0] = p[0];
  }
}

// =============================== anchor scores =====================================
// CTA (unit u, chunk ch): anchors ch*64 .. ch*64 + 63, warp w rows 16 w .. 16 w + 15, straight
// from global memory into the mma A fragments (rows are stored swizzled in 16-byte chunks by
// slot % 8; the k order is permuted the same way in A and B so that a thread's dims are
// contiguous: thread (r8, c4) of k-pair step j holds dims 32 j + 8 c4 .. + 7 of rows r8, r8 + 8).
template <int GS>
__global__ void __launch_bounds__(128) akv_scores_kernel(const ScoreParams P) {
  pdl_wait_prev();
  pdl_allow_next();
  __shared__ float wmax[4][8];
  const int u = blockIdx.x / P.n_ch, ch = blockIdx.x % P.n_ch;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, r8 = lane >> 2, c4 = lane & 3;
  const akv_unit_desc* d = unit_desc(P.arena, u);
  const int k = d->n_anchors;
  if (ch == 0 && threadIdx.x == 0) P.cnt[u] = 0u;
  const int a0 = ch * CHA + 16 * warp;
  float mx0 = -INFINITY, mx1 = -INFINITY;  // heads 2 c4, 2 c4 + 1
  if (a0 < k) {
    const size_t qb = qrow_base(u, P.n_kv_heads, P.n_q_heads);
    uint2 bq[8];
#pragma unroll
    for (int ks = 0; ks < 8; ++ks)
      bq[ks] = r8 < GS ? *reinterpret_cast<const uint2*>(P.q + qb + (size_t)r8 * 128 + 32 * (ks >> 1) + 8 * c4 + 4 * (ks & 1))
                       : make_uint2(0u, 0u);
    const uint8_t* AK = P.arena + d->off_anchor_k;
    const int ra = min(a0 + r8, k - 1), rb = min(a0 + r8 + 8, k - 1);
    uint4 lo[4], hi[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int cc = 4 * j + c4;
      lo[j] = ldg_stream(AK + (size_t)ra * 256 + 16 * (cc ^ (ra & 7)));
      hi[j] = ldg_stream(AK + (size_t)rb * 256 + 16 * (cc ^ (rb & 7)));
    }
    float dd[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      mma_bf16(dd, lo[j].x, hi[j].x, lo[j].y, hi[j].y, bq[2 * j].x, bq[2 * j].y);
      mma_bf16(dd, lo[j].z, hi[j].z, lo[j].w, hi[j].w, bq[2 * j + 1].x, bq[2 * j + 1].y);
    }
    float* sa = P.sa + (size_t)u * P.ka_stride * GS;
    const int g0 = 2 * c4;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int a = a0 + r8 + 8 * h;
      if (a < k) {
        const float s0 = dd[2 * h] * P.scale_log2, s1 = dd[2 * h + 1] * P.scale_log2;
        if (g0 < GS) {
          sa[(size_t)a * GS + g0] = s0;
          mx0 = fmaxf(mx0, s0);
        }
        if (g0 + 1 < GS) {
          sa[(size_t)a * GS + g0 + 1] = s1;
          mx1 = fmaxf(mx1, s1);
        }
      }
    }
  }
#pragma unroll
  for (int o = 4; o < 32; o <<= 1) {
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, o));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, o));
  }
  if (lane < 4) {
    wmax[warp][2 * lane] = mx0;
    wmax[warp][2 * lane + 1] = mx1;
  }
  __syncthreads();
  if (threadIdx.x < GS) {
    const int g = threadIdx.x;
    P.cmax[((size_t)u * P.n_ch + ch) * GS + g] = fmaxf(fmaxf(wmax[0][g], wmax[1][g]), fmaxf(wmax[2][g], wmax[3][g]));
  }
}

// ============================ the unit's output ====================================
// Sum of the unit's partial slots in a fixed order (CTAs, then groups and the overflow slot),
// the inverse rotation of the value-residual part once, the normalisation, bf16 RNE output.
// Run by nw warps (index widx); warp widx takes heads widx, widx + nw, ...
template <int GS>
__device__ void combine_unit(const DecodeParams& P, int u, int first, int nseg, int widx, int nw) {
  const int lane = threadIdx.x & 31;
  constexpr int PF = part_floats(GS);
  const size_t ob = qrow_base(u, P.n_kv_heads, P.n_q_heads);
  for (int h = widx; h < GS; h += nw) {
    float4 a = make_float4(0.f, 0.f, 0.f, 0.f), r = a;
    float L = 0.f, PM = 0.f;
    bool bad = false;
    for (int c = first; c < first + nseg; ++c)
      for (int j = 0; j <= NG; ++j) {
        const float* sp = P.part + ((size_t)(c + u) * (NG + 1) + j) * PF;
        const float4 x = __ldcg(reinterpret_cast<const float4*>(sp + h * 128 + 4 * lane));
        const float4 y = __ldcg(reinterpret_cast<const float4*>(sp + GS * 128 + h * 128 + 4 * lane));
        a.x += x.x; a.y += x.y; a.z += x.z; a.w += x.w;
        r.x += y.x; r.y += y.y; r.z += y.z; r.w += y.w;
        if (j < NG)
          for (int w = 0; w < WPG; ++w) {
            L += __ldcg(sp + 256 * GS + w * GS + h);
            PM += __ldcg(sp + 256 * GS + WPG * GS + w * GS + h);
          }
        bad |= __ldcg(sp + part_flag(GS)) != 0.f;
      }
    float x[4] = {r.x + PM, r.y + PM, r.z + PM, r.w + PM};
    if (P.rotate) {
      warp_wht128(x, lane);
      apply_signs(x, lane, P.sign_lo, P.sign_hi);
#pragma unroll
      for (int e = 0; e < 4; ++e) x[e] *= (1.0f / 128.0f);
    }
    bad |= !(L < INFINITY);  // a logit so far above the reference that the sums overflowed
    const float yv[4] = {a.x + x[0], a.y + x[1], a.z + x[2], a.w + x[3]};
    const size_t o = ob + (size_t)h * 128 + 4 * lane;
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const float y = bad ? __int_as_float(0x7FC00000) : yv[e] / L;
      P.out[o + e] = __float2bfloat16_rn(y);
      if (P.out_f32) P.out_f32[o + e] = y;
    }
  }
}

// Counts one slot of unit u in (after this thread's group stored it); true if it completed the
// unit, whose slots the caller then combines.
__device__ __forceinline__ bool count_in(const DecodeParams& P, int u, int nseg) {
  __threadfence();
  const unsigned old = atomicAdd(P.cnt + u, 1u);
  const bool last = old == (unsigned)((NG + 1) * nseg - 1);
  if (last) __threadfence();
  return last;
}

// ================================ decode ============================================
template <int GS>
__global__ void __launch_bounds__(NT, 1) akv_decode_kernel(const DecodeParams P) {
  extern __shared__ __align__(128) uint8_t smem[];
  constexpr int NP = GS >= 2 ? GS / 2 : 1;      // pairs of heads for the packed arithmetic
  constexpr int HPL = GS >= 2 ? GS / 2 : 1;     // heads per lane when building value operands
  constexpr int PF = part_floats(GS);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int c4 = lane & 3, r8 = lane >> 2;
  const int c = blockIdx.x;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + P.o_bar);
  Meta* meta = reinterpret_cast<Meta*>(smem + P.o_meta);
  volatile int* failed = reinterpret_cast<volatile int*>(smem + P.o_misc);
  float* SAs = reinterpret_cast<float*>(smem + P.o_sa);
  float* ovf = reinterpret_cast<float*>(smem + P.o_ovf);  // [2][GS][128]: anchor-value and value-residual overflow sums
  uint8_t* ring = smem + P.o_ring;
  // per slot: block + anchor rows landed (full), slot free again (empty: its group's warps are
  // done); per unit: its anchor-score table landed (sa_full), compute warps done with it (sa_free)
  auto bar_full = [&](int s) { return smem_u32(bars + s); };
  auto bar_empty = [&](int s) { return smem_u32(bars + NSLOT + s); };
  const uint32_t bar_sa_full = smem_u32(bars + 2 * NSLOT), bar_sa_free = smem_u32(bars + 2 * NSLOT + 1);

  if (tid == 0) {
    for (int s = 0; s < NSLOT; ++s) {
      mbar_init(bar_full(s), 1);
      mbar_init(bar_empty(s), WPG);
    }
    mbar_init(bar_sa_full, 1);
    mbar_init(bar_sa_free, NCW);
    *failed = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  for (int e = tid; e < 2 * GS * 128; e += NT) ovf[e] = 0.f;
  // zeroed p rows: rows past a tile's records are read (and multiplied by zero codes)
  for (int gi = 0; gi < NG; ++gi) {
    float* pvz = reinterpret_cast<float*>(smem + P.o_grp + gi * P.grp_bytes + P.g_pv);
    for (int e = tid; e < P.R * 8; e += NT) pvz[e] = 0.f;
  }
  __syncthreads();
  pdl_allow_next();
  // Everything above touches only this CTA's shared memory; from here on the launch reads
  // the cache, the query and the anchor scores, and writes outputs.
  pdl_wait_prev();

  // This CTA's range of the concatenated tiles, walked as segments (one per unit it touches).
  const long long B0 = (long long)c * P.ttot / P.grid, B1 = (long long)(c + 1) * P.ttot / P.grid;
  struct Seg {
    int u, jb, je, ib;  // unit, its tiles [jb, je), CTA-local index of tile jb
    long long t0;       // global index of the unit's tile 0
    int nt, first, nseg;
  };
  auto seg_fill = [&](Seg& s) {
    s.nt = unit_desc(P.arena, s.u)->n_tiles;
    s.je = (int)min((long long)s.nt, B1 - s.t0);
    s.first = (int)(((s.t0 + 1) * P.grid - 1) / P.ttot);
    s.nseg = (int)(((s.t0 + s.nt) * P.grid - 1) / P.ttot) - s.first + 1;
  };
  auto seg_begin = [&](Seg& s) {
    s.u = P.cta_unit[c];
    s.jb = P.cta_tile[c];
    s.t0 = B0 - s.jb;
    s.ib = 0;
    seg_fill(s);
  };
  auto seg_next = [&](Seg& s) -> bool {  // false past the last segment
    if (s.t0 + s.je >= B1) return false;
    s.ib += s.je - s.jb;
    s.t0 += s.nt;
    ++s.u;
    s.jb = 0;
    seg_fill(s);
    return true;
  };

  // =========================== producer warp ===================================
  if (warp == W_PROD) {
    struct InFlight {
      int i;
      uint32_t a, e;
    };
    InFlight fq[NSLOT];  // tiles whose slot may not be free yet, oldest first (lane 0)
    int qh = 0, qn = 0;
    uint32_t head = 0;
    int n_cta_tiles = (int)(B1 - B0);
    Seg sg;
    seg_begin(sg);
    int sigma = 0, prev_u = -1, prev_first = 0, prev_nseg = 0;
    // the overflow sums of a finished segment into this CTA's third slot of its unit, then the
    // unit's counter (whole warp)
    auto flush_ovf = [&](int u, int first, int nseg) {
      float* dst = P.part + ((size_t)(c + u) * (NG + 1) + NG) * PF;
      for (int e = 4 * lane; e < GS * 128; e += 128) {
        float4* oa = reinterpret_cast<float4*>(ovf + e);
        float4* orr = reinterpret_cast<float4*>(ovf + GS * 128 + e);
        *reinterpret_cast<float4*>(dst + e) = *oa;
        *reinterpret_cast<float4*>(dst + GS * 128 + e) = *orr;
        *oa = make_float4(0.f, 0.f, 0.f, 0.f);
        *orr = make_float4(0.f, 0.f, 0.f, 0.f);
      }
      if (lane == 0) dst[part_flag(GS)] = *failed ? 1.f : 0.f;
      __syncwarp();
      int last = 0;
      if (lane == 0) last = count_in(P, u, nseg) ? 1 : 0;
      if (__shfl_sync(0xffffffffu, last, 0)) {
        __threadfence();
        combine_unit<GS>(P, u, first, nseg, 0, 1);
      }
    };
    for (;; ++sigma) {
      const UnitView U = unit_view(P.arena, sg.u);
      if (sigma > 0) {
        // every compute warp is done with the previous unit's anchor scores and overflow sums
        if (!warp_failed(failed) && !mbar_wait_w(bar_sa_free, (uint32_t)(sigma - 1) & 1u)) *failed = 1;
        flush_ovf(prev_u, prev_first, prev_nseg);
      }
      if (lane == 0) {
        if (P.smem_sa && !*failed) {
          const uint32_t bytes = round16(4u * (uint32_t)(U.k * GS));
          mbar_expect_tx(bar_sa_full, bytes);
          bulk_g2s(smem_u32(SAs), P.sa + (size_t)sg.u * P.ka_stride * GS, bytes, bar_sa_full);
        } else {
          mbar_arrive(bar_sa_full);  // the unit's start, for the compute warps
        }
      }
      for (int j = sg.jb; j < sg.je; ++j) {
        const int i = sg.ib + (j - sg.jb), s = i % NSLOT;
        if (lane == 0 && !*failed) {
          const uint32_t blk0 = U.table[j], blkn = U.table[j + 1] - blk0, sr = U.table[U.nt + 1 + j];
          const uint32_t lo = sr & 0xFFFFu, hi = sr >> 16;
          const uint32_t staged = min(blkn, (uint32_t)P.cap);
          const uint32_t nrows = min(hi - lo + 1u, (uint32_t)P.X);
          const uint32_t sz = staged + 256u * nrows;
          if (head + sz > (uint32_t)P.ring_bytes) head = 0;
          const uint32_t a = head;
          // wait for the in-flight tiles whose bytes overlap [a, a + sz), and for the slot's
          // previous tile, oldest first
          int last = -1;
          for (int t = 0; t < qn; ++t) {
            const InFlight& f = fq[(qh + t) % NSLOT];
            if (f.a < a + sz && a < f.e) last = t;
          }
          if (qn == NSLOT && last < 0) last = 0;
          bool ok = true;
          for (int t = 0; t <= last && ok; ++t) {
            const InFlight& f = fq[qh];
            ok = mbar_wait(bar_empty(f.i % NSLOT), (uint32_t)(f.i / NSLOT) & 1u);
            qh = (qh + 1) % NSLOT;
            --qn;
          }
          if (!ok) {
            *failed = 1;
          } else {
            head = a + sz;
            fq[(qh + qn) % NSLOT] = InFlight{i, a, a + sz};
            ++qn;
            meta[s] = Meta{a, blk0, blkn, staged, lo, nrows, (uint32_t)j, 0u};
            // (drop_last: a test withholds the last tile of the range)
            if (!(P.drop_last > 0 && i == n_cta_tiles - P.drop_last)) {
              mbar_expect_tx(bar_full(s), sz);
              bulk_g2s(smem_u32(ring + a), U.tiles + blk0, staged, bar_full(s));
              if (nrows) bulk_g2s(smem_u32(ring + a + staged), U.AV + (size_t)lo * 256, 256u * nrows, bar_full(s));
            } else {
              fq[(qh + qn - 1) % NSLOT].e = fq[(qh + qn - 1) % NSLOT].a;  // nothing in flight there
            }
          }
        }
        __syncwarp();
      }
      prev_u = sg.u;
      prev_first = sg.first;
      prev_nseg = sg.nseg;
      if (!seg_next(sg)) break;
    }
    if (!warp_failed(failed) && !mbar_wait_w(bar_sa_free, (uint32_t)sigma & 1u)) *failed = 1;
    flush_ovf(prev_u, prev_first, prev_nseg);
    // every copy this warp started has landed before the CTA may exit (bounded)
    if (lane == 0)
      for (int t = 0; t < qn; ++t) {
        const InFlight& f = fq[(qh + t) % NSLOT];
        if (f.e > f.a) mbar_wait(bar_full(f.i % NSLOT), (uint32_t)(f.i / NSLOT) & 1u);
      }
    if (lane == 0 && P.smem_sa) mbar_wait(bar_sa_full, (uint32_t)sigma & 1u);
    return;
  }

  // =========================== compute groups ==================================
  const int grp = warp / WPG, wg = warp % WPG, gt = tid - grp * WPG * 32;
  uint8_t* GB = smem + P.o_grp + grp * P.grp_bytes;
  float* qp = reinterpret_cast<float*>(GB + P.g_qp);      // [GS][128] rotated query q'
  float* rows = reinterpret_cast<float*>(GB + P.g_rows);  // [0,8): -m, [8,16): -inf, [16,24): sum q', [24,32): m
  int* lastf = reinterpret_cast<int*>(GB + P.g_red);
  float* wb = reinterpret_cast<float*>(GB + P.g_wb);      // [2][X][GS] value weights of a tile's slots
  float* pv = reinterpret_cast<float*>(GB + P.g_pv);      // [R][8] p rows of the value records, then A operands
  uint2* qf = reinterpret_cast<uint2*>(GB + P.g_qf);      // [NBF][8][32] key-residual B fragments
  const int bar_id = 1 + grp;
  auto gsync = [&]() { named_sync(bar_id, WPG * 32); };
  constexpr int NBF = GS == 8 ? 2 : 1;  // key-residual fragment sets: GS = 8 keeps high and low parts apart

  float accA[4][4], accR[4][4];  // anchor-value and value-residual sums, dims 32 wg .. 32 wg + 31
  float2 l2[NP];
  float pminv[HPL];
  int lt = 0;  // this group's tiles so far (weight-table buffer parity)
  Seg sg;
  seg_begin(sg);
  for (int sigma = 0;; ++sigma) {
    const UnitView U = unit_view(P.arena, sg.u);
    const int k = U.k;
    // ---- segment set-up: q' rows (warp wg: heads wg, wg + 4), their sums, the reference m ----
    {
      const size_t qb = qrow_base(sg.u, P.n_kv_heads, P.n_q_heads);
      const float f = P.rotate ? P.scale_log2 * (1.0f / 128.0f) : P.scale_log2;
      for (int g = wg; g < GS; g += WPG) {
        const uint2 raw = *reinterpret_cast<const uint2*>(P.q + qb + (size_t)g * 128 + 4 * lane);
        float x[4] = {__bfloat162float(__ushort_as_bfloat16((unsigned short)(raw.x & 0xFFFFu))),
                      __bfloat162float(__ushort_as_bfloat16((unsigned short)(raw.x >> 16))),
                      __bfloat162float(__ushort_as_bfloat16((unsigned short)(raw.y & 0xFFFFu))),
                      __bfloat162float(__ushort_as_bfloat16((unsigned short)(raw.y >> 16)))};
        if (P.rotate) {
          apply_signs(x, lane, P.sign_lo, P.sign_hi);
          warp_wht128(x, lane);
        }
#pragma unroll
        for (int j = 0; j < 4; ++j) x[j] *= f;
        *reinterpret_cast<float4*>(qp + g * 128 + 4 * lane) = make_float4(x[0], x[1], x[2], x[3]);
        const float sg_ = warp_sum((x[0] + x[1]) + (x[2] + x[3]));
        float m = -INFINITY;
        const int nch = (k + CHA - 1) / CHA;
        for (int ch = lane; ch < nch; ch += 32) m = fmaxf(m, P.cmax[((size_t)sg.u * P.n_ch + ch) * GS + g]);
        m = warp_max(m);
        if (lane == 0) {
          rows[g] = -m;
          rows[8 + g] = -INFINITY;
          rows[16 + g] = sg_;
          rows[24 + g] = m;
        }
      }
    }
#pragma unroll
    for (int nb = 0; nb < 4; ++nb)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        accA[nb][e] = 0.f;
        accR[nb][e] = 0.f;
      }
#pragma unroll
    for (int i = 0; i < NP; ++i) l2[i] = make_float2(0.f, 0.f);
#pragma unroll
    for (int i = 0; i < HPL; ++i) pminv[i] = 0.f;
    gsync();
    // key-residual B fragments (k-step ks): column n = lane / 4 is head n as the fp16 high part
    // (set 0) and low part (set 1) for GS = 8, else head n % 4 high (n < 4) or low (n >= 4);
    // k pairs (2t, 2t+1) <-> dims (16 ks + 2t, 16 ks + 2t + 8), (2t+8, 2t+9) <-> (16 ks + 2t + 1,
    // 16 ks + 2t + 9), t = lane % 4; warp wg builds k-steps wg, wg + 4
    {
      const int gcol = lane >> 2, cc = lane & 3;
#pragma unroll
      for (int hl = 0; hl < NBF; ++hl)
        for (int ks = wg; ks < 8; ks += WPG) {
          uint2 fk = make_uint2(0u, 0u);
          const int head = GS == 8 ? gcol : (gcol & 3);
          const bool low = GS == 8 ? hl == 1 : gcol >= 4;
          if (head < GS) {
            const float* x = qp + head * 128 + 16 * ks + 2 * cc;
            auto part = [&](float v) {
              const __half hi = __float2half_rn(v);
              return low ? __float2half_rn(v - __half2float(hi)) : hi;
            };
            fk.x = pack_h2(part(x[0]), part(x[8]));
            fk.y = pack_h2(part(x[1]), part(x[9]));
          }
          qf[(hl * 8 + ks) * 32 + lane] = fk;
        }
    }
    // the unit's anchor-score table (every warp waits, tiles or not, so its phase count stays right)
    if (!warp_failed(failed) && !mbar_wait_w(bar_sa_full, (uint32_t)sigma & 1u)) *failed = 1;
    gsync();  // fragments built
    const float* SAt = P.smem_sa ? SAs : P.sa + (size_t)sg.u * P.ka_stride * GS;

    const int i_end = sg.ib + (sg.je - sg.jb);
    int i0 = sg.ib + ((grp - sg.ib % NG) + NG) % NG;  // this group's first tile of the segment
    for (int i = i0; i < i_end; i += NG, ++lt) {
      const int s = i % NSLOT;
      const bool go = !warp_failed(failed) && mbar_wait_w(bar_full(s), (uint32_t)(i / NSLOT) & 1u);
      if (!go) *failed = 1;
      const Meta mt = meta[s];
      const uint8_t* st = ring + mt.ring_off;
      TileView tv;
      int nKs = 0, nVs = 0;
      float* W = wb + (lt & 1) * P.X * GS;
      if (go) {
        tv = tile_view(st, mt, U);
        const uint32_t codes_staged = tv.staged > tv.cd_k ? (tv.staged - tv.cd_k) / 32u : 0u;
        nKs = min(min(tv.nk, P.R), (int)codes_staged);
        nVs = min(tv.nv, P.R);
        for (int e = gt; e < P.X * GS; e += WPG * 32) W[e] = 0.f;
        // ---- key residuals: q' . c of the staged key records, tensor cores; the terms
        // scale (q' . c) + min sum(q') - m are written over the records' codes ----
        float* rsb = reinterpret_cast<float*>(const_cast<uint8_t*>(st) + tv.cd_k);
        for (int g16 = wg; g16 * 16 < nKs; g16 += 2 * WPG) {
          uint32_t wd[2][2][8];  // [group][record r8 / r8 + 8][16-dim step]
#pragma unroll
          for (int q = 0; q < 2; ++q)
#pragma unroll
            for (int hr = 0; hr < 2; ++hr) {
              const int sl = (g16 + q * WPG) * 16 + r8 + 8 * hr;
              uint4 w0 = make_uint4(0u, 0u, 0u, 0u), w1 = w0;
              if (sl < nKs) {
                w0 = *reinterpret_cast<const uint4*>(st + tv.cd_k + 32u * (uint32_t)sl);
                w1 = *reinterpret_cast<const uint4*>(st + tv.cd_k + 32u * (uint32_t)sl + 16u);
              }
              wd[q][hr][0] = w0.x; wd[q][hr][1] = w0.y; wd[q][hr][2] = w0.z; wd[q][hr][3] = w0.w;
              wd[q][hr][4] = w1.x; wd[q][hr][5] = w1.y; wd[q][hr][6] = w1.z; wd[q][hr][7] = w1.w;
            }
          float d[2][2][4] = {};
#pragma unroll
          for (int ks = 0; ks < 8; ++ks) {
            const uint2 b0 = qf[ks * 32 + lane], b1 = qf[((NBF - 1) * 8 + ks) * 32 + lane];
#pragma unroll
            for (int q = 0; q < 2; ++q) {
              const uint32_t xa = wd[q][0][ks] >> (4 * c4), xb = wd[q][1][ks] >> (4 * c4);
              const uint4 a = make_uint4(codes2_to_h2(xa), codes2_to_h2(xb), codes2_to_h2(xa >> 2), codes2_to_h2(xb >> 2));
              if constexpr (GS == 8) {
                mma_f16(d[q][0], a, b0.x, b0.y);
                mma_f16(d[q][1], a, b1.x, b1.y);
              } else {
                mma_f16(d[q][ks & 1], a, b0.x, b0.y);
              }
            }
          }
          __syncwarp();  // every lane has its codes before any term overwrites them
#pragma unroll
          for (int q = 0; q < 2; ++q) {
            float v[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              v[e] = d[q][0][e] + d[q][1][e];
              if constexpr (GS != 8) v[e] += __shfl_xor_sync(0xffffffffu, v[e], 2);
            }
            if (GS == 8 || c4 < 2) {
#pragma unroll
              for (int hr = 0; hr < 2; ++hr) {
                const int sl = (g16 + q * WPG) * 16 + r8 + 8 * hr;
                if (sl < nKs) {
                  const uint32_t smn = *reinterpret_cast<const uint32_t*>(st + tv.sm_k + 4u * (uint32_t)sl);
#pragma unroll
                  for (int e = 0; e < 2; ++e) {
                    const int g = 2 * c4 + e;
                    if (g < GS) rsb[sl * 8 + g] = half_hi(smn) * rows[16 + g] + half_lo(smn) * v[2 * hr + e] + rows[g];
                  }
                }
              }
            }
          }
        }
      }
      gsync();  // (A) key-residual terms written, weight table zeroed
      if (go) {
        // ---- tokens: lane -> stored tokens t0 .. t0 + 7, every head ----
        const int t0 = wg * (32 * LCH) + LCH * lane;
        if (t0 < tv.n) {
          const int nvalid = min(LCH, tv.n - t0);
          const uint4 ka0 = *reinterpret_cast<const uint4*>(st + 4 * t0);
          const uint4 ka1 = *reinterpret_cast<const uint4*>(st + 4 * t0 + 16);
          const uint4 va0 = *reinterpret_cast<const uint4*>(st + 4 * (tv.n64 + t0));
          const uint4 va1 = *reinterpret_cast<const uint4*>(st + 4 * (tv.n64 + t0) + 16);
          const uint32_t ek[LCH] = {ka0.x, ka0.y, ka0.z, ka0.w, ka1.x, ka1.y, ka1.z, ka1.w};
          const uint32_t ev[LCH] = {va0.x, va0.y, va0.z, va0.w, va1.x, va1.y, va1.z, va1.w};
          const int wi = t0 >> 6, sh = t0 & 63;
          const uint64_t wk = tv.bm(0, wi), wv = tv.bm(1, wi);
          const uint32_t kbits = (uint32_t)(wk >> sh) & 0xFFu, vbits = (uint32_t)(wv >> sh) & 0xFFu;
          int rkn = tv.rk(0, wi) + __popcll(wk & ((1ull << sh) - 1ull));
          int rvn = tv.rk(1, wi) + __popcll(wv & ((1ull << sh) - 1ull));
          const float* rsb = reinterpret_cast<const float*>(st + tv.cd_k);
          const float* negrow = rows;
          const float* ninfrow = rows + 8;
          const uint32_t lo = mt.lo;
          const int nrows = (int)mt.nrows;
          uint32_t key = ev[0] & 0xFFFFu;  // value slot of the run being summed
          float2 acc[NP];
#pragma unroll
          for (int i2 = 0; i2 < NP; ++i2) acc[i2] = make_float2(0.f, 0.f);
          // a finished run's weights into the tile's table (or, beyond its staged rows, its
          // anchor-value products into the overflow sums)
          auto flush = [&](uint32_t kk, const float2 (&v)[NP]) {
            const int ix = (int)(kk - lo);
            if (ix < nrows) {
              float* w = W + ix * GS;
#pragma unroll
              for (int g = 0; g < GS; ++g) red_local(w + g, (g & 1) ? v[g >> 1].y : v[g >> 1].x);
            } else {
              float vv[GS];
#pragma unroll
              for (int g = 0; g < GS; ++g) vv[g] = (g & 1) ? v[g >> 1].y : v[g >> 1].x;
              anchor_value_add<GS>(U.AV, (int)kk, vv, ovf);
            }
          };
#pragma unroll
          for (int e = 0; e < LCH; ++e) {
            const int a = min((int)(ek[e] & 0xFFFFu), k - 1);  // indices are < k by construction
            float sa[GS], rt[GS];
            load_row<GS>(SAt + a * GS, sa);
            const bool kb = (kbits >> e) & 1u;
            const int r = rkn;
            rkn += (int)kb;
            if (kb && r >= nKs && e < nvalid) {  // beyond the staged records: CUDA cores (rare)
#pragma unroll
              for (int g = 0; g < GS; ++g) rt[g] = key_record_term(tv, r, qp + g * 128, rows[16 + g]) + rows[g];
            } else {  // the key-residual terms, -m, or -inf for a token past the tile's end
              load_row<GS>(e >= nvalid ? ninfrow : (kb ? rsb + r * 8 : negrow), rt);
            }
            const float gk = half_hi(ek[e]), gv = half_hi(ev[e]);
            float2 pe[NP], cw[NP];
#pragma unroll
            for (int i2 = 0; i2 < NP; ++i2) {
              const float2 s2 = make_float2(sa[2 * i2], GS >= 2 ? sa[2 * i2 + 1] : 0.f);
              const float2 r2 = make_float2(rt[2 * i2], GS >= 2 ? rt[2 * i2 + 1] : -INFINITY);
              const float2 x = f2fma(make_float2(gk, gk), s2, r2);
              const float2 p = make_float2(exp2_approx(x.x), GS >= 2 ? exp2_approx(x.y) : 0.f);
              l2[i2] = f2add(l2[i2], p);
              cw[i2] = make_float2(p.x * gv, p.y * gv);
              pe[i2] = p;
            }
            const bool vb = (vbits >> e) & 1u;
            const int rv = rvn;
            rvn += (int)vb;
            if (vb && e < nvalid) {
              if (rv < nVs) {
                store_row<GS>(pv + rv * 8, pe);
              } else {  // beyond the staged records: CUDA cores (rare)
#pragma unroll
                for (int g = 0; g < GS; ++g)
                  value_record_add(tv, rv, (g & 1) ? pe[g >> 1].y : pe[g >> 1].x, ovf + GS * 128 + g * 128);
              }
            }
            // tokens past the tile join the current run with zero weight
            const uint32_t av = e < nvalid ? (ev[e] & 0xFFFFu) : key;
            if (av != key) {
              flush(key, acc);
              key = av;
#pragma unroll
              for (int i2 = 0; i2 < NP; ++i2) acc[i2] = cw[i2];
            } else {
#pragma unroll
              for (int i2 = 0; i2 < NP; ++i2) acc[i2] = f2add(acc[i2], cw[i2]);
            }
          }
          flush(key, acc);
        }
      }
      gsync();  // (B) the tile's weights and p rows are complete
      if (go) {
        // ---- value operands: p scale as bf16 high + low parts in the mma A layout, written
        // over the p rows of the same 16 records; sum of p min per head ----
        const int sl16 = lane & 15, hb = lane >> 4;
        for (int grp16 = wg; grp16 * 16 < nVs; grp16 += WPG) {
          const int r = grp16 * 16 + sl16;
          const bool rec_ok = r < nVs;
          uint32_t smn = 0u;
          if (rec_ok) smn = *reinterpret_cast<const uint32_t*>(tv.at(tv.sm_v + 4u * (uint32_t)r));
          const float scl = half_lo(smn), mn = half_hi(smn);
          float pr[HPL];
#pragma unroll
          for (int i2 = 0; i2 < HPL; ++i2) {
            const int g = hb + 2 * i2;
            pr[i2] = (rec_ok && g < GS) ? pv[r * 8 + g] : 0.f;
          }
          __syncwarp();  // the group's p rows are read before they are overwritten
#pragma unroll
          for (int i2 = 0; i2 < HPL; ++i2) {
            const int g = hb + 2 * i2;
            if (g < GS) {
              // A-operand place of (record r, head g): lane 4 g + (r % 8) / 2, register
              // 2 ((r / 8) % 2) (high part) or + 1 (low part), half r % 2
              __nv_bfloat16 phi, plo;
              split_b(pr[i2] * scl, phi, plo);
              pminv[i2] = fmaf(pr[i2], mn, pminv[i2]);
              unsigned short* dst = reinterpret_cast<unsigned short*>(
                  reinterpret_cast<uint8_t*>(pv) + grp16 * 512 + (4 * g + ((sl16 & 7) >> 1)) * 16 + ((sl16 >> 3) & 1) * 8 +
                  (sl16 & 1) * 2);
              dst[0] = __bfloat16_as_ushort(phi);
              dst[2] = __bfloat16_as_ushort(plo);
            }
          }
        }
        // ---- anchor values: w^T V_A over the tile's staged slots (bf16, weights hi + lo) ----
        const uint8_t* Vr = st + mt.staged;
        const int nr = (int)mt.nrows;
        const int mi = lane >> 3, ri = lane & 7;
        for (int blk = 0; 16 * blk < nr; ++blk) {
          const int ka = 16 * blk + 2 * c4;
          uint32_t ah0 = 0, al0 = 0, ah2 = 0, al2 = 0;
          if (r8 < GS) {
            const int kk[4] = {ka, ka + 1, ka + 8, ka + 9};
            __nv_bfloat16 hi[4], lo_[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) split_b(kk[e] < nr ? W[kk[e] * GS + r8] : 0.f, hi[e], lo_[e]);
            ah0 = pack_b2(hi[0], hi[1]);
            al0 = pack_b2(lo_[0], lo_[1]);
            ah2 = pack_b2(hi[2], hi[3]);
            al2 = pack_b2(lo_[2], lo_[3]);
          }
          const uint32_t m0 = (ka < nr ? 0xFFFFu : 0u) | (ka + 1 < nr ? 0xFFFF0000u : 0u);
          const uint32_t m1 = (ka + 8 < nr ? 0xFFFFu : 0u) | (ka + 9 < nr ? 0xFFFF0000u : 0u);
          const int row = 16 * blk + (mi & 1) * 8 + ri;
#pragma unroll
          for (int hf = 0; hf < 2; ++hf) {
            const int cc = (4 * wg + 2 * hf + (mi >> 1)) ^ (int)((mt.lo + (uint32_t)ri) & 7u);
            uint32_t b00, b01, b10, b11;
            ldsm_x4_trans(smem_u32(Vr + row * 256 + 16 * cc), b00, b01, b10, b11);
            // rows past the staged slots hold other bytes: clear their halves of B
            b00 &= m0;
            b10 &= m0;
            b01 &= m1;
            b11 &= m1;
            mma_bf16(accA[2 * hf], ah0, al0, ah2, al2, b00, b01);
            mma_bf16(accA[2 * hf + 1], ah0, al0, ah2, al2, b10, b11);
          }
        }
      }
      gsync();  // (C) every value operand is built
      if (go) {
        // ---- value residuals: (p scale) c over the staged records, in the rotated domain;
        // this lane's four code words hold dimensions 32 wg + 8 nb + r8 of 16 records ----
        const uint32_t woff = tv.cd_v + 4u * (uint32_t)(32 * wg + 4 * r8);
        const bool all_staged = tv.cd_v + 512u * (uint32_t)((nVs + 15) / 16) <= tv.staged;
        for (int g16 = 0; g16 * 16 < nVs; g16 += 2) {
#pragma unroll
          for (int q = 0; q < 2; ++q) {
            if ((g16 + q) * 16 >= nVs) break;  // warp-uniform
            const uint4 a = *reinterpret_cast<const uint4*>(reinterpret_cast<const uint8_t*>(pv) + (g16 + q) * 512 + lane * 16);
            const uint32_t off = woff + 512u * (uint32_t)(g16 + q);
            const uint4 w4 = all_staged ? *reinterpret_cast<const uint4*>(st + off) : *reinterpret_cast<const uint4*>(tv.at(off));
            const uint32_t wd[4] = {w4.x, w4.y, w4.z, w4.w};
#pragma unroll
            for (int nb = 0; nb < 4; ++nb) {
              // records 2c, 2c+1 at bits 2c and 2c + 16, records 2c+8, 2c+9 eight bits higher
              const uint32_t x = wd[nb] >> (2 * c4);
              mma_bf16(accR[nb], a.x, a.y, a.z, a.w, codes2_to_b2(x), codes2_to_b2(x >> 8));
            }
          }
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(bar_empty(s));
    }
    // this warp is done with the unit's anchor scores and overflow sums
    __syncwarp();
    if (lane == 0) mbar_arrive(bar_sa_free);

    // ---- the group's partial for this unit into its slot, then the unit's counter ----
    {
      float* dst = P.part + ((size_t)(c + sg.u) * (NG + 1) + grp) * PF;
      if (r8 < GS) {
#pragma unroll
        for (int nb = 0; nb < 4; ++nb) {
          const int col = 32 * wg + 8 * nb + 2 * c4;
          *reinterpret_cast<float2*>(dst + r8 * 128 + col) =
              make_float2(accA[nb][0] + accA[nb][2], accA[nb][1] + accA[nb][3]);
          *reinterpret_cast<float2*>(dst + GS * 128 + r8 * 128 + col) =
              make_float2(accR[nb][0] + accR[nb][2], accR[nb][1] + accR[nb][3]);
        }
      }
#pragma unroll
      for (int g = 0; g < GS; ++g) {
        const float sl = warp_sum((g & 1) ? l2[g >> 1].y : l2[g >> 1].x);
        if (lane == 0) dst[256 * GS + wg * GS + g] = sl;
      }
#pragma unroll
      for (int i2 = 0; i2 < HPL; ++i2) {
        float v = pminv[i2];
#pragma unroll
        for (int o = 1; o < 16; o <<= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
        const int g = (lane >> 4) + 2 * i2;
        if ((lane & 15) == 0 && g < GS) dst[256 * GS + WPG * GS + wg * GS + g] = v;
      }
      gsync();
      if (gt == 0) {
        dst[part_flag(GS)] = *failed ? 1.f : 0.f;
        *lastf = count_in(P, sg.u, sg.nseg) ? 1 : 0;
      }
      gsync();
      if (*lastf) {
        __threadfence();
        combine_unit<GS>(P, sg.u, sg.first, sg.nseg, wg, WPG);
      }
      gsync();  // lastf and the set-up buffers are reused by the next segment
    }
    if (!seg_next(sg)) break;
  }
}

struct DeviceInfo {
  int sms = 0;
  int smem_optin = 0;
};

DeviceInfo device_info() {
  static std::mutex mu;
  static DeviceInfo cache[64];
  static bool have[64] = {};
  int dev = 0;
  cudaGetDevice(&dev);
  std::lock_guard<std::mutex> lk(mu);
  if (dev >= 0 && dev < 64 && have[dev]) return cache[dev];
  DeviceInfo d;
  cudaDeviceGetAttribute(&d.sms, cudaDevAttrMultiProcessorCount, dev);
  cudaDeviceGetAttribute(&d.smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  if (dev >= 0 && dev < 64) {
    cache[dev] = d;
    have[dev] = true;
  }
  return d;
}

size_t align128(size_t x) { return (x + 127) & ~(size_t)127; }

double max_density(const Layout& L) {
  double dens = 0.0;
  for (const auto& s : L.shape) dens = std::max(dens, (double)std::max(s.nk, s.nv) / (double)s.S);
  return dens;
}
double max_anchor_density(const Layout& L) {
  double dens = 0.0;
  for (const auto& s : L.shape) dens = std::max(dens, (double)s.k / (double)s.S);
  return dens;
}

// Records staged per tile and side: 1.35x the densest unit's mean plus slack, at most 320;
// records of a denser tile beyond these take the CUDA-core paths, which cost far more.
int full_r(const Layout& L) {
  const int R = (int)(T * max_density(L) * 1.35) + 32;
  return std::min(320, std::max(16, (R + 15) & ~15));
}
// Anchor-value rows staged per tile: 1.5x the mean number of value slots a tile covers plus
// slack, at most 256; runs on slots beyond these take a CUDA-core path.
int full_x(const Layout& L) {
  const int X = (int)(1.5 * (T * max_anchor_density(L) + 1.0)) + 16;
  return std::min(256, std::max(16, (X + 15) & ~15));
}

struct Plan {
  DecodeParams P;
  size_t smem = 0;
  int grid = 0;
};

// Shared-memory carve-up for (R, X, table in shared memory or not); false if the ring
// would hold fewer than `min_tiles` of the largest staged tiles.
bool make_plan_rx(const Layout& L, int GS, int R, int X, bool smem_sa, int smem_optin, int min_tiles, Plan* out) {
  DecodeParams& P = out->P;
  P.R = R;
  P.X = X;
  P.cap = (int)(F_MAX + 2 * round16(4u * (uint32_t)R) + 64u * (uint32_t)R);
  P.ka_stride = (L.max_k + 3) & ~3;
  P.smem_sa = smem_sa ? 1 : 0;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off = align128(off + bytes);
    return (int)o;
  };
  P.o_bar = take((2 * NSLOT + 2) * 8);
  P.o_meta = take(NSLOT * sizeof(Meta));
  P.o_misc = take(16);
  P.o_sa = take(smem_sa ? (size_t)P.ka_stride * GS * 4 : 0);
  P.o_ovf = take((size_t)2 * GS * 128 * 4);
  // a group's block: q' rows, small rows, last flag, two weight tables, p rows / A operands
  size_t g = 0;
  auto gtake = [&](size_t bytes) {
    const size_t o = g;
    g = align128(g + bytes);
    return (int)o;
  };
  P.g_qp = gtake((size_t)GS * 128 * 4);
  P.g_rows = gtake(32 * 4);
  P.g_red = gtake(16);
  P.g_wb = gtake((size_t)2 * X * GS * 4);
  P.g_pv = gtake((size_t)R * 32);
  P.g_qf = gtake((size_t)(GS == 8 ? 2 : 1) * 8 * 32 * 8);
  P.grp_bytes = (int)g;
  P.o_grp = take((size_t)NG * g);
  P.o_ring = (int)off;
  const long long room = (long long)smem_optin - (long long)P.o_ring - kRingSlack;
  const long long tile_max = (long long)P.cap + 256LL * X;
  if (room < (long long)min_tiles * tile_max) return false;
  P.ring_bytes = (int)(room & ~127LL);
  out->smem = (size_t)P.o_ring + (size_t)P.ring_bytes + kRingSlack;
  return true;
}

// Preference: the anchor-score table in shared memory (the token gathers' fast path), with
// room for three, then two of the largest staged tiles, staged counts trimmed from their full
// values towards the mean (records first, then anchor-value rows: a run beyond those takes
// the slowest fallback); then the table in global memory (gathers through L1 and L2) the
// same way; then anything that holds two tiles, then one.
bool make_plan(const Layout& L, int GS, int smem_optin, Plan* out, std::string* why) {
  const int R0 = full_r(L), X0 = full_x(L);
  const int Rmin = std::max(16, ((R0 * 3 / 4) + 15) & ~15), Xmin = std::max(16, ((X0 * 3 / 4) + 15) & ~15);
  for (int sa = 1; sa >= 0; --sa)
    for (int min_tiles : {3, 2})
      for (int X = X0; X >= Xmin; X -= 16)
        for (int R = R0; R >= Rmin; R -= 16)
          if (make_plan_rx(L, GS, R, X, sa == 1, smem_optin, min_tiles, out)) return true;
  for (int min_tiles : {2, 1})
    for (int X = X0; X >= 16; X -= 16)
      for (int R = R0; R >= 16; R -= 16)
        if (make_plan_rx(L, GS, R, X, false, smem_optin, min_tiles, out)) return true;
  *why = "shared memory: no room for the decode pipeline";
  return false;
}

using DecodeFn = void (*)(const DecodeParams);
using ScoreFn = void (*)(const ScoreParams);
template <int GS>
DecodeFn decode_kernel() {
  return akv_decode_kernel<GS>;
}
template <int GS>
ScoreFn score_kernel() {
  return akv_scores_kernel<GS>;
}

// Launch configuration per (device, G, layout shape): computed once, then reused, so that a
// call made during CUDA-graph capture only issues the launches.
struct LaunchKey {
  int dev, G, units, max_len, max_k, ctas;
  long long dens_key, adens_key, ttot;
  bool operator<(const LaunchKey& o) const {
    return std::tie(dev, G, units, max_len, max_k, ctas, dens_key, adens_key, ttot) <
           std::tie(o.dev, o.G, o.units, o.max_len, o.max_k, o.ctas, o.dens_key, o.adens_key, o.ttot);
  }
};

}  // namespace

std::atomic<int> g_debug_cluster{0}, g_debug_withhold{0};

// Workspace of a decode call: anchor scores, chunk maxima, arrival counters, partial slots.
DecodeWs decode_ws_layout(const Layout& L) {
  DecodeWs w;
  const size_t units = L.shape.size();
  const size_t ka = (size_t)((L.max_k + 3) & ~3);
  const size_t nch = (size_t)((L.max_k + CHA - 1) / CHA);
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off = (off + bytes + 255) & ~(size_t)255;
    return o;
  };
  w.o_sa = take(units * ka * (size_t)L.G * 4);
  w.o_cmax = take(units * nch * (size_t)L.G * 4);
  w.o_cnt = take(units * 4);
  w.o_part = take((size_t)(kMaxGrid + units) * (NG + 1) * (size_t)part_floats(L.G) * 4);
  w.total = off;
  return w;
}

template <int GS>
int launch_g(const Layout& L, const akv_params& p, const void* arena, const void* q, void* out, float* out_f32,
             float sm_scale, void* ws, void* stream, std::string* why) {
  static std::mutex mu;
  static std::map<LaunchKey, Plan> cache;
  const int units = (int)L.shape.size();
  int dev = 0;
  cudaGetDevice(&dev);
  long long ttot = 0;
  for (const auto& s : L.shape) ttot += s.nt;
  // testing controls (akv_decode_set_debug): a requested number of CTAs, and the failure-detection
  // hook with which every CTA withholds the last tile of its range, so the waits on it run out
  // after their bound and the outputs of its units become NaN
  const int ctas = g_debug_cluster.load(std::memory_order_relaxed);
  const int drop = g_debug_withhold.load(std::memory_order_relaxed);
  const LaunchKey key{dev, L.G, units, L.max_len, L.max_k, ctas, (long long)(max_density(L) * 1e6),
                      (long long)(max_anchor_density(L) * 1e6), ttot};
  Plan pl;
  bool have = false;
  {
    std::lock_guard<std::mutex> lk(mu);
    auto it = cache.find(key);
    if (it != cache.end()) {
      pl = it->second;
      have = true;
    }
  }
  if (!have) {
    const DeviceInfo di = device_info();
    cudaError_t e = cudaFuncSetAttribute(decode_kernel<GS>(), cudaFuncAttributeMaxDynamicSharedMemorySize, di.smem_optin);
    if (e != cudaSuccess) return (int)e;
    if (!make_plan(L, GS, di.smem_optin, &pl, why)) return -1;
    int grid = (int)std::min<long long>(std::min(di.sms, kMaxGrid), ttot);
    if (ctas > 0) grid = (int)std::min<long long>(ctas, ttot);
    pl.grid = grid;
    // first unit and tile of every CTA's range
    long long t0 = 0;
    int u = 0;
    for (int c = 0; c < grid; ++c) {
      const long long b = (long long)c * ttot / grid;
      while (t0 + L.shape[u].nt <= b) t0 += L.shape[u++].nt;
      pl.P.cta_unit[c] = u;
      pl.P.cta_tile[c] = (int)(b - t0);
    }
    pl.P.ttot = ttot;
    pl.P.grid = grid;
    pl.P.n_ch = (L.max_k + CHA - 1) / CHA;
    std::lock_guard<std::mutex> lk(mu);
    cache[key] = pl;
  }
  const DecodeWs W = decode_ws_layout(L);
  uint8_t* wsb = (uint8_t*)ws;
  DecodeParams& P = pl.P;
  P.arena = (const uint8_t*)arena;
  P.q = (const __nv_bfloat16*)q;
  P.out = (__nv_bfloat16*)out;
  P.out_f32 = out_f32;
  P.sa = (const float*)(wsb + W.o_sa);
  P.cmax = (const float*)(wsb + W.o_cmax);
  P.part = (float*)(wsb + W.o_part);
  P.cnt = (unsigned*)(wsb + W.o_cnt);
  P.n_kv_heads = p.n_kv_heads;
  P.n_q_heads = p.n_q_heads;
  P.rotate = (p.flags & AKV_FLAG_ROTATE) ? 1 : 0;
  P.scale_log2 = sm_scale * kLog2e;
  P.sign_lo = L.header.sign_bits[0];
  P.sign_hi = L.header.sign_bits[1];
  P.drop_last = drop;

  ScoreParams S;
  S.arena = P.arena;
  S.q = P.q;
  S.sa = (float*)(wsb + W.o_sa);
  S.cmax = (float*)(wsb + W.o_cmax);
  S.cnt = P.cnt;
  S.n_kv_heads = p.n_kv_heads;
  S.n_q_heads = p.n_q_heads;
  S.G = L.G;
  S.ka_stride = P.ka_stride;
  S.n_ch = P.n_ch;
  S.scale_log2 = P.scale_log2;

  cudaLaunchAttribute attr[1];
  // each launch may overlap the tail of the preceding one (griddepcontrol in the kernels)
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(units * P.n_ch), 1, 1);
  cfg.blockDim = dim3(128, 1, 1);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = (cudaStream_t)stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaError_t e = cudaLaunchKernelEx(&cfg, score_kernel<GS>(), S);
  if (e != cudaSuccess) return (int)e;
  cfg.gridDim = dim3((unsigned)pl.grid, 1, 1);
  cfg.blockDim = dim3(NT, 1, 1);
  cfg.dynamicSmemBytes = pl.smem;
  e = cudaLaunchKernelEx(&cfg, decode_kernel<GS>(), P);
  if (e != cudaSuccess) {
    cudaFuncAttributes fa{};
    cudaFuncGetAttributes(&fa, decode_kernel<GS>());
    *why = "(decode kernel: " + std::to_string(fa.numRegs) + " registers, max " + std::to_string(fa.maxThreadsPerBlock) +
           " threads, " + std::to_string(pl.smem) + " B dynamic shared memory of " +
           std::to_string(fa.maxDynamicSharedSizeBytes) + ", grid " + std::to_string(pl.grid) + ")";
    return (int)e;
  }
  return (int)cudaGetLastError();
}

int launch_decode(const Layout& L, const akv_params& p, const void* arena, const void* q, void* out, float* out_f32,
                  float sm_scale, void* ws, void* stream, std::string* why) {
  switch (L.G) {
    case 1: return launch_g<1>(L, p, arena, q, out, out_f32, sm_scale, ws, stream, why);
    case 2: return launch_g<2>(L, p, arena, q, out, out_f32, sm_scale, ws, stream, why);
    case 4: return launch_g<4>(L, p, arena, q, out, out_f32, sm_scale, ws, stream, why);
    case 8: return launch_g<8>(L, p, arena, q, out, out_f32, sm_scale, ws, stream, why);
  }
  *why = "unsupported group size";
  return -1;
}

const char* cuda_error_string(int err) { return cudaGetErrorString((cudaError_t)err); }

}  // namespace akv
