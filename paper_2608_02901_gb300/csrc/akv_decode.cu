// Decode attention read directly from the AnchorKV compressed cache (Eq. 3 folded into
// Eq. 4: no key or value row is ever rebuilt in memory).  Two launches per call, in stream
// order (three with a dense suffix, whose chunks take a launch of their own between them):
//
// 1. akv_scores_tc_kernel.  The anchor scores S_A[a][g] = q_g . k_a of every anchor of every
//    unit, once per anchor (Eq. 2-3), in log2 units with sm_scale folded in, into the
//    workspace, with the largest score per query head of each chunk of 64 anchors: tiles of
//    128 anchors brought by tensor copies (TMA) into shared memory, products by tcgen05.mma
//    into tensor memory, one persistent warp-specialised CTA per SM.  It streams the anchor
//    keys, a fifth of the compressed bytes.  It also writes each unit's query header (the
//    rotated query q' = H(s o q)/128 of Appendix A.1 Eq. 12, its sums per head, and q' as
//    tensor-core fragments for the key residuals) and zeroes the unit's arrival counter.
//    (With RoPE at decode akv_rope_logits_kernel takes its place.)
//
// 2. akv_decode_kernel.  Persistent: one CTA per SM.  The tile blocks of all units, in unit
//    order, are split into equal contiguous ranges, one per CTA (stream-K): a unit's tiles may
//    lie in several CTAs and a CTA's range may cross units (its segments).  A CTA has two
//    groups of four warps; each group takes every other tile of the range, end to end:
//      staging        the group's warp 0 issues its own tiles into its half of a byte ring of
//                     shared memory: one bulk asynchronous copy of the tile block and one of
//                     the anchor-value rows of the value slots the tile covers (the tile
//                     table records the range), completing a transaction-counted mbarrier;
//                     table entries are read one issue ahead;
//      key residuals  q' . c of the tile's staged key records on tensor cores, the terms
//                     scale (q' . c) + min sum(q') written over the records' own codes;
//      tokens         each lane 8 consecutive stored tokens, every head: logits
//                     gamma_i S_A[a(i)] + residual term, p = 2^(l - m), the normaliser, p
//                     rows of the value records, and the value weights w[a] = sum_i p_i
//                     gamma_i (Eq. 3): tokens are stored sorted by value anchor, so runs
//                     inside a lane are summed in registers and stored, and runs across
//                     lanes merged by a warp segmented scan, without shared atomics;
//      value side     the value-residual sum (p scale) c over the records and the anchor-
//                     value product w^T V_A over the tile's slots, both on tensor cores
//                     (weights and p scale as bf16 high + low parts, codes exact),
//                     accumulated in registers across the segment's tiles.
//    At the end of a segment both groups add their sums into the CTA's shared sums; the group
//    that finishes last applies the inverse rotation once (Appendix E.1), stores the CTA's
//    partial numerator and normaliser into its workspace slot for the unit, and counts it in
//    on the unit's counter; the CTA that completes the count sums the unit's slots in a fixed
//    order and writes the output.  Tiles denser than the staged counts, and runs on value
//    slots beyond a tile's staged anchor-value rows, take CUDA-core paths.
//
// The exponent reference m is the largest anchor score of each query row.  Anchors are
// tokens of the unit, so it is a lower bound of the largest logit (sums cannot overflow unless
// a logit exceeds m by more than 2^120, which is flagged); every CTA of a unit takes the same
// m, so partial sums combine by plain addition.  Every wait on an mbarrier is bounded; a wait
// that runs out marks the CTA failed and the outputs of its units NaN.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
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
constexpr int NCW = NG * WPG;       // warps 0 .. 7; two per SM sub-partition, so 255 registers each
constexpr int NT = NCW * 32;        // 256 threads
constexpr int T = kTile;            // tokens per tile block
constexpr int LCH = T / (WPG * 32); // consecutive stored tokens per lane
static_assert(LCH == 8, "a lane's tokens are one byte of a bitmap word");
constexpr int NSG = 4;              // tiles a group has in flight at most (its stage descriptors)
constexpr int kMaxGrid = 256;       // CTAs of the decode launch at most
constexpr int CHA = 64;             // anchors per chunk maximum of the score launch
// Score launch on tensor cores: a tile of 128 anchors (TMEM lanes) x 16 query rows (columns),
// anchor rows and query rows brought by tensor copies into two 128-byte halves each
constexpr int kScTile = 128;
constexpr uint32_t kScHalfA = kScTile * 128;             // 128 rows x 64 bf16
constexpr uint32_t kScHalfB = 16 * 128;                  // 16 rows x 64 bf16
constexpr uint32_t kScStage = 2 * kScHalfA + 2 * kScHalfB;  // 36 KB, a multiple of 1024
constexpr int kScStages = 6;                             // tiles in flight (one CTA per SM)
constexpr int kScThreads = 192;  // warps 0-3 epilogue (TMEM lanes 32 w ..), 4 copies and products, 5 query headers
constexpr int kScMaxTiles = 512;  // tiles of one CTA (its table in shared memory); the grid grows past this
constexpr uint32_t kScDynSmem = kScStages * kScStage + 1024;  // + alignment of the first stage
constexpr uint32_t kScTmemCols = 32;                     // two accumulators of 16 fp32 columns
// Instruction descriptor of kind::f16: fp32 accumulator (bits 4-5 = 1), bf16 A and B (7-9 = 1,
// 10-12 = 1), both K-major (15, 16 = 0), N / 8 (17-22), M / 16 (24-28).
constexpr uint32_t kScIdesc = (1u << 4) | (1u << 7) | (1u << 10) | ((16u >> 3) << 17) | ((uint32_t)(kScTile >> 4) << 24);
constexpr int kOvl = 32;            // a tile's entries per overflow list (value records, anchor-value runs)
constexpr int kRingSlack = 4096;    // shared memory after the ring: the masked rows of the last
                                    // 16-row block of staged anchor values are read from here
constexpr unsigned long long kWaitNs = 2000000000ull;  // an mbarrier wait gives up after 2 s
constexpr float kLog2e = 1.4426950408889634f;
constexpr uint32_t F_MAX = tile_fixed_bytes(T);  // streams, bitmaps, rank words of a full tile

// floats of one CTA's partial slot for a unit: numerator y [GS][128] (the inverse rotation already
// applied), normaliser l [GS] (8 places), failure flag, pad to 16 bytes
__host__ __device__ constexpr int part_floats(int GS) { return 128 * GS + 12; }
__host__ __device__ constexpr int part_l(int GS) { return 128 * GS; }
__host__ __device__ constexpr int part_flag(int GS) { return 128 * GS + 8; }

// Bytes of a unit's query header (from the score kernel): the rotated query q' [GS][128] f32, its
// sums [8] f32, and the key-residual mma B fragments [GS == 8 ? 2 : 1][8][32] uint2.
__host__ __device__ constexpr int hdr_bytes(int GS) { return GS * 512 + 32 + (GS == 8 ? 2 : 1) * 2048; }

// Dense suffix: tokens per chunk, and the floats of a chunk's partial slot: the value sum
// o [GS][128] under the chunk's own maximum, its normaliser l [8] and that maximum m [8] (log2 units).
constexpr int SCH = kSuffixChunk;
__host__ __device__ constexpr int suf_floats(int GS) { return 128 * GS + 16; }
__host__ __device__ constexpr int suf_l(int GS) { return 128 * GS; }
__host__ __device__ constexpr int suf_m(int GS) { return 128 * GS + 8; }

struct ScoreParams {
  const uint8_t* arena;
  const __nv_bfloat16* q;
  uint8_t* uh;     // [units] query headers, uh_stride bytes apart
  int uh_stride, rotate;
  unsigned long long sign_lo, sign_hi;
  float* sa;      // [units][ka_stride][G] anchor scores (log2 units)
  float* cmax;    // [units][n_ch][G] largest score of each chunk of CHA anchors
  unsigned* cnt;  // [units] arrival counters of the decode launch, zeroed here
  int n_kv_heads, n_q_heads, G, ka_stride, n_ch;
  float scale_log2;
  // dense suffix (null ksuf: none): rows [units][suf_cap][128], lengths per request, n_sch
  // chunks of SCH tokens per unit, each a partial slot of suf_floats(G) floats
  const __nv_bfloat16* ksuf;
  const __nv_bfloat16* vsuf;
  const int32_t* suf_len;
  float* suf_part;
  int suf_cap, n_sch;
  int units, n_t;  // units; tiles of kScTile anchors per unit (the largest unit's)
  long long arena_rows;  // 256-byte rows of the arena the anchor map covers
  // RoPE at decode (the suffix launch): suffix token t of a unit sits at position S + t
  unsigned long long turn[64];  // theta_j / (2 pi) as a 64-bit binary fraction of a turn
};

// The RoPE logits launch (AKV_FLAG_ROPE): every stored token's logit per head.
struct RopeParams {
  const uint8_t* arena;
  const __nv_bfloat16* q;
  float* lg;      // [units][s_stride][G] logits (log2 units, sm_scale folded in), stored order
  float* cmax;    // [units][n_tch][G] largest logit of each chunk of 64 stored tokens
  unsigned* cnt;  // [units] arrival counters of the decode launch, zeroed here
  int n_kv_heads, n_q_heads, rotate, lloyd, s_stride, n_tch;
  float scale_log2;
  unsigned long long sign_lo, sign_hi;
  unsigned long long turn[64];  // theta_j / (2 pi) as a 64-bit binary fraction of a turn
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
  const uint8_t* uh;  // query headers (score kernel)
  int uh_stride;
  long long ttot;  // tiles of all units
  int grid, n_kv_heads, n_q_heads, rotate, ka_stride, n_ch;
  float scale_log2;
  unsigned long long sign_lo, sign_hi;
  int R;           // value records per tile handled on tensor cores (their p rows); sizes the staging cap
  int X;           // anchor-value rows per tile that are staged (the weight table's rows)
  int cap;         // staged bytes of a tile block at most
  int ring_bytes, drop_last, smem_sa;
  int o_bar, o_meta, o_misc, o_sa, o_ovf, o_grp, grp_bytes, o_ring;
  int g_qp, g_rows, g_red, g_wb, g_pv, g_qf, g_ovl;  // offsets inside a group's block
  const float* lg;         // RoPE at decode: logits [units][s_stride][G] in stored order (else null)
  int s_stride;
  const float* suf_part;   // dense suffix partials [units][n_sch][suf_floats] (null: no suffix)
  const int32_t* suf_len;  // suffix tokens per request
  int suf_cap, n_sch;
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
// ---- tensor copies (TMA), tensor memory and the fifth-generation tensor-core MMA (tcgen05) ----
// Tiled 2-D tensor copy global -> this CTA's shared memory at element column x (a multiple of 8
// bf16, so 16-byte aligned) and row y, completing its bytes on the mbarrier.
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const void* tmap, int x, int y, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];"
      ::"r"(dst), "l"(tmap), "r"(x), "r"(y), "r"(bar)
      : "memory");
}
// Shared-memory matrix descriptor of a K-major bf16 operand in the 128-byte swizzled layout:
// rows of 128 bytes (64 elements of K), 8-row groups 1024 bytes apart, 16-byte chunk j of row r
// at chunk j ^ (r & 7) of the 1024-byte-aligned group.  Bits: start address / 16 (0-13),
// leading-dimension offset / 16 (16-29, unused by this layout), stride-dimension offset / 16
// (32-45), descriptor version 1 (46-47), swizzle mode 2 = 128 bytes (61-63).  A K step of 16
// elements advances the start address by 32 bytes; the swizzle applies to the full address.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
  return (uint64_t)((saddr >> 4) & 0x3FFFu) | ((uint64_t)1u << 16) | ((uint64_t)(1024u >> 4) << 32) |
         ((uint64_t)1u << 46) | ((uint64_t)2u << 61);
}
// D[tmem] (+)= A[smem] B[smem]^T, kind::f16 (bf16 operands), issued by one thread.
__device__ __forceinline__ void tc_mma(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc, uint32_t acc) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n"
      ::"r"(d_tmem), "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(acc)
      : "memory");
}
// One arrival on the mbarrier once every MMA this thread issued before it has completed.
__device__ __forceinline__ void tc_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
// Tensor-memory columns for this CTA (a whole warp; ncols a power of two >= 32); the address is
// written to shared memory.  The permit to allocate is given up at once (one allocation per CTA).
__device__ __forceinline__ void tc_alloc(uint32_t dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem), "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tc_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
// Eight consecutive 32-bit columns of the calling thread's tensor-memory lane (a whole warp;
// warp w of the CTA reads lanes 32 (w % 4) .. + 31), waited for before the values are used.
__device__ __forceinline__ void tc_ld8(uint32_t taddr, float (&v)[8]) {
  uint32_t r0, r1, r2, r3, r4, r5, r6, r7;
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8];\n"
      "tcgen05.wait::ld.sync.aligned;\n"
      : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3), "=r"(r4), "=r"(r5), "=r"(r6), "=r"(r7)
      : "r"(taddr)
      : "memory");
  v[0] = __uint_as_float(r0); v[1] = __uint_as_float(r1); v[2] = __uint_as_float(r2); v[3] = __uint_as_float(r3);
  v[4] = __uint_as_float(r4); v[5] = __uint_as_float(r5); v[6] = __uint_as_float(r6); v[7] = __uint_as_float(r7);
}
__device__ __forceinline__ void named_sync(int id, int n) { asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(n) : "memory"); }
// Named barrier of n threads that also returns whether any of them passed a true predicate.
__device__ __forceinline__ bool named_sync_or(int id, int n, bool pred) {
  uint32_t r;
  asm volatile(
      "{ .reg .pred p, q; setp.ne.u32 p, %1, 0; bar.red.or.pred q, %2, %3, p; selp.u32 %0, 1, 0, q; }"
      : "=r"(r)
      : "r"((uint32_t)pred), "r"(id), "r"(n)
      : "memory");
  return r != 0;
}
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
// The Lloyd-Max codec (AKV_FLAG_LLOYD): a code c stands for level L[c] of
// {-1.5078125, -0.453125, 0.453125, 1.5078125}.  Two codes (bits 0-1 and 16-17 of x) become a
// 16-bit pair by a byte permutation out of the four-entry table held in two registers: the
// selector nibbles 2c, 2c + 1 of both codes come from one integer multiply-add and one gather.
__device__ __forceinline__ uint32_t lm_selector(uint32_t x) {
  const uint32_t u = (x & 0x00030003u) * 0x22u + 0x00100010u;  // bytes 0 and 2: nibbles 2c, 2c + 1
  uint32_t sel;
  asm("prmt.b32 %0, %1, %2, %3;" : "=r"(sel) : "r"(u), "r"(0u), "r"(0x00000020u));
  return sel;
}
__device__ __forceinline__ uint32_t lm_pair(uint32_t x, uint32_t tab_lo, uint32_t tab_hi) {
  uint32_t r;
  asm("prmt.b32 %0, %1, %2, %3;" : "=r"(r) : "r"(tab_lo), "r"(tab_hi), "r"(lm_selector(x)));
  return r;
}
// Code pair as the fp16 (key-residual A operand) or bf16 (value-residual B operand) pair of the
// codec's reconstruction values: the codes themselves, or their Lloyd-Max levels (exact in both).
template <int CODEC>
__device__ __forceinline__ uint32_t code_pair_h2(uint32_t x) {
  if constexpr (CODEC == 0) return codes2_to_h2(x);
  else return lm_pair(x, 0xB740BE08u, 0x3E083740u);
}
template <int CODEC>
__device__ __forceinline__ uint32_t code_pair_b2(uint32_t x) {
  if constexpr (CODEC == 0) return codes2_to_b2(x);
  else return lm_pair(x, 0xBEE8BFC1u, 0x3FC13EE8u);
}
// One code's reconstruction value on CUDA cores (the rare paths).
__device__ __forceinline__ float code_level(uint32_t c, int lloyd) {
  if (!lloyd) return (float)c;
  return c == 0u ? -1.5078125f : (c == 1u ? -0.453125f : (c == 2u ? 0.453125f : 1.5078125f));
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
    const float sg = (lane & m) ? -1.f : 1.f;  // v - x (upper partner) or x + v, one exact fma each
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float v = __shfl_xor_sync(0xffffffffu, x[j], m);
      x[j] = fmaf(sg, x[j], v);
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

// Bytes of a tile block at offset `off`: shared memory for its first `staged` bytes, else the
// block in global memory.
__device__ __forceinline__ const uint8_t* blk_at(const uint8_t* st, const uint8_t* gb, uint32_t staged, uint32_t off) {
  return off < staged ? st + off : gb + off;
}
// Records beyond the staged ones (a locally dense tile whose codes did not fit the staging
// cap) take these rare paths on CUDA cores, kept out of line so that the token loop stays
// small.  Their arguments are plain pointers and offsets: a struct passed by value would be
// built in local memory at every call.
// Key residual term scale (q'_g . c) + min sum(q'_g) of the key record whose scale-min word
// is at `smn_off` and whose codes start at `cd_off`.
__device__ __noinline__ float key_record_term(const uint8_t* st, const uint8_t* gb, uint32_t staged, uint32_t smn_off,
                                              uint32_t cd_off, const float* qpg, float sqg, int lloyd) {
  const uint32_t smn = *reinterpret_cast<const uint32_t*>(blk_at(st, gb, staged, smn_off));
  float dot = 0.f;
  for (int bb = 0; bb < 32; ++bb) {
    const uint32_t byte = *blk_at(st, gb, staged, cd_off + (uint32_t)bb);
#pragma unroll
    for (int c = 0; c < 4; ++c) dot += qpg[4 * bb + c] * code_level((byte >> (2 * c)) & 3u, lloyd);
  }
  return half_hi(smn) * sqg + half_lo(smn) * dot;
}
// accg += p (min + scale c) of value record r, in the rotated domain (value codes are
// dimension-major groups of 16 records; the group of r starts at `grp_off`).
__device__ __noinline__ void value_record_add(const uint8_t* st, const uint8_t* gb, uint32_t staged, uint32_t smn_off,
                                              uint32_t grp_off, int r, float p, float* accg, int lloyd) {
  const uint32_t smn = *reinterpret_cast<const uint32_t*>(blk_at(st, gb, staged, smn_off));
  const float ps = p * half_lo(smn), pm = p * half_hi(smn);
  for (int d = 0; d < 128; ++d) {
    const uint32_t w = *reinterpret_cast<const uint32_t*>(blk_at(st, gb, staged, grp_off + 4u * value_code_word(d)));
    atomicAdd(&accg[d], fmaf(ps, code_level((w >> value_code_bit(r % 16)) & 3u, lloyd), pm));
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

// Anchor-score table of a unit, ka rows: [a][GS] floats, except at GS = 8, where heads 0-3 and
// 4-7 are two arrays [2][ka][4]: a gathered 16-byte half-row then lies in any of the eight
// 16-byte bank groups of shared memory (a 32-byte row would start in only four of them).
template <int GS>
__device__ __forceinline__ size_t sa_at(int a, int g, int ka) {
  if constexpr (GS == 8) return (size_t)(g >> 2) * ka * 4 + (size_t)a * 4 + (g & 3);
  else return (size_t)a * GS + g;
}
template <int GS>
__device__ __forceinline__ void load_sa_row(const float* t, int a, int ka, float (&out)[GS]) {
  if constexpr (GS == 8) {
    const float4 v = *reinterpret_cast<const float4*>(t + a * 4), w = *reinterpret_cast<const float4*>(t + (ka + a) * 4);
    out[0] = v.x; out[1] = v.y; out[2] = v.z; out[3] = v.w;
    out[4] = w.x; out[5] = w.y; out[6] = w.z; out[7] = w.w;
  } else {
    if constexpr (GS == 4) {
      const float4 v = *reinterpret_cast<const float4*>(t + a * 4);
      out[0] = v.x; out[1] = v.y; out[2] = v.z; out[3] = v.w;
    } else if constexpr (GS == 2) {
      const float2 v = *reinterpret_cast<const float2*>(t + a * 2);
      out[0] = v.x; out[1] = v.y;
    } else {
      out[0] = t[a];
    }
  }
}

// N consecutive 32-bit words (4 N-byte aligned) from shared memory.
template <int N>
__device__ __forceinline__ void load_words(const uint8_t* p, uint32_t (&w)[N]) {
  if constexpr (N == 4) {
    const uint4 v = *reinterpret_cast<const uint4*>(p);
    w[0] = v.x; w[1] = v.y; w[2] = v.z; w[3] = v.w;
  } else {
    const uint2 v = *reinterpret_cast<const uint2*>(p);
    w[0] = v.x; w[1] = v.y;
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
// Dense suffix chunk sc of unit u (Appendix E.1 and E.2): suffix tokens j0 .. j0 + 63 of its
// request, scored against the unit's GS query rows on tensor cores (rows plain [token][128] bf16;
// the same permuted k order as the anchor chunks), p = 2^(s - m_c) under the chunk's own maximum
// m_c, then o[g][d] = sum_t p_t[g] V[t][d] (thread d) and l[g] = sum_t p_t[g] into the chunk's
// partial slot.  Chunks at or past the request's length write nothing (the combine reads the
// chunks below it only).  ROPE: the keys are pre-RoPE and turn to positions S + t first.
template <int GS, bool ROPE>
__device__ __forceinline__ void suffix_chunk(const ScoreParams& P, int u, int sc, __nv_bfloat16 (*vsm)[128]) {
  __shared__ float ps[SCH][8];
  __shared__ float wm[4][8];
  __shared__ float mc[8];
  const int len = max(0, min(P.suf_len[u / P.n_kv_heads], P.suf_cap));
  const int j0 = sc * SCH;
  if (j0 >= len) return;
  const int nv = min(SCH, len - j0);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, r8 = lane >> 2, c4 = lane & 3;
  const uint8_t* Kr = reinterpret_cast<const uint8_t*>(P.ksuf) + (size_t)u * P.suf_cap * 256;
  const uint8_t* Vr = reinterpret_cast<const uint8_t*>(P.vsuf) + (size_t)u * P.suf_cap * 256;
  // the chunk's value rows, all in flight at once (row t / 16 + 8 i, 16-byte column t % 16),
  // while the keys are scored
  uint4 vrow[SCH / 8];
#pragma unroll
  for (int i = 0; i < SCH / 8; ++i) {
    const int row = tid / 16 + 8 * i;
    vrow[i] = row < nv ? ldg_stream(Vr + (size_t)(j0 + row) * 256 + 16 * (tid % 16)) : make_uint4(0u, 0u, 0u, 0u);
  }
  const size_t qb = qrow_base(u, P.n_kv_heads, P.n_q_heads);
  uint2 bq[8];
#pragma unroll
  for (int ks = 0; ks < 8; ++ks)
    bq[ks] = r8 < GS ? *reinterpret_cast<const uint2*>(P.q + qb + (size_t)r8 * 128 + 32 * (ks >> 1) + 8 * c4 + 4 * (ks & 1))
                     : make_uint2(0u, 0u);
  const int t0 = j0 + 16 * warp;
  const int ra = min(t0 + r8, len - 1), rb = min(t0 + r8 + 8, len - 1);
  uint4 lo[4], hi[4];
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const int cc = 4 * j + c4;
    lo[j] = ldg_stream(Kr + (size_t)ra * 256 + 16 * cc);
    hi[j] = ldg_stream(Kr + (size_t)rb * 256 + 16 * cc);
  }
  float dd[4] = {0.f, 0.f, 0.f, 0.f};
  if constexpr (ROPE) {
    // RoPE at positions S + t: a thread's chunks c4 + 4 j (j < 2) and c4 + 4 j + 8 hold the two
    // members of pairs (d, d + 64), so each row turns in registers; the turned keys enter the
    // products as bf16 high and low parts
    const uint32_t S_u = (uint32_t)unit_desc(P.arena, u)->len;
    uint4 kr[2][4];  // [row ra / rb][chunk j]: the loaded rows
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      kr[0][j] = lo[j];
      kr[1][j] = hi[j];
    }
    uint32_t khi[2][4][4], klo[2][4][4];  // [row][chunk][bf16 pair]
#pragma unroll
    for (int rr = 0; rr < 2; ++rr) {
      const uint32_t p = S_u + (uint32_t)(rr ? rb : ra);
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        const uint32_t* wa = reinterpret_cast<const uint32_t*>(&kr[rr][j]);
        const uint32_t* wb = reinterpret_cast<const uint32_t*>(&kr[rr][j + 2]);
#pragma unroll
        for (int w = 0; w < 4; ++w) {
          float ya[2], yb[2];
#pragma unroll
          for (int hh = 0; hh < 2; ++hh) {
            const int dim = 8 * (4 * j + c4) + 2 * w + hh;  // < 64; its partner is dim + 64
            const float xa = __bfloat162float(__ushort_as_bfloat16((unsigned short)(hh ? wa[w] >> 16 : wa[w] & 0xFFFFu)));
            const float xb = __bfloat162float(__ushort_as_bfloat16((unsigned short)(hh ? wb[w] >> 16 : wb[w] & 0xFFFFu)));
            float sn, cs;
            __sincosf((float)(uint32_t)(((unsigned long long)p * P.turn[dim]) >> 40) * (6.2831853071795865f / 16777216.0f), &sn, &cs);
            ya[hh] = fmaf(xa, cs, -xb * sn);
            yb[hh] = fmaf(xb, cs, xa * sn);
          }
          __nv_bfloat162 ha = __floats2bfloat162_rn(ya[0], ya[1]), hb = __floats2bfloat162_rn(yb[0], yb[1]);
          const float2 fa = __bfloat1622float2(ha), fb = __bfloat1622float2(hb);
          __nv_bfloat162 la = __floats2bfloat162_rn(ya[0] - fa.x, ya[1] - fa.y), lb = __floats2bfloat162_rn(yb[0] - fb.x, yb[1] - fb.y);
          khi[rr][j][w] = *reinterpret_cast<const uint32_t*>(&ha);
          khi[rr][j + 2][w] = *reinterpret_cast<const uint32_t*>(&hb);
          klo[rr][j][w] = *reinterpret_cast<const uint32_t*>(&la);
          klo[rr][j + 2][w] = *reinterpret_cast<const uint32_t*>(&lb);
        }
      }
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      mma_bf16(dd, khi[0][j][0], khi[1][j][0], khi[0][j][1], khi[1][j][1], bq[2 * j].x, bq[2 * j].y);
      mma_bf16(dd, khi[0][j][2], khi[1][j][2], khi[0][j][3], khi[1][j][3], bq[2 * j + 1].x, bq[2 * j + 1].y);
      mma_bf16(dd, klo[0][j][0], klo[1][j][0], klo[0][j][1], klo[1][j][1], bq[2 * j].x, bq[2 * j].y);
      mma_bf16(dd, klo[0][j][2], klo[1][j][2], klo[0][j][3], klo[1][j][3], bq[2 * j + 1].x, bq[2 * j + 1].y);
    }
  } else {
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      mma_bf16(dd, lo[j].x, hi[j].x, lo[j].y, hi[j].y, bq[2 * j].x, bq[2 * j].y);
      mma_bf16(dd, lo[j].z, hi[j].z, lo[j].w, hi[j].w, bq[2 * j + 1].x, bq[2 * j + 1].y);
    }
  }
  const int g0 = 2 * c4;
  float sv[2][2];
  float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const bool ok = t0 + r8 + 8 * h < len;
    sv[h][0] = ok && g0 < GS ? dd[2 * h] * P.scale_log2 : -INFINITY;
    sv[h][1] = ok && g0 + 1 < GS ? dd[2 * h + 1] * P.scale_log2 : -INFINITY;
    mx0 = fmaxf(mx0, sv[h][0]);
    mx1 = fmaxf(mx1, sv[h][1]);
  }
#pragma unroll
  for (int o = 4; o < 32; o <<= 1) {
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, o));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, o));
  }
  if (lane < 4) {
    wm[warp][2 * lane] = mx0;
    wm[warp][2 * lane + 1] = mx1;
  }
#pragma unroll
  for (int i = 0; i < SCH / 8; ++i) *reinterpret_cast<uint4*>(&vsm[tid / 16 + 8 * i][8 * (tid % 16)]) = vrow[i];
  __syncthreads();
  if (tid < 8) mc[tid] = fmaxf(fmaxf(wm[0][tid], wm[1][tid]), fmaxf(wm[2][tid], wm[3][tid]));
  __syncthreads();
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int row = 16 * warp + r8 + 8 * h;
    if (g0 < GS) ps[row][g0] = sv[h][0] > -INFINITY ? exp2_approx(sv[h][0] - mc[g0]) : 0.f;
    if (g0 + 1 < GS) ps[row][g0 + 1] = sv[h][1] > -INFINITY ? exp2_approx(sv[h][1] - mc[g0 + 1]) : 0.f;
  }
  __syncthreads();
  float o[GS];
#pragma unroll
  for (int g = 0; g < GS; ++g) o[g] = 0.f;
  for (int j = 0; j < nv; ++j) {  // thread tid: dimension tid of every row
    const float v = __bfloat162float(vsm[j][tid]);
#pragma unroll
    for (int g = 0; g < GS; ++g) o[g] = fmaf(ps[j][g], v, o[g]);
  }
  float* dst = P.suf_part + ((size_t)u * P.n_sch + sc) * suf_floats(GS);
#pragma unroll
  for (int g = 0; g < GS; ++g) dst[g * 128 + tid] = o[g];
  if (tid < GS) {
    float l = 0.f;
    for (int j = 0; j < nv; ++j) l += ps[j][tid];
    dst[suf_l(GS) + tid] = l;
    dst[suf_m(GS) + tid] = mc[tid];
  }
}

// The dense suffix's chunks (grid: units x n_sch), a launch of their own after the score or RoPE
// logits launch (ROPE: the keys are pre-RoPE).
template <int GS, bool ROPE>
__global__ void __launch_bounds__(128) akv_suffix_kernel(const ScoreParams P) {
  extern __shared__ __align__(16) uint8_t score_dyn[];  // the chunk's value rows
  suffix_chunk<GS, ROPE>(P, blockIdx.x / P.n_sch, blockIdx.x % P.n_sch,
                         reinterpret_cast<__nv_bfloat16 (*)[128]>(score_dyn));
}

// The unit's query header, by one warp: the rotated query q' = H(s o q) / 128 scaled to log2 units
// (Appendix A.1, Eq. 12; warp-local Walsh-Hadamard transform), its sums, and the key-residual mma
// B fragments: column n = lane / 4 is head n as the fp16 high part (set 0) and low part (set 1) for
// GS = 8, else head n % 4 high (n < 4) or low (n >= 4); k pairs (2t, 2t+1) <-> dims
// (16 ks + 2t, 16 ks + 2t + 8), (2t+8, 2t+9) <-> (16 ks + 2t + 1, 16 ks + 2t + 9).  qs: 8 x 128
// floats of shared memory for the rotated rows.
template <int GS>
__device__ __noinline__ void unit_query_header_warp(const ScoreParams& P, int u, float* qs) {
  const int lane = threadIdx.x & 31;
  constexpr int NBF = GS == 8 ? 2 : 1;
  uint8_t* H = P.uh + (size_t)u * P.uh_stride;
  float* hq = reinterpret_cast<float*>(H);
  float* hs = hq + GS * 128;
  uint2* hf = reinterpret_cast<uint2*>(hs + 8);
  const size_t qb = qrow_base(u, P.n_kv_heads, P.n_q_heads);
  const float f = P.rotate ? P.scale_log2 * (1.0f / 128.0f) : P.scale_log2;
  uint2 raw[GS];  // every row's loads in flight at once
#pragma unroll
  for (int g = 0; g < GS; ++g) raw[g] = *reinterpret_cast<const uint2*>(P.q + qb + (size_t)g * 128 + 4 * lane);
#pragma unroll
  for (int g = 0; g < GS; ++g) {
    float x[4] = {__bfloat162float(__ushort_as_bfloat16((unsigned short)(raw[g].x & 0xFFFFu))),
                  __bfloat162float(__ushort_as_bfloat16((unsigned short)(raw[g].x >> 16))),
                  __bfloat162float(__ushort_as_bfloat16((unsigned short)(raw[g].y & 0xFFFFu))),
                  __bfloat162float(__ushort_as_bfloat16((unsigned short)(raw[g].y >> 16)))};
    if (P.rotate) {
      apply_signs(x, lane, P.sign_lo, P.sign_hi);
      warp_wht128(x, lane);
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) x[j] *= f;
    const float4 v = make_float4(x[0], x[1], x[2], x[3]);
    *reinterpret_cast<float4*>(qs + g * 128 + 4 * lane) = v;
    *reinterpret_cast<float4*>(hq + g * 128 + 4 * lane) = v;
    const float sg = warp_sum((x[0] + x[1]) + (x[2] + x[3]));
    if (lane == 0) hs[g] = sg;
  }
  if (lane >= GS && lane < 8) hs[lane] = 0.f;
  __syncwarp();  // the rotated rows are in shared memory for every lane
  const int gcol = lane >> 2, cc = lane & 3;
#pragma unroll
  for (int idx = 0; idx < NBF * 8; ++idx) {
    const int hl = idx >> 3, ks = idx & 7;
    uint2 fk = make_uint2(0u, 0u);
    const int head = GS == 8 ? gcol : (gcol & 3);
    const bool low = GS == 8 ? hl == 1 : gcol >= 4;
    if (head < GS) {
      const float* x = qs + head * 128 + 16 * ks + 2 * cc;
      auto part = [&](float v) {
        const __half hi = __float2half_rn(v);
        return low ? __float2half_rn(v - __half2float(hi)) : hi;
      };
      fk.x = pack_h2(part(x[0]), part(x[8]));
      fk.y = pack_h2(part(x[1]), part(x[9]));
    }
    hf[(hl * 8 + ks) * 32 + lane] = fk;
  }
  __syncwarp();  // the next unit's rows may overwrite qs
}

// Anchor scores on tensor cores (Eq. 2-3: S_A = q . k_a once per anchor).  One persistent CTA per
// SM takes tiles T = blockIdx.x, + gridDim.x, ... of units x n_t; tile (u, t) is anchors
// 128 t .. 128 t + 127 of unit u (tile 0 of every unit is taken even when empty).  Warps have
// roles, coupled only by mbarriers:
//  * warp 4, lane 0, copies and products: it keeps kScStages tiles in flight (two tensor copies
//    bring the anchor rows' 128-byte halves, stored with the 16-byte chunks of row a at chunk
//    j ^ (a & 7), which is the 128-byte swizzled operand layout as it is; two bring the query
//    rows, swizzled by the copy, with the next 16 - G rows of q or zeros in columns that are not
//    read), and as each tile lands and one of two TMEM accumulators is free it issues the 8 K steps
//    of D[128 anchors][16 columns] and commits them to that accumulator's "full" barrier and to the
//    stage's "free" barrier; the stage of the previous tile is refilled once its products are done;
//  * warps 0-3, the epilogue: warp w reads TMEM lanes 32 w .. 32 w + 31 (one anchor per thread),
//    frees the accumulator, writes S_A in log2 units and, after a named barrier of the four warps,
//    the maxima of the tile's two 64-anchor chunks;
//  * warp 5 writes the query header of every unit whose tile 0 is this CTA's and zeroes the unit's
//    arrival counter.
// Both the copying lane and the epilogue walk the same tiles, from a table of the CTA's tiles that
// all threads fill at the start (every descriptor load in flight at once).  Every wait is bounded; a CTA whose wait runs out, or that finds a unit's anchor rows
// outside the arena the map covers, writes +inf as the chunk maxima of all its tiles (the decode's
// outputs for those units become NaN) and stops.
template <int GS>
__global__ void __launch_bounds__(kScThreads) akv_scores_tc_kernel(const __grid_constant__ ScoreParams P,
                                                                   const __grid_constant__ CUtensorMap tmA,
                                                                   const __grid_constant__ CUtensorMap tmB) {
  extern __shared__ __align__(16) uint8_t score_dyn[];
  __shared__ __align__(8) uint64_t bars[2 * kScStages + 4];  // full[s], free[s], acc_full[b], acc_empty[b]
  __shared__ uint32_t tmem_sh;
  __shared__ float wmx[2][4][8];
  __shared__ int failed_sh;
  __shared__ int2 tab[kScMaxTiles];  // this CTA's tiles: the unit's anchors, anchor row (-1: outside the map)
  __shared__ __align__(16) float hdr_q[8 * 128];  // the header warp's rotated query rows
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t sbase = (smem_u32(score_dyn) + 1023u) & ~1023u;
  auto full = [&](int s) { return smem_u32(bars + s); };
  auto freed = [&](int s) { return smem_u32(bars + kScStages + s); };
  auto acc_full = [&](int b) { return smem_u32(bars + 2 * kScStages + b); };
  auto acc_empty = [&](int b) { return smem_u32(bars + 2 * kScStages + 2 + b); };
  volatile int* failed = &failed_sh;
  const int n_tiles = P.units * P.n_t;
  const int n_my = n_tiles > (int)blockIdx.x ? (n_tiles - 1 - (int)blockIdx.x) / (int)gridDim.x + 1 : 0;
  for (int i = tid; i < n_my && i < kScMaxTiles; i += kScThreads) {  // all descriptors in one round trip
    const akv_unit_desc* d = unit_desc(P.arena, ((int)blockIdx.x + i * (int)gridDim.x) / P.n_t);
    const int k = d->n_anchors;
    const uint64_t off = d->off_anchor_k;
    tab[i] = make_int2(k, !(off & 255u) && (long long)(off >> 8) + k <= P.arena_rows ? (int)(off >> 8) : -1);
  }
  if (tid == 0) {
    for (int s = 0; s < kScStages; ++s) {
      mbar_init(full(s), 1);
      mbar_init(freed(s), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(acc_full(b), 1);
      mbar_init(acc_empty(b), 4);  // one arrival per epilogue warp
    }
    *failed = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 0) tc_alloc(smem_u32(&tmem_sh), kScTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_sh;

  // the next of this CTA's tiles that hold anchors (or are a unit's tile 0), from the table: ci is
  // the next entry to look at; row is the anchor row (-1: outside the map)
  int ci = 0;
  const int n_tab = min(n_my, kScMaxTiles);
  auto next_tile = [&](int& u, int& t, int& k, int& row) {
    while (ci < n_tab) {
      const int T = (int)blockIdx.x + ci * (int)gridDim.x;
      const int2 e = tab[ci++];
      k = e.x;
      row = e.y;
      u = T / P.n_t;
      t = T % P.n_t;
      if (t == 0 || t * kScTile < k) return true;
    }
    return false;
  };

  if (warp == 4) {
    if (lane == 0) {  // ---- copies and products
      int u, t, k, row0, n_iss = 0, n_mma = 0;
      auto issue = [&](int j) {  // the tile just found into stage j % kScStages
        const int s = j % kScStages;
        const uint32_t st = sbase + (uint32_t)s * kScStage;
        if (row0 >= 0) {
          const int row = row0 + t * kScTile;  // 256-byte rows
          const int qrow = (int)(qrow_base(u, P.n_kv_heads, P.n_q_heads) >> 7);
          mbar_expect_tx(full(s), kScStage);
          tma_load_2d(st, &tmA, 0, row, full(s));
          tma_load_2d(st + kScHalfA, &tmA, 64, row, full(s));
          tma_load_2d(st + 2 * kScHalfA, &tmB, 0, qrow, full(s));
          tma_load_2d(st + 2 * kScHalfA + kScHalfB, &tmB, 64, qrow, full(s));
        } else {
          mbar_arrive(full(s));  // nothing copied: the epilogue fails the CTA
        }
      };
      bool more = true;
      while (n_iss < kScStages && (more = next_tile(u, t, k, row0))) issue(n_iss++);
      for (int j = 0; j < n_iss; ++j) {
        const int s = j % kScStages, b = j & 1;
        if (*failed || !mbar_wait(full(s), (uint32_t)(j / kScStages) & 1u) ||
            !mbar_wait(acc_empty(b), ((uint32_t)(j >> 1) & 1u) ^ 1u)) {
          *failed = 1;
          break;
        }
        tc_fence_after();
        const uint32_t a = sbase + (uint32_t)s * kScStage, bq = a + 2 * kScHalfA;
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {  // K steps of 16: 32 bytes into a half, then the other half
          const uint32_t ka = (uint32_t)(kk >> 2) * kScHalfA + (uint32_t)(kk & 3) * 32;
          const uint32_t kb = (uint32_t)(kk >> 2) * kScHalfB + (uint32_t)(kk & 3) * 32;
          tc_mma(tmem + 16u * (uint32_t)b, sw128_desc(a + ka), sw128_desc(bq + kb), kScIdesc, kk > 0 ? 1u : 0u);
        }
        tc_commit(acc_full(b));
        tc_commit(freed(s));
        ++n_mma;
        // refill the previous tile's stage once its products are done (this tile's run meanwhile)
        if (j > 0 && more && (more = next_tile(u, t, k, row0))) {
          const int sp = (j - 1) % kScStages;
          if (!mbar_wait(freed(sp), (uint32_t)((j - 1) / kScStages) & 1u)) {
            *failed = 1;
            break;
          }
          issue(n_iss++);  // n_iss = j - 1 + kScStages: stage sp
        }
      }
      // (bounded) nothing of this CTA's is left in flight at exit: copies never consumed (after a
      // failure), and the last commit's arrivals (every earlier one has landed before it)
      if (*failed)
        for (int j = n_mma; j < n_iss; ++j) mbar_wait(full(j % kScStages), (uint32_t)(j / kScStages) & 1u);
      if (n_mma > 0) mbar_wait(freed((n_mma - 1) % kScStages), (uint32_t)((n_mma - 1) / kScStages) & 1u);
    }
    __syncwarp();
  } else if (warp == 5) {  // ---- query headers
    for (int T = (int)blockIdx.x; T < n_tiles; T += (int)gridDim.x) {
      if (T % P.n_t) continue;
      if (lane == 0) P.cnt[T / P.n_t] = 0u;
      unit_query_header_warp<GS>(P, T / P.n_t, hdr_q);
    }
  } else {  // ---- epilogue, warps 0-3
    int u, t, k, row0;
    for (int j = 0; next_tile(u, t, k, row0); ++j) {
      const int b = j & 1;
      const bool got = mbar_wait_w(acc_full(b), (uint32_t)(j >> 1) & 1u);
      tc_fence_after();
      float v[8];
      tc_ld8(tmem + ((uint32_t)(32 * warp) << 16) + 16u * (uint32_t)b, v);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(acc_empty(b));  // this warp's lanes of accumulator b are read
      const bool ok_tile = got && row0 >= 0;
      const int a = t * kScTile + 32 * warp + lane;
      const bool ok = ok_tile && a < k;
      float sc[8];
#pragma unroll
      for (int g = 0; g < 8; ++g) sc[g] = v[g] * P.scale_log2;
      if (ok) {
        float* sa = P.sa + (size_t)u * P.ka_stride * GS;
        if constexpr (GS == 8) {
          *reinterpret_cast<float4*>(sa + (size_t)a * 4) = make_float4(sc[0], sc[1], sc[2], sc[3]);
          *reinterpret_cast<float4*>(sa + ((size_t)P.ka_stride + a) * 4) = make_float4(sc[4], sc[5], sc[6], sc[7]);
        } else if constexpr (GS == 4) {
          *reinterpret_cast<float4*>(sa + (size_t)a * 4) = make_float4(sc[0], sc[1], sc[2], sc[3]);
        } else if constexpr (GS == 2) {
          *reinterpret_cast<float2*>(sa + (size_t)a * 2) = make_float2(sc[0], sc[1]);
        } else {
          sa[a] = sc[0];
        }
      }
#pragma unroll
      for (int g = 0; g < GS; ++g) {
        const float m = warp_max(ok ? sc[g] : -INFINITY);
        if (lane == 0) wmx[b][warp][g] = m;
      }
      // the four warps' maxima are in place; a failure seen by any thread stops all four
      if (named_sync_or(1, 128, !ok_tile || *failed)) {
        if (tid == 0) *failed = 1;
        break;
      }
      if (tid < 2 * GS) {
        const int c = tid / GS, g = tid % GS, ch = 2 * t + c;
        if (ch * CHA < k) P.cmax[((size_t)u * P.n_ch + ch) * GS + g] = fmaxf(wmx[b][2 * c][g], wmx[b][2 * c + 1][g]);
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (*failed) {
    for (int T2 = (int)blockIdx.x; T2 < n_tiles; T2 += (int)gridDim.x) {
      const int u = T2 / P.n_t, t = T2 % P.n_t;
      if (tid < 2 * GS && 2 * t + tid / GS < P.n_ch)
        P.cmax[((size_t)u * P.n_ch + 2 * t + tid / GS) * GS + tid % GS] = INFINITY;
    }
  }
  if (warp == 0) tc_dealloc(tmem, kScTmemCols);
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
  auto slot = [&](int s) { return P.part + (size_t)(first + s + u) * PF; };  // CTA first + s
  // normalisers and failure flags of every slot: lanes in parallel, then a fixed-order reduction
  float Lh[GS];
#pragma unroll
  for (int g = 0; g < GS; ++g) Lh[g] = 0.f;
  bool bad = false;
  for (int s = lane; s < nseg; s += 32) {
    const float* sp = slot(s);
    bad |= __ldcg(sp + part_flag(GS)) != 0.f;
#pragma unroll
    for (int g = 0; g < GS; ++g) Lh[g] += __ldcg(sp + part_l(GS) + g);
  }
  bad = __any_sync(0xffffffffu, bad);
#pragma unroll
  for (int g = 0; g < GS; ++g) Lh[g] = warp_sum(Lh[g]);
  for (int h = widx; h < GS; h += nw) {
    float4 a = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int s0 = 0; s0 < nseg; s0 += 8) {  // eight slots' loads in flight at a time
      float4 xa[8];
#pragma unroll
      for (int j = 0; j < 8; ++j)
        xa[j] = s0 + j < nseg ? __ldcg(reinterpret_cast<const float4*>(slot(s0 + j) + h * 128 + 4 * lane))
                              : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        a.x += xa[j].x; a.y += xa[j].y; a.z += xa[j].z; a.w += xa[j].w;
      }
    }
    float L = 0.f;
#pragma unroll
    for (int g = 0; g < GS; ++g)
      if (g == h) L = Lh[g];
    if (P.suf_part) {  // the dense suffix joins the same softmax (Appendix E.1 and E.2)
      const int len = max(0, min(P.suf_len[u / P.n_kv_heads], P.suf_cap));
      if (len > 0) {
        // the compressed part's reference m (the unit's largest anchor score), the common maximum
        // M over it and the chunks' maxima, and every part rescaled to M
        // (with RoPE at decode: the chunk maxima are those of every token's logit)
        const int nch = P.lg ? (unit_desc(P.arena, u)->len + 63) / 64 : (unit_desc(P.arena, u)->n_anchors + CHA - 1) / CHA;
        float m = -INFINITY;
        for (int ch = lane; ch < nch; ch += 32) m = fmaxf(m, P.cmax[((size_t)u * P.n_ch + ch) * GS + h]);
        m = warp_max(m);
        const float* sp0 = P.suf_part + (size_t)u * P.n_sch * suf_floats(GS);
        const int nsc = (len + SCH - 1) / SCH;
        float M = m;
        for (int c = lane; c < nsc; c += 32) M = fmaxf(M, sp0[(size_t)c * suf_floats(GS) + suf_m(GS) + h]);
        M = warp_max(M);
        const float f0 = exp2_approx(m - M);
        a.x *= f0;
        a.y *= f0;
        a.z *= f0;
        a.w *= f0;
        L *= f0;
        for (int c = 0; c < nsc; ++c) {
          const float* sp = sp0 + (size_t)c * suf_floats(GS);
          const float f = exp2_approx(sp[suf_m(GS) + h] - M);
          const float4 o = *reinterpret_cast<const float4*>(sp + h * 128 + 4 * lane);
          a.x = fmaf(f, o.x, a.x);
          a.y = fmaf(f, o.y, a.y);
          a.z = fmaf(f, o.z, a.z);
          a.w = fmaf(f, o.w, a.w);
          L = fmaf(f, sp[suf_l(GS) + h], L);
        }
      }
    }
    const bool badh = bad || !(L < INFINITY);  // a logit so far above the reference that the sums overflowed
    const float yv[4] = {a.x, a.y, a.z, a.w};
    const size_t o = ob + (size_t)h * 128 + 4 * lane;
    float y[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) y[e] = badh ? __int_as_float(0x7FC00000) : yv[e] / L;
    *reinterpret_cast<uint2*>(P.out + o) = make_uint2(pack_b2(__float2bfloat16_rn(y[0]), __float2bfloat16_rn(y[1])),
                                                      pack_b2(__float2bfloat16_rn(y[2]), __float2bfloat16_rn(y[3])));
    if (P.out_f32) *reinterpret_cast<float4*>(P.out_f32 + o) = make_float4(y[0], y[1], y[2], y[3]);
  }
}

// Counts one slot of unit u in (after this thread's group stored it); true if it completed the
// unit, whose slots the caller then combines.
__device__ __forceinline__ bool count_in(const DecodeParams& P, int u, int nseg) {
  __threadfence();
  const unsigned old = atomicAdd(P.cnt + u, 1u);
  const bool last = old == (unsigned)(nseg - 1);
  if (last) __threadfence();
  return last;
}

// Probabilities of one token for every head: p_g = 2^(gamma S_A[a][g] + rt_g) (rt: the key-residual
// term minus m, or -m), added into the normaliser sums.
template <int GS, int NP>
__device__ __forceinline__ void head_probs(float gk, const float (&sa)[GS], const float (&rt)[GS], float2 (&pe)[NP],
                                           float2 (&l2)[NP]) {
  if constexpr (GS == 1) {
    const float p = exp2_approx(fmaf(gk, sa[0], rt[0]));
    pe[0] = make_float2(p, 0.f);
    l2[0].x += p;
  } else {
    const float2 gk2 = make_float2(gk, gk);
#pragma unroll
    for (int i2 = 0; i2 < NP; ++i2) {
      const float2 x = __ffma2_rn(gk2, make_float2(sa[2 * i2], sa[2 * i2 + 1]), make_float2(rt[2 * i2], rt[2 * i2 + 1]));
      pe[i2] = make_float2(exp2_approx(x.x), exp2_approx(x.y));
      l2[i2] = __fadd2_rn(l2[i2], pe[i2]);
    }
  }
}

// ============================ RoPE at decode (AKV_FLAG_ROPE) ============================
// Keys are stored pre-RoPE, so a token's score no longer factors through its anchor's score:
// q . R(p_i) x^_i with x^_i = gamma_i x_a(i) + r~_i (Eq. 3) and R(p) the rotate-half RoPE turn
// of dimension pairs (j, j + 64) by p theta_j (Section 3.2; Appendix E.1's score kernel rebuilds
// keys and applies RoPE from the stored positions the same way).  CTA (unit u, chunk c): stored
// tokens 64 c .. 64 c + 63; warp w rebuilds tokens 16 w .. 16 w + 15, lane l holding dimensions
// 4 l .. 4 l + 3 (pair partners sit 16 lanes apart), into shared memory; then its 16 x G logits
// come from tensor-core products (keys as fp16 high + low parts, q exact).  The angle of pair j
// at position p is taken as a binary fraction of a turn, p * turn_j mod 2^64 (exact integer
// arithmetic), so the sine and cosine are evaluated on [0, 2 pi) whatever the position.
template <int GS, int CODEC>
__global__ void __launch_bounds__(128) akv_rope_logits_kernel(const RopeParams P) {
  __shared__ __align__(16) float ys[64][132];  // rows 16-byte aligned; 128-bit reads conflict-free
  __shared__ __align__(16) float qsm[8][128];
  __shared__ float wmx4[4][8];
  __shared__ unsigned long long turn[64];
  const int u = blockIdx.x / P.n_tch, c = blockIdx.x % P.n_tch;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const akv_unit_desc* d = unit_desc(P.arena, u);
  const int S = d->len, k = d->n_anchors;
  if (c == 0 && tid == 0) P.cnt[u] = 0u;
  const int ts0 = 64 * c;
  if (ts0 >= S) return;  // past this unit's end (a shorter request)
  const size_t qb = qrow_base(u, P.n_kv_heads, P.n_q_heads);
  for (int e = tid; e < GS * 128; e += 128) qsm[e / 128][e % 128] = __bfloat162float(P.q[qb + e]);
  if (tid < 64) turn[tid] = P.turn[tid];
  // the chunk inside its tile block: one bitmap word (64 tokens) per side
  const int j = ts0 / T, tl0 = ts0 % T;
  const int n = min(T, S - j * T), nw = (int)tile_words(n), n64 = 64 * nw;
  const uint8_t* blk = P.arena + d->off_tiles + reinterpret_cast<const uint32_t*>(P.arena + d->off_tile_table)[j];
  const uint64_t* bm = reinterpret_cast<const uint64_t*>(blk + 8 * n64);
  const uint16_t* rkk = reinterpret_cast<const uint16_t*>(blk + 8 * n64 + 16 * nw);
  const uint16_t* rkv = reinterpret_cast<const uint16_t*>(blk + 8 * n64 + 16 * nw + round16(2u * nw));
  const int nk = rkk[nw - 1] + __popcll(bm[nw - 1]), nv = rkv[nw - 1] + __popcll(bm[nw + nw - 1]);
  const uint32_t F = tile_fixed_bytes(n);
  const uint32_t sm_k = F, cd_k = F + round16(4u * (uint32_t)nk) + round16(4u * (uint32_t)nv);
  const uint64_t word = bm[tl0 / 64];
  const int rbase = rkk[tl0 / 64];
  const uint8_t* AK = P.arena + d->off_anchor_k;
  const uint32_t* pos = reinterpret_cast<const uint32_t*>(P.arena + d->off_pos);
  __syncthreads();
  // per lane: the turns of the two pair angles it evaluates (lanes 0-15 pairs 0, 1 of their four,
  // lanes 16-31 pairs 2, 3), the rotation signs of its dimensions with the 1/128 folded in
  const bool low = lane < 16;
  const unsigned long long tn0 = turn[(4 * lane + (low ? 0 : 2)) & 63], tn1 = turn[(4 * lane + (low ? 1 : 3)) & 63];
  const float rsgn = low ? -1.f : 1.f;  // y = x cos - x' sin below the partner, x cos + x' sin above
  float sgn128[4];
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const unsigned long long sb = lane < 16 ? P.sign_lo : P.sign_hi;
    sgn128[e] = (P.rotate ? (((sb >> ((4 * lane + e) & 63)) & 1ull) ? -1.f : 1.f) : 1.f) * (P.rotate ? 1.0f / 128.0f : 1.f);
  }
  // the warp's 16 tokens: lane i < 16 fetches token i's stream word and position; every lane then
  // loads its 8 bytes of all 16 anchor rows, and the records of the tokens with a residual, before
  // any arithmetic (the loads do not wait on one another)
  const int tw = tl0 + 16 * warp;
  const int nwt = max(0, min(16, n - tw));  // the warp's tokens inside the tile
  uint32_t ek_l = 0u, pos_l = 0u;
  if (lane < nwt) {
    ek_l = reinterpret_cast<const uint32_t*>(blk)[tw + lane];
    pos_l = pos[j * T + tw + lane];
  }
  uint2 xa[16];
  uint32_t smn[16], cbyte[16];
  const uint32_t wbits = (uint32_t)(word >> (tw % 64)) & 0xFFFFu;  // residual flags of the 16 tokens
#pragma unroll
  for (int i = 0; i < 16; ++i) {
    const uint32_t ek = __shfl_sync(0xffffffffu, ek_l, i);
    const int a = min((int)(ek & 0xFFFFu), k - 1);
    xa[i] = i < nwt ? *reinterpret_cast<const uint2*>(AK + (size_t)a * 256 + 16 * ((lane >> 1) ^ (a & 7)) + 8 * (lane & 1))
                    : make_uint2(0u, 0u);
    smn[i] = 0u;
    cbyte[i] = 0u;
    if (i < nwt && ((wbits >> i) & 1u)) {
      const int r = rbase + __popcll(word & ((1ull << ((tw % 64) + i)) - 1ull));
      smn[i] = *reinterpret_cast<const uint32_t*>(blk + sm_k + 4u * (uint32_t)r);
      cbyte[i] = blk[cd_k + 32u * (uint32_t)r + (uint32_t)lane];
    }
  }
#pragma unroll
  for (int i = 0; i < 16; ++i) {  // (fully unrolled: the per-token arrays stay in registers)
    float y[4] = {0.f, 0.f, 0.f, 0.f};
    const uint32_t ek = __shfl_sync(0xffffffffu, ek_l, i);
    const uint32_t p = __shfl_sync(0xffffffffu, pos_l, i);
    if (i < nwt) {  // (the same for the whole warp)
      const float gk = half_hi(ek);
      float x[4];
      x[0] = gk * __bfloat162float(__ushort_as_bfloat16((unsigned short)(xa[i].x & 0xFFFFu)));
      x[1] = gk * __bfloat162float(__ushort_as_bfloat16((unsigned short)(xa[i].x >> 16)));
      x[2] = gk * __bfloat162float(__ushort_as_bfloat16((unsigned short)(xa[i].y & 0xFFFFu)));
      x[3] = gk * __bfloat162float(__ushort_as_bfloat16((unsigned short)(xa[i].y >> 16)));
      if ((wbits >> i) & 1u) {  // plus r~ = s o H(c^) / 128, c^ = min + scale L[code] (warp-uniform)
        float cr[4];
#pragma unroll
        for (int e = 0; e < 4; ++e)
          cr[e] = fmaf(half_lo(smn[i]), code_level((cbyte[i] >> (2 * e)) & 3u, CODEC), half_hi(smn[i]));
        if (P.rotate) warp_wht128(cr, lane);
#pragma unroll
        for (int e = 0; e < 4; ++e) x[e] = fmaf(cr[e], sgn128[e], x[e]);
      }
      // RoPE at the token's position: lanes 0-15 hold dims j < 64, lanes 16-31 their partners j + 64;
      // the two halves each evaluate two of the four pairs' angles and trade them
      float sa[2], ca[2], sb[2], cb[2];
      __sincosf((float)(uint32_t)(((unsigned long long)p * tn0) >> 40) * (6.2831853071795865f / 16777216.0f), &sa[0], &ca[0]);
      __sincosf((float)(uint32_t)(((unsigned long long)p * tn1) >> 40) * (6.2831853071795865f / 16777216.0f), &sa[1], &ca[1]);
#pragma unroll
      for (int h = 0; h < 2; ++h) {  // the partner half's two angles
        sb[h] = __shfl_xor_sync(0xffffffffu, sa[h], 16);
        cb[h] = __shfl_xor_sync(0xffffffffu, ca[h], 16);
      }
      // pair e of this lane: pairs 0, 1 from the lower half's angles, pairs 2, 3 from the upper half's
      const float sn[4] = {low ? sa[0] : sb[0], low ? sa[1] : sb[1], low ? sb[0] : sa[0], low ? sb[1] : sa[1]};
      const float cs[4] = {low ? ca[0] : cb[0], low ? ca[1] : cb[1], low ? cb[0] : ca[0], low ? cb[1] : ca[1]};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float xp = __shfl_xor_sync(0xffffffffu, x[e], 16);
        y[e] = fmaf(x[e], cs[e], rsgn * xp * sn[e]);
      }
    }
    *reinterpret_cast<float4*>(&ys[16 * warp + i][4 * lane]) = make_float4(y[0], y[1], y[2], y[3]);
  }
  __syncwarp();
  // the warp's 16 logits rows on tensor cores: A = its rotated keys (fp16 high and low parts, from
  // shared memory), B = the query rows (exact in fp16), fp32 sums: D[token][head] (heads >= GS zero)
  {
    const int r8 = lane >> 2, c4 = lane & 3;
    float d[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int ks = 0; ks < 8; ++ks) {
      const float* y0 = &ys[16 * warp + r8][16 * ks + 2 * c4];
      const float* y1 = &ys[16 * warp + r8 + 8][16 * ks + 2 * c4];
      const float2 v[4] = {*reinterpret_cast<const float2*>(y0), *reinterpret_cast<const float2*>(y1),
                           *reinterpret_cast<const float2*>(y0 + 8), *reinterpret_cast<const float2*>(y1 + 8)};
      uint32_t hi[4], lo[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const __half2 h = __float22half2_rn(v[e]);
        const float2 hf = __half22float2(h);
        const __half2 l = __float22half2_rn(make_float2(v[e].x - hf.x, v[e].y - hf.y));
        hi[e] = *reinterpret_cast<const uint32_t*>(&h);
        lo[e] = *reinterpret_cast<const uint32_t*>(&l);
      }
      const bool hv = r8 < GS;  // column n = r8 of B: head r8
      const __half2 b0 = __float22half2_rn(hv ? make_float2(qsm[hv ? r8 : 0][16 * ks + 2 * c4], qsm[hv ? r8 : 0][16 * ks + 2 * c4 + 1])
                                              : make_float2(0.f, 0.f));
      const __half2 b1 = __float22half2_rn(hv ? make_float2(qsm[hv ? r8 : 0][16 * ks + 2 * c4 + 8], qsm[hv ? r8 : 0][16 * ks + 2 * c4 + 9])
                                              : make_float2(0.f, 0.f));
      const uint32_t ub0 = *reinterpret_cast<const uint32_t*>(&b0), ub1 = *reinterpret_cast<const uint32_t*>(&b1);
      mma_f16(d, make_uint4(hi[0], hi[1], hi[2], hi[3]), ub0, ub1);
      mma_f16(d, make_uint4(lo[0], lo[1], lo[2], lo[3]), ub0, ub1);
    }
    // D rows r8, r8 + 8 (tokens), columns 2 c4, 2 c4 + 1 (heads)
    float mx[2] = {-INFINITY, -INFINITY};
#pragma unroll
    for (int hr = 0; hr < 2; ++hr) {
      const int ts = ts0 + 16 * warp + r8 + 8 * hr;
      const bool ok = ts < S;
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int g = 2 * c4 + e;
        const float l = d[2 * hr + e] * P.scale_log2;
        if (ok && g < GS) {
          P.lg[((size_t)u * P.s_stride + ts) * GS + g] = l;
          mx[e] = fmaxf(mx[e], l);
        }
      }
    }
#pragma unroll
    for (int o = 4; o < 32; o <<= 1) {
      mx[0] = fmaxf(mx[0], __shfl_xor_sync(0xffffffffu, mx[0], o));
      mx[1] = fmaxf(mx[1], __shfl_xor_sync(0xffffffffu, mx[1], o));
    }
    if (lane < 4) {
      wmx4[warp][2 * lane] = mx[0];
      wmx4[warp][2 * lane + 1] = mx[1];
    }
  }
  __syncthreads();
  if (tid < GS)
    P.cmax[((size_t)u * P.n_tch + c) * GS + tid] =
        fmaxf(fmaxf(wmx4[0][tid], wmx4[1][tid]), fmaxf(wmx4[2][tid], wmx4[3][tid]));
}

// A lane's tokens of a tile: bitmap bytes and first record indices.
struct TokLane {
  uint32_t kbits, vbits;
  int rk, rv, t0;
};
// What the general token path reads of its tile.
struct TokTile {
  TileView tv;
  uint32_t lo, nrows;
  const float* SAt;   // anchor scores [k][GS]
  const float* rows;  // [0,8): -m, [8,16): -inf, [16,24): sum q'
  const float* qp;    // [GS][128] rotated query
  float* pv;          // [R][8] p rows of the value records
  float* W;           // [X][GS] the tile's value weights
  float* ovf;         // [2][GS][128] overflow sums
  const uint8_t* AV;  // the unit's anchor values (global)
  const float* lgt;   // RoPE at decode: the tile's logit rows [T][GS] (global), else null
  int* ovl_n;         // the tile's overflow lists: value records beyond the staged ones, and runs
  float* ovl;         // beyond the staged anchor-value rows, applied by the whole group after the tokens
  int k, nKs, nVs, ka, lloyd;
};

// The general token path (kept out of line: a tile with records beyond the staged ones, runs
// beyond the staged anchor-value rows, or a lane past the tile's end): the same arithmetic as
// the fast path, with the rare cases on CUDA cores; it returns the lane's share of the
// normaliser (a shared-memory sum would take every lane's addition on the same words).  The
// arguments arrive by value and are copied into locals first: the shared-memory reductions below clobber memory, so a field read
// through the argument itself would be reloaded from its local-memory copy (L2 latency, the
// L1 here being small) after every reduction.
template <int NP>
struct LShare {
  float2 v[NP];
};
template <int GS>
__device__ __noinline__ LShare<(GS >= 2 ? GS / 2 : 1)> token_chunk_general(const TokTile tt_arg, const TokLane tl_arg) {
  constexpr int NP = GS >= 2 ? GS / 2 : 1;
  const TokTile tt = tt_arg;
  const TokLane tl = tl_arg;
  const TileView tv = tt.tv;
  const uint8_t* st = tv.st;
  const uint8_t* gb = tv.gb;
  const uint32_t staged = tv.staged;
  const int t0 = tl.t0;
  const int nvalid = min(LCH, tv.n - t0);
  const float* rsb = reinterpret_cast<const float*>(st + tv.cd_k);
  const float* negrow = tt.rows;
  const float* ninfrow = tt.rows + 8;
  const float* qp = tt.qp;
  const float* SAt = tt.SAt;
  float* W = tt.W;
  float* pv = tt.pv;
  float* ovf = tt.ovf;
  const uint8_t* AV = tt.AV;
  const float* lgt = tt.lgt;
  int* ovl_n = tt.ovl_n;
  float* ovl = tt.ovl;
  const int k = tt.k, nKs = tt.nKs, nVs = tt.nVs, ka = tt.ka, lloyd = tt.lloyd;
  const uint32_t lo = tt.lo;
  const int nrows = (int)tt.nrows;
  int rkn = tl.rk, rvn = tl.rv;
  const uint32_t kbits = tl.kbits, vbits = tl.vbits;
  float2 l2[NP];
#pragma unroll
  for (int i2 = 0; i2 < NP; ++i2) l2[i2] = make_float2(0.f, 0.f);
  uint32_t key = *reinterpret_cast<const uint32_t*>(st + 4 * (tv.n64 + t0)) & 0xFFFFu;
  float2 acc[NP];
#pragma unroll
  for (int i2 = 0; i2 < NP; ++i2) acc[i2] = make_float2(0.f, 0.f);
  auto flush = [&](uint32_t kk, const float2 (&v)[NP]) {
    const int ix = (int)(kk - lo);
    float vv[GS];
#pragma unroll
    for (int g = 0; g < GS; ++g) vv[g] = (g & 1) ? v[g >> 1].y : v[g >> 1].x;
    if (ix < nrows) {
      float* w = W + ix * GS;
#pragma unroll
      for (int g = 0; g < GS; ++g) red_local(w + g, vv[g]);
    } else {  // beyond the staged anchor-value rows: listed for the group (else on CUDA cores here)
      const int e = atomicAdd(ovl_n + 1, 1);
      if (e < kOvl) {
        float* en = ovl + (kOvl + e) * 9;
        en[0] = __int_as_float((int)kk);
#pragma unroll
        for (int g = 0; g < GS; ++g) en[1 + g] = vv[g];
      } else {
        anchor_value_add<GS>(AV, (int)kk, vv, ovf);
      }
    }
  };
  for (int e = 0; e < LCH; ++e) {
    const uint32_t ek = e < nvalid ? *reinterpret_cast<const uint32_t*>(st + 4 * (t0 + e)) : 0u;
    const uint32_t ev = e < nvalid ? *reinterpret_cast<const uint32_t*>(st + 4 * (tv.n64 + t0 + e)) : 0u;
    const int a = min((int)(ek & 0xFFFFu), k - 1);
    float sa[GS], rt[GS];
    if (lgt) {  // RoPE: the token's logits (no anchor-score table)
#pragma unroll
      for (int g = 0; g < GS; ++g) sa[g] = 0.f;
    } else {
      load_sa_row<GS>(SAt, a, ka, sa);
    }
    const bool kb = (kbits >> e) & 1u;
    const int r = rkn;
    rkn += (int)kb;
    if (lgt) {  // RoPE: the logits minus m, or -inf for a token past the tile's end
      load_row<GS>(e >= nvalid ? ninfrow : negrow, rt);
      if (e < nvalid) {
#pragma unroll
        for (int g = 0; g < GS; ++g) rt[g] += lgt[(t0 + e) * GS + g];
      }
    } else if (kb && r >= nKs && e < nvalid) {  // beyond the staged records
#pragma unroll
      for (int g = 0; g < GS; ++g)
        rt[g] = key_record_term(st, gb, staged, tv.sm_k + 4u * (uint32_t)r, tv.cd_k + 32u * (uint32_t)r, qp + g * 128,
                                qp[GS * 128 + g], lloyd) +
                negrow[g];
    } else {  // the key-residual terms minus m, -m, or -inf for a token past the tile's end
      load_row<GS>(e >= nvalid ? ninfrow : negrow, rt);
      if (kb && e < nvalid) {
        float rs[GS];
        load_row<GS>(rsb + r * 8, rs);
#pragma unroll
        for (int g = 0; g < GS; ++g) rt[g] += rs[g];
      }
    }
    const float gk = lgt ? 0.f : half_hi(ek), gv = half_hi(ev);
    float2 pe[NP];
    head_probs<GS, NP>(gk, sa, rt, pe, l2);
    const bool vb = (vbits >> e) & 1u;
    const int rv = rvn;
    rvn += (int)vb;
    if (vb && e < nvalid) {
      if (rv < nVs) {
        store_row<GS>(pv + rv * 8, pe);
      } else {  // beyond the staged records: listed for the group (else on CUDA cores here)
        const int en_i = atomicAdd(ovl_n, 1);
        if (en_i < kOvl) {
          float* en = ovl + en_i * 9;
          en[0] = __int_as_float(rv);
#pragma unroll
          for (int g = 0; g < GS; ++g) en[1 + g] = (g & 1) ? pe[g >> 1].y : pe[g >> 1].x;
        } else {
#pragma unroll
          for (int g = 0; g < GS; ++g)
            value_record_add(st, gb, staged, tv.sm_v + 4u * (uint32_t)rv, tv.cd_v + 512u * (uint32_t)(rv / 16), rv,
                             (g & 1) ? pe[g >> 1].y : pe[g >> 1].x, ovf + GS * 128 + g * 128, lloyd);
        }
      }
    }
    // tokens past the tile join the current run with zero weight
    const uint32_t av = e < nvalid ? (ev & 0xFFFFu) : key;
    if (av != key) {
      flush(key, acc);
      key = av;
#pragma unroll
      for (int i2 = 0; i2 < NP; ++i2) acc[i2] = make_float2(0.f, 0.f);
    }
    const float2 gv2 = make_float2(gv, gv);
#pragma unroll
    for (int i2 = 0; i2 < NP; ++i2) acc[i2] = __ffma2_rn(pe[i2], gv2, acc[i2]);
  }
  flush(key, acc);
  LShare<NP> ls;
#pragma unroll
  for (int i2 = 0; i2 < NP; ++i2) ls.v[i2] = l2[i2];
  return ls;
}

// ================================ decode ============================================
// CODEC: 0 = uniform codes (c^ = min + c scale), 1 = Lloyd-Max levels (c^ = scale L[c]).
// ROPE: 1 = pre-RoPE keys: every token's logit comes from the RoPE logits launch (P.lg) instead
// of gamma S_A plus its key-residual term; the key-residual phase has nothing to do.
template <int GS, int CODEC, int ROPE>
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
  // per group and slot: a tile block and its anchor-value rows landed (full); per unit: its
  // anchor-score table landed (sa_full; a plain arrival when the table stays in global memory)
  auto bar_full = [&](int g, int s) { return smem_u32(bars + g * NSG + s); };
  const uint32_t bar_sa_full = smem_u32(bars + NG * NSG);
  auto bar_hdr = [&](int g) { return smem_u32(bars + NG * NSG + 1 + g); };  // a group's query header landed
  int* segcnt = reinterpret_cast<int*>(smem + P.o_misc + 4);  // groups done with a segment, in total

  if (tid == 0) {
    for (int s = 0; s < NG * NSG + 1 + NG; ++s) mbar_init(smem_u32(bars + s), 1);
    *failed = 0;
    *segcnt = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  for (int e = tid; e < 2 * GS * 128 + 16; e += NT) ovf[e] = 0.f;  // (the CTA's sums start at zero)
  // zeroed p rows: rows past a tile's records are read (and multiplied by zero codes)
  for (int gi = 0; gi < NG; ++gi) {
    float* pvz = reinterpret_cast<float*>(smem + P.o_grp + gi * P.grp_bytes + P.g_pv);
    for (int e = tid; e < P.R * 8; e += NT) pvz[e] = 0.f;
  }
  __syncthreads();

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

  // the first unit's anchor-score table (later ones: the group that finishes the previous unit last)
  auto start_table = [&](int u) {
    const int k = unit_desc(P.arena, u)->n_anchors;
    if (P.smem_sa && !*failed) {
      const float* src = P.sa + (size_t)u * P.ka_stride * GS;
      if (GS == 8) {  // the two four-head arrays, k rows of each
        const uint32_t half = 16u * (uint32_t)k;
        mbar_expect_tx(bar_sa_full, 2 * half);
        bulk_g2s(smem_u32(SAs), src, half, bar_sa_full);
        bulk_g2s(smem_u32(SAs + (size_t)P.ka_stride * 4), src + (size_t)P.ka_stride * 4, half, bar_sa_full);
      } else {
        const uint32_t bytes = round16(4u * (uint32_t)(k * GS));
        mbar_expect_tx(bar_sa_full, bytes);
        bulk_g2s(smem_u32(SAs), src, bytes, bar_sa_full);
      }
    } else {
      mbar_arrive(bar_sa_full);  // the unit's start, for the warps that wait on it
    }
  };
  if (tid == 0) start_table(P.cta_unit[c]);
  const int n_cta_tiles = (int)(B1 - B0);

  // =========================== compute groups ==================================
  const int grp = warp / WPG, wg = warp % WPG, gt = tid - grp * WPG * 32;
  uint8_t* GB = smem + P.o_grp + grp * P.grp_bytes;
  float* qp = reinterpret_cast<float*>(GB + P.g_qp);      // [GS][128] rotated query q'
  float* sq = qp + GS * 128;                              // [8] sums of q' per head
  float* rows = reinterpret_cast<float*>(GB + P.g_rows);  // [0,8): -m, [8,16): -inf, [24,32): m
  int* lastf = reinterpret_cast<int*>(GB + P.g_red);
  float* wb = reinterpret_cast<float*>(GB + P.g_wb);      // [2][X][GS] value weights of a tile's slots
  float* pv = reinterpret_cast<float*>(GB + P.g_pv);      // [R][8] p rows of the value records, then A operands
  int* ovl_n = reinterpret_cast<int*>(GB + P.g_ovl);       // [2] entries in the two overflow lists
  float* ovl = reinterpret_cast<float*>(GB + P.g_ovl + 16);  // [2][kOvl][9]: index bits, then p (or weights) per head
  uint2* qf = reinterpret_cast<uint2*>(GB + P.g_qf);      // [NBF][8][32] key-residual B fragments
  const int bar_id = 1 + grp;
  auto gsync = [&]() { named_sync(bar_id, WPG * 32); };
  constexpr int NBF = GS == 8 ? 2 : 1;  // key-residual fragment sets: GS = 8 keeps high and low parts apart

  float accA[4][4], accR[4][4];  // anchor-value and value-residual sums, dims 32 wg .. 32 wg + 31
  float2 l2[NP];
  float pminv[HPL];
  int lt = 0;  // this group's tiles so far (weight-table buffer parity, stage descriptor)

  // ---- the group as its own producer (warp wg = 0; lane 0 issues the copies) ----
  // Its tiles are the CTA's tiles i = grp, grp + NG, ...; each goes, with the anchor-value rows
  // of the value slots it covers, into this group's half of the ring, oldest first: the tile
  // table entries of the next tile to issue are read one issue ahead, so a copy never waits on
  // a global load.
  const uint32_t RH = ((uint32_t)P.ring_bytes / NG) & ~127u, rbase = (uint32_t)grp * RH;  // 128-byte aligned halves
  Meta* gmeta = meta + grp * NSG;
  Seg si{};                       // segment of the next tile to issue
  int ii = grp;                   // CTA-local index of the next tile to issue
  int nis = 0, nrel = 0;          // tiles issued, tiles released (group-local)
  uint32_t head = 0, used = 0;    // ring bytes: next free place, bytes in flight
  uint32_t pe0 = 0, pe1 = 0, pe2 = 0;  // table entries of tile ii: block offset, next offset, slot range
  int pj = 0;
  const uint8_t* ptiles = nullptr;
  const uint8_t* pav = nullptr;
  auto prefetch = [&]() {
    if (ii >= n_cta_tiles) return;
    while (ii >= si.ib + (si.je - si.jb)) seg_next(si);
    const UnitView V = unit_view(P.arena, si.u);
    pj = si.jb + (ii - si.ib);
    pe0 = V.table[pj];
    pe1 = V.table[pj + 1];
    pe2 = V.table[V.nt + 1 + pj];
    ptiles = V.tiles;
    pav = V.AV;
  };
  auto issue_more = [&]() {
    while (ii < n_cta_tiles && nis - nrel < NSG && !warp_failed(failed)) {
      const uint32_t blkn = pe1 - pe0, lo = pe2 & 0xFFFFu, hi = pe2 >> 16;
      const uint32_t staged = min(blkn, (uint32_t)P.cap);
      const uint32_t nrows = min(hi - lo + 1u, (uint32_t)P.X);
      const uint32_t sz = staged + 256u * nrows;
      uint32_t at = 0;
      bool fits = true;
      if (used == 0) {
        at = 0;
      } else {
        const uint32_t tail = gmeta[nrel % NSG].ring_off - rbase;  // the oldest tile in flight
        if (head > tail) {
          if (head + sz <= RH) at = head;
          else if (sz <= tail) at = 0;
          else fits = false;
        } else if (head < tail) {
          at = head;
          fits = head + sz <= tail;
        } else {
          fits = false;
        }
      }
      if (!fits) break;
      const int sl = nis % NSG;
      if (lane == 0) {
        gmeta[sl] = Meta{rbase + at, pe0, blkn, staged, lo, nrows, (uint32_t)pj, sz};
        // (drop_last: a test withholds the last tile of the range)
        if (P.drop_last > 0 && ii == n_cta_tiles - P.drop_last) {
          gmeta[sl].nrows |= 0x80000000u;  // withheld: nothing in flight
        } else {
          const uint32_t bar = bar_full(grp, sl);
          mbar_expect_tx(bar, sz);
          bulk_g2s(smem_u32(ring + rbase + at), ptiles + pe0, staged, bar);
          if (nrows) bulk_g2s(smem_u32(ring + rbase + at + staged), pav + (size_t)lo * 256, 256u * nrows, bar);
        }
      }
      __syncwarp();
      head = at + sz;
      used += sz;
      ++nis;
      ii += NG;
      prefetch();
    }
  };
  auto release_to = [&](int upto) {  // this group's tiles before `upto` are done with
    for (; nrel < upto; ++nrel) used -= gmeta[nrel % NSG].pad;
  };
  if (wg == 0) {
    seg_begin(si);
    prefetch();
    issue_more();
  }
  Seg sg;
  seg_begin(sg);
  int sigma = 0;
  for (;; ++sigma) {
    const UnitView U = unit_view(P.arena, sg.u);
    const int k = U.k;
    // ---- segment set-up: the unit's query header (q', its sums, key-residual fragments, from
    // the score kernel) by one bulk copy; meanwhile the reference m of each head from the chunk
    // maxima (warp wg: heads wg, wg + 4) ----
    if (wg == 0 && lane == 0) {
      if (!*failed && !ROPE) {  // (RoPE: no key-side header is needed)
        mbar_expect_tx(bar_hdr(grp), (uint32_t)hdr_bytes(GS));
        bulk_g2s(smem_u32(qp), P.uh + (size_t)sg.u * P.uh_stride, (uint32_t)hdr_bytes(GS), bar_hdr(grp));
      } else {
        mbar_arrive(bar_hdr(grp));
      }
    }
    for (int g = wg; g < GS; g += WPG) {
      float m = -INFINITY;
      // the largest anchor score (a lower bound of the largest logit), or with RoPE the largest logit
      const int nch = ROPE ? (U.S + 63) / 64 : (k + CHA - 1) / CHA;
      for (int ch = lane; ch < nch; ch += 32) m = fmaxf(m, P.cmax[((size_t)sg.u * P.n_ch + ch) * GS + g]);
      m = warp_max(m);
      if (lane == 0) {
        rows[g] = -m;
        rows[8 + g] = -INFINITY;
        rows[24 + g] = m;
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
    // the header, then the unit's anchor-score table (every warp waits on both, tiles or not, so
    // the phase counts stay right)
    if (!warp_failed(failed) && !mbar_wait_w(bar_hdr(grp), (uint32_t)sigma & 1u)) *failed = 1;
    if (!warp_failed(failed) && !mbar_wait_w(bar_sa_full, (uint32_t)sigma & 1u)) *failed = 1;
    gsync();  // m of every head written
    const float* SAt = P.smem_sa ? SAs : P.sa + (size_t)sg.u * P.ka_stride * GS;

    const int i_end = sg.ib + (sg.je - sg.jb);
    int i0 = sg.ib + ((grp - sg.ib % NG) + NG) % NG;  // this group's first tile of the segment
    for (int i = i0; i < i_end; i += NG, ++lt) {
      const bool go = !warp_failed(failed) && mbar_wait_w(bar_full(grp, lt % NSG), (uint32_t)(lt / NSG) & 1u);
      if (!go) *failed = 1;
      const Meta mt = gmeta[lt % NSG];
      const uint8_t* st = ring + mt.ring_off;
      TileView tv;
      int nKs = 0, nVs = 0;
      bool fast_tile = false;
      float* W = wb + (lt & 1) * P.X * GS;
      if (go) {
        tv = tile_view(st, mt, U);
        const uint32_t codes_staged = tv.staged > tv.cd_k ? (tv.staged - tv.cd_k) / 32u : 0u;
        nKs = ROPE ? 0 : min(tv.nk, (int)codes_staged);  // their terms go over their own codes: no cap but staging
        nVs = min(tv.nv, P.R);
        fast_tile = (ROPE || nKs == tv.nk) && nVs == tv.nv &&
                    (int)(((reinterpret_cast<const uint32_t*>(st + 4 * tv.n64))[tv.n - 1] & 0xFFFFu) - mt.lo) < (int)mt.nrows;
        for (int e = gt; e < P.X * GS; e += WPG * 32) W[e] = 0.f;
        if (gt < 2) ovl_n[gt] = 0;
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
              const uint4 a = make_uint4(code_pair_h2<CODEC>(xa), code_pair_h2<CODEC>(xb), code_pair_h2<CODEC>(xa >> 2),
                                         code_pair_h2<CODEC>(xb >> 2));
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
                    if (g < GS) rsb[sl * 8 + g] = half_hi(smn) * sq[g] + half_lo(smn) * v[2 * hr + e];
                  }
                }
              }
            }
          }
        }
      }
      gsync();  // (A) key-residual terms written, weight table zeroed
      if (wg == 0) {  // every warp is done with the group's previous tile: its bytes take new ones
        release_to(lt);
        issue_more();
        // the next tile did not fit beside this one (the ring's free bytes are split): it is
        // issued once this tile is done (rare)
        if (lane == 0) lastf[2] = (nis <= lt + 1 && ii < n_cta_tiles) ? 1 : 0;
      }
      if (go) {
        // ---- tokens: lane -> stored tokens t0 .. t0 + 7, every head ----
        const int t0 = wg * (32 * LCH) + LCH * lane;
        TokLane tl;
        if (t0 < tv.n) {
          const int wi = t0 >> 6, sh = t0 & 63;
          const uint64_t wk = tv.bm(0, wi), wv = tv.bm(1, wi);
          tl.kbits = (uint32_t)(wk >> sh) & 0xFFu;
          tl.vbits = (uint32_t)(wv >> sh) & 0xFFu;
          tl.rk = tv.rk(0, wi) + __popcll(wk & ((1ull << sh) - 1ull));
          tl.rv = tv.rk(1, wi) + __popcll(wv & ((1ull << sh) - 1ull));
          tl.t0 = t0;
        }
        if (fast_tile && tv.n == T) {  // warp-uniform
          // A full tile, every record staged, every run on a staged anchor-value row.  No shared
          // atomics: a run that starts and ends inside a lane's tokens is stored as it is (no
          // other lane has its slot); runs that cross lanes are merged by a segmented scan.
          const float* rsb = reinterpret_cast<const float*>(st + tv.cd_k);
          const uint32_t lo = mt.lo;
          const int km1 = k - 1;
          uint32_t kb8 = tl.kbits, vb8 = tl.vbits;
          int rk = tl.rk, rv = tl.rv;
          uint32_t key = *reinterpret_cast<const uint32_t*>(st + 4 * (tv.n64 + t0)) & 0xFFFFu;
          uint32_t hk = key;  // the lane's first run (its head), kept for the merge
          bool multi = false;  // the lane's tokens hold more than one run
          float2 acc[NP], hs[NP];
#pragma unroll
          for (int i2 = 0; i2 < NP; ++i2) acc[i2] = hs[i2] = make_float2(0.f, 0.f);
          float2 negm2[NP];  // -m: the logit offset of every token
#pragma unroll
          for (int i2 = 0; i2 < NP; ++i2) negm2[i2] = make_float2(rows[2 * i2], GS >= 2 ? rows[2 * i2 + 1] : 0.f);
          constexpr int TPI = 4;  // stream words per load (16 bytes)
          // RoPE: the lane's tokens' logit rows (global, stored order)
          const float* lgt = ROPE ? P.lg + ((size_t)sg.u * P.s_stride + (size_t)mt.j * T + t0) * GS : nullptr;
          // the table pointer as shared memory (32-bit addressing, shared loads) or global memory
          auto token_loop = [&](const float* SAtab) {
#pragma unroll 1
          for (int qd = 0; qd < LCH / TPI; ++qd) {
            uint32_t ek[TPI], ev[TPI];
            load_words<TPI>(st + 4 * (t0 + TPI * qd), ek);
            load_words<TPI>(st + 4 * (tv.n64 + t0 + TPI * qd), ev);
#pragma unroll
            for (int e = 0; e < TPI; ++e) {
              const float gv = half_hi(ev[e]);
              float2 x[NP];
              if constexpr (ROPE) {  // the token's logits from the RoPE logits launch, minus m
                float lr[GS];
                load_row<GS>(lgt + (TPI * qd + e) * GS, lr);
#pragma unroll
                for (int i2 = 0; i2 < NP; ++i2)
                  x[i2] = __fadd2_rn(make_float2(lr[2 * i2], GS >= 2 ? lr[2 * i2 + 1] : 0.f), negm2[i2]);
              } else {
                const int a = min((int)(ek[e] & 0xFFFFu), km1);  // indices are < k by construction
                float sa[GS];
                load_sa_row<GS>(SAtab, a, P.ka_stride, sa);
                const bool kb = kb8 & 1u;
                kb8 >>= 1;
                const float gk = half_hi(ek[e]);
                // logits gamma S_A - m, plus the key-residual term for the lanes whose token has one
                const float2 gk2 = make_float2(gk, gk);
#pragma unroll
                for (int i2 = 0; i2 < NP; ++i2)
                  x[i2] = __ffma2_rn(gk2, make_float2(sa[2 * i2], GS >= 2 ? sa[2 * i2 + 1] : 0.f), negm2[i2]);
                if (kb) {
                  float rs[GS];
                  load_row<GS>(rsb + rk * 8, rs);
#pragma unroll
                  for (int i2 = 0; i2 < NP; ++i2)
                    x[i2] = __fadd2_rn(x[i2], make_float2(rs[2 * i2], GS >= 2 ? rs[2 * i2 + 1] : 0.f));
                }
                rk += (int)kb;
              }
              float2 pe[NP];
#pragma unroll
              for (int i2 = 0; i2 < NP; ++i2) {
                pe[i2] = make_float2(exp2_approx(x[i2].x), GS >= 2 ? exp2_approx(x[i2].y) : 0.f);
                l2[i2] = __fadd2_rn(l2[i2], pe[i2]);
              }
              const bool vb = vb8 & 1u;
              vb8 >>= 1;
              if (vb) store_row<GS>(pv + rv * 8, pe);
              rv += (int)vb;
              // the run of `key` ends here when the slot changes (branch-free): the lane's first
              // run is kept as its head (it may continue the previous lane's); a later one started
              // and ended in this lane, so its slot is this lane's alone and is stored as it is
              const uint32_t av = ev[e] & 0xFFFFu;
              const bool chg = av != key;
              if (chg && multi) store_row<GS>(W + (int)(key - lo) * GS, acc);
              const float f_first = (chg && !multi) ? 1.f : 0.f, f_keep = chg ? 0.f : 1.f;
              const float2 first2 = make_float2(f_first, f_first), keep2 = make_float2(f_keep, f_keep);
              const float2 gv2 = make_float2(gv, gv);
#pragma unroll
              for (int i2 = 0; i2 < NP; ++i2) {
                hs[i2] = __ffma2_rn(acc[i2], first2, hs[i2]);
                acc[i2] = __ffma2_rn(pe[i2], gv2, __fmul2_rn(acc[i2], keep2));
              }
              multi |= chg;
              key = av;
            }
          }
          };
          if (ROPE || !P.smem_sa) token_loop(P.sa + (size_t)sg.u * P.ka_stride * GS);  // (RoPE: no table read)
          else token_loop(SAs);
          // merge across lanes: the next lane's head continues this lane's last run when their
          // slots match; a head that does not continue the previous lane's run is complete
          const uint32_t ptk = __shfl_up_sync(0xffffffffu, key, 1);
          const uint32_t nhk = __shfl_down_sync(0xffffffffu, hk, 1);
          const bool nmulti = __shfl_down_sync(0xffffffffu, (int)multi, 1) != 0;
          const float f_tn = (lane < 31 && nmulti && nhk == key) ? 1.f : 0.f;
          const float2 tn2 = make_float2(f_tn, f_tn);
#pragma unroll
          for (int i2 = 0; i2 < NP; ++i2) {
            const float2 nh = make_float2(__shfl_down_sync(0xffffffffu, hs[i2].x, 1),
                                          __shfl_down_sync(0xffffffffu, hs[i2].y, 1));
            acc[i2] = __ffma2_rn(nh, tn2, acc[i2]);
          }
          if (multi && !(lane > 0 && ptk == hk)) {
            float* w = W + (int)(hk - lo) * GS;
            if (lane == 0) {  // may continue the previous warp's last run
#pragma unroll
              for (int g = 0; g < GS; ++g) red_local(w + g, (g & 1) ? hs[g >> 1].y : hs[g >> 1].x);
            } else {
              store_row<GS>(w, hs);
            }
          }
          // segmented inclusive scan of the last runs over lanes with equal slots
#pragma unroll
          for (int d = 1; d < 32; d <<= 1) {
            const uint32_t kd = __shfl_up_sync(0xffffffffu, key, d);
            const float f_add = (lane >= d && kd == key) ? 1.f : 0.f;
            const float2 add2 = make_float2(f_add, f_add);
#pragma unroll
            for (int i2 = 0; i2 < NP; ++i2) {
              const float2 vd = make_float2(__shfl_up_sync(0xffffffffu, acc[i2].x, d),
                                            __shfl_up_sync(0xffffffffu, acc[i2].y, d));
              acc[i2] = __ffma2_rn(vd, add2, acc[i2]);
            }
          }
          const uint32_t nkey = __shfl_down_sync(0xffffffffu, key, 1);
          const uint32_t key0 = __shfl_sync(0xffffffffu, key, 0);
          if (lane == 31 || nkey != key) {  // the last lane of a segment holds its total
            float* w = W + (int)(key - lo) * GS;
            if (lane == 31 || key == key0) {  // the warp's first or last run: shared with a neighbour warp
#pragma unroll
              for (int g = 0; g < GS; ++g) red_local(w + g, (g & 1) ? acc[g >> 1].y : acc[g >> 1].x);
            } else {
              store_row<GS>(w, acc);
            }
          }
        } else if (t0 < tv.n) {
          const auto ls = token_chunk_general<GS>(TokTile{tv, mt.lo, mt.nrows, SAt, rows, qp, pv, W, ovf, U.AV,
                                                      ROPE ? P.lg + ((size_t)sg.u * P.s_stride + (size_t)mt.j * T) * GS : nullptr,
                                                      ovl_n, ovl, k, nKs, nVs, P.ka_stride, CODEC}, tl);
#pragma unroll
          for (int i2 = 0; i2 < NP; ++i2) l2[i2] = __fadd2_rn(l2[i2], ls.v[i2]);
        }
      }
      gsync();  // (B) the tile's weights and p rows are complete
      if (go && !fast_tile) {  // the overflow lists: thread gt takes dimension gt of every entry
        const int nv_o = min(ovl_n[0], kOvl), na_o = min(ovl_n[1], kOvl);
        if (nv_o + na_o > 0) {
          float av[GS], aa[GS];
#pragma unroll
          for (int g = 0; g < GS; ++g) av[g] = aa[g] = 0.f;
          for (int e = 0; e < nv_o; ++e) {  // p (min + scale L(c)) of a value record, rotated domain
            const float* en = ovl + e * 9;
            const uint32_t r = (uint32_t)__float_as_int(en[0]);
            const uint32_t smn = *reinterpret_cast<const uint32_t*>(tv.at(tv.sm_v + 4u * r));
            const uint32_t w = *reinterpret_cast<const uint32_t*>(tv.at(tv.cd_v + 512u * (r / 16u) + 4u * value_code_word(gt)));
            const float val = fmaf(half_lo(smn), code_level((w >> value_code_bit((int)(r % 16u))) & 3u, CODEC), half_hi(smn));
#pragma unroll
            for (int g = 0; g < GS; ++g) av[g] = fmaf(en[1 + g], val, av[g]);
          }
          for (int e = 0; e < na_o; ++e) {  // weight x the anchor's value row (global, swizzled by the slot)
            const float* en = ovl + (kOvl + e) * 9;
            const int kk = __float_as_int(en[0]);
            const uint8_t* row = U.AV + (size_t)kk * 256;
            const float x = __bfloat162float(
                *reinterpret_cast<const __nv_bfloat16*>(row + 16 * ((gt >> 3) ^ (kk & 7)) + 2 * (gt & 7)));
#pragma unroll
            for (int g = 0; g < GS; ++g) aa[g] = fmaf(en[1 + g], x, aa[g]);
          }
#pragma unroll
          for (int g = 0; g < GS; ++g) {
            if (nv_o) red_local(ovf + GS * 128 + g * 128 + gt, av[g]);
            if (na_o) red_local(ovf + g * 128 + gt, aa[g]);
          }
        }
      }
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
              mma_bf16(accR[nb], a.x, a.y, a.z, a.w, code_pair_b2<CODEC>(x), code_pair_b2<CODEC>(x >> 8));
            }
          }
        }
      }
      if (lastf[2]) {  // (written before barrier C by warp 0, the same for every warp)
        gsync();
        if (wg == 0) {
          release_to(lt + 1);
          issue_more();
        }
      }
    }

    // ---- the group's sums for this unit into the CTA's sums in shared memory (anchor-value and
    // rotated value-residual numerators, normaliser, sum of p min); the overflow paths added there
    // already.  Adds of the two groups meet only element by element. ----
    float* cl = ovf + 2 * GS * 128;  // [8] normaliser, then [8] sum of p min, per head
    {
      if (r8 < GS) {
#pragma unroll
        for (int nb = 0; nb < 4; ++nb) {
          const int col = 32 * wg + 8 * nb + 2 * c4;
          red_local(ovf + r8 * 128 + col, accA[nb][0] + accA[nb][2]);
          red_local(ovf + r8 * 128 + col + 1, accA[nb][1] + accA[nb][3]);
          red_local(ovf + GS * 128 + r8 * 128 + col, accR[nb][0] + accR[nb][2]);
          red_local(ovf + GS * 128 + r8 * 128 + col + 1, accR[nb][1] + accR[nb][3]);
        }
      }
#pragma unroll
      for (int g = 0; g < GS; ++g) {
        const float sl = warp_sum((g & 1) ? l2[g >> 1].y : l2[g >> 1].x);
        if (lane == 0) red_local(cl + g, sl);
      }
#pragma unroll
      for (int i2 = 0; i2 < HPL; ++i2) {
        float v = pminv[i2];
#pragma unroll
        for (int o = 1; o < 16; o <<= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
        const int g = (lane >> 4) + 2 * i2;
        if ((lane & 15) == 0 && g < GS) red_local(cl + 8 + g, v);
      }
    }
    if (wg == 0) {  // the segment's last tile is done with: top the ring up
      release_to(lt);
      issue_more();
    }
    // ---- the group that finishes the segment last (the other has added its sums) turns the
    // CTA's sums into its slot of the unit: the value-residual part gets its sum of p min and the
    // inverse rotation (s o H(.) / 128, once per head and CTA), the anchor-value part is added;
    // then it clears the sums, counts the slot in, and starts the next unit's anchor scores ----
    gsync();
    if (gt == 0) {
      __threadfence_block();
      lastf[1] = atomicAdd(segcnt, 1) % NG == NG - 1 ? 1 : 0;
      __threadfence_block();
    }
    gsync();
    const bool has_next = sg.t0 + sg.je < B1;
    if (lastf[1]) {
      float* dst = P.part + (size_t)(c + sg.u) * PF;
      for (int h = wg; h < GS; h += WPG) {
        float4* oa = reinterpret_cast<float4*>(ovf + h * 128 + 4 * lane);
        float4* orr = reinterpret_cast<float4*>(ovf + GS * 128 + h * 128 + 4 * lane);
        const float4 va = *oa, vr = *orr;
        const float pm = cl[8 + h];
        float x[4] = {vr.x + pm, vr.y + pm, vr.z + pm, vr.w + pm};
        if (P.rotate) {
          warp_wht128(x, lane);
          apply_signs(x, lane, P.sign_lo, P.sign_hi);
#pragma unroll
          for (int e = 0; e < 4; ++e) x[e] *= (1.0f / 128.0f);
        }
        *reinterpret_cast<float4*>(dst + h * 128 + 4 * lane) = make_float4(va.x + x[0], va.y + x[1], va.z + x[2], va.w + x[3]);
        *oa = make_float4(0.f, 0.f, 0.f, 0.f);
        *orr = make_float4(0.f, 0.f, 0.f, 0.f);
      }
      gsync();
      if (gt < GS) {
        dst[part_l(GS) + gt] = cl[gt];
        cl[gt] = 0.f;
        cl[8 + gt] = 0.f;
      }
      gsync();
      if (gt == 0) {
        dst[part_flag(GS)] = *failed ? 1.f : 0.f;
        lastf[0] = count_in(P, sg.u, sg.nseg) ? 1 : 0;
        if (has_next) start_table(sg.u + 1);  // the CTA's sums are clear for it
      }
      gsync();
      if (lastf[0]) {
        __threadfence();
        combine_unit<GS>(P, sg.u, sg.first, sg.nseg, wg, WPG);
      }
    }
    gsync();  // lastf and the set-up buffers are reused by the next segment
    if (!has_next) break;
    seg_next(sg);
  }
  // every copy this group started has landed before the CTA may exit (bounded; they all have
  // unless a wait ran out)
  if (wg == 0 && lane == 0) {
    for (int t = max(0, nis - NSG); t < nis; ++t)
      if (!(gmeta[t % NSG].nrows >> 31)) mbar_wait(bar_full(grp, t % NSG), (uint32_t)(t / NSG) & 1u);
    mbar_wait(bar_hdr(grp), (uint32_t)sigma & 1u);
    if (grp == 0) mbar_wait(bar_sa_full, (uint32_t)sigma & 1u);
  }
}

struct DeviceInfo {
  int sms = 0;
  int smem_optin = 0;
  int smem_sm = 0;  // shared memory per SM
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
  cudaDeviceGetAttribute(&d.smem_sm, cudaDevAttrMaxSharedMemoryPerMultiprocessor, dev);
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
  int sms = 0;  // SMs of the device (the score launch: one CTA each)
};

// Shared-memory carve-up for (R, X, table in shared memory or not); false if the ring
// would hold fewer than `min_tiles` of the largest staged tiles per group.
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
  P.o_bar = take((NG * NSG + 1 + NG) * 8);
  P.o_meta = take(NG * NSG * sizeof(Meta));
  P.o_misc = take(16);
  P.o_sa = take(smem_sa ? (size_t)P.ka_stride * GS * 4 : 0);
  P.o_ovf = take((size_t)2 * GS * 128 * 4 + 2 * 8 * 4);  // + normaliser and sum of p min per head
  // a group's block: q' rows, small rows, last flag, two weight tables, p rows / A operands
  size_t g = 0;
  auto gtake = [&](size_t bytes) {
    const size_t o = g;
    g = align128(g + bytes);
    return (int)o;
  };
  P.g_qp = gtake((size_t)hdr_bytes(GS));  // the unit's query header: q', its sums, B fragments
  P.g_qf = P.g_qp + GS * 512 + 32;
  P.g_rows = gtake(32 * 4);
  P.g_red = gtake(16);
  P.g_wb = gtake((size_t)2 * X * GS * 4);
  P.g_pv = gtake((size_t)R * 32);
  P.g_ovl = gtake((size_t)(16 + 2 * kOvl * 9 * 4));  // the tile's overflow lists (counts, then entries)
  P.grp_bytes = (int)g;
  P.o_grp = take((size_t)NG * g);
  P.o_ring = (int)off;
  const long long room = (long long)smem_optin - (long long)P.o_ring - kRingSlack;
  const long long tile_max = (long long)P.cap + 256LL * X;
  if (((room / NG) & ~127LL) < (long long)min_tiles * tile_max) return false;  // each group's part of the ring
  P.ring_bytes = (int)(room & ~127LL);
  out->smem = (size_t)P.o_ring + (size_t)P.ring_bytes + kRingSlack;
  return true;
}

// Preference: the anchor-score table in shared memory (the token gathers' fast path), with
// room for two, then one of the largest staged tiles in each group's half of the ring, staged
// counts trimmed from their full values towards the mean (records first, then anchor-value
// rows: a run beyond those takes the slowest fallback); then the table in global memory
// (gathers through L1 and L2) the same way; then anything that holds one tile per group.
// table false: no anchor-score table is read (RoPE at decode), so none is placed in shared memory.
bool make_plan(const Layout& L, int GS, int smem_optin, bool table, Plan* out, std::string* why) {
  const int R0 = full_r(L), X0 = full_x(L);
  const int Rmin = std::max(16, ((R0 * 3 / 4) + 15) & ~15), Xmin = std::max(16, ((X0 * 3 / 4) + 15) & ~15);
  for (int sa = table ? 1 : 0; sa >= 0; --sa)
    for (int min_tiles : {2, 1})
      for (int X = X0; X >= Xmin; X -= 16)
        for (int R = R0; R >= Rmin; R -= 16)
          if (make_plan_rx(L, GS, R, X, sa == 1, smem_optin, min_tiles, out)) return true;
  for (int min_tiles : {1})
    for (int X = X0; X >= 16; X -= 16)
      for (int R = R0; R >= 16; R -= 16)
        if (make_plan_rx(L, GS, R, X, false, smem_optin, min_tiles, out)) return true;
  *why = "shared memory: no room for the decode pipeline";
  return false;
}

using DecodeFn = void (*)(const DecodeParams);
using ScoreFn = void (*)(const ScoreParams);
using ScoreTcFn = void (*)(const ScoreParams, const CUtensorMap, const CUtensorMap);
using RopeFn = void (*)(const RopeParams);
template <int GS>
DecodeFn decode_kernel(int codec, int rope) {
  if (rope) return codec ? akv_decode_kernel<GS, 1, 1> : akv_decode_kernel<GS, 0, 1>;
  return codec ? akv_decode_kernel<GS, 1, 0> : akv_decode_kernel<GS, 0, 0>;
}
template <int GS>
RopeFn rope_kernel(int codec) {
  return codec ? akv_rope_logits_kernel<GS, 1> : akv_rope_logits_kernel<GS, 0>;
}
template <int GS>
ScoreTcFn score_kernel() {
  return akv_scores_tc_kernel<GS>;
}

// cuTensorMapEncodeTiled of the driver, found once through the runtime (no link to libcuda).
PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static std::once_flag once;
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  std::call_once(once, [] {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q = cudaDriverEntryPointSymbolNotFound;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = (PFN_cuTensorMapEncodeTiled_v12000)f;
  });
  return fn;
}

// A 2-D map over `rows` rows of 128 bf16 (256 bytes apart) at `base` (16-byte aligned), copied
// as boxes of 64 elements (one 128-byte half) x box_rows rows; rows past the end read as zero.
bool encode_row_map(CUtensorMap* m, const void* base, uint64_t rows, uint32_t box_rows, CUtensorMapSwizzle sw) {
  const PFN_cuTensorMapEncodeTiled_v12000 enc = tensor_map_encoder();
  if (!enc || rows == 0) return false;
  const cuuint64_t dims[2] = {128, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {256};
  const cuuint32_t box[2] = {64, box_rows};
  const cuuint32_t estr[2] = {1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}
template <int GS>
ScoreFn suffix_kernel(bool rope) {
  return rope ? akv_suffix_kernel<GS, true> : akv_suffix_kernel<GS, false>;
}

// Launch configuration per (device, G, layout shape): computed once, then reused, so that a
// call made during CUDA-graph capture only issues the launches.
struct LaunchKey {
  int dev, G, codec, rope, units, max_len, max_k, ctas;
  long long dens_key, adens_key, ttot;
  bool operator<(const LaunchKey& o) const {
    return std::tie(dev, G, codec, rope, units, max_len, max_k, ctas, dens_key, adens_key, ttot) <
           std::tie(o.dev, o.G, o.codec, o.rope, o.units, o.max_len, o.max_k, o.ctas, o.dens_key, o.adens_key, o.ttot);
  }
};

}  // namespace

std::atomic<int> g_debug_cluster{0}, g_debug_withhold{0};
namespace {
std::mutex g_events_mu;
cudaEvent_t g_ev_scores = nullptr, g_ev_decode = nullptr;
}  // namespace
void set_decode_events(void* after_scores, void* after_decode) {
  std::lock_guard<std::mutex> lk(g_events_mu);
  g_ev_scores = (cudaEvent_t)after_scores;
  g_ev_decode = (cudaEvent_t)after_decode;
}

// Workspace of a decode call: anchor scores, chunk maxima, arrival counters, partial slots.
DecodeWs decode_ws_layout(const Layout& L, int32_t suffix_cap) {
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
  const bool rope = (L.header.params.flags & AKV_FLAG_ROPE) != 0;
  const size_t s_stride = (size_t)((L.max_len + 63) & ~63);
  w.o_sa = take(rope ? 0 : units * ka * (size_t)L.G * 4);
  w.o_uh = take(units * (size_t)((hdr_bytes(L.G) + 255) & ~255));
  // chunk maxima: of 64 anchors, or with RoPE of 64 stored tokens
  w.o_cmax = take(units * (rope ? s_stride / 64 : nch) * (size_t)L.G * 4);
  w.o_lg = take(rope ? units * s_stride * (size_t)L.G * 4 : 0);  // RoPE: every token's logits
  w.o_cnt = take(units * 4);
  w.o_part = take((size_t)(kMaxGrid + units) * (size_t)part_floats(L.G) * 4);
  w.o_suf = take(units * (size_t)((suffix_cap + SCH - 1) / SCH) * (size_t)suf_floats(L.G) * 4);
  w.total = off;
  return w;
}

template <int GS>
int launch_g(const Layout& L, const akv_params& p, const void* arena, size_t arena_bytes, const void* q, void* out, float* out_f32,
             float sm_scale, const DecodeSuffix& sfx, void* ws, void* stream, std::string* why) {
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
  const int codec = (p.flags & AKV_FLAG_LLOYD) ? 1 : 0;
  const int rope = (p.flags & AKV_FLAG_ROPE) ? 1 : 0;
  const LaunchKey key{dev, L.G, codec, rope, units, L.max_len, L.max_k, ctas, (long long)(max_density(L) * 1e6),
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
    cudaError_t e =
        cudaFuncSetAttribute(decode_kernel<GS>(codec, rope), cudaFuncAttributeMaxDynamicSharedMemorySize, di.smem_optin);
    if (e != cudaSuccess) return (int)e;
    if (!make_plan(L, GS, di.smem_optin, !rope, &pl, why)) return -1;
    if ((e = cudaFuncSetAttribute(score_kernel<GS>(), cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  (int)kScDynSmem)) != cudaSuccess)  // the score launch's stages
      return (int)e;
    int grid = (int)std::min<long long>(std::min(di.sms, kMaxGrid), ttot);
    if (ctas > 0) grid = (int)std::min<long long>(ctas, ttot);
    pl.grid = grid;
    pl.sms = di.sms;
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
    // chunk maxima per unit: of 64 anchors, or with RoPE of 64 stored tokens
    pl.P.n_ch = rope ? (L.max_len + 63) / 64 : (L.max_k + CHA - 1) / CHA;
    std::lock_guard<std::mutex> lk(mu);
    cache[key] = pl;
  }
  const DecodeWs W = decode_ws_layout(L, sfx.cap);
  const int n_sch = sfx.K ? (sfx.cap + SCH - 1) / SCH : 0;
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
  P.uh = wsb + W.o_uh;
  P.uh_stride = (hdr_bytes(GS) + 255) & ~255;
  P.n_kv_heads = p.n_kv_heads;
  P.n_q_heads = p.n_q_heads;
  P.rotate = (p.flags & AKV_FLAG_ROTATE) ? 1 : 0;
  P.scale_log2 = sm_scale * kLog2e;
  P.sign_lo = L.header.sign_bits[0];
  P.sign_hi = L.header.sign_bits[1];
  P.drop_last = drop;
  P.lg = rope ? (const float*)(wsb + W.o_lg) : nullptr;
  P.s_stride = (L.max_len + 63) & ~63;
  P.suf_part = n_sch ? (const float*)(wsb + W.o_suf) : nullptr;
  P.suf_len = sfx.len;
  P.suf_cap = sfx.cap;
  P.n_sch = n_sch;

  ScoreParams S;
  S.arena = P.arena;
  S.q = P.q;
  S.sa = (float*)(wsb + W.o_sa);
  S.cmax = (float*)(wsb + W.o_cmax);
  S.cnt = P.cnt;
  S.n_kv_heads = p.n_kv_heads;
  S.n_q_heads = p.n_q_heads;
  S.G = L.G;
  S.ksuf = (const __nv_bfloat16*)sfx.K;
  S.vsuf = (const __nv_bfloat16*)sfx.V;
  S.suf_len = sfx.len;
  S.suf_part = (float*)(wsb + W.o_suf);
  S.suf_cap = sfx.cap;
  S.n_sch = n_sch;
  S.ka_stride = P.ka_stride;
  S.n_ch = P.n_ch;
  S.scale_log2 = P.scale_log2;
  S.uh = wsb + W.o_uh;
  S.uh_stride = P.uh_stride;
  S.rotate = P.rotate;
  S.sign_lo = P.sign_lo;
  S.sign_hi = P.sign_hi;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(units * P.n_ch), 1, 1);
  cfg.blockDim = dim3(128, 1, 1);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = (cudaStream_t)stream;
  cudaEvent_t ev_scores = nullptr, ev_decode = nullptr;
  {
    std::lock_guard<std::mutex> lk(g_events_mu);
    ev_scores = g_ev_scores;
    ev_decode = g_ev_decode;
  }
  cudaError_t e;
  if (rope) {  // the logits of every stored token (no anchor scores)
    RopeParams R;
    R.arena = P.arena;
    R.q = P.q;
    R.lg = (float*)(wsb + W.o_lg);
    R.cmax = (float*)(wsb + W.o_cmax);
    R.cnt = P.cnt;
    R.n_kv_heads = p.n_kv_heads;
    R.n_q_heads = p.n_q_heads;
    R.rotate = P.rotate;
    R.lloyd = codec;
    R.s_stride = P.s_stride;
    R.n_tch = P.n_ch;
    R.scale_log2 = P.scale_log2;
    R.sign_lo = P.sign_lo;
    R.sign_hi = P.sign_hi;
    // theta_j / (2 pi) < 1 as a 64-bit binary fraction of a turn (truncated past 2^-64)
    for (int j = 0; j < 64; ++j)
      R.turn[j] = (unsigned long long)std::ldexp(
          std::pow((double)p.rope_theta, -2.0 * (double)j / 128.0) / 6.283185307179586476925, 64);
    cfg.gridDim = dim3((unsigned)(units * P.n_ch), 1, 1);
    e = cudaLaunchKernelEx(&cfg, rope_kernel<GS>(codec), R);
    for (int j = 0; j < 64; ++j) S.turn[j] = R.turn[j];
  } else {
    // anchor rows of every unit through one map over the caller's arena as 256-byte rows (each
    // unit's anchor-key section starts its 256-byte-aligned segment; a full-selection arena places
    // its units by the budgets it chose, past the plain layout's size), query rows through one over q
    CUtensorMap tmA, tmB;
    if (!encode_row_map(&tmA, arena, arena_bytes / 256, kScTile, CU_TENSOR_MAP_SWIZZLE_NONE) ||
        !encode_row_map(&tmB, q, (uint64_t)p.batch * (uint64_t)p.n_q_heads, 16, CU_TENSOR_MAP_SWIZZLE_128B)) {
      *why = "(tensor maps of the score launch could not be encoded)";
      return -1;
    }
    S.units = units;
    S.n_t = (P.n_ch + 1) / 2;
    S.arena_rows = (long long)(arena_bytes / 256);
    // persistent, one CTA per SM over the units' anchor tiles (more CTAs, one after another on an
    // SM, when one CTA would take more tiles than its table holds)
    const long long n_tiles = (long long)units * S.n_t;
    cfg.gridDim = dim3((unsigned)std::max<long long>({1, std::min<long long>(n_tiles, pl.sms),
                                                      (n_tiles + kScMaxTiles - 1) / kScMaxTiles}), 1, 1);
    cfg.blockDim = dim3(kScThreads, 1, 1);
    cfg.dynamicSmemBytes = kScDynSmem;
    e = cudaLaunchKernelEx(&cfg, score_kernel<GS>(), S, tmA, tmB);
    cfg.blockDim = dim3(128, 1, 1);
    cfg.dynamicSmemBytes = 0;
  }
  if (e == cudaSuccess && n_sch) {  // the dense suffix's chunks (with RoPE: keys turned to positions S + t)
    cfg.gridDim = dim3((unsigned)(units * n_sch), 1, 1);
    cfg.dynamicSmemBytes = (size_t)SCH * 256;  // a chunk's value rows
    e = cudaLaunchKernelEx(&cfg, suffix_kernel<GS>(rope != 0), S);
    cfg.dynamicSmemBytes = 0;
  }
  if (e != cudaSuccess) return (int)e;
  if (ev_scores && (e = cudaEventRecord(ev_scores, cfg.stream)) != cudaSuccess) return (int)e;
  cfg.gridDim = dim3((unsigned)pl.grid, 1, 1);
  cfg.blockDim = dim3(NT, 1, 1);
  cfg.dynamicSmemBytes = pl.smem;
  e = cudaLaunchKernelEx(&cfg, decode_kernel<GS>(codec, rope), P);
  if (e != cudaSuccess) {
    cudaFuncAttributes fa{};
    cudaFuncGetAttributes(&fa, decode_kernel<GS>(codec, rope));
    *why = "(decode kernel: " + std::to_string(fa.numRegs) + " registers, max " + std::to_string(fa.maxThreadsPerBlock) +
           " threads, " + std::to_string(pl.smem) + " B dynamic shared memory of " +
           std::to_string(fa.maxDynamicSharedSizeBytes) + ", grid " + std::to_string(pl.grid) + ")";
    return (int)e;
  }
  if (ev_decode && (e = cudaEventRecord(ev_decode, cfg.stream)) != cudaSuccess) return (int)e;
  return (int)cudaGetLastError();
}

int launch_decode(const Layout& L, const akv_params& p, const void* arena, size_t arena_bytes, const void* q, void* out, float* out_f32,
                  float sm_scale, const DecodeSuffix& sfx, void* ws, void* stream, std::string* why) {
  switch (L.G) {
    case 1: return launch_g<1>(L, p, arena, arena_bytes, q, out, out_f32, sm_scale, sfx, ws, stream, why);
    case 2: return launch_g<2>(L, p, arena, arena_bytes, q, out, out_f32, sm_scale, sfx, ws, stream, why);
    case 4: return launch_g<4>(L, p, arena, arena_bytes, q, out, out_f32, sm_scale, sfx, ws, stream, why);
    case 8: return launch_g<8>(L, p, arena, arena_bytes, q, out, out_f32, sm_scale, sfx, ws, stream, why);
  }
  *why = "unsupported group size";
  return -1;
}

// The append path of the dense suffix (Appendix E.2): CTA b copies the new key and value rows of
// request b's KV heads to row len[b] of their suffix blocks, then counts the token in.  Every
// thread reads len[b] before the barrier; thread 0 writes it after.
__global__ void __launch_bounds__(256) akv_suffix_append_kernel(int H, const uint4* K_new, const uint4* V_new,
                                                                 uint4* K_suf, uint4* V_suf, int32_t* len, int cap) {
  const int b = blockIdx.x;
  const int n = len[b];
  const bool room = n >= 0 && n < cap;
  if (room) {
    for (int e = threadIdx.x; e < H * 16; e += blockDim.x) {  // 16 x 16 bytes per row
      const size_t row = (size_t)b * H + e / 16;
      K_suf[(row * cap + n) * 16 + e % 16] = K_new[row * 16 + e % 16];
      V_suf[(row * cap + n) * 16 + e % 16] = V_new[row * 16 + e % 16];
    }
  }
  __syncthreads();
  if (threadIdx.x == 0 && room) len[b] = n + 1;
}

int launch_suffix_append(int32_t B, int32_t H, const void* K_new, const void* V_new, void* K_suf, void* V_suf,
                         int32_t* len, int32_t cap, void* stream) {
  akv_suffix_append_kernel<<<B, 256, 0, (cudaStream_t)stream>>>(H, (const uint4*)K_new, (const uint4*)V_new,
                                                                (uint4*)K_suf, (uint4*)V_suf, len, cap);
  return (int)cudaGetLastError();
}

const char* cuda_error_string(int err) { return cudaGetErrorString((cudaError_t)err); }

}  // namespace akv
