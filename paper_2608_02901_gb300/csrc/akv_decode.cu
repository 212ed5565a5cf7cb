// Split-K decode attention read directly from the AnchorKV compressed cache.
//
// One thread-block cluster per (request, KV head) -- for G = 8, when eight heads' tables do
// not fit, per (request, KV head, four query heads); its C CTAs split the unit's tile blocks
// and its anchors.  Eq. 3 is folded into Eq. 4: no key or value row is ever rebuilt in
// memory.
//
// Warp-specialised CTA (16 warps):
//   producer warp     one elected lane streams a sequence of items through a ring of
//                     shared-memory stages, one bulk asynchronous copy per item, each
//                     completing a transaction-counted mbarrier:
//                     [anchor-key chunks] [tile blocks] [anchor-value chunks]
//   3 key-residual warps  first the rotated query q' = H(s o q)/128 (Appendix A.1, Eq. 12;
//                     a warp-local Walsh-Hadamard transform) and its fp16 high + low
//                     fragments; then per tile: q' . c for the staged key records on tensor
//                     cores, straight from the packed 2-bit codes
//   8 token warps     phase 1: anchor scores S_A = q . k_a of the CTA's anchor slice (bf16
//                     tensor cores), pushed into every peer's table (DSMEM stores);
//                     per tile: logits gamma_i S_A[a(i)] + residual term, p = 2^(l - m),
//                     the value-residual warps' p, and the value weights
//                     w[a] = sum_i p_i gamma_i (Eq. 3) -- tokens are stored sorted by
//                     value anchor, so w is a sum over runs: per lane its head and tail
//                     runs, merged across lanes by a warp segmented scan, one shared-memory
//                     reduction per run into the CTA's own table of the value slots its
//                     tiles cover (a slot at the edge of two CTAs' tiles gets a share in
//                     each: the products add up);
//                     phase 3: the anchor-value product over those slots, the inverse
//                     rotation of the value-residual sum, cluster combine
//   4 value-residual warps  per tile: sum of (p scale) c over the staged value records on
//                     tensor cores, in the rotated domain
// Stages are handed between the roles with mbarriers, so different roles work on
// different tiles at the same time.
//
// The exponent reference m is the largest anchor score of each query row.  Anchors
// are tokens of the unit, so it is a lower bound of the largest logit (sums cannot
// overflow unless a logit exceeds m by more than 2^120, which is flagged), and all
// CTAs of a cluster share it: no running-max rescaling is needed and the cluster
// combine (Eq. 4 normaliser and numerator) is a plain sum.
// Every wait on an mbarrier is bounded; a wait that runs out marks the CTA failed,
// the CTA stops issuing and consuming, and its outputs become NaN.
#include <cooperative_groups.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <cstdio>
#include <cstdlib>
#include <map>
#include <mutex>
#include <queue>
#include <vector>
#include <string>
#include <tuple>
#include <type_traits>

#include "akv_internal.h"

namespace cg = cooperative_groups;

namespace akv {
namespace {

// warp roles
constexpr int NTW = 8;                 // token warps (warps 0 .. 7)
constexpr int NTT = NTW * 32;          // token threads
constexpr int NKR = 3;                 // key-residual warps: 10, 11, 15
constexpr int NVR = 4;                 // value-residual warps: 8, 9, 12, 13
constexpr int W_PROD = 14;             // producer warp
constexpr int NT = 16 * 32;            // 512 threads: four warpgroups
// A warp issues on sub-partition (warp % 4): each sub-partition carries two token warps and
// two of the others.
__device__ __forceinline__ int kres_index(int warp) { return warp == 10 ? 0 : warp == 11 ? 1 : warp == 15 ? 2 : -1; }
__device__ __forceinline__ int vres_index(int warp) {
  return warp == 8 ? 0 : warp == 9 ? 1 : warp == 12 ? 2 : warp == 13 ? 3 : -1;
}
static_assert(NTW == 8 && NKR == 3 && NVR == 4 && W_PROD == 14, "role placement above assumes 8 + 3 + 4 + 1 warps");
constexpr int T = kTile;               // tokens per tile block
constexpr int REG = T / NTW;           // tokens of a tile per token warp
static_assert(REG == 128, "a token lane's chunk (REG * GS / 32 tokens) lies in one bitmap word");
static_assert(NTW % NVR == 0, "value-residual warps release a stage with NTW / NVR arrivals each");
constexpr int CH = 80;                 // anchor rows per chunk item (a multiple of 16)
constexpr int kMaxCluster = 16;
constexpr unsigned long long kWaitNs = 2000000000ull;  // an mbarrier wait gives up after 2 s
constexpr float kLog2e = 1.4426950408889634f;
constexpr uint32_t F_MAX = tile_fixed_bytes(T);  // streams, bitmaps, rank words of a full tile

struct DecodeParams {
  const uint8_t* arena;
  const __nv_bfloat16* q;
  __nv_bfloat16* out;
  float* out_f32;
  int n_kv_heads, n_q_heads, G, nhg, cluster, rotate;
  float scale_log2;
  unsigned long long sign_lo, sign_hi;
  int R, NS, stage_bytes, cap;
  int o_sa, o_w, o_qfa, o_qfk, o_qp, o_acc, o_opart, o_misc, o_meta, o_bar, o_ring;
  int o_pfb;       // value-residual operands, two buffers (tiles alternate)
  int o_rs, o_pv;  // inside a stage: key-residual terms, p of the value-record tokens
  int o_hdr;       // [NS][2] uint4: tile header per stage (put_header)
  int o_mslot;     // [kMaxCluster][GS] largest anchor score of each CTA's slice, per head
  int o_lslot;     // [kMaxCluster][GS] each CTA's normaliser share
  int o_fslot;     // [kMaxCluster] each CTA's failure flag
  int o_ofin;      // [C][per] staging: partial output numerators of this CTA's share, per rank
  int drop_last;   // test hook: the producer withholds its tile item n_kas + n_t - drop_last (0: none)
  int o_ovf;       // [GS][128] anchor-value products of runs beyond the value-weight table
  int wrows;       // rows of the value-weight table (value slots o0 .. o0 + wrows - 1)
};

// ---- device helpers ---------------------------------------------------------------

__device__ __forceinline__ uint32_t smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ void mbar_arrive_cnt(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
// One arrival that also announces `bytes` of transactions the bulk copies will complete.
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}
// Test for completion of the phase with the given parity (the hardware may hold the thread
// for a short while before answering no).  A longer sleep hint measured slower: waking on
// completion lags behind polling.
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
// Bounded wait of one thread for completion of the phase with the given parity; false if
// kWaitNs passed first (the clock is read every 64 tries, so a try costs a few instructions).
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity) {
  if (mbar_try(bar, parity)) return true;
  const unsigned long long t0 = global_ns();
  for (unsigned i = 1;; ++i) {
    if (mbar_try(bar, parity)) return true;
    if ((i & 63u) == 0 && global_ns() - t0 >= kWaitNs) return false;
  }
}
// The same by a whole warp: every lane observes the completion itself (its acquire), and
// all lanes return together with the same result (the clock is lane 0's).
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
__device__ __forceinline__ void tw_sync() { asm volatile("bar.sync 1, %0;" ::"n"(NTT) : "memory"); }
__device__ __forceinline__ void named_sync(int id, int n) { asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(n) : "memory"); }
__device__ __forceinline__ void named_arrive(int id, int n) {
  asm volatile("bar.arrive %0, %1;" ::"r"(id), "r"(n) : "memory");
}
// Programmatic dependent launch: the next launch in the stream may be scheduled, and set up
// its shared memory and barriers, while this one runs; before it reads the cache
// or the query, or writes an output, every thread waits for the preceding work to complete.
__device__ __forceinline__ void pdl_allow_next() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void pdl_wait_prev() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void cluster_arrive() { asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory"); }
__device__ __forceinline__ void cluster_wait() { asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory"); }
// A row of GS floats (16-byte aligned for GS >= 4, else 8 or 4) stored into the same place in the shared
// memory of CTA `rank` of the cluster.
template <int GS>
__device__ __forceinline__ void st_cluster_row(const float* local, int rank) {
  uint32_t remote;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(smem_u32(local)), "r"(rank));
  if constexpr (GS == 8) {
    const float4 v = *reinterpret_cast<const float4*>(local), w = *reinterpret_cast<const float4*>(local + 4);
    asm volatile("st.shared::cluster.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(remote), "f"(v.x), "f"(v.y), "f"(v.z), "f"(v.w)
                 : "memory");
    asm volatile("st.shared::cluster.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(remote + 16u), "f"(w.x), "f"(w.y), "f"(w.z),
                 "f"(w.w)
                 : "memory");
  } else if constexpr (GS == 4) {
    const float4 v = *reinterpret_cast<const float4*>(local);
    asm volatile("st.shared::cluster.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(remote), "f"(v.x), "f"(v.y), "f"(v.z), "f"(v.w)
                 : "memory");
  } else if constexpr (GS == 2) {
    const float2 v = *reinterpret_cast<const float2*>(local);
    asm volatile("st.shared::cluster.v2.f32 [%0], {%1, %2};" ::"r"(remote), "f"(v.x), "f"(v.y) : "memory");
  } else {
    asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(remote), "f"(local[0]) : "memory");
  }
}
// v stored at the place of `local` in the shared memory of CTA `rank` of the cluster.
__device__ __forceinline__ void st_cluster_v4(const float* local, int rank, float4 v) {
  uint32_t remote;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(smem_u32(local)), "r"(rank));
  asm volatile("st.shared::cluster.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(remote), "f"(v.x), "f"(v.y), "f"(v.z), "f"(v.w)
               : "memory");
}
// An int stored into the same place in the shared memory of CTA `rank` of the cluster.
__device__ __forceinline__ void st_cluster_int(const int* local, int rank) {
  uint32_t remote;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(smem_u32(local)), "r"(rank));
  asm volatile("st.shared::cluster.s32 [%0], %1;" ::"r"(remote), "r"(local[0]) : "memory");
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

// Two 2-bit codes, at bits 0-1 and 16-17 of x, as an fp16 pair of exact small integers: OR
// them into the mantissa of 1024.0 (0x6400, unit spacing), then subtract 1024.  (Leaving the
// 1024 in and taking 1024 x sum(q') off afterwards saves the subtraction but costs the
// tensor-core sums about two decimal digits: they do not hold full fp32 precision against an
// offset that large.)
__device__ __forceinline__ uint32_t codes2_to_h2(uint32_t x) {
  uint32_t t, r;
  asm("lop3.b32 %0, %1, %2, %3, 0xEA;" : "=r"(t) : "r"(x), "r"(0x00030003u), "r"(0x64006400u));
  asm("sub.f16x2 %0, %1, %2;" : "=r"(r) : "r"(t), "r"(0x64006400u));
  return r;
}
// Two 2-bit codes as the exact bf16 pair c: OR into the mantissa of 128.0 (0x4300, unit
// spacing), then t * 1 - 128.  (The value-residual sum runs over many more products than a
// key term, so it keeps exact operands: an offset there would cost fp32 accuracy.)
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
__device__ __forceinline__ float2 f2mul(float2 a, float2 b) {
  unsigned long long ra, rb, rd;
  asm("mov.b64 %0, {%1, %2};" : "=l"(ra) : "f"(a.x), "f"(a.y));
  asm("mov.b64 %0, {%1, %2};" : "=l"(rb) : "f"(b.x), "f"(b.y));
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(rd) : "l"(ra), "l"(rb));
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

// Sections of one unit.
struct UnitView {
  int S, k, nt;
  const uint8_t* AK;
  const uint8_t* AV;
  const uint32_t* table;
  const uint8_t* tiles;
};

__device__ __forceinline__ UnitView unit_view(const uint8_t* A, int u) {
  const akv_unit_desc* d = reinterpret_cast<const akv_unit_desc*>(A + 256) + u;
  UnitView v;
  v.S = d->len;
  v.k = d->n_anchors;
  v.nt = d->n_tiles;
  v.AK = A + d->off_anchor_k;
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

// `meta` = {block offset, block bytes} as the producer recorded them for this stage.
__device__ __forceinline__ TileView tile_view(const uint8_t* st, const uint2 meta, const UnitView& U, int j, int cap) {
  TileView v;
  v.st = st;
  v.gb = U.tiles + meta.x;
  v.staged = min(meta.y, (uint32_t)cap);
  v.n = min(T, U.S - j * T);
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

// A tile block's header as the key-residual warps publish it per stage (two 16-byte words:
// block offset, block bytes, n | nw << 16, nk | nv << 16, then the four section offsets), so
// that the token and value-residual warps skip the dependent loads of tile_view.
__device__ __forceinline__ void put_header(uint4* hdr, const TileView& v, uint2 meta) {
  const int lane = threadIdx.x & 31;
  if (lane == 0)
    hdr[0] = make_uint4(meta.x, meta.y, (uint32_t)v.n | ((uint32_t)v.nw << 16), (uint32_t)v.nk | ((uint32_t)v.nv << 16));
  if (lane == 1) hdr[1] = make_uint4(v.sm_k, v.sm_v, v.cd_k, v.cd_v);
}
__device__ __forceinline__ TileView header_view(const uint8_t* st, const uint4* hdr, const UnitView& U, int cap, uint2* meta_out) {
  const uint4 h0 = hdr[0], h1 = hdr[1];
  TileView v;
  v.st = st;
  v.gb = U.tiles + h0.x;
  v.staged = min(h0.y, (uint32_t)cap);
  v.n = (int)(h0.z & 0xFFFFu);
  v.nw = (int)(h0.z >> 16);
  v.n64 = 64 * v.nw;
  v.nk = (int)(h0.w & 0xFFFFu);
  v.nv = (int)(h0.w >> 16);
  v.sm_k = h1.x;
  v.sm_v = h1.y;
  v.cd_k = h1.z;
  v.cd_v = h1.w;
  *meta_out = make_uint2(h0.x, h0.y);
  return v;
}

// Records beyond the staged count (a locally dense tile) take these rare paths on CUDA
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
// accg += ps * c of value record r (rotated domain); value codes are dimension-major
// groups of 16 records.
__device__ __noinline__ void value_record_add(const TileView& tv, int r, float ps, float* accg) {
  const uint32_t base = tv.cd_v + 512u * (uint32_t)(r / 16);
  for (int d = 0; d < 128; ++d) {
    const uint32_t w = *reinterpret_cast<const uint32_t*>(tv.at(base + 4u * value_code_word(d)));
    atomicAdd(&accg[d], ps * (float)((w >> value_code_bit(r % 16)) & 3u));
  }
}

// GS probabilities (pairs) as one row of GS floats (16-byte aligned for GS >= 4, else 8 or 4).
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

template <int GS>
__global__ void __launch_bounds__(NT, 1) akv_decode_kernel(const DecodeParams P) {
  extern __shared__ __align__(128) uint8_t smem[];
  cg::cluster_group cluster = cg::this_cluster();
  const int C = P.cluster;
  const int rank = (int)cluster.block_rank();
  const int vu = blockIdx.x / C;
  const int u = vu / P.nhg, hg = vu % P.nhg;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int c4 = lane & 3, r8 = lane >> 2;
  float* SA = reinterpret_cast<float*>(smem + P.o_sa);  // [k][GS] anchor scores (log2 units)
  float* Wt = reinterpret_cast<float*>(smem + P.o_w);   // [wrows][GS] value weights of covered slots
  uint2* qfa = reinterpret_cast<uint2*>(smem + P.o_qfa);
  uint2* qfk = reinterpret_cast<uint2*>(smem + P.o_qfk);
  float* qp = reinterpret_cast<float*>(smem + P.o_qp);
  float* accs = reinterpret_cast<float*>(smem + P.o_acc);
  float* opart = reinterpret_cast<float*>(smem + P.o_opart);
  float* red = reinterpret_cast<float*>(smem + P.o_misc);  // [NTW][GS]
  float* sq = red + NTW * GS;                             // [GS]
  float* mref = sq + GS;                                  // [GS]
  float* cl = mref + GS;                                  // [GS]
  float* pms = cl + GS;                                   // [GS]
  float* ltot = pms + GS;                                 // [GS]
  volatile int* failed = reinterpret_cast<volatile int*>(ltot + GS);
  // rows of max(GS, 4) floats: zeros (no key residual) and -inf (a token past the tile's end)
  float* zrow = reinterpret_cast<float*>(smem + P.o_misc + (((NTW * GS + 6 * GS + 4) * 4 + 15) & ~15));
  float* ninfrow = zrow + (GS > 4 ? GS : 4);
  uint2* meta = reinterpret_cast<uint2*>(smem + P.o_meta);  // [NS] tile block offset, bytes
  float* mslot = reinterpret_cast<float*>(smem + P.o_mslot);
  uint4* hdrs = reinterpret_cast<uint4*>(smem + P.o_hdr);  // [NS][2]
  float* lslot = reinterpret_cast<float*>(smem + P.o_lslot);
  int* fslot = reinterpret_cast<int*>(smem + P.o_fslot);
  float* ofin = reinterpret_cast<float*>(smem + P.o_ofin);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + P.o_bar);
  uint8_t* ring = smem + P.o_ring;
  float* ovf = reinterpret_cast<float*>(smem + P.o_ovf);
  const int NS = P.NS;
  // per stage: an anchor chunk landed (full_c) / a tile block landed (full_t); stage free
  // again (empty: all token and value-residual warps are done with it); key-residual
  // terms ready (rs); probabilities of the value-record tokens written (p).  Chunk items and
  // tiles complete different barriers, so every waiter sees every phase it waits on.
  auto bar_full_c = [&](int s) { return smem_u32(bars + s); };
  auto bar_full_t = [&](int s) { return smem_u32(bars + NS + s); };
  auto bar_empty = [&](int s) { return smem_u32(bars + 2 * NS + s); };
  auto bar_rs = [&](int s) { return smem_u32(bars + 3 * NS + s); };
  auto bar_p = [&](int s) { return smem_u32(bars + 4 * NS + s); };
  auto stage = [&](int s) { return ring + (size_t)s * P.stage_bytes; };


  if (tid == 0) {
    for (int s = 0; s < NS; ++s) {
      mbar_init(bar_full_c(s), 1);  // the producer's expect_tx arrival; bytes complete the phase
      mbar_init(bar_full_t(s), 1);
      mbar_init(bar_empty(s), NTW + NVR);
      mbar_init(bar_rs(s), NKR);
      mbar_init(bar_p(s), NTW);
    }
    *failed = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  pdl_allow_next();
  // Everything above touches only this CTA's shared memory; from here on the launch reads
  // the cache and the query, and writes outputs: first the preceding work must be complete.
  pdl_wait_prev();
  const UnitView U = unit_view(P.arena, u);
  const int k = U.k;

  // This CTA's stream of items: the anchor-key chunks of its score slice (ceil(k / C) anchors),
  // its tile blocks, then the anchor-value chunks of the value slots its tiles cover.  Tokens
  // are stored in value-slot order, so those slots run from the slot of its first stored token,
  // o0, to that of its last; it weights them with its own tokens only, and the products of the
  // CTAs whose ranges meet at a slot add up to that slot's share of the output.
  const int kc = (k + C - 1) / C;
  const int a0 = min(k, rank * kc), a1 = min(k, a0 + kc);
  const int j0 = (int)((long long)rank * U.nt / C), j1 = (int)((long long)(rank + 1) * U.nt / C);
  const int n_kas = (a1 - a0 + CH - 1) / CH;
  const int n_t = j1 - j0;
  const int R = P.R;
  // phase index, on its stage's barrier, of item `it` (anchor chunks and tiles counted apart)
  auto item_phase = [&](int it) -> uint32_t {
    if (it < n_kas) return (uint32_t)(it / NS);
    if (it < n_kas + n_t) return (uint32_t)((it - n_kas) / NS);
    const int s = it % NS, cj = it - n_kas - n_t;
    const int ka_on_s = n_kas > s ? (n_kas - 1 - s) / NS + 1 : 0;
    return (uint32_t)(ka_on_s + cj / NS);
  };
  auto is_tile = [&](int it) { return it >= n_kas && it < n_kas + n_t; };
  // Stage and phase parity of the tiles in order, without divisions: tile tl is item n_kas + tl
  // on stage (n_kas + tl) % NS, and its parity on the tile barriers is (tl / NS) & 1.
  struct TileCursor {
    int s, cnt, ns;
    uint32_t par;
    __device__ void next() {
      s = s + 1 == ns ? 0 : s + 1;
      if (++cnt == ns) {
        cnt = 0;
        par ^= 1u;
      }
    }
  };
  const TileCursor cursor0{n_kas % NS, 0, NS, 0u};
  // B0: every CTA of the cluster has started (its shared memory may take remote stores)
  cluster_arrive();
  // first element of this CTA's query (and output) rows, computed where used
  auto qrow_base = [&]() -> size_t {
    const int b = u / P.n_kv_heads, h = u % P.n_kv_heads;
    return ((size_t)b * P.n_q_heads + (size_t)h * P.G + (size_t)hg * GS) * 128;
  };

  // =========================== producer warp ===================================
  if (warp == W_PROD) {
    // The first NS items need no free stage.  Before the first wait for one (a stage whose
    // tile is consumed only after B1) this warp passes B0 and arrives on B1.
    bool ok = true, b1_arrived = false, b1_done = false;
    const int n_front = n_kas + n_t;
    const int b1_at = min(NS, n_front);
    auto arrive_b1 = [&]() {
      cluster_wait();  // B0
      cluster_arrive();  // B1
      b1_arrived = true;
    };
    int issued = 0;
    int s = 0;
    uint32_t use = 0;  // it = NS use + s
    // value words of the first and the last stored token (lane 0, read as their tiles are
    // issued), then the covered slots [o0, oe) and their chunks, from item n_front on
    uint32_t w_first = 0, w_last = 0;
    int o0 = 0, oe = 0, n_kao = 0;
    for (int it = 0;; ++it, ++s) {
      if (it == n_front) {
        int f = 0, e = 0;
        if (lane == 0 && n_t > 0) {
          f = (int)(w_first & 0xFFFFu);
          e = min(k, min((int)(w_last & 0xFFFFu) + 1, f + P.wrows));
        }
        o0 = __shfl_sync(0xffffffffu, f, 0);
        oe = __shfl_sync(0xffffffffu, e, 0);
        n_kao = oe > o0 ? (oe - o0 + CH - 1) / CH : 0;
      }
      if (it >= n_front + n_kao) break;
      if (s == NS) {
        s = 0;
        ++use;
      }
      if (it == b1_at) arrive_b1();
      if (it == n_front) {  // anchor values are consumed after B2: let B1 complete, arrive on B2
        cluster_wait();
        cluster_arrive();
        b1_done = true;
      }
      if (it >= NS) ok = mbar_wait_w(bar_empty(s), (use - 1) & 1u);
      if (!ok || warp_failed(failed)) {
        *failed = 1;
        break;
      }
      // (drop_last: a test withholds one tile)
      if (lane == 0 && !(P.drop_last > 0 && it == n_front - P.drop_last)) {
        const uint32_t dst = smem_u32(stage(s));
        if (!is_tile(it)) {
          const bool val = it >= n_front;
          const int r0 = val ? o0 + (it - n_front) * CH : a0 + it * CH;
          const int nr = min((val ? oe : a1) - r0, CH);
          const uint32_t bytes = (uint32_t)nr * 256u;
          mbar_expect_tx(bar_full_c(s), bytes);
          bulk_g2s(dst, (val ? U.AV : U.AK) + (size_t)r0 * 256, bytes, bar_full_c(s));
        } else {
          const int j = j0 + it - n_kas;
          const uint32_t b0 = U.table[j], blk = U.table[j + 1] - b0;
          const uint32_t bytes = min(blk, (uint32_t)P.cap);
          meta[s] = make_uint2(b0, blk);
          mbar_expect_tx(bar_full_t(s), bytes);
          bulk_g2s(dst, U.tiles + b0, bytes, bar_full_t(s));
        }
      }
      if (lane == 0 && is_tile(it) && (it == n_kas || it == n_front - 1)) {
        const int j = j0 + it - n_kas, n = min(T, U.S - j * T);
        const uint8_t* vs = U.tiles + U.table[j] + 4 * ((n + 63) & ~63);  // the value stream
        if (it == n_kas) w_first = *reinterpret_cast<const uint32_t*>(vs);
        if (it == n_front - 1) w_last = *reinterpret_cast<const uint32_t*>(vs + 4 * (n - 1));
      }
      issued = it + 1;
      __syncwarp();
    }
    if (!b1_arrived) arrive_b1();
    if (!b1_done) {
      cluster_wait();
      cluster_arrive();
    }
    // every copy this warp started has landed before the CTA may exit (bounded)
    if (lane == 0)
      for (int it = max(0, issued - NS); it < issued; ++it)
        mbar_wait(is_tile(it) ? bar_full_t(it % NS) : bar_full_c(it % NS), item_phase(it) & 1u);
    __syncwarp();
    cluster_wait();  // B2
    cluster_arrive();
    cluster_wait();  // B3 (the last cluster barrier: nothing remote follows it)
    return;
  }

  // =========================== key-residual warps ================================
  // q' . c for the staged key records of each tile on tensor cores: A = the 2-bit codes of
  // 16 records (rows), converted in registers; B = q' (columns: heads as fp16 high parts, then
  // low parts), fragments held in registers.  k order within a 16-dim step: the pair (2c, 2c+1)
  // is dims (2c, 2c+8), the pair (2c+8, 2c+9) is dims (2c+1, 2c+9), so one shift of a code word
  // gives both codes of a pair at bits 0 and 16.
  if (kres_index(warp) >= 0) {
    const int kw = kres_index(warp);
    cluster_wait();    // B0
    cluster_arrive();  // B1
    // ---- the rotated query (off the token warps' way to the anchor scores) ----
    // row g (warp g % NKR): signs, 128-point Walsh-Hadamard transform in registers, scale ->
    // q' (Appendix A.1, Eq. 12) into qp, its sum into sq
    const float f = P.rotate ? P.scale_log2 * (1.0f / 128.0f) : P.scale_log2;
    for (int g = kw; g < GS; g += NKR) {
      const uint2 raw = *reinterpret_cast<const uint2*>(P.q + qrow_base() + (size_t)g * 128 + 4 * lane);
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
      const float sg = warp_sum((x[0] + x[1]) + (x[2] + x[3]));
      if (lane == 0) sq[g] = sg;
    }
    named_sync(5, NKR * 32);
    // key-residual B fragments (k-step ks, lane): column c = lane / 4 is head c % 4 as the fp16
    // high part (c < 4) or low part -- for GS = 8, set hl (0: high parts, 1: low parts) of
    // head c; k pairs (2t, 2t+1) <-> dims (16ks + 2t, 16ks + 2t + 8), (2t+8, 2t+9) <->
    // (16ks + 2t + 1, 16ks + 2t + 9), t = lane % 4.
    {
      const int g = lane >> 2, c = lane & 3;
      for (int ks = kw; ks < 8; ks += NKR)
#pragma unroll
        for (int hl = 0; hl < (GS == 8 ? 2 : 1); ++hl) {
          uint2 fk = make_uint2(0u, 0u);
          const int head = GS == 8 ? g : (g & 3);
          const bool low = GS == 8 ? hl == 1 : g >= 4;
          if (head < GS) {
            const float* x = qp + head * 128 + 16 * ks + 2 * c;
            auto part = [&](float v) {
              const __half hi = __float2half_rn(v);
              return low ? __float2half_rn(v - __half2float(hi)) : hi;
            };
            const __half h0 = part(x[0]), h8 = part(x[8]), h1 = part(x[1]), h9 = part(x[9]);
            fk.x = pack_h2(h0, h8);
            fk.y = pack_h2(h1, h9);
          }
          qfk[hl * 256 + ks * 32 + lane] = fk;
        }
    }
    named_sync(5, NKR * 32);
    named_arrive(2, NTW * 32 + NKR * 32);  // the token warps may use qp and sq
    constexpr int NBF = GS == 8 ? 2 : 1;  // fragment sets: GS = 8 keeps high and low parts apart
    uint2 bf[NBF][8];
#pragma unroll
    for (int hl = 0; hl < NBF; ++hl)
#pragma unroll
      for (int ks = 0; ks < 8; ++ks) bf[hl][ks] = qfk[hl * 256 + ks * 32 + lane];
    bool ok = true;
    TileCursor cur = cursor0;
    for (int tl = 0; tl < n_t; ++tl, cur.next()) {
      const int s = cur.s;
      if (ok && !warp_failed(failed)) {
        ok = mbar_wait_w(bar_full_t(s), cur.par);
        if (!ok) *failed = 1;
      }
      if (ok && !warp_failed(failed)) {
        const TileView tv = tile_view(stage(s), meta[s], U, j0 + tl, P.cap);
        if (kw == 0) put_header(hdrs + 2 * s, tv, meta[s]);
        const int nK = min(tv.nk, R);
        float* rs = reinterpret_cast<float*>(stage(s) + P.o_rs);
        // records addressed in shared memory when the whole block is staged (the common case)
        auto groups = [&](auto staged_all) {
          auto rec = [&](uint32_t off) -> const uint8_t* {
            if constexpr (decltype(staged_all)::value) return tv.st + off;
            else return tv.at(off);
          };
          // two groups of 16 records at a time, each as two independent mma chains
          for (int g16 = kw; g16 * 16 < nK; g16 += 2 * NKR) {
            uint32_t wd[2][2][8];  // [group][record r8 / r8 + 8][16-dim step]
#pragma unroll
            for (int q = 0; q < 2; ++q)
#pragma unroll
              for (int hr = 0; hr < 2; ++hr) {
                const int sl = (g16 + q * NKR) * 16 + r8 + 8 * hr;
                uint4 w0 = make_uint4(0u, 0u, 0u, 0u), w1 = w0;
                if (sl < nK) {
                  w0 = *reinterpret_cast<const uint4*>(rec(tv.cd_k + 32u * (uint32_t)sl));
                  w1 = *reinterpret_cast<const uint4*>(rec(tv.cd_k + 32u * (uint32_t)sl + 16u));
                }
                wd[q][hr][0] = w0.x; wd[q][hr][1] = w0.y; wd[q][hr][2] = w0.z; wd[q][hr][3] = w0.w;
                wd[q][hr][4] = w1.x; wd[q][hr][5] = w1.y; wd[q][hr][6] = w1.z; wd[q][hr][7] = w1.w;
              }
            // two independent chains per group: alternate k-steps, or (GS = 8) high and low parts
            float d[2][2][4] = {};
#pragma unroll
            for (int ks = 0; ks < 8; ++ks)
#pragma unroll
              for (int q = 0; q < 2; ++q) {
                const uint32_t xa = wd[q][0][ks] >> (4 * c4), xb = wd[q][1][ks] >> (4 * c4);
                const uint4 a = make_uint4(codes2_to_h2(xa), codes2_to_h2(xb), codes2_to_h2(xa >> 2), codes2_to_h2(xb >> 2));
                if constexpr (GS == 8) {
                  mma_f16(d[q][0], a, bf[0][ks].x, bf[0][ks].y);
                  mma_f16(d[q][1], a, bf[NBF - 1][ks].x, bf[NBF - 1][ks].y);
                } else {
                  mma_f16(d[q][ks & 1], a, bf[0][ks].x, bf[0][ks].y);
                }
              }
            // columns 2c, 2c+1: heads 2c, 2c+1 (GS = 8: high + low parts of the two chains);
            // otherwise high parts of heads 2c, 2c+1 (c < 2) or low parts (c >= 2)
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
                  const int sl = (g16 + q * NKR) * 16 + r8 + 8 * hr;
                  if (sl < nK) {
                    const uint32_t smn = *reinterpret_cast<const uint32_t*>(rec(tv.sm_k + 4u * (uint32_t)sl));
#pragma unroll
                    for (int e = 0; e < 2; ++e) {
                      const int g = 2 * c4 + e;
                      if (g < GS) rs[sl * GS + g] = half_hi(smn) * sq[g] + half_lo(smn) * v[2 * hr + e];
                    }
                  }
                }
              }
            }
          }
        };
        if (tv.staged == meta[s].y) groups(std::true_type{});
        else groups(std::false_type{});
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(bar_rs(s));
    }
    cluster_wait();  // B1
    cluster_arrive();
    cluster_wait();  // B2
    cluster_arrive();
    cluster_wait();  // B3 (the last cluster barrier: nothing remote follows it)
    return;
  }

  // =========================== value-residual warps ==============================
  // Per tile, for the staged value records: sum over records of (p scale) c on tensor cores
  // (bf16 operands: p scale as high + low parts, codes exact), in the rotated domain, with p
  // as the token warps stored it.  Step 1: each warp builds the A operands of every NVR-th
  // group of 16 records into a shared buffer (two buffers, tiles alternate); step 2: each
  // warp multiplies all groups into the 32 coordinates 32 vw .. 32 vw + 31 it owns.  The token
  // warps add records beyond the staged count themselves, on CUDA cores.
  if (vres_index(warp) >= 0) {
    const int vw = vres_index(warp);
    cluster_wait();    // B0
    cluster_arrive();  // B1
    named_sync(3, NTW * 32 + NVR * 32);  // anchor-score table, references and accs are ready
    float accV[2][4][4] = {};  // two independent sets (alternate groups), summed at the end
    // step-1 roles: record slot (lane % 16) of a group, heads hb, hb + 2, ... (hb = lane / 16)
    constexpr int HPL = GS >= 2 ? GS / 2 : 1;
    const int sl16 = lane & 15, hb = lane >> 4;
    const bool head_lane = hb < GS;
    float pminv[HPL];
#pragma unroll
    for (int i = 0; i < HPL; ++i) pminv[i] = 0.f;
    const int ngrp_st = (R + 15) / 16;
    bool ok = true;
    TileCursor cur = cursor0;
    for (int tl = 0; tl < n_t; ++tl, cur.next()) {
      const int s = cur.s;
      const uint32_t par = cur.par;
      if (ok && !warp_failed(failed)) {
        ok = mbar_wait_w(bar_full_t(s), par) && mbar_wait_w(bar_p(s), par);
        if (!ok) *failed = 1;
      }
      const bool go = ok && !warp_failed(failed);
      TileView tv;
      uint2 mt = make_uint2(0u, 0u);  // block offset and bytes, from the header
      uint8_t* pf = smem + P.o_pfb + (tl & 1) * ngrp_st * 512;
      int nV = 0;
      if (go) {
        tv = header_view(stage(s), hdrs + 2 * s, U, P.cap, &mt);
        nV = min(tv.nv, R);
        const float* pvb = reinterpret_cast<const float*>(stage(s) + P.o_pv);
        for (int grp = vw; grp * 16 < nV; grp += NVR) {
          const int r = grp * 16 + sl16;
          // slots past the last record get zero operands
          if (head_lane) {
            const bool rec_ok = r < nV;
            uint32_t smn = 0u;
            if (rec_ok)
              smn = *reinterpret_cast<const uint32_t*>(tv.staged == mt.y ? tv.st + tv.sm_v + 4u * (uint32_t)r
                                                                             : tv.at(tv.sm_v + 4u * (uint32_t)r));
            const float scl = half_lo(smn), mn = half_hi(smn);
#pragma unroll
            for (int i = 0; i < HPL; ++i) {
              const int g = hb + 2 * i;
              const float p = rec_ok ? pvb[r * GS + g] : 0.f;
              // A-operand place of (record r, head g): group r / 16, lane 4 g + (r % 8) / 2,
              // register 2 ((r / 8) % 2) (high part) or + 1 (low part), half r % 2
              __nv_bfloat16 phi, plo;
              split_b(p * scl, phi, plo);
              pminv[i] = fmaf(p, mn, pminv[i]);
              unsigned short* dst = reinterpret_cast<unsigned short*>(
                  pf + grp * 512 + (4 * g + ((r & 7) >> 1)) * 16 + ((r >> 3) & 1) * 8 + (r & 1) * 2);
              dst[0] = __bfloat16_as_ushort(phi);
              dst[2] = __bfloat16_as_ushort(plo);
            }
          }
        }
      }
      // every warp's operands of this tile are written, and every warp is done with the
      // other buffer (its previous tile)
      named_sync(4, NVR * 32);
      if (go) {
        // B operand straight from the dimension-major code words: this lane's four words hold
        // dimensions 32 vw + 8 nb + r8 (nb = 0..3) of 16 records; records 2c, 2c+1 feed b0,
        // records 2c+8, 2c+9 feed b1
        auto groups = [&](auto staged_all) {  // code words in shared memory when all staged
          auto rec = [&](uint32_t off) -> const uint8_t* {
            if constexpr (decltype(staged_all)::value) return tv.st + off;
            else return tv.at(off);
          };
          const uint32_t woff = tv.cd_v + 4u * (uint32_t)(32 * vw + 4 * r8);
          for (int grp = 0; grp * 16 < nV; grp += 2) {
#pragma unroll
            for (int q = 0; q < 2; ++q) {
              if ((grp + q) * 16 >= nV) break;  // warp-uniform
              const uint4 a = *reinterpret_cast<const uint4*>(pf + (grp + q) * 512 + lane * 16);
              const uint4 w4 = *reinterpret_cast<const uint4*>(rec(woff + 512u * (uint32_t)(grp + q)));
              const uint32_t wd[4] = {w4.x, w4.y, w4.z, w4.w};
#pragma unroll
              for (int nb = 0; nb < 4; ++nb) {
                // records 2c, 2c+1 at bits 2c and 2c + 16, records 2c+8, 2c+9 eight bits higher
                const uint32_t x = wd[nb] >> (2 * c4);
                mma_bf16(accV[q][nb], a.x, a.y, a.z, a.w, codes2_to_b2(x), codes2_to_b2(x >> 8));
              }
            }
          }
        };
        if (tv.staged == mt.y) groups(std::true_type{});
        else groups(std::false_type{});
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(bar_empty(s));
    }
    // rows r8 (high parts) + r8 + 8 (low parts); records beyond the staged count were added
    // in step 1; sum p min per head
    if (r8 < GS) {
#pragma unroll
      for (int nb = 0; nb < 4; ++nb) {
        const int col = 32 * vw + 8 * nb + 2 * c4;
        atomicAdd(&accs[r8 * 128 + col], (accV[0][nb][0] + accV[0][nb][2]) + (accV[1][nb][0] + accV[1][nb][2]));
        atomicAdd(&accs[r8 * 128 + col + 1], (accV[0][nb][1] + accV[0][nb][3]) + (accV[1][nb][1] + accV[1][nb][3]));
      }
    }
#pragma unroll
    for (int i = 0; i < HPL; ++i) {
#pragma unroll
      for (int o = 1; o < 16; o <<= 1) pminv[i] += __shfl_xor_sync(0xffffffffu, pminv[i], o);
      if (sl16 == 0 && head_lane) atomicAdd(&pms[hb + 2 * i], pminv[i]);
    }
    cluster_wait();  // B1
    cluster_arrive();
    cluster_wait();  // B2
    cluster_arrive();
    cluster_wait();  // B3 (the last cluster barrier: nothing remote follows it)
    return;
  }

  // =========================== token warps =======================================
  // ---- phase 0: zeroed tables, anchor-score B fragments (the rotated query is the
  // key-residual warps' job) ----
  for (int e = tid; e < GS * 128; e += NTT) accs[e] = ovf[e] = 0.f;
  for (int e = a0 * GS + tid; e < a1 * GS; e += NTT) SA[e] = 0.f;
  for (int e = tid; e < P.wrows * GS; e += NTT) Wt[e] = 0.f;
  for (int e = tid; e < ((R + 15) / 16) * 256; e += NTT) reinterpret_cast<uint32_t*>(smem + P.o_pfb)[e] = 0u;
  if (tid < GS) pms[tid] = 0.f;
  if (tid < (GS > 4 ? GS : 4)) {
    zrow[tid] = 0.f;
    ninfrow[tid] = -INFINITY;
  }
  {
    // fragment (k-step ks, lane ln): one per token thread (8 k-steps x 32 lanes); q in bf16,
    // k order permuted so that a thread's dims are contiguous
    const int ks = tid >> 5, ln = tid & 31, g = ln >> 2, c = ln & 3;
    uint2 fa = make_uint2(0u, 0u);
    if (g < GS) {
      const uint2 raw = *reinterpret_cast<const uint2*>(P.q + qrow_base() + (size_t)g * 128 + 32 * (ks >> 1) + 8 * c + 4 * (ks & 1));
      fa = raw;  // dims d0 .. d0 + 3 as two bf16 pairs
    }
    qfa[ks * 32 + ln] = fa;
  }
  tw_sync();

  bool ok = true;
  auto wait_item = [&](int i) -> const uint8_t* {
    const int s = i % NS;
    if (ok && !warp_failed(failed)) ok = mbar_wait_w(is_tile(i) ? bar_full_t(s) : bar_full_c(s), item_phase(i) & 1u);
    if (!ok) *failed = 1;
    return stage(s);
  };
  auto release_chunk = [&](int i) {  // the value-residual warps' share of a chunk's release: warp 0
    __syncwarp();
    if (lane == 0) mbar_arrive_cnt(bar_empty(i % NS), warp == 0 ? 1 + NVR : 1);
  };

  // ---- phase 1: anchor scores of this CTA's slice (bf16 tensor cores) ----
  // work item (16-row block rb, half kh of the 128 dims) -> warp item % NTW; rows are
  // swizzled in 16-byte chunks by (absolute row % 8)
  for (int it = 0; it < n_kas; ++it) {
    const uint8_t* st = wait_item(it);
    if (ok && !warp_failed(failed)) {
      const int r0 = a0 + it * CH, nr = min(a1 - r0, CH);
      for (int item = warp; item < 2 * (CH / 16); item += NTW) {
        const int rb = item >> 1, kh = item & 1;
        if (16 * rb >= nr) break;
        float d[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int jj = 0; jj < 2; ++jj) {
          const int j = 2 * kh + jj, cc = (4 * j + c4) ^ ((r0 + r8) & 7);  // rows r8, r8 + 8: same swizzle
          const uint4 lo = *reinterpret_cast<const uint4*>(st + (16 * rb + r8) * 256 + 16 * cc);
          const uint4 hi = *reinterpret_cast<const uint4*>(st + (16 * rb + r8 + 8) * 256 + 16 * cc);
          const uint2 b0 = qfa[(2 * j) * 32 + lane], b1 = qfa[(2 * j + 1) * 32 + lane];
          mma_bf16(d, lo.x, hi.x, lo.y, hi.y, b0.x, b0.y);
          mma_bf16(d, lo.z, hi.z, lo.w, hi.w, b1.x, b1.y);
        }
        const int ra = 16 * rb + r8, gc = 2 * c4;
        // two partial sums (the dim halves) per entry, added onto 0: the same in either order
        if (ra < nr) {
          if (gc < GS) atomicAdd(&SA[(r0 + ra) * GS + gc], d[0] * P.scale_log2);
          if (gc + 1 < GS) atomicAdd(&SA[(r0 + ra) * GS + gc + 1], d[1] * P.scale_log2);
        }
        if (ra + 8 < nr) {
          if (gc < GS) atomicAdd(&SA[(r0 + ra + 8) * GS + gc], d[2] * P.scale_log2);
          if (gc + 1 < GS) atomicAdd(&SA[(r0 + ra + 8) * GS + gc + 1], d[3] * P.scale_log2);
        }
      }
    }
    release_chunk(it);
  }
  tw_sync();
  // The slice goes into every peer's table (remote stores, done before B1 completes), and
  // its largest score per head into slot `rank` of every CTA.  Reference for the exponentials:
  // the largest anchor score per query row.  Anchors are tokens of the unit, so it never
  // exceeds the true maximum logit; every CTA of the cluster takes the same reference, which
  // makes the cluster combine a plain sum.
  cluster_wait();  // B0: the peers have started
  {
    float mx[GS];
#pragma unroll
    for (int g = 0; g < GS; ++g) mx[g] = -INFINITY;
    for (int a = a0 + tid; a < a1; a += NTT) {
      float row[GS];
      load_row<GS>(SA + a * GS, row);
#pragma unroll
      for (int g = 0; g < GS; ++g) mx[g] = fmaxf(mx[g], row[g]);
      for (int r = 0; r < C; ++r)
        if (r != rank) st_cluster_row<GS>(SA + a * GS, r);
    }
#pragma unroll
    for (int g = 0; g < GS; ++g) {
      const float m = warp_max(mx[g]);
      if (lane == 0) red[warp * GS + g] = m;
    }
    tw_sync();
    if (tid < GS) {
      float m = red[tid];
      for (int w = 1; w < NTW; ++w) m = fmaxf(m, red[w * GS + tid]);
      mslot[rank * GS + tid] = m;
      for (int r = 0; r < C; ++r)
        if (r != rank) st_cluster_row<1>(mslot + rank * GS + tid, r);
    }
  }
  cluster_arrive();  // B1
  cluster_wait();
  if (tid < GS) {
    float m = mslot[tid];
    for (int r = 1; r < C; ++r) m = fmaxf(m, mslot[r * GS + tid]);
    mref[tid] = m;
  }
  tw_sync();
  named_arrive(3, NTW * 32 + NVR * 32);  // the value-residual warps may use SA, mref and accs
  // pairs of heads for the packed arithmetic (GS = 1: one head, the pair's second lane idle)
  constexpr int NP = GS >= 2 ? GS / 2 : 1;
  float2 negm[NP], l2[NP];
#pragma unroll
  for (int i = 0; i < NP; ++i) {
    negm[i] = make_float2(-mref[2 * i], GS >= 2 ? -mref[2 * i + 1] : 0.f);
    l2[i] = make_float2(0.f, 0.f);
  }
  // Value weights of a run: one reduction per head into this CTA's table, whose row i is value
  // slot o0 + i (o0: the slot of this CTA's first stored token, so no run lies below it).  A run
  // beyond the table's wrows rows (tiles that cover more slots than it holds: rare) takes its
  // anchor's value row from global memory and adds its products into ovf on CUDA cores.
  int o0 = 0, o_last = -1;  // value slots of this CTA's first and last stored tokens
  auto flush = [&](int anchor, const float2 (&v)[NP]) {
    const int i = anchor - o0;
    if (anchor >= k || i < 0) return;
    if (i < P.wrows) {
      float* w = &Wt[i * GS];
#pragma unroll
      for (int g = 0; g < GS; ++g) red_local(w + g, (g & 1) ? v[g >> 1].y : v[g >> 1].x);
    } else {
      // (kept compact: this code sits in the token loop but almost never runs)
      const uint8_t* row = U.AV + (size_t)anchor * 256;
#pragma unroll 1
      for (int d = 0; d < 128; ++d) {  // dim d: element d % 8 of chunk d / 8, stored at (d / 8) ^ (row % 8)
        const float x = __bfloat162float(*reinterpret_cast<const __nv_bfloat16*>(row + 16 * ((d >> 3) ^ (anchor & 7)) + 2 * (d & 7)));
#pragma unroll
        for (int g = 0; g < GS; ++g) atomicAdd(&ovf[g * 128 + d], ((g & 1) ? v[g >> 1].y : v[g >> 1].x) * x);
      }
    }
  };

  // ---- phase 2: tile blocks ----
  named_sync(2, NTW * 32 + NKR * 32);  // q' rows and their sums from the key-residual warps
  // lane -> four consecutive stored tokens of the warp's 128-token region, every head
  TileCursor cur = cursor0;
  for (int tl = 0; tl < n_t; ++tl, cur.next()) {
    const int s = cur.s;
    const uint8_t* st = stage(s);
    if (ok && !warp_failed(failed)) {
      ok = mbar_wait_w(bar_full_t(s), cur.par) && mbar_wait_w(bar_rs(s), cur.par);
      if (!ok) *failed = 1;
    }
    bool released = false;
    if (ok && !warp_failed(failed)) {
      uint2 mt;
      const TileView tv = header_view(st, hdrs + 2 * s, U, P.cap, &mt);
      const float* rsb = reinterpret_cast<const float*>(st + P.o_rs);
      const int t0 = warp * REG + 4 * lane;
      if (tl == 0) o0 = (int)(*reinterpret_cast<const uint32_t*>(tv.st + 4 * tv.n64) & 0xFFFFu);
      if (tl == n_t - 1) o_last = (int)(*reinterpret_cast<const uint32_t*>(tv.st + 4 * (tv.n64 + tv.n - 1)) & 0xFFFFu);
      // tail: the run that ends this lane's tokens (its anchor `key`), head: the run that
      // starts them when it differs (multi)
      uint32_t key = 0xFFFFFFFFu;
      int hkey = -1;
      bool multi = false;
      float2 val[NP], headv[NP];
#pragma unroll
      for (int i = 0; i < NP; ++i) val[i] = headv[i] = make_float2(0.f, 0.f);
      if (t0 < tv.n) {
        const uint4 ka = *reinterpret_cast<const uint4*>(tv.st + 4 * t0);
        const uint4 va = *reinterpret_cast<const uint4*>(tv.st + 4 * (tv.n64 + t0));
        const uint32_t ek[4] = {ka.x, ka.y, ka.z, ka.w}, ev[4] = {va.x, va.y, va.z, va.w};
        const int wi = t0 >> 6, sh = t0 & 63;
        const uint64_t wk = tv.bm(0, wi), wv = tv.bm(1, wi);
        const uint32_t kbits = (uint32_t)(wk >> sh) & 0xFu, vbits = (uint32_t)(wv >> sh) & 0xFu;
        int rkn = tv.rk(0, wi) + __popcll(wk & ((1ull << sh) - 1ull));
        int rvn = tv.rk(1, wi) + __popcll(wv & ((1ull << sh) - 1ull));
        float* pvb = reinterpret_cast<float*>(const_cast<uint8_t*>(st) + P.o_pv);
        const int nvalid = min(4, tv.n - t0);
        float2 cw[4][NP];
        uint32_t av[4];
        // one token: logits, p, l, run weights and, for a value record, its p (every record
        // staged: tokens without a value record write the spare row R; otherwise the records
        // beyond the staged ones take the CUDA-core paths)
        auto token = [&](int e, auto dense) {
          constexpr bool kDense = decltype(dense)::value;
          const int a = min((int)(ek[e] & 0xFFFFu), k - 1);  // indices are < k by construction
          float sa[GS], rt[GS];
          load_row<GS>(SA + a * GS, sa);
          const bool kb = (kbits >> e) & 1u;
          const int r = rkn;
          rkn += (int)kb;
          if (kDense && kb && r >= R) {
#pragma unroll
            for (int g = 0; g < GS; ++g) rt[g] = key_record_term(tv, r, qp + g * 128, sq[g]);
          } else {  // the key-residual terms, zeros, or -inf for a token past the tile's end
            load_row<GS>(e >= nvalid ? ninfrow : (kb ? rsb + r * GS : zrow), rt);
          }
          const float gk = half_hi(ek[e]), gv = half_hi(ev[e]);
          float2 pe[NP];
#pragma unroll
          for (int i = 0; i < NP; ++i) {
            const float2 s2 = make_float2(sa[2 * i], GS >= 2 ? sa[2 * i + 1] : 0.f);
            const float2 r2 = make_float2(rt[2 * i], GS >= 2 ? rt[2 * i + 1] : 0.f);
            const float2 x = f2add(f2fma(make_float2(gk, gk), s2, r2), negm[i]);
            const float2 p = make_float2(exp2_approx(x.x), GS >= 2 ? exp2_approx(x.y) : 0.f);
            l2[i] = f2add(l2[i], p);
            cw[e][i] = f2mul(p, make_float2(gv, gv));
            pe[i] = p;
          }
          av[e] = ev[e] & 0xFFFFu;
          const bool vb = (vbits >> e) & 1u;
          const int rv = rvn;
          rvn += (int)vb;
          if (!kDense) {
            store_row<GS>(pvb + (vb ? rv : R) * GS, pe);
          } else if (vb) {
            if (rv < R) {
              store_row<GS>(pvb + rv * GS, pe);
            } else {  // beyond the staged records (a locally dense tile): CUDA cores
              const uint32_t smn = *reinterpret_cast<const uint32_t*>(tv.at(tv.sm_v + 4u * (uint32_t)rv));
#pragma unroll
              for (int g = 0; g < GS; ++g) {
                const float pg = (g & 1) ? pe[g >> 1].y : pe[g >> 1].x;
                value_record_add(tv, rv, pg * half_lo(smn), accs + g * 128);
                atomicAdd(&pms[g], pg * half_hi(smn));
              }
            }
          }
        };
        if (tv.nk <= R && tv.nv <= R) {
#pragma unroll
          for (int e = 0; e < 4; ++e) token(e, std::false_type{});
        } else {
#pragma unroll
          for (int e = 0; e < 4; ++e) token(e, std::true_type{});
        }
        // tokens past the tile join the last token's run with zero weight
#pragma unroll
        for (int e = 1; e < 4; ++e)
          if (e >= nvalid) av[e] = av[e - 1];
        hkey = (int)av[0];
        key = av[3];
        multi = av[0] != av[3];
        float hw[4], tw[4];  // 0/1 membership of the head run and the tail run
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          hw[e] = av[e] == av[0] ? 1.f : 0.f;
          tw[e] = av[e] == av[3] ? 1.f : 0.f;
        }
#pragma unroll
        for (int i = 0; i < NP; ++i) {
          float2 hs = make_float2(0.f, 0.f), ts = hs;
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            hs = f2fma(cw[e][i], make_float2(hw[e], hw[e]), hs);
            ts = f2fma(cw[e][i], make_float2(tw[e], tw[e]), ts);
          }
          val[i] = ts;
          headv[i] = multi ? hs : make_float2(0.f, 0.f);
        }
        if (multi) {  // runs strictly inside the lane's four tokens (rare)
#pragma unroll
          for (int e = 1; e < 3; ++e)
            if (av[e] != av[0] && av[e] != av[3]) flush((int)av[e], cw[e]);
        }
      }
      // the stage is not read again: release it before the reductions, which then never
      // delay the hand-over to the value-residual warps and the producer
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(bar_p(s));
        mbar_arrive(bar_empty(s));
      }
      released = true;
      // Runs across lanes (anchors never decrease from lane to lane): the next lane's head run
      // continues this lane's tail run when their anchors match; a head run that does not
      // continue the previous lane's tail is complete
      const uint32_t pkey = __shfl_up_sync(0xffffffffu, key, 1);
      const int nhkey = __shfl_down_sync(0xffffffffu, hkey, 1);
      const bool nmulti = __shfl_down_sync(0xffffffffu, (int)multi, 1) != 0;
      const bool take_next = lane < 31 && nmulti && (uint32_t)nhkey == key;
#pragma unroll
      for (int i = 0; i < NP; ++i) {
        const float2 nh = make_float2(__shfl_down_sync(0xffffffffu, headv[i].x, 1),
                                      __shfl_down_sync(0xffffffffu, headv[i].y, 1));
        if (take_next) val[i] = f2add(val[i], nh);
      }
      if (multi && !(lane > 0 && pkey == (uint32_t)hkey)) flush(hkey, headv);
      // segmented inclusive scan of the tail sums over lanes with equal anchors
#pragma unroll
      for (int d = 1; d < 32; d <<= 1) {
        const uint32_t kd = __shfl_up_sync(0xffffffffu, key, d);
        const bool add = lane >= d && kd == key;
#pragma unroll
        for (int i = 0; i < NP; ++i) {
          const float2 vd = make_float2(__shfl_up_sync(0xffffffffu, val[i].x, d),
                                        __shfl_up_sync(0xffffffffu, val[i].y, d));
          if (add) val[i] = f2add(val[i], vd);
        }
      }
      const uint32_t nkey = __shfl_down_sync(0xffffffffu, key, 1);
      if (key != 0xFFFFFFFFu && (lane == 31 || nkey != key)) flush((int)key, val);
    }
    if (!released) {  // a failed CTA still hands the stage on (warp-uniform)
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(bar_p(s));
        mbar_arrive(bar_empty(s));
      }
    }
  }
  // a logit so far above the reference that the sums overflow leaves a non-finite normaliser
  bool overflow_risk = false;
#pragma unroll
  for (int i = 0; i < NP; ++i) overflow_risk |= !(l2[i].x < INFINITY) || !(l2[i].y < INFINITY);
  if (overflow_risk) *failed = 1;

  // ---- per-CTA totals ----
#pragma unroll
  for (int g = 0; g < GS; ++g) {
    const float sl = warp_sum((g & 1) ? l2[g >> 1].y : l2[g >> 1].x);
    if (lane == 0) red[warp * GS + g] = sl;
  }
  tw_sync();
  if (tid < GS) {  // this CTA's normaliser share, into slot `rank` of every CTA
    float sl = 0.f;
    for (int w = 0; w < NTW; ++w) sl += red[w * GS + tid];
    lslot[rank * GS + tid] = sl;
    for (int r = 0; r < C; ++r)
      if (r != rank) st_cluster_row<1>(lslot + rank * GS + tid, r);
  }
  tw_sync();

  // ---- phase 3: combine across the cluster (one common reference: plain sums) ----
  cluster_arrive();  // B2: every normaliser share has landed
  cluster_wait();
  if (tid < GS) {
    float Lt = 0.f;
    for (int r = 0; r < C; ++r) Lt += lslot[r * GS + tid];
    ltot[tid] = Lt;
  }
  // weights of the covered slots times their values (bf16 tensor cores, weights as hi + lo);
  // warp -> dims 16 warp .. 16 warp + 15
  float oacc[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
  // (the producer derives the same covered slots [o0, oe) from the same two tokens)
  const int oe = n_t > 0 ? min(k, min(o_last + 1, o0 + P.wrows)) : 0;
  const int n_kao = oe > o0 ? (oe - o0 + CH - 1) / CH : 0;
  for (int ci = 0; ci < n_kao; ++ci) {
    const int it = n_kas + n_t + ci;
    const uint8_t* st = wait_item(it);
    if (ok && !warp_failed(failed)) {
      const int r0 = o0 + ci * CH, nr = min(oe - r0, CH);
      for (int blk = 0; blk < CH / 16 && 16 * blk < nr; ++blk) {
        const int mi = lane >> 3, ri = lane & 7;
        const int row = 16 * blk + (mi & 1) * 8 + ri;
        const int cc = (2 * warp + (mi >> 1)) ^ ((r0 + ri) & 7);  // absolute row % 8
        uint32_t b00, b01, b10, b11;
        ldsm_x4_trans(smem_u32(st + row * 256 + 16 * cc), b00, b01, b10, b11);
        // rows past the slice hold stale bytes: clear their halves of B
        const int ka = 16 * blk + 2 * c4;
        const uint32_t m0 = (ka < nr ? 0xFFFFu : 0u) | (ka + 1 < nr ? 0xFFFF0000u : 0u);
        const uint32_t m1 = (ka + 8 < nr ? 0xFFFFu : 0u) | (ka + 9 < nr ? 0xFFFF0000u : 0u);
        b00 &= m0;
        b10 &= m0;
        b01 &= m1;
        b11 &= m1;
        uint32_t ah0 = 0, al0 = 0, ah2 = 0, al2 = 0;
        if (r8 < GS) {
          const int kk[4] = {ka, ka + 1, ka + 8, ka + 9};
          __nv_bfloat16 hi[4], lo[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float w = kk[e] < nr ? Wt[(r0 - o0 + kk[e]) * GS + r8] : 0.f;
            split_b(w, hi[e], lo[e]);
          }
          ah0 = pack_b2(hi[0], hi[1]);
          al0 = pack_b2(lo[0], lo[1]);
          ah2 = pack_b2(hi[2], hi[3]);
          al2 = pack_b2(lo[2], lo[3]);
        }
        mma_bf16(oacc[0], ah0, al0, ah2, al2, b00, b01);
        mma_bf16(oacc[1], ah0, al0, ah2, al2, b10, b11);
      }
    }
    release_chunk(it);
  }
  // this CTA's value residuals (staged records from the value-residual warps, overflow
  // records and sum p * min from the token warps), then the inverse rotation once
  // (warp g < GS: row g in registers; the inverse of q' = H (s o q) / 128 on the value side
  // is s o H(.) / 128)
  if (warp < GS) {
    const float4 v = *reinterpret_cast<const float4*>(accs + warp * 128 + 4 * lane);
    const float pm = pms[warp];
    float x[4] = {v.x + pm, v.y + pm, v.z + pm, v.w + pm};
    if (P.rotate) {
      warp_wht128(x, lane);
      apply_signs(x, lane, P.sign_lo, P.sign_hi);
#pragma unroll
      for (int j = 0; j < 4; ++j) x[j] *= (1.0f / 128.0f);
    }
    *reinterpret_cast<float4*>(opart + warp * 128 + 4 * lane) = make_float4(x[0], x[1], x[2], x[3]);
  }
  tw_sync();
  if (r8 < GS) {
#pragma unroll
    for (int nb = 0; nb < 2; ++nb) {
      const int col = 16 * warp + 8 * nb + 2 * c4;
      opart[r8 * 128 + col] += oacc[nb][0] + oacc[nb][2];
      opart[r8 * 128 + col + 1] += oacc[nb][1] + oacc[nb][3];
    }
  }
  tw_sync();
  for (int e = tid; e < GS * 128; e += NTT) opart[e] += ovf[e];
  tw_sync();
  // Elements are shared out in blocks of `per` (a multiple of 4); each block of this CTA's
  // partial output goes, as 16-byte remote stores, into slot `rank` of the staging rows of
  // the CTA that writes it, and this CTA's failure flag into slot `rank` of every CTA.  After
  // B3 no CTA touches another's shared memory, so none waits for the others before it exits.
  const int E = GS * 128;
  const int per = 4 * ((E / 4 + C - 1) / C);
  for (int e = 4 * tid; e < E; e += 4 * NTT) {
    const int owner = e / per;
    float* dst = ofin + rank * per + (e - owner * per);  // the same place in the owner's rows
    const float4 v = *reinterpret_cast<const float4*>(opart + e);
    if (owner == rank) *reinterpret_cast<float4*>(dst) = v;
    else st_cluster_v4(dst, owner, v);
  }
  if (tid == 0) {
    fslot[rank] = *failed;
    for (int r = 0; r < C; ++r)
      if (r != rank) st_cluster_int(fslot + rank, r);
  }
  cluster_arrive();  // B3
  cluster_wait();
  {
    const int e0 = rank * per, e1 = min(E, e0 + per);
    bool bad = false;
    for (int r = 0; r < C; ++r) bad |= fslot[r] != 0;
    for (int e = e0 + tid; e < e1; e += NTT) {
      float sum = 0.f;
      for (int r = 0; r < C; ++r) sum += ofin[r * per + (e - e0)];
      const float y = bad ? __int_as_float(0x7FC00000) : sum / ltot[e >> 7];
      const size_t o = qrow_base() + e;
      P.out[o] = __float2bfloat16_rn(y);
      if (P.out_f32) P.out_f32[o] = y;
    }
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

// Launch plan: shared-memory carve-up, ring depth, staged records per tile, cluster size.
struct Plan {
  DecodeParams P;
  size_t smem = 0;
  int C = 1;
};

size_t align128(size_t x) { return (x + 127) & ~(size_t)127; }

double max_density(const Layout& L) {
  double dens = 0.0;
  for (const auto& s : L.shape) dens = std::max(dens, (double)std::max(s.nk, s.nv) / (double)s.S);
  return dens;
}

bool make_plan_r(const Layout& L, int GS, int C, int R, int smem_optin, Plan* out) {
  Plan pl;
  DecodeParams& P = pl.P;
  // staged bytes of a tile: all of a tile with at most R records per side
  const int cap = (int)(F_MAX + 2 * round16(4u * (uint32_t)R) + 64u * (uint32_t)R);
  const int kc_max = (L.max_k + C - 1) / C;
  // a stage: staged bytes (a tile block's head, or an anchor chunk), then the key-residual
  // terms of a tile
  const int sb = (int)align128((size_t)std::max(cap, CH * 256));
  P.o_rs = sb;
  P.o_pv = (int)align128((size_t)sb + (size_t)R * GS * 4);
  const int stage = (int)align128((size_t)P.o_pv + (size_t)(R + 1) * GS * 4);  // row R: spare
  // The value-weight table holds kt + 2 m rows for the value slots a CTA's tiles cover: kt, the
  // larger tile share of a CTA (where C does not divide a unit's tiles) times the unit's slots
  // per tile, plus the slot a first run continues; m, a margin for uneven runs, takes what the
  // ring leaves of the shared memory (at most kc_max).
  int kt = 1;
  for (const auto& sh : L.shape) {
    const long long tmax = (sh.nt + C - 1) / C;
    kt = std::max(kt, (int)(((long long)sh.k * tmax + sh.nt - 1) / std::max(1, sh.nt)) + 1);
  }
  auto layout = [&](int m) -> bool {
    size_t off = 0;
    auto take = [&](size_t bytes) {
      const size_t o = off;
      off = align128(off + bytes);
      return (int)o;
    };
    P.wrows = kt + 2 * m;
    P.o_sa = take((size_t)L.max_k * GS * 4);
    P.o_w = take((size_t)P.wrows * GS * 4);
    P.o_qfa = take(8 * 32 * 8);
    P.o_qfk = take((GS == 8 ? 2 : 1) * 8 * 32 * 8);  // [hi, lo for GS = 8][k-step][lane]
    P.o_qp = take((size_t)GS * 128 * 4);
    P.o_acc = take((size_t)GS * 128 * 4);
    P.o_opart = take((size_t)std::max(GS * 128, NTW * GS) * 4);
    P.o_misc = take((size_t)(((NTW * GS + 6 * GS + 4) * 4 + 15) & ~15) + 2 * 4 * std::max(GS, 4));
    P.o_meta = take(8 * 8);
    P.o_hdr = take(8 * 32);
    P.o_mslot = take((size_t)kMaxCluster * GS * 4);
    P.o_lslot = take((size_t)kMaxCluster * GS * 4);
    P.o_fslot = take((size_t)kMaxCluster * 4);
    P.o_ofin = take((size_t)(GS * 128 + 4 * kMaxCluster) * 4);  // C x per <= GS 128 + 4 C
    P.o_bar = take(5 * 8 * 8);
    P.o_ovf = take((size_t)GS * 128 * 4);
    P.o_pfb = take((size_t)2 * ((R + 15) / 16) * 512);
    P.o_ring = (int)off;
    return true;
  };
  layout(0);
  const long long room = (long long)smem_optin - (long long)P.o_ring;
  if (room < 2LL * stage) return false;
  const int NS = (int)std::min<long long>(8, room / stage);
  // the margin: whole 128-byte steps of the table within what NS stages leave over
  const long long spare = room - (long long)NS * stage;
  const int m = (int)std::min<long long>(kc_max, std::max<long long>(0, (spare - 128) / (2LL * GS * 4)));
  layout(m);
  if ((long long)P.o_ring + (long long)NS * stage > (long long)smem_optin) return false;
  P.NS = NS;
  P.stage_bytes = stage;
  P.R = R;
  P.cap = cap;
  pl.smem = (size_t)P.o_ring + (size_t)NS * stage;
  pl.C = C;
  *out = pl;
  return true;
}

// Records staged per tile and side: 1.35x the densest unit's mean plus slack, at most 320;
// records of a denser tile beyond these take the CUDA-core paths, which cost far more.
int full_r(const Layout& L) {
  const int R = (int)(T * max_density(L) * 1.35) + 32;
  return std::min(320, std::max(16, (R + 15) & ~15));
}

// full_only: only the full staged count; else fewer records when the ring would otherwise hold
// less than two stages (the last resort: most records then take the CUDA-core paths).
bool make_plan(const Layout& L, int GS, int C, int smem_optin, Plan* out, std::string* why, bool full_only = false) {
  for (int R = full_r(L); R >= (full_only ? full_r(L) : 16); R -= 16)
    if (make_plan_r(L, GS, C, R, smem_optin, out)) return true;
  *why = "shared memory: anchor tables of k = " + std::to_string(L.max_k) + " with " + std::to_string(GS) +
         " query heads per CTA leave room for fewer than 2 pipeline stages";
  return false;
}

// Estimated makespan, in tile times, of a launch with clusters of C CTAs of which nc can be
// resident at once: clusters start in launch order (unit-major, then head group) on the first
// free slot, and a cluster lasts as long as its CTA with the most tiles, plus a fixed cost
// (query preparation, cluster barriers, combine: about six tiles) and its anchor chunks.
double estimate_makespan(const Layout& L, int nhg, int C, int nc) {
  constexpr double kFixed = 6.0, kPerChunk = 0.3;
  std::priority_queue<double, std::vector<double>, std::greater<double>> slots;
  for (int i = 0; i < nc; ++i) slots.push(0.0);
  double end = 0.0;
  for (const auto& s : L.shape) {
    const double cost = (double)((s.nt + C - 1) / C) + kFixed + kPerChunk * (double)(((s.k + C - 1) / C + CH - 1) / CH);
    for (int g = 0; g < nhg; ++g) {
      const double t = slots.top() + cost;
      slots.pop();
      slots.push(t);
      end = std::max(end, t);
    }
  }
  return end;
}

// Launch configuration per (device, G, units, lengths, density, cluster override):
// computed once (attributes, occupancy query), then reused, so that a call made
// during CUDA-graph capture only issues the launch itself.
struct LaunchKey {
  int dev, G, units, max_len, max_k, cluster_env;
  long long dens_key;
  bool operator<(const LaunchKey& o) const {
    return std::tie(dev, G, units, max_len, max_k, cluster_env, dens_key) <
           std::tie(o.dev, o.G, o.units, o.max_len, o.max_k, o.cluster_env, o.dens_key);
  }
};

using KernelFn = void (*)(const DecodeParams);
template <int GS>
KernelFn decode_kernel() {
  return akv_decode_kernel<GS>;
}

template <int GS>
int plan_for(const Layout& L, const LaunchKey& key, int vunits, Plan* out, std::string* why) {
  static std::mutex mu;
  static std::map<LaunchKey, Plan> cache;
  {
    std::lock_guard<std::mutex> lk(mu);
    auto it = cache.find(key);
    if (it != cache.end()) {
      *out = it->second;
      return 0;
    }
  }
  const DeviceInfo di = device_info();
  // The attribute is per kernel, not per launch: raise it to the device limit
  // once, so that every cached configuration stays launchable.
  const KernelFn kfn = decode_kernel<GS>();
  cudaError_t e = cudaFuncSetAttribute(kfn, cudaFuncAttributeMaxDynamicSharedMemorySize, di.smem_optin);
  if (e != cudaSuccess) return (int)e;
  e = cudaFuncSetAttribute(kfn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  if (e != cudaSuccess) return (int)e;
  // Cluster size: the most CTAs per unit such that every cluster is resident at once (one CTA
  // per SM), no more CTAs than tiles in the longest unit.  Sizes are tried downwards one by
  // one: a GPU whose processor clusters cannot hold 16 CTAs each may still hold 12 or 13.
  // A size whose tables leave room for the full staged count comes first: the value-weight table
  // shrinks with C (ceil(k / C) anchors), so when it is too large at every all-resident size a
  // larger C is taken even if its clusters run in more than one wave; only when no size fits is
  // the staged count cut.
  const int C0 = std::max(1, std::min<int>(std::min<long long>(kMaxCluster, std::max<long long>(1, di.sms / std::max(1, vunits))),
                                           L.max_tiles));
  auto clusters_fit = [&](int C, const Plan& pl) -> int {  // clusters resident at once (C > 1)
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(C * vunits), 1, 1);
    cfg.blockDim = dim3(NT, 1, 1);
    cfg.dynamicSmemBytes = pl.smem;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = C;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int nclusters = 0;
    if (cudaOccupancyMaxActiveClusters(&nclusters, kfn, &cfg) != cudaSuccess) {
      cudaGetLastError();
      return 0;
    }
    return nclusters;
  };
  Plan pl;
  int C = 0;
  if (key.cluster_env >= 1 && key.cluster_env <= kMaxCluster) {  // requested size, or the next that fits once
    for (int c = key.cluster_env; c >= 1 && !C; --c)
      if (make_plan(L, GS, c, di.smem_optin, &pl, why) && (c == 1 || clusters_fit(c, pl) >= 1)) C = c;
    if (!C) return -1;
  } else {
    // 1. among the sizes whose tables leave room for the full staged count, the one with the
    //    shortest estimated makespan (estimate_makespan; resident clusters from the occupancy
    //    query, so sizes whose clusters cannot all be resident pay for their extra waves)
    double best = 0.0;
    for (int c = std::min(kMaxCluster, std::max(1, L.max_tiles)); c >= 1; --c) {
      Plan cand;
      std::string w;
      if (!make_plan(L, GS, c, di.smem_optin, &cand, &w, true)) continue;
      const int nc = c == 1 ? di.sms : clusters_fit(c, cand);
      if (nc < 1) continue;
      const double t = estimate_makespan(L, vunits / (int)L.shape.size(), c, nc);
      if (!C || t < best * 0.97) {  // near-ties keep the larger size: the anchor work spreads wider
        C = c;
        best = t;
        pl = cand;
      }
    }
    // 2. else a cut staged count at the largest all-resident size
    for (int c = C0; c >= 1 && !C; --c)
      if (make_plan(L, GS, c, di.smem_optin, &pl, why) && (c == 1 || clusters_fit(c, pl) >= vunits)) C = c;
    if (!C) return -1;
  }
  std::lock_guard<std::mutex> lk(mu);
  cache[key] = pl;
  *out = pl;
  return 0;
}

template <int GS>
int launch_g(const Layout& L, const akv_params& p, const void* arena, const void* q, void* out, float* out_f32,
             float sm_scale, void* stream, std::string* why) {
  const int units = (int)L.shape.size();
  const int nhg = L.G / GS;
  const int vunits = units * nhg;
  int dev = 0;
  cudaGetDevice(&dev);
  // testing controls (akv_decode_set_debug): a requested cluster size, and the failure-detection
  // hook with which every CTA withholds the last tile of its stream (its stage is not used
  // again), so the waits on it run out after their bound and the outputs become NaN
  const int cenv = g_debug_cluster.load(std::memory_order_relaxed);
  const int drop = g_debug_withhold.load(std::memory_order_relaxed);
  const LaunchKey key{dev, L.G, units, L.max_len, L.max_k, cenv, (long long)(max_density(L) * 1e6)};
  Plan pl;
  int err = plan_for<GS>(L, key, vunits, &pl, why);
  if (err) return err;
  DecodeParams P = pl.P;
  P.arena = (const uint8_t*)arena;
  P.q = (const __nv_bfloat16*)q;
  P.out = (__nv_bfloat16*)out;
  P.out_f32 = out_f32;
  P.n_kv_heads = p.n_kv_heads;
  P.n_q_heads = p.n_q_heads;
  P.G = L.G;
  P.nhg = nhg;
  P.rotate = (p.flags & AKV_FLAG_ROTATE) ? 1 : 0;
  P.scale_log2 = sm_scale * kLog2e;
  P.sign_lo = L.header.sign_bits[0];
  P.sign_hi = L.header.sign_bits[1];
  P.cluster = pl.C;
  P.drop_last = drop;

  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(pl.C * vunits), 1, 1);
  cfg.blockDim = dim3(NT, 1, 1);
  cfg.dynamicSmemBytes = pl.smem;
  cfg.stream = (cudaStream_t)stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = pl.C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  // the launch may overlap the tail of a preceding decode launch (griddepcontrol in the kernel)
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  cudaError_t e = cudaLaunchKernelEx(&cfg, decode_kernel<GS>(), P);
  if (e != cudaSuccess) return (int)e;
  return (int)cudaGetLastError();
}

}  // namespace

std::atomic<int> g_debug_cluster{0}, g_debug_withhold{0};

int launch_decode(const Layout& L, const akv_params& p, const void* arena, const void* q, void* out, float* out_f32,
                  float sm_scale, void* stream, std::string* why) {
  // a CTA serves all G query heads of its KV head; for G = 8, when the anchor tables of eight
  // heads leave no room for the pipeline, two CTA groups of four heads each
  switch (L.G) {
    case 1: return launch_g<1>(L, p, arena, q, out, out_f32, sm_scale, stream, why);
    case 2: return launch_g<2>(L, p, arena, q, out, out_f32, sm_scale, stream, why);
    case 4: return launch_g<4>(L, p, arena, q, out, out_f32, sm_scale, stream, why);
    case 8: {
      const int e = launch_g<8>(L, p, arena, q, out, out_f32, sm_scale, stream, why);
      if (e != -1) return e;
      why->clear();
      return launch_g<4>(L, p, arena, q, out, out_f32, sm_scale, stream, why);
    }
  }
  *why = "unsupported group size";
  return -1;
}

const char* cuda_error_string(int err) { return cudaGetErrorString((cudaError_t)err); }

}  // namespace akv
