// Split-K decode attention read directly from the AnchorKV compressed cache.
//
// One thread-block cluster per (request, KV head) unit; its C CTAs split the
// unit's positions and its anchors.  Eq. 3 is folded into Eq. 4: no key or
// value row is ever rebuilt in memory.
//
// Warp-specialised CTA (15 warps):
//   producer warp     streams one sequence of items through a ring of shared-
//                     memory stages with 16-byte asynchronous copies (cp.async),
//                     each lane's copies completing an mbarrier arrival:
//                     [anchor-key chunks] [position tiles] [anchor-value chunks]
//   2 key-residual warps  per tile: q' . c for the staged key slots on tensor
//                     cores, straight from the packed 2-bit codes (q' = H(s o q)/128,
//                     Appendix A.1 Eq. 12, as fp16 high + low parts)
//   8 token warps     phase 1: anchor scores S_A = q . k_a of the CTA's anchor slice
//                     (bf16 tensor cores), gathered cluster-wide through DSMEM;
//                     per tile: logits gamma_i S_A[a(i)] + residual term, p = 2^(l - m),
//                     value weights scattered per anchor, value-residual operands;
//                     phase 3: cluster combine and the anchor-value product
//   4 value-residual warps  per tile: sum of (p scale) c over the staged value
//                     slots on tensor cores, in the rotated domain
// Stages are handed between the roles with mbarriers, so different roles work on
// different tiles at the same time.
//
// The exponent reference m is the largest anchor score of each query row.  Anchors
// are tokens of the unit, so m never exceeds the true maximum logit (sums cannot
// overflow unless a logit exceeds m by more than 2^120, which is flagged), and all
// CTAs of a cluster share the same m: no running-max rescaling is needed and the
// cluster combine (Eq. 4 normaliser and numerator) is a plain sum.
// Every wait on an mbarrier is bounded; a wait that runs out marks the CTA failed,
// the CTA stops issuing and consuming, and its outputs become NaN.
#include <cooperative_groups.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdio>
#include <cstdlib>
#include <map>
#include <mutex>
#include <string>
#include <tuple>

#include "akv_internal.h"

namespace cg = cooperative_groups;

namespace akv {
namespace {

// warp roles
constexpr int NTW = 8;                 // token warps (warps 0 .. 7)
constexpr int NTT = NTW * 32;          // token threads
constexpr int W_KRES = NTW;            // key-residual warps
constexpr int NKR = 2;
constexpr int W_VRES = W_KRES + NKR;   // value-residual warps
constexpr int NVR = 4;
constexpr int W_PROD = W_VRES + NVR;   // producer warp
constexpr int NT = (W_PROD + 1) * 32;  // 480 threads
constexpr int T = 512;                 // positions per tile
constexpr int PPT = T / NTT;           // positions per token thread
static_assert(PPT == 2, "the token pass reads two stream words per thread");
static_assert(NTW % NVR == 0, "value-residual warps release a stage with NTW / NVR arrivals each");
constexpr int ROWS = 32;   // anchor rows per chunk
constexpr int ROWB = 272;  // shared-memory stride of a staged anchor row (256 B + 16 B pad)
constexpr int ROWE = 80;   // stride of an expanded row of 32 codes (64 B + 16 B pad)
constexpr int kMaxCluster = 16;
constexpr unsigned kWaitLimit = 1u << 22;
constexpr float kLog2e = 1.4426950408889634f;

// stage sub-buffers of a position tile (bytes)
constexpr int ST_K = 0;                 // [T] u32
constexpr int ST_V = ST_K + 4 * T;      // [T] u32
constexpr int ST_BMK = ST_V + 4 * T;    // [T/64] u64
constexpr int ST_PFK = ST_BMK + T / 8;  // [T/64] u32 (+pad)
constexpr int ST_BMV = ST_PFK + 64;
constexpr int ST_PFV = ST_BMV + T / 8;
constexpr int ST_REC = ST_PFV + 64;  // records follow, 128-aligned

struct DecodeParams {
  const uint8_t* arena;
  const __nv_bfloat16* q;
  __nv_bfloat16* out;
  float* out_f32;
  int n_kv_heads, n_q_heads, cluster, rotate, max_k;
  float scale_log2;
  unsigned long long sign_lo, sign_hi;
  int R, NS, stage_bytes, max_tiles;
  int o_sa, o_w, o_bk, o_bv, o_qfa, o_qfk, o_qp, o_acc, o_opart, o_e, o_misc, o_bar, o_ring;
  int o_cdk, o_sck, o_cdv, o_scv, o_rsb, o_pfb;  // inside a stage
};

// ---- device helpers ---------------------------------------------------------------

__device__ __forceinline__ uint32_t smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
// Bounded wait for completion of the phase with the given parity; false if the bound ran out.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity) {
  for (unsigned i = 0; i < kWaitLimit; ++i) {
    uint32_t done;
    asm volatile(
        "{ .reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2; selp.u32 %0, 1, 0, p; }"
        : "=r"(done)
        : "r"(bar), "r"(parity)
        : "memory");
    if (done) return true;
  }
  return false;
}
// 16-byte asynchronous copy global -> shared (L2 only); completion is tracked by
// cp_arrive_on on an mbarrier.  Many small copies from all lanes keep far more bytes in
// flight per SM than a few bulk copies of the small pieces a tile is made of.
__device__ __forceinline__ void cp16(uint32_t dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}
// Copies `bytes` (a multiple of 16) with the lanes of one warp.
__device__ __forceinline__ void warp_copy(uint32_t dst, const void* src, uint32_t bytes, int lane) {
  const uint8_t* s = reinterpret_cast<const uint8_t*>(src);
  for (uint32_t o = (uint32_t)lane * 16u; o < bytes; o += 512u) cp16(dst + o, s + o);
}
// The mbarrier counts one arrival from this thread once all of its earlier cp.async copies landed.
__device__ __forceinline__ void cp_arrive_on(uint32_t bar) {
  asm volatile("cp.async.mbarrier.arrive.noinc.shared::cta.b64 [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ void red_add(float* p, float v) {
  asm volatile("red.shared.add.f32 [%0], %1;" ::"r"(smem_u32(p)), "f"(v) : "memory");
}
__device__ __forceinline__ void tw_sync() { asm volatile("bar.sync 1, %0;" ::"n"(NTT) : "memory"); }
__device__ __forceinline__ void named_sync(int id, int n) { asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(n) : "memory"); }
__device__ __forceinline__ void named_arrive(int id, int n) {
  asm volatile("bar.arrive %0, %1;" ::"r"(id), "r"(n) : "memory");
}
__device__ __forceinline__ void mbar_arrive_cnt(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void cluster_arrive() { asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory"); }
__device__ __forceinline__ void cluster_wait() { asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory"); }

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

// Two 2-bit codes, at bits 0-1 and 16-17 of x, as an fp16 pair of exact small
// integers: OR them into the mantissa of 1024.0 (0x6400), then subtract 1024.
__device__ __forceinline__ uint32_t codes2_to_h2(uint32_t x) {
  uint32_t t, r;
  asm("lop3.b32 %0, %1, %2, %3, 0xEA;" : "=r"(t) : "r"(x), "r"(0x00030003u), "r"(0x64006400u));
  asm("sub.f16x2 %0, %1, %2;" : "=r"(r) : "r"(t), "r"(0x64006400u));
  return r;
}
__device__ __forceinline__ uint32_t pack_h2(__half lo, __half hi) {
  return (uint32_t)__half_as_ushort(lo) | ((uint32_t)__half_as_ushort(hi) << 16);
}
__device__ __forceinline__ uint32_t pack_b2(__nv_bfloat16 lo, __nv_bfloat16 hi) {
  return (uint32_t)__bfloat16_as_ushort(lo) | ((uint32_t)__bfloat16_as_ushort(hi) << 16);
}
__device__ __forceinline__ float half_lo(uint32_t w) {
  return __half2float(__ushort_as_half((unsigned short)(w & 0xFFFFu)));
}
__device__ __forceinline__ float half_hi(uint32_t w) { return __half2float(__ushort_as_half((unsigned short)(w >> 16))); }

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

// Unnormalised 128-point Walsh-Hadamard transform of `rows` rows in shared
// memory, by the token warps.
__device__ void tw_wht_rows(float* v, int rows) {
  for (int h = 1; h < 128; h <<= 1) {
    tw_sync();
    for (int e = threadIdx.x; e < rows * 64; e += NTT) {
      const int r = e >> 6, pr = e & 63;
      const int j = (pr / h) * 2 * h + (pr % h);
      float* x = v + r * 128;
      const float a = x[j], b = x[j + h];
      x[j] = a + b;
      x[j + h] = a - b;
    }
  }
  tw_sync();
}

// Sections of one unit.
struct UnitView {
  int S, k, nk, nv;
  const __nv_bfloat16* AK;
  const __nv_bfloat16* AV;
  const uint32_t* stK;
  const uint32_t* stV;
  const uint64_t* bmK;
  const uint32_t* pfK;
  const uint64_t* bmV;
  const uint32_t* pfV;
  const uint8_t* cdK;
  const uint32_t* scK;
  const uint8_t* cdV;
  const uint32_t* scV;
};

__device__ __forceinline__ UnitView unit_view(const uint8_t* A, int u) {
  const akv_unit_desc* d = reinterpret_cast<const akv_unit_desc*>(A + 256) + u;
  UnitView v;
  v.S = d->len;
  v.k = d->n_anchors;
  v.nk = d->n_res_k;
  v.nv = d->n_res_v;
  v.AK = reinterpret_cast<const __nv_bfloat16*>(A + d->off_anchor_k);
  v.AV = reinterpret_cast<const __nv_bfloat16*>(A + d->off_anchor_v);
  v.stK = reinterpret_cast<const uint32_t*>(A + d->off_stream_k);
  v.stV = reinterpret_cast<const uint32_t*>(A + d->off_stream_v);
  v.bmK = reinterpret_cast<const uint64_t*>(A + d->off_bitmap_k);
  v.pfK = reinterpret_cast<const uint32_t*>(A + d->off_prefix_k);
  v.bmV = reinterpret_cast<const uint64_t*>(A + d->off_bitmap_v);
  v.pfV = reinterpret_cast<const uint32_t*>(A + d->off_prefix_v);
  v.cdK = A + d->off_codes_k;
  v.scK = reinterpret_cast<const uint32_t*>(A + d->off_scales_k);
  v.cdV = A + d->off_codes_v;
  v.scV = reinterpret_cast<const uint32_t*>(A + d->off_scales_v);
  return v;
}

__host__ __device__ constexpr uint32_t round16(uint32_t x) { return (x + 15u) & ~15u; }

// One of the ten copies of a position tile, chosen by lane (0-9): K and V streams,
// bitmaps and prefix words of both sides, then codes and (scale, min) words of the staged
// residual slots of both sides.  Used for both the stage copy and the L2 prefetch.
struct LaneCopy {
  const void* src;
  uint32_t bytes;
  uint32_t dst;
};

__device__ __forceinline__ LaneCopy tile_copy_lane(const DecodeParams& P, const UnitView& U, int lane, int t0, int te,
                                                   int skl, int skh, int svl, int svh) {
  LaneCopy c{nullptr, 0u, 0u};
  const int npos = te - t0;
  const int w0 = t0 >> 6, nw = (npos + 63) >> 6;
  const int nK = min(skh - skl, P.R), nV = min(svh - svl, P.R);
  switch (lane) {
    case 0: c = {U.stK + t0, round16(npos * 4), (uint32_t)ST_K}; break;
    case 1: c = {U.stV + t0, round16(npos * 4), (uint32_t)ST_V}; break;
    case 2: c = {U.bmK + w0, round16(nw * 8), (uint32_t)ST_BMK}; break;
    case 3: c = {U.pfK + w0, round16(nw * 4), (uint32_t)ST_PFK}; break;
    case 4: c = {U.bmV + w0, round16(nw * 8), (uint32_t)ST_BMV}; break;
    case 5: c = {U.pfV + w0, round16(nw * 4), (uint32_t)ST_PFV}; break;
    case 6:
      if (nK > 0) c = {U.cdK + (size_t)skl * 32, (uint32_t)nK * 32, (uint32_t)P.o_cdk};
      break;
    case 7:
      if (nK > 0) c = {U.scK + (skl & ~3), (uint32_t)(((skl + nK + 3) & ~3) - (skl & ~3)) * 4, (uint32_t)P.o_sck};
      break;
    case 8:
      if (nV > 0) c = {U.cdV + (size_t)svl * 32, (uint32_t)nV * 32, (uint32_t)P.o_cdv};
      break;
    case 9:
      if (nV > 0) c = {U.scV + (svl & ~3), (uint32_t)(((svl + nV + 3) & ~3) - (svl & ~3)) * 4, (uint32_t)P.o_scv};
      break;
    default: break;
  }
  return c;
}

template <int G>
__global__ void __launch_bounds__(NT, 1) akv_decode_kernel(const DecodeParams P) {
  extern __shared__ __align__(128) uint8_t smem[];
  cg::cluster_group cluster = cg::this_cluster();
  const int C = P.cluster;
  const int rank = (int)cluster.block_rank();
  const int u = blockIdx.x / C;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int c4 = lane & 3, r8 = lane >> 2;
  const UnitView U = unit_view(P.arena, u);
  const int S = U.S, k = U.k;

  float* SA = reinterpret_cast<float*>(smem + P.o_sa);
  float* Wt = reinterpret_cast<float*>(smem + P.o_w);
  int* bK = reinterpret_cast<int*>(smem + P.o_bk);
  int* bV = reinterpret_cast<int*>(smem + P.o_bv);
  uint2* qfa = reinterpret_cast<uint2*>(smem + P.o_qfa);
  uint4* qfk = reinterpret_cast<uint4*>(smem + P.o_qfk);
  float* qp = reinterpret_cast<float*>(smem + P.o_qp);
  float* accs = reinterpret_cast<float*>(smem + P.o_acc);
  float* opart = reinterpret_cast<float*>(smem + P.o_opart);
  uint8_t* ebuf = smem + P.o_e;
  float* red = reinterpret_cast<float*>(smem + P.o_misc);  // [NTW][G]
  float* sq = red + NTW * G;                              // [G]
  float* mref = sq + G;                                   // [G]
  float* cl = mref + G;                                   // [G]
  float* pms = cl + G;                                    // [G]
  float* ltot = pms + G;                                  // [G]
  volatile int* failed = reinterpret_cast<volatile int*>(ltot + G);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + P.o_bar);
  uint8_t* ring = smem + P.o_ring;
  const int NS = P.NS;
  const int max_k = P.max_k;
  // per stage: copies of an anchor chunk landed (full_c) / of a position tile landed (full_t);
  // stage free again (empty); key-residual terms ready (rsr); probabilities written (pr).
  // Chunk items and tiles complete different barriers, so every waiter sees every phase of
  // the barriers it waits on.
  auto bar_full_c = [&](int s) { return smem_u32(bars + s); };
  auto bar_full_t = [&](int s) { return smem_u32(bars + NS + s); };
  auto bar_empty = [&](int s) { return smem_u32(bars + 2 * NS + s); };
  auto bar_rs = [&](int s) { return smem_u32(bars + 3 * NS + s); };
  auto bar_p = [&](int s) { return smem_u32(bars + 4 * NS + s); };
  auto stage = [&](int s) { return ring + (size_t)s * P.stage_bytes; };

  // this CTA's anchor slice and position range
  const int a_per = ((k + C - 1) / C + 15) / 16 * 16;
  const int a0 = min(k, rank * a_per), a1 = min(k, a0 + a_per);
  const int chunk = ((S + C - 1) / C + T - 1) / T * T;
  const int p0 = min(S, rank * chunk), p1 = min(S, p0 + chunk);
  const int n_ka = (a1 - a0 + ROWS - 1) / ROWS;
  const int n_t = (p1 - p0 + T - 1) / T;
  const int n_items = 2 * n_ka + n_t;
  const int R = P.R;
  // phase index, on its stage's barrier, of item `it` (anchor chunks and tiles counted apart)
  auto item_phase = [&](int it) -> uint32_t {
    if (it < n_ka) return (uint32_t)(it / NS);
    if (it < n_ka + n_t) return (uint32_t)((it - n_ka) / NS);
    const int s = it % NS, cj = it - n_ka - n_t;
    const int ka_on_s = n_ka > s ? (n_ka - 1 - s) / NS + 1 : 0;
    return (uint32_t)(ka_on_s + cj / NS);
  };
  auto is_tile = [&](int it) { return it >= n_ka && it < n_ka + n_t; };

  if (tid == 0) {
    for (int s = 0; s < NS; ++s) {
      mbar_init(bar_full_c(s), 32);  // one arrival per producer lane, when its copies landed
      mbar_init(bar_full_t(s), 32);
      mbar_init(bar_empty(s), NTW);
      mbar_init(bar_rs(s), NKR);
      mbar_init(bar_p(s), NTW);
    }
    *failed = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();

  // =========================== producer warp ===================================
  if (warp == W_PROD) {
    cluster_arrive();  // B1: this warp never blocks on anything behind B1 before it waits on B1
    for (int i = lane; i <= n_t; i += 32) {
      const int pos = min(p0 + i * T, p1);
      bK[i] = pos >= S ? U.nk : (int)U.pfK[pos >> 6];
      bV[i] = pos >= S ? U.nv : (int)U.pfV[pos >> 6];
    }
    __syncwarp();
    bool ok = true, b1_done = false;
    for (int it = 0; it < n_items; ++it) {
      if (it == n_ka + n_t) {  // anchor values are consumed after B2: let B1 complete, arrive on B2
        cluster_wait();
        cluster_arrive();
        b1_done = true;
      }
      const int s = it % NS;
      const uint32_t use = (uint32_t)(it / NS);
      if (it >= NS) ok = mbar_wait(bar_empty(s), (use - 1) & 1u);
      if (!ok || *failed) {
        *failed = 1;
        break;
      }
      uint8_t* st = stage(s);
      if (it < n_ka || it >= n_ka + n_t) {
        // anchor rows into padded shared-memory rows (272-byte stride: conflict-free fragment loads)
        const bool val = it >= n_ka + n_t;
        const int ci = val ? it - n_ka - n_t : it;
        const int r0 = a0 + ci * ROWS, nr = min(a1 - r0, ROWS);
        const uint8_t* src = reinterpret_cast<const uint8_t*>((val ? U.AV : U.AK) + (size_t)r0 * 128);
        for (int q = lane; q < nr * 16; q += 32) cp16(smem_u32(st + (q >> 4) * ROWB + (q & 15) * 16), src + q * 16);
        cp_arrive_on(bar_full_c(s));
      } else {
        const int tl = it - n_ka;
        const int t0 = p0 + tl * T, te = min(t0 + T, p1);
#pragma unroll 1
        for (int j = 0; j < 10; ++j) {
          const LaneCopy c = tile_copy_lane(P, U, j, t0, te, bK[tl], bK[tl + 1], bV[tl], bV[tl + 1]);
          if (c.bytes) warp_copy(smem_u32(st + c.dst), c.src, c.bytes, lane);
        }
        cp_arrive_on(bar_full_t(s));
      }
      __syncwarp();
    }
    if (!b1_done) {
      cluster_wait();
      cluster_arrive();
    }
    // every copy this warp started has landed before the CTA may exit
    asm volatile("cp.async.wait_all;" ::: "memory");
    cluster_wait();  // B2
    cluster_arrive();
    cluster_wait();  // B3
    cluster_arrive();
    cluster_wait();  // B4
    return;
  }

  // =========================== key-residual warps ================================
  // q' . c for the staged key slots of each tile, 8 slots per mma group, fragments of q'
  // (fp16 high and low parts) held in registers.
  if (warp >= W_KRES && warp < W_KRES + NKR) {
    const int kw = warp - W_KRES;
    cluster_arrive();  // B1
    named_sync(2, NTW * 32 + NKR * 32);  // q' fragments written by the token warps
    uint4 af[8];
#pragma unroll
    for (int ks = 0; ks < 8; ++ks) af[ks] = qfk[ks * 32 + lane];
    bool ok = true;
    for (int tl = 0; tl < n_t; ++tl) {
      const int s = (n_ka + tl) % NS;
      if (ok && !*failed) {
        ok = mbar_wait(bar_full_t(s), (uint32_t)(tl / NS) & 1u);
        if (!ok) *failed = 1;
      }
      if (ok && !*failed) {
        const uint8_t* st = stage(s);
        const int skl = bK[tl], nK = min(bK[tl + 1] - skl, R);
        const uint8_t* cd = st + P.o_cdk;
        const uint32_t* sc = reinterpret_cast<const uint32_t*>(st + P.o_sck) + (skl & 3);
        float* rs = reinterpret_cast<float*>(const_cast<uint8_t*>(st) + P.o_rsb);
        for (int g8 = kw; g8 * 8 < nK; g8 += NKR) {
          const int sl = g8 * 8 + r8;  // the slot whose codes this lane feeds (B column r8)
          uint4 w0 = make_uint4(0u, 0u, 0u, 0u), w1 = w0;
          if (sl < nK) {
            w0 = *reinterpret_cast<const uint4*>(cd + (size_t)sl * 32);
            w1 = *reinterpret_cast<const uint4*>(cd + (size_t)sl * 32 + 16);
          }
          const uint32_t wd[8] = {w0.x, w0.y, w0.z, w0.w, w1.x, w1.y, w1.z, w1.w};
          float d[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
          for (int ks = 0; ks < 8; ++ks) {
            const uint32_t x = wd[ks] >> (4 * c4);
            mma_f16(d, af[ks], codes2_to_h2(x), codes2_to_h2(x >> 2));
          }
          if (r8 < G) {  // D rows r8 (high parts) and r8 + 8 (low parts), columns 2c, 2c+1
#pragma unroll
            for (int e2 = 0; e2 < 2; ++e2) {
              const int sl2 = g8 * 8 + 2 * c4 + e2;
              if (sl2 < nK) {
                const uint32_t smn = sc[sl2];
                rs[sl2 * G + r8] = half_hi(smn) * sq[r8] + half_lo(smn) * (d[e2] + d[2 + e2]);
              }
            }
          }
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(bar_rs(s));
    }
    cluster_wait();  // B1
    cluster_arrive();
    cluster_wait();  // B2
    cluster_arrive();
    cluster_wait();  // B3
    cluster_arrive();
    cluster_wait();  // B4
    return;
  }

  // =========================== value-residual warps ==============================
  // sum over staged value slots of (p scale) c, 16 slots per mma group; warp vw owns
  // the 32 coordinates 32 vw .. 32 vw + 31 of the rotated-domain accumulator.
  if (warp >= W_VRES && warp < W_VRES + NVR) {
    const int vw = warp - W_VRES;
    cluster_arrive();  // B1
    float accV[4][4];
#pragma unroll
    for (int nb = 0; nb < 4; ++nb)
#pragma unroll
      for (int e = 0; e < 4; ++e) accV[nb][e] = 0.f;
    uint8_t* ew = ebuf + vw * 16 * ROWE;
    bool ok = true;
    for (int tl = 0; tl < n_t; ++tl) {
      const int s = (n_ka + tl) % NS;
      const uint32_t par = (uint32_t)(tl / NS) & 1u;
      if (ok && !*failed) {
        ok = mbar_wait(bar_full_t(s), par) && mbar_wait(bar_p(s), par);
        if (!ok) *failed = 1;
      }
      if (ok && !*failed) {
        const uint8_t* st = stage(s);
        const int nV = min(bV[tl + 1] - bV[tl], R);
        const uint8_t* cd = st + P.o_cdv;
        const uint8_t* pf = st + P.o_pfb;
        for (int grp = 0; grp * 16 < nV; ++grp) {
          const int n = lane >> 1, hh = lane & 1;
          const int sl = grp * 16 + n;
          uint32_t x = 0;
          if (sl < nV) x = *reinterpret_cast<const uint32_t*>(cd + (size_t)sl * 32 + 8 * vw + 4 * hh);
          uint4 v0, v1;
          {
            const uint32_t lo = x & 0xFFFFu, y = lo | (lo << 14);  // code 2m at bit 4m, code 2m+1 at 4m + 16
            v0 = make_uint4(codes2_to_h2(y), codes2_to_h2(y >> 4), codes2_to_h2(y >> 8), codes2_to_h2(y >> 12));
            const uint32_t hi = x >> 16, z = hi | (hi << 14);
            v1 = make_uint4(codes2_to_h2(z), codes2_to_h2(z >> 4), codes2_to_h2(z >> 8), codes2_to_h2(z >> 12));
          }
          *reinterpret_cast<uint4*>(ew + n * ROWE + hh * 32) = v0;
          *reinterpret_cast<uint4*>(ew + n * ROWE + hh * 32 + 16) = v1;
          __syncwarp();
          const uint4 a = *reinterpret_cast<const uint4*>(pf + grp * 512 + lane * 16);
          const int mi = lane >> 3, ri = lane & 7;
#pragma unroll
          for (int half = 0; half < 2; ++half) {
            uint32_t b00, b01, b10, b11;
            ldsm_x4_trans(smem_u32(ew + ((mi & 1) * 8 + ri) * ROWE + half * 32 + (mi >> 1) * 16), b00, b01, b10, b11);
            mma_f16(accV[2 * half], a, b00, b01);
            mma_f16(accV[2 * half + 1], a, b10, b11);
          }
          __syncwarp();
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive_cnt(bar_empty(s), NTW / NVR);
    }
    // rows r8 (high parts) + r8 + 8 (low parts); overflow slots were added by the token warps,
    // which zeroed the accumulator in phase 0
    named_sync(3, NTW * 32 + NVR * 32);
    if (r8 < G) {
#pragma unroll
      for (int nb = 0; nb < 4; ++nb) {
        const int col = 32 * vw + 8 * nb + 2 * c4;
        accs[r8 * 128 + col] += accV[nb][0] + accV[nb][2];
        accs[r8 * 128 + col + 1] += accV[nb][1] + accV[nb][3];
      }
    }
    cluster_wait();  // B1
    cluster_arrive();
    cluster_wait();  // B2
    cluster_arrive();
    cluster_wait();  // B3
    cluster_arrive();
    cluster_wait();  // B4
    return;
  }

  // =========================== token warps =======================================
  const int b = u / P.n_kv_heads, h = u % P.n_kv_heads;
  const size_t qrow0 = ((size_t)b * P.n_q_heads + (size_t)h * G) * 128;

  // ---- phase 0: query rows, rotated query, tensor-core fragments ----
  for (int e = tid; e < G * 128; e += NTT) {
    const int j = e & 127;
    const float x = __bfloat162float(P.q[qrow0 + e]);
    const unsigned long long sb = j < 64 ? P.sign_lo : P.sign_hi;
    qp[e] = (P.rotate && ((sb >> (j & 63)) & 1ull)) ? -x : x;
    accs[e] = 0.f;
  }
  for (int e = a0 * G + tid; e < a1 * G; e += NTT) SA[e] = 0.f;
  for (int s = 0; s < NS; ++s)
    for (int e = tid; e < ((R + 15) / 16) * 128; e += NTT)
      reinterpret_cast<uint32_t*>(stage(s) + P.o_pfb)[e] = 0u;
  if (P.rotate) tw_wht_rows(qp, G);
  else tw_sync();
  {
    const float f = P.rotate ? P.scale_log2 * (1.0f / 128.0f) : P.scale_log2;
    for (int e = tid; e < G * 128; e += NTT) qp[e] *= f;
  }
  tw_sync();
  if (warp < G) {
    float s = 0.f;
    for (int j = lane; j < 128; j += 32) s += qp[warp * 128 + j];
    s = warp_sum(s);
    if (lane == 0) sq[warp] = s;
  }
  {
    // fragment (k-step ks, lane ln): one per token thread (8 k-steps x 32 lanes)
    const int ks = tid >> 5, ln = tid & 31, g = ln >> 2, c = ln & 3;
    uint2 fa = make_uint2(0u, 0u);
    uint4 fk = make_uint4(0u, 0u, 0u, 0u);
    if (g < G) {
      // anchor-score B operand: q in bf16, k order permuted so a thread's dims are contiguous
      const __nv_bfloat16* qr = P.q + qrow0 + (size_t)g * 128;
      const int d0 = 32 * (ks >> 1) + 8 * c + 4 * (ks & 1);
      fa.x = pack_b2(qr[d0], qr[d0 + 1]);
      fa.y = pack_b2(qr[d0 + 2], qr[d0 + 3]);
      // key-residual A operand: rows g = q' high parts, rows g + 8 = low parts; k index pairs
      // (2c, 2c+1) <-> coords (16ks + 2c, 16ks + 2c + 8), (2c+8, 2c+9) <-> (16ks + 2c + 1, 16ks + 2c + 9)
      const float* x = qp + g * 128 + 16 * ks + 2 * c;
      const __half h0 = __float2half_rn(x[0]), h8 = __float2half_rn(x[8]);
      const __half h1 = __float2half_rn(x[1]), h9 = __float2half_rn(x[9]);
      fk.x = pack_h2(h0, h8);
      fk.y = pack_h2(__float2half_rn(x[0] - __half2float(h0)), __float2half_rn(x[8] - __half2float(h8)));
      fk.z = pack_h2(h1, h9);
      fk.w = pack_h2(__float2half_rn(x[1] - __half2float(h1)), __float2half_rn(x[9] - __half2float(h9)));
    }
    qfa[ks * 32 + ln] = fa;
    qfk[ks * 32 + ln] = fk;
  }
  tw_sync();
  named_arrive(2, NTW * 32 + NKR * 32);  // the key-residual warps may read q' fragments and sq
  named_arrive(3, NTW * 32 + NVR * 32);  // the value-residual warps may add into accs

  bool ok = true;
  auto wait_item = [&](int i) -> const uint8_t* {
    const int s = i % NS;
    if (ok && !*failed) ok = mbar_wait(is_tile(i) ? bar_full_t(s) : bar_full_c(s), item_phase(i) & 1u);
    if (!ok) *failed = 1;
    return stage(s);
  };
  auto release_chunk = [&](int i) {
    __syncwarp();
    if (lane == 0) mbar_arrive(bar_empty(i % NS));
  };

  // ---- phase 1: anchor scores of this CTA's slice (bf16 tensor cores) ----
  for (int it = 0; it < n_ka; ++it) {
    const uint8_t* st = wait_item(it);
    if (!*failed) {
      const int r0 = a0 + it * ROWS, nr = min(a1 - r0, ROWS);
      const int blk = warp >> 2, j = warp & 3;  // 2 blocks of 16 rows x 4 pairs of k-steps
      const uint8_t* row0 = st + (16 * blk + r8) * ROWB + 64 * j + 16 * c4;
      const uint4 lo = *reinterpret_cast<const uint4*>(row0);
      const uint4 hi = *reinterpret_cast<const uint4*>(row0 + 8 * ROWB);
      float d[4] = {0.f, 0.f, 0.f, 0.f};
      const uint2 b0 = qfa[(2 * j) * 32 + lane], b1 = qfa[(2 * j + 1) * 32 + lane];
      mma_bf16(d, lo.x, hi.x, lo.y, hi.y, b0.x, b0.y);
      mma_bf16(d, lo.z, hi.z, lo.w, hi.w, b1.x, b1.y);
      const int ra = 16 * blk + r8, gc = 2 * c4;
      if (ra < nr) {
        if (gc < G) atomicAdd(&SA[(r0 + ra) * G + gc], d[0] * P.scale_log2);
        if (gc + 1 < G) atomicAdd(&SA[(r0 + ra) * G + gc + 1], d[1] * P.scale_log2);
      }
      if (ra + 8 < nr) {
        if (gc < G) atomicAdd(&SA[(r0 + ra + 8) * G + gc], d[2] * P.scale_log2);
        if (gc + 1 < G) atomicAdd(&SA[(r0 + ra + 8) * G + gc + 1], d[3] * P.scale_log2);
      }
    }
    release_chunk(it);
  }
  tw_sync();
  cluster_arrive();  // B1
  cluster_wait();
  // every entry outside this CTA's slice comes from the peer that owns its anchor
#pragma unroll 4
  for (int e = tid; e < k * G; e += NTT) {
    const int r = (e / G) / a_per;
    if (r != rank) SA[e] = cluster.map_shared_rank(SA, r)[e];
  }
  for (int e = tid; e < G * max_k; e += NTT) Wt[e] = 0.f;  // [G][max_k]: the scatter spreads over banks
  tw_sync();
  // Reference for the exponentials: the largest anchor score per query row.  Anchors are
  // tokens of the unit, so it never exceeds the true maximum logit; every CTA of the
  // cluster holds the same table and so the same reference, which makes the cluster
  // combine a plain sum.
  {
    float mx[G];
#pragma unroll
    for (int g = 0; g < G; ++g) mx[g] = -INFINITY;
    for (int a = tid; a < k; a += NTT)
#pragma unroll
      for (int g = 0; g < G; ++g) mx[g] = fmaxf(mx[g], SA[a * G + g]);
#pragma unroll
    for (int g = 0; g < G; ++g) {
      const float m = warp_max(mx[g]);
      if (lane == 0) red[warp * G + g] = m;
    }
    tw_sync();
    if (tid < G) {
      float m = red[tid];
      for (int w = 1; w < NTW; ++w) m = fmaxf(m, red[w * G + tid]);
      mref[tid] = m;
    }
    tw_sync();
  }
  float m_ref[G], l_part[G], pmin[G];
#pragma unroll
  for (int g = 0; g < G; ++g) {
    m_ref[g] = mref[g];
    l_part[g] = 0.f;
    pmin[g] = 0.f;
  }

  // ---- phase 2: position tiles ----
  bool overflow_risk = false;
  for (int tl = 0; tl < n_t; ++tl) {
    const int it = n_ka + tl;
    const int s = it % NS;
    const uint8_t* st = wait_item(it);
    if (ok && !*failed) {
      ok = mbar_wait(bar_rs(s), item_phase(it) & 1u);
      if (!ok) *failed = 1;
    }
    if (!*failed) {
      const int t0 = p0 + tl * T, te = min(t0 + T, p1);
      const int skl = bK[tl], svl = bV[tl];
      const int i0 = t0 + PPT * tid;
      const float* rsb = reinterpret_cast<const float*>(st + P.o_rsb);
      uint8_t* pfb = const_cast<uint8_t*>(st) + P.o_pfb;
      const uint32_t* scv = reinterpret_cast<const uint32_t*>(st + P.o_scv) + (svl & 3);
      const uint2 ek = *reinterpret_cast<const uint2*>(st + ST_K + 8 * tid);
      const uint2 ev = *reinterpret_cast<const uint2*>(st + ST_V + 8 * tid);
      const int wi = (PPT * tid) >> 6, bit0 = (PPT * tid) & 63;
      const uint64_t wk = reinterpret_cast<const uint64_t*>(st + ST_BMK)[wi];
      const uint64_t wv = reinterpret_cast<const uint64_t*>(st + ST_BMV)[wi];
      const int pk = (int)reinterpret_cast<const uint32_t*>(st + ST_PFK)[wi] - skl;
      const int pv = (int)reinterpret_cast<const uint32_t*>(st + ST_PFV)[wi] - svl;
#pragma unroll
      for (int pp = 0; pp < PPT; ++pp) {
        const int i = i0 + pp;
        if (i >= te) continue;
        const int bit = bit0 + pp;
        const uint64_t below = (1ull << bit) - 1ull;
        float lg[G];
        {
          const uint32_t e = pp ? ek.y : ek.x;
          const int a = min((int)(e & 0xFFFFu), k - 1);  // indices are < k by construction; never read past the table
          const float gam = half_hi(e);
          if constexpr (G % 4 == 0) {
#pragma unroll
            for (int g4 = 0; g4 < G; g4 += 4) {
              const float4 s4 = *reinterpret_cast<const float4*>(SA + a * G + g4);
              lg[g4] = gam * s4.x;
              lg[g4 + 1] = gam * s4.y;
              lg[g4 + 2] = gam * s4.z;
              lg[g4 + 3] = gam * s4.w;
            }
          } else {
#pragma unroll
            for (int g = 0; g < G; ++g) lg[g] = gam * SA[a * G + g];
          }
        }
        if ((wk >> bit) & 1ull) {  // key residual term
          const int sl = pk + __popcll(wk & below);
          if (sl < R) {
#pragma unroll
            for (int g = 0; g < G; ++g) lg[g] += rsb[sl * G + g];
          } else {  // beyond the staged slots (a locally dense tile): from global memory, on CUDA cores
            const int gs = skl + sl;
            const uint8_t* rec = U.cdK + (size_t)gs * 32;
            const uint32_t smn = U.scK[gs];
#pragma unroll
            for (int g = 0; g < G; ++g) {
              float dot = 0.f;
              for (int bb = 0; bb < 32; ++bb) {
                const uint32_t byte = rec[bb];
#pragma unroll
                for (int c = 0; c < 4; ++c) dot += qp[g * 128 + 4 * bb + c] * (float)((byte >> (2 * c)) & 3u);
              }
              lg[g] += half_hi(smn) * sq[g] + half_lo(smn) * dot;
            }
          }
        }
        const uint32_t e = pp ? ev.y : ev.x;
        const int a = min((int)(e & 0xFFFFu), k - 1);
        const float gam = half_hi(e);
        float p[G];
#pragma unroll
        for (int g = 0; g < G; ++g) {
          const float x = lg[g] - m_ref[g];
          overflow_risk |= x > 120.f;
          p[g] = exp2f(x);
          l_part[g] += p[g];
          red_add(&Wt[g * max_k + a], p[g] * gam);
        }
        if ((wv >> bit) & 1ull) {  // value residual: A operand of its 16-slot group, or overflow
          const int sl = pv + __popcll(wv & below);
          if (sl < R) {
            const uint32_t smn = scv[sl];
            const float scl = half_lo(smn), mn = half_hi(smn);
            const int grp = sl >> 4, kk = sl & 15;
            const int comp = (kk >> 3) * 2, hf = kk & 1, cc = (kk & 7) >> 1;
#pragma unroll
            for (int g = 0; g < G; ++g) {
              const float x = p[g] * scl;
              const __half hi = __float2half_rn(x);
              const __half lo = __float2half_rn(x - __half2float(hi));
              unsigned short* dst = reinterpret_cast<unsigned short*>(pfb + grp * 512 + (4 * g + cc) * 16);
              dst[comp * 2 + hf] = __half_as_ushort(hi);
              dst[(comp + 1) * 2 + hf] = __half_as_ushort(lo);
              pmin[g] += p[g] * mn;
            }
          } else {
            const int gs = svl + sl;
            const uint8_t* rec = U.cdV + (size_t)gs * 32;
            const uint32_t smn = U.scV[gs];
            const float scl = half_lo(smn), mn = half_hi(smn);
#pragma unroll
            for (int g = 0; g < G; ++g) {
              pmin[g] += p[g] * mn;
              const float ps = p[g] * scl;
              for (int bb = 0; bb < 32; ++bb) {
                const uint32_t byte = rec[bb];
#pragma unroll
                for (int c = 0; c < 4; ++c) atomicAdd(&accs[g * 128 + 4 * bb + c], ps * (float)((byte >> (2 * c)) & 3u));
              }
            }
          }
        }
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(bar_p(s));
  }
  if (overflow_risk) *failed = 1;  // a logit beyond 2^120 of the reference would overflow the sums

  // ---- per-CTA totals ----
#pragma unroll
  for (int g = 0; g < G; ++g) {
    const float sl = warp_sum(l_part[g]);
    const float pm = warp_sum(pmin[g]);
    if (lane == 0) {
      red[warp * G + g] = sl;
      opart[warp * G + g] = pm;  // scratch until phase 3
    }
  }
  tw_sync();
  if (tid < G) {
    float sl = 0.f, pm = 0.f;
    for (int w = 0; w < NTW; ++w) {
      sl += red[w * G + tid];
      pm += opart[w * G + tid];
    }
    cl[tid] = sl;
    pms[tid] = pm;
  }
  tw_sync();

  // ---- phase 3: combine across the cluster (one common reference: plain sums) ----
  cluster_arrive();  // B2
  cluster_wait();
  if (tid < G) {
    float Lt = 0.f;
    for (int r = 0; r < C; ++r) Lt += cluster.map_shared_rank(cl, r)[tid];
    ltot[tid] = Lt;
  }
  for (int e = tid; e < (a1 - a0) * G; e += NTT) {
    const int idx = (e / (a1 - a0)) * max_k + a0 + e % (a1 - a0);
    float v[kMaxCluster];
#pragma unroll
    for (int r = 0; r < kMaxCluster; ++r) v[r] = r < C ? cluster.map_shared_rank(Wt, r)[idx] : 0.f;
    float sw = 0.f;
#pragma unroll
    for (int r = 0; r < kMaxCluster; ++r) sw += v[r];
    Wt[idx] = sw;
  }
  tw_sync();
  // reduced weights of the slice times its anchor values (bf16 tensor cores, weights as hi + lo)
  float oacc[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
  for (int ci = 0; ci < n_ka; ++ci) {
    const int it = n_ka + n_t + ci;
    const uint8_t* st = wait_item(it);
    if (!*failed) {
      const int r0 = a0 + ci * ROWS, nr = min(a1 - r0, ROWS);
      for (int blk = 0; blk < 2 && 16 * blk < nr; ++blk) {
        const int mi = lane >> 3, ri = lane & 7;
        uint32_t b00, b01, b10, b11;
        ldsm_x4_trans(smem_u32(st + (16 * blk + (mi & 1) * 8 + ri) * ROWB + (16 * warp + (mi >> 1) * 8) * 2), b00,
                      b01, b10, b11);
        // rows past the slice hold stale bytes: clear their halves of B
        const int ka = 16 * blk + 2 * c4;
        const uint32_t m0 = (ka < nr ? 0xFFFFu : 0u) | (ka + 1 < nr ? 0xFFFF0000u : 0u);
        const uint32_t m1 = (ka + 8 < nr ? 0xFFFFu : 0u) | (ka + 9 < nr ? 0xFFFF0000u : 0u);
        b00 &= m0;
        b10 &= m0;
        b01 &= m1;
        b11 &= m1;
        uint32_t ah0 = 0, al0 = 0, ah2 = 0, al2 = 0;
        if (r8 < G) {
          const int kk[4] = {ka, ka + 1, ka + 8, ka + 9};
          __nv_bfloat16 hi[4], lo[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float w = kk[e] < nr ? Wt[r8 * max_k + r0 + kk[e]] : 0.f;
            hi[e] = __float2bfloat16_rn(w);
            lo[e] = __float2bfloat16_rn(w - __bfloat162float(hi[e]));
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
  // this CTA's value residuals (staged slots from the value-residual warps, overflow slots and
  // sum p * min from the token warps), then the inverse rotation once
  for (int e = tid; e < G * 128; e += NTT) accs[e] += pms[e >> 7];
  if (P.rotate) tw_wht_rows(accs, G);
  else tw_sync();
  for (int e = tid; e < G * 128; e += NTT) {
    const int j = e & 127;
    float r = accs[e];
    if (P.rotate) {
      const unsigned long long sb = j < 64 ? P.sign_lo : P.sign_hi;
      r = ((sb >> (j & 63)) & 1ull) ? -r : r;
      r *= (1.0f / 128.0f);
    }
    opart[e] = r;
  }
  tw_sync();
  if (r8 < G) {
#pragma unroll
    for (int nb = 0; nb < 2; ++nb) {
      const int col = 16 * warp + 8 * nb + 2 * c4;
      opart[r8 * 128 + col] += oacc[nb][0] + oacc[nb][2];
      opart[r8 * 128 + col + 1] += oacc[nb][1] + oacc[nb][3];
    }
  }
  tw_sync();
  cluster_arrive();  // B3
  cluster_wait();
  {
    const int E = G * 128;
    const int per = (E + C - 1) / C;
    const int e0 = rank * per, e1 = min(E, e0 + per);
    bool bad = false;
    for (int r = 0; r < C; ++r) bad |= cluster.map_shared_rank(const_cast<int*>(failed), r)[0] != 0;
    for (int e = e0 + tid; e < e1; e += NTT) {
      float v[kMaxCluster];
#pragma unroll
      for (int r = 0; r < kMaxCluster; ++r) v[r] = r < C ? cluster.map_shared_rank(opart, r)[e] : 0.f;
      float sum = 0.f;
#pragma unroll
      for (int r = 0; r < kMaxCluster; ++r) sum += v[r];
      const float y = bad ? __int_as_float(0x7FC00000) : sum / ltot[e >> 7];
      const size_t o = qrow0 + e;
      P.out[o] = __float2bfloat16_rn(y);
      if (P.out_f32) P.out_f32[o] = y;
    }
  }
  cluster_arrive();  // B4
  cluster_wait();
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

// Launch plan: shared-memory carve-up, ring depth, staged residual slots per tile, cluster size.
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

bool make_plan(const Layout& L, int G, int C, int smem_optin, Plan* out, std::string* why) {
  Plan pl;
  DecodeParams& P = pl.P;
  // residual slots staged per tile and side: 1.35x the densest unit's mean plus slack;
  // slots of a locally denser tile beyond these are taken from global memory by the token warps
  int R = (int)(T * max_density(L) * 1.35) + 24;
  R = std::min(T, std::max(16, (R + 15) & ~15));
  const int chunk = ((L.max_len + C - 1) / C + T - 1) / T * T;
  const int max_tiles = chunk / T;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off = align128(off + bytes);
    return (int)o;
  };
  const size_t tab = (size_t)((L.max_k * G + 3) & ~3) * 4;
  P.o_sa = take(tab);
  P.o_w = take(tab);
  P.o_bk = take((size_t)(max_tiles + 1) * 4);
  P.o_bv = take((size_t)(max_tiles + 1) * 4);
  P.o_qfa = take(8 * 32 * 8);
  P.o_qfk = take(8 * 32 * 16);
  P.o_qp = take((size_t)G * 128 * 4);
  P.o_acc = take((size_t)G * 128 * 4);
  P.o_opart = take((size_t)std::max(G * 128, NTW * G) * 4);
  P.o_e = take((size_t)NVR * 16 * ROWE);
  P.o_misc = take((size_t)(NTW * G + 6 * G + 4) * 4);
  P.o_bar = take(5 * 8 * 8);
  // a stage: streams, bitmaps and prefix words, staged records, then (beyond the footprint
  // of an anchor chunk, so chunk copies never touch them) residual terms and value operands
  P.o_cdk = (int)align128(ST_REC);
  P.o_sck = (int)align128(P.o_cdk + R * 32);
  P.o_cdv = (int)align128(P.o_sck + (R + 8) * 4);
  P.o_scv = (int)align128(P.o_cdv + R * 32);
  P.o_rsb = (int)align128(std::max(P.o_scv + (R + 8) * 4, ROWS * ROWB));
  P.o_pfb = (int)align128(P.o_rsb + R * G * 4);
  const int stage = (int)align128(P.o_pfb + ((R + 15) / 16) * 512);
  P.o_ring = (int)off;
  const long long room = (long long)smem_optin - (long long)off;
  if (room < 2LL * stage) {
    *why = "shared memory: anchor tables of k * G = " + std::to_string(L.max_k * G) +
           " leave room for fewer than 2 pipeline stages";
    return false;
  }
  const int NS = (int)std::min<long long>(8, room / stage);
  P.NS = NS;
  P.stage_bytes = stage;
  P.R = R;
  P.max_tiles = max_tiles;
  pl.smem = (size_t)P.o_ring + (size_t)NS * stage;
  pl.C = C;
  *out = pl;
  return true;
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

template <int G>
int plan_for(const Layout& L, const LaunchKey& key, Plan* out, std::string* why) {
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
  cudaError_t e = cudaFuncSetAttribute(akv_decode_kernel<G>, cudaFuncAttributeMaxDynamicSharedMemorySize, di.smem_optin);
  if (e != cudaSuccess) return (int)e;
  e = cudaFuncSetAttribute(akv_decode_kernel<G>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  if (e != cudaSuccess) return (int)e;
  // Cluster size: one CTA per SM for one wave, no more CTAs than tiles in the longest unit.
  int C = 1;
  while (C < kMaxCluster && (long long)key.units * (C * 2) <= di.sms && (C * 2) * T <= L.max_len + T - 1) C *= 2;
  if (key.cluster_env >= 1 && key.cluster_env <= kMaxCluster) C = key.cluster_env;
  Plan pl;
  for (;;) {
    if (!make_plan(L, G, C, di.smem_optin, &pl, why)) return -1;
    if (C == 1) break;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(C * key.units), 1, 1);
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
    e = cudaOccupancyMaxActiveClusters(&nclusters, akv_decode_kernel<G>, &cfg);
    // prefer a size whose clusters all fit at once; an explicit override only needs one to fit
    if (e == cudaSuccess && (nclusters >= key.units || (key.cluster_env == C && nclusters >= 1))) break;
    cudaGetLastError();
    C = (C & (C - 1)) ? C - 1 : C / 2;
  }
  std::lock_guard<std::mutex> lk(mu);
  cache[key] = pl;
  *out = pl;
  return 0;
}

template <int G>
int launch_g(const Layout& L, const akv_params& p, const void* arena, const void* q, void* out, float* out_f32,
             float sm_scale, void* stream, std::string* why) {
  const int units = (int)L.shape.size();
  int dev = 0;
  cudaGetDevice(&dev);
  int cenv = 0;
  if (const char* env = std::getenv("AKV_CLUSTER")) cenv = std::atoi(env);
  const LaunchKey key{dev, G, units, L.max_len, L.max_k, cenv, (long long)(max_density(L) * 1e6)};
  Plan pl;
  int err = plan_for<G>(L, key, &pl, why);
  if (err) return err;
  DecodeParams P = pl.P;
  P.arena = (const uint8_t*)arena;
  P.q = (const __nv_bfloat16*)q;
  P.out = (__nv_bfloat16*)out;
  P.out_f32 = out_f32;
  P.n_kv_heads = p.n_kv_heads;
  P.n_q_heads = p.n_q_heads;
  P.rotate = (p.flags & AKV_FLAG_ROTATE) ? 1 : 0;
  P.max_k = L.max_k;
  P.scale_log2 = sm_scale * kLog2e;
  P.sign_lo = L.header.sign_bits[0];
  P.sign_hi = L.header.sign_bits[1];
  P.cluster = pl.C;

  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(pl.C * units), 1, 1);
  cfg.blockDim = dim3(NT, 1, 1);
  cfg.dynamicSmemBytes = pl.smem;
  cfg.stream = (cudaStream_t)stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = pl.C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaError_t e = cudaLaunchKernelEx(&cfg, akv_decode_kernel<G>, P);
  if (e != cudaSuccess) return (int)e;
  return (int)cudaGetLastError();
}

}  // namespace

int launch_decode(const Layout& L, const akv_params& p, const void* arena, const void* q, void* out, float* out_f32,
                  float sm_scale, void* stream, std::string* why) {
  switch (L.G) {
    case 1: return launch_g<1>(L, p, arena, q, out, out_f32, sm_scale, stream, why);
    case 2: return launch_g<2>(L, p, arena, q, out, out_f32, sm_scale, stream, why);
    case 4: return launch_g<4>(L, p, arena, q, out, out_f32, sm_scale, stream, why);
    case 8: return launch_g<8>(L, p, arena, q, out, out_f32, sm_scale, stream, why);
  }
  *why = "unsupported group size";
  return -1;
}

const char* cuda_error_string(int err) { return cudaGetErrorString((cudaError_t)err); }

}  // namespace akv
