// Split-K decode attention read directly from the AnchorKV compressed cache.
//
// One thread-block cluster per (request, KV head) unit; its C CTAs split the
// unit's positions and its anchors.  Eq. 3 is folded into Eq. 4: no key or
// value row is ever rebuilt in memory.
//
// Warp roles per CTA: 8 compute warps and 1 producer warp.  The producer
// streams one sequence of items through a ring of shared-memory stages with
// bulk asynchronous copies (cp.async.bulk completing on mbarrier transaction
// counts) and prefetches later items into L2:
//   [anchor-key chunks of this CTA's slice] [position tiles] [anchor-value chunks]
// The compute warps consume the same sequence:
//   phase 0  q rows and the rotated-domain query q' = H(s o q)/128 (Appendix A.1,
//            Eq. 12); tensor-core fragments of q (bf16) and of q' (fp16 hi + lo)
//   phase 1  anchor scores S_A = q . k_a of the slice (bf16 mma.sync), then every
//            CTA gathers the full S_A table from its peers (DSMEM)
//   phase 2  per tile: key logits gamma_i S_A[a(i)] plus the residual term
//            min sum(q') + scale (q' . c), with q' . c on tensor cores straight
//            from the packed 2-bit codes; running max; p = 2^(l - m); value
//            weights scattered per anchor; value residuals accumulated in the
//            rotated domain on tensor cores (p * scale as fp16 hi + lo)
//   phase 3  cluster combine (max / sum rescale of Eq. 4) through DSMEM; each CTA
//            reduces its slice of the value weights and multiplies it by its
//            anchor values on tensor cores, inverse-rotates its residual
//            accumulator once (Appendix E.1), then partial outputs are summed
//            and normalised.
// Every wait on an mbarrier is bounded; a wait that runs out marks the CTA
// failed, the CTA stops issuing and consuming, and its outputs become NaN.
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

constexpr int NCW = 8;         // compute warps
constexpr int NCT = NCW * 32;  // compute threads
constexpr int NT = NCT + 32;   // plus the producer warp
constexpr int T = 512;         // positions per tile
constexpr int PPT = T / NCT;   // positions per compute thread
static_assert(PPT == 2, "the token pass reads two stream words per thread");
constexpr int ROWS = 32;   // anchor rows per chunk
constexpr int ROWB = 272;  // shared-memory stride of a staged anchor row (256 B + 16 B pad)
constexpr int ROWE = 48;   // stride of an expanded row of 16 codes (32 B + 16 B pad)
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
  int R, NS, stage_bytes, max_tiles, pf_items;
  int o_sa, o_w, o_bk, o_bv, o_qfa, o_qfk, o_qs, o_qp, o_rs, o_pf, o_e, o_acc, o_opart, o_misc, o_bar, o_ring;
  int o_cdk, o_sck, o_cdv, o_scv;  // record buffers inside a stage
};

// ---- device helpers ---------------------------------------------------------------

__device__ __forceinline__ uint32_t smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
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
__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
               "l"(src), "r"(bytes), "r"(bar)
               : "memory");
}
__device__ __forceinline__ void bulk_prefetch(const void* src, uint32_t bytes) {
  if (bytes) asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(src), "r"(bytes) : "memory");
}
__device__ __forceinline__ void cw_sync() { asm volatile("bar.sync 1, %0;" ::"n"(NCT) : "memory"); }
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
// memory, by the compute warps.
__device__ void cw_wht_rows(float* v, int rows) {
  for (int h = 1; h < 128; h <<= 1) {
    cw_sync();
    for (int e = threadIdx.x; e < rows * 64; e += NCT) {
      const int r = e >> 6, pr = e & 63;
      const int j = (pr / h) * 2 * h + (pr % h);
      float* x = v + r * 128;
      const float a = x[j], b = x[j + h];
      x[j] = a + b;
      x[j + h] = a - b;
    }
  }
  cw_sync();
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

// Byte ranges of one position tile (used for both the stage copy and the L2 prefetch):
// streams, bitmaps and prefix words of both sides (6), codes and scales of both sides (4).
constexpr int kTileCopies = 10;
struct TileCopy {
  const void* src[kTileCopies];
  uint32_t bytes[kTileCopies];
  uint32_t dst[kTileCopies];
  int n;
  uint32_t total;
};

__device__ __forceinline__ void tile_copy_plan(const DecodeParams& P, const UnitView& U, int t0, int te, int skl,
                                               int skh, int svl, int svh, TileCopy& c) {
  c.n = 0;
  c.total = 0;
  auto add = [&](const void* src, uint32_t bytes, uint32_t dst) {
    if (!bytes || c.n == kTileCopies) return;
    c.src[c.n] = src;
    c.bytes[c.n] = bytes;
    c.dst[c.n] = dst;
    c.total += bytes;
    ++c.n;
  };
  const int npos = te - t0;
  const int w0 = t0 >> 6, nw = (npos + 63) >> 6;
  add(U.stK + t0, round16(npos * 4), ST_K);
  add(U.stV + t0, round16(npos * 4), ST_V);
  add(U.bmK + w0, round16(nw * 8), ST_BMK);
  add(U.pfK + w0, round16(nw * 4), ST_PFK);
  add(U.bmV + w0, round16(nw * 8), ST_BMV);
  add(U.pfV + w0, round16(nw * 4), ST_PFV);
  const int nK = min(skh - skl, P.R), nV = min(svh - svl, P.R);
  if (nK > 0) {
    add(U.cdK + (size_t)skl * 32, (uint32_t)nK * 32, P.o_cdk);
    const int s0 = skl & ~3, s1 = (skl + nK + 3) & ~3;
    add(U.scK + s0, (uint32_t)(s1 - s0) * 4, P.o_sck);
  }
  if (nV > 0) {
    add(U.cdV + (size_t)svl * 32, (uint32_t)nV * 32, P.o_cdv);
    const int s0 = svl & ~3, s1 = (svl + nV + 3) & ~3;
    add(U.scV + s0, (uint32_t)(s1 - s0) * 4, P.o_scv);
  }
}

template <int G>
__global__ void __launch_bounds__(NT, 1) akv_decode_kernel(const DecodeParams P) {
  extern __shared__ __align__(128) uint8_t smem[];
  cg::cluster_group cluster = cg::this_cluster();
  const int C = P.cluster;
  const int rank = (int)cluster.block_rank();
  const int u = blockIdx.x / C;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const UnitView U = unit_view(P.arena, u);
  const int S = U.S, k = U.k;

  float* SA = reinterpret_cast<float*>(smem + P.o_sa);
  float* Wt = reinterpret_cast<float*>(smem + P.o_w);
  int* bK = reinterpret_cast<int*>(smem + P.o_bk);
  int* bV = reinterpret_cast<int*>(smem + P.o_bv);
  uint2* qfa = reinterpret_cast<uint2*>(smem + P.o_qfa);
  uint4* qfk = reinterpret_cast<uint4*>(smem + P.o_qfk);
  float* qs = reinterpret_cast<float*>(smem + P.o_qs);
  float* qp = reinterpret_cast<float*>(smem + P.o_qp);
  float* rs = reinterpret_cast<float*>(smem + P.o_rs);
  uint8_t* pfrag = smem + P.o_pf;
  uint8_t* ebuf = smem + P.o_e;
  float* accs = reinterpret_cast<float*>(smem + P.o_acc);
  float* opart = reinterpret_cast<float*>(smem + P.o_opart);
  float* red = reinterpret_cast<float*>(smem + P.o_misc);
  float* sq = red + NCW * G;
  float* cm = sq + G;
  float* cl = cm + G;
  float* ltot = cl + G;
  float* peer_m = ltot + G;
  float* peer_l = peer_m + kMaxCluster * G;
  float* facs = peer_l + kMaxCluster * G;
  volatile int* failed = reinterpret_cast<volatile int*>(facs + kMaxCluster * G);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + P.o_bar);
  uint8_t* ring = smem + P.o_ring;
  const int NS = P.NS;

  // this CTA's anchor slice and position range
  const int a_per = ((k + C - 1) / C + 15) / 16 * 16;
  const int a0 = min(k, rank * a_per), a1 = min(k, a0 + a_per);
  const int chunk = ((S + C - 1) / C + T - 1) / T * T;
  const int p0 = min(S, rank * chunk), p1 = min(S, p0 + chunk);
  const int n_ka = (a1 - a0 + ROWS - 1) / ROWS;
  const int n_t = (p1 - p0 + T - 1) / T;
  const int n_items = 2 * n_ka + n_t;

  if (tid == 0) {
    for (int s = 0; s < NS; ++s) {
      mbar_init(smem_u32(bars + s), 1);
      mbar_init(smem_u32(bars + NS + s), NCW);
    }
    *failed = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();

  // =========================== producer warp ===================================
  if (warp == NCW) {
    cluster_arrive();  // B1; this warp never waits on anything behind B1 before it waits on B1
    for (int i = lane; i <= n_t; i += 32) {
      const int pos = min(p0 + i * T, p1);
      bK[i] = pos >= S ? U.nk : (int)U.pfK[pos >> 6];
      bV[i] = pos >= S ? U.nv : (int)U.pfV[pos >> 6];
    }
    __syncwarp();
    auto prefetch_item = [&](int it) {
      if (it >= n_items || lane != 0) return;
      if (it < n_ka || it >= n_ka + n_t) {
        const bool val = it >= n_ka + n_t;
        const int ci = val ? it - n_ka - n_t : it;
        const int r0 = a0 + ci * ROWS, r1 = min(a1, r0 + ROWS);
        bulk_prefetch((val ? U.AV : U.AK) + (size_t)r0 * 128, (uint32_t)(r1 - r0) * 256);
      } else {
        const int tl = it - n_ka;
        const int t0 = p0 + tl * T, te = min(t0 + T, p1);
        TileCopy c;
        tile_copy_plan(P, U, t0, te, bK[tl], bK[tl + 1], bV[tl], bV[tl + 1], c);
        for (int j = 0; j < c.n; ++j) bulk_prefetch(c.src[j], c.bytes[j]);
      }
    };
    for (int it = 0; it < min(P.pf_items, n_items); ++it) prefetch_item(it);
    bool ok = true, b1_done = false;
    int issued = 0;
    for (int it = 0; it < n_items; ++it) {
      if (it == n_ka + n_t) {  // anchor values are consumed after B2: let B1 complete and arrive on B2
        cluster_wait();
        cluster_arrive();
        b1_done = true;
      }
      const int s = it % NS;
      const uint32_t use = (uint32_t)(it / NS);
      if (it >= NS) ok = mbar_wait(smem_u32(bars + NS + s), (use - 1) & 1u);
      if (!ok || *failed) {
        *failed = 1;
        break;
      }
      prefetch_item(it + P.pf_items);
      uint8_t* st = ring + (size_t)s * P.stage_bytes;
      if (it < n_ka || it >= n_ka + n_t) {
        const bool val = it >= n_ka + n_t;
        const int ci = val ? it - n_ka - n_t : it;
        const int r0 = a0 + ci * ROWS, nr = min(a1 - r0, ROWS);
        if (lane == 0) mbar_expect_tx(smem_u32(bars + s), (uint32_t)nr * 256);
        __syncwarp();
        if (lane < nr)
          bulk_g2s(smem_u32(st + lane * ROWB), (val ? U.AV : U.AK) + (size_t)(r0 + lane) * 128, 256,
                   smem_u32(bars + s));
      } else if (lane == 0) {
        const int tl = it - n_ka;
        const int t0 = p0 + tl * T, te = min(t0 + T, p1);
        TileCopy c;
        tile_copy_plan(P, U, t0, te, bK[tl], bK[tl + 1], bV[tl], bV[tl + 1], c);
        mbar_expect_tx(smem_u32(bars + s), c.total);
        for (int j = 0; j < c.n; ++j) bulk_g2s(smem_u32(st + c.dst[j]), c.src[j], c.bytes[j], smem_u32(bars + s));
      }
      __syncwarp();
      ++issued;
    }
    if (!b1_done) {
      cluster_wait();
      cluster_arrive();
    }
    // every copy this warp started has landed before the CTA may exit
    for (int s = 0; s < NS && s < issued; ++s) {
      const int last = s + ((issued - 1 - s) / NS) * NS;
      mbar_wait(smem_u32(bars + s), (uint32_t)(last / NS) & 1u);
    }
    cluster_wait();    // B2
    cluster_arrive();  // B3
    cluster_wait();
    cluster_arrive();  // B4
    cluster_wait();
    return;
  }

  // =========================== compute warps ===================================
  const int b = u / P.n_kv_heads, h = u % P.n_kv_heads;
  const size_t qrow0 = ((size_t)b * P.n_q_heads + (size_t)h * G) * 128;
  const int c4 = lane & 3, r8 = lane >> 2;

  // ---- phase 0: query rows, rotated query, tensor-core fragments ----
  for (int e = tid; e < G * 128; e += NCT) {
    const int j = e & 127;
    const float x = __bfloat162float(P.q[qrow0 + e]);
    qs[e] = x;
    const unsigned long long sb = j < 64 ? P.sign_lo : P.sign_hi;
    qp[e] = (P.rotate && ((sb >> (j & 63)) & 1ull)) ? -x : x;
  }
  for (int e = a0 * G + tid; e < a1 * G; e += NCT) SA[e] = 0.f;
  if (P.rotate) cw_wht_rows(qp, G);
  else cw_sync();
  {
    const float f = P.rotate ? P.scale_log2 * (1.0f / 128.0f) : P.scale_log2;
    for (int e = tid; e < G * 128; e += NCT) qp[e] *= f;
  }
  cw_sync();
  if (warp < G) {
    float s = 0.f;
    for (int j = lane; j < 128; j += 32) s += qp[warp * 128 + j];
    s = warp_sum(s);
    if (lane == 0) sq[warp] = s;
  }
  {
    // fragment (k-step ks, lane ln): one per compute thread (8 k-steps x 32 lanes)
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
  for (int e = tid; e < ((P.R + 15) / 16) * 128; e += NCT) reinterpret_cast<uint32_t*>(pfrag)[e] = 0u;
  cw_sync();

  int it = 0;
  bool ok = true;
  auto wait_item = [&](int i) -> const uint8_t* {
    const int s = i % NS;
    if (ok && !*failed) ok = mbar_wait(smem_u32(bars + s), (uint32_t)(i / NS) & 1u);
    if (!ok) *failed = 1;
    return ring + (size_t)s * P.stage_bytes;
  };
  auto release_item = [&](int i) {
    __syncwarp();
    if (lane == 0) mbar_arrive(smem_u32(bars + NS + (i % NS)));
  };

  // ---- phase 1: anchor scores of this CTA's slice (bf16 tensor cores) ----
  for (; it < n_ka; ++it) {
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
    release_item(it);
  }
  cw_sync();
  cluster_arrive();  // B1
  cluster_wait();
  for (int r = 0; r < C; ++r) {
    if (r == rank) continue;
    const int b0r = min(k, r * a_per), b1r = min(k, b0r + a_per);
    const float* rem = cluster.map_shared_rank(SA, r);
    for (int e = b0r * G + tid; e < b1r * G; e += NCT) SA[e] = rem[e];
  }
  for (int e = tid; e < k * G; e += NCT) Wt[e] = 0.f;
  cw_sync();

  // ---- phase 2: position tiles ----
  float accV[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
  float m_run[G], l_part[G], pmin[G];
#pragma unroll
  for (int g = 0; g < G; ++g) {
    m_run[g] = -1e30f;
    l_part[g] = 0.f;
    pmin[g] = 0.f;
  }
  const int R = P.R;
  uint8_t* ew = ebuf + warp * 16 * ROWE;
  for (int tl = 0; tl < n_t; ++tl, ++it) {
    const uint8_t* st = wait_item(it);
    if (*failed) {
      release_item(it);
      continue;
    }
    const int t0 = p0 + tl * T, te = min(t0 + T, p1);
    const int skl = bK[tl], skh = bK[tl + 1], svl = bV[tl], svh = bV[tl + 1];
    const int i0 = t0 + PPT * tid;
    float lg[PPT][G];
    int slotK[PPT], slotV[PPT];
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
      const int bit = bit0 + pp;
      const uint64_t below = (1ull << bit) - 1ull;
      slotK[pp] = (i < te && ((wk >> bit) & 1ull)) ? pk + __popcll(wk & below) : -1;
      slotV[pp] = (i < te && ((wv >> bit) & 1ull)) ? pv + __popcll(wv & below) : -1;
      if (i < te) {
        const uint32_t e = pp ? ek.y : ek.x;
        const int a = min((int)(e & 0xFFFFu), k - 1);  // indices are < k by construction; never read past the table
        const float gam = half_hi(e);
        if constexpr (G % 4 == 0) {
#pragma unroll
          for (int g4 = 0; g4 < G; g4 += 4) {
            const float4 s4 = *reinterpret_cast<const float4*>(SA + a * G + g4);
            lg[pp][g4] = gam * s4.x;
            lg[pp][g4 + 1] = gam * s4.y;
            lg[pp][g4 + 2] = gam * s4.z;
            lg[pp][g4 + 3] = gam * s4.w;
          }
        } else {
#pragma unroll
          for (int g = 0; g < G; ++g) lg[pp][g] = gam * SA[a * G + g];
        }
      } else {
#pragma unroll
        for (int g = 0; g < G; ++g) lg[pp][g] = -INFINITY;
      }
    }
    // key residual terms on tensor cores, in rounds of at most R slots (rounds after the
    // first read their records from global memory)
    const int nK = skh - skl;
    for (int r0 = 0; r0 < nK; r0 += R) {
      const int nr = min(R, nK - r0);
      const uint8_t* cd = r0 == 0 ? st + P.o_cdk : U.cdK + (size_t)(skl + r0) * 32;
      const uint32_t* sc = r0 == 0 ? reinterpret_cast<const uint32_t*>(st + P.o_sck) + (skl & 3) : U.scK + skl + r0;
      for (int g8 = warp; g8 * 8 < nr; g8 += NCW) {
        const int sl = g8 * 8 + r8;  // the slot whose codes this lane feeds (B column r8)
        uint4 w0 = make_uint4(0u, 0u, 0u, 0u), w1 = w0;
        if (sl < nr) {
          w0 = *reinterpret_cast<const uint4*>(cd + (size_t)sl * 32);
          w1 = *reinterpret_cast<const uint4*>(cd + (size_t)sl * 32 + 16);
        }
        const uint32_t wd[8] = {w0.x, w0.y, w0.z, w0.w, w1.x, w1.y, w1.z, w1.w};
        float d[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int ks = 0; ks < 8; ++ks) {
          const uint32_t x = wd[ks] >> (4 * c4);
          mma_f16(d, qfk[ks * 32 + lane], codes2_to_h2(x), codes2_to_h2(x >> 2));
        }
        if (r8 < G) {  // D rows r8 (high parts) and r8 + 8 (low parts), columns 2c, 2c+1
#pragma unroll
          for (int e2 = 0; e2 < 2; ++e2) {
            const int sl2 = g8 * 8 + 2 * c4 + e2;
            if (sl2 < nr) {
              const uint32_t smn = sc[sl2];
              rs[sl2 * G + r8] = half_hi(smn) * sq[r8] + half_lo(smn) * (d[e2] + d[2 + e2]);
            }
          }
        }
      }
      cw_sync();
#pragma unroll
      for (int pp = 0; pp < PPT; ++pp) {
        const int sl = slotK[pp] - r0;
        if (sl >= 0 && sl < nr) {
#pragma unroll
          for (int g = 0; g < G; ++g) lg[pp][g] += rs[sl * G + g];
        }
      }
      if (r0 + R < nK) cw_sync();
    }
    // running max over the tile
#pragma unroll
    for (int g = 0; g < G; ++g) {
      float mx = lg[0][g];
#pragma unroll
      for (int pp = 1; pp < PPT; ++pp) mx = fmaxf(mx, lg[pp][g]);
      mx = warp_max(mx);
      if (lane == 0) red[warp * G + g] = mx;
    }
    cw_sync();
    bool grow = false;
    float fac[G];
#pragma unroll
    for (int g = 0; g < G; ++g) {
      float mx = red[g];
#pragma unroll
      for (int w = 1; w < NCW; ++w) mx = fmaxf(mx, red[w * G + g]);
      const float nm = fmaxf(m_run[g], mx);
      fac[g] = exp2f(m_run[g] - nm);
      grow |= nm > m_run[g];
      m_run[g] = nm;
    }
    if (grow) {  // uniform across the compute warps
      for (int e = tid; e < k * G; e += NCT) Wt[e] *= fac[e % G];
      float fq = 0.f;
#pragma unroll
      for (int g = 0; g < G; ++g) {
        l_part[g] *= fac[g];
        pmin[g] *= fac[g];
        if (g == r8) fq = fac[g];
      }
#pragma unroll
      for (int nb = 0; nb < 2; ++nb)
#pragma unroll
        for (int e = 0; e < 4; ++e) accV[nb][e] *= fq;
      cw_sync();
    }
    // probabilities and the value-weight scatter
#pragma unroll
    for (int pp = 0; pp < PPT; ++pp) {
      if (i0 + pp < te) {
        const uint32_t e = pp ? ev.y : ev.x;
        const int a = min((int)(e & 0xFFFFu), k - 1);
        const float gam = half_hi(e);
#pragma unroll
        for (int g = 0; g < G; ++g) {
          const float p = exp2f(lg[pp][g] - m_run[g]);
          lg[pp][g] = p;
          l_part[g] += p;
          atomicAdd(&Wt[a * G + g], p * gam);
        }
      }
    }
    // value residuals on tensor cores, in rounds of at most R slots
    const int nV = svh - svl;
    for (int r0 = 0; r0 < nV; r0 += R) {
      const int nr = min(R, nV - r0);
      const uint8_t* cd = r0 == 0 ? st + P.o_cdv : U.cdV + (size_t)(svl + r0) * 32;
      const uint32_t* sc = r0 == 0 ? reinterpret_cast<const uint32_t*>(st + P.o_scv) + (svl & 3) : U.scV + svl + r0;
      // A operand of each group of 16 slots: rows g = (p * scale) high parts, rows g + 8 = low parts
#pragma unroll
      for (int pp = 0; pp < PPT; ++pp) {
        const int sl = slotV[pp] - r0;
        if (sl >= 0 && sl < nr) {
          const uint32_t smn = sc[sl];
          const float scl = half_lo(smn), mn = half_hi(smn);
          const int grp = sl >> 4, kk = sl & 15;
          const int comp = (kk >> 3) * 2, hf = kk & 1, cc = (kk & 7) >> 1;
#pragma unroll
          for (int g = 0; g < G; ++g) {
            const float x = lg[pp][g] * scl;
            const __half hi = __float2half_rn(x);
            const __half lo = __float2half_rn(x - __half2float(hi));
            unsigned short* dst = reinterpret_cast<unsigned short*>(pfrag + grp * 512 + (4 * g + cc) * 16);
            dst[comp * 2 + hf] = __half_as_ushort(hi);
            dst[(comp + 1) * 2 + hf] = __half_as_ushort(lo);
            pmin[g] += lg[pp][g] * mn;
          }
        }
      }
      cw_sync();
      // each warp owns the 16 coordinates 16w .. 16w + 15 for every group
      const int ngrp = (nr + 15) >> 4;
      for (int grp = 0; grp < ngrp; ++grp) {
        const int n = lane >> 1, hh = lane & 1;
        const int sl = grp * 16 + n;
        uint32_t x = 0;
        if (sl < nr) x = *reinterpret_cast<const unsigned short*>(cd + (size_t)sl * 32 + 4 * warp + 2 * hh);
        const uint32_t y = x | (x << 14);  // code 2k at bit 4k, code 2k+1 at bit 4k+16
        uint4 v;
        v.x = codes2_to_h2(y);
        v.y = codes2_to_h2(y >> 4);
        v.z = codes2_to_h2(y >> 8);
        v.w = codes2_to_h2(y >> 12);
        *reinterpret_cast<uint4*>(ew + n * ROWE + hh * 16) = v;
        __syncwarp();
        uint32_t b00, b01, b10, b11;
        const int mi = lane >> 3, ri = lane & 7;
        ldsm_x4_trans(smem_u32(ew + ((mi & 1) * 8 + ri) * ROWE + (mi >> 1) * 16), b00, b01, b10, b11);
        const uint4 a = *reinterpret_cast<const uint4*>(pfrag + grp * 512 + lane * 16);
        mma_f16(accV[0], a, b00, b01);
        mma_f16(accV[1], a, b10, b11);
        __syncwarp();
      }
      if (r0 + R < nV) cw_sync();
    }
    release_item(it);
  }

  // ---- per-CTA totals ----
#pragma unroll
  for (int g = 0; g < G; ++g) {
    const float s = warp_sum(l_part[g]);
    const float pm = warp_sum(pmin[g]);
    if (lane == 0) {
      red[warp * G + g] = s;
      opart[warp * G + g] = pm;  // scratch until phase 3
    }
  }
  cw_sync();
  if (tid < G) {
    float s = 0.f, pm = 0.f;
    for (int w = 0; w < NCW; ++w) {
      s += red[w * G + tid];
      pm += opart[w * G + tid];
    }
    cl[tid] = s;
#pragma unroll
    for (int g = 0; g < G; ++g)
      if (g == tid) cm[tid] = m_run[g];
    peer_l[tid] = pm;  // scratch: this CTA's sum of p * min per row
  }
  cw_sync();
  if (r8 < G) {  // rotated-domain residual accumulator: high + low rows, plus sum p * min on every coordinate
#pragma unroll
    for (int nb = 0; nb < 2; ++nb) {
      const int col = 16 * warp + 8 * nb + 2 * c4;
      accs[r8 * 128 + col] = accV[nb][0] + accV[nb][2] + peer_l[r8];
      accs[r8 * 128 + col + 1] = accV[nb][1] + accV[nb][3] + peer_l[r8];
    }
  }
  cw_sync();

  // ---- phase 3: combine across the cluster ----
  cluster_arrive();  // B2
  cluster_wait();
  if (tid < C * G) {
    const int r = tid / G, g = tid % G;
    peer_m[tid] = cluster.map_shared_rank(cm, r)[g];
    peer_l[tid] = cluster.map_shared_rank(cl, r)[g];
  }
  cw_sync();
  if (tid < G) {
    float M = -1e30f;
    for (int r = 0; r < C; ++r) M = fmaxf(M, peer_m[r * G + tid]);
    float Lt = 0.f;
    for (int r = 0; r < C; ++r) {
      const float f = exp2f(peer_m[r * G + tid] - M);
      facs[r * G + tid] = f;
      Lt += f * peer_l[r * G + tid];
    }
    ltot[tid] = Lt;
  }
  cw_sync();
  for (int e = a0 * G + tid; e < a1 * G; e += NCT) {
    const int g = e % G;
    float s = 0.f;
    for (int r = 0; r < C; ++r) s += facs[r * G + g] * cluster.map_shared_rank(Wt, r)[e];
    Wt[e] = s;
  }
  cw_sync();
  // reduced weights of the slice times its anchor values (bf16 tensor cores, weights as hi + lo)
  float oacc[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
  for (int ci = 0; ci < n_ka; ++ci, ++it) {
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
            const float w = kk[e] < nr ? Wt[(r0 + kk[e]) * G + r8] : 0.f;
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
    release_item(it);
  }
  // this CTA's value residuals: its own rescale factor, then the inverse rotation once
  for (int e = tid; e < G * 128; e += NCT) accs[e] *= facs[rank * G + (e >> 7)];
  if (P.rotate) cw_wht_rows(accs, G);
  else cw_sync();
  for (int e = tid; e < G * 128; e += NCT) {
    const int j = e & 127;
    float r = accs[e];
    if (P.rotate) {
      const unsigned long long sb = j < 64 ? P.sign_lo : P.sign_hi;
      r = ((sb >> (j & 63)) & 1ull) ? -r : r;
      r *= (1.0f / 128.0f);
    }
    opart[e] = r;
  }
  cw_sync();
  if (r8 < G) {
#pragma unroll
    for (int nb = 0; nb < 2; ++nb) {
      const int col = 16 * warp + 8 * nb + 2 * c4;
      opart[r8 * 128 + col] += oacc[nb][0] + oacc[nb][2];
      opart[r8 * 128 + col + 1] += oacc[nb][1] + oacc[nb][3];
    }
  }
  cw_sync();
  cluster_arrive();  // B3
  cluster_wait();
  {
    const int E = G * 128;
    const int per = (E + C - 1) / C;
    const int e0 = rank * per, e1 = min(E, e0 + per);
    bool bad = false;
    for (int r = 0; r < C; ++r) bad |= cluster.map_shared_rank(const_cast<int*>(failed), r)[0] != 0;
    for (int e = e0 + tid; e < e1; e += NCT) {
      float s = 0.f;
      for (int r = 0; r < C; ++r) s += cluster.map_shared_rank(opart, r)[e];
      const float y = bad ? __int_as_float(0x7FC00000) : s / ltot[e >> 7];
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
  // a denser tile processes its extra slots from global memory in further rounds
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
  P.o_qs = take((size_t)G * 128 * 4);
  P.o_qp = take((size_t)G * 128 * 4);
  P.o_rs = take((size_t)R * G * 4);
  P.o_pf = take((size_t)((R + 15) / 16) * 512);
  P.o_e = take((size_t)NCW * 16 * ROWE);
  P.o_acc = take((size_t)G * 128 * 4);
  P.o_opart = take((size_t)std::max(G * 128, NCW * G) * 4);
  P.o_misc = take((size_t)(NCW * G + 4 * G + 3 * kMaxCluster * G + 4) * 4);
  P.o_bar = take(2 * 8 * 8);
  P.o_cdk = (int)align128(ST_REC);
  P.o_sck = (int)align128(P.o_cdk + R * 32);
  P.o_cdv = (int)align128(P.o_sck + (R + 8) * 4);
  P.o_scv = (int)align128(P.o_cdv + R * 32);
  int stage = (int)align128(P.o_scv + (R + 8) * 4);
  stage = std::max(stage, (int)align128(ROWS * ROWB));
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
  P.pf_items = NS + 6;
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
    if (e == cudaSuccess && nclusters >= 1) break;
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
