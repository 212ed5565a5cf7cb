// Split-K decode attention read directly from the AnchorKV compressed cache.
//
// One thread-block cluster per (request, KV head) unit; its C CTAs split the
// unit's positions.  Per CTA (Eq. 3 folded into Eq. 4):
//   phase 0  q rows of the GQA group, q' = H(s o q)/128 (Appendix A.1, Eq. 12)
//   phase 1  anchor scores S_A = q . k_a for this CTA's slice of anchors,
//            then every CTA gathers the full S_A table from its peers (DSMEM)
//   phase 2  tiles of positions: key logits gamma_i S_A[a(i)] + residual term,
//            running max, p = 2^(l - m), value weights scattered per anchor
//            and rotated-domain residual accumulation
//   phase 3  cluster combine (max / sum rescale, Eq. 4) through DSMEM: each CTA
//            reduces its slice of the anchor weights, multiplies by its anchor
//            values, inverse-rotates its residual accumulator once (Appendix E.1
//            linearity), then the partial outputs are summed and normalised.
// No decompressed key or value is ever written to global memory, and the
// kernel uses no global scratch.
#include <cooperative_groups.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

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

constexpr int NT = 256;  // threads per CTA
constexpr int NWARP = NT / 32;
constexpr int TILE = 512;  // positions per tile
constexpr int PPT = TILE / NT;
constexpr float kLog2e = 1.4426950408889634f;
constexpr int kMaxCluster = 16;

struct DecodeParams {
  const uint8_t* arena;
  const __nv_bfloat16* q;
  __nv_bfloat16* out;
  float* out_f32;
  int n_kv_heads;
  int n_q_heads;
  int cluster;
  int rotate;
  int max_k;
  float scale_log2;
  unsigned long long sign_lo, sign_hi;
};

__device__ __forceinline__ float half_lo(uint32_t w) { return __half2float(__ushort_as_half((unsigned short)(w & 0xFFFFu))); }
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

// Number of residual positions < pos, from the bitmap and its prefix words.
__device__ __forceinline__ int res_rank(const uint64_t* bm, const uint32_t* pf, int S, int n, int pos) {
  if (pos >= S) return n;
  const int w = pos >> 6, bit = pos & 63;
  const uint64_t word = bm[w];
  return (int)pf[w] + __popcll(bit ? (word & ((1ull << bit) - 1ull)) : 0ull);
}

// Unnormalised 128-point Walsh-Hadamard transform of `rows` rows in shared
// memory, all threads of the CTA participating.
__device__ void cta_wht_rows(float* v, int rows) {
  for (int h = 1; h < 128; h <<= 1) {
    __syncthreads();
    for (int e = threadIdx.x; e < rows * 64; e += NT) {
      const int r = e >> 6, pr = e & 63;
      const int j = (pr / h) * 2 * h + (pr % h);
      float* x = v + r * 128;
      const float a = x[j], b = x[j + h];
      x[j] = a + b;
      x[j + h] = a - b;
    }
  }
  __syncthreads();
}

// Shared-memory carve-up, in floats; every region starts on a 16-byte boundary.
__host__ __device__ constexpr size_t r4(size_t x) { return (x + 3) & ~(size_t)3; }

template <int G>
struct Smem {
  static __host__ __device__ size_t sa(int) { return 0; }
  static __host__ __device__ size_t w(int max_k) { return r4((size_t)max_k * G); }
  static __host__ __device__ size_t qs(int max_k) { return 2 * r4((size_t)max_k * G); }
  static __host__ __device__ size_t qp(int max_k) { return qs(max_k) + G * 128; }
  static __host__ __device__ size_t rsk(int max_k) { return qp(max_k) + G * 128; }
  static __host__ __device__ size_t pv(int max_k) { return rsk(max_k) + (size_t)TILE * G; }
  static __host__ __device__ size_t acc(int max_k) { return pv(max_k) + (size_t)TILE * G; }
  static __host__ __device__ size_t opart(int max_k) { return acc(max_k) + G * 128; }
  static __host__ __device__ size_t misc(int max_k) { return opart(max_k) + G * 128; }
  // misc: red[NWARP*G], sq[G], cm[G], cl[G], ltot[G], peer_m[16*G], peer_l[16*G], facs[16*G]
  static __host__ __device__ size_t total_floats(int max_k) {
    return misc(max_k) + NWARP * G + 4 * G + 3 * kMaxCluster * G;
  }
  static __host__ __device__ size_t bytes(int max_k) { return total_floats(max_k) * sizeof(float); }
};

template <int G>
__global__ void __launch_bounds__(NT, 1) akv_decode_kernel(const DecodeParams P) {
  extern __shared__ __align__(16) float smem[];
  cg::cluster_group cluster = cg::this_cluster();
  const int C = P.cluster;
  const int rank = (int)cluster.block_rank();
  const int u = blockIdx.x / C;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  const akv_unit_desc* dsc = reinterpret_cast<const akv_unit_desc*>(P.arena + 256) + u;
  const int S = dsc->len, k = dsc->n_anchors, nk = dsc->n_res_k, nv = dsc->n_res_v;
  const uint8_t* A = P.arena;
  const __nv_bfloat16* AK = reinterpret_cast<const __nv_bfloat16*>(A + dsc->off_anchor_k);
  const __nv_bfloat16* AV = reinterpret_cast<const __nv_bfloat16*>(A + dsc->off_anchor_v);
  const uint32_t* stK = reinterpret_cast<const uint32_t*>(A + dsc->off_stream_k);
  const uint32_t* stV = reinterpret_cast<const uint32_t*>(A + dsc->off_stream_v);
  const uint64_t* bmK = reinterpret_cast<const uint64_t*>(A + dsc->off_bitmap_k);
  const uint32_t* pfK = reinterpret_cast<const uint32_t*>(A + dsc->off_prefix_k);
  const uint64_t* bmV = reinterpret_cast<const uint64_t*>(A + dsc->off_bitmap_v);
  const uint32_t* pfV = reinterpret_cast<const uint32_t*>(A + dsc->off_prefix_v);
  const uint8_t* cdK = A + dsc->off_codes_k;
  const uint32_t* scK = reinterpret_cast<const uint32_t*>(A + dsc->off_scales_k);
  const uint8_t* cdV = A + dsc->off_codes_v;
  const uint32_t* scV = reinterpret_cast<const uint32_t*>(A + dsc->off_scales_v);

  const int max_k = P.max_k;
  float* SA = smem + Smem<G>::sa(max_k);
  float* Wt = smem + Smem<G>::w(max_k);
  float* qs = smem + Smem<G>::qs(max_k);
  float* qp = smem + Smem<G>::qp(max_k);
  float* rsK = smem + Smem<G>::rsk(max_k);
  float* pV = smem + Smem<G>::pv(max_k);
  float* accs = smem + Smem<G>::acc(max_k);
  float* opart = smem + Smem<G>::opart(max_k);
  float* red = smem + Smem<G>::misc(max_k);
  float* sq = red + NWARP * G;
  float* cm = sq + G;
  float* cl = cm + G;
  float* ltot = cl + G;
  float* peer_m = ltot + G;
  float* peer_l = peer_m + kMaxCluster * G;
  float* facs = peer_l + kMaxCluster * G;

  const int b = u / P.n_kv_heads, h = u % P.n_kv_heads;
  const size_t qrow0 = ((size_t)b * P.n_q_heads + (size_t)h * G) * 128;

  // ---- phase 0: query rows and the rotated-domain query ---------------------
  for (int e = tid; e < G * 128; e += NT) {
    const int j = e & 127;
    const float x = __bfloat162float(P.q[qrow0 + e]);
    qs[e] = x;
    const unsigned long long sb = j < 64 ? P.sign_lo : P.sign_hi;
    qp[e] = (P.rotate && ((sb >> (j & 63)) & 1ull)) ? -x : x;
  }
  if (P.rotate) cta_wht_rows(qp, G);
  else __syncthreads();
  {
    const float f = P.rotate ? P.scale_log2 * (1.0f / 128.0f) : P.scale_log2;
    for (int e = tid; e < G * 128; e += NT) qp[e] *= f;
  }
  __syncthreads();
  if (warp < G) {
    float s = 0.f;
    for (int j = lane; j < 128; j += 32) s += qp[warp * 128 + j];
    s = warp_sum(s);
    if (lane == 0) sq[warp] = s;
  }

  // ---- phase 1: anchor scores for this CTA's slice, then gather the rest ----
  const int a_per = ((k + C - 1) / C + 15) / 16 * 16;
  const int a0 = min(k, rank * a_per), a1 = min(k, a0 + a_per);
  for (int a = a0 + warp; a < a1; a += NWARP) {
    const uint2 raw = *reinterpret_cast<const uint2*>(AK + (size_t)a * 128 + lane * 4);
    const float x0 = __bfloat162float(__ushort_as_bfloat16((unsigned short)(raw.x & 0xFFFFu)));
    const float x1 = __bfloat162float(__ushort_as_bfloat16((unsigned short)(raw.x >> 16)));
    const float x2 = __bfloat162float(__ushort_as_bfloat16((unsigned short)(raw.y & 0xFFFFu)));
    const float x3 = __bfloat162float(__ushort_as_bfloat16((unsigned short)(raw.y >> 16)));
#pragma unroll
    for (int g = 0; g < G; ++g) {
      const float4 qq = *reinterpret_cast<const float4*>(qs + g * 128 + lane * 4);
      float d = x0 * qq.x + x1 * qq.y + x2 * qq.z + x3 * qq.w;
      d = warp_sum(d);
      if (lane == 0) SA[a * G + g] = d * P.scale_log2;
    }
  }
  cluster.sync();
  for (int r = 0; r < C; ++r) {
    if (r == rank) continue;
    const int b0 = min(k, r * a_per), b1 = min(k, b0 + a_per);
    const float* rem = cluster.map_shared_rank(SA, r);
    for (int e = b0 * G + tid; e < b1 * G; e += NT) SA[e] = rem[e];
  }
  for (int e = tid; e < k * G; e += NT) Wt[e] = 0.f;
  __syncthreads();

  // ---- phase 2: tiles of positions -----------------------------------------
  constexpr int Q = G * 32;                     // (row, code byte) quads of the V accumulator
  constexpr int NGRP = NT / Q > 0 ? NT / Q : 1;  // slot groups
  const int quad = tid % Q, grp = tid / Q;
  const int gq = quad >> 5, bq = quad & 31;
  const bool acc_owner = tid < Q * NGRP;
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
  float pmin = 0.f;
  float m_run[G], l_part[G];
#pragma unroll
  for (int g = 0; g < G; ++g) {
    m_run[g] = -1e30f;
    l_part[g] = 0.f;
  }

  const int chunk = ((S + C - 1) / C + TILE - 1) / TILE * TILE;
  const int p0 = min(S, rank * chunk), p1 = min(S, p0 + chunk);
  for (int t0 = p0; t0 < p1; t0 += TILE) {
    const int te = min(t0 + TILE, p1);
    const int skl = res_rank(bmK, pfK, S, nk, t0), skh = res_rank(bmK, pfK, S, nk, te);
    const int svl = res_rank(bmV, pfV, S, nv, t0), svh = res_rank(bmV, pfV, S, nv, te);

    // (a) key residual terms, one warp per slot: min * sum(q') + scale * (q' . c)
    for (int s = skl + warp; s < skh; s += NWARP) {
      const uint32_t byte = cdK[(size_t)s * 32 + lane];
      const uint32_t sm = scK[s];
      const float sc = half_lo(sm), mn = half_hi(sm);
      const float c0 = (float)(byte & 3u), c1 = (float)((byte >> 2) & 3u), c2 = (float)((byte >> 4) & 3u),
                  c3 = (float)((byte >> 6) & 3u);
#pragma unroll
      for (int g = 0; g < G; ++g) {
        const float4 qq = *reinterpret_cast<const float4*>(qp + g * 128 + lane * 4);
        float d = c0 * qq.x + c1 * qq.y + c2 * qq.z + c3 * qq.w;
        d = warp_sum(d);
        if (lane == 0) rsK[(s - skl) * G + g] = mn * sq[g] + sc * d;
      }
    }
    __syncthreads();

    // (b) key logits
    float lg[PPT][G];
#pragma unroll
    for (int pp = 0; pp < PPT; ++pp) {
      const int i = t0 + tid * PPT + pp;
      if (i < te) {
        const uint32_t e = stK[i];
        const int a = min((int)(e & 0xFFFFu), k - 1);  // indices are < k by construction; never read past the table
        const float gam = half_hi(e);
#pragma unroll
        for (int g = 0; g < G; ++g) lg[pp][g] = gam * SA[a * G + g];
        const uint64_t word = bmK[i >> 6];
        if ((word >> (i & 63)) & 1ull) {
          const int bit = i & 63;
          const int slot = (int)pfK[i >> 6] + __popcll(bit ? (word & ((1ull << bit) - 1ull)) : 0ull) - skl;
#pragma unroll
          for (int g = 0; g < G; ++g) lg[pp][g] += rsK[slot * G + g];
        }
      } else {
#pragma unroll
        for (int g = 0; g < G; ++g) lg[pp][g] = -INFINITY;
      }
    }
    // (c) running max over the tile
#pragma unroll
    for (int g = 0; g < G; ++g) {
      float mx = lg[0][g];
#pragma unroll
      for (int pp = 1; pp < PPT; ++pp) mx = fmaxf(mx, lg[pp][g]);
      mx = warp_max(mx);
      if (lane == 0) red[warp * G + g] = mx;
    }
    __syncthreads();
    bool grow = false;
    float fac[G];
#pragma unroll
    for (int g = 0; g < G; ++g) {
      float mx = red[g];
#pragma unroll
      for (int w = 1; w < NWARP; ++w) mx = fmaxf(mx, red[w * G + g]);
      const float nm = fmaxf(m_run[g], mx);
      fac[g] = exp2f(m_run[g] - nm);
      grow |= nm > m_run[g];
      m_run[g] = nm;
    }
    if (grow) {  // uniform across the CTA
      for (int e = tid; e < k * G; e += NT) Wt[e] *= fac[e % G];
#pragma unroll
      for (int g = 0; g < G; ++g) l_part[g] *= fac[g];
      float fq = 1.f;
#pragma unroll
      for (int g = 0; g < G; ++g)
        if (g == gq) fq = fac[g];
#pragma unroll
      for (int c = 0; c < 4; ++c) acc[c] *= fq;
      pmin *= fq;
      __syncthreads();
    }
    // (d) probabilities, value-weight scatter, residual probabilities
#pragma unroll
    for (int pp = 0; pp < PPT; ++pp) {
      const int i = t0 + tid * PPT + pp;
      if (i < te) {
        float p[G];
#pragma unroll
        for (int g = 0; g < G; ++g) {
          p[g] = exp2f(lg[pp][g] - m_run[g]);
          l_part[g] += p[g];
        }
        const uint32_t e = stV[i];
        const int a = min((int)(e & 0xFFFFu), k - 1);
        const float gam = half_hi(e);
#pragma unroll
        for (int g = 0; g < G; ++g) atomicAdd(&Wt[a * G + g], p[g] * gam);
        const uint64_t word = bmV[i >> 6];
        if ((word >> (i & 63)) & 1ull) {
          const int bit = i & 63;
          const int slot = (int)pfV[i >> 6] + __popcll(bit ? (word & ((1ull << bit) - 1ull)) : 0ull) - svl;
#pragma unroll
          for (int g = 0; g < G; ++g) pV[slot * G + g] = p[g];
        }
      }
    }
    __syncthreads();
    // (e) value residual accumulation in the rotated domain
    if (acc_owner) {
      for (int s = svl + grp; s < svh; s += NGRP) {
        const uint32_t byte = cdV[(size_t)s * 32 + bq];
        const uint32_t sm = scV[s];
        const float sc = half_lo(sm), mn = half_hi(sm);
        const float pp = pV[(s - svl) * G + gq];
        const float ps = pp * sc;
        acc[0] += ps * (float)(byte & 3u);
        acc[1] += ps * (float)((byte >> 2) & 3u);
        acc[2] += ps * (float)((byte >> 4) & 3u);
        acc[3] += ps * (float)((byte >> 6) & 3u);
        pmin += pp * mn;
      }
    }
    __syncthreads();
  }

  // ---- per-CTA totals -------------------------------------------------------
#pragma unroll
  for (int g = 0; g < G; ++g) {
    const float s = warp_sum(l_part[g]);
    if (lane == 0) red[warp * G + g] = s;
  }
  for (int e = tid; e < G * 128; e += NT) accs[e] = 0.f;
  __syncthreads();
  if (tid < G) {
    float s = 0.f;
    for (int w = 0; w < NWARP; ++w) s += red[w * G + tid];
    cl[tid] = s;
    cm[tid] = m_run[tid];
  }
  if (acc_owner) {
#pragma unroll
    for (int c = 0; c < 4; ++c) atomicAdd(&accs[gq * 128 + bq * 4 + c], acc[c] + pmin);
  }
  __syncthreads();

  // ---- phase 3: combine across the cluster ----------------------------------
  cluster.sync();
  if (tid < C * G) {
    const int r = tid / G, g = tid % G;
    peer_m[tid] = cluster.map_shared_rank(cm, r)[g];
    peer_l[tid] = cluster.map_shared_rank(cl, r)[g];
  }
  __syncthreads();
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
  __syncthreads();
  // anchor weights of this CTA's slice, summed over the cluster
  for (int e = a0 * G + tid; e < a1 * G; e += NT) {
    const int g = e % G;
    float s = 0.f;
    for (int r = 0; r < C; ++r) s += facs[r * G + g] * cluster.map_shared_rank(Wt, r)[e];
    Wt[e] = s;
  }
  __syncthreads();
  // partial output: anchor values of the slice plus this CTA's inverse-rotated residuals
  for (int e = tid; e < G * 128; e += NT) accs[e] *= facs[rank * G + e / 128];
  if (P.rotate) cta_wht_rows(accs, G);
  else __syncthreads();
  for (int e = tid; e < G * 128; e += NT) {
    const int g = e >> 7, j = e & 127;
    float o = 0.f;
    for (int a = a0; a < a1; ++a) o += Wt[a * G + g] * __bfloat162float(AV[(size_t)a * 128 + j]);
    float r = accs[e];
    if (P.rotate) {
      const unsigned long long sb = j < 64 ? P.sign_lo : P.sign_hi;
      r = ((sb >> (j & 63)) & 1ull) ? -r : r;
      r *= (1.0f / 128.0f);
    }
    opart[e] = o + r;
  }
  __syncthreads();
  cluster.sync();
  {
    const int E = G * 128;
    const int per = (E + C - 1) / C;
    const int e0 = rank * per, e1 = min(E, e0 + per);
    for (int e = e0 + tid; e < e1; e += NT) {
      float s = 0.f;
      for (int r = 0; r < C; ++r) s += cluster.map_shared_rank(opart, r)[e];
      const float y = s / ltot[e >> 7];
      const size_t o = qrow0 + e;
      P.out[o] = __float2bfloat16_rn(y);
      if (P.out_f32) P.out_f32[o] = y;
    }
  }
  cluster.sync();
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

// Launch configuration per (device, G, shared-memory size, unit count, longest
// context): computed once (attributes, occupancy query), then reused, so that a
// call made during CUDA-graph capture only issues the launch itself.
struct LaunchKey {
  int dev, G, units, max_len, cluster_env;
  size_t smem;
  bool operator<(const LaunchKey& o) const {
    return std::tie(dev, G, units, max_len, cluster_env, smem) <
           std::tie(o.dev, o.G, o.units, o.max_len, o.cluster_env, o.smem);
  }
};

template <int G>
int choose_cluster(const LaunchKey& key, int* C_out) {
  static std::mutex mu;
  static std::map<LaunchKey, int> cache;
  {
    std::lock_guard<std::mutex> lk(mu);
    auto it = cache.find(key);
    if (it != cache.end()) {
      *C_out = it->second;
      return 0;
    }
  }
  const DeviceInfo di = device_info();
  // The attribute is per kernel, not per launch: raise it to the device limit once,
  // so that every cached configuration stays launchable.
  cudaError_t e = cudaFuncSetAttribute(akv_decode_kernel<G>, cudaFuncAttributeMaxDynamicSharedMemorySize, di.smem_optin);
  if (e != cudaSuccess) return (int)e;
  e = cudaFuncSetAttribute(akv_decode_kernel<G>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  if (e != cudaSuccess) return (int)e;
  // Cluster size: enough CTAs for one wave over the SMs, no more than the tiles of the longest unit.
  const int per_sm = std::max(1, (int)((228 * 1024) / (key.smem + 1024)));
  const int slots = di.sms * std::min(per_sm, 2048 / NT);
  int C = 1;
  while (C < kMaxCluster && (long long)key.units * (C * 2) <= slots && (C * 2) * TILE <= key.max_len + TILE - 1) C *= 2;
  if (key.cluster_env >= 1 && key.cluster_env <= kMaxCluster) C = key.cluster_env;
  for (; C > 1; C = (C == 3 ? 1 : C / 2)) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(C * key.units), 1, 1);
    cfg.blockDim = dim3(NT, 1, 1);
    cfg.dynamicSmemBytes = key.smem;
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
  }
  std::lock_guard<std::mutex> lk(mu);
  cache[key] = C;
  *C_out = C;
  return 0;
}

template <int G>
int launch_g(const Layout& L, const akv_params& p, const void* arena, const void* q, void* out, float* out_f32,
             float sm_scale, void* stream, std::string* why) {
  const int units = (int)L.shape.size();
  const size_t smem = Smem<G>::bytes(L.max_k);
  const DeviceInfo di = device_info();
  if ((int)smem > di.smem_optin) {
    *why = "anchor tables need " + std::to_string(smem) + " B of shared memory (k * G too large)";
    return -1;
  }
  int dev = 0;
  cudaGetDevice(&dev);
  int cenv = 0;
  if (const char* env = std::getenv("AKV_CLUSTER")) cenv = std::atoi(env);
  const LaunchKey key{dev, G, units, L.max_len, cenv, smem};
  int C = 1;
  int err = choose_cluster<G>(key, &C);
  if (err) return err;

  DecodeParams P;
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
  P.cluster = C;

  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(C * units), 1, 1);
  cfg.blockDim = dim3(NT, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = (cudaStream_t)stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = C;
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
