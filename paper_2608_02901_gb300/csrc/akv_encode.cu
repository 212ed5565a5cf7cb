// Plain GPU encoder of the AnchorKV compressed cache (Algorithm 1 with the
// anchor and slot rules of this build).  Correct, not tuned: every decision
// (assignment, gamma, residual energy ranking, rotation, codes) is taken in
// IEEE fp64 with a fixed operation order, so the packed bytes are
// reproducible bit for bit.  Compiled with --fmad=false; where a fused
// multiply-add is used explicitly its product is exact, so rounding once or
// twice gives the same result.
//
// Kernels, in launch order, each over all units of the batch:
//   enc_hash       anchor-selection hashes of the non-window positions
//   enc_anchors    select the k - W smallest hashes, number anchor slots by position
//   enc_rows       copy anchor rows into the arena (16-byte chunks swizzled), squared norms
//   enc_assign     Eq. 1 nearest anchor, Eq. 2 gamma, residual energies (per position)
//   enc_slots      top-N residual energies per side -> residual flags and slot list
//   enc_order      stored order: stable counting sort of positions by value anchor slot
//   enc_tile_count residual records per tile and side
//   enc_tile_table tile block offsets
//   enc_tile_fill  streams, bitmaps and rank words of every tile block
//   enc_quant      Eq. 12 rotation and 2-bit quantization of every slot, into its tile
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <cstring>
#include <mutex>
#include <vector>

#include "akv_internal.h"

namespace akv {
namespace {

// The Lloyd-Max codec's outer decision threshold: the midpoint of its levels 0.453125 and
// 1.5078125 (the Gaussian four-level Lloyd-Max levels 0.4528, 1.5104 to 8 significant bits).
constexpr double kLloydT = 0.98046875;

// Per-unit scratch pointers, derived from the workspace table the host writes.
struct EncUnitWs {
  uint64_t* key0;     // [S] anchor hashes, then key residual energies
  uint64_t* key1;     // [S] value residual energies
  int32_t* slot_of;   // [S] anchor slot or -1
  int32_t* res_pos;   // [N_K + N_V] residual positions (keys, then values)
  double* n2[2];      // [k] squared anchor norms per side
  double* rn[2];      // [k] their square roots
  uint32_t* ctrl;     // [0]: side 0 has a nonzero anchor, [1]: side 1
  uint32_t* st[2];    // [S] stream word (slot | fp16 gamma << 16) per position and side
  uint8_t* flag;      // [S] bit 0: key residual, bit 1: value residual
  int32_t* perm;      // [S] position of stored token t
  int32_t* inv;       // [S] stored index of position i
  uint32_t* cursor;   // [k + 1] value-anchor counts, then start of each run
  uint32_t* tcnt;     // [2 * n_tiles] residual records per tile (keys, values)
  double* alpha;      // full selection: [m][S] observation rows' attention
  double* yobs;       // full selection: [m][128] their exact outputs
};

struct EncArgs {
  const uint8_t* arena_c;
  uint8_t* arena;
  const uint8_t* ws_base;
  const uint64_t* ws_off;  // [units] byte offsets of each unit's scratch
  const __nv_bfloat16* K;
  const __nv_bfloat16* V;
  int32_t s_max;
  int32_t n_kv_heads;
  int32_t window;
  int32_t rotate;
  int32_t lloyd;  // AKV_FLAG_LLOYD: the Lloyd-Max codec
  uint64_t seed;
  unsigned long long sign_lo, sign_hi;
  // full selection (m_obs > 0): observation rows Q [units][m_obs][128], pooling width,
  // scored share, retained fraction
  const __nv_bfloat16* Q;
  int32_t m_obs, kappa;
  float rho, theta;
};

__device__ __forceinline__ const akv_unit_desc* unit_desc(const EncArgs& A, int u) {
  return reinterpret_cast<const akv_unit_desc*>(A.arena_c + 256) + u;
}

__device__ __forceinline__ uint64_t au(uint64_t x, uint64_t a) { return (x + a - 1) / a * a; }

__device__ EncUnitWs unit_ws(const EncArgs& A, int u, const akv_unit_desc* d) {
  uint8_t* p = const_cast<uint8_t*>(A.ws_base) + A.ws_off[u];
  EncUnitWs w;
  const uint64_t S = (uint64_t)d->len, k = (uint64_t)d->n_anchors, n = (uint64_t)(d->n_res_k + d->n_res_v);
  w.key0 = (uint64_t*)p;
  p += au(S * 8, 256);
  w.key1 = (uint64_t*)p;
  p += au(S * 8, 256);
  w.slot_of = (int32_t*)p;
  p += au(S * 4, 256);
  w.res_pos = (int32_t*)p;
  p += au(n * 4 + 16, 256);
  for (int s = 0; s < 2; ++s) {
    w.n2[s] = (double*)p;
    p += au(k * 8, 256);
    w.rn[s] = (double*)p;
    p += au(k * 8, 256);
  }
  w.ctrl = (uint32_t*)p;
  p += 256;
  for (int s = 0; s < 2; ++s) {
    w.st[s] = (uint32_t*)p;
    p += au(S * 4, 256);
  }
  w.flag = p;
  p += au(S, 256);
  w.perm = (int32_t*)p;
  p += au(S * 4, 256);
  w.inv = (int32_t*)p;
  p += au(S * 4, 256);
  w.cursor = (uint32_t*)p;
  p += au((k + 1) * 4, 256);
  w.tcnt = (uint32_t*)p;
  p += au((uint64_t)d->n_tiles * 8, 256);
  w.alpha = (double*)p;
  p += au((uint64_t)A.m_obs * S * 8, 256);
  w.yobs = (double*)p;
  return w;
}

// Anchor row a of a side in the source K or V (the arena holds it swizzled).
__device__ __forceinline__ const __nv_bfloat16* anchor_src(const EncArgs& A, int u, int side, const int32_t* apos, int a) {
  return (side ? A.V : A.K) + ((size_t)u * A.s_max + (size_t)apos[a]) * 128;
}

__device__ __forceinline__ uint64_t splitmix64_dev(uint64_t x) {
  uint64_t z = x + 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

__device__ __forceinline__ double bf16_to_f64(__nv_bfloat16 v) { return (double)__bfloat162float(v); }
__device__ __forceinline__ double fp16_bits_to_f64(uint32_t h) {
  return (double)__half2float(__ushort_as_half((unsigned short)(h & 0xFFFFu)));
}

// fp64 -> fp16 bits, round to nearest even on the integer significand,
// saturating at +-65504 (values are finite here; NaN maps to 0x7E00).
__device__ uint32_t f64_to_fp16_bits(double x) {
  const unsigned long long bits = (unsigned long long)__double_as_longlong(x);
  const uint32_t sign = (uint32_t)(bits >> 63) << 15;
  const int ex = (int)((bits >> 52) & 0x7FF);
  const unsigned long long frac = bits & 0xFFFFFFFFFFFFFull;
  if (ex == 0x7FF) return frac ? 0x7E00u : (sign | 0x7BFFu);
  if (fabs(x) >= 65504.0) return sign | 0x7BFFu;
  if (ex == 0) return sign;  // fp64 subnormals are far below half an fp16 ulp
  const int e = ex - 1023;
  if (e < -25) return sign;
  const unsigned long long m = frac | (1ull << 52);  // 53-bit significand
  const int sh = (e >= -14) ? 42 : 42 + (-14 - e);   // bits dropped
  unsigned long long r = m >> sh;
  const unsigned long long rem = m & ((1ull << sh) - 1ull);
  const unsigned long long half = 1ull << (sh - 1);
  if (rem > half || (rem == half && (r & 1ull))) ++r;
  uint32_t out;
  if (e >= -14) out = (uint32_t)(((e + 14) << 10) + (int)r);  // r carries the implicit 1024
  else out = (uint32_t)r;                                      // subnormal (1024 -> smallest normal)
  if (out >= 0x7C00u) out = 0x7BFFu;
  return sign | out;
}

// r-th smallest (1-based) of the n 64-bit keys key_at(0 .. n-1) (optionally of their
// complements), MSB-first radix select by 8-bit digits; returns the key and the rank of
// the answer among keys equal to it (*rank_in_eq, 1-based).  Block-wide.
template <class KeyAt>
__device__ uint64_t block_select_f(KeyAt key_at, int64_t n, uint32_t r, bool complement, uint32_t* hist,
                                   uint32_t* bcast, uint32_t* rank_in_eq) {
  uint64_t prefix = 0, mask = 0;
  for (int shift = 56; shift >= 0; shift -= 8) {
    for (int i = threadIdx.x; i < 256; i += blockDim.x) hist[i] = 0;
    __syncthreads();
    for (int64_t i = threadIdx.x; i < n; i += blockDim.x) {
      uint64_t key = key_at(i);
      if (complement) key = ~key;
      if ((key & mask) == prefix) atomicAdd(&hist[(key >> shift) & 255u], 1u);
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      uint32_t cum = 0, sel = 255;
      for (uint32_t bkt = 0; bkt < 256; ++bkt) {
        if (cum + hist[bkt] >= r) {
          sel = bkt;
          break;
        }
        cum += hist[bkt];
      }
      bcast[0] = sel;
      bcast[1] = r - cum;
    }
    __syncthreads();
    prefix |= (uint64_t)bcast[0] << shift;
    mask |= 0xFFull << shift;
    r = bcast[1];
    __syncthreads();
  }
  *rank_in_eq = r;
  return complement ? ~prefix : prefix;
}
__device__ uint64_t block_select(const uint64_t* keys, int n, uint32_t r, bool complement, uint32_t* hist,
                                 uint32_t* bcast, uint32_t* rank_in_eq) {
  return block_select_f([keys](int64_t i) { return keys[i]; }, n, r, complement, hist, bcast, rank_in_eq);
}

// Exclusive block scan of 0/1 flags for a block of 1024 threads; returns the
// prefix and writes the block total to *total.
__device__ int block_scan_flag(int flag, int* warp_tot, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const unsigned bal = __ballot_sync(0xffffffffu, flag);
  const int pre_lane = __popc(bal & ((1u << lane) - 1u));
  if (lane == 0) warp_tot[warp] = __popc(bal);
  __syncthreads();
  if (warp == 0) {
    const int nw = blockDim.x >> 5;
    int v = lane < nw ? warp_tot[lane] : 0;
    int incl = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int t = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += t;
    }
    if (lane < nw) warp_tot[lane] = incl - v;
    if (lane == 31) warp_tot[32] = incl;
  }
  __syncthreads();
  const int pre = warp_tot[warp] + pre_lane;
  *total = warp_tot[32];
  __syncthreads();
  return pre;
}

// ---- kernels -----------------------------------------------------------------

// Anchors of the full selection picked by score: floor(rho (k - w)) (Section 3.2); none in
// the plain encoder.
__device__ __forceinline__ int n_scored(const EncArgs& A, int rest) {
  return (A.m_obs > 0 && rest > 0) ? (int)floor((double)A.rho * (double)rest) : 0;
}

__global__ void enc_hash(const EncArgs A) {
  const int u = blockIdx.y;
  const akv_unit_desc* d = unit_desc(A, u);
  const int S = d->len;
  const int p = blockIdx.x * blockDim.x + threadIdx.x;
  if (p >= S) return;
  EncUnitWs w = unit_ws(A, u, d);
  const int win = min(A.window, S);
  const uint64_t base = A.seed ^ ((uint64_t)d->b << 40) ^ ((uint64_t)d->h << 32);
  // (full selection: positions already chosen by their score take no part in the sampling)
  const bool scored = A.m_obs > 0 && w.slot_of[p] == -2;
  w.key0[p] = (p < S - win && !scored) ? splitmix64_dev(base ^ (uint64_t)p) : ~0ull;
}

__global__ void __launch_bounds__(1024) enc_anchors(const EncArgs A) {
  __shared__ uint32_t hist[256];
  __shared__ uint32_t bc[2];
  __shared__ int wt[33];
  const int u = blockIdx.x;
  const akv_unit_desc* d = unit_desc(A, u);
  const int S = d->len, k = d->n_anchors;
  EncUnitWs w = unit_ws(A, u, d);
  const int win = min(A.window, S);
  const int pool = S - win;
  // the sampled share: all k - w non-window anchors, less those the full selection scored
  const int rest = k - win - n_scored(A, k - win);
  uint64_t thr = 0;
  bool any = rest > 0;
  if (any) {
    uint32_t req;
    thr = block_select(w.key0, pool, (uint32_t)rest, false, hist, bc, &req);
  }
  int32_t* apos = reinterpret_cast<int32_t*>(A.arena + d->off_anchor_pos);
  int base = 0;
  for (int c0 = 0; c0 < S; c0 += 1024) {
    const int p = c0 + threadIdx.x;
    int flag = 0;
    if (p < S) flag = (p >= pool) || (A.m_obs > 0 && w.slot_of[p] == -2) || (any && w.key0[p] <= thr);
    int tot;
    const int pre = block_scan_flag(flag, wt, &tot);
    if (p < S) {
      w.slot_of[p] = flag ? base + pre : -1;
      if (flag) apos[base + pre] = p;
    }
    base += tot;
  }
  if (threadIdx.x < 2) w.ctrl[threadIdx.x] = 0;
}

// One warp per anchor: copy rows, squared norms (sequential in j) per side.
__global__ void enc_rows(const EncArgs A) {
  const int u = blockIdx.y;
  const akv_unit_desc* d = unit_desc(A, u);
  const int k = d->n_anchors;
  const int a = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (a >= k) return;
  EncUnitWs w = unit_ws(A, u, d);
  const int pos = reinterpret_cast<const int32_t*>(A.arena_c + d->off_anchor_pos)[a];
  for (int side = 0; side < 2; ++side) {
    const __nv_bfloat16* X = (side ? A.V : A.K) + ((size_t)u * A.s_max + pos) * 128;
    __nv_bfloat16* dst = reinterpret_cast<__nv_bfloat16*>(A.arena + (side ? d->off_anchor_v : d->off_anchor_k)) +
                         (size_t)a * 128;
    // dim j is in chunk j / 8, stored at chunk place (j / 8) ^ (a % 8)
    for (int j = lane; j < 128; j += 32) dst[8 * ((j >> 3) ^ (a & 7)) + (j & 7)] = X[j];
    if (lane == 0) {
      double n = 0.0;
      for (int j = 0; j < 128; ++j) {
        const double t = bf16_to_f64(X[j]);
        n = __dadd_rn(n, __dmul_rn(t, t));
      }
      w.n2[side][a] = n;
      w.rn[side][a] = __dsqrt_rn(n);
      if (n != 0.0) atomicOr(&w.ctrl[side], 1u);
    }
  }
}

constexpr int AS_POS = 64;  // positions per assignment block
constexpr int AS_ANC = 32;  // anchors per smem chunk
constexpr int AS_THREADS = 256;
constexpr size_t AS_SMEM = (size_t)128 * AS_POS * 8 + (size_t)AS_ANC * 128 * 8 + 4 * AS_POS * (8 + 8 + 4) + 64;

__global__ void __launch_bounds__(AS_THREADS) enc_assign(const EncArgs A) {
  extern __shared__ __align__(16) unsigned char sm_raw[];
  double* xs = reinterpret_cast<double*>(sm_raw);                 // [128][64] positions, transposed
  double* xa = xs + 128 * AS_POS;                                 // [32][128] anchor chunk
  double* bcv = xa + AS_ANC * 128;                                // [4][64]
  double* bdv = bcv + 4 * AS_POS;                                 // [4][64]
  int* bav = reinterpret_cast<int*>(bdv + 4 * AS_POS);            // [4][64]

  const int u = blockIdx.y, side = blockIdx.z;
  const akv_unit_desc* d = unit_desc(A, u);
  const int S = d->len, k = d->n_anchors;
  const int p0 = blockIdx.x * AS_POS;
  if (p0 >= S) return;
  EncUnitWs w = unit_ws(A, u, d);
  const __nv_bfloat16* X = (side ? A.V : A.K) + (size_t)u * A.s_max * 128;
  const int32_t* apos = reinterpret_cast<const int32_t*>(A.arena_c + d->off_anchor_pos);
  const double* n2 = w.n2[side];
  const double* rn = w.rn[side];
  const int tid = threadIdx.x;

  for (int e = tid; e < AS_POS * 128; e += AS_THREADS) {
    const int pi = e >> 7, j = e & 127;
    const int p = p0 + pi;
    xs[j * AS_POS + pi] = (p < S) ? bf16_to_f64(X[(size_t)p * 128 + j]) : 0.0;
  }
  const int pi = tid % AS_POS, ag = tid / AS_POS;
  double bestc = -1.0, bestd = 0.0;
  int besta = -1;
  for (int ac = 0; ac < k; ac += AS_ANC) {
    __syncthreads();
    for (int e = tid; e < AS_ANC * 128; e += AS_THREADS) {
      const int t = e >> 7, j = e & 127;
      xa[e] = (ac + t < k) ? bf16_to_f64(anchor_src(A, u, side, apos, ac + t)[j]) : 0.0;
    }
    __syncthreads();
    double dd[8];
#pragma unroll
    for (int t = 0; t < 8; ++t) dd[t] = 0.0;
    const double* xr = xa + (ag * 8) * 128;
    for (int j = 0; j < 128; ++j) {
      const double x = xs[j * AS_POS + pi];
#pragma unroll
      for (int t = 0; t < 8; ++t) dd[t] = __fma_rn(x, xr[t * 128 + j], dd[t]);  // product of two bf16: exact
    }
#pragma unroll
    for (int t = 0; t < 8; ++t) {
      const int a = ac + ag * 8 + t;
      if (a < k && n2[a] != 0.0) {
        const double c = __ddiv_rn(fabs(dd[t]), rn[a]);
        if (c > bestc) {
          bestc = c;
          besta = a;
          bestd = dd[t];
        }
      }
    }
  }
  bcv[ag * AS_POS + pi] = bestc;
  bdv[ag * AS_POS + pi] = bestd;
  bav[ag * AS_POS + pi] = besta;
  __syncthreads();
  if (tid >= AS_POS) return;
  const int p = p0 + tid;
  if (p >= S) return;
  double c = -1.0, dbest = 0.0;
  int a = -1;
  for (int g = 0; g < 4; ++g) {
    const int ga = bav[g * AS_POS + tid];
    if (ga < 0) continue;
    const double gc = bcv[g * AS_POS + tid];
    if (a < 0 || gc > c || (gc == c && ga < a)) {
      c = gc;
      a = ga;
      dbest = bdv[g * AS_POS + tid];
    }
  }
  uint32_t* stream = w.st[side];
  uint64_t* key = side ? w.key1 : w.key0;
  const int sl = w.slot_of[p];
  if (sl >= 0) {
    stream[p] = (uint32_t)sl | (0x3C00u << 16);
    key[p] = 0;
    return;
  }
  const uint32_t gh = (a >= 0) ? f64_to_fp16_bits(__ddiv_rn(dbest, n2[a])) : 0u;
  stream[p] = (uint32_t)(a >= 0 ? a : 0) | (gh << 16);
  const double g = fp16_bits_to_f64(gh);
  const __nv_bfloat16* xar = anchor_src(A, u, side, apos, a >= 0 ? a : 0);
  double e = 0.0;
  for (int j = 0; j < 128; ++j) {
    const double pj = (a >= 0) ? __dmul_rn(g, bf16_to_f64(xar[j])) : 0.0;
    const double r = __dsub_rn(xs[j * AS_POS + tid], pj);
    e = __dadd_rn(e, __dmul_rn(r, r));
  }
  key[p] = (uint64_t)__double_as_longlong(e) + 1ull;
}

// Per (unit, side): the N largest keys (ties: lower position) -> flags and the
// ascending slot list.
__global__ void __launch_bounds__(1024) enc_slots(const EncArgs A, int side) {
  __shared__ uint32_t hist[256];
  __shared__ uint32_t bc[2];
  __shared__ int wt[33];
  const int u = blockIdx.x;
  const akv_unit_desc* d = unit_desc(A, u);
  const int S = d->len, N = side ? d->n_res_v : d->n_res_k;
  EncUnitWs w = unit_ws(A, u, d);
  const uint64_t* key = side ? w.key1 : w.key0;
  int32_t* rp = w.res_pos + (side ? d->n_res_k : 0);
  uint64_t thr = ~0ull;
  uint32_t need = 0;
  if (N > 0) thr = block_select(key, S, (uint32_t)N, true, hist, bc, &need);
  int base = 0, eq_seen = 0;
  for (int c0 = 0; c0 < S; c0 += 1024) {
    const int p = c0 + threadIdx.x;
    const uint64_t kv = (p < S) ? key[p] : 0ull;
    const int is_eq = (N > 0 && p < S && kv == thr) ? 1 : 0;
    int eq_tot;
    const int eq_pre = block_scan_flag(is_eq, wt, &eq_tot);
    const int sel = (N > 0 && p < S) && (kv > thr || (is_eq && (uint32_t)(eq_seen + eq_pre) < need));
    eq_seen += eq_tot;
    int tot;
    const int pre = block_scan_flag(sel, wt, &tot);
    if (sel) rp[base + pre] = p;
    // flags of both sides share bytes: the side-0 launch writes them, the side-1 launch
    // (ordered after it on the stream) ORs its bit in
    if (p < S) {
      if (side == 0) w.flag[p] = (uint8_t)sel;
      else if (sel) w.flag[p] |= 2u;
    }
    base += tot;
    __syncthreads();
  }
}

// Exclusive block scan of non-negative counts (1024 threads); returns the prefix and
// writes the block total to *total.
__device__ uint32_t block_scan_u32(uint32_t v, uint32_t* warp_tot, uint32_t* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint32_t incl = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t t = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += t;
  }
  if (lane == 31) warp_tot[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    uint32_t x = warp_tot[lane], xi = x;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t t = __shfl_up_sync(0xffffffffu, xi, o);
      if (lane >= o) xi += t;
    }
    warp_tot[lane] = xi - x;
    if (lane == 31) warp_tot[32] = xi;
  }
  __syncthreads();
  const uint32_t pre = warp_tot[warp] + incl - v;
  *total = warp_tot[32];
  __syncthreads();
  return pre;
}

// Stored order of one unit: positions sorted by value anchor slot, ties by position
// (a stable counting sort).  One block per unit; the scatter is done by one warp in
// position order, 32 positions at a time, so equal slots keep their position order.
__global__ void __launch_bounds__(1024) enc_order(const EncArgs A) {
  __shared__ uint32_t wt[33];
  const int u = blockIdx.x;
  const akv_unit_desc* d = unit_desc(A, u);
  const int S = d->len, k = d->n_anchors;
  EncUnitWs w = unit_ws(A, u, d);
  for (int a = threadIdx.x; a <= k; a += blockDim.x) w.cursor[a] = 0u;
  __syncthreads();
  for (int p = threadIdx.x; p < S; p += blockDim.x) atomicAdd(&w.cursor[w.st[1][p] & 0xFFFFu], 1u);
  __syncthreads();
  uint32_t run = 0;
  for (int c0 = 0; c0 < k; c0 += 1024) {
    const int a = c0 + threadIdx.x;
    const uint32_t v = a < k ? w.cursor[a] : 0u;
    uint32_t tot;
    const uint32_t pre = block_scan_u32(v, wt, &tot);
    if (a < k) w.cursor[a] = run + pre;
    run += tot;
  }
  __syncthreads();
  if (threadIdx.x >= 32) return;
  const int lane = threadIdx.x;
  for (int c0 = 0; c0 < S; c0 += 32) {
    const int p = c0 + lane;
    const uint32_t a = p < S ? (w.st[1][p] & 0xFFFFu) : 0xFFFFFFFFu;
    const unsigned peers = __match_any_sync(0xffffffffu, a);
    const uint32_t base = p < S ? w.cursor[a] : 0u;
    __syncwarp();
    const int rank = __popc(peers & ((1u << lane) - 1u));
    if (p < S) {
      w.perm[base + rank] = p;
      w.inv[p] = (int32_t)(base + rank);
      if (rank == 0) w.cursor[a] = base + (uint32_t)__popc(peers);
    }
    __syncwarp();
  }
}

__device__ __forceinline__ int tile_len(int S, int j) { return min(kTile, S - j * kTile); }

// Residual records of each tile and side (one thread per stored token).
__global__ void __launch_bounds__(kTile) enc_tile_count(const EncArgs A) {
  const int u = blockIdx.y, j = blockIdx.x;
  const akv_unit_desc* d = unit_desc(A, u);
  if (j >= d->n_tiles) return;
  EncUnitWs w = unit_ws(A, u, d);
  const int t = j * kTile + threadIdx.x;
  const uint32_t f = t < d->len ? w.flag[w.perm[t]] : 0u;
  const int nk = __syncthreads_count(f & 1u), nv = __syncthreads_count(f & 2u);
  if (threadIdx.x == 0) {
    w.tcnt[2 * j] = (uint32_t)nk;
    w.tcnt[2 * j + 1] = (uint32_t)nv;
  }
}

// Tile block offsets of every unit (one thread per unit).
__global__ void enc_tile_table(const EncArgs A, int units) {
  const int u = blockIdx.x * blockDim.x + threadIdx.x;
  if (u >= units) return;
  const akv_unit_desc* d = unit_desc(A, u);
  EncUnitWs w = unit_ws(A, u, d);
  uint32_t* table = reinterpret_cast<uint32_t*>(A.arena + d->off_tile_table);
  uint32_t off = 0;
  for (int j = 0; j < d->n_tiles; ++j) {
    table[j] = off;
    off += tile_block_bytes(tile_len(d->len, j), (int)w.tcnt[2 * j], (int)w.tcnt[2 * j + 1]);
    // value slots of the tile's first and last stored tokens
    const int t0 = j * kTile, t1 = t0 + tile_len(d->len, j) - 1;
    table[d->n_tiles + 1 + j] = (w.st[1][w.perm[t0]] & 0xFFFFu) | ((w.st[1][w.perm[t1]] & 0xFFFFu) << 16);
  }
  table[d->n_tiles] = off;
}

// Streams, bitmaps and rank words of one tile block (one thread per stored token).
__global__ void __launch_bounds__(kTile) enc_tile_fill(const EncArgs A) {
  __shared__ uint32_t halves[2][kTile / 32];
  const int u = blockIdx.y, j = blockIdx.x;
  const akv_unit_desc* d = unit_desc(A, u);
  if (j >= d->n_tiles) return;
  EncUnitWs w = unit_ws(A, u, d);
  const int n = tile_len(d->len, j), nw = (int)tile_words(n), n64 = 64 * nw;
  const uint32_t off = reinterpret_cast<const uint32_t*>(A.arena_c + d->off_tile_table)[j];
  uint8_t* blk = A.arena + d->off_tiles + off;
  uint32_t* kst = reinterpret_cast<uint32_t*>(blk);
  uint32_t* vst = kst + n64;
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
  uint32_t f = 0;
  if (t < n) {
    const int i = w.perm[j * kTile + t];
    kst[t] = w.st[0][i];
    vst[t] = w.st[1][i];
    f = w.flag[i];
    if (d->off_pos) reinterpret_cast<uint32_t*>(A.arena + d->off_pos)[j * kTile + t] = (uint32_t)i;  // RoPE positions
  }
  const unsigned bk = __ballot_sync(0xffffffffu, f & 1u), bv = __ballot_sync(0xffffffffu, f & 2u);
  if (lane == 0) {
    halves[0][warp] = bk;
    halves[1][warp] = bv;
  }
  __syncthreads();
  if (t < 2 * nw) {
    const int side = t / nw, wi = t % nw;
    uint64_t* bm = reinterpret_cast<uint64_t*>(blk + 8u * n64) + side * nw;
    uint16_t* rk = reinterpret_cast<uint16_t*>(blk + 8u * n64 + 16u * nw + side * round16(2u * nw));
    const uint64_t word = (uint64_t)halves[side][2 * wi] | ((uint64_t)halves[side][2 * wi + 1] << 32);
    bm[wi] = word;
    int before = 0;
    for (int x = 0; x < 2 * wi; ++x) before += __popc(halves[side][x]);
    rk[wi] = (uint16_t)before;
  }
}

// One warp per residual slot: r = x - gamma x_a (fp64), v = H(s o r), quantize.
__global__ void enc_quant(const EncArgs A) {
  __shared__ double vbuf[8][128];
  const int u = blockIdx.y, side = blockIdx.z;
  const akv_unit_desc* d = unit_desc(A, u);
  EncUnitWs w = unit_ws(A, u, d);
  // slots of this unit: the parameters' count, or the count the full selection chose
  const int N = A.m_obs > 0 ? (int)w.ctrl[2 + side] : (side ? d->n_res_v : d->n_res_k);
  const int wi = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int s = blockIdx.x * 8 + wi;
  if (s >= N) return;
  const int p = w.res_pos[(side ? d->n_res_k : 0) + s];
  const uint32_t st = w.st[side][p];
  const int a = (int)(st & 0xFFFFu);
  const double g = fp16_bits_to_f64(st >> 16);
  const bool valid = w.ctrl[side] != 0u;
  const __nv_bfloat16* X = (side ? A.V : A.K) + ((size_t)u * A.s_max + p) * 128;
  const __nv_bfloat16* XA = anchor_src(A, u, side, reinterpret_cast<const int32_t*>(A.arena_c + d->off_anchor_pos), a);
  double* v = vbuf[wi];
  for (int j = lane; j < 128; j += 32) {
    const double pj = valid ? __dmul_rn(g, bf16_to_f64(XA[j])) : 0.0;
    double r = __dsub_rn(bf16_to_f64(X[j]), pj);
    if (A.rotate) {
      const unsigned long long sb = j < 64 ? A.sign_lo : A.sign_hi;
      if ((sb >> (j & 63)) & 1ull) r = -r;
    }
    v[j] = r;
  }
  __syncwarp();
  if (A.rotate) {
    for (int hh = 1; hh < 128; hh <<= 1) {
      for (int pr = lane; pr < 64; pr += 32) {
        const int j = (pr / hh) * 2 * hh + (pr % hh);
        const double x = v[j], y = v[j + hh];
        v[j] = __dadd_rn(x, y);
        v[j + hh] = __dsub_rn(x, y);
      }
      __syncwarp();
    }
  }
  uint32_t mnh, sch, byte = 0;
  if (A.lloyd) {
    // Lloyd-Max codec (Section 3.1, Appendix A.1): per-token RMS scale fp16(sqrt(sum v^2 / 128)),
    // the sum in index order (lane 0), min 0, codes by the decision regions of v / scale
    double ss = 0.0;
    if (lane == 0)
      for (int j = 0; j < 128; ++j) ss = __dadd_rn(ss, __dmul_rn(v[j], v[j]));
    ss = __shfl_sync(0xffffffffu, ss, 0);
    sch = f64_to_fp16_bits(__dsqrt_rn(__ddiv_rn(ss, 128.0)));
    mnh = 0u;
    const double sc = fp16_bits_to_f64(sch);
    for (int c = 0; c < 4; ++c) {
      int code = 2;  // a zero scale: every level reconstructs 0
      if (sc != 0.0) {
        const double t = __ddiv_rn(v[4 * lane + c], sc);
        code = t < -kLloydT ? 0 : (t < 0.0 ? 1 : (t < kLloydT ? 2 : 3));
      }
      byte |= (uint32_t)code << (2 * c);
    }
  } else {
    // min / max with the first index winning ties (as a sequential scan does)
    double mnv = v[4 * lane], mxv = mnv;
    int mni = 4 * lane, mxi = mni;
    for (int c = 1; c < 4; ++c) {
      const double x = v[4 * lane + c];
      if (x < mnv) { mnv = x; mni = 4 * lane + c; }
      if (x > mxv) { mxv = x; mxi = 4 * lane + c; }
    }
    for (int o = 16; o > 0; o >>= 1) {
      const double omn = __shfl_xor_sync(0xffffffffu, mnv, o);
      const int omi = __shfl_xor_sync(0xffffffffu, mni, o);
      const double omx = __shfl_xor_sync(0xffffffffu, mxv, o);
      const int oxi = __shfl_xor_sync(0xffffffffu, mxi, o);
      if (omn < mnv || (omn == mnv && omi < mni)) { mnv = omn; mni = omi; }
      if (omx > mxv || (omx == mxv && oxi < mxi)) { mxv = omx; mxi = oxi; }
    }
    mnh = f64_to_fp16_bits(mnv);
    const double mn = fp16_bits_to_f64(mnh);
    double t = __ddiv_rn(__dsub_rn(mxv, mn), 3.0);
    if (!(t > 0.0)) t = 0.0;
    sch = f64_to_fp16_bits(t);
    const double sc = fp16_bits_to_f64(sch);
    for (int c = 0; c < 4; ++c) {
      int code = 0;
      if (sc != 0.0) {
        double qv = rint(__ddiv_rn(__dsub_rn(v[4 * lane + c], mn), sc));
        qv = fmin(fmax(qv, 0.0), 3.0);
        code = (int)qv;
      }
      byte |= (uint32_t)code << (2 * c);
    }
  }
  // record r of its tile: the rank of the token among the tile's tokens with this side's bit
  const int ts = w.inv[p], j = ts / kTile, tl = ts % kTile;
  const int n = tile_len(d->len, j), nw = (int)tile_words(n), n64 = 64 * nw;
  const int nkj = (int)w.tcnt[2 * j], nvj = (int)w.tcnt[2 * j + 1];
  const uint8_t* blkc = A.arena_c + d->off_tiles + reinterpret_cast<const uint32_t*>(A.arena_c + d->off_tile_table)[j];
  const uint64_t word = reinterpret_cast<const uint64_t*>(blkc + 8u * n64)[side * nw + (tl >> 6)];
  const uint16_t* rk = reinterpret_cast<const uint16_t*>(blkc + 8u * n64 + 16u * nw + side * round16(2u * nw));
  const int r = (int)rk[tl >> 6] + __popcll(word & ((1ull << (tl & 63)) - 1ull));
  const uint32_t F = tile_fixed_bytes(n);
  const uint32_t sm_off = F + (side ? round16(4u * (uint32_t)nkj) : 0u) + 4u * (uint32_t)r;
  const uint32_t cd_off = F + round16(4u * (uint32_t)nkj) + round16(4u * (uint32_t)nvj) +
                          (side ? 32u * (uint32_t)nkj : 0u) + 32u * (uint32_t)r;
  uint8_t* blk = const_cast<uint8_t*>(blkc);
  if (side == 0) {
    blk[cd_off + lane] = (uint8_t)byte;
  } else {  // value codes: dimension-major groups of 16 records
    uint32_t* grp = reinterpret_cast<uint32_t*>(blk + cd_off - 32u * (uint32_t)r + 512u * (uint32_t)(r / 16));
    for (int c = 0; c < 4; ++c)
      atomicOr(&grp[value_code_word(4 * lane + c)], ((byte >> (2 * c)) & 3u) << value_code_bit(r % 16));
  }
  if (lane == 0) *reinterpret_cast<uint32_t*>(blk + sm_off) = sch | (mnh << 16);
}

// ---- the paper's full selection (Algorithm 1; Section 3.2-3.4, Appendix A.2) --------------
// Each fp64 sum runs in a fixed order (positions, then rows, then dimensions ascending, one
// thread per output), and the exponential is evaluated by fixed steps, so every decision
// (scored anchors, pooled residual slots) comes out the same on any IEEE machine.

// e^x for x <= 0: Cody-Waite argument reduction (ln 2 split into a 42-bit leading part,
// whose product with n is exact, and the remainder), a degree-22 Taylor series of e^r by
// Horner's rule, then the exact scaling by 2^n; about 1 ulp.  Arguments below -700 give 0.
__device__ double exp_neg_dev(double x) {
  if (!(x >= -700.0)) return 0.0;
  const double ln2_hi = 0.693147180559890330187045037746429443359375;
  const double ln2_lo = 5.4979230187083711552420206887987e-14;
  const double n = rint(__ddiv_rn(x, 0.6931471805599453094172321));
  const double r = __dsub_rn(__dsub_rn(x, __dmul_rn(n, ln2_hi)), __dmul_rn(n, ln2_lo));
  double y = 1.0;
  for (int j = 22; j >= 1; --j) y = __dadd_rn(1.0, __dmul_rn(__ddiv_rn(r, (double)j), y));
  return ldexp(y, (int)n);
}

// Logits q_w . K_t / sqrt(D) of every observation row and position (Eq. 4), into alpha.
__global__ void __launch_bounds__(128) enc_obs_logit(const EncArgs A) {
  __shared__ double qs[128];
  const int u = blockIdx.z, wr = blockIdx.y;
  const akv_unit_desc* d = unit_desc(A, u);
  const int S = d->len;
  const int t = blockIdx.x * 128 + threadIdx.x;
  if (blockIdx.x * 128 >= S) return;
  EncUnitWs w = unit_ws(A, u, d);
  qs[threadIdx.x] = bf16_to_f64(A.Q[((size_t)u * A.m_obs + wr) * 128 + threadIdx.x]);
  __syncthreads();
  if (t >= S) return;
  const __nv_bfloat16* X = A.K + ((size_t)u * A.s_max + t) * 128;
  double acc = 0.0;
  for (int j = 0; j < 128; ++j) acc = __dadd_rn(acc, __dmul_rn(qs[j], bf16_to_f64(X[j])));
  w.alpha[(size_t)wr * S + t] = __dmul_rn(acc, __ddiv_rn(1.0, __dsqrt_rn(128.0)));
}

// Softmax of each observation row's logits over all S positions.
__global__ void __launch_bounds__(1024) enc_obs_softmax(const EncArgs A) {
  __shared__ double red[32];
  __shared__ double den_s;
  const int u = blockIdx.y, wr = blockIdx.x;
  const akv_unit_desc* d = unit_desc(A, u);
  const int S = d->len;
  EncUnitWs w = unit_ws(A, u, d);
  double* a = w.alpha + (size_t)wr * S;
  double mx = -INFINITY;
  for (int t = threadIdx.x; t < S; t += blockDim.x) mx = fmax(mx, a[t]);
  for (int o = 16; o > 0; o >>= 1) mx = fmax(mx, __shfl_xor_sync(0xffffffffu, mx, o));
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = mx;
  __syncthreads();
  if (threadIdx.x == 0) {
    double m = red[0];
    for (int i = 1; i < (int)(blockDim.x >> 5); ++i) m = fmax(m, red[i]);
    red[0] = m;
  }
  __syncthreads();
  mx = red[0];
  for (int t = threadIdx.x; t < S; t += blockDim.x) a[t] = exp_neg_dev(__dsub_rn(a[t], mx));
  __syncthreads();
  if (threadIdx.x == 0) {  // the normaliser, summed in position order
    double den = 0.0;
    for (int t = 0; t < S; ++t) den = __dadd_rn(den, a[t]);
    den_s = den;
  }
  __syncthreads();
  const double den = den_s;
  for (int t = threadIdx.x; t < S; t += blockDim.x) a[t] = __ddiv_rn(a[t], den);
}

// Exact output y_w = sum_t alpha_wt V_t of each observation row (positions in order).
__global__ void __launch_bounds__(128) enc_obs_y(const EncArgs A) {
  const int u = blockIdx.y, wr = blockIdx.x, j = threadIdx.x;
  const akv_unit_desc* d = unit_desc(A, u);
  const int S = d->len;
  EncUnitWs w = unit_ws(A, u, d);
  const double* a = w.alpha + (size_t)wr * S;
  const __nv_bfloat16* V = A.V + (size_t)u * A.s_max * 128;
  double acc = 0.0;
  for (int t = 0; t < S; ++t) acc = __dadd_rn(acc, __dmul_rn(a[t], bf16_to_f64(V[(size_t)t * 128 + j])));
  w.yobs[wr * 128 + j] = acc;
}

// Selector score, step 1: the rows' attention averaged over the m rows (into key1 as fp64).
__global__ void enc_score_mean(const EncArgs A) {
  const int u = blockIdx.y;
  const akv_unit_desc* d = unit_desc(A, u);
  const int S = d->len, P = S - min(A.window, S);
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= P) return;
  EncUnitWs w = unit_ws(A, u, d);
  double acc = 0.0;
  for (int wr = 0; wr < A.m_obs; ++wr) acc = __dadd_rn(acc, w.alpha[(size_t)wr * S + t]);
  w.key1[t] = (uint64_t)__double_as_longlong(__ddiv_rn(acc, (double)A.m_obs));
}

// Selector score, step 2: average pooling of width kappa centred on t over [0, P), zero
// outside, divided by kappa (Appendix A.2); the score's bits into key0 (scores are >= 0,
// so their bit patterns order like the values).
__global__ void enc_score_pool(const EncArgs A) {
  const int u = blockIdx.y;
  const akv_unit_desc* d = unit_desc(A, u);
  const int S = d->len, P = S - min(A.window, S);
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= P) return;
  EncUnitWs w = unit_ws(A, u, d);
  const int h = A.kappa / 2;
  double acc = 0.0;
  for (int j = t - h; j <= t + h; ++j)
    if (j >= 0 && j < P) acc = __dadd_rn(acc, __longlong_as_double((long long)w.key1[j]));
  w.key0[t] = (uint64_t)__double_as_longlong(__ddiv_rn(acc, (double)A.kappa));
}

// The floor(rho (k - w)) highest scores (ties: lower position) become anchors: slot_of = -2
// marks them for enc_hash and enc_anchors, every other position gets -1.
__global__ void __launch_bounds__(1024) enc_score_pick(const EncArgs A) {
  __shared__ uint32_t hist[256];
  __shared__ uint32_t bc[2];
  __shared__ int wt[33];
  const int u = blockIdx.x;
  const akv_unit_desc* d = unit_desc(A, u);
  const int S = d->len, k = d->n_anchors, win = min(A.window, S), P = S - win;
  EncUnitWs w = unit_ws(A, u, d);
  const int ns = n_scored(A, k - win);
  uint64_t thr = ~0ull;
  uint32_t need = 0;
  if (ns > 0) thr = block_select(w.key0, P, (uint32_t)ns, true, hist, bc, &need);
  int eq_seen = 0;
  for (int c0 = 0; c0 < S; c0 += 1024) {
    const int p = c0 + threadIdx.x;
    const uint64_t kv = (p < P) ? w.key0[p] : 0ull;
    const int is_eq = (ns > 0 && p < P && kv == thr) ? 1 : 0;
    int eq_tot;
    const int eq_pre = block_scan_flag(is_eq, wt, &eq_tot);
    const int sel = (ns > 0 && p < P) && (kv > thr || (is_eq && (uint32_t)(eq_seen + eq_pre) < need));
    eq_seen += eq_tot;
    if (p < S) w.slot_of[p] = sel ? -2 : -1;
    __syncthreads();
  }
}

// Eq. 6 utilities of the non-anchor positions (one thread per position, rows and
// dimensions in order): key0 = bits(u^K) + 1, key1 = bits(u^V) + 1, anchors 0.
constexpr int UT_ROWS = 16;  // observation rows staged in shared memory at a time
__global__ void __launch_bounds__(128) enc_util(const EncArgs A) {
  __shared__ double qs[UT_ROWS][128];
  __shared__ double ys[UT_ROWS][128];
  const int u = blockIdx.y;
  const akv_unit_desc* d = unit_desc(A, u);
  const int S = d->len;
  if (blockIdx.x * 128 >= S) return;
  EncUnitWs w = unit_ws(A, u, d);
  const int p = blockIdx.x * 128 + threadIdx.x;
  const bool live = p < S && w.slot_of[p] < 0;
  const int32_t* apos = reinterpret_cast<const int32_t*>(A.arena_c + d->off_anchor_pos);
  const __nv_bfloat16 *xk = nullptr, *xv = nullptr, *ak = nullptr, *av = nullptr;
  double gk = 0.0, gv = 0.0, ev = 0.0;
  if (live) {
    xk = A.K + ((size_t)u * A.s_max + p) * 128;
    xv = A.V + ((size_t)u * A.s_max + p) * 128;
    const uint32_t sk = w.st[0][p], sv = w.st[1][p];
    ak = anchor_src(A, u, 0, apos, (int)(sk & 0xFFFFu));
    av = anchor_src(A, u, 1, apos, (int)(sv & 0xFFFFu));
    gk = fp16_bits_to_f64(sk >> 16);
    gv = fp16_bits_to_f64(sv >> 16);
    for (int j = 0; j < 128; ++j) {
      const double rv = __dsub_rn(bf16_to_f64(xv[j]), __dmul_rn(gv, bf16_to_f64(av[j])));
      ev = __dadd_rn(ev, __dmul_rn(rv, rv));
    }
  }
  double uk = 0.0, uv = 0.0;
  for (int w0 = 0; w0 < A.m_obs; w0 += UT_ROWS) {
    const int nr = min(UT_ROWS, A.m_obs - w0);
    __syncthreads();
    for (int e = threadIdx.x; e < nr * 128; e += 128) {
      qs[e >> 7][e & 127] = bf16_to_f64(A.Q[((size_t)u * A.m_obs + w0 + (e >> 7)) * 128 + (e & 127)]);
      ys[e >> 7][e & 127] = w.yobs[(w0 + (e >> 7)) * 128 + (e & 127)];
    }
    __syncthreads();
    if (!live) continue;
    for (int r = 0; r < nr; ++r) {
      const double a = w.alpha[(size_t)(w0 + r) * S + p];
      const double a2 = __dmul_rn(a, a);
      double dq = 0.0, dv = 0.0;
      for (int j = 0; j < 128; ++j) {
        const double rk = __dsub_rn(bf16_to_f64(xk[j]), __dmul_rn(gk, bf16_to_f64(ak[j])));
        dq = __dadd_rn(dq, __dmul_rn(qs[r][j], rk));
        const double c = __dsub_rn(bf16_to_f64(xv[j]), ys[r][j]);
        dv = __dadd_rn(dv, __dmul_rn(c, c));
      }
      uk = __dadd_rn(uk, __dmul_rn(__dmul_rn(a2, __ddiv_rn(__dmul_rn(dq, dq), 128.0)), dv));
      uv = __dadd_rn(uv, __dmul_rn(a2, ev));
    }
  }
  if (p >= S) return;
  if (!live) {
    w.key0[p] = 0ull;
    w.key1[p] = 0ull;
    return;
  }
  uk = __ddiv_rn(uk, (double)A.m_obs);
  uv = __ddiv_rn(uv, (double)A.m_obs);
  w.key0[p] = (uint64_t)__double_as_longlong(uk) + 1ull;
  w.key1[p] = (uint64_t)__double_as_longlong(uv) + 1ull;
}

// One block per request: the side's Eq. 9 share of the budget goes to the highest
// utilities over all KV heads of the request (ties: lower head, then lower position) ->
// per-unit flags, ascending slot lists and counts (ctrl[2 + side]).
__global__ void __launch_bounds__(1024) enc_pool(const EncArgs A, int side) {
  __shared__ uint32_t hist[256];
  __shared__ uint32_t bc[2];
  __shared__ int wt[33];
  __shared__ const uint64_t* keys[256];
  __shared__ int32_t* lists[256];
  __shared__ uint32_t* ctrls[256];
  __shared__ uint8_t* flags[256];
  const int H = A.n_kv_heads, u0 = blockIdx.x * H;
  const akv_unit_desc* d0 = unit_desc(A, u0);
  const int S = d0->len, k = d0->n_anchors;
  for (int h = threadIdx.x; h < H; h += blockDim.x) {
    const akv_unit_desc* d = unit_desc(A, u0 + h);
    EncUnitWs w = unit_ws(A, u0 + h, d);
    keys[h] = side ? w.key1 : w.key0;
    lists[h] = w.res_pos + (side ? d->n_res_k : 0);
    ctrls[h] = w.ctrl;
    flags[h] = w.flag;
  }
  __syncthreads();
  const int64_t N = budget_residuals(A.theta, S, H, A.window, k);
  const int64_t cand = (int64_t)H * (S - k);
  int64_t want = side ? N - N / 2 : N / 2;
  if (want > cand) want = cand;
  const int64_t n = (int64_t)H * S;
  auto key_at = [&](int64_t i) { return keys[i / S][i % S]; };
  uint64_t thr = ~0ull;
  uint32_t need = 0;
  if (want > 0) thr = block_select_f(key_at, n, (uint32_t)want, true, hist, bc, &need);
  int eq_seen = 0;
  for (int h = 0; h < H; ++h) {
    int base = 0;
    for (int c0 = 0; c0 < S; c0 += 1024) {
      const int p = c0 + threadIdx.x;
      const uint64_t kv = p < S ? keys[h][p] : 0ull;
      const int is_eq = (want > 0 && p < S && kv == thr) ? 1 : 0;
      int eq_tot;
      const int eq_pre = block_scan_flag(is_eq, wt, &eq_tot);
      const int sel = (want > 0 && p < S) && (kv > thr || (is_eq && (uint32_t)(eq_seen + eq_pre) < need));
      eq_seen += eq_tot;
      int tot;
      const int pre = block_scan_flag(sel, wt, &tot);
      if (sel) lists[h][base + pre] = p;
      // flags of both sides share bytes: the side-0 launch writes them, side 1 ORs its bit in
      if (p < S) {
        if (side == 0) flags[h][p] = (uint8_t)sel;
        else if (sel) flags[h][p] |= 2u;
      }
      base += tot;
      __syncthreads();
    }
    if (threadIdx.x == 0) ctrls[h][2 + side] = (uint32_t)base;
  }
}

// The arena descriptors take the residual counts the full selection chose (last launch:
// every earlier kernel sizes its scratch from the reserved counts).
__global__ void enc_set_counts(const EncArgs A, int units) {
  const int u = blockIdx.x * blockDim.x + threadIdx.x;
  if (u >= units) return;
  const akv_unit_desc* d = unit_desc(A, u);
  EncUnitWs w = unit_ws(A, u, d);
  akv_unit_desc* dm = reinterpret_cast<akv_unit_desc*>(A.arena + 256) + u;
  const int32_t nk = (int32_t)w.ctrl[2], nv = (int32_t)w.ctrl[3];
  dm->n_res_k = nk;
  dm->n_res_v = nv;
}

}  // namespace

// Scratch of akv_encode_noalloc, for callers that cannot hand the library a
// device workspace.  It is part of the module image: no allocation call makes
// it, and each device that loads the library keeps it until the process exits.
static __device__ __align__(256) unsigned char g_noalloc_scratch[AKV_NOALLOC_SCRATCH_BYTES];

int noalloc_scratch(void** ptr, size_t* bytes) {
  // Host code must not use g_noalloc_scratch's name as a device address: it is
  // a host-side stand-in.  The device address is looked up on every call, with
  // the caller's device current, rather than cached: after cudaDeviceReset the
  // module is loaded again and the array may move, and a context other than the
  // primary one holds its own copy, so a cached address could point at memory
  // this call does not own.  The lookup costs far less than the encode.  The
  // first lookup on a device loads the library's module there.
  void* p = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
  if (e != cudaSuccess) return (int)e;
  *ptr = p;
  *bytes = AKV_NOALLOC_SCRATCH_BYTES;
  return 0;
}

int launch_encode(const Layout& L, const EncodeWs& W, const akv_params& p, const void* K, const void* V, int32_t s_max,
                  void* arena, void* ws, void* stream, const akv_select_params* sel, const void* Q, int32_t m_obs) {
  cudaStream_t st = (cudaStream_t)stream;
  const int units = (int)L.shape.size();
  cudaError_t e;
  // header + descriptors, then the per-unit workspace table at the start of ws
  std::vector<uint8_t> head(kHeaderBytes + kDescBytes * (size_t)units);
  std::memcpy(head.data(), &L.header, sizeof(L.header));
  std::memcpy(head.data() + kHeaderBytes, L.desc.data(), kDescBytes * (size_t)units);
  if ((e = cudaMemsetAsync(arena, 0, (size_t)L.total_bytes, st)) != cudaSuccess) return (int)e;
  if ((e = cudaMemcpyAsync(arena, head.data(), head.size(), cudaMemcpyHostToDevice, st)) != cudaSuccess) return (int)e;
  std::vector<uint64_t> table(W.unit_off.begin(), W.unit_off.end());
  if ((e = cudaMemcpyAsync(ws, table.data(), (size_t)units * 8, cudaMemcpyHostToDevice, st)) != cudaSuccess)
    return (int)e;

  EncArgs A;
  A.arena_c = (const uint8_t*)arena;
  A.arena = (uint8_t*)arena;
  A.ws_base = (const uint8_t*)ws;
  A.ws_off = (const uint64_t*)ws;
  A.K = (const __nv_bfloat16*)K;
  A.V = (const __nv_bfloat16*)V;
  A.s_max = s_max;
  A.n_kv_heads = p.n_kv_heads;
  A.window = p.window;
  A.rotate = (p.flags & AKV_FLAG_ROTATE) ? 1 : 0;
  A.lloyd = (p.flags & AKV_FLAG_LLOYD) ? 1 : 0;
  A.seed = p.seed;
  A.sign_lo = L.header.sign_bits[0];
  A.sign_hi = L.header.sign_bits[1];
  const bool full = sel != nullptr && Q != nullptr && m_obs > 0;
  A.Q = (const __nv_bfloat16*)Q;
  A.m_obs = full ? m_obs : 0;
  A.kappa = full ? sel->kappa : 1;
  A.rho = full ? sel->rho : 0.0f;
  A.theta = full ? sel->theta : 0.0f;

  const unsigned maxS = (unsigned)L.max_len;
  if (full) {  // observation rows' attention, selector scores, the scored anchors
    const unsigned m = (unsigned)m_obs;
    enc_obs_logit<<<dim3((maxS + 127) / 128, m, units), 128, 0, st>>>(A);
    enc_obs_softmax<<<dim3(m, units), 1024, 0, st>>>(A);
    enc_obs_y<<<dim3(m, units), 128, 0, st>>>(A);
    enc_score_mean<<<dim3((maxS + 255) / 256, units), 256, 0, st>>>(A);
    enc_score_pool<<<dim3((maxS + 255) / 256, units), 256, 0, st>>>(A);
    enc_score_pick<<<units, 1024, 0, st>>>(A);
  }
  enc_hash<<<dim3((maxS + 255) / 256, units), 256, 0, st>>>(A);
  enc_anchors<<<units, 1024, 0, st>>>(A);
  enc_rows<<<dim3((unsigned)(L.max_k + 7) / 8, units), 256, 0, st>>>(A);
  if ((e = cudaFuncSetAttribute(enc_assign, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)AS_SMEM)) != cudaSuccess)
    return (int)e;
  enc_assign<<<dim3((maxS + AS_POS - 1) / AS_POS, units, 2), AS_THREADS, AS_SMEM, st>>>(A);
  if (full) {  // Eq. 6 utilities, then each side's pooled top-N per request
    enc_util<<<dim3((maxS + 127) / 128, units), 128, 0, st>>>(A);
    enc_pool<<<units / p.n_kv_heads, 1024, 0, st>>>(A, 0);  // writes the flag bytes
    enc_pool<<<units / p.n_kv_heads, 1024, 0, st>>>(A, 1);  // ORs the value bit in
  } else {
    enc_slots<<<units, 1024, 0, st>>>(A, 0);  // writes the flag bytes
    enc_slots<<<units, 1024, 0, st>>>(A, 1);  // ORs the value bit in
  }
  enc_order<<<units, 1024, 0, st>>>(A);
  enc_tile_count<<<dim3((unsigned)L.max_tiles, units), kTile, 0, st>>>(A);
  enc_tile_table<<<(units + 127) / 128, 128, 0, st>>>(A, units);
  enc_tile_fill<<<dim3((unsigned)L.max_tiles, units), kTile, 0, st>>>(A);
  const int maxN = std::max(L.max_nk, L.max_nv);
  if (maxN > 0) enc_quant<<<dim3((unsigned)(maxN + 7) / 8, units, 2), 256, 0, st>>>(A);
  if (full) enc_set_counts<<<(units + 127) / 128, 128, 0, st>>>(A, units);
  return (int)cudaGetLastError();
}

}  // namespace akv
