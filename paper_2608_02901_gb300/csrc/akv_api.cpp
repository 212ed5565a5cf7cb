// Host side of the C ABI: parameter validation, arena layout, the host packer
// and the thin wrappers that hand validated work to the kernel launchers.
#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <memory>
#include <mutex>
#include <string>
#include <vector>

#include "akv_internal.h"

namespace akv {

namespace {
thread_local std::string g_last_error;

uint64_t align_up(uint64_t x, uint64_t a) { return (x + a - 1) / a * a; }
}  // namespace

akv_status fail(akv_status s, const std::string& msg) {
  g_last_error = msg;
  return s;
}

uint64_t splitmix64(uint64_t x) {
  // SplitMix64 finaliser applied to x advanced by the golden-ratio increment.
  uint64_t z = x + 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

void rotation_signs(uint64_t rot_seed, uint64_t bits[2]) {
  bits[0] = splitmix64(rot_seed);
  bits[1] = splitmix64(rot_seed + 1);
}

akv_status make_layout(const akv_params* p, const int32_t* ctx_lens, Layout* out, const akv_select_params* sel) {
  if (!p || !ctx_lens || !out) return fail(AKV_ERR_INVALID, "null params, ctx_lens or output");
  if (p->head_dim != kD) return fail(AKV_ERR_UNSUPPORTED, "head_dim must be 128");
  if (p->batch < 1 || p->n_kv_heads < 1 || p->n_q_heads < 1)
    return fail(AKV_ERR_INVALID, "batch, n_kv_heads and n_q_heads must be >= 1");
  if (p->n_q_heads % p->n_kv_heads != 0) return fail(AKV_ERR_INVALID, "n_q_heads must be a multiple of n_kv_heads");
  int G = p->n_q_heads / p->n_kv_heads;
  if (G != 1 && G != 2 && G != 4 && G != 8) return fail(AKV_ERR_UNSUPPORTED, "query group size must be 1, 2, 4 or 8");
  if (p->n_kv_heads > 256 || p->batch > (1 << 24)) return fail(AKV_ERR_UNSUPPORTED, "too many heads or requests");
  auto frac_ok = [](float f) { return std::isfinite(f) && f >= 0.0f && f <= 1.0f; };
  if (!frac_ok(p->anchor_frac) || !frac_ok(p->res_frac_k) || !frac_ok(p->res_frac_v))
    return fail(AKV_ERR_INVALID, "fractions must be finite and in [0, 1]");
  if (p->window < 0) return fail(AKV_ERR_INVALID, "window must be >= 0");
  if ((p->flags & ~(AKV_FLAG_ROTATE | AKV_FLAG_LLOYD | AKV_FLAG_ROPE)) != 0) return fail(AKV_ERR_INVALID, "unknown flags");
  if ((p->flags & AKV_FLAG_ROPE) ? !(std::isfinite(p->rope_theta) && p->rope_theta > 1.0f) : p->rope_theta != 0.0f)
    return fail(AKV_ERR_INVALID, "rope_theta must be finite and > 1 with AKV_FLAG_ROPE, and 0 without it");
  if (sel) {
    if (!(std::isfinite(sel->theta) && sel->theta > 0.0f && sel->theta <= 1.0f))
      return fail(AKV_ERR_INVALID, "theta must be in (0, 1]");
    if (!(std::isfinite(sel->rho) && sel->rho >= 0.0f && sel->rho <= 1.0f))
      return fail(AKV_ERR_INVALID, "rho must be in [0, 1]");
    if (sel->kappa < 1 || sel->kappa > 255 || sel->kappa % 2 == 0)
      return fail(AKV_ERR_INVALID, "kappa must be odd and in [1, 255]");
    if (sel->reserved != 0) return fail(AKV_ERR_INVALID, "reserved select field must be 0");
    if (p->window < 1) return fail(AKV_ERR_INVALID, "the full selection needs W >= 1 observation positions");
  }

  Layout& L = *out;
  L = Layout();
  L.G = G;
  const int32_t n_units = p->batch * p->n_kv_heads;
  L.shape.resize(n_units);
  L.desc.resize(n_units);
  uint64_t off = kHeaderBytes + kDescBytes * (uint64_t)n_units;
  for (int32_t b = 0; b < p->batch; ++b) {
    const int32_t S = ctx_lens[b];
    if (S < 1 || S > (1 << 30)) return fail(AKV_ERR_INVALID, "context lengths must be in [1, 2^30]");
    // Anchor budget including the window; residual budgets capped by the non-anchors.
    const int32_t w = p->window < S ? p->window : S;
    int64_t k = (int64_t)std::ceil((double)p->anchor_frac * (double)S);
    if (k < w) k = w;
    if (k > S) k = S;
    int64_t nk = (int64_t)std::floor((double)p->res_frac_k * (double)S);
    int64_t nv = (int64_t)std::floor((double)p->res_frac_v * (double)S);
    if (sel) {  // capacities: the most the request's pooled budget can give one head
      const int64_t N = budget_residuals(sel->theta, S, p->n_kv_heads, p->window, (int32_t)std::min<int64_t>(k, S));
      nk = N / 2;
      nv = N - N / 2;
    }
    if (nk > S - k) nk = S - k;
    if (nv > S - k) nv = S - k;
    if (k < 1) return fail(AKV_ERR_INVALID, "anchor budget is zero (window 0 and anchor_frac * S < 1)");
    if (k > AKV_MAX_ANCHORS) return fail(AKV_ERR_UNSUPPORTED, "more than 65535 anchors in one unit");
    for (int32_t h = 0; h < p->n_kv_heads; ++h) {
      const int32_t u = b * p->n_kv_heads + h;
      UnitShape& sh = L.shape[u];
      sh.S = S;
      sh.k = (int32_t)k;
      sh.nk = (int32_t)nk;
      sh.nv = (int32_t)nv;
      const int32_t nt = (S + kTile - 1) / kTile;
      sh.nt = nt;
      // tile blocks: fixed parts exactly, records, at most 24 bytes of scale padding and
      // 480 bytes of value-code group padding per tile
      uint64_t cap = 0;
      for (int32_t j = 0; j < nt; ++j) cap += tile_fixed_bytes(std::min(kTile, S - j * kTile));
      cap += 36ull * (uint64_t)(nk + nv) + 504ull * (uint64_t)nt;
      if (cap >= (1ull << 32)) return fail(AKV_ERR_UNSUPPORTED, "a unit's tile blocks could exceed 2^32 bytes");
      const uint64_t sizes[kNumSections] = {(uint64_t)k * 256, (uint64_t)k * 256, (uint64_t)k * 4,
                                            tile_table_bytes(nt), cap};
      akv_unit_desc& d = L.desc[u];
      std::memset(&d, 0, sizeof(d));
      d.len = S;
      d.n_anchors = (int32_t)k;
      d.n_res_k = (int32_t)nk;
      d.n_res_v = (int32_t)nv;
      d.n_tiles = nt;
      d.b = b;
      d.h = h;
      off = align_up(off, kSegmentAlign);
      uint64_t* offs = &d.off_anchor_k;
      for (int s = 0; s < kNumSections; ++s) {
        off = align_up(off, kSectionAlign);
        offs[s] = off;
        off += sizes[s];
      }
      d.tiles_capacity = cap;
      d.data_bytes = sizes[kAnchorK] + sizes[kAnchorV] + sizes[kTileTable] + cap;
      if (p->flags & AKV_FLAG_ROPE) {  // original positions of the stored tokens
        off = align_up(off, kSectionAlign);
        d.off_pos = off;
        off += (uint64_t)S * 4;
        d.data_bytes += (uint64_t)S * 4;
      }
      if (nt > L.max_tiles) L.max_tiles = nt;
      if (S > L.max_len) L.max_len = S;
      if (k > L.max_k) L.max_k = (int32_t)k;
      if (nk > L.max_nk) L.max_nk = (int32_t)nk;
      if (nv > L.max_nv) L.max_nv = (int32_t)nv;
    }
  }
  L.total_bytes = align_up(off, kSegmentAlign) + kTailPad;
  akv_arena_header& H = L.header;
  std::memset(&H, 0, sizeof(H));
  H.magic = AKV_ARENA_MAGIC;
  H.version = AKV_ARENA_VERSION;
  H.total_bytes = L.total_bytes;
  H.params = *p;
  H.n_units = n_units;
  H.max_len = L.max_len;
  H.desc_offset = kHeaderBytes;
  H.tile_tokens = kTile;
  rotation_signs(p->rot_seed, H.sign_bits);
  return AKV_OK;
}

void encode_ws_layout(const Layout& L, EncodeWs* ws, int32_t m_obs) {
  // Per unit: two u64 key arrays [S] (anchor hashes, then residual energies
  // per side), slot map i32 [S], residual positions i32 [N_K + N_V],
  // anchor norms (squared, and square roots) f64 [k] per side, 256 B control,
  // stream words u32 [S] per side, flags u8 [S], stored order and inverse
  // i32 [S], run starts u32 [k + 1], record counts u32 [2 n_tiles].
  // A table of per-unit byte offsets (u64 each) leads the workspace.
  ws->unit_off.resize(L.shape.size());
  uint64_t off = align_up((uint64_t)L.shape.size() * 8, 256);
  for (size_t u = 0; u < L.shape.size(); ++u) {
    const UnitShape& s = L.shape[u];
    ws->unit_off[u] = off;
    uint64_t b = 0;
    b += align_up((uint64_t)s.S * 8, 256) * 2;
    b += align_up((uint64_t)s.S * 4, 256);
    b += align_up((uint64_t)(s.nk + s.nv) * 4 + 16, 256);
    b += align_up((uint64_t)s.k * 8, 256) * 4;
    b += 256;
    b += align_up((uint64_t)s.S * 4, 256) * 2;        // stream words per side
    b += align_up((uint64_t)s.S, 256);                // residual flags
    b += align_up((uint64_t)s.S * 4, 256) * 2;        // stored order and its inverse
    b += align_up((uint64_t)(s.k + 1) * 4, 256);      // value-anchor run starts
    b += align_up((uint64_t)s.nt * 8, 256);           // records per tile and side
    if (m_obs > 0) {                                  // full selection: observation rows'
      b += align_up((uint64_t)m_obs * s.S * 8, 256);  // attention alpha [m][S] f64
      b += align_up((uint64_t)m_obs * kD * 8, 256);   // and exact outputs y [m][128] f64
    }
    off += b;
  }
  ws->total = off + 256;
}

// Layouts of recent decode calls.  A decode loop repeats the same (params, lengths) call after
// call; the layout (one descriptor per unit) is then built once instead of on every call.
std::shared_ptr<const Layout> decode_layout(const akv_params* p, const int32_t* ctx_lens, akv_status* st) {
  static std::mutex mu;
  struct Entry {
    akv_params p;
    std::vector<int32_t> lens;
    std::shared_ptr<const Layout> L;
  };
  static std::vector<Entry> recent;  // most recent last, at most kKeep
  constexpr size_t kKeep = 16;
  *st = AKV_OK;
  const bool cacheable = p && ctx_lens && p->batch >= 1 && p->batch <= 4096;
  if (cacheable) {
    std::lock_guard<std::mutex> lk(mu);
    for (size_t i = recent.size(); i-- > 0;) {
      const Entry& e = recent[i];
      if (std::memcmp(&e.p, p, sizeof(akv_params)) == 0 &&
          std::memcmp(e.lens.data(), ctx_lens, sizeof(int32_t) * (size_t)p->batch) == 0 &&
          e.lens.size() == (size_t)p->batch)
        return e.L;
    }
  }
  auto L = std::make_shared<Layout>();
  *st = make_layout(p, ctx_lens, L.get());
  if (*st != AKV_OK) return nullptr;
  if (cacheable) {
    std::lock_guard<std::mutex> lk(mu);
    if (recent.size() >= kKeep) recent.erase(recent.begin());
    recent.push_back(Entry{*p, std::vector<int32_t>(ctx_lens, ctx_lens + p->batch), L});
  }
  return L;
}

}  // namespace akv

using namespace akv;

extern "C" {

const char* akv_status_string(akv_status s) {
  switch (s) {
    case AKV_OK: return "AKV_OK";
    case AKV_ERR_INVALID: return "AKV_ERR_INVALID";
    case AKV_ERR_UNSUPPORTED: return "AKV_ERR_UNSUPPORTED";
    case AKV_ERR_TOO_SMALL: return "AKV_ERR_TOO_SMALL";
    case AKV_ERR_CUDA: return "AKV_ERR_CUDA";
  }
  return "AKV_ERR_UNKNOWN";
}

const char* akv_last_error(void) { return g_last_error.c_str(); }

akv_status akv_unit_shapes(const akv_params* p, const int32_t* ctx_lens_host, int32_t* out_shapes) {
  g_last_error.clear();
  if (!out_shapes) return fail(AKV_ERR_INVALID, "null out_shapes");
  Layout L;
  akv_status st = make_layout(p, ctx_lens_host, &L);
  if (st != AKV_OK) return st;
  for (size_t u = 0; u < L.shape.size(); ++u) {
    out_shapes[4 * u + 0] = L.shape[u].S;
    out_shapes[4 * u + 1] = L.shape[u].k;
    out_shapes[4 * u + 2] = L.shape[u].nk;
    out_shapes[4 * u + 3] = L.shape[u].nv;
  }
  return AKV_OK;
}

akv_status akv_cache_size(const akv_params* p, const int32_t* ctx_lens_host, size_t* arena_bytes,
                          size_t* encode_ws_bytes) {
  g_last_error.clear();
  Layout L;
  akv_status st = make_layout(p, ctx_lens_host, &L);
  if (st != AKV_OK) return st;
  if (arena_bytes) *arena_bytes = (size_t)L.total_bytes;
  if (encode_ws_bytes) {
    EncodeWs W;
    encode_ws_layout(L, &W);
    *encode_ws_bytes = (size_t)W.total;
  }
  return AKV_OK;
}

akv_status akv_cache_header_host(const akv_params* p, const int32_t* ctx_lens_host, void* header_host,
                                 size_t header_bytes) {
  g_last_error.clear();
  Layout L;
  akv_status st = make_layout(p, ctx_lens_host, &L);
  if (st != AKV_OK) return st;
  if (!header_host) return fail(AKV_ERR_INVALID, "null header buffer");
  const size_t need = kHeaderBytes + kDescBytes * L.desc.size();
  if (header_bytes < need) return fail(AKV_ERR_TOO_SMALL, "header buffer shorter than 256 * (1 + B*H)");
  std::memcpy(header_host, &L.header, sizeof(L.header));
  std::memcpy((char*)header_host + kHeaderBytes, L.desc.data(), kDescBytes * L.desc.size());
  return AKV_OK;
}

akv_status akv_cache_pack_host(const akv_params* p, const int32_t* ctx_lens_host, const akv_unit_host* units,
                               void* arena_host, size_t arena_bytes) {
  g_last_error.clear();
  Layout L;
  akv_status st = make_layout(p, ctx_lens_host, &L);
  if (st != AKV_OK) return st;
  if (!units || !arena_host) return fail(AKV_ERR_INVALID, "null units or arena");
  if (arena_bytes < L.total_bytes) return fail(AKV_ERR_TOO_SMALL, "arena shorter than akv_cache_size");
  uint8_t* A = (uint8_t*)arena_host;
  std::memset(A, 0, (size_t)L.total_bytes);
  std::memcpy(A, &L.header, sizeof(L.header));
  std::memcpy(A + kHeaderBytes, L.desc.data(), kDescBytes * L.desc.size());
  for (size_t u = 0; u < L.shape.size(); ++u) {
    const UnitShape& sh = L.shape[u];
    const akv_unit_desc& d = L.desc[u];
    const akv_unit_host& in = units[u];
    const int32_t S = sh.S, k = sh.k;
    if (!in.anchor_k || !in.anchor_v || !in.anchor_pos || !in.idx_k || !in.gamma_k || !in.idx_v || !in.gamma_v ||
        (sh.nk && (!in.res_pos_k || !in.codes_k || !in.scale_k || !in.min_k)) ||
        (sh.nv && (!in.res_pos_v || !in.codes_v || !in.scale_v || !in.min_v)))
      return fail(AKV_ERR_INVALID, "null array in unit " + std::to_string(u));
    // anchor rows, 16-byte chunks swizzled by the slot (chunk c at place c ^ (a % 8))
    for (int side = 0; side < 2; ++side) {
      const uint16_t* src = side ? in.anchor_v : in.anchor_k;
      uint8_t* dst = A + (side ? d.off_anchor_v : d.off_anchor_k);
      for (int32_t a = 0; a < k; ++a)
        for (int c = 0; c < 16; ++c)
          std::memcpy(dst + (size_t)a * 256 + 16 * (c ^ (a & 7)), src + (size_t)a * 128 + 8 * c, 16);
    }
    std::memcpy(A + d.off_anchor_pos, in.anchor_pos, (size_t)k * 4);
    // residual slot of each position per side (-1: none)
    std::vector<int32_t> slot[2];
    for (int side = 0; side < 2; ++side) {
      const uint16_t* idx = side ? in.idx_v : in.idx_k;
      for (int32_t i = 0; i < S; ++i)
        if (idx[i] >= k) return fail(AKV_ERR_INVALID, "anchor index out of range in unit " + std::to_string(u));
      const int32_t n = side ? sh.nv : sh.nk;
      const int32_t* pos = side ? in.res_pos_v : in.res_pos_k;
      slot[side].assign((size_t)S, -1);
      for (int32_t t = 0; t < n; ++t) {
        if (pos[t] < 0 || pos[t] >= S || (t > 0 && pos[t] <= pos[t - 1]))
          return fail(AKV_ERR_INVALID, "residual positions must be ascending and < S in unit " + std::to_string(u));
        slot[side][(size_t)pos[t]] = t;
      }
    }
    // stored order: stable counting sort of positions by value anchor slot
    std::vector<int32_t> start((size_t)k + 1, 0), perm((size_t)S);
    for (int32_t i = 0; i < S; ++i) ++start[(size_t)in.idx_v[i] + 1];
    for (int32_t a = 0; a < k; ++a) start[(size_t)a + 1] += start[(size_t)a];
    for (int32_t i = 0; i < S; ++i) perm[(size_t)start[in.idx_v[i]]++] = i;
    if (d.off_pos) std::memcpy(A + d.off_pos, perm.data(), (size_t)S * 4);  // position of each stored token
    // tile blocks
    uint32_t* table = (uint32_t*)(A + d.off_tile_table);
    uint8_t* tiles = A + d.off_tiles;
    uint32_t off = 0;
    for (int32_t j = 0; j < sh.nt; ++j) {
      const int32_t t0 = j * kTile, n = std::min(kTile, S - t0);
      const uint32_t nw = tile_words(n), n64 = 64 * nw;
      int32_t cnt[2] = {0, 0};
      for (int32_t t = 0; t < n; ++t)
        for (int side = 0; side < 2; ++side) cnt[side] += slot[side][(size_t)perm[(size_t)(t0 + t)]] >= 0;
      table[j] = off;
      table[sh.nt + 1 + j] = (uint32_t)in.idx_v[perm[(size_t)t0]] | ((uint32_t)in.idx_v[perm[(size_t)(t0 + n - 1)]] << 16);
      if ((uint64_t)off + tile_block_bytes(n, cnt[0], cnt[1]) > d.tiles_capacity)
        return fail(AKV_ERR_INVALID, "tile blocks exceed their reserved capacity");  // cannot happen: bound
      uint8_t* blk = tiles + off;
      uint32_t* kst = (uint32_t*)blk;
      uint32_t* vst = kst + n64;
      uint64_t* bm[2] = {(uint64_t*)(vst + n64), (uint64_t*)(vst + n64) + nw};
      uint16_t* rk[2] = {(uint16_t*)(bm[1] + nw), (uint16_t*)(bm[1] + nw) + round16(2 * nw) / 2};
      const uint32_t F = tile_fixed_bytes(n);
      uint32_t* sm[2] = {(uint32_t*)(blk + F), (uint32_t*)(blk + F + round16(4 * (uint32_t)cnt[0]))};
      uint8_t* cd[2];
      cd[0] = blk + F + round16(4 * (uint32_t)cnt[0]) + round16(4 * (uint32_t)cnt[1]);
      cd[1] = cd[0] + 32 * (size_t)cnt[0];
      int32_t r[2] = {0, 0};
      for (int32_t t = 0; t < n; ++t) {
        const int32_t i = perm[(size_t)(t0 + t)];
        kst[t] = (uint32_t)in.idx_k[i] | ((uint32_t)in.gamma_k[i] << 16);
        vst[t] = (uint32_t)in.idx_v[i] | ((uint32_t)in.gamma_v[i] << 16);
        if ((t & 63) == 0)
          for (int side = 0; side < 2; ++side) rk[side][t >> 6] = (uint16_t)r[side];
        for (int side = 0; side < 2; ++side) {
          const int32_t sl = slot[side][(size_t)i];
          if (sl < 0) continue;
          bm[side][t >> 6] |= 1ull << (t & 63);
          const uint16_t sc = side ? in.scale_v[sl] : in.scale_k[sl];
          const uint16_t mn = side ? in.min_v[sl] : in.min_k[sl];
          sm[side][r[side]] = (uint32_t)sc | ((uint32_t)mn << 16);
          const uint8_t* src = (side ? in.codes_v : in.codes_k) + 32 * (size_t)sl;
          if (side == 0) {
            std::memcpy(cd[0] + 32 * (size_t)r[0], src, 32);
          } else {  // dimension-major groups of 16 records
            uint32_t* grp = (uint32_t*)(cd[1] + 512 * (size_t)(r[1] / 16));
            for (int dd = 0; dd < 128; ++dd)
              grp[value_code_word(dd)] |= (uint32_t)((src[dd / 4] >> (2 * (dd % 4))) & 3u) << value_code_bit(r[1] % 16);
          }
          ++r[side];
        }
      }
      off += tile_block_bytes(n, cnt[0], cnt[1]);
    }
    table[sh.nt] = off;
  }
  return AKV_OK;
}

akv_status akv_encode(const akv_params* p, const int32_t* ctx_lens_host, const void* K, const void* V,
                      int32_t s_max, void* arena, size_t arena_bytes, void* ws, size_t ws_bytes,
                      akv_stream_t stream) {
  g_last_error.clear();
  Layout L;
  akv_status st = make_layout(p, ctx_lens_host, &L);
  if (st != AKV_OK) return st;
  if (!K || !V || !arena || !ws) return fail(AKV_ERR_INVALID, "null K, V, arena or workspace");
  if (((uintptr_t)arena % 256) || ((uintptr_t)ws % 256) || ((uintptr_t)K % 16) || ((uintptr_t)V % 16))
    return fail(AKV_ERR_INVALID, "arena and workspace must be 256-byte aligned, K and V 16-byte aligned");
  if (s_max < L.max_len) return fail(AKV_ERR_INVALID, "s_max is smaller than the longest context");
  if (L.shape.size() > 65535) return fail(AKV_ERR_UNSUPPORTED, "encode handles at most 65535 (request, head) units");
  if (arena_bytes < L.total_bytes) return fail(AKV_ERR_TOO_SMALL, "arena shorter than akv_cache_size");
  EncodeWs W;
  encode_ws_layout(L, &W);
  if (ws_bytes < W.total) return fail(AKV_ERR_TOO_SMALL, "encode workspace shorter than akv_cache_size");
  int err = launch_encode(L, W, *p, K, V, s_max, arena, ws, (void*)stream);
  if (err) return fail(AKV_ERR_CUDA, std::string("encode launch failed: ") + cuda_error_string(err));
  return AKV_OK;
}

akv_status akv_cache_size_select(const akv_params* p, const akv_select_params* sel, const int32_t* ctx_lens_host,
                                 size_t* arena_bytes, size_t* encode_ws_bytes) {
  g_last_error.clear();
  if (!sel) return fail(AKV_ERR_INVALID, "null select parameters");
  Layout L;
  akv_status st = make_layout(p, ctx_lens_host, &L, sel);
  if (st != AKV_OK) return st;
  if (arena_bytes) *arena_bytes = (size_t)L.total_bytes;
  if (encode_ws_bytes) {
    EncodeWs W;
    encode_ws_layout(L, &W, p->window * L.G);
    *encode_ws_bytes = (size_t)W.total;
  }
  return AKV_OK;
}

akv_status akv_encode_select(const akv_params* p, const akv_select_params* sel, const int32_t* ctx_lens_host,
                             const void* K, const void* V, const void* Q, int32_t s_max, void* arena, size_t arena_bytes,
                             void* ws, size_t ws_bytes, akv_stream_t stream) {
  g_last_error.clear();
  if (!sel) return fail(AKV_ERR_INVALID, "null select parameters");
  Layout L;
  akv_status st = make_layout(p, ctx_lens_host, &L, sel);
  if (st != AKV_OK) return st;
  if (!K || !V || !Q || !arena || !ws) return fail(AKV_ERR_INVALID, "null K, V, Q, arena or workspace");
  if (((uintptr_t)arena % 256) || ((uintptr_t)ws % 256) || ((uintptr_t)K % 16) || ((uintptr_t)V % 16) ||
      ((uintptr_t)Q % 16))
    return fail(AKV_ERR_INVALID, "arena and workspace must be 256-byte aligned, K, V and Q 16-byte aligned");
  if (s_max < L.max_len) return fail(AKV_ERR_INVALID, "s_max is smaller than the longest context");
  if (L.shape.size() > 65535) return fail(AKV_ERR_UNSUPPORTED, "encode handles at most 65535 (request, head) units");
  if (arena_bytes < L.total_bytes) return fail(AKV_ERR_TOO_SMALL, "arena shorter than akv_cache_size_select");
  const int32_t m_obs = p->window * L.G;
  EncodeWs W;
  encode_ws_layout(L, &W, m_obs);
  if (ws_bytes < W.total) return fail(AKV_ERR_TOO_SMALL, "encode workspace shorter than akv_cache_size_select");
  int err = launch_encode(L, W, *p, K, V, s_max, arena, ws, (void*)stream, sel, Q, m_obs);
  if (err) return fail(AKV_ERR_CUDA, std::string("encode launch failed: ") + cuda_error_string(err));
  return AKV_OK;
}

akv_status akv_encode_noalloc(const akv_params* p, const int32_t* ctx_lens_host, const void* K, const void* V,
                              int32_t s_max, void* arena, size_t arena_bytes, akv_stream_t stream) {
  // Same validation and kernels as akv_encode; the workspace is the library's
  // static scratch array, so nothing here or in the caller allocates device memory.
  g_last_error.clear();
  Layout L;
  akv_status st = make_layout(p, ctx_lens_host, &L);
  if (st != AKV_OK) return st;
  EncodeWs W;
  encode_ws_layout(L, &W);
  if (W.total > AKV_NOALLOC_SCRATCH_BYTES)
    return fail(AKV_ERR_UNSUPPORTED, "encode needs " + std::to_string(W.total) +
                                         " B of scratch, more than the " +
                                         std::to_string((size_t)AKV_NOALLOC_SCRATCH_BYTES) +
                                         " B static array of akv_encode_noalloc; use akv_encode with a workspace");
  void* ws = nullptr;
  size_t ws_bytes = 0;
  int err = noalloc_scratch(&ws, &ws_bytes);
  if (err) return fail(AKV_ERR_CUDA, std::string("scratch address lookup failed: ") + cuda_error_string(err));
  return akv_encode(p, ctx_lens_host, K, V, s_max, arena, arena_bytes, ws, ws_bytes, stream);
}

akv_status akv_decode_set_debug(int32_t ctas, int32_t withhold_last) {
  g_last_error.clear();
  if (ctas < 0 || ctas > 256) return fail(AKV_ERR_INVALID, "ctas must be in [0, 256]");
  if (withhold_last < 0 || withhold_last > 1) return fail(AKV_ERR_INVALID, "withhold_last must be 0 or 1");
  g_debug_cluster.store(ctas);
  g_debug_withhold.store(withhold_last);
  return AKV_OK;
}

akv_status akv_decode_set_events(void* after_scores, void* after_decode) {
  g_last_error.clear();
  if ((after_scores == nullptr) != (after_decode == nullptr))
    return fail(AKV_ERR_INVALID, "both events must be given, or neither");
  set_decode_events(after_scores, after_decode);
  return AKV_OK;
}

// ---- The paper's Table 1 layer layout (byte parity with Appendix A.1) ----

namespace {
// Exact value of an fp16 bit pattern (every fp16 value is a float).
float fp16_bits_to_float(uint16_t h) {
  const int e = (h >> 10) & 31, m = h & 1023;
  const float mag = e == 0 ? std::ldexp((float)m, -24) : (e == 31 ? (m ? NAN : INFINITY) : std::ldexp((float)(1024 + m), e - 25));
  return (h & 0x8000) ? -mag : mag;
}
struct Table1Sizes {
  uint64_t anchors, pos, stream, words, offsets, ids, codes, scales, vslots, total;
};
// Bytes of each Table 1 tensor of one request's layer (H units, context S, k anchors, N_K and N_V
// residual records over its heads), with P = S - W the non-window positions.
Table1Sizes table1_sizes(int64_t S, int64_t H, int64_t W, int64_t k, int64_t NK, int64_t NV) {
  Table1Sizes t;
  const int64_t P = S - W, nw = (P + 63) / 64;
  t.anchors = (uint64_t)(H * k * 128 * 2);  // each of anchor keys and anchor values
  t.pos = (uint64_t)(8 * H * (k - W));
  t.stream = (uint64_t)(2 * H * P * 2);  // each of anchor index and coefficient
  t.words = (uint64_t)(2 * H * nw * 8);  // residual mask
  t.offsets = (uint64_t)(8 * (H + 1));
  t.ids = (uint64_t)(4 * P);
  t.codes = (uint64_t)((NK + NV) * 32);
  t.scales = (uint64_t)((NK + NV) * 4);
  t.vslots = (uint64_t)NV;
  t.total = 2 * t.anchors + t.pos + 2 * t.stream + t.words + t.words / 2 + t.offsets + t.ids + t.codes + t.scales +
            t.vslots;
  return t;
}
// Table 1 needs every request's window inside its context and one scale per record (no min).
akv_status table1_check(const akv_params* p, const Layout& L) {
  if (!(p->flags & AKV_FLAG_LLOYD))
    return fail(AKV_ERR_UNSUPPORTED, "the Table 1 layout stores one scale per record: the Lloyd-Max codec only");
  for (const auto& sh : L.shape)
    if (sh.S < p->window) return fail(AKV_ERR_UNSUPPORTED, "the Table 1 layout needs S >= W in every request");
  return AKV_OK;
}
}  // namespace

akv_status akv_table1_bytes(const akv_params* p, const int32_t* ctx_lens_host, size_t* bytes_per_request) {
  g_last_error.clear();
  Layout L;
  akv_status st = make_layout(p, ctx_lens_host, &L);
  if (st != AKV_OK) return st;
  if (!bytes_per_request) return fail(AKV_ERR_INVALID, "null output");
  if ((st = table1_check(p, L)) != AKV_OK) return st;
  const int H = p->n_kv_heads;
  for (int b = 0; b < p->batch; ++b) {
    int64_t NK = 0, NV = 0;
    for (int h = 0; h < H; ++h) {
      NK += L.shape[(size_t)b * H + h].nk;
      NV += L.shape[(size_t)b * H + h].nv;
    }
    const UnitShape& sh = L.shape[(size_t)b * H];
    bytes_per_request[b] = (size_t)table1_sizes(sh.S, H, p->window, sh.k, NK, NV).total;
  }
  return AKV_OK;
}

akv_status akv_pack_table1_host(const akv_params* p, const int32_t* ctx_lens_host, const akv_unit_host* units,
                                void* out_host, size_t out_bytes) {
  g_last_error.clear();
  Layout L;
  akv_status st = make_layout(p, ctx_lens_host, &L);
  if (st != AKV_OK) return st;
  if (!units || !out_host) return fail(AKV_ERR_INVALID, "null units or output");
  if ((st = table1_check(p, L)) != AKV_OK) return st;
  const int H = p->n_kv_heads;
  const int64_t W = p->window;
  uint8_t* o = (uint8_t*)out_host;
  size_t used = 0;
  for (int b = 0; b < p->batch; ++b) {
    const UnitShape& sh0 = L.shape[(size_t)b * H];
    const int64_t S = sh0.S, k = sh0.k, P = S - W, nw = (P + 63) / 64;
    int64_t NK = 0, NV = 0;
    for (int h = 0; h < H; ++h) {
      const akv_unit_host& in = units[(size_t)b * H + h];
      const UnitShape& sh = L.shape[(size_t)b * H + h];
      NK += sh.nk;
      NV += sh.nv;
      if (!in.anchor_k || !in.anchor_v || !in.anchor_pos || !in.idx_k || !in.gamma_k || !in.idx_v || !in.gamma_v ||
          (sh.nk && (!in.res_pos_k || !in.codes_k || !in.scale_k || !in.min_k)) ||
          (sh.nv && (!in.res_pos_v || !in.codes_v || !in.scale_v || !in.min_v)))
        return fail(AKV_ERR_INVALID, "null array in unit " + std::to_string(b * H + h));
    }
    const Table1Sizes t = table1_sizes(S, H, W, k, NK, NV);
    if (used + t.total > out_bytes) return fail(AKV_ERR_TOO_SMALL, "output shorter than akv_table1_bytes");
    uint8_t* base = o + used;
    size_t at = 0;
    auto put = [&](const void* src, size_t n) {
      std::memcpy(base + at, src, n);
      at += n;
    };
    // anchor keys, anchor values: [H][k][128] bf16
    for (int side = 0; side < 2; ++side)
      for (int h = 0; h < H; ++h) put(side ? units[(size_t)b * H + h].anchor_v : units[(size_t)b * H + h].anchor_k, (size_t)k * 256);
    // anchor positions [H][k - W] int64 (the non-window anchors: the first k - W slots)
    for (int h = 0; h < H; ++h)
      for (int64_t a = 0; a < k - W; ++a) {
        const int64_t v = units[(size_t)b * H + h].anchor_pos[a];
        put(&v, 8);
      }
    // anchor index and coefficient [2][H][P] (b_a = b_gamma = 2), positions 0 .. P-1
    for (int side = 0; side < 2; ++side)
      for (int h = 0; h < H; ++h) put(side ? units[(size_t)b * H + h].idx_v : units[(size_t)b * H + h].idx_k, (size_t)P * 2);
    for (int side = 0; side < 2; ++side)
      for (int h = 0; h < H; ++h)
        put(side ? units[(size_t)b * H + h].gamma_v : units[(size_t)b * H + h].gamma_k, (size_t)P * 2);
    // residual mask [2][H][nw] u64 and exclusive prefix counts [2][H][nw] i32 (within the head)
    std::vector<uint64_t> mask((size_t)(2 * H * nw), 0);
    for (int side = 0; side < 2; ++side)
      for (int h = 0; h < H; ++h) {
        const akv_unit_host& in = units[(size_t)b * H + h];
        const int32_t n = side ? L.shape[(size_t)b * H + h].nv : L.shape[(size_t)b * H + h].nk;
        const int32_t* rp = side ? in.res_pos_v : in.res_pos_k;
        for (int32_t r = 0; r < n; ++r) {
          if (rp[r] < 0 || rp[r] >= P || (r && rp[r] <= rp[r - 1]))
            return fail(AKV_ERR_INVALID, "residual positions must be ascending non-window positions");
          mask[(size_t)((side * H + h) * nw + rp[r] / 64)] |= 1ull << (rp[r] % 64);
        }
      }
    put(mask.data(), mask.size() * 8);
    for (int side = 0; side < 2; ++side)
      for (int h = 0; h < H; ++h) {
        int32_t run = 0;
        for (int64_t wi = 0; wi < nw; ++wi) {
          put(&run, 4);
          run += __builtin_popcountll(mask[(size_t)((side * H + h) * nw + wi)]);
        }
      }
    // head offsets [2][H + 1] i32: each side's records head by head
    for (int side = 0; side < 2; ++side) {
      int32_t off = 0;
      for (int h = 0; h <= H; ++h) {
        put(&off, 4);
        if (h < H) off += side ? L.shape[(size_t)b * H + h].nv : L.shape[(size_t)b * H + h].nk;
      }
    }
    // position ids [P] i32 (every non-window position is kept)
    for (int32_t i = 0; i < (int32_t)P; ++i) put(&i, 4);
    // residual codes [N][32]: key records head by head, then value records (position order);
    // scales [N] fp32; value slot positions [N_V] u8 (position within its 64-position chunk)
    for (int side = 0; side < 2; ++side)
      for (int h = 0; h < H; ++h) {
        const akv_unit_host& in = units[(size_t)b * H + h];
        const int32_t n = side ? L.shape[(size_t)b * H + h].nv : L.shape[(size_t)b * H + h].nk;
        put(side ? in.codes_v : in.codes_k, (size_t)n * 32);
      }
    for (int side = 0; side < 2; ++side)
      for (int h = 0; h < H; ++h) {
        const akv_unit_host& in = units[(size_t)b * H + h];
        const int32_t n = side ? L.shape[(size_t)b * H + h].nv : L.shape[(size_t)b * H + h].nk;
        for (int32_t r = 0; r < n; ++r) {
          if ((side ? in.min_v : in.min_k)[r] & 0x7FFFu)
            return fail(AKV_ERR_INVALID, "a record with a nonzero min: not a Lloyd-Max record");
          const float sc = fp16_bits_to_float((side ? in.scale_v : in.scale_k)[r]);
          put(&sc, 4);
        }
      }
    for (int h = 0; h < H; ++h) {
      const akv_unit_host& in = units[(size_t)b * H + h];
      for (int32_t r = 0; r < L.shape[(size_t)b * H + h].nv; ++r) {
        const uint8_t v = (uint8_t)(in.res_pos_v[r] % 64);
        put(&v, 1);
      }
    }
    if (at != t.total) return fail(AKV_ERR_INVALID, "internal: Table 1 sizes disagree");  // cannot happen
    used += t.total;
  }
  return AKV_OK;
}

akv_status akv_decode_workspace_size(const akv_params* p, const int32_t* ctx_lens_host, size_t* ws_bytes) {
  return akv_decode_workspace_size_suffix(p, ctx_lens_host, 0, ws_bytes);
}

akv_status akv_decode_workspace_size_suffix(const akv_params* p, const int32_t* ctx_lens_host, int32_t suffix_cap,
                                            size_t* ws_bytes) {
  g_last_error.clear();
  Layout L;
  akv_status st = make_layout(p, ctx_lens_host, &L);
  if (st != AKV_OK) return st;
  if (!ws_bytes) return fail(AKV_ERR_INVALID, "null ws_bytes");
  if (suffix_cap < 0 || suffix_cap > AKV_MAX_SUFFIX) return fail(AKV_ERR_INVALID, "suffix_cap out of range");
  *ws_bytes = decode_ws_layout(L, suffix_cap).total;
  return AKV_OK;
}

akv_status akv_decode_attn(const akv_params* p, const int32_t* ctx_lens_host, const void* arena,
                           size_t arena_bytes, const void* q, void* out, float* out_f32, float sm_scale,
                           void* ws, size_t ws_bytes, akv_stream_t stream) {
  return akv_decode_attn_suffix(p, ctx_lens_host, arena, arena_bytes, q, out, out_f32, sm_scale, nullptr, ws, ws_bytes,
                                stream);
}

akv_status akv_decode_attn_suffix(const akv_params* p, const int32_t* ctx_lens_host, const void* arena,
                                  size_t arena_bytes, const void* q, void* out, float* out_f32, float sm_scale,
                                  const akv_suffix* suffix, void* ws, size_t ws_bytes, akv_stream_t stream) {
  if (!g_last_error.empty()) g_last_error.clear();
  akv_status st;
  const std::shared_ptr<const Layout> Lp = decode_layout(p, ctx_lens_host, &st);
  if (st != AKV_OK) return st;
  const Layout& L = *Lp;
  if (!arena || !q || !out) return fail(AKV_ERR_INVALID, "null arena, q or out");
  if (((uintptr_t)arena % 256) || ((uintptr_t)q % 16) || ((uintptr_t)out % 16) || ((uintptr_t)out_f32 % 16))
    return fail(AKV_ERR_INVALID, "arena must be 256-byte aligned; q, out, out_f32 16-byte aligned");
  if (arena_bytes < L.total_bytes) return fail(AKV_ERR_TOO_SMALL, "arena shorter than akv_cache_size");
  if (!std::isfinite(sm_scale)) return fail(AKV_ERR_INVALID, "sm_scale must be finite");
  DecodeSuffix sfx;
  if (suffix) {
    if (!suffix->K || !suffix->V || !suffix->len) return fail(AKV_ERR_INVALID, "suffix: null K, V or len");
    if (((uintptr_t)suffix->K % 16) || ((uintptr_t)suffix->V % 16) || ((uintptr_t)suffix->len % 4))
      return fail(AKV_ERR_INVALID, "suffix: K and V must be 16-byte aligned, len 4-byte aligned");
    if (suffix->cap < 1 || suffix->cap > AKV_MAX_SUFFIX) return fail(AKV_ERR_INVALID, "suffix: cap out of range");
    sfx.K = suffix->K;
    sfx.V = suffix->V;
    sfx.len = suffix->len;
    sfx.cap = suffix->cap;
  }
  if (!ws || ((uintptr_t)ws % 256)) return fail(AKV_ERR_INVALID, "decode workspace must be non-null and 256-byte aligned");
  if (ws_bytes < decode_ws_layout(L, sfx.cap).total)
    return fail(AKV_ERR_TOO_SMALL, "decode workspace shorter than akv_decode_workspace_size(_suffix)");
  std::string why;
  int err = launch_decode(L, *p, arena, arena_bytes, q, out, out_f32, sm_scale, sfx, ws, (void*)stream, &why);
  if (err == -1) return fail(AKV_ERR_UNSUPPORTED, why);
  if (err) return fail(AKV_ERR_CUDA, std::string("decode launch failed: ") + cuda_error_string(err) + " " + why);
  return AKV_OK;
}

akv_status akv_suffix_append(const akv_params* p, const void* K_new, const void* V_new, void* K_suf, void* V_suf,
                             int32_t* len, int32_t cap, akv_stream_t stream) {
  g_last_error.clear();
  if (!p) return fail(AKV_ERR_INVALID, "null params");
  if (p->batch < 1 || p->n_kv_heads < 1 || p->head_dim != AKV_HEAD_DIM)
    return fail(AKV_ERR_INVALID, "batch and n_kv_heads must be >= 1, head_dim 128");
  if (!K_new || !V_new || !K_suf || !V_suf || !len) return fail(AKV_ERR_INVALID, "null pointer");
  if (((uintptr_t)K_new % 16) || ((uintptr_t)V_new % 16) || ((uintptr_t)K_suf % 16) || ((uintptr_t)V_suf % 16) ||
      ((uintptr_t)len % 4))
    return fail(AKV_ERR_INVALID, "rows must be 16-byte aligned, len 4-byte aligned");
  if (cap < 1 || cap > AKV_MAX_SUFFIX) return fail(AKV_ERR_INVALID, "cap out of range");
  const int err = launch_suffix_append(p->batch, p->n_kv_heads, K_new, V_new, K_suf, V_suf, len, cap, (void*)stream);
  if (err) return fail(AKV_ERR_CUDA, std::string("suffix append launch failed: ") + cuda_error_string(err));
  return AKV_OK;
}

}  // extern "C"
