// Internal declarations shared by the host API and the CUDA translation units.
#pragma once

#include <atomic>
#include <cmath>
#include <cstddef>
#include <cstdint>
#include <string>
#include <vector>

#include "akv.h"

namespace akv {

constexpr int kD = 128;
constexpr uint64_t kSectionAlign = 128;
constexpr uint64_t kSegmentAlign = 256;
constexpr uint64_t kHeaderBytes = 256;
constexpr uint64_t kDescBytes = 256;
constexpr uint64_t kTailPad = 256;  // bytes after the last section, so 16-byte rounded copies stay inside

static_assert(sizeof(akv_arena_header) == 256, "header must be 256 bytes");
static_assert(sizeof(akv_unit_desc) == 256, "descriptor must be 256 bytes");

#ifdef __CUDACC__
#define AKV_HD __host__ __device__
#else
#define AKV_HD
#endif

constexpr int kTile = AKV_TILE_TOKENS;

// Geometry of one tile block (the layout documented with akv_unit_desc).
AKV_HD constexpr uint32_t round16(uint32_t x) { return (x + 15u) & ~15u; }
AKV_HD constexpr uint32_t tile_words(int n) { return (uint32_t)(n + 63) / 64u; }
// streams, bitmaps and rank words of a tile of n tokens
AKV_HD constexpr uint32_t tile_fixed_bytes(int n) {
  return 8u * 64u * tile_words(n) + 16u * tile_words(n) + 2u * round16(2u * tile_words(n));
}
// value codes: groups of 16 records, 512 bytes each (the last group padded)
AKV_HD constexpr uint32_t value_code_bytes(int nv) { return 512u * (((uint32_t)nv + 15u) / 16u); }
AKV_HD constexpr uint32_t tile_block_bytes(int n, int nk, int nv) {
  return tile_fixed_bytes(n) + round16(4u * (uint32_t)nk) + round16(4u * (uint32_t)nv) + 32u * (uint32_t)nk +
         value_code_bytes(nv);
}
// tile table section: n_tiles + 1 block offsets, then one value-slot range word per tile
AKV_HD constexpr uint64_t tile_table_bytes(int nt) { return 4ull * (uint64_t)(2 * nt + 1); }
// word of dimension d in a group of value codes
AKV_HD constexpr uint32_t value_code_word(int d) { return 32u * (uint32_t)(d / 32) + 4u * (uint32_t)(d % 8) + (uint32_t)((d % 32) / 8); }
// bit of record slot s (0..15) in a value-code word: even slots in the low half word
AKV_HD constexpr uint32_t value_code_bit(int s) { return 2u * (uint32_t)(s / 2) + 16u * (uint32_t)(s % 2); }

// Eq. 9 residual count of one layer (one request's H KV heads at context S), with the fixed
// bytes M_base of Eq. 11 and the residual cost of the Appendix A.1 accounting.  M_base per
// head: bf16 anchor keys and values (4 k D bytes), int64 positions of the k - w non-window
// anchors, a 2-byte index and a 2-byte coefficient per side for each of the P = S - w other
// positions, and per side a 64-bit mask word and a 32-bit prefix word per 64 positions;
// shared by the heads: H + 1 int64 head offsets and P int32 position ids.  M_full = 4 S H D
// (bf16 keys and values).  One residual costs the mean of a key record (D/4 code bytes and
// an fp32 scale) and a value record (one more byte of position).  Every term is an integer
// below 2^53 except theta * M_full, so host and device evaluate it identically.  Keys take
// floor(N / 2) slots, values the rest (Section 3.4).
AKV_HD inline int64_t budget_residuals(float theta, int32_t S, int32_t H, int32_t W, int32_t k) {
  const int64_t w = W < S ? W : S;
  const int64_t P = (int64_t)S - w;
  const int64_t m_full = 4ll * S * H * kD;
  const int64_t m_base = (int64_t)H * (4ll * k * kD + 8ll * (k - w) + 8ll * P) + 24ll * H * ((P + 63) / 64) +
                         8ll * (H + 1) + 4ll * P;
  const double b_res = (double)((kD / 4 + 4) + (kD / 4 + 5)) / 2.0;
  const double n = floor(((double)theta * (double)m_full - (double)m_base) / b_res);
  return n > 0.0 ? (int64_t)n : 0;
}

// Section indices inside one unit segment, in storage order.
enum Section { kAnchorK = 0, kAnchorV, kAnchorPos, kTileTable, kTiles, kNumSections };

struct UnitShape {
  int32_t S = 0, k = 0, nk = 0, nv = 0, nt = 0;
};

struct Layout {
  std::vector<UnitShape> shape;        // per unit
  std::vector<akv_unit_desc> desc;     // per unit, offsets from the arena base
  akv_arena_header header{};
  uint64_t total_bytes = 0;
  int32_t max_len = 0, max_k = 0, max_nk = 0, max_nv = 0, max_tiles = 0;
  int G = 0;
};

// Records a failure text for akv_last_error() and returns the status.
akv_status fail(akv_status s, const std::string& msg);

// Validates parameters and context lengths and fills the layout.  With `sel` (the
// paper's full selection), each unit's residual capacity per side is the most the pooled
// Eq. 9 budget of its request can give one head: min(N_side, S - k); the descriptors of an
// encoded arena then hold the counts the selection chose.
akv_status make_layout(const akv_params* p, const int32_t* ctx_lens, Layout* out,
                       const akv_select_params* sel = nullptr);

// 128-bit rotation sign mask: bit j set <=> s_j = -1.
void rotation_signs(uint64_t rot_seed, uint64_t bits[2]);

uint64_t splitmix64(uint64_t x);

// Encode workspace layout (device), per unit.
struct EncodeWs {
  std::vector<uint64_t> unit_off;  // byte offset of each unit's scratch in ws
  uint64_t total = 0;
};
// m_obs > 0: scratch of the full selection (observation rows' attention and outputs) as well.
void encode_ws_layout(const Layout& L, EncodeWs* ws, int32_t m_obs = 0);

// Kernel launchers (defined in the .cu files).  Return cudaError_t as int.
// sel / Q non-null: the paper's full selection with m_obs observation rows per KV head.
int launch_encode(const Layout& L, const EncodeWs& W, const akv_params& p, const void* K, const void* V, int32_t s_max,
                  void* arena, void* ws, void* stream, const akv_select_params* sel = nullptr,
                  const void* Q = nullptr, int32_t m_obs = 0);
// Decode workspace (device): anchor scores [units][ka][G] f32, query headers, chunk maxima,
// arrival counters, partial slots; byte offsets from the workspace base (256-byte aligned).
struct DecodeWs {
  size_t o_sa = 0, o_uh = 0, o_cmax = 0, o_cnt = 0, o_part = 0, o_suf = 0, o_lg = 0, total = 0;
};
// The dense suffix of a decode call (akv_suffix): bf16 rows [B][H_kv][cap][128] and the tokens
// held per request (device int32 [B]); null K = no suffix.
struct DecodeSuffix {
  const void* K = nullptr;
  const void* V = nullptr;
  const int32_t* len = nullptr;
  int32_t cap = 0;
};
// Tokens per suffix chunk (one score-launch CTA each, one partial slot each).
constexpr int kSuffixChunk = 64;
// Workspace of a decode call whose suffix holds at most `suffix_cap` tokens per request.
DecodeWs decode_ws_layout(const Layout& L, int32_t suffix_cap = 0);
int launch_decode(const Layout& L, const akv_params& p, const void* arena, size_t arena_bytes, const void* q, void* out, float* out_f32,
                  float sm_scale, const DecodeSuffix& sfx, void* ws, void* stream, std::string* why);
// Appends one token per request to the dense suffix (akv_suffix_append); returns a cudaError_t.
int launch_suffix_append(int32_t B, int32_t H, const void* K_new, const void* V_new, void* K_suf, void* V_suf,
                         int32_t* len, int32_t cap, void* stream);
const char* cuda_error_string(int err);
// Testing controls of the decode launch (akv_decode_set_debug), 0 = normal operation.
extern std::atomic<int> g_debug_cluster, g_debug_withhold;
// Timing aid of the decode launch (akv_decode_set_events): events recorded after each of
// its two launches; both null = off.
void set_decode_events(void* after_scores, void* after_decode);
// Device address of the library's static encode scratch on the current device
// and context (looked up on every call); returns a cudaError_t as int.
int noalloc_scratch(void** ptr, size_t* bytes);

}  // namespace akv
