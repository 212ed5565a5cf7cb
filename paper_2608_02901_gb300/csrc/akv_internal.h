// Internal declarations shared by the host API and the CUDA translation units.
#pragma once

#include <atomic>
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
// word of dimension d in a group of value codes
AKV_HD constexpr uint32_t value_code_word(int d) { return 32u * (uint32_t)(d / 32) + 4u * (uint32_t)(d % 8) + (uint32_t)((d % 32) / 8); }
// bit of record slot s (0..15) in a value-code word: even slots in the low half word
AKV_HD constexpr uint32_t value_code_bit(int s) { return 2u * (uint32_t)(s / 2) + 16u * (uint32_t)(s % 2); }

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

// Validates parameters and context lengths and fills the layout.
akv_status make_layout(const akv_params* p, const int32_t* ctx_lens, Layout* out);

// 128-bit rotation sign mask: bit j set <=> s_j = -1.
void rotation_signs(uint64_t rot_seed, uint64_t bits[2]);

uint64_t splitmix64(uint64_t x);

// Encode workspace layout (device), per unit.
struct EncodeWs {
  std::vector<uint64_t> unit_off;  // byte offset of each unit's scratch in ws
  uint64_t total = 0;
};
void encode_ws_layout(const Layout& L, EncodeWs* ws);

// Kernel launchers (defined in the .cu files).  Return cudaError_t as int.
int launch_encode(const Layout& L, const EncodeWs& W, const akv_params& p, const void* K, const void* V, int32_t s_max,
                  void* arena, void* ws, void* stream);
int launch_decode(const Layout& L, const akv_params& p, const void* arena, const void* q, void* out, float* out_f32,
                  float sm_scale, void* stream, std::string* why);
const char* cuda_error_string(int err);
// Testing controls of the decode launch (akv_decode_set_debug), 0 = normal operation.
extern std::atomic<int> g_debug_cluster, g_debug_withhold;
// Device address of the library's static encode scratch on the current device
// and context (looked up on every call); returns a cudaError_t as int.
int noalloc_scratch(void** ptr, size_t* bytes);

}  // namespace akv
