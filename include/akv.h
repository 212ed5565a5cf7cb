/*
 * akv.h — C ABI of the AnchorKV decode-attention hot path on GB300 (sm_103a).
 *
 * AnchorKV (arXiv 2608.02901) stores, per layer and KV head, a few anchor
 * vectors exactly and every other key/value as an anchor index plus one
 * projection coefficient, with a 2-bit rotated residual for budgeted
 * positions (Section 3.1, Eq. 1-3; Appendix A.1, Eq. 12-14).  This library
 * provides the two calls of the paper's problem statement (Section 3, the
 * opening of "Method"; Algorithm 1):
 *
 *   akv_encode      : dense bf16 K, V            -> packed compressed cache
 *   akv_decode_attn : one query per head + cache -> attention output
 *
 * plus a host packer for caches whose logical arrays are given directly.
 * Neither call ever writes a decompressed K or V row to device memory: the
 * reconstruction of Eq. 3 is folded into the attention arithmetic.
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 *  - All pointers are plain addresses.  "device" pointers are CUDA global
 *    memory of the current device; "host" pointers are CPU memory.  The
 *    caller owns every buffer; the library allocates no device memory and
 *    never synchronises the stream it is given (all work is stream-ordered).
 *  - Every call validates its arguments on the host before any launch and
 *    reports problems as an akv_status; it never throws and never aborts.
 *    akv_last_error() returns a thread-local text for the last failure.
 *  - bf16 / fp16 values are passed as their 16-bit IEEE encodings.
 *  - head_dim is 128.  The query-group size G = n_q_heads / n_kv_heads must be
 *    1, 2, 4 or 8; query head j reads KV head floor(j / G).
 *
 * The byte layout of the arena is normative and documented with the
 * akv_arena_header and akv_unit_desc structures below.
 */
#ifndef AKV_H_
#define AKV_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* akv_stream_t; /* a cudaStream_t; NULL = legacy default stream */

typedef enum akv_status {
  AKV_OK = 0,
  AKV_ERR_INVALID = 1,     /* malformed argument: null pointer, bad size, short buffer, bad alignment */
  AKV_ERR_UNSUPPORTED = 2, /* well-formed but outside what this build implements (head_dim, G, k*G) */
  AKV_ERR_TOO_SMALL = 3,   /* a caller buffer (arena, workspace) is smaller than required */
  AKV_ERR_CUDA = 4         /* a CUDA runtime call or kernel launch failed */
} akv_status;

#define AKV_HEAD_DIM 128
#define AKV_FLAG_ROTATE 1u /* residuals carry the randomized Hadamard rotation (Appendix A.1, Eq. 12) */
/* Residual codec (Section 3.1, Appendix A.1 "Codebook"): without this flag, 4 uniform levels
 * on [min, max] per token (c^ = min + code * scale, fp16 scale and min); with it, the
 * four-level Lloyd-Max codebook of a unit Gaussian over a per-token RMS scale:
 * scale = fp16(sqrt(sum_j v_j^2 / 128)) of the rotated residual v, min = 0, code = the
 * decision region of v_j / scale (thresholds 0, +-0.98046875), c^ = scale * L[code] with
 * L = {-1.5078125, -0.453125, 0.453125, 1.5078125} (Max's levels +-0.4528, +-1.5104 to 8
 * significant bits, exact in bf16 and fp16).  Encode and decode must use the same flags. */
#define AKV_FLAG_LLOYD 2u
/* RoPE applied at decode (Section 3.2; Appendix E.1's score kernel): the keys given to the
 * encoder are pre-RoPE and are compressed as they are; the arena keeps each stored token's
 * original position (its index in the request: 0 .. S-1), and the decode scores token i at
 * position p_i as q . R(p_i) x^_i, R(p) the rotate-half RoPE rotation of dimension pairs
 * (j, j + 64) by the angle p theta_j, theta_j = rope_theta^(-2j/128).  q is given already
 * rotated to its own position, as a model computes it.  rope_theta must be finite and > 1. */
#define AKV_FLAG_ROPE 4u
#define AKV_ARENA_MAGIC 0x32564B41u /* "AKV2" */
#define AKV_ARENA_VERSION 4u
#define AKV_MAX_ANCHORS 65535 /* anchor indices are uint16 (Table 1, b_a = 2) */
#define AKV_TILE_TOKENS 1024  /* tokens per tile block of the packed token stream */

/*
 * Compression parameters of one layer (Section 3.2 "Anchor selection",
 * Section 3.4 "Byte-Budgeted Residual Allocation").
 *
 *  k   = min(S, max(min(W, S), ceil(anchor_frac * S)))   anchors per (request, KV head),
 *        the last min(W, S) positions always among them (Section 3.2);
 *  N_K = min(floor(res_frac_k * S), S - k)               key residual slots;
 *  N_V = min(floor(res_frac_v * S), S - k)               value residual slots.
 *  Products are evaluated in double precision from the float fractions.
 *
 *  seed      picks the uniformly sampled anchors (the "random rest" of Algorithm 1);
 *  rot_seed  picks the Hadamard sign pattern s, shared by every layer and head
 *            (Appendix A.1, "Rotation");
 *  flags     AKV_FLAG_ROTATE on: residuals are rotated before quantization.
 */
typedef struct akv_params {
  int32_t batch;      /* B >= 1 */
  int32_t n_kv_heads; /* H >= 1 */
  int32_t n_q_heads;  /* H_q = G * H, G in {1,2,4,8} */
  int32_t head_dim;   /* must be 128 */
  float anchor_frac;  /* in [0, 1] */
  float res_frac_k;   /* in [0, 1] */
  float res_frac_v;   /* in [0, 1] */
  int32_t window;     /* W >= 0 (32 in the paper, Section 4.1) */
  uint64_t seed;
  uint64_t rot_seed;
  uint32_t flags;
  float rope_theta;   /* AKV_FLAG_ROPE: the RoPE base; 0 otherwise */
} akv_params;

/*
 * Arena header, at byte 0 of every arena (256 bytes).  The arena is
 * self-describing: header, then n_units descriptors of 256 bytes each, then
 * one 256-byte-aligned segment per (request b, KV head h), unit u = b*H + h.
 */
typedef struct akv_arena_header {
  uint32_t magic;   /* AKV_ARENA_MAGIC */
  uint32_t version; /* AKV_ARENA_VERSION */
  uint64_t total_bytes;
  akv_params params;
  int32_t n_units; /* B * H */
  int32_t max_len; /* max_b S_b */
  uint64_t desc_offset; /* = 256 */
  uint64_t sign_bits[2]; /* bit j of the 128-bit word: s_j = -1 when set (rotation signs) */
  int32_t tile_tokens;   /* AKV_TILE_TOKENS */
  int32_t reserved1;
  uint8_t pad[256 - 8 - 8 - sizeof(akv_params) - 8 - 8 - 16 - 8];
} akv_arena_header;

/*
 * Per-unit descriptor (256 bytes).  Offsets are bytes from the arena base.
 *
 * Token order.  The S tokens of a unit (anchors included) are stored sorted
 * by their VALUE anchor slot, ties by position: the stored order is the
 * stable sort of positions by a_V(i).  Attention over all S positions with
 * no mask (Eq. 4) does not depend on the order of its terms, and in this
 * order every anchor's value weight w[a] = sum p_i gamma_i (Eq. 3) is a sum
 * over one contiguous run.  Positions themselves are not stored (decode never
 * needs them); anchor_pos keeps the anchors' positions.
 *
 * Sections, in order (each 128-byte aligned):
 *   anchor_k   [k][128] bf16  anchor keys, slots in ascending position (Table 1: anchor keys).
 *                             Row a is stored as 16 chunks of 16 bytes; chunk c (dims
 *                             8c .. 8c+7) sits at chunk place c XOR (a mod 8), so that a
 *                             linear copy to shared memory reads back without bank conflicts.
 *   anchor_v   [k][128] bf16  anchor values, same swizzle
 *   anchor_pos [k] int32      anchor positions (not read by decode)
 *   tile_table [n_tiles + 1] uint32  byte offset of tile block j from off_tiles
 *                             (multiples of 16); entry n_tiles = bytes used;
 *              then [n_tiles] uint32  value-slot range of tile j: the a_V slot of its
 *                             first stored token in bits 0-15, of its last in bits
 *                             16-31 (the anchor-value rows its tokens weight, known
 *                             before the block is read)
 *   tiles                     n_tiles = ceil(S / AKV_TILE_TOKENS) tile blocks
 *
 * Tile block j holds the stored tokens [j T, min(S, (j+1) T)), T = AKV_TILE_TOKENS:
 * n tokens, n64 = n rounded up to 64, nw = n64 / 64, nk / nv residual records.
 *   +0              kst [n64] uint32  key anchor slot a_K in bits 0-15, fp16 gamma^K in
 *                                     bits 16-31 (Eq. 1, Eq. 2); an anchor stores (own slot,
 *                                     1.0); entries n .. n64-1 are 0
 *   +4 n64          vst [n64] uint32  the same for values (a_V non-decreasing over the tile)
 *   +8 n64          bmk [nw] uint64   bit t%64 of word t/64 set <=> token t has a key residual
 *   +8 n64 + 8 nw   bmv [nw] uint64   value residuals
 *   +8 n64 + 16 nw  rkk [nw] uint16   exclusive popcount prefix of bmk words (zero-padded to 16 B)
 *   then            rkv [nw] uint16   of bmv words (zero-padded to 16 B)
 *   F = 8 n64 + 16 nw + 2 * round16(2 nw) bytes so far
 *   +F              smk [nk] uint32   fp16 scale in bits 0-15, fp16 min in bits 16-31 (padded to 16 B)
 *   then            smv [nv] uint32   (padded to 16 B)
 *   then            cdk [nk][32] uint8  2-bit codes of the rotated key residual, code j in
 *                                     byte j/4, bits 2(j%4)..2(j%4)+1
 *   then            cdv  value codes in groups of 16 records (the last group padded with
 *                        zero codes): group G is 128 uint32 words; word
 *                        32 (d/32) + 4 (d%8) + (d%32)/8 holds the code of dimension d of
 *                        record 16 G + s at bits 2 (s/2) + 16 (s%2) .. +1 (even records
 *                        in the low half word, odd ones in the high half).
 *                        ceil(nv/16) * 512 bytes.
 *                        (Dimension-major, because the value side sums over records:
 *                        one 16-byte load gives a thread the codes of 16 records for
 *                        the four dimensions it multiplies.)
 * Record r of a side belongs to the r-th token (in stored order) whose bit is set;
 * token t's record is rk[t/64] + popcount(bm[t/64] & ((1 << (t%64)) - 1)) (the O(1)
 * position-to-slot lookup of Appendix A.1, "Layout", local to the tile).
 * Dequantized rotated residual: c^_j = min + code_j * scale; the residual is
 * r~ = s o (H_128 c^) / 128 with H_128 the unnormalised Sylvester Hadamard matrix
 * (or r~ = c^ when AKV_FLAG_ROTATE is off).
 */
typedef struct akv_unit_desc {
  int32_t len;       /* S */
  int32_t n_anchors; /* k */
  int32_t n_res_k;   /* N_K */
  int32_t n_res_v;   /* N_V */
  int32_t n_tiles;   /* ceil(S / AKV_TILE_TOKENS) */
  int32_t b, h;
  int32_t reserved0;
  uint64_t off_anchor_k, off_anchor_v, off_anchor_pos, off_tile_table, off_tiles;
  uint64_t tiles_capacity; /* bytes reserved for the tile blocks (an upper bound of their use) */
  uint64_t data_bytes;     /* anchors + tile table + tiles_capacity (+ positions): the most one decode reads */
  uint64_t off_pos;        /* AKV_FLAG_ROPE: u32 [S], the original position of each stored token; else 0 */
  uint8_t pad[256 - 32 - 8 * 8];
} akv_unit_desc;

/* ---- Introspection ------------------------------------------------------ */

/* Human-readable name of a status code.  Never NULL. */
const char* akv_status_string(akv_status s);

/* Thread-local detail text of the last failing call on this thread ("" if none). */
const char* akv_last_error(void);

/* ---- Layout ------------------------------------------------------------- */

/*
 * Per-unit shape implied by the parameters (the k, N_K, N_V formulas above).
 *   ctx_lens_host : host [B] int32, 1 <= S_b <= 2^30
 *   out_shapes    : host [B*H][4] int32, filled with (S, k, N_K, N_V) per unit
 * Errors: AKV_ERR_INVALID for null pointers or out-of-range parameters,
 * AKV_ERR_UNSUPPORTED for head_dim != 128, G not in {1,2,4,8}, k > 65535, or a
 * unit whose tile blocks could exceed 2^32 bytes.
 */
akv_status akv_unit_shapes(const akv_params* p, const int32_t* ctx_lens_host, int32_t* out_shapes);

/*
 * Bytes of the arena for these parameters and context lengths, and bytes of
 * the device workspace akv_encode needs for the same inputs.  Either output
 * pointer may be NULL.  The arena size includes header, descriptors and
 * 128/256-byte section padding.
 */
akv_status akv_cache_size(const akv_params* p, const int32_t* ctx_lens_host, size_t* arena_bytes,
                          size_t* encode_ws_bytes);

/*
 * Writes the arena header and descriptor table (the first 256 * (1 + B*H)
 * bytes) into a HOST buffer, so that a caller can read offsets without
 * touching the device.  header_bytes must be >= 256 * (1 + B*H).
 */
akv_status akv_cache_header_host(const akv_params* p, const int32_t* ctx_lens_host, void* header_host,
                                 size_t header_bytes);

/* ---- Encode ------------------------------------------------------------- */

/*
 * Compresses dense keys and values into the arena (Algorithm 1, with anchor
 * selection "last W + uniform rest" and residual slots ranked by residual
 * norm, the paper's ablation variant (ii) of Section 4.3).
 *
 *   K, V  : device bf16 [B][H][s_max][128] (row-major; positions >= S_b unused)
 *   arena : device, arena_bytes >= akv_cache_size(...).arena_bytes, 256-byte aligned
 *   ws    : device scratch, ws_bytes >= encode_ws_bytes, 256-byte aligned;
 *           contents on entry are ignored and on exit are unspecified
 * Decisions (assignment, gamma, slot ranking, codes) are taken in IEEE fp64
 * with a fixed operation order, so the packed bytes are reproducible bit for
 * bit.  Errors: AKV_ERR_INVALID (null, misaligned, s_max < max S_b),
 * AKV_ERR_TOO_SMALL (arena or ws short), AKV_ERR_CUDA (launch failure).
 */
akv_status akv_encode(const akv_params* p, const int32_t* ctx_lens_host, const void* K, const void* V,
                      int32_t s_max, void* arena, size_t arena_bytes, void* ws, size_t ws_bytes,
                      akv_stream_t stream);

/*
 * Encode without any device allocation by the caller or the library.
 * The paper has no counterpart to this entry point; it exists for callers
 * that cannot obtain device memory for a workspace -- for example a process
 * whose memory is owned by another allocator that hands out no scratch, or
 * a caller that must not call cudaMalloc on its critical path.  It runs the
 * same kernels as akv_encode, with the workspace taken from a scratch array
 * of AKV_NOALLOC_SCRATCH_BYTES that lives inside this library
 * (a file-scope __device__ array; every GPU that loads the library holds it
 * until the process exits).
 *
 *   K, V, s_max, arena, arena_bytes : as for akv_encode
 * Limits and behaviour:
 *  - The encode workspace that akv_cache_size reports for (p, ctx_lens_host)
 *    must fit AKV_NOALLOC_SCRATCH_BYTES; otherwise AKV_ERR_UNSUPPORTED and
 *    nothing is launched.
 *  - Every call looks up the array's address on the current device and
 *    context (cudaGetSymbolAddress), so the address stays right after a device
 *    reset or in a non-primary context.  The first call on a device also
 *    loads the library's module there: make that first call before any
 *    stream capture.
 *  - Every call on a device shares the one array and leaves its contents
 *    behind; the kernels need none of it cleared.  Calls whose work overlaps
 *    on the GPU (different streams, no ordering between them) race on the
 *    array: order them on one stream or with events.
 * Errors: as for akv_encode, plus AKV_ERR_CUDA if the set-up lookup fails.
 */
#define AKV_NOALLOC_SCRATCH_BYTES ((size_t)16 << 20)
akv_status akv_encode_noalloc(const akv_params* p, const int32_t* ctx_lens_host, const void* K, const void* V,
                              int32_t s_max, void* arena, size_t arena_bytes, akv_stream_t stream);

/* ---- Encode with the paper's full selection ------------------------------ */

/*
 * The paper's full selection (Algorithm 1; Section 3.2 "Anchor selection",
 * Appendix A.2; Section 3.3 Eq. 6; Section 3.4 Eq. 9):
 *  - anchors: the last min(W, S) positions; floor(rho (k - W)) positions of
 *    [0, S - W) with the highest selector score (the observation rows'
 *    softmax attention, q.K / sqrt(D) over all S positions, averaged over the
 *    m rows and average-pooled over kappa positions centred on each one, zero
 *    outside [0, S - W), divided by kappa; ties: lower position); the rest
 *    sampled uniformly as in akv_encode (smallest SplitMix64 hashes among the
 *    positions not yet chosen);
 *  - residual budget of each request's layer: N of Eq. 9 (Appendix A.1
 *    accounting: anchors, metadata, 36.5 bytes per residual), keys floor(N/2),
 *    values the rest;
 *  - each side's N slots go to the positions with the highest utility of
 *    Eq. 6 over all KV heads of the request (ties: lower head, then lower
 *    position), so heads receive different counts:
 *      u^K_t = 1/m sum_w alpha_wt^2 (q_w . r^K_t)^2 / D |V_t - y_w|^2,
 *      u^V_t = 1/m sum_w alpha_wt^2 |r^V_t|^2,
 *    with alpha_w, y_w the exact attention and output of observation row w.
 * The anchor budget k comes from akv_params.anchor_frac and window as for
 * akv_encode; res_frac_k and res_frac_v are not used.  Every decision is taken
 * in fp64 with a fixed operation order (the exponential is evaluated by a
 * Cody-Waite reduction and a Taylor series), so the packed bytes are
 * reproducible bit for bit.
 */
typedef struct akv_select_params {
  float theta;      /* retained fraction of the bf16 cache, in (0, 1] (Eq. 9) */
  float rho;        /* share of the k - W non-window anchors picked by score, in [0, 1] (0.7) */
  int32_t kappa;    /* pooling width of the selector score, odd, 1..255 (7) */
  int32_t reserved; /* must be 0 */
} akv_select_params;

/*
 * Arena and workspace bytes of akv_encode_select.  The arena reserves, per
 * unit and side, room for min(N_side, S - k) residual records (the most the
 * pooled budget can give one head); the workspace adds the observation rows'
 * attention (8 m S bytes per unit).  m = W * G.
 */
akv_status akv_cache_size_select(const akv_params* p, const akv_select_params* sel, const int32_t* ctx_lens_host,
                                 size_t* arena_bytes, size_t* encode_ws_bytes);

/*
 * Compresses K, V with the full selection.
 *   K, V  : device bf16 [B][H][s_max][128], as for akv_encode
 *   Q     : device bf16 [B][H][m][128], m = W * G: the observation rows of each
 *           KV head, i.e. the queries of the last W positions of the G query
 *           heads that read it (W >= 1)
 *   arena, ws : sizes from akv_cache_size_select, 256-byte aligned
 * The descriptors of the written arena hold each unit's chosen residual
 * counts; akv_decode_attn reads such an arena like any other.  Its launch
 * planner stages, per tile, the residual records that the akv_params
 * fractions it is given suggest: pass fractions near the densities the
 * selection chose (at most N / (2 H S) per side keeps the size check within
 * this arena) for speed; records beyond the staged count are read from
 * global memory, so any such fractions, 0 included, give the same results.
 * Errors: as for akv_encode; AKV_ERR_INVALID for bad select parameters or
 * W = 0 (no observation rows).
 */
akv_status akv_encode_select(const akv_params* p, const akv_select_params* sel, const int32_t* ctx_lens_host,
                             const void* K, const void* V, const void* Q, int32_t s_max, void* arena, size_t arena_bytes,
                             void* ws, size_t ws_bytes, akv_stream_t stream);

/* ---- Host packer -------------------------------------------------------- */

/*
 * Logical arrays of one unit, all HOST memory, sizes from akv_unit_shapes.
 * res_pos_* hold the residual positions in strictly ascending order; every
 * other array is indexed by position (stream arrays) or by slot.
 */
typedef struct akv_unit_host {
  const uint16_t* anchor_k;   /* [k][128] bf16 */
  const uint16_t* anchor_v;   /* [k][128] bf16 */
  const int32_t* anchor_pos;  /* [k] ascending */
  const uint16_t* idx_k;      /* [S] anchor slot per position */
  const uint16_t* gamma_k;    /* [S] fp16 */
  const uint16_t* idx_v;      /* [S] */
  const uint16_t* gamma_v;    /* [S] */
  const int32_t* res_pos_k;   /* [N_K] */
  const uint8_t* codes_k;     /* [N_K][32] */
  const uint16_t* scale_k;    /* [N_K] fp16 */
  const uint16_t* min_k;      /* [N_K] fp16 */
  const int32_t* res_pos_v;   /* [N_V] */
  const uint8_t* codes_v;     /* [N_V][32] */
  const uint16_t* scale_v;    /* [N_V] fp16 */
  const uint16_t* min_v;      /* [N_V] fp16 */
} akv_unit_host;

/*
 * Builds a complete arena image in HOST memory from per-unit logical arrays
 * (units[B*H]), indexed by position; the packer puts the tokens into stored
 * order (stable sort by value anchor slot) and builds the tile blocks.  The
 * caller copies the image to the device.  Validates anchor slot indices (< k),
 * ascending residual positions (< S) and buffer size.
 */
akv_status akv_cache_pack_host(const akv_params* p, const int32_t* ctx_lens_host, const akv_unit_host* units,
                               void* arena_host, size_t arena_bytes);

/* ---- The paper's Table 1 layer layout (byte parity) ---------------------- */

/*
 * Appendix A.1 "Layout", Table 1: the tensors of one compressed layer, charging every byte, with
 * P = S - W non-window positions:
 *   anchor keys [H][k][128] bf16, anchor values [H][k][128] bf16, anchor positions [H][k-W] int64
 *   (the non-window anchors), anchor index [2][H][P] u16 (b_a = 2), coefficient [2][H][P] fp16
 *   (b_gamma = 2), residual mask [2][H][ceil(P/64)] u64 words, prefix counts [2][H][ceil(P/64)]
 *   int32 (exclusive, within the head), head offsets [2][H+1] int32, position ids [P] int32, then
 *   residual codes [N][32] (key records head by head in position order, then value records),
 *   scales [N] fp32, value slot positions [N_V] u8 (position mod 64 of each value record).
 * Its size is exactly M_base of Eq. 11 + N_K (D/4 + 4) + N_V (D/4 + 5): the accounting behind Eq. 9.
 * It is an interchange layout, not read by the decode (whose own format is documented above).
 * Table 1 stores one scale per record, so it needs AKV_FLAG_LLOYD (min = 0), and S >= W.
 * One layer block per request, concatenated in request order.
 */
akv_status akv_table1_bytes(const akv_params* p, const int32_t* ctx_lens_host, size_t* bytes_per_request);
/* Packs logical units (as for akv_cache_pack_host, minima 0) into the Table 1 layout in HOST memory.
 * Errors: AKV_ERR_INVALID (null arrays, residual positions not ascending non-window positions, a
 * nonzero min), AKV_ERR_UNSUPPORTED (not the Lloyd-Max codec, S < W), AKV_ERR_TOO_SMALL. */
akv_status akv_pack_table1_host(const akv_params* p, const int32_t* ctx_lens_host, const akv_unit_host* units,
                                void* out_host, size_t out_bytes);

/* ---- Decode ------------------------------------------------------------- */

/*
 * Bytes of device workspace akv_decode_attn needs for these parameters and
 * context lengths: the anchor scores of every unit (4 G bytes per anchor),
 * their maxima per chunk of 64 anchors, one arrival counter per unit, and
 * the partial sums of the CTAs that share a unit (about 8.5 KB per query head
 * and (CTA or unit) slot, at most 256 CTAs).  Contents on entry are ignored.
 */
akv_status akv_decode_workspace_size(const akv_params* p, const int32_t* ctx_lens_host, size_t* ws_bytes);

/*
 * Single-query decode attention read directly from the compressed cache
 * (Eq. 3 inside Eq. 4): for each request b and query head j with KV head
 * h = j / G,
 *     l_i = sm_scale * q . x^K_i,   out = sum_i softmax(l)_i x^V_i,
 * over all S_b positions (no mask), with x^ reconstructed per Eq. 3.
 *
 *   arena     : device, as written by akv_encode or copied from akv_cache_pack_host
 *               for the same (p, ctx_lens_host), or by akv_encode_select
 *   arena_bytes : the arena's whole size (akv_cache_size, or akv_cache_size_select
 *               for a full-selection arena): the score launch reads anchor rows
 *               through a tensor map of exactly this many bytes, and a unit whose
 *               anchor rows lie outside it gets NaN outputs
 *   q         : device bf16 [B][H_q][128]
 *   out       : device bf16 [B][H_q][128], round-to-nearest-even of the fp32 result
 *   out_f32   : device fp32 [B][H_q][128] or NULL
 *   ws        : device workspace, 256-byte aligned, of >= akv_decode_workspace_size
 *               bytes; calls that overlap on the GPU need separate workspaces
 * Two launches: the anchor scores of every unit (persistent, tensor cores with
 * tensor-memory accumulators, tiles of 128 anchors brought by tensor copies), then
 * the decode itself, one CTA per SM over equal shares of all units' tile blocks.
 * Errors: AKV_ERR_INVALID (null/misaligned pointers, bad sizes), AKV_ERR_TOO_SMALL
 * (arena or workspace short), AKV_ERR_UNSUPPORTED (no shared-memory plan fits),
 * AKV_ERR_CUDA (launch failure).
 * Ordering: both launches are ordinary launches on `stream`: they start after all
 * preceding work in the stream and complete before any later work starts.
 */
akv_status akv_decode_attn(const akv_params* p, const int32_t* ctx_lens_host, const void* arena,
                           size_t arena_bytes, const void* q, void* out, float* out_f32, float sm_scale,
                           void* ws, size_t ws_bytes, akv_stream_t stream);

/* ---- Exact dense suffix (generated tokens) -------------------------------- */

/*
 * Tokens produced during decoding stay exact: their keys and values are
 * appended in bf16 to a dense suffix and never compressed, and the compressed
 * prefix and the suffix are attended in one softmax (Appendix E.1, the combine
 * kernel; Appendix E.2, generated tokens).  The suffix is caller-owned device
 * memory; its lengths live on the device, so that an append and a decode can be
 * replayed from one CUDA graph step after step.
 *   K, V : device bf16 [B][H_kv][cap][128]: row t of (request b, KV head h) at
 *          ((b H_kv + h) cap + t) 128 elements (keys as the caller's model uses
 *          them, the same as the keys given to akv_encode)
 *   len  : device int32 [B]: the tokens held by each request, 0 .. cap; rows at
 *          or past len are never read
 *   cap  : tokens per (request, KV head), 1 .. AKV_MAX_SUFFIX
 */
#define AKV_MAX_SUFFIX (1 << 20)
typedef struct akv_suffix {
  const void* K;
  const void* V;
  const int32_t* len;
  int32_t cap;
} akv_suffix;

/*
 * Workspace of akv_decode_attn_suffix for a suffix of at most suffix_cap tokens
 * per request: akv_decode_workspace_size's, plus one partial slot (about
 * 0.5 KB per query head) per unit and chunk of 64 suffix tokens.  suffix_cap 0
 * gives akv_decode_workspace_size's value.
 * Errors: AKV_ERR_INVALID (bad parameters, suffix_cap < 0 or > AKV_MAX_SUFFIX).
 */
akv_status akv_decode_workspace_size_suffix(const akv_params* p, const int32_t* ctx_lens_host, int32_t suffix_cap,
                                            size_t* ws_bytes);

/*
 * akv_decode_attn over the compressed prefix and the dense suffix together:
 * for request b with n = suffix->len[b] suffix tokens,
 *     out = sum_{i < S_b} w_i x^V_i + sum_{t < n} w_{S_b + t} V_suf[t],
 *     w = softmax over the S_b + n logits sm_scale q . x^K_i and sm_scale q . K_suf[t].
 * suffix NULL is akv_decode_attn.  A third launch scores each chunk of 64 suffix
 * tokens and sums its values under the chunk's own maximum; the unit's combine
 * rescales those partials to the common maximum (one softmax, exactly).
 *   ws : >= akv_decode_workspace_size_suffix(p, ctx_lens_host, suffix->cap)
 * Errors: those of akv_decode_attn, and AKV_ERR_INVALID for a suffix with null
 * or misaligned pointers (K, V 16-byte aligned; len 4-byte) or cap out of range.
 * With AKV_FLAG_ROPE the suffix keys are pre-RoPE too: suffix token t of request b sits at
 * position S_b + t and is turned there before it is scored.
 * Lengths above cap are taken as cap.
 */
akv_status akv_decode_attn_suffix(const akv_params* p, const int32_t* ctx_lens_host, const void* arena,
                                  size_t arena_bytes, const void* q, void* out, float* out_f32, float sm_scale,
                                  const akv_suffix* suffix, void* ws, size_t ws_bytes, akv_stream_t stream);

/*
 * The append path (Appendix E.2): one new token per request.  For every request b
 * with len[b] < cap, rows K_new[b][h] and V_new[b][h] (device bf16 [B][H_kv][128])
 * are copied to row len[b] of (b, h) in K_suf and V_suf, and len[b] is then
 * incremented, on the device.  A request whose suffix is full (len[b] >= cap) is
 * left unchanged; its len stays at cap, which is how the caller sees it.
 * One launch on `stream`; the lengths are read and written only by it.
 * Errors: AKV_ERR_INVALID (bad parameters, null or misaligned pointers: rows
 * 16-byte aligned, len 4-byte aligned; cap out of range), AKV_ERR_CUDA.
 */
akv_status akv_suffix_append(const akv_params* p, const void* K_new, const void* V_new, void* K_suf, void* V_suf,
                             int32_t* len, int32_t cap, akv_stream_t stream);

/* ---- Testing and tuning controls ------------------------------------------ */

/*
 * Process-wide controls of akv_decode_attn, for tests and tuning (the paper has
 * no counterpart).  Both are 0 by default, which is normal operation; a call
 * applies to every decode launch issued after it, on every thread.
 *   ctas          : 0 = one decode CTA per SM; 1..256 = that many CTAs (at most
 *                   one per tile block), which moves the boundaries of the ranges
 *                   of tile blocks the CTAs share out
 *   withhold_last : 1 = every CTA withholds the last tile block of its range, so
 *                   the waits on it run out after their bound (about 2 s): the
 *                   call returns and the outputs of the units of those tiles are
 *                   NaN.  This tests the bounded waits (failure detection) without
 *                   any GPU fault.
 * Errors: AKV_ERR_INVALID for values out of range.
 */
akv_status akv_decode_set_debug(int32_t ctas, int32_t withhold_last);

/*
 * Timing aid (process-wide, like akv_decode_set_debug): with non-null events, every
 * later akv_decode_attn call records `after_scores` on its stream right after its
 * first launch (the anchor scores) and `after_decode` right after its second (the
 * decode), so that a caller who records an event before the call can time each
 * launch with cudaEventElapsedTime.  Nothing is skipped or changed in the work.
 *   after_scores, after_decode : cudaEvent_t handles created by the caller (both
 *                                null = off; ownership stays with the caller, who
 *                                must clear them before destroying the events)
 * Errors: AKV_ERR_INVALID if exactly one of the two is null.  A failed record makes
 * the decode call return AKV_ERR_CUDA.
 */
akv_status akv_decode_set_events(void* after_scores, void* after_decode);

#ifdef __cplusplus
} /* extern "C" */
#endif

#endif /* AKV_H_ */
