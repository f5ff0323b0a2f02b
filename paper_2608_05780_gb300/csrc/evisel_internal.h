// Internal structures shared by the host planner (evisel_capi.cpp) and the
// sm_103a kernels. Not part of the public ABI.
#pragma once

#include <atomic>
#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>
#include <mutex>

namespace evisel {

// One kept kv tile of a work item: keys [start, start + len) (global token
// indices, one video). `diag` marks the tile that holds the query tile's own
// positions: causal masking inside it. `visual` marks visual-token tiles, whose
// logits the text rows spill for the evidence pass.
struct KvTile {
  int32_t start;
  int16_t len;
  uint8_t diag;
  uint8_t visual;
};
static_assert(sizeof(KvTile) == 8, "KvTile is packed into 8 bytes");

// Query-head slots per work item. A slot is one 128-row MMA tile: one head
// for 128-token tiles, two consecutive heads for 64-token tiles. Both slots of
// an item belong to one KV group and share every K/V tile the CTA loads.
constexpr int kSlots = 2;

// One CTA's work: a query row tile of up to kSlots * (128 / tile) consecutive
// query heads of one KV group against a contiguous range of its kept kv tiles.
// Heads past the end of the group are left out.
struct WorkItem {
  int32_t q_start;    // global index of the tile's first query token
  int32_t q_len;      // valid rows (<= tile)
  int32_t head;       // first query head
  int32_t kv_begin;   // index into the KvTile list
  int32_t kv_count;   // >= 1
  int32_t part;       // split-KV partial of slot 0 (slot s uses part + s), -1 when the item writes O/LSE
  int32_t video;      // video index
  int32_t text_row0;  // index of the first row among the video's text rows, -1 for visual rows
};
static_assert(sizeof(WorkItem) == 32, "WorkItem is 32 bytes");

// Per-video layout used by the spill and the evidence pass.
struct VideoInfo {
  int64_t spill_off;  // float offset of this video's logit block [hq, text_pitch / 32, n_vis, 32]
  int32_t vis_start;  // global index of its first visual token
  int32_t n_vis;
  int32_t n_text;
  int32_t text_pitch; // n_text rounded up to a multiple of 32 (rows of the spill, in blocks of 32)
  int32_t vis_off;    // column offset of its tokens in the token map
  int32_t frame_off;  // column offset of its frames in the frame map
};
static_assert(sizeof(VideoInfo) == 32, "VideoInfo is 32 bytes");

// One slot of a text row tile whose kv range was split over several items:
// the partial of split k sits in partial slot part0 + k * stride.
struct CombineGroup {
  int32_t q_start;
  int32_t q_len;
  int32_t head;
  int32_t part0;
  int32_t nsplit;
  int32_t stride;
  int32_t pad1, pad2;
};
static_assert(sizeof(CombineGroup) == 32, "CombineGroup is 32 bytes");

// Column chunk of the evidence pass: 128 visual tokens of one video.
struct EvChunk {
  int32_t video;
  int32_t col0;       // first visual column within the video
};

struct ProbeLaunch {
  CUtensorMap tm_q, tm_k, tm_v;     // 3-D maps {d, heads, tokens}, box {64, 1, tile}, 128B swizzle
  CUtensorMap tm_o;                 // O, laid out and boxed like Q (epilogue stores)
  const WorkItem* items;
  const KvTile* kv;
  const VideoInfo* videos;
  void* o;                          // bf16 [N, hq, d]
  float* lse;                       // [hq, N]
  float* spill;                     // text-row logits
  float* part_o;                    // [slots, 128, d] fp32, unnormalised
  float2* part_ml;                  // [slots, 128] (running max in log2 units, row sum)
  int* status;                      // device status word
  int n_items;
  int n_tok;
  int hq, hkv, head_dim, tile;
  float scale_log2;                 // softmax_scale * log2(e)
  float scale;                      // softmax_scale
  // Cross-frame partials of the visual rows (null when not requested):
  // [hq, fs_nnz, tile / fs_span, tile] fp32, fs_nnz = kept visual kv tiles
  // (the mask's nonzeros, in mask order), fs_span = min(N_v, 64) keys per
  // partial (a key frame is N_v / fs_span consecutive spans).
  float* fspill;
  int fs_nnz, fs_span;
  // Per-row block masks (null: the tile mask alone): keep[h][word][row], bit j
  // of word w = block 32 w + j of the row's video, blocks of keep_block tokens.
  const uint32_t* keep;
  int keep_words, keep_block;
};

struct CombineLaunch {
  const CombineGroup* groups;
  const float* part_o;
  const float2* part_ml;
  void* o;
  float* lse;
  int n_groups;
  int n_tok, hq, hkv, head_dim, tile;
};

struct EvidenceLaunch {
  const EvChunk* chunks;
  const VideoInfo* videos;
  const float* spill;
  const float* lse;
  float* tok;
  float* frame;
  float* head;
  float* aqf;
  int n_chunks;
  int n_videos;
  int n_tok, hq, tokens_per_frame;
  int total_vis, total_frames;
  int accumulate;
};

// Kernel launchers (defined in the .cu files).
// Intra-frame cue kernel: one CTA per 128-token block of a video's visual rows.
struct IntraFrameLaunch {
  CUtensorMap tm_q, tm_k;           // 3-D maps {d, heads, tokens}, box {64, 1, 128}, 128B swizzle
  const VideoInfo* videos;
  const float* lse;                 // [hq, N] from the probe
  float* aif;                       // [sum T, N_v, N_v]
  int* status;
  int n_videos;
  int total_blocks;                 // 128-row blocks over all videos' visual rows
  int n_tok, hq, hkv, head_dim, tokens_per_frame;
  float scale_log2;                 // softmax_scale * log2(e)
  int accumulate;
};

// One visual row tile of the mask, for the cross-frame reduction.
struct VisRow {
  int32_t q_start;    // global index of the tile's first token
  int32_t q_len;      // rows (<= tile)
  int32_t video;
  int32_t row_tile;   // video-local tile index
  int32_t kv_begin;   // its first kept tile: index into the mask nonzeros (and the KvTile list)
  int32_t kv_count;
  int32_t pad0, pad1;
};
static_assert(sizeof(VisRow) == 32, "VisRow is 32 bytes");

// Kept tiles per row tile up to which the cross-frame pairs kernel also
// writes the zeros of A_ff (beyond it the entry point clears A_ff first).
constexpr int kCrossFrameMaxKept = 1024;

struct CrossFrameLaunch {
  const VisRow* rows;
  const KvTile* kv;
  const VideoInfo* videos;
  const int64_t* aff_off;           // [videos] float offset of each video's (T-1)^2 block
  const float* fspill;              // [hq, nnz, fpt, tile] from the probe (spans of tile / fpt keys)
  const float* lse;                 // [hq, N]
  float* aff;
  float* eff;                       // may be null
  int n_rows, n_videos, max_frames;
  int max_kv;                       // longest kept-tile list of a row tile
  int nnz, fpt, tokens_per_frame, tile;   // fpt: partial spans per tile
  int spans_per_frame;              // N_v / span
  int n_tok, hq;
  int accumulate;
  int* status;                      // device status word (a timed-out wait records EVISEL_ETIMEOUT)
};

// Text-row evidence by recompute (no logit spill): one CTA per (128 visual
// keys, KV group).
struct TextEvidenceLaunch {
  CUtensorMap tm_q, tm_k;           // 3-D maps {d, heads, tokens}, box {64, 1, 128}, 128B swizzle
  const EvChunk* chunks;
  const VideoInfo* videos;
  const float* lse;                 // [hq, N]
  float* tok;                       // [hq, total_vis]
  float* frame;                     // [hq, total_frames]
  int* status;
  int n_chunks, n_tok, hq, hkv, head_dim, tokens_per_frame, total_vis, total_frames;
  float scale_log2;
  int accumulate;
};

// Top-p block retention (mask builder).
struct ToppVideo {
  int32_t start;      // global index of the video's first token
  int32_t n_vis, n_text;
  int32_t blk_off;    // global index of its first block (k_bar rows)
  int32_t row_tile0;  // global index of its first visual row tile of the attention's tiling
  int32_t pad0, pad1, pad2;
};
static_assert(sizeof(ToppVideo) == 32, "ToppVideo is 32 bytes");

struct ToppRowTile {  // 128 rows of one video (visual rows, or text rows)
  int32_t video;
  int32_t q_start;    // global index of the first row
  int32_t q_len;
  int32_t local0;     // video-local position of the first row
  int32_t text;       // 1: text rows
  int32_t pad0, pad1, pad2;
};
static_assert(sizeof(ToppRowTile) == 32, "ToppRowTile is 32 bytes");

struct ToppLaunch {
  CUtensorMap tm_q, tm_kbar;        // q {d, hq, N}; k_bar {d, hkv, blocks}; boxes {64, 1, 128}
  const void* k;                    // bf16 [N, hkv, d]
  void* kbar;                       // bf16 [blocks, hkv, d]
  const ToppVideo* vids;
  const ToppRowTile* tiles;
  uint32_t* keep;                   // [hq, n_words, N]
  uint32_t* tile_union;             // [visual row tiles, n_tile_words] or null
  int* status;
  int n_videos, n_tiles, n_blocks_total, n_words, n_tile_words;
  int n_tok, hq, hkv, head_dim, block, tile;
  float scale_log2, tau;
};

cudaError_t launch_intra_frame(const IntraFrameLaunch& L, cudaStream_t stream);
cudaError_t launch_text_evidence(const TextEvidenceLaunch& L, cudaStream_t stream);
cudaError_t launch_topp(const ToppLaunch& L, cudaStream_t stream);

// Evidence from the coarse token-level map (Eq. 10-11), on the builder's k_bar and keep bits.
struct CoarseLaunch {
  const void* q;                    // bf16 [N, hq, d]
  const void* k;                    // bf16 [N, hkv, d]
  const void* kbar;                 // bf16 [blocks, hkv, d] (from the builder)
  const ToppVideo* vids;
  const int* text_off;              // [videos + 1] first text row of each video (text rows back to back)
  const int* vis_off;               // [videos + 1] column offsets of the token map
  const int* frame_off;             // [videos + 1] column offsets of the frame map
  const uint32_t* keep;             // [hq, n_words, N]
  float* gbuf;                      // [hq, total_text, pitch] block affinities of the text rows
  float* row_m;                     // [hq, total_text]
  float* row_z;                     // [hq, total_text]
  float* tok;
  float* frame;
  float* head;
  float* aqf;
  int n_videos, total_text, pitch, n_words, n_tok, hq, hkv, head_dim, block, tokens_per_frame;
  int total_vis, total_frames, max_frames, accumulate;
  float scale;
};

cudaError_t launch_coarse(const CoarseLaunch& L, cudaStream_t stream);
cudaError_t launch_cross_frame(const CrossFrameLaunch& L, cudaStream_t stream);
cudaError_t launch_probe_attn(const ProbeLaunch& L, cudaStream_t stream);
cudaError_t launch_attn_combine(const CombineLaunch& L, cudaStream_t stream);
cudaError_t launch_evidence(const EvidenceLaunch& L, cudaStream_t stream);

// Host helpers defined in evisel_capi.cpp.
int encode_tensor_map(CUtensorMap* map, const void* base, int n_tok, int heads, int d, int rows);
int set_last_error(int code, const char* msg);
void clear_last_error();

// A kernel's dynamic shared-memory limit is an attribute of the current
// device: raise it once per device (ordinals below 64; others every launch),
// under a lock so that concurrent first launches on one device agree.
struct PerDeviceAttr {
  std::atomic<uint64_t> done{0};
  std::mutex mu;
};

inline cudaError_t raise_smem_limit(PerDeviceAttr& once, const void* kern, int bytes) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const uint64_t bit = dev < 64 ? (1ull << dev) : 0ull;
  if (bit && (once.done.load(std::memory_order_acquire) & bit)) return cudaSuccess;
  std::lock_guard<std::mutex> lock(once.mu);
  if (bit && (once.done.load(std::memory_order_relaxed) & bit)) return cudaSuccess;
  e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess && bit) once.done.fetch_or(bit, std::memory_order_release);
  return e;
}

// Bounded waits give up after this many nanoseconds of %globaltimer.
constexpr uint64_t kWaitTimeoutNs = 2000000000ull;

constexpr int kStatusTimeout = -6;   // == EVISEL_ETIMEOUT
constexpr int kStatusBounds = -7;    // == EVISEL_EBOUNDS

}  // namespace evisel
