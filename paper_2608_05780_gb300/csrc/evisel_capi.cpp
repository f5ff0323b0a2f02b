// Host side of the C ABI: argument and mask validation, work planning (one
// item per query row tile x head block x kv range, longest first), the
// workspace arena, TMA descriptor encoding and kernel launches.
#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <string>
#include <vector>

#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>
#include <nvtx3/nvToolsExt.h>

#include "../../include/evisel.h"
#include "evisel_internal.h"
#include "evisel_plan.h"

using namespace evisel;

namespace {

// An NVTX range named after the entry point around each compute call, so that
// profilers can attribute and filter the kernels by call (header-only NVTX v3:
// a no-op unless a tool is attached).
struct NvtxRange {
  explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};

thread_local std::string g_last_error;

int fail(int code, const std::string& msg) {
  g_last_error = msg;
  return code;
}

int cuda_fail(cudaError_t e, const char* what) {
  return fail(EVISEL_ECUDA, std::string(what) + ": " + cudaGetErrorString(e));
}

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

// 3-D bf16 tensor [tokens, heads, d] viewed as {d, heads, tokens}; box {64, 1, rows}.
int encode_map(CUtensorMap* map, const void* base, int n_tok, int heads, int d, int rows,
               CUtensorMapL2promotion promotion = CU_TENSOR_MAP_L2_PROMOTION_L2_256B) {
  auto enc = tensor_map_encoder();
  if (!enc) return fail(EVISEL_ECUDA, "cuTensorMapEncodeTiled unavailable from the driver");
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(heads),
                        static_cast<cuuint64_t>(std::max(n_tok, 1))};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(d) * 2, static_cast<cuuint64_t>(heads) * d * 2};
  cuuint32_t box[3] = {64, 1, static_cast<cuuint32_t>(rows)};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, promotion,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(EVISEL_ECUDA, "cuTensorMapEncodeTiled failed: " + std::to_string(r));
  return EVISEL_OK;
}

// Host-side plan of one probe call.
struct Plan {
  std::vector<WorkItem> items;
  std::vector<KvTile> kv;
  std::vector<VideoInfo> videos;
  std::vector<CombineGroup> groups;
  std::vector<EvChunk> chunks;
  int n_parts = 0;
  int64_t spill_floats = 0;
  int total_vis = 0;
  int total_frames = 0;
  int n_tok = 0;
  bool text_recompute = false;      // args->text_evidence: no spill, evidence from q and k
  // cross-frame partials (args->cross_frame)
  bool cross_frame = false;
  std::vector<VisRow> vrows;        // visual row tiles in mask order
  std::vector<int64_t> aff_off;     // per video: float offset of its (T-1)^2 block of A_ff
  int64_t aff_floats = 0;
  int64_t fspill_floats = 0;
  int nnz_vis = 0;                  // kept visual kv tiles (mask nonzeros)
  int max_kv = 0;                   // longest mask row
  int max_frames = 0;
};

int validate(const evisel_probe_args* a) {
  if (!a) return fail(EVISEL_EINVAL, "args is NULL");
  if (a->num_videos < 0) return fail(EVISEL_EINVAL, "num_videos < 0");
  if (a->num_videos > 0 && (!a->cu_seqlens_h || !a->n_vis_h))
    return fail(EVISEL_EINVAL, "cu_seqlens_h / n_vis_h is NULL");
  if (a->head_dim != 64 && a->head_dim != 128)
    return fail(EVISEL_EUNSUPPORTED, "head_dim must be 64 or 128, got " + std::to_string(a->head_dim));
  if (a->tile != 64 && a->tile != 128)
    return fail(EVISEL_EUNSUPPORTED, "tile must be 64 or 128, got " + std::to_string(a->tile));
  if (a->hq < 1 || a->hkv < 1) return fail(EVISEL_EINVAL, "hq and hkv must be >= 1");
  if (a->hq % a->hkv != 0) return fail(EVISEL_EUNSUPPORTED, "hq must be a multiple of hkv");
  const int npf = a->tokens_per_frame;
  if (npf < 4 || npf > a->tile || (npf & (npf - 1)) != 0)
    return fail(EVISEL_EUNSUPPORTED, "tokens_per_frame must be a power of two in [4, tile]");
  if (!(a->softmax_scale >= 0.f) || !std::isfinite(a->softmax_scale))
    return fail(EVISEL_EINVAL, "softmax_scale must be finite and >= 0");
  if (a->cross_frame != 0 && a->cross_frame != 1) return fail(EVISEL_EINVAL, "cross_frame must be 0 or 1");
  if (a->text_evidence != 0 && a->text_evidence != 1) return fail(EVISEL_EINVAL, "text_evidence must be 0 or 1");
  if (a->keep) {
    const int kb = a->keep_block;
    if (kb < 16 || kb > npf || (kb & (kb - 1)) != 0)
      return fail(EVISEL_EUNSUPPORTED, "keep_block must be a power of two in [16, tokens_per_frame]");
    if (a->cross_frame || a->text_evidence)
      return fail(EVISEL_EUNSUPPORTED, "per-row block masks do not combine with cross_frame or text_evidence");
    if (reinterpret_cast<uintptr_t>(a->keep) & 3u) return fail(EVISEL_EINVAL, "keep must be 4-byte aligned");
    int max_blocks = 0;
    for (int b = 0; b < a->num_videos; ++b) {
      const int nv = a->n_vis_h[b], nt = a->cu_seqlens_h[b + 1] - a->cu_seqlens_h[b] - nv;
      max_blocks = std::max(max_blocks, nv / kb + (nt + kb - 1) / kb);
    }
    if (a->keep_words < (max_blocks + 31) / 32) return fail(EVISEL_EINVAL, "keep_words too small for the blocks");
  }
  if (a->cross_frame && npf < 16)
    return fail(EVISEL_EUNSUPPORTED, "cross-frame partials need tokens_per_frame >= 16");
  if (a->num_videos == 0) return EVISEL_OK;
  if (a->cu_seqlens_h[0] != 0) return fail(EVISEL_EINVAL, "cu_seqlens[0] must be 0");
  int64_t rows = 0;
  for (int b = 0; b < a->num_videos; ++b) {
    const int64_t len = static_cast<int64_t>(a->cu_seqlens_h[b + 1]) - a->cu_seqlens_h[b];
    if (len < 0) return fail(EVISEL_EINVAL, "cu_seqlens must be non-decreasing");
    const int nv = a->n_vis_h[b];
    if (nv < 0 || nv > len) return fail(EVISEL_EINVAL, "n_vis[" + std::to_string(b) + "] out of range");
    if (nv % npf != 0) return fail(EVISEL_EINVAL, "n_vis must be a multiple of tokens_per_frame");
    rows += (nv + a->tile - 1) / a->tile;
  }
  const int64_t n_tok = a->cu_seqlens_h[a->num_videos];
  if (n_tok > (int64_t(1) << 30)) return fail(EVISEL_EINVAL, "too many tokens");
  if (n_tok > 0) {
    if (!a->q || !a->k || !a->v || !a->o || !a->lse) return fail(EVISEL_EINVAL, "a device pointer is NULL");
    auto mis = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) != 0; };
    if (mis(a->q) || mis(a->k) || mis(a->v) || mis(a->o) || mis(a->lse))
      return fail(EVISEL_EINVAL, "device pointers must be 16-byte aligned");
  }
  if (rows > 0 && (!a->mask_row_ptr_h || !a->mask_col_idx_h)) return fail(EVISEL_EINVAL, "mask is NULL");
  if (rows > 0) {
    const int32_t* rp = a->mask_row_ptr_h;
    const int32_t* ci = a->mask_col_idx_h;
    if (rp[0] != 0) return fail(EVISEL_EMASK, "mask row_ptr[0] must be 0");
    int64_t r = 0;
    for (int b = 0; b < a->num_videos; ++b) {
      const int n_vt = (a->n_vis_h[b] + a->tile - 1) / a->tile;
      for (int t = 0; t < n_vt; ++t, ++r) {
        const int32_t s = rp[r], e = rp[r + 1];
        if (e <= s) return fail(EVISEL_EMASK, "mask row " + std::to_string(r) + " is empty");
        for (int32_t i = s; i < e; ++i) {
          const int32_t c = ci[i];
          if (c < 0 || c > t)
            return fail(EVISEL_EMASK, "mask row " + std::to_string(r) + " has non-causal or negative tile " +
                                          std::to_string(c));
          if (i > s && c <= ci[i - 1])
            return fail(EVISEL_EMASK, "mask row " + std::to_string(r) + " is not strictly ascending");
        }
        if (ci[e - 1] != t)
          return fail(EVISEL_EMASK, "mask row " + std::to_string(r) + " lacks its diagonal tile");
      }
    }
  }
  return EVISEL_OK;
}

void build_plan(const evisel_probe_args* a, Plan& P) {
  const int T = a->tile;
  const int hq = a->hq, gq = a->hq / a->hkv;
  const int hp = 128 / T;                      // heads per slot
  P.n_tok = a->num_videos ? a->cu_seqlens_h[a->num_videos] : 0;

  // Head blocks: up to kSlots * hp consecutive heads of one KV group.
  std::vector<int> head_blocks;
  for (int g = 0; g < a->hkv; ++g)
    for (int hh = 0; hh < gq; hh += kSlots * hp) head_blocks.push_back(g * gq + hh);

  // Videos.
  int64_t spill = 0;
  int vis_off = 0, frame_off = 0;
  for (int b = 0; b < a->num_videos; ++b) {
    VideoInfo v{};
    v.vis_start = a->cu_seqlens_h[b];
    v.n_vis = a->n_vis_h[b];
    v.n_text = a->cu_seqlens_h[b + 1] - a->cu_seqlens_h[b] - v.n_vis;
    v.text_pitch = (v.n_text + 31) & ~31;
    v.spill_off = spill;
    v.vis_off = vis_off;
    v.frame_off = frame_off;
    if (!a->text_evidence) spill += static_cast<int64_t>(hq) * v.n_vis * v.text_pitch;
    vis_off += v.n_vis;
    frame_off += v.n_vis / a->tokens_per_frame;
    P.videos.push_back(v);
  }
  P.spill_floats = spill;
  P.text_recompute = a->text_evidence != 0;
  P.total_vis = vis_off;
  P.total_frames = frame_off;

  // Visual row tiles: kv lists straight from the mask.
  int max_visual = 1;
  int64_t r = 0;
  std::vector<WorkItem> items;
  for (int b = 0; b < a->num_videos; ++b) {
    const VideoInfo& v = P.videos[b];
    const int n_vt = (v.n_vis + T - 1) / T;
    for (int t = 0; t < n_vt; ++t, ++r) {
      const int kv_begin = static_cast<int>(P.kv.size());
      for (int32_t i = a->mask_row_ptr_h[r]; i < a->mask_row_ptr_h[r + 1]; ++i) {
        const int c = a->mask_col_idx_h[i];
        KvTile k{};
        k.start = v.vis_start + c * T;
        k.len = static_cast<int16_t>(std::min(T, v.n_vis - c * T));
        k.diag = c == t;
        k.visual = 1;
        P.kv.push_back(k);
      }
      const int cnt = static_cast<int>(P.kv.size()) - kv_begin;
      max_visual = std::max(max_visual, cnt);
      if (a->cross_frame) {
        VisRow vr{};
        vr.q_start = v.vis_start + t * T;
        vr.q_len = std::min(T, v.n_vis - t * T);
        vr.video = b;
        vr.row_tile = t;
        vr.kv_begin = kv_begin;
        vr.kv_count = cnt;
        P.vrows.push_back(vr);
        P.max_kv = std::max(P.max_kv, cnt);
      }
      for (int h : head_blocks) {
        WorkItem it{};
        it.q_start = v.vis_start + t * T;
        it.q_len = std::min(T, v.n_vis - t * T);
        it.head = h;
        it.kv_begin = kv_begin;
        it.kv_count = cnt;
        it.part = -1;
        it.video = b;
        it.text_row0 = -1;
        items.push_back(it);
      }
    }
  }

  P.nnz_vis = static_cast<int>(P.kv.size());   // the visual kv lists come first, in mask order
  if (a->cross_frame) {
    P.cross_frame = true;
    const int span = std::min(a->tokens_per_frame, 64);
    P.fspill_floats = static_cast<int64_t>(hq) * P.nnz_vis * (T / span) * T;   // [hq, nnz, T / span, T]
    int64_t off = 0;
    for (int b = 0; b < a->num_videos; ++b) {
      const int64_t tb = P.videos[b].n_vis / a->tokens_per_frame;
      P.aff_off.push_back(off);
      off += tb > 1 ? (tb - 1) * (tb - 1) : 0;
      P.max_frames = std::max<int>(P.max_frames, static_cast<int>(tb));
    }
    P.aff_floats = off;
  }

  // Text row tiles: dense causal over the video, split into kv ranges of
  // text_split_len tiles.
  int64_t work = static_cast<int64_t>(P.kv.size());
  for (int b = 0; b < a->num_videos; ++b) {
    const VideoInfo& v = P.videos[b];
    const int64_t n_vt = (v.n_vis + T - 1) / T, n_tt = (v.n_text + T - 1) / T;
    work += n_tt * n_vt + n_tt * (n_tt + 1) / 2;
  }
  const int split_len = text_split_len(max_visual, work * static_cast<int64_t>(head_blocks.size()));
  for (int b = 0; b < a->num_videos; ++b) {
    const VideoInfo& v = P.videos[b];
    const int n_vt = (v.n_vis + T - 1) / T;
    const int n_tt = (v.n_text + T - 1) / T;
    for (int t = 0; t < n_tt; ++t) {
      const int kv_begin = static_cast<int>(P.kv.size());
      for (int c = 0; c < n_vt; ++c) {
        KvTile k{};
        k.start = v.vis_start + c * T;
        k.len = static_cast<int16_t>(std::min(T, v.n_vis - c * T));
        k.diag = 0;
        k.visual = 1;
        P.kv.push_back(k);
      }
      for (int u = 0; u <= t; ++u) {
        KvTile k{};
        k.start = v.vis_start + v.n_vis + u * T;
        k.len = static_cast<int16_t>(std::min(T, v.n_text - u * T));
        k.diag = u == t;
        k.visual = 0;
        P.kv.push_back(k);
      }
      const int cnt = static_cast<int>(P.kv.size()) - kv_begin;
      const int nsplit = (cnt + split_len - 1) / split_len;
      for (int h : head_blocks) {
        int part0 = -1;
        if (nsplit > 1) {
          // kSlots partial slots per split, interleaved: split k of slot s
          // sits in part0 + k * kSlots + s.
          part0 = P.n_parts;
          P.n_parts += kSlots * nsplit;
          for (int slot = 0; slot < kSlots && (h % gq) + slot * hp < gq; ++slot) {
            CombineGroup g{};
            g.q_start = v.vis_start + v.n_vis + t * T;
            g.q_len = std::min(T, v.n_text - t * T);
            g.head = h + slot * hp;
            g.part0 = part0 + slot;
            g.nsplit = nsplit;
            g.stride = kSlots;
            P.groups.push_back(g);
          }
        }
        for (int s = 0; s < nsplit; ++s) {
          // Even split of cnt tiles into nsplit chunks.
          const int lo = static_cast<int>(static_cast<int64_t>(cnt) * s / nsplit);
          const int hi = static_cast<int>(static_cast<int64_t>(cnt) * (s + 1) / nsplit);
          WorkItem it{};
          it.q_start = v.vis_start + v.n_vis + t * T;
          it.q_len = std::min(T, v.n_text - t * T);
          it.head = h;
          it.kv_begin = kv_begin + lo;
          it.kv_count = hi - lo;
          it.part = nsplit > 1 ? part0 + kSlots * s : -1;
          it.video = b;
          it.text_row0 = t * T;
          items.push_back(it);
        }
      }
    }
  }
  // Longest first; stable so that the heads of one row tile stay adjacent and
  // share their K/V tiles through L2. A probe on top-p masks (keep bits) runs
  // over tile unions that cover most of each row's causal history: there the
  // items go KV group by group (longest first within a group), so that the
  // CTAs in flight read one group's K/V (33.5 MB at 65K tokens), which L2
  // holds, instead of all groups' (A/B on 65K tokens: same time, static mask
  // or union; the static masks keep the plain order).
  if (a->keep) {
    std::stable_sort(items.begin(), items.end(), [gq](const WorkItem& x, const WorkItem& y) {
      const int gx = x.head / gq, gy = y.head / gq;
      return gx != gy ? gx < gy : x.kv_count > y.kv_count;
    });
  } else {
    std::stable_sort(items.begin(), items.end(),
                     [](const WorkItem& x, const WorkItem& y) { return x.kv_count > y.kv_count; });
  }
  P.items = std::move(items);

  // Evidence column chunks.
  for (int b = 0; b < a->num_videos; ++b)
    for (int c = 0; c < P.videos[b].n_vis; c += 128) P.chunks.push_back(EvChunk{b, c});
}

}  // namespace

// Helpers shared with the other host entry points of the library.
namespace evisel {
int validate_probe_args(const evisel_probe_args* a) { return validate(a); }
int encode_tensor_map(CUtensorMap* map, const void* base, int n_tok, int heads, int d, int rows) {
  return encode_map(map, base, n_tok, heads, d, rows);
}
int set_last_error(int code, const char* msg) { return fail(code, msg); }
void clear_last_error() { g_last_error.clear(); }
}  // namespace evisel

struct evisel_ws {
  int device = -1;
  // device arena
  void* arena = nullptr;
  size_t arena_bytes = 0;
  int* status = nullptr;
  // pinned staging of the plan metadata
  void* stage = nullptr;
  size_t stage_bytes = 0;
  cudaEvent_t stage_done = nullptr;
  // current plan
  std::vector<int32_t> key;
  bool have_plan = false;
  Plan plan;
  WorkItem* d_items = nullptr;
  KvTile* d_kv = nullptr;
  VideoInfo* d_videos = nullptr;
  CombineGroup* d_groups = nullptr;
  EvChunk* d_chunks = nullptr;
  float* d_part_o = nullptr;
  float2* d_part_ml = nullptr;
  float* d_spill = nullptr;
  VisRow* d_vrows = nullptr;
  int64_t* d_aff_off = nullptr;
  float* d_fspill = nullptr;
  // last probe, for the evidence pass
  bool probed = false;
  const float* lse = nullptr;
  bool probe_keep = false;          // the last probe ran with per-row block masks
  const void* q = nullptr;          // the probe's q and k (read by the recompute evidence)
  const void* k = nullptr;
  int hkv = 0, head_dim = 0;
  float scale = 0.f;
  int hq = 0;
  int tokens_per_frame = 0;
  cudaStream_t last_stream = nullptr;
  // top-p mask builder: [videos | row tiles | k_bar] on the device, staged through pinned memory
  void* topp_buf = nullptr;
  size_t topp_bytes = 0;
  void* topp_stage = nullptr;
  size_t topp_stage_bytes = 0;
  cudaEvent_t topp_done = nullptr;
  int topp_block = 0;               // the last evisel_topp_mask on this workspace
  int topp_n_videos = 0, topp_n_words = 0, topp_n_tok = 0;
  size_t topp_kbar_off = 0;
  // coarse map scratch: offsets, block affinities and row normalisers of the text rows
  void* coarse_buf = nullptr;
  size_t coarse_bytes = 0;
};

namespace {

std::vector<int32_t> plan_key(const evisel_probe_args* a) {
  std::vector<int32_t> k = {a->num_videos, a->tokens_per_frame, a->hq, a->hkv, a->head_dim, a->tile, a->cross_frame,
                            a->text_evidence, a->keep != nullptr};   // the item order differs with keep bits
  for (int b = 0; b <= a->num_videos && a->num_videos > 0; ++b) k.push_back(a->cu_seqlens_h[b]);
  for (int b = 0; b < a->num_videos; ++b) k.push_back(a->n_vis_h[b]);
  int64_t rows = 0;
  for (int b = 0; b < a->num_videos; ++b) rows += (a->n_vis_h[b] + a->tile - 1) / a->tile;
  if (rows > 0) {
    k.insert(k.end(), a->mask_row_ptr_h, a->mask_row_ptr_h + rows + 1);
    k.insert(k.end(), a->mask_col_idx_h, a->mask_col_idx_h + a->mask_row_ptr_h[rows]);
  }
  return k;
}

template <typename T>
size_t bytes_of(const std::vector<T>& v) { return v.size() * sizeof(T); }

// Lays out the arena and uploads the plan metadata on `stream`.
int install_plan(evisel_ws* ws, cudaStream_t stream) {
  const Plan& P = ws->plan;
  const int d = 128;   // partial rows are sized for the largest head_dim
  size_t off = 0;
  auto take = [&](size_t bytes) { size_t o = off; off = align_up(off + bytes, 256); return o; };
  const size_t o_items = take(bytes_of(P.items));
  const size_t o_kv = take(bytes_of(P.kv));
  const size_t o_videos = take(bytes_of(P.videos));
  const size_t o_groups = take(bytes_of(P.groups));
  const size_t o_chunks = take(bytes_of(P.chunks));
  const size_t o_vrows = take(bytes_of(P.vrows));
  const size_t o_aff_off = take(bytes_of(P.aff_off));
  const size_t meta_bytes = off;
  const size_t o_part_o = take(static_cast<size_t>(P.n_parts) * 128 * d * sizeof(float));
  const size_t o_part_ml = take(static_cast<size_t>(P.n_parts) * 128 * sizeof(float2));
  const size_t o_spill = take(static_cast<size_t>(P.spill_floats) * sizeof(float));
  const size_t o_fspill = take(static_cast<size_t>(P.fspill_floats) * sizeof(float));
  const size_t total = std::max<size_t>(off, 256);

  if (total > ws->arena_bytes) {
    if (ws->arena) {
      cudaError_t e = cudaStreamSynchronize(stream);
      if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
      cudaFree(ws->arena);
      ws->arena = nullptr;
      ws->arena_bytes = 0;
    }
    cudaError_t e = cudaMalloc(&ws->arena, total);
    if (e != cudaSuccess) {
      cudaGetLastError();
      return fail(EVISEL_ENOMEM, "workspace allocation of " + std::to_string(total) + " bytes failed");
    }
    ws->arena_bytes = total;
  }
  if (meta_bytes > ws->stage_bytes) {
    if (ws->stage) {
      cudaEventSynchronize(ws->stage_done);
      cudaFreeHost(ws->stage);
      ws->stage = nullptr;
    }
    if (cudaMallocHost(&ws->stage, meta_bytes) != cudaSuccess) {
      cudaGetLastError();
      ws->stage_bytes = 0;
      return fail(EVISEL_ENOMEM, "pinned staging allocation failed");
    }
    ws->stage_bytes = meta_bytes;
  }
  // The staging buffer may still feed the previous upload.
  cudaEventSynchronize(ws->stage_done);
  char* h = static_cast<char*>(ws->stage);
  if (!P.items.empty()) std::memcpy(h + o_items, P.items.data(), bytes_of(P.items));
  if (!P.kv.empty()) std::memcpy(h + o_kv, P.kv.data(), bytes_of(P.kv));
  if (!P.videos.empty()) std::memcpy(h + o_videos, P.videos.data(), bytes_of(P.videos));
  if (!P.groups.empty()) std::memcpy(h + o_groups, P.groups.data(), bytes_of(P.groups));
  if (!P.chunks.empty()) std::memcpy(h + o_chunks, P.chunks.data(), bytes_of(P.chunks));
  if (!P.vrows.empty()) std::memcpy(h + o_vrows, P.vrows.data(), bytes_of(P.vrows));
  if (!P.aff_off.empty()) std::memcpy(h + o_aff_off, P.aff_off.data(), bytes_of(P.aff_off));
  char* base = static_cast<char*>(ws->arena);
  if (meta_bytes > 0) {
    cudaError_t e = cudaMemcpyAsync(base, h, meta_bytes, cudaMemcpyHostToDevice, stream);
    if (e != cudaSuccess) return cuda_fail(e, "plan upload");
    e = cudaEventRecord(ws->stage_done, stream);
    if (e != cudaSuccess) return cuda_fail(e, "cudaEventRecord");
  }
  ws->d_items = reinterpret_cast<WorkItem*>(base + o_items);
  ws->d_kv = reinterpret_cast<KvTile*>(base + o_kv);
  ws->d_videos = reinterpret_cast<VideoInfo*>(base + o_videos);
  ws->d_groups = reinterpret_cast<CombineGroup*>(base + o_groups);
  ws->d_chunks = reinterpret_cast<EvChunk*>(base + o_chunks);
  ws->d_part_o = reinterpret_cast<float*>(base + o_part_o);
  ws->d_part_ml = reinterpret_cast<float2*>(base + o_part_ml);
  ws->d_spill = reinterpret_cast<float*>(base + o_spill);
  ws->d_vrows = reinterpret_cast<VisRow*>(base + o_vrows);
  ws->d_aff_off = reinterpret_cast<int64_t*>(base + o_aff_off);
  ws->d_fspill = reinterpret_cast<float*>(base + o_fspill);
  return EVISEL_OK;
}

int create_ws(evisel_ws** out) {
  evisel_ws* ws = new evisel_ws();
  cudaError_t e = cudaGetDevice(&ws->device);
  if (e == cudaSuccess) e = cudaMalloc(&ws->status, sizeof(int));
  if (e == cudaSuccess) e = cudaMemset(ws->status, 0, sizeof(int));
  if (e == cudaSuccess) e = cudaEventCreateWithFlags(&ws->stage_done, cudaEventDisableTiming);
  if (e != cudaSuccess) {
    cudaGetLastError();
    if (ws->status) cudaFree(ws->status);
    delete ws;
    return cuda_fail(e, "workspace creation");
  }
  *out = ws;
  return EVISEL_OK;
}

}  // namespace

extern "C" {

int evisel_probe_attention(const evisel_probe_args* args, void* stream_ptr, evisel_ws** ws_inout) {
  const NvtxRange nvtx_range("evisel_probe_attention");
  g_last_error.clear();
  if (!ws_inout) return fail(EVISEL_EINVAL, "ws_inout is NULL");
  int rc = validate(args);
  if (rc != EVISEL_OK) return rc;
  cudaStream_t stream = static_cast<cudaStream_t>(stream_ptr);
  if (!*ws_inout) {
    rc = create_ws(ws_inout);
    if (rc != EVISEL_OK) return rc;
  }
  evisel_ws* ws = *ws_inout;
  int dev = -1;
  cudaGetDevice(&dev);
  if (dev != ws->device) return fail(EVISEL_EINVAL, "workspace belongs to another device");

  std::vector<int32_t> key = plan_key(args);
  if (!ws->have_plan || key != ws->key) {
    ws->plan = Plan();
    build_plan(args, ws->plan);
    ws->have_plan = false;
    rc = install_plan(ws, stream);
    if (rc != EVISEL_OK) return rc;
    ws->key.swap(key);
    ws->have_plan = true;
  }
  if (ws->last_stream != stream) {
    // The plan metadata may have been uploaded on another stream.
    cudaError_t e = cudaStreamWaitEvent(stream, ws->stage_done, 0);
    if (e != cudaSuccess) return cuda_fail(e, "cudaStreamWaitEvent");
  }
  const Plan& P = ws->plan;
  const float scale = args->softmax_scale > 0.f ? args->softmax_scale : 1.0f / std::sqrt(float(args->head_dim));

  if (!P.items.empty()) {
    ProbeLaunch L;
    std::memset(&L, 0, sizeof(L));
    rc = encode_map(&L.tm_q, args->q, P.n_tok, args->hq, args->head_dim, args->tile);
    if (rc == EVISEL_OK) rc = encode_map(&L.tm_k, args->k, P.n_tok, args->hkv, args->head_dim, args->tile);
    if (rc == EVISEL_OK) rc = encode_map(&L.tm_v, args->v, P.n_tok, args->hkv, args->head_dim, args->tile);
    if (rc == EVISEL_OK) rc = encode_map(&L.tm_o, args->o, P.n_tok, args->hq, args->head_dim, args->tile);
    if (rc != EVISEL_OK) return rc;
    L.items = ws->d_items;
    L.kv = ws->d_kv;
    L.videos = ws->d_videos;
    L.o = args->o;
    L.lse = args->lse;
    L.spill = P.text_recompute ? nullptr : ws->d_spill;
    L.part_o = ws->d_part_o;
    L.part_ml = ws->d_part_ml;
    L.status = ws->status;
    L.n_items = static_cast<int>(P.items.size());
    L.n_tok = P.n_tok;
    L.hq = args->hq;
    L.hkv = args->hkv;
    L.head_dim = args->head_dim;
    L.tile = args->tile;
    L.scale = scale;
    L.scale_log2 = scale * 1.4426950408889634f;
    if (args->keep) {
      L.keep = args->keep;
      L.keep_words = args->keep_words;
      L.keep_block = args->keep_block;
    }
    if (P.cross_frame && P.nnz_vis > 0) {
      L.fspill = ws->d_fspill;
      L.fs_nnz = P.nnz_vis;
      L.fs_span = std::min(args->tokens_per_frame, 64);
    }
    cudaError_t e = launch_probe_attn(L, stream);
    if (e != cudaSuccess) return cuda_fail(e, "probe_attn launch");
    if (!P.groups.empty()) {
      CombineLaunch C{};
      C.groups = ws->d_groups;
      C.part_o = ws->d_part_o;
      C.part_ml = ws->d_part_ml;
      C.o = args->o;
      C.lse = args->lse;
      C.n_groups = static_cast<int>(P.groups.size());
      C.n_tok = P.n_tok;
      C.hq = args->hq;
      C.hkv = args->hkv;
      C.head_dim = args->head_dim;
      C.tile = args->tile;
      e = launch_attn_combine(C, stream);
      if (e != cudaSuccess) return cuda_fail(e, "attn_combine launch");
    }
  }
  ws->probed = true;
  ws->probe_keep = args->keep != nullptr;
  ws->lse = args->lse;
  ws->q = args->q;
  ws->k = args->k;
  ws->hkv = args->hkv;
  ws->head_dim = args->head_dim;
  ws->scale = scale;
  ws->hq = args->hq;
  ws->tokens_per_frame = args->tokens_per_frame;
  ws->last_stream = stream;
  return EVISEL_OK;
}

int evisel_evidence_reduce(const evisel_ws* ws_c, float* tok, float* frame, float* head, float* aqf,
                           int accumulate, void* stream_ptr) {
  const NvtxRange nvtx_range("evisel_evidence_reduce");
  g_last_error.clear();
  evisel_ws* ws = const_cast<evisel_ws*>(ws_c);
  if (!ws) return fail(EVISEL_EINVAL, "workspace is NULL");
  if (!ws->probed || !ws->have_plan) return fail(EVISEL_ESTATE, "no probe has run on this workspace");
  const Plan& P = ws->plan;
  if (P.videos.empty()) return EVISEL_OK;
  if ((P.total_vis > 0 && (!tok || !frame)) || !head || (P.total_frames > 0 && !aqf))
    return fail(EVISEL_EINVAL, "an output map is NULL");
  if ((reinterpret_cast<uintptr_t>(tok) & 15u) != 0) return fail(EVISEL_EINVAL, "tok must be 16-byte aligned");
  cudaStream_t stream = static_cast<cudaStream_t>(stream_ptr);
  EvidenceLaunch L{};
  L.chunks = ws->d_chunks;
  L.videos = ws->d_videos;
  L.spill = ws->d_spill;
  L.lse = ws->lse;
  L.tok = tok;
  L.frame = frame;
  L.head = head;
  L.aqf = aqf;
  L.n_chunks = static_cast<int>(P.chunks.size());
  L.n_videos = static_cast<int>(P.videos.size());
  L.n_tok = P.n_tok;
  L.hq = ws->hq;
  L.tokens_per_frame = ws->tokens_per_frame;
  L.total_vis = P.total_vis;
  L.total_frames = P.total_frames;
  L.accumulate = accumulate != 0;
  if (P.text_recompute) {
    // Token and frame maps from q and k (no spill); the finalize below forms
    // the head map and A_qf from the frame map.
    TextEvidenceLaunch T;
    std::memset(&T, 0, sizeof(T));
    int rc = encode_map(&T.tm_q, ws->q, P.n_tok, ws->hq, ws->head_dim, 128);
    if (rc == EVISEL_OK) rc = encode_map(&T.tm_k, ws->k, P.n_tok, ws->hkv, ws->head_dim, 128);
    if (rc != EVISEL_OK) return rc;
    T.chunks = ws->d_chunks;
    T.videos = ws->d_videos;
    T.lse = ws->lse;
    T.tok = tok;
    T.frame = frame;
    T.status = ws->status;
    T.n_chunks = static_cast<int>(P.chunks.size());
    T.n_tok = P.n_tok;
    T.hq = ws->hq;
    T.hkv = ws->hkv;
    T.head_dim = ws->head_dim;
    T.tokens_per_frame = ws->tokens_per_frame;
    T.total_vis = P.total_vis;
    T.total_frames = P.total_frames;
    T.scale_log2 = ws->scale * 1.4426950408889634f;
    T.accumulate = accumulate != 0;
    cudaError_t te = launch_text_evidence(T, stream);
    if (te != cudaSuccess) return cuda_fail(te, "text_evidence launch");
    L.n_chunks = 0;
  }
  cudaError_t e = launch_evidence(L, stream);
  if (e != cudaSuccess) return cuda_fail(e, "evidence launch");
  ws->last_stream = stream;
  return EVISEL_OK;
}

int evisel_intra_frame_evidence(const evisel_probe_args* args, const evisel_ws* ws_c, float* aif, int accumulate,
                                void* stream_ptr) {
  const NvtxRange nvtx_range("evisel_intra_frame_evidence");
  g_last_error.clear();
  evisel_ws* ws = const_cast<evisel_ws*>(ws_c);
  if (!ws) return fail(EVISEL_EINVAL, "workspace is NULL");
  int rc = validate(args);
  if (rc != EVISEL_OK) return rc;
  if (!ws->probed || !ws->have_plan) return fail(EVISEL_ESTATE, "no probe has run on this workspace");
  if (ws->probe_keep) return fail(EVISEL_EUNSUPPORTED, "the probe ran with per-row block masks");
  const Plan& P = ws->plan;
  if (static_cast<int>(P.videos.size()) != args->num_videos)
    return fail(EVISEL_EINVAL, "args do not match the probe that ran on this workspace");
  if (P.total_frames > 0 && !aif) return fail(EVISEL_EINVAL, "aif is NULL");
  int total_blocks = 0;
  for (const VideoInfo& v : P.videos) total_blocks += (v.n_vis + 127) / 128;
  if (total_blocks == 0) return EVISEL_OK;
  cudaStream_t stream = static_cast<cudaStream_t>(stream_ptr);
  IntraFrameLaunch L;
  std::memset(&L, 0, sizeof(L));
  // No L2 promotion: each Q row of a head is read once, by one CTA (measured
  // faster than 256-byte promotion for this pass).
  rc = encode_map(&L.tm_q, args->q, P.n_tok, args->hq, args->head_dim, 128, CU_TENSOR_MAP_L2_PROMOTION_NONE);
  if (rc == EVISEL_OK)
    rc = encode_map(&L.tm_k, args->k, P.n_tok, args->hkv, args->head_dim, 128, CU_TENSOR_MAP_L2_PROMOTION_NONE);
  if (rc != EVISEL_OK) return rc;
  const float scale = args->softmax_scale > 0.f ? args->softmax_scale : 1.0f / std::sqrt(float(args->head_dim));
  L.videos = ws->d_videos;
  L.lse = args->lse;
  L.aif = aif;
  L.status = ws->status;
  L.n_videos = static_cast<int>(P.videos.size());
  L.total_blocks = total_blocks;
  L.n_tok = P.n_tok;
  L.hq = args->hq;
  L.hkv = args->hkv;
  L.head_dim = args->head_dim;
  L.tokens_per_frame = args->tokens_per_frame;
  L.scale_log2 = scale * 1.4426950408889634f;
  L.accumulate = accumulate != 0;
  if (ws->last_stream != stream) {
    cudaError_t e = cudaStreamWaitEvent(stream, ws->stage_done, 0);
    if (e != cudaSuccess) return cuda_fail(e, "cudaStreamWaitEvent");
  }
  cudaError_t e = launch_intra_frame(L, stream);
  if (e != cudaSuccess) return cuda_fail(e, "intra_frame launch");
  ws->last_stream = stream;
  return EVISEL_OK;
}

int evisel_cross_frame_evidence(const evisel_probe_args* args, evisel_ws* ws, float* aff, float* eff,
                                int accumulate, void* stream_ptr) {
  const NvtxRange nvtx_range("evisel_cross_frame_evidence");
  g_last_error.clear();
  if (!ws) return fail(EVISEL_EINVAL, "workspace is NULL");
  int rc = validate(args);
  if (rc != EVISEL_OK) return rc;
  if (!ws->probed || !ws->have_plan) return fail(EVISEL_ESTATE, "no probe has run on this workspace");
  const Plan& P = ws->plan;
  if (!P.cross_frame) return fail(EVISEL_ESTATE, "the probe on this workspace ran without cross_frame");
  if (ws->probe_keep) return fail(EVISEL_EUNSUPPORTED, "the probe ran with per-row block masks");
  if (static_cast<int>(P.videos.size()) != args->num_videos || plan_key(args) != ws->key)
    return fail(EVISEL_EINVAL, "args do not match the probe that ran on this workspace");
  if (P.aff_floats > 0 && !aff) return fail(EVISEL_EINVAL, "aff is NULL");
  cudaStream_t stream = static_cast<cudaStream_t>(stream_ptr);
  if (ws->last_stream != stream) {
    cudaError_t e = cudaStreamWaitEvent(stream, ws->stage_done, 0);
    if (e != cudaSuccess) return cuda_fail(e, "cudaStreamWaitEvent");
  }
  // Without accumulate the pairs kernel writes every entry of A_ff (zeros
  // included) when no row tile keeps more tiles than it stages; else clear first.
  if (!accumulate && P.aff_floats > 0 && P.max_kv > kCrossFrameMaxKept) {
    cudaError_t e = cudaMemsetAsync(aff, 0, static_cast<size_t>(P.aff_floats) * sizeof(float), stream);
    if (e != cudaSuccess) return cuda_fail(e, "A_ff clear");
  }
  CrossFrameLaunch L{};
  L.rows = ws->d_vrows;
  L.kv = ws->d_kv;
  L.videos = ws->d_videos;
  L.aff_off = ws->d_aff_off;
  L.fspill = ws->d_fspill;
  L.lse = args->lse;
  L.aff = aff;
  L.eff = P.total_frames > 0 ? eff : nullptr;
  L.n_rows = P.aff_floats > 0 ? static_cast<int>(P.vrows.size()) : 0;
  L.n_videos = static_cast<int>(P.videos.size());
  L.max_frames = P.max_frames;
  L.max_kv = P.max_kv;
  L.nnz = P.nnz_vis;
  L.fpt = args->tile / std::min(args->tokens_per_frame, 64);
  L.spans_per_frame = args->tokens_per_frame / std::min(args->tokens_per_frame, 64);
  L.tokens_per_frame = args->tokens_per_frame;
  L.tile = args->tile;
  L.n_tok = P.n_tok;
  L.hq = args->hq;
  L.accumulate = accumulate != 0;
  L.status = ws->status;
  cudaError_t e = launch_cross_frame(L, stream);
  if (e != cudaSuccess) return cuda_fail(e, "cross_frame launch");
  ws->last_stream = stream;
  return EVISEL_OK;
}

int evisel_topp_mask(const evisel_probe_args* a, int32_t block, float tau_p, uint32_t* keep, uint32_t* tile_union,
                     void* stream_ptr, evisel_ws** ws_inout) {
  const NvtxRange nvtx_range("evisel_topp_mask");
  g_last_error.clear();
  if (!a) return fail(EVISEL_EINVAL, "args is NULL");
  if (!ws_inout) return fail(EVISEL_EINVAL, "ws_inout is NULL");
  if (a->num_videos < 0 || (a->num_videos > 0 && (!a->cu_seqlens_h || !a->n_vis_h)))
    return fail(EVISEL_EINVAL, "num_videos / cu_seqlens_h / n_vis_h");
  if (a->head_dim != 64 && a->head_dim != 128) return fail(EVISEL_EUNSUPPORTED, "head_dim must be 64 or 128");
  if (a->tile != 64 && a->tile != 128) return fail(EVISEL_EUNSUPPORTED, "tile must be 64 or 128");
  if (a->hq < 1 || a->hkv < 1 || a->hq % a->hkv != 0) return fail(EVISEL_EUNSUPPORTED, "hq must be a multiple of hkv");
  const int npf = a->tokens_per_frame;
  if (npf < 4 || npf > a->tile || (npf & (npf - 1)) != 0)
    return fail(EVISEL_EUNSUPPORTED, "tokens_per_frame must be a power of two in [4, tile]");
  if (block < 16 || block > npf || (block & (block - 1)) != 0)
    return fail(EVISEL_EUNSUPPORTED, "block must be a power of two in [16, tokens_per_frame] (it divides N_v)");
  if (!(tau_p > 0.f && tau_p <= 1.f)) return fail(EVISEL_EINVAL, "tau_p must be in (0, 1]");
  if (!(a->softmax_scale >= 0.f) || !std::isfinite(a->softmax_scale))
    return fail(EVISEL_EINVAL, "softmax_scale must be finite and >= 0");
  if (a->num_videos == 0) return EVISEL_OK;
  if (a->cu_seqlens_h[0] != 0) return fail(EVISEL_EINVAL, "cu_seqlens[0] must be 0");
  for (int b = 0; b < a->num_videos; ++b) {
    const int64_t len = static_cast<int64_t>(a->cu_seqlens_h[b + 1]) - a->cu_seqlens_h[b];
    if (len < 0 || a->n_vis_h[b] < 0 || a->n_vis_h[b] > len || a->n_vis_h[b] % npf != 0)
      return fail(EVISEL_EINVAL, "cu_seqlens / n_vis of video " + std::to_string(b));
  }
  const int n_tok = a->cu_seqlens_h[a->num_videos];
  if (n_tok == 0) return EVISEL_OK;
  if (!a->q || !a->k || !keep) return fail(EVISEL_EINVAL, "q, k or keep is NULL");
  if ((reinterpret_cast<uintptr_t>(a->q) & 15u) || (reinterpret_cast<uintptr_t>(a->k) & 15u))
    return fail(EVISEL_EINVAL, "q and k must be 16-byte aligned");

  // Videos, their blocks and row tiles (128 rows: the visual rows, then the text rows).
  std::vector<ToppVideo> vids;
  std::vector<ToppRowTile> tiles;
  int blk_off = 0, row_tile0 = 0, max_blocks = 0, max_vis_tiles = 0;
  for (int b = 0; b < a->num_videos; ++b) {
    ToppVideo v{};
    v.start = a->cu_seqlens_h[b];
    v.n_vis = a->n_vis_h[b];
    v.n_text = a->cu_seqlens_h[b + 1] - v.start - v.n_vis;
    v.blk_off = blk_off;
    v.row_tile0 = row_tile0;
    const int nb = v.n_vis / block + (v.n_text + block - 1) / block;
    blk_off += nb;
    max_blocks = std::max(max_blocks, nb);
    const int n_vt = (v.n_vis + a->tile - 1) / a->tile;
    row_tile0 += n_vt;
    max_vis_tiles = std::max(max_vis_tiles, n_vt);
    for (int s = 0; s < v.n_vis; s += 128)
      tiles.push_back(ToppRowTile{b, v.start + s, std::min(128, v.n_vis - s), s, 0, 0, 0, 0});
    for (int s = 0; s < v.n_text; s += 128)
      tiles.push_back(ToppRowTile{b, v.start + v.n_vis + s, std::min(128, v.n_text - s), v.n_vis + s, 1, 0, 0, 0});
    vids.push_back(v);
  }
  const int n_words = std::max(1, (max_blocks + 31) / 32);
  const int n_tile_words = std::max(1, (max_vis_tiles + 31) / 32);

  if (!*ws_inout) {
    int rc = create_ws(ws_inout);
    if (rc != EVISEL_OK) return rc;
  }
  evisel_ws* ws = *ws_inout;
  cudaStream_t stream = static_cast<cudaStream_t>(stream_ptr);
  const size_t meta = align_up(vids.size() * sizeof(ToppVideo), 256) + align_up(tiles.size() * sizeof(ToppRowTile), 256);
  const size_t kbar_bytes = static_cast<size_t>(blk_off) * a->hkv * a->head_dim * 2;
  const size_t need = meta + kbar_bytes;
  if (!ws->topp_done && cudaEventCreateWithFlags(&ws->topp_done, cudaEventDisableTiming) != cudaSuccess)
    return cuda_fail(cudaGetLastError(), "event");
  cudaEventSynchronize(ws->topp_done);             // the staging buffer may still feed the last upload
  if (need > ws->topp_bytes) {
    cudaStreamSynchronize(ws->last_stream);
    cudaStreamSynchronize(stream);
    if (ws->topp_buf) cudaFree(ws->topp_buf);
    ws->topp_buf = nullptr;
    ws->topp_bytes = 0;
    if (cudaMalloc(&ws->topp_buf, need) != cudaSuccess) {
      cudaGetLastError();
      return fail(EVISEL_ENOMEM, "top-p scratch of " + std::to_string(need) + " bytes");
    }
    ws->topp_bytes = need;
  }
  if (meta > ws->topp_stage_bytes) {
    if (ws->topp_stage) cudaFreeHost(ws->topp_stage);
    ws->topp_stage = nullptr;
    ws->topp_stage_bytes = 0;
    if (cudaMallocHost(&ws->topp_stage, meta) != cudaSuccess) {
      cudaGetLastError();
      return fail(EVISEL_ENOMEM, "top-p staging");
    }
    ws->topp_stage_bytes = meta;
  }
  char* h = static_cast<char*>(ws->topp_stage);
  const size_t o_tiles = align_up(vids.size() * sizeof(ToppVideo), 256);
  std::memcpy(h, vids.data(), vids.size() * sizeof(ToppVideo));
  std::memcpy(h + o_tiles, tiles.data(), tiles.size() * sizeof(ToppRowTile));
  char* d = static_cast<char*>(ws->topp_buf);
  cudaError_t e = cudaMemcpyAsync(d, h, meta, cudaMemcpyHostToDevice, stream);
  if (e == cudaSuccess) e = cudaEventRecord(ws->topp_done, stream);
  if (e == cudaSuccess)
    e = cudaMemsetAsync(keep, 0, static_cast<size_t>(a->hq) * n_words * n_tok * sizeof(uint32_t), stream);
  const int r_vis = row_tile0;
  if (e == cudaSuccess && tile_union && r_vis > 0)
    e = cudaMemsetAsync(tile_union, 0, static_cast<size_t>(r_vis) * n_tile_words * sizeof(uint32_t), stream);
  if (e != cudaSuccess) return cuda_fail(e, "top-p upload");

  ToppLaunch L;
  std::memset(&L, 0, sizeof(L));
  int rc = encode_map(&L.tm_q, a->q, n_tok, a->hq, a->head_dim, 128);
  if (rc == EVISEL_OK && blk_off > 0) rc = encode_map(&L.tm_kbar, d + meta, blk_off, a->hkv, a->head_dim, 128);
  if (rc != EVISEL_OK) return rc;
  const float scale = a->softmax_scale > 0.f ? a->softmax_scale : 1.0f / std::sqrt(float(a->head_dim));
  L.k = a->k;
  L.kbar = d + meta;
  L.vids = reinterpret_cast<const ToppVideo*>(d);
  L.tiles = reinterpret_cast<const ToppRowTile*>(d + o_tiles);
  L.keep = keep;
  L.tile_union = tile_union;
  L.status = ws->status;
  L.n_videos = a->num_videos;
  L.n_tiles = static_cast<int>(tiles.size());
  L.n_blocks_total = blk_off;
  L.n_words = n_words;
  L.n_tile_words = n_tile_words;
  L.n_tok = n_tok;
  L.hq = a->hq;
  L.hkv = a->hkv;
  L.head_dim = a->head_dim;
  L.block = block;
  L.tile = a->tile;
  L.scale_log2 = scale * 1.4426950408889634f;
  L.tau = tau_p;
  e = launch_topp(L, stream);
  if (e != cudaSuccess) return cuda_fail(e, "top-p launch");
  ws->last_stream = stream;
  ws->topp_block = block;
  ws->topp_n_videos = a->num_videos;
  ws->topp_n_words = n_words;
  ws->topp_n_tok = n_tok;
  ws->topp_kbar_off = meta;
  return EVISEL_OK;
}

int evisel_coarse_evidence(const evisel_probe_args* a, evisel_ws* ws, int32_t block, const uint32_t* keep, float* tok,
                           float* frame, float* head, float* aqf, int accumulate, void* stream_ptr) {
  const NvtxRange nvtx_range("evisel_coarse_evidence");
  g_last_error.clear();
  if (!a || !ws) return fail(EVISEL_EINVAL, "args or workspace is NULL");
  if (ws->topp_block == 0) return fail(EVISEL_ESTATE, "no evisel_topp_mask has run on this workspace");
  if (block != ws->topp_block || a->num_videos != ws->topp_n_videos ||
      (a->num_videos > 0 && a->cu_seqlens_h[a->num_videos] != ws->topp_n_tok))
    return fail(EVISEL_EINVAL, "args / block do not match the evisel_topp_mask call on this workspace");
  if (a->num_videos == 0) return EVISEL_OK;
  const int npf = a->tokens_per_frame;
  std::vector<int> text_off(1, 0), vis_off(1, 0), frame_off(1, 0);
  int max_frames = 0;
  for (int b = 0; b < a->num_videos; ++b) {
    const int nv = a->n_vis_h[b], nt = a->cu_seqlens_h[b + 1] - a->cu_seqlens_h[b] - nv;
    text_off.push_back(text_off.back() + nt);
    vis_off.push_back(vis_off.back() + nv);
    frame_off.push_back(frame_off.back() + nv / npf);
    max_frames = std::max(max_frames, nv / npf);
  }
  const int total_text = text_off.back();
  if ((vis_off.back() > 0 && (!tok || !frame)) || !head || (frame_off.back() > 0 && !aqf) || !keep || !a->q || !a->k)
    return fail(EVISEL_EINVAL, "an output map, keep, q or k is NULL");
  const int pitch = ws->topp_n_words * 32;
  const size_t ints = align_up(3 * (a->num_videos + 1) * sizeof(int), 256);
  const size_t gbytes = align_up(static_cast<size_t>(a->hq) * total_text * pitch * sizeof(float), 256);
  const size_t mz = align_up(static_cast<size_t>(a->hq) * total_text * sizeof(float), 256);
  const size_t need = ints + gbytes + 2 * mz;
  cudaStream_t stream = static_cast<cudaStream_t>(stream_ptr);
  if (need > ws->coarse_bytes) {
    cudaStreamSynchronize(ws->last_stream);
    cudaStreamSynchronize(stream);
    if (ws->coarse_buf) cudaFree(ws->coarse_buf);
    ws->coarse_buf = nullptr;
    ws->coarse_bytes = 0;
    if (cudaMalloc(&ws->coarse_buf, need) != cudaSuccess) {
      cudaGetLastError();
      return fail(EVISEL_ENOMEM, "coarse-map scratch of " + std::to_string(need) + " bytes");
    }
    ws->coarse_bytes = need;
  }
  std::vector<int> offs;
  offs.insert(offs.end(), text_off.begin(), text_off.end());
  offs.insert(offs.end(), vis_off.begin(), vis_off.end());
  offs.insert(offs.end(), frame_off.begin(), frame_off.end());
  char* d = static_cast<char*>(ws->coarse_buf);
  cudaError_t e = cudaMemcpyAsync(d, offs.data(), offs.size() * sizeof(int), cudaMemcpyHostToDevice, stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(stream);   // the host vector goes out of scope
  if (e != cudaSuccess) return cuda_fail(e, "coarse-map offsets");
  CoarseLaunch L{};
  L.q = a->q;
  L.k = a->k;
  L.kbar = static_cast<char*>(ws->topp_buf) + ws->topp_kbar_off;
  L.vids = static_cast<const ToppVideo*>(ws->topp_buf);
  L.text_off = reinterpret_cast<const int*>(d);
  L.vis_off = L.text_off + (a->num_videos + 1);
  L.frame_off = L.vis_off + (a->num_videos + 1);
  L.keep = keep;
  L.gbuf = reinterpret_cast<float*>(d + ints);
  L.row_m = reinterpret_cast<float*>(d + ints + gbytes);
  L.row_z = reinterpret_cast<float*>(d + ints + gbytes + mz);
  L.tok = tok;
  L.frame = frame;
  L.head = head;
  L.aqf = aqf;
  L.n_videos = a->num_videos;
  L.total_text = total_text;
  L.pitch = pitch;
  L.n_words = ws->topp_n_words;
  L.n_tok = ws->topp_n_tok;
  L.hq = a->hq;
  L.hkv = a->hkv;
  L.head_dim = a->head_dim;
  L.block = block;
  L.tokens_per_frame = npf;
  L.total_vis = vis_off.back();
  L.total_frames = frame_off.back();
  L.max_frames = max_frames;
  L.accumulate = accumulate != 0;
  L.scale = a->softmax_scale > 0.f ? a->softmax_scale : 1.0f / std::sqrt(float(a->head_dim));
  e = launch_coarse(L, stream);
  if (e != cudaSuccess) return cuda_fail(e, "coarse-map launch");
  ws->last_stream = stream;
  return EVISEL_OK;
}

void evisel_free(evisel_ws* ws) {
  if (!ws) return;
  int prev = -1;
  cudaGetDevice(&prev);
  if (ws->device >= 0 && prev != ws->device) cudaSetDevice(ws->device);
  cudaStreamSynchronize(ws->last_stream);
  if (ws->stage_done) cudaEventSynchronize(ws->stage_done);
  if (ws->arena) cudaFree(ws->arena);
  if (ws->status) cudaFree(ws->status);
  if (ws->stage) cudaFreeHost(ws->stage);
  if (ws->stage_done) cudaEventDestroy(ws->stage_done);
  if (ws->topp_done) cudaEventSynchronize(ws->topp_done);
  if (ws->topp_buf) cudaFree(ws->topp_buf);
  if (ws->coarse_buf) cudaFree(ws->coarse_buf);
  if (ws->topp_stage) cudaFreeHost(ws->topp_stage);
  if (ws->topp_done) cudaEventDestroy(ws->topp_done);
  if (prev >= 0 && prev != ws->device) cudaSetDevice(prev);
  cudaGetLastError();
  delete ws;
}

int evisel_status(evisel_ws* ws) {
  g_last_error.clear();
  if (!ws) return fail(EVISEL_EINVAL, "workspace is NULL");
  cudaError_t e = cudaStreamSynchronize(ws->last_stream);
  if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
  int st = 0;
  e = cudaMemcpy(&st, ws->status, sizeof(int), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(e, "status read");
  if (st != 0) {
    const int zero = 0;
    cudaMemcpy(ws->status, &zero, sizeof(int), cudaMemcpyHostToDevice);
  }
  return st;
}

const char* evisel_strerror(int code) {
  switch (code) {
    case EVISEL_OK: return "success";
    case EVISEL_EINVAL: return "invalid argument";
    case EVISEL_EUNSUPPORTED: return "unsupported shape or parameter";
    case EVISEL_EMASK: return "invalid block mask";
    case EVISEL_ECUDA: return "CUDA error";
    case EVISEL_ENOMEM: return "out of memory";
    case EVISEL_ETIMEOUT: return "device wait timed out";
    case EVISEL_EBOUNDS: return "device index check failed";
    case EVISEL_ESTATE: return "no probe has run on this workspace";
    default: return "unknown status";
  }
}

const char* evisel_last_error(void) { return g_last_error.c_str(); }

#ifndef EVISEL_BUILD_ID
#define EVISEL_BUILD_ID "unversioned"
#endif
// The prefix lets the build script find the id in the binary without loading it.
static const char kBuildIdString[] = "evisel-build-id:" EVISEL_BUILD_ID;

const char* evisel_build_id(void) { return kBuildIdString + sizeof("evisel-build-id:") - 1; }

int64_t evisel_workspace_bytes(const evisel_ws* ws) {
  return ws ? static_cast<int64_t>(ws->arena_bytes) : 0;
}

}  // extern "C"
