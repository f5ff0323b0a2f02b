// evisel_probe_evidence_noalloc: the probe attention and the evidence pass in
// one call that allocates nothing.
//
// Some callers cannot call cudaMalloc: inference servers that hand out all
// device memory up front from their own pool, real-time serving paths where an
// allocation (or the device-wide synchronisation of cudaFree) is not acceptable,
// or hosts that forbid a library any allocator use of its own. For them this
// entry point keeps all of its scratch -- the work
// plan, the split-KV partials of the text rows and the text-row logit spill --
// in one file-scope device array of fixed size (kScratchBytes), and its host
// staging in one file-scope host array. The caller still passes Q/K/V, the mask
// and every output (O, LSE and the four evidence maps).
//
// The first call on a device looks up the array's device address with
// cudaGetSymbolAddress (with that device current) and caches it; later calls on
// that device reuse it. Every call shares the array, which keeps the previous
// call's contents; calls that overlap on the GPU (two streams, or two host
// threads without ordering) race on it.
#include <algorithm>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <mutex>
#include <string>

#include <cuda_runtime.h>
#include <nvtx3/nvToolsExt.h>

#include "../../include/evisel.h"
#include "evisel_internal.h"
#include "evisel_plan.h"

namespace evisel {
int validate_probe_args(const evisel_probe_args* a);
}

// The device scratch: status word, plan, partials, spill. Held by every GPU
// that loads this library until the process exits.
static __device__ __align__(256) unsigned char g_scratch[static_cast<size_t>(EVISEL_NOALLOC_SCRATCH_BYTES)];

using namespace evisel;

namespace {

constexpr size_t kScratchBytes = static_cast<size_t>(EVISEL_NOALLOC_SCRATCH_BYTES);
constexpr size_t kStageBytes = size_t(4) << 20;     // largest plan (work list, kv lists, tables)
constexpr int kMaxDevices = 64;

alignas(256) unsigned char g_stage[kStageBytes];    // host staging of the plan
std::mutex g_mutex;
void* g_scratch_ptr[kMaxDevices] = {};

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

struct Counts {
  size_t items = 0, kv = 0, groups = 0, chunks = 0;
  int64_t parts = 0;
  int64_t spill_floats = 0;
  int total_vis = 0, total_frames = 0;
};

struct Out {
  WorkItem* items;
  KvTile* kv;
  VideoInfo* videos;
  CombineGroup* groups;
  EvChunk* chunks;
};

// Work plan: one item per (query row tile, block of heads of one KV group, kv
// range); text row tiles are split into kv ranges of text_split_len tiles, as
// in the allocating entry point. Counts only when `o` is null.
void make_plan(const evisel_probe_args* a, Counts& c, const Out* o) {
  const int T = a->tile, hq = a->hq, gq = a->hq / a->hkv, hp = 128 / T;
  const int nb = a->num_videos;
  c = Counts();
  int64_t spill = 0;
  int vis_off = 0, frame_off = 0;
  auto info = [&](int b) {
    VideoInfo v{};
    v.vis_start = a->cu_seqlens_h[b];
    v.n_vis = a->n_vis_h[b];
    v.n_text = a->cu_seqlens_h[b + 1] - a->cu_seqlens_h[b] - v.n_vis;
    v.text_pitch = (v.n_text + 31) & ~31;
    return v;
  };
  for (int b = 0; b < nb; ++b) {
    VideoInfo v = info(b);
    v.spill_off = spill;
    v.vis_off = vis_off;
    v.frame_off = frame_off;
    if (!a->text_evidence) spill += static_cast<int64_t>(hq) * v.n_vis * v.text_pitch;
    vis_off += v.n_vis;
    frame_off += v.n_vis / a->tokens_per_frame;
    if (o) o->videos[b] = v;
  }
  c.spill_floats = spill;
  c.total_vis = vis_off;
  c.total_frames = frame_off;

  int max_visual = 1;
  int64_t r = 0;
  for (int b = 0; b < nb; ++b) {
    const VideoInfo v = info(b);
    const int n_vt = (v.n_vis + T - 1) / T;
    for (int t = 0; t < n_vt; ++t, ++r) {
      const int kv_begin = static_cast<int>(c.kv);
      for (int32_t i = a->mask_row_ptr_h[r]; i < a->mask_row_ptr_h[r + 1]; ++i, ++c.kv) {
        const int col = a->mask_col_idx_h[i];
        if (o) o->kv[c.kv] = KvTile{v.vis_start + col * T, static_cast<int16_t>(std::min(T, v.n_vis - col * T)),
                                    static_cast<uint8_t>(col == t), 1};
      }
      const int cnt = static_cast<int>(c.kv) - kv_begin;
      max_visual = std::max(max_visual, cnt);
      for (int g = 0; g < a->hkv; ++g)
        for (int hh = 0; hh < gq; hh += kSlots * hp, ++c.items)
          if (o) o->items[c.items] = WorkItem{v.vis_start + t * T, std::min(T, v.n_vis - t * T), g * gq + hh,
                                              kv_begin, cnt, -1, b, -1};
    }
  }
  int64_t work = c.kv;
  for (int b = 0; b < nb; ++b) {
    const VideoInfo v = info(b);
    const int64_t n_vt = (v.n_vis + T - 1) / T, n_tt = (v.n_text + T - 1) / T;
    work += n_tt * n_vt + n_tt * (n_tt + 1) / 2;
  }
  const int64_t head_blocks = static_cast<int64_t>(a->hkv) * ((gq + kSlots * hp - 1) / (kSlots * hp));
  const int split_len = text_split_len(max_visual, work * head_blocks);
  for (int b = 0; b < nb; ++b) {
    const VideoInfo v = info(b);
    const int n_vt = (v.n_vis + T - 1) / T;
    const int n_tt = (v.n_text + T - 1) / T;
    for (int t = 0; t < n_tt; ++t) {
      const int kv_begin = static_cast<int>(c.kv);
      for (int col = 0; col < n_vt; ++col, ++c.kv)
        if (o) o->kv[c.kv] = KvTile{v.vis_start + col * T, static_cast<int16_t>(std::min(T, v.n_vis - col * T)), 0, 1};
      for (int u = 0; u <= t; ++u, ++c.kv)
        if (o) o->kv[c.kv] = KvTile{v.vis_start + v.n_vis + u * T, static_cast<int16_t>(std::min(T, v.n_text - u * T)),
                                    static_cast<uint8_t>(u == t), 0};
      const int cnt = static_cast<int>(c.kv) - kv_begin;
      const int nsplit = (cnt + split_len - 1) / split_len;
      const int q_start = v.vis_start + v.n_vis + t * T;
      const int q_len = std::min(T, v.n_text - t * T);
      for (int g = 0; g < a->hkv; ++g) {
        for (int hh = 0; hh < gq; hh += kSlots * hp) {
          const int h = g * gq + hh;
          int part0 = -1;
          if (nsplit > 1) {
            part0 = static_cast<int>(c.parts);
            c.parts += kSlots * nsplit;
            for (int slot = 0; slot < kSlots && hh + slot * hp < gq; ++slot, ++c.groups)
              if (o) o->groups[c.groups] = CombineGroup{q_start, q_len, h + slot * hp, part0 + slot, nsplit, kSlots, 0, 0};
          }
          for (int s = 0; s < nsplit; ++s, ++c.items) {
            const int lo = static_cast<int>(static_cast<int64_t>(cnt) * s / nsplit);
            const int hi = static_cast<int>(static_cast<int64_t>(cnt) * (s + 1) / nsplit);
            if (o) o->items[c.items] = WorkItem{q_start, q_len, h, kv_begin + lo, hi - lo,
                                                nsplit > 1 ? part0 + kSlots * s : -1, b, t * T};
          }
        }
      }
    }
  }
  for (int b = 0; b < nb; ++b) {
    const int nv = a->n_vis_h[b];
    for (int col = 0; col < nv; col += 128, ++c.chunks)
      if (o) o->chunks[c.chunks] = EvChunk{b, col};
  }
  if (o) {
    // Longest first (a strict total order, so the in-place sort is deterministic).
    std::sort(o->items, o->items + c.items, [](const WorkItem& x, const WorkItem& y) {
      if (x.kv_count != y.kv_count) return x.kv_count > y.kv_count;
      const bool tx = x.text_row0 >= 0, ty = y.text_row0 >= 0;
      if (tx != ty) return ty;
      if (x.q_start != y.q_start) return x.q_start < y.q_start;
      if (x.head != y.head) return x.head < y.head;
      return x.kv_begin < y.kv_begin;
    });
  }
}

}  // namespace

extern "C" int evisel_probe_evidence_noalloc(const evisel_probe_args* args, float* tok, float* frame, float* head,
                                             float* aqf, int accumulate, void* stream_ptr, int* device_status) {
  nvtxRangePushA("evisel_probe_evidence_noalloc");
  struct Pop {
    ~Pop() { nvtxRangePop(); }
  } const nvtx_pop;
  clear_last_error();
  int rc = validate_probe_args(args);
  if (rc != EVISEL_OK) return rc;
  if (args->cross_frame)
    return set_last_error(EVISEL_EUNSUPPORTED, "cross-frame partials need a workspace (evisel_probe_attention)");
  if (args->keep)
    return set_last_error(EVISEL_EUNSUPPORTED, "per-row block masks need a workspace (evisel_probe_attention)");
  Counts c;
  make_plan(args, c, nullptr);
  if ((c.total_vis > 0 && (!tok || !frame)) || (args->num_videos > 0 && !head) || (c.total_frames > 0 && !aqf))
    return set_last_error(EVISEL_EINVAL, "an output map is NULL");
  if ((reinterpret_cast<uintptr_t>(tok) & 15u) != 0) return set_last_error(EVISEL_EINVAL, "tok must be 16-byte aligned");

  // Scratch layout: [status | items | kv | videos | groups | chunks | partial O | partial (m, l) | spill]
  const int nb = args->num_videos;
  size_t off = 256;
  auto take = [&](size_t bytes) { const size_t at = off; off = align256(off + bytes); return at; };
  const size_t o_items = take(c.items * sizeof(WorkItem));
  const size_t o_kv = take(c.kv * sizeof(KvTile));
  const size_t o_videos = take(static_cast<size_t>(nb) * sizeof(VideoInfo));
  const size_t o_groups = take(c.groups * sizeof(CombineGroup));
  const size_t o_chunks = take(c.chunks * sizeof(EvChunk));
  const size_t meta_end = off;
  const size_t o_part_o = take(static_cast<size_t>(c.parts) * 128 * args->head_dim * sizeof(float));
  const size_t o_part_ml = take(static_cast<size_t>(c.parts) * 128 * sizeof(float2));
  const size_t o_spill = take(static_cast<size_t>(c.spill_floats) * sizeof(float));
  if (off > kScratchBytes || meta_end - 256 > kStageBytes) {
    const std::string msg = "problem needs " + std::to_string(off) + " bytes of scratch (plan " +
                            std::to_string(meta_end - 256) + " bytes); the static scratch holds " +
                            std::to_string(kScratchBytes) + " bytes (plan at most " + std::to_string(kStageBytes) +
                            "); use evisel_probe_attention for larger problems";
    return set_last_error(EVISEL_ENOMEM, msg.c_str());
  }

  std::lock_guard<std::mutex> lock(g_mutex);
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess || dev < 0 || dev >= kMaxDevices)
    return set_last_error(EVISEL_ECUDA, "cudaGetDevice failed or device index out of range");
  if (!g_scratch_ptr[dev]) {
    // Device address of the array on the current device (a host-side use of
    // the symbol's name would only give the host stand-in).
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_scratch);
    if (e != cudaSuccess) {
      cudaGetLastError();
      return set_last_error(EVISEL_ECUDA, (std::string("cudaGetSymbolAddress: ") + cudaGetErrorString(e)).c_str());
    }
    g_scratch_ptr[dev] = p;
  }
  unsigned char* base = static_cast<unsigned char*>(g_scratch_ptr[dev]);
  cudaStream_t stream = static_cast<cudaStream_t>(stream_ptr);

  Out out{reinterpret_cast<WorkItem*>(g_stage + (o_items - 256)), reinterpret_cast<KvTile*>(g_stage + (o_kv - 256)),
          reinterpret_cast<VideoInfo*>(g_stage + (o_videos - 256)),
          reinterpret_cast<CombineGroup*>(g_stage + (o_groups - 256)),
          reinterpret_cast<EvChunk*>(g_stage + (o_chunks - 256))};
  make_plan(args, c, &out);

  // The status word must start at zero; the rest is fully written before it is read.
  e = cudaMemsetAsync(base, 0, sizeof(int), stream);
  // Pageable source: the copy is staged before cudaMemcpyAsync returns, so g_stage
  // may be rewritten by the next call.
  if (e == cudaSuccess && meta_end > 256)
    e = cudaMemcpyAsync(base + 256, g_stage, meta_end - 256, cudaMemcpyHostToDevice, stream);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return set_last_error(EVISEL_ECUDA, (std::string("plan upload: ") + cudaGetErrorString(e)).c_str());
  }

  const int n_tok = nb ? args->cu_seqlens_h[nb] : 0;
  const float scale = args->softmax_scale > 0.f ? args->softmax_scale : 1.0f / std::sqrt(float(args->head_dim));
  if (c.items > 0) {
    ProbeLaunch L;
    std::memset(&L, 0, sizeof(L));
    rc = encode_tensor_map(&L.tm_q, args->q, n_tok, args->hq, args->head_dim, args->tile);
    if (rc == EVISEL_OK) rc = encode_tensor_map(&L.tm_k, args->k, n_tok, args->hkv, args->head_dim, args->tile);
    if (rc == EVISEL_OK) rc = encode_tensor_map(&L.tm_v, args->v, n_tok, args->hkv, args->head_dim, args->tile);
    if (rc == EVISEL_OK) rc = encode_tensor_map(&L.tm_o, args->o, n_tok, args->hq, args->head_dim, args->tile);
    if (rc != EVISEL_OK) return rc;
    L.items = reinterpret_cast<const WorkItem*>(base + o_items);
    L.kv = reinterpret_cast<const KvTile*>(base + o_kv);
    L.videos = reinterpret_cast<const VideoInfo*>(base + o_videos);
    L.o = args->o;
    L.lse = args->lse;
    L.spill = args->text_evidence ? nullptr : reinterpret_cast<float*>(base + o_spill);
    L.part_o = reinterpret_cast<float*>(base + o_part_o);
    L.part_ml = reinterpret_cast<float2*>(base + o_part_ml);
    L.status = reinterpret_cast<int*>(base);
    L.n_items = static_cast<int>(c.items);
    L.n_tok = n_tok;
    L.hq = args->hq;
    L.hkv = args->hkv;
    L.head_dim = args->head_dim;
    L.tile = args->tile;
    L.scale = scale;
    L.scale_log2 = scale * 1.4426950408889634f;
    e = launch_probe_attn(L, stream);
    if (e == cudaSuccess && c.groups > 0) {
      CombineLaunch C{};
      C.groups = reinterpret_cast<const CombineGroup*>(base + o_groups);
      C.part_o = L.part_o;
      C.part_ml = L.part_ml;
      C.o = args->o;
      C.lse = args->lse;
      C.n_groups = static_cast<int>(c.groups);
      C.n_tok = n_tok;
      C.hq = args->hq;
      C.hkv = args->hkv;
      C.head_dim = args->head_dim;
      C.tile = args->tile;
      e = launch_attn_combine(C, stream);
    }
    if (e != cudaSuccess) {
      cudaGetLastError();
      return set_last_error(EVISEL_ECUDA, (std::string("probe launch: ") + cudaGetErrorString(e)).c_str());
    }
  }
  if (nb > 0) {
    EvidenceLaunch E{};
    E.chunks = reinterpret_cast<const EvChunk*>(base + o_chunks);
    E.videos = reinterpret_cast<const VideoInfo*>(base + o_videos);
    E.spill = reinterpret_cast<const float*>(base + o_spill);
    E.lse = args->lse;
    E.tok = tok;
    E.frame = frame;
    E.head = head;
    E.aqf = aqf;
    E.n_chunks = static_cast<int>(c.chunks);
    E.n_videos = nb;
    E.n_tok = n_tok;
    E.hq = args->hq;
    E.tokens_per_frame = args->tokens_per_frame;
    E.total_vis = c.total_vis;
    E.total_frames = c.total_frames;
    E.accumulate = accumulate != 0;
    if (args->text_evidence && c.chunks > 0) {
      // Token and frame maps recomputed from q and k (no spill).
      TextEvidenceLaunch T;
      std::memset(&T, 0, sizeof(T));
      rc = encode_tensor_map(&T.tm_q, args->q, n_tok, args->hq, args->head_dim, 128);
      if (rc == EVISEL_OK) rc = encode_tensor_map(&T.tm_k, args->k, n_tok, args->hkv, args->head_dim, 128);
      if (rc != EVISEL_OK) return rc;
      T.chunks = E.chunks;
      T.videos = E.videos;
      T.lse = args->lse;
      T.tok = tok;
      T.frame = frame;
      T.status = reinterpret_cast<int*>(base);
      T.n_chunks = static_cast<int>(c.chunks);
      T.n_tok = n_tok;
      T.hq = args->hq;
      T.hkv = args->hkv;
      T.head_dim = args->head_dim;
      T.tokens_per_frame = args->tokens_per_frame;
      T.total_vis = c.total_vis;
      T.total_frames = c.total_frames;
      const float scale = args->softmax_scale > 0.f ? args->softmax_scale : 1.0f / std::sqrt(float(args->head_dim));
      T.scale_log2 = scale * 1.4426950408889634f;
      T.accumulate = accumulate != 0;
      e = launch_text_evidence(T, stream);
      if (e != cudaSuccess) {
        cudaGetLastError();
        return set_last_error(EVISEL_ECUDA, (std::string("text_evidence launch: ") + cudaGetErrorString(e)).c_str());
      }
      E.n_chunks = 0;
    }
    e = launch_evidence(E, stream);
    if (e != cudaSuccess) {
      cudaGetLastError();
      return set_last_error(EVISEL_ECUDA, (std::string("evidence launch: ") + cudaGetErrorString(e)).c_str());
    }
  }
  if (device_status) {
    e = cudaStreamSynchronize(stream);
    if (e == cudaSuccess) e = cudaMemcpy(device_status, base, sizeof(int), cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) {
      cudaGetLastError();
      return set_last_error(EVISEL_ECUDA, (std::string("status read: ") + cudaGetErrorString(e)).c_str());
    }
  }
  return EVISEL_OK;
}
