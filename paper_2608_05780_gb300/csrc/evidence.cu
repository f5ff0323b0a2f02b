// Evidence pass over the text rows (Sec. 3.2, "Evidence Decomposition").
//
// evidence_reduce: re-forms the text-row probabilities P_im = exp(s_im - LSE_i)
// from the spilled logits and the saved LSE and sums them over the text rows
// (token map), then over each frame's N_v tokens (frame map). HBM-bound: one
// streaming read of the spill, laid out [hq, text rows / 32, n_vis, 32] (the
// attention kernel writes one key of a warp's 32 rows as 128 contiguous
// bytes). One block handles 128 visual keys of one video for one head: per
// 32-row block those keys are 16 KB in a row; each of the 4 warps reads its
// 32 keys' 4 KB with 16-byte loads (lane l: 4 rows of keys 4i + l / 8), sums
// over all row blocks in registers, closes each key over its 8 lanes, and the
// block forms the frames (N_v divides 128) from the 128 token sums.
//
// evidence_finalize: head map (sum of a video's frames per head; one warp per
// video and head) and the query-frame cue A_qf (sum over heads / (Hq * n_text);
// one thread per frame), both recomputed from the frame map so that they
// accumulate over layers exactly as it does.
#include <cstdint>
#include <cuda_runtime.h>

#include "evisel_internal.h"

namespace evisel {
namespace {

constexpr int kChunk = 128;                        // visual keys per block
constexpr int kWarps = kChunk / 32;                // one warp per 32 keys

// 16 blocks of 128 threads per SM (32 registers): the full 2,048 threads,
// which the HBM stream needs (at 45 registers it ran 11 blocks and 26% slower).
__global__ void __launch_bounds__(kWarps * 32, 16) evidence_reduce_kernel(const __grid_constant__ EvidenceLaunch L) {
  __shared__ float tok_s[kChunk];
  const int h = blockIdx.y;
  const EvChunk ck = L.chunks[blockIdx.x];
  const VideoInfo vi = L.videos[ck.video];
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int n_rb = vi.text_pitch >> 5;
  const float* lse = L.lse + static_cast<int64_t>(h) * L.n_tok + vi.vis_start + vi.n_vis;
  const int key0 = ck.col0 + warp * 32;             // this warp's first key (within the video)
  const int sub = lane & 7;                         // rows 4 sub .. 4 sub + 3 of each row block
  // float4 i of the warp's 4 KB in a row block: keys key0 + 4 i + lane / 8.
  const float4* base = reinterpret_cast<const float4*>(L.spill + vi.spill_off +
                                                       static_cast<int64_t>(h) * vi.n_vis * vi.text_pitch +
                                                       static_cast<int64_t>(key0) * 32) + lane;

  float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  for (int rb = 0; rb < n_rb; ++rb) {
    const int row = rb * 32 + 4 * sub;
    float m[4];
    bool in[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      in[u] = row + u < vi.n_text;   // rows past n_text are padding that was never written
      m[u] = in[u] ? __ldg(lse + row + u) : 0.f;
    }
    const float4* src = base + static_cast<int64_t>(rb) * vi.n_vis * 8;
    float4 sv[8];
#pragma unroll
    for (int i = 0; i < 8; ++i)
      sv[i] = key0 + 4 * i + (lane >> 3) < vi.n_vis ? __ldcs(src + i * 32)
                                                   : make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const float e0 = in[0] ? __expf(sv[i].x - m[0]) : 0.f;
      const float e1 = in[1] ? __expf(sv[i].y - m[1]) : 0.f;
      const float e2 = in[2] ? __expf(sv[i].z - m[2]) : 0.f;
      const float e3 = in[3] ? __expf(sv[i].w - m[3]) : 0.f;
      acc[i] += (e0 + e1) + (e2 + e3);
    }
  }
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    float t = acc[i];
    t += __shfl_xor_sync(0xffffffffu, t, 4);
    t += __shfl_xor_sync(0xffffffffu, t, 2);
    t += __shfl_xor_sync(0xffffffffu, t, 1);
    if (sub == 0) tok_s[warp * 32 + 4 * i + (lane >> 3)] = t;
  }
  __syncthreads();

  const int nkeys = min(kChunk, vi.n_vis - ck.col0);   // a multiple of N_v
  const int c = threadIdx.x;
  // Token map.
  if (c < nkeys) {
    float* dst = L.tok + static_cast<int64_t>(h) * L.total_vis + vi.vis_off + ck.col0 + c;
    *dst = L.accumulate ? *dst + tok_s[c] : tok_s[c];
  }
  // Frame map: frame f of the chunk is keys [f N_v, (f + 1) N_v).
  const int npf = L.tokens_per_frame;
  if (c < nkeys / npf) {
    float f = 0.f;
    for (int i = 0; i < npf; ++i) f += tok_s[c * npf + i];
    float* dst = L.frame + static_cast<int64_t>(h) * L.total_frames + vi.frame_off + ck.col0 / npf + c;
    *dst = L.accumulate ? *dst + f : f;
  }
}

// Blocks [0, n_videos * head_blocks): head map, one warp per (video, head),
// four independent partial sums per lane. Blocks after those: A_qf, one
// thread per frame.
constexpr int kFinalizeWarps = 8;

__global__ void __launch_bounds__(kFinalizeWarps * 32) evidence_finalize_kernel(const __grid_constant__ EvidenceLaunch L) {
  const int head_blocks = (L.hq + kFinalizeWarps - 1) / kFinalizeWarps;
  if (blockIdx.x < static_cast<unsigned>(L.n_videos * head_blocks)) {
    const int b = blockIdx.x / head_blocks;
    const int h = (blockIdx.x % head_blocks) * kFinalizeWarps + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (h >= L.hq) return;
    const VideoInfo vi = L.videos[b];
    const int frames = vi.n_vis / L.tokens_per_frame;
    const float* fr = L.frame + static_cast<int64_t>(h) * L.total_frames + vi.frame_off;
    float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
    int t = lane;
    for (; t + 96 < frames; t += 128) {
      s0 += fr[t];
      s1 += fr[t + 32];
      s2 += fr[t + 64];
      s3 += fr[t + 96];
    }
    for (; t < frames; t += 32) s0 += fr[t];
    float s = (s0 + s1) + (s2 + s3);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
    if (lane == 0) L.head[static_cast<int64_t>(b) * L.hq + h] = s;
    return;
  }
  const int t = (blockIdx.x - L.n_videos * head_blocks) * blockDim.x + threadIdx.x;
  if (t >= L.total_frames) return;
  int lo = 0, hi = L.n_videos - 1;                 // video owning frame t
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (L.videos[mid].frame_off <= t) lo = mid; else hi = mid - 1;
  }
  // (the last video whose frame offset is <= t always owns >= 1 frame)
  const VideoInfo vi = L.videos[lo];
  float s0 = 0.f, s1 = 0.f;
  int h = 0;
  for (; h + 1 < L.hq; h += 2) {
    s0 += L.frame[static_cast<int64_t>(h) * L.total_frames + t];
    s1 += L.frame[static_cast<int64_t>(h + 1) * L.total_frames + t];
  }
  if (h < L.hq) s0 += L.frame[static_cast<int64_t>(h) * L.total_frames + t];
  L.aqf[t] = vi.n_text > 0 ? (s0 + s1) / (static_cast<float>(L.hq) * static_cast<float>(vi.n_text)) : 0.f;
}

}  // namespace

cudaError_t launch_evidence(const EvidenceLaunch& L, cudaStream_t stream) {
  if (L.n_chunks > 0) {
    dim3 grid(L.n_chunks, L.hq);
    evidence_reduce_kernel<<<grid, kWarps * 32, 0, stream>>>(L);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  const int head_blocks = (L.hq + kFinalizeWarps - 1) / kFinalizeWarps;
  const int aqf_blocks = (L.total_frames + kFinalizeWarps * 32 - 1) / (kFinalizeWarps * 32);
  if (L.n_videos * head_blocks + aqf_blocks > 0) {
    evidence_finalize_kernel<<<L.n_videos * head_blocks + aqf_blocks, kFinalizeWarps * 32, 0, stream>>>(L);
    return cudaGetLastError();
  }
  return cudaSuccess;
}

}  // namespace evisel
