// Evidence pass over the text rows (Sec. 3.2, "Evidence Decomposition").
//
// evidence_reduce: re-forms the text-row probabilities P_im = exp(s_im - LSE_i)
// from the spilled logits and the saved LSE and sums them over the text rows
// (token map), then over each frame's N_v tokens (frame map). HBM-bound: one
// streaming read of the spill. One block handles 128 visual columns of one
// video for one head; its 8 warps split the text rows, each lane owns 4
// consecutive columns (16-byte loads); partial sums meet in shared memory and
// frames are closed with a segmented warp-shuffle sum (N_v / 4 lanes).
//
// evidence_finalize: head map (sum of a video's frames per head) and the
// query-frame cue A_qf (sum over heads / (Hq * n_text)), both recomputed from
// the frame map so that they accumulate over layers exactly as it does.
#include <cstdint>
#include <cuda_runtime.h>

#include "evisel_internal.h"

namespace evisel {
namespace {

constexpr int kWarps = 8;

__device__ __forceinline__ float4 ld_stream(const float* p) {
  return __ldcs(reinterpret_cast<const float4*>(p));
}

__global__ void __launch_bounds__(kWarps * 32) evidence_reduce_kernel(const __grid_constant__ EvidenceLaunch L) {
  __shared__ float4 part[kWarps][32];
  const int h = blockIdx.y;
  const EvChunk ck = L.chunks[blockIdx.x];
  const VideoInfo vi = L.videos[ck.video];
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int col = ck.col0 + lane * 4;            // visual column within the video
  const bool col_ok = col < vi.n_vis;            // n_vis is a multiple of 4

  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  if (col_ok) {
    const float* base = L.spill + vi.spill_off + static_cast<int64_t>(h) * vi.n_text * vi.vis_pitch + col;
    const float* lse = L.lse + static_cast<int64_t>(h) * L.n_tok + vi.vis_start + vi.n_vis;
    int i = warp;
    for (; i + 3 * kWarps < vi.n_text; i += 4 * kWarps) {
      float4 s[4];
      float m[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        s[u] = ld_stream(base + static_cast<int64_t>(i + u * kWarps) * vi.vis_pitch);
        m[u] = __ldg(lse + i + u * kWarps);
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        acc.x += __expf(s[u].x - m[u]);
        acc.y += __expf(s[u].y - m[u]);
        acc.z += __expf(s[u].z - m[u]);
        acc.w += __expf(s[u].w - m[u]);
      }
    }
    for (; i < vi.n_text; i += kWarps) {
      const float4 s = ld_stream(base + static_cast<int64_t>(i) * vi.vis_pitch);
      const float m = __ldg(lse + i);
      acc.x += __expf(s.x - m);
      acc.y += __expf(s.y - m);
      acc.z += __expf(s.z - m);
      acc.w += __expf(s.w - m);
    }
  }
  part[warp][lane] = acc;
  __syncthreads();
  if (warp != 0) return;
  float4 t = part[0][lane];
#pragma unroll
  for (int w = 1; w < kWarps; ++w) {
    const float4 o = part[w][lane];
    t.x += o.x; t.y += o.y; t.z += o.z; t.w += o.w;
  }
  // Token map.
  if (col_ok) {
    float4* dst = reinterpret_cast<float4*>(L.tok + static_cast<int64_t>(h) * L.total_vis + vi.vis_off + col);
    if (L.accumulate) {
      const float4 o = *dst;
      *dst = make_float4(o.x + t.x, o.y + t.y, o.z + t.z, o.w + t.w);
    } else {
      *dst = t;
    }
  }
  // Frame map: frames of N_v tokens are N_v / 4 consecutive lanes.
  float f = t.x + t.y + t.z + t.w;
  const int lanes = L.tokens_per_frame >> 2;
  for (int off = 1; off < lanes; off <<= 1) f += __shfl_xor_sync(0xffffffffu, f, off);
  if (col_ok && (lane & (lanes - 1)) == 0) {
    float* dst = L.frame + static_cast<int64_t>(h) * L.total_frames + vi.frame_off + col / L.tokens_per_frame;
    *dst = L.accumulate ? *dst + f : f;
  }
}

// Blocks [0, n_videos): head map of one video (one warp per head).
// Blocks [n_videos, ...): A_qf, one thread per frame.
__global__ void __launch_bounds__(256) evidence_finalize_kernel(const __grid_constant__ EvidenceLaunch L) {
  if (blockIdx.x < static_cast<unsigned>(L.n_videos)) {
    const VideoInfo vi = L.videos[blockIdx.x];
    const int frames = vi.n_vis / L.tokens_per_frame;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    for (int h = warp; h < L.hq; h += 8) {
      const float* fr = L.frame + static_cast<int64_t>(h) * L.total_frames + vi.frame_off;
      float s = 0.f;
      for (int t = lane; t < frames; t += 32) s += fr[t];
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
      if (lane == 0) L.head[static_cast<int64_t>(blockIdx.x) * L.hq + h] = s;
    }
    return;
  }
  const int t = (blockIdx.x - L.n_videos) * blockDim.x + threadIdx.x;
  if (t >= L.total_frames) return;
  int lo = 0, hi = L.n_videos - 1;                 // video owning frame t
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (L.videos[mid].frame_off <= t) lo = mid; else hi = mid - 1;
  }
  // (the last video whose frame offset is <= t always owns >= 1 frame)
  const VideoInfo vi = L.videos[lo];
  float s = 0.f;
  for (int h = 0; h < L.hq; ++h) s += L.frame[static_cast<int64_t>(h) * L.total_frames + t];
  L.aqf[t] = vi.n_text > 0 ? s / (static_cast<float>(L.hq) * static_cast<float>(vi.n_text)) : 0.f;
}

}  // namespace

cudaError_t launch_evidence(const EvidenceLaunch& L, cudaStream_t stream) {
  if (L.n_chunks > 0) {
    dim3 grid(L.n_chunks, L.hq);
    evidence_reduce_kernel<<<grid, kWarps * 32, 0, stream>>>(L);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  const int aqf_blocks = (L.total_frames + 255) / 256;
  if (L.n_videos + aqf_blocks > 0) {
    evidence_finalize_kernel<<<L.n_videos + aqf_blocks, 256, 0, stream>>>(L);
    return cudaGetLastError();
  }
  return cudaSuccess;
}

}  // namespace evisel
