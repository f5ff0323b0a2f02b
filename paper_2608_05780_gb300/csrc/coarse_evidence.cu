// Evidence from the coarse token-level map of the sparse prefill (Appendix,
// "Detailed Sparse Prefilling", Eq. 10-11). For a text row i of head h:
//   a_im = scale q_i k_m              for the keys of its own block up to i (E_i),
//   a_im = g_ij = scale q_i k_bar_j   for the tokens of each retained block j in S_i,
//   -inf elsewhere;  A~_im = exp(a_im) / sum_n exp(a_in)                (Eq. 11)
// and the maps of Sec. 3.2: tok[h, m] = sum over the text rows of A~_im for the
// visual tokens m, frame sums, head sums and A_qf. All tokens of a retained
// visual block share its weight exp(g_ij - M_i) / Z_i.
//
// coarse_rows_kernel: one warp per (text row, head). Lanes split d; for every
//   block of the row's history the warp forms g_ij (stored for the next
//   kernel) and, over S_i (the keep bits), the running max M_i and the sum
//   Z_i = sum_{S_i} B exp(g - M) + sum_{E_i} exp(s - M) with the exact own-block
//   logits s.
// coarse_map_kernel: one thread per (frame, head, video): for each block of
//   the frame, c_j = sum over the video's text rows of [j in S_i]
//   exp(g_ij - M_i) / Z_i (rows in order: deterministic); writes c_j to the
//   block's tokens and B sum_j c_j to the frame.
// coarse_finalize_kernel: head[b, h] = sum of the video's frames; A_qf[t] =
//   sum_h frame[h, t] / (Hq n_text), from the (possibly accumulated) frame map.
#include <algorithm>
#include <cstdint>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "evisel_internal.h"

namespace evisel {
namespace {

constexpr unsigned kFull = 0xffffffffu;

__device__ __forceinline__ float warp_sum(float x) {
  for (int off = 16; off > 0; off >>= 1) x += __shfl_xor_sync(kFull, x, off);
  return x;
}

__global__ void __launch_bounds__(256) coarse_rows_kernel(const __grid_constant__ CoarseLaunch L) {
  const int warp_global = blockIdx.x * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  const int h = blockIdx.y;
  if (warp_global >= L.total_text) return;       // warp-uniform
  // The text row: find its video (text rows of the videos back to back).
  int v = 0;
  while (v + 1 < L.n_videos && L.text_off[v + 1] <= warp_global) ++v;
  const ToppVideo vid = L.vids[v];
  const int t = warp_global - L.text_off[v];     // text row within the video
  const int pos = vid.n_vis + t;                 // video-local position
  const int row = vid.start + pos;               // global token
  const int B = L.block, nvb = vid.n_vis / B;
  const int nh = nvb + t / B;                    // blocks that end before the row
  const int own0 = vid.n_vis + (t / B) * B;      // first token of its own block
  const int g = h / (L.hq / L.hkv);
  const int d = L.head_dim;
  const __nv_bfloat16* q = static_cast<const __nv_bfloat16*>(L.q) + (static_cast<int64_t>(row) * L.hq + h) * d;
  const __nv_bfloat16* kbar = static_cast<const __nv_bfloat16*>(L.kbar);
  const __nv_bfloat16* k = static_cast<const __nv_bfloat16*>(L.k);
  // This lane's d / 32 query elements (d = 64 or 128: 2 or 4 per lane).
  float qv[4] = {0.f, 0.f, 0.f, 0.f};
  const int per = d / 32;
  for (int e = 0; e < per; ++e) qv[e] = __bfloat162float(q[lane * per + e]);
  auto dot = [&](const __nv_bfloat16* kr) {
    float s = 0.f;
    for (int e = 0; e < per; ++e) s += qv[e] * __bfloat162float(kr[lane * per + e]);
    return warp_sum(s) * L.scale;
  };
  float* grow = L.gbuf + (static_cast<int64_t>(h) * L.total_text + warp_global) * L.pitch;
  const uint32_t* keep = L.keep + static_cast<int64_t>(h) * L.n_words * L.n_tok + row;
  float m = -INFINITY, z = 0.f;
  uint32_t word = 0u;
  for (int j = 0; j < nh; ++j) {
    if ((j & 31) == 0) word = keep[static_cast<int64_t>(j >> 5) * L.n_tok];
    const float gj = dot(kbar + (static_cast<int64_t>(vid.blk_off + j) * L.hkv + g) * d);
    if (lane == 0) grow[j] = gj;
    if ((word >> (j & 31)) & 1u) {               // j in S_i: B tokens share g_ij
      if (gj > m) {
        z = (m == -INFINITY) ? 0.f : z * __expf(m - gj);
        m = gj;
      }
      z += static_cast<float>(B) * __expf(gj - m);
    }
  }
  for (int mm = own0; mm <= pos; ++mm) {          // E_i: exact logits of the own block's causal prefix
    const float s = dot(k + (static_cast<int64_t>(vid.start + mm) * L.hkv + g) * d);
    if (s > m) {
      z = (m == -INFINITY) ? 0.f : z * __expf(m - s);
      m = s;
    }
    z += __expf(s - m);
  }
  if (lane == 0) {
    L.row_m[static_cast<int64_t>(h) * L.total_text + warp_global] = m;
    L.row_z[static_cast<int64_t>(h) * L.total_text + warp_global] = z;
  }
}

__global__ void __launch_bounds__(128) coarse_map_kernel(const __grid_constant__ CoarseLaunch L) {
  const int v = blockIdx.z, h = blockIdx.y;
  const ToppVideo vid = L.vids[v];
  const int npf = L.tokens_per_frame, B = L.block;
  const int n_frames = vid.n_vis / npf;
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= n_frames) return;
  const int n_text = vid.n_text;
  const int tr0 = L.text_off[v];
  float fsum = 0.f;
  for (int jj = 0; jj < npf / B; ++jj) {
    const int j = t * (npf / B) + jj;            // visual block
    float c = 0.f;
    for (int i = 0; i < n_text; ++i) {
      const int row = vid.start + vid.n_vis + i;
      const uint32_t word = L.keep[(static_cast<int64_t>(h) * L.n_words + (j >> 5)) * L.n_tok + row];
      if ((word >> (j & 31)) & 1u) {
        const int64_t r = static_cast<int64_t>(h) * L.total_text + tr0 + i;
        c += __expf(L.gbuf[r * L.pitch + j] - L.row_m[r]) / L.row_z[r];
      }
    }
    float* tok = L.tok + static_cast<int64_t>(h) * L.total_vis + L.vis_off[v] + j * B;
    for (int e = 0; e < B; ++e) tok[e] = L.accumulate ? tok[e] + c : c;
    fsum += static_cast<float>(B) * c;
  }
  float* fr = L.frame + static_cast<int64_t>(h) * L.total_frames + L.frame_off[v] + t;
  *fr = L.accumulate ? *fr + fsum : fsum;
}

__global__ void __launch_bounds__(128) coarse_finalize_kernel(const __grid_constant__ CoarseLaunch L) {
  const int v = blockIdx.y;
  const ToppVideo vid = L.vids[v];
  const int n_frames = vid.n_vis / L.tokens_per_frame;
  const int f0 = L.frame_off[v];
  if (blockIdx.x == 0) {                         // head map: one thread per head
    for (int h = threadIdx.x; h < L.hq; h += blockDim.x) {
      float s = 0.f;
      for (int t = 0; t < n_frames; ++t) s += L.frame[static_cast<int64_t>(h) * L.total_frames + f0 + t];
      L.head[static_cast<int64_t>(v) * L.hq + h] = s;
    }
  }
  const float inv = vid.n_text > 0 ? 1.f / (static_cast<float>(L.hq) * vid.n_text) : 0.f;
  for (int t = blockIdx.x * blockDim.x + threadIdx.x; t < n_frames; t += gridDim.x * blockDim.x) {
    float s = 0.f;
    for (int h = 0; h < L.hq; ++h) s += L.frame[static_cast<int64_t>(h) * L.total_frames + f0 + t];
    L.aqf[f0 + t] = s * inv;
  }
}

}  // namespace

cudaError_t launch_coarse(const CoarseLaunch& L, cudaStream_t stream) {
  if (L.n_videos == 0) return cudaSuccess;
  if (L.total_text > 0) {
    dim3 g1((L.total_text + 7) / 8, L.hq);
    coarse_rows_kernel<<<g1, 256, 0, stream>>>(L);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  if (L.max_frames > 0) {
    dim3 g2((L.max_frames + 127) / 128, L.hq, L.n_videos);
    coarse_map_kernel<<<g2, 128, 0, stream>>>(L);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  dim3 g3(std::max(1, (L.max_frames + 127) / 128), L.n_videos);
  coarse_finalize_kernel<<<g3, 128, 0, stream>>>(L);
  return cudaGetLastError();
}

}  // namespace evisel
