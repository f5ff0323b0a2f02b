// Evidence from the coarse token-level map of the sparse prefill (Appendix,
// "Detailed Sparse Prefilling", Eq. 10-11). For a text row i of head h:
//   a_im = scale q_i k_m              for the keys of its own block up to i (E_i),
//   a_im = g_ij = scale q_i k_bar_j   for the tokens of each retained block j in S_i,
//   -inf elsewhere;  A~_im = exp(a_im) / sum_n exp(a_in)                (Eq. 11)
// and the maps of Sec. 3.2: tok[h, m] = sum over the text rows of A~_im for the
// visual tokens m, frame sums, head sums and A_qf. All tokens of a retained
// visual block share its weight exp(g_ij - M_i) / Z_i.
//
// coarse_rows_kernel: one CTA per (8 text rows of a video, head), a warp per
//   row. The CTA stages the k_bar rows of the head's KV group in chunks of 32
//   blocks (one keep word) in shared memory; lane j of a warp takes block
//   j of each chunk: it forms g_ij = scale q_i k_bar_j (stored for the next
//   kernel) and, over its blocks in S_i, a running max and sum. The lanes'
//   pairs then merge (a butterfly: each step's merge is symmetric, so all
//   lanes agree) and the warp adds the exact logits s of the own block's
//   causal prefix E_i, giving M_i and
//   Z_i = sum_{S_i} B exp(g - M) + sum_{E_i} exp(s - M).
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

// s + sum of the 8 bf16 products of a and b, in order.
__device__ __forceinline__ float dot8(const uint4& a, const uint4& b, float s) {
  const __nv_bfloat162* a2 = reinterpret_cast<const __nv_bfloat162*>(&a);
  const __nv_bfloat162* b2 = reinterpret_cast<const __nv_bfloat162*>(&b);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float2 fa = __bfloat1622float2(a2[i]), fb = __bfloat1622float2(b2[i]);
    s = fmaf(fa.x, fb.x, s);
    s = fmaf(fa.y, fb.y, s);
  }
  return s;
}

// (m, z) <- the softmax pair of (m, z) and (m2, z2): max and rescaled sum.
__device__ __forceinline__ void merge_mz(float& m, float& z, float m2, float z2) {
  const float mm = fmaxf(m, m2);
  z = mm == -INFINITY ? 0.f : z * __expf(m - mm) + z2 * __expf(m2 - mm);
  m = mm;
}

constexpr int kRowsPerCta = 8;                   // text rows (warps) per CTA
constexpr int kChunk = 32;                       // k_bar rows staged at a time: one keep word

__global__ void __launch_bounds__(256) coarse_rows_kernel(const __grid_constant__ CoarseLaunch L) {
  __shared__ __align__(16) __nv_bfloat16 q_s[kRowsPerCta][128];   // each warp's query row
  __shared__ uint4 kb_s[kChunk][128 / 8 + 1];                     // k_bar rows, padded by 16 B
  const int wib = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int h = blockIdx.y;
  // This CTA's video and row group (groups of 8 text rows, videos back to back).
  int v = 0, grp = blockIdx.x;
  for (; v < L.n_videos; ++v) {
    const int cnt = (L.text_off[v + 1] - L.text_off[v] + kRowsPerCta - 1) / kRowsPerCta;
    if (grp < cnt) break;
    grp -= cnt;
  }
  if (v >= L.n_videos) return;                   // CTA-uniform, before any barrier
  const ToppVideo vid = L.vids[v];
  const int n_text = L.text_off[v + 1] - L.text_off[v];
  const int t_last = min(grp * kRowsPerCta + kRowsPerCta - 1, n_text - 1);
  const int t = min(grp * kRowsPerCta + wib, t_last);   // text row within the video (clamped)
  const bool active = grp * kRowsPerCta + wib <= t_last;   // warp-uniform
  const int trow = L.text_off[v] + t;            // text row over all videos
  const int pos = vid.n_vis + t;                 // video-local position
  const int row = vid.start + pos;               // global token
  const int B = L.block, nvb = vid.n_vis / B;
  const int nh = nvb + t / B;                    // blocks that end before the row
  const int nh_cta = nvb + t_last / B;           // the most over the CTA's rows
  const int own0 = vid.n_vis + (t / B) * B;      // first token of its own block
  const int g = h / (L.hq / L.hkv);
  const int d = L.head_dim, dc = d / 8;          // d = 64 or 128
  const __nv_bfloat16* q = static_cast<const __nv_bfloat16*>(L.q) + (static_cast<int64_t>(row) * L.hq + h) * d;
  for (int c = lane; c < dc; c += 32) reinterpret_cast<uint4*>(q_s[wib])[c] = reinterpret_cast<const uint4*>(q)[c];
  __syncwarp();
  const uint4* q4 = reinterpret_cast<const uint4*>(q_s[wib]);
  const __nv_bfloat16* kbar = static_cast<const __nv_bfloat16*>(L.kbar);
  const __nv_bfloat16* k = static_cast<const __nv_bfloat16*>(L.k);
  float* grow = L.gbuf + (static_cast<int64_t>(h) * L.total_text + trow) * L.pitch;
  const uint32_t* keep = L.keep + static_cast<int64_t>(h) * L.n_words * L.n_tok + row;
  float m = -INFINITY, z = 0.f;
  for (int j0 = 0; j0 < nh_cta; j0 += kChunk) {
    __syncthreads();                             // the previous chunk is consumed
    for (int i = threadIdx.x; i < kChunk * dc; i += blockDim.x) {   // coalesced: 16 B per thread
      const int jj = i / dc, c = i % dc;
      if (j0 + jj < nh_cta)
        kb_s[jj][c] = reinterpret_cast<const uint4*>(kbar + (static_cast<int64_t>(vid.blk_off + j0 + jj) * L.hkv + g) * d)[c];
    }
    __syncthreads();
    const int j = j0 + lane;
    if (active && j < nh) {
      const uint32_t word = keep[static_cast<int64_t>(j0 >> 5) * L.n_tok];
      float s = 0.f;
      for (int c = 0; c < dc; ++c) s = dot8(q4[c], kb_s[lane][c], s);
      const float gj = s * L.scale;
      grow[j] = gj;
      if ((word >> lane) & 1u) {                 // j in S_i: B tokens share g_ij
        if (gj > m) {
          z = (m == -INFINITY) ? 0.f : z * __expf(m - gj);
          m = gj;
        }
        z += static_cast<float>(B) * __expf(gj - m);
      }
    }
  }
  if (!active) return;                           // warp-uniform; no barrier follows
  for (int off = 16; off > 0; off >>= 1) {
    const float m2 = __shfl_xor_sync(kFull, m, off), z2 = __shfl_xor_sync(kFull, z, off);
    merge_mz(m, z, m2, z2);
  }
  // E_i: exact logits of the own block's causal prefix; lanes split d.
  const int per = d / 32;
  float qv[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
  for (int e = 0; e < 4; ++e)
    if (e < per) qv[e] = __bfloat162float(q_s[wib][lane * per + e]);
  for (int mm = own0; mm <= pos; ++mm) {
    const __nv_bfloat16* kr = k + (static_cast<int64_t>(vid.start + mm) * L.hkv + g) * d;
    float s = 0.f;
#pragma unroll
    for (int e = 0; e < 4; ++e)
      if (e < per) s += qv[e] * __bfloat162float(kr[lane * per + e]);
    s = warp_sum(s) * L.scale;
    if (s > m) {
      z = (m == -INFINITY) ? 0.f : z * __expf(m - s);
      m = s;
    }
    z += __expf(s - m);
  }
  if (lane == 0) {
    L.row_m[static_cast<int64_t>(h) * L.total_text + trow] = m;
    L.row_z[static_cast<int64_t>(h) * L.total_text + trow] = z;
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
    // groups of 8 text rows per video: at most total_text / 8 + one partial group per video;
    // CTAs past the last group return at once
    dim3 g1((L.total_text + 7) / 8 + L.n_videos, L.hq);
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
