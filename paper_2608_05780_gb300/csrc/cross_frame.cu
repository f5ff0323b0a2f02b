// Cross-frame cue A_ff and its timestamp-aligned evidence E_ff (Sec. 3.2,
// "Evidence Decomposition"):
//   A_ff[a-1, b] = (1 / (N_v Hq)) sum_h sum_{i in frame a} sum_{j in frame b} P^h_ij,  b < a,
//   E_ff[t]      = ( sum_{b<t} A_ff[t-1, b] + sum_{a>t} A_ff[a-1, t] ) / 2.
//
// The probe, run with cross-frame partials on, leaves for every visual row i,
// kept kv tile p of its row tile and key span f of that tile (min(N_v, 64)
// keys, so a key frame is one or two spans) the value m + log2(sum of the
// row's 2^(s scale log2e - m) over the span's keys), m the running max it used
// there. The span's share of the row's softmax (Eq. 11) is then
// 2^(value - LSE_i log2 e), with LSE the probe's final normaliser.
//
// cross_frame_pairs_kernel: one CTA per (visual row tile, 8 kept tiles), one
// thread per row. A thread sums its row's shares over the heads, the CTA sums
// them over the N_v rows of each query frame (shuffles, then a shared-memory
// step for N_v > 32), and the first row of the frame writes A_ff[a-1, b]. A
// frame pair (a, b) belongs to exactly one (row tile, kept tile), so every
// entry has one writer and a fixed summation order (deterministic).
// e_ff_kernel: one CTA per (32 frames, video) forms E_ff from A_ff: the
// received attention by column sums (8 warps over the rows, coalesced), the
// given attention by row sums (a warp per row), partials added in a fixed order.
#include <cstdint>
#include <cuda_runtime.h>

#include "evisel_internal.h"
#include "sm103_ptx.cuh"

namespace evisel {
namespace {

constexpr int kKvPerCta = 8;
constexpr unsigned kFull = 0xffffffffu;

template <int TILE>
__global__ void __launch_bounds__(TILE) cross_frame_pairs_kernel(const __grid_constant__ CrossFrameLaunch L) {
  extern __shared__ float lse2[];                  // [hq][TILE]: each thread's own column
  __shared__ float red[TILE / 32];
  const VisRow R = L.rows[blockIdx.x];
  const int k0 = blockIdx.y * kKvPerCta;
  if (k0 >= R.kv_count) return;                    // uniform over the CTA
  const int k1 = min(R.kv_count, k0 + kKvPerCta);
  const VideoInfo vi = L.videos[R.video];
  const int npf = L.tokens_per_frame, fpt = L.fpt;
  const int T = vi.n_vis / npf;
  const int row = threadIdx.x, lane = row & 31, warp = row >> 5;
  const bool valid = row < R.q_len;
  for (int h = 0; h < L.hq; ++h)
    lse2[h * TILE + row] = valid ? L.lse[static_cast<int64_t>(h) * L.n_tok + R.q_start + row] * 1.4426950408889634f
                                 : 0.f;
  const int a = (R.row_tile * TILE + row) / npf;  // the row's frame (video-local)
  const float inv_norm = 1.f / static_cast<float>(npf * L.hq);
  const int64_t head_stride = static_cast<int64_t>(L.nnz) * fpt * TILE;
  float* aff = L.aff + L.aff_off[R.video];
  for (int k = k0; k < k1; ++k) {
    const int p = R.kv_begin + k;
    const int c_tile = (L.kv[p].start - vi.vis_start) / TILE;
    const int spf = L.spans_per_frame;
    float v = 0.f;
    for (int f = 0; f < fpt; ++f) {
      if (valid) {
        const float* src = L.fspill + (static_cast<int64_t>(p) * fpt + f) * TILE + row;
#pragma unroll 4
        for (int h = 0; h < L.hq; ++h) v += ptx::ex2(__ldcs(src + h * head_stride) - lse2[h * TILE + row]);
      }
      if ((f + 1) % spf != 0) continue;            // the key frame has another span
      const int b = (c_tile * fpt + f) / spf;      // key frame (video-local)
      // Sum over the N_v rows of the query frame (aligned groups of threads).
      const int w = npf < 32 ? npf : 32;
      for (int off = w / 2; off > 0; off >>= 1) v += __shfl_xor_sync(kFull, v, off);
      if (npf > 32) {
        if (lane == 0) red[warp] = v;
        __syncthreads();
        if (row % npf == 0) {
          float t = 0.f;
          for (int ww = warp; ww < warp + npf / 32; ++ww) t += red[ww];
          v = t;
        }
        __syncthreads();
      }
      if (row % npf == 0 && b < a && a < T) {
        float* dst = aff + static_cast<int64_t>(a - 1) * (T - 1) + b;
        const float val = v * inv_norm;
        *dst = L.accumulate ? *dst + val : val;
      }
      v = 0.f;
    }
  }
}

__global__ void __launch_bounds__(256) e_ff_kernel(const __grid_constant__ CrossFrameLaunch L) {
  __shared__ float part[8][33];
  __shared__ float give[32];
  const VideoInfo vi = L.videos[blockIdx.y];
  const int T = vi.n_vis / L.tokens_per_frame;
  const int t0 = blockIdx.x * 32;
  if (t0 >= T) return;                             // uniform over the CTA
  const float* A = L.aff + L.aff_off[blockIdx.y];  // [(T-1), (T-1)]
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int t = t0 + lane;
  // Received: column t over the rows of frames a > t (row index a - 1 >= t).
  float recv = 0.f;
  for (int ra = t0 + warp; ra <= T - 2; ra += 8)
    if (t <= T - 2 && ra >= t) recv += A[static_cast<int64_t>(ra) * (T - 1) + t];
  part[warp][lane] = recv;
  // Given: row t - 1 over the frames b < t.
  for (int tt = warp; tt < 32; tt += 8) {
    const int tg = t0 + tt;
    float g = 0.f;
    if (tg >= 1 && tg < T)
      for (int b = lane; b < tg; b += 32) g += A[static_cast<int64_t>(tg - 1) * (T - 1) + b];
    for (int off = 16; off > 0; off >>= 1) g += __shfl_xor_sync(kFull, g, off);
    if (lane == 0) give[tt] = g;
  }
  __syncthreads();
  if (warp == 0 && t < T) {
    float r = 0.f;
#pragma unroll
    for (int w = 0; w < 8; ++w) r += part[w][lane];
    L.eff[vi.frame_off + t] = 0.5f * (give[lane] + r);
  }
}

template <int TILE>
cudaError_t launch_pairs(const CrossFrameLaunch& L, cudaStream_t stream) {
  const size_t smem = static_cast<size_t>(L.hq) * TILE * sizeof(float);
  auto kern = cross_frame_pairs_kernel<TILE>;
  if (smem > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    if (e != cudaSuccess) return e;
  }
  dim3 grid(L.n_rows, (L.max_kv + kKvPerCta - 1) / kKvPerCta);
  kern<<<grid, TILE, smem, stream>>>(L);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_cross_frame(const CrossFrameLaunch& L, cudaStream_t stream) {
  if (L.n_rows > 0 && L.max_kv > 0) {
    cudaError_t e = L.tile == 128 ? launch_pairs<128>(L, stream)
                  : L.tile == 64  ? launch_pairs<64>(L, stream)
                                  : cudaErrorInvalidValue;
    if (e != cudaSuccess) return e;
  }
  if (L.eff && L.n_videos > 0 && L.max_frames > 0) {
    dim3 grid((L.max_frames + 31) / 32, L.n_videos);
    e_ff_kernel<<<grid, 256, 0, stream>>>(L);
    return cudaGetLastError();
  }
  return cudaSuccess;
}

}  // namespace evisel
