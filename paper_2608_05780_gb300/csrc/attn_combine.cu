// Merge of split-KV partials of the text row tiles.
//
// A text row tile attends to every visual tile and to its causal text tiles,
// many more kv tiles than any visual row tile, so its kv range is split over
// several CTAs. Each split leaves, per row, an unnormalised accumulator O_s, its
// running max m_s (log2 units) and row sum l_s. With M = max_s m_s and
// w_s = 2^(m_s - M):  O = sum_s w_s O_s / sum_s w_s l_s,
// LSE = (M + log2 sum_s w_s l_s) ln 2 -- the same softmax normalisation as a
// single pass over the whole row (Eq. 11).
#include <cstdint>
#include <cuda_runtime.h>

#include "evisel_internal.h"

namespace evisel {
namespace {

constexpr int kRows = 128;
constexpr int kRowsPerBlock = 8;

__device__ __forceinline__ uint32_t pack2(float lo, float hi) {
  uint32_t r;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
  return r;
}

// grid.x = groups * (128 / kRowsPerBlock); block = kRowsPerBlock rows x (d / 4) threads.
__global__ void attn_combine_kernel(const __grid_constant__ CombineLaunch L) {
  const int blocks_per_group = kRows / kRowsPerBlock;
  const int gi = blockIdx.x / blocks_per_group;
  const int row = (blockIdx.x % blocks_per_group) * kRowsPerBlock + threadIdx.y;
  const int c4 = threadIdx.x;                      // float4 column
  const CombineGroup g = L.groups[gi];
  const int hp = row / L.tile;
  const int row_local = row % L.tile;
  const int gq = L.hq / L.hkv;
  const bool head_ok = hp == 0 || ((g.head + 1) < L.hq && (g.head + 1) / gq == g.head / gq);
  if (!head_ok || row_local >= g.q_len) return;
  const int head = g.head + hp;
  const int qpos = g.q_start + row_local;

  float mmax = -INFINITY;
  for (int s = 0; s < g.nsplit; ++s)
    mmax = fmaxf(mmax, L.part_ml[(g.part0 + static_cast<int64_t>(s) * g.stride) * kRows + row].x);
  const float msafe = mmax == -INFINITY ? 0.f : mmax;
  float lsum = 0.f;
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  for (int s = 0; s < g.nsplit; ++s) {
    const int64_t slot = g.part0 + static_cast<int64_t>(s) * g.stride;
    const float2 ml = L.part_ml[slot * kRows + row];
    const float w = exp2f(ml.x - msafe);
    lsum += w * ml.y;
    const float4 o = reinterpret_cast<const float4*>(L.part_o + (slot * kRows + row) * L.head_dim)[c4];
    acc.x += w * o.x; acc.y += w * o.y; acc.z += w * o.z; acc.w += w * o.w;
  }
  const float inv = lsum > 0.f ? 1.f / lsum : 0.f;
  uint2 packed;
  packed.x = pack2(acc.x * inv, acc.y * inv);
  packed.y = pack2(acc.z * inv, acc.w * inv);
  reinterpret_cast<uint2*>(static_cast<uint16_t*>(L.o) + ((int64_t)qpos * L.hq + head) * L.head_dim)[c4] = packed;
  if (c4 == 0) L.lse[(int64_t)head * L.n_tok + qpos] = (mmax + log2f(lsum)) * 0.69314718055994531f;
}

}  // namespace

cudaError_t launch_attn_combine(const CombineLaunch& L, cudaStream_t stream) {
  if (L.n_groups == 0) return cudaSuccess;
  dim3 block(L.head_dim / 4, kRowsPerBlock);
  attn_combine_kernel<<<L.n_groups * (kRows / kRowsPerBlock), block, 0, stream>>>(L);
  return cudaGetLastError();
}

}  // namespace evisel
