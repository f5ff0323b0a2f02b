// Intra-frame cue A_if (Sec. 3.2, "Evidence Decomposition"): for every frame
// the head-averaged token-level causal attention among its N_v visual tokens,
//   A_if[t, i, j] = (1 / Hq) sum_h exp(s^h_ij - LSE^h_i),  j <= i  (0 above),
// re-formed from the probe's saved LSE (the row's full softmax normaliser,
// Eq. 11) and recomputed logits s = q k^T scale (Eq. 8). A frame's keys are
// the row's own frame, which every mask keeps (the diagonal tile), so the
// mask enters only through the LSE.
//
// One CTA per 128-token block of a video's visual rows (grid: row blocks x
// videos) loops over all query heads:
//   warp 4  TMA: Q_h per head into a 2-deep ring, K_g per KV group into a
//           2-deep ring (128B swizzle, no multicast)
//   warp 5  MMA: S_h = Q_h K_g^T (tcgen05, bf16 in, fp32 in TMEM) into a
//           double-buffered TMEM S; one elected lane issues, the warp walks
//           the heads on warp-uniform values
//   warps 0-3  one thread per row (TMEM lane): reads its frame's window of
//           S_h, adds exp2(s scale log2e - LSE log2e) over its frame keys
//           j <= i, and after the last head stores sum / Hq.
// Heads are summed in a fixed order, so the result is deterministic. Every
// wait is bounded; on timeout the CTA records EVISEL_ETIMEOUT, drains its own
// copies and MMAs and exits.
#include <cstdint>
#include <cuda_runtime.h>

#include "evisel_internal.h"
#include "sm103_ptx.cuh"

namespace evisel {
namespace {

constexpr int kRows = 128;
constexpr int kThreads = 192;
constexpr int kWarpProducer = 4;
constexpr int kWarpMma = 5;

template <int D>
struct IfCfg {
  static constexpr int KB = D / 64;              // 128-byte swizzle column blocks along d
  static constexpr int TILE_BYTES = kRows * D * 2;
  static constexpr int BLOCK = kRows * 128;      // one column block of a 128-row tile
  static constexpr int OFF_Q = 0;                // 2 stages
  static constexpr int OFF_K = OFF_Q + 2 * TILE_BYTES;   // 2 stages
  static constexpr int OFF_BAR = OFF_K + 2 * TILE_BYTES;
  static constexpr int B_QF = 0, B_QE = 2, B_KF = 4, B_KE = 6, B_SF = 8, B_SE = 10, B_DRAIN = 12;
  static constexpr int N_BARS = 13;
  static constexpr int OFF_MISC = OFF_BAR + N_BARS * 8;
  static constexpr int SMEM_BYTES = OFF_MISC + 16 + 1024;
  static constexpr int TMEM_COLS = 256;          // S double buffer
  static_assert(SMEM_BYTES <= 232448, "shared memory budget");
};

__device__ __forceinline__ void record_failure(volatile int* abort_flag, int* status) {
  *abort_flag = 1;
  atomicExch(status, kStatusTimeout);
}

__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag) {
  const bool ok = ptx::mbar_wait(bar, parity, abort_flag, kWaitTimeoutNs);
  return __all_sync(0xffffffffu, ok);
}

template <int D>
__device__ __forceinline__ void producer(const IntraFrameLaunch& L, int row0, uint32_t sbase, volatile int* abort_flag) {
  using C = IfCfg<D>;
  auto bar = [&](int i) { return sbase + C::OFF_BAR + 8u * i; };
  const int gq = L.hq / L.hkv;
  const uint64_t pol_q = ptx::l2_policy_evict_first();
  const uint64_t pol_k = ptx::l2_policy_evict_last();
  uint32_t leader = 0;
  int q_issued = 0, k_issued = 0;
  bool ok = true;
  for (int h = 0; ok && h < L.hq; ++h) {
    const int g = h / gq;
    if (h % gq == 0) {   // first head of a KV group: its K tile into stage g % 2
      if (g >= 2 && !warp_wait(bar(C::B_KE + g % 2), ((g - 2) / 2) & 1, abort_flag)) {
        ok = false;
        break;
      }
      if (ptx::elect_one(leader)) {
        ptx::mbar_arrive_expect_tx(bar(C::B_KF + g % 2), C::TILE_BYTES);
#pragma unroll
        for (int kb = 0; kb < C::KB; ++kb)
          ptx::tma_load_3d(sbase + C::OFF_K + (g % 2) * C::TILE_BYTES + kb * C::BLOCK, &L.tm_k, bar(C::B_KF + g % 2),
                           kb * 64, g, row0, pol_k);
      }
      __syncwarp();
      ++k_issued;
    }
    if (h >= 2 && !warp_wait(bar(C::B_QE + h % 2), ((h - 2) / 2) & 1, abort_flag)) {
      ok = false;
      break;
    }
    if (ptx::elect_one(leader)) {
      ptx::mbar_arrive_expect_tx(bar(C::B_QF + h % 2), C::TILE_BYTES);
#pragma unroll
      for (int kb = 0; kb < C::KB; ++kb)
        ptx::tma_load_3d(sbase + C::OFF_Q + (h % 2) * C::TILE_BYTES + kb * C::BLOCK, &L.tm_q, bar(C::B_QF + h % 2),
                         kb * 64, h, row0, pol_q);
    }
    __syncwarp();
    ++q_issued;
  }
  if (!ok && (threadIdx.x & 31) == 0) record_failure(abort_flag, L.status);
  // Drain: the last phase issued into each stage, so that no copy is in flight at exit.
  const volatile int never = 0;
  for (int s = 0; s < 2; ++s) {
    if (s < q_issued) ptx::mbar_wait(bar(C::B_QF + s), (((q_issued - 1 - s) / 2)) & 1, &never, kWaitTimeoutNs);
    if (s < k_issued) ptx::mbar_wait(bar(C::B_KF + s), (((k_issued - 1 - s) / 2)) & 1, &never, kWaitTimeoutNs);
  }
}

template <int D>
__device__ __forceinline__ void mma_issuer(const IntraFrameLaunch& L, uint32_t sbase, uint32_t tmem,
                                           volatile int* abort_flag) {
  using C = IfCfg<D>;
  auto bar = [&](int i) { return sbase + C::OFF_BAR + 8u * i; };
  constexpr uint32_t kIdesc = ptx::idesc_bf16_f32(kRows, kRows, false, false);
  const int gq = L.hq / L.hkv;
  uint32_t leader = 0;
  int first_leader = -1;
  bool same = true;
  bool issued = false;
  bool ok = true;
  for (int h = 0; ok && h < L.hq; ++h) {
    const int g = h / gq;
    const int b = h % 2;
    // Q_h and K_g landed; S buffer b was read by the rows (head h - 2).
    if ((h % gq == 0 && !warp_wait(bar(C::B_KF + g % 2), (g / 2) & 1, abort_flag)) ||
        !warp_wait(bar(C::B_QF + b), (h / 2) & 1, abort_flag) ||
        (h >= 2 && !warp_wait(bar(C::B_SE + b), ((h - 2) / 2) & 1, abort_flag))) {
      ok = false;
      break;
    }
    ptx::tc_fence_after();
    const bool me = ptx::elect_one(leader);
    if (first_leader < 0) first_leader = static_cast<int>(leader);
    same = same && static_cast<int>(leader) == first_leader;
    if (me && same) {
      const uint32_t qbase = sbase + C::OFF_Q + b * C::TILE_BYTES;
      const uint32_t kbase = sbase + C::OFF_K + (g % 2) * C::TILE_BYTES;
#pragma unroll
      for (int kk = 0; kk < D / 16; ++kk) {
        const uint64_t a = ptx::sdesc_sw128(qbase + (kk / 4) * C::BLOCK + (kk % 4) * 32, 16, 1024);
        const uint64_t bd = ptx::sdesc_sw128(kbase + (kk / 4) * C::BLOCK + (kk % 4) * 32, 16, 1024);
        ptx::mma_ss(tmem + b * kRows, a, bd, kIdesc, kk > 0 ? 1u : 0u);
      }
      ptx::mma_commit(bar(C::B_SF + b));
      ptx::mma_commit(bar(C::B_QE + b));
      if (h % gq == gq - 1) ptx::mma_commit(bar(C::B_KE + g % 2));
    }
    __syncwarp();
    issued = true;
    ok = same;
  }
  const int lane = threadIdx.x & 31;
  if (!ok) {
    if (lane == 0) record_failure(abort_flag, L.status);
    if (issued && lane == first_leader) {
      const volatile int never = 0;
      ptx::mma_commit(bar(C::B_DRAIN));
      ptx::mbar_wait(bar(C::B_DRAIN), 0, &never, kWaitTimeoutNs);
    }
  }
  __syncwarp();
}

// The rows: W = max(32, N_v) columns of S around each warp's frames.
template <int D, int W>
__device__ __forceinline__ void rows(const IntraFrameLaunch& L, const VideoInfo& vi, int rb, uint32_t sbase,
                                     uint32_t tmem_base, volatile int* abort_flag) {
  using C = IfCfg<D>;
  auto bar = [&](int i) { return sbase + C::OFF_BAR + 8u * i; };
  const int warp = threadIdx.x >> 5;
  const int row = threadIdx.x;                       // row within the block = TMEM lane
  const int npf = L.tokens_per_frame;
  const int col_base = ((32 * warp) / W) * W;        // the warp's window of key columns
  const int f0 = (row / npf) * npf;                  // first key of the row's frame (block-local)
  const int pos = rb * kRows + row;                  // visual position within the video
  const bool row_ok = pos < vi.n_vis;
  const uint32_t tmem = tmem_base + (static_cast<uint32_t>(warp * 32) << 16) + col_base;
  const float* lse_row = L.lse + vi.vis_start + pos;
  float acc[W];
#pragma unroll
  for (int c = 0; c < W; ++c) acc[c] = 0.f;
  bool ok = true;
  for (int h = 0; h < L.hq; ++h) {
    const int b = h % 2;
    const float m = row_ok ? __ldg(lse_row + static_cast<int64_t>(h) * L.n_tok) * 1.4426950408889634f : 0.f;
    if (!warp_wait(bar(C::B_SF + b), (h / 2) & 1, abort_flag)) {
      ok = false;
      break;
    }
    ptx::tc_fence_after();
#pragma unroll
    for (int c0 = 0; c0 < W; c0 += 32) {
      uint32_t r[32];
      ptx::tmem_ld32(tmem + b * kRows + c0, r);
      ptx::tmem_wait_ld();
#pragma unroll
      for (int e = 0; e < 32; ++e) {
        const int col = col_base + c0 + e;           // key column within the block
        if (col >= f0 && col <= row) acc[c0 + e] += ptx::ex2(__uint_as_float(r[e]) * L.scale_log2 - m);
      }
    }
    ptx::tc_fence_before();
    ptx::mbar_arrive(bar(C::B_SE + b));
  }
  if (!ok) {
    record_failure(abort_flag, L.status);
    return;
  }
  if (!row_ok) return;
  // Row i = row - f0 of frame (frame_off + (pos - (row - f0)) / npf): keys j = col - f0.
  const int64_t frame = vi.frame_off + (pos - (row - f0)) / npf;
  float* dst = L.aif + (frame * npf + (row - f0)) * npf;
  const float inv_h = 1.f / static_cast<float>(L.hq);
#pragma unroll
  for (int c = 0; c < W; ++c) {
    const int j = col_base + c - f0;
    if (j >= 0 && j < npf) dst[j] = L.accumulate ? dst[j] + acc[c] * inv_h : acc[c] * inv_h;
  }
}

template <int D, int W>
__global__ void __launch_bounds__(kThreads, 1) intra_frame_kernel(const __grid_constant__ IntraFrameLaunch L) {
  using C = IfCfg<D>;
  const VideoInfo vi = L.videos[blockIdx.y];
  const int rb = blockIdx.x;
  if (rb * kRows >= vi.n_vis) return;                // this video has fewer row blocks
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t sbase = ptx::smem_addr(smem);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + C::OFF_MISC);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::OFF_MISC + 4);
  const int warp = threadIdx.x >> 5;
  if (threadIdx.x == 0) {
    for (int i = 0; i < C::N_BARS; ++i)
      ptx::mbar_init(sbase + C::OFF_BAR + 8u * i, (i == C::B_SE || i == C::B_SE + 1) ? kRows : 1u);
    *abort_flag = 0;
    ptx::fence_mbar_init();
  }
  if (warp == 0) {
    ptx::tmem_alloc<C::TMEM_COLS>(ptx::smem_addr(tmem_slot));
    ptx::tmem_relinquish();
  }
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  if (warp == kWarpProducer) {
    producer<D>(L, vi.vis_start + rb * kRows, sbase, abort_flag);
  } else if (warp == kWarpMma) {
    mma_issuer<D>(L, sbase, tmem, abort_flag);
  } else {
    rows<D, W>(L, vi, rb, sbase, tmem, abort_flag);
  }
  ptx::tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc<C::TMEM_COLS>(tmem);
  }
}

template <int D, int W>
cudaError_t launch_dw(const IntraFrameLaunch& L, cudaStream_t stream) {
  using C = IfCfg<D>;
  auto kern = intra_frame_kernel<D, W>;
  static bool configured = false;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM_BYTES);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  dim3 grid((L.max_vis + kRows - 1) / kRows, L.n_videos);
  kern<<<grid, kThreads, C::SMEM_BYTES, stream>>>(L);
  return cudaGetLastError();
}

template <int D>
cudaError_t launch_d(const IntraFrameLaunch& L, cudaStream_t stream) {
  if (L.tokens_per_frame <= 32) return launch_dw<D, 32>(L, stream);
  if (L.tokens_per_frame == 64) return launch_dw<D, 64>(L, stream);
  return launch_dw<D, 128>(L, stream);
}

}  // namespace

cudaError_t launch_intra_frame(const IntraFrameLaunch& L, cudaStream_t stream) {
  if (L.n_videos == 0 || L.max_vis == 0) return cudaSuccess;
  if (L.head_dim == 128) return launch_d<128>(L, stream);
  if (L.head_dim == 64) return launch_d<64>(L, stream);
  return cudaErrorInvalidValue;
}

}  // namespace evisel
