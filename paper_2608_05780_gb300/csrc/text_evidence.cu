// Text-row evidence by recompute (Sec. 3.2, "Evidence Decomposition"), the
// variant of the evidence pass that needs no logit spill:
//   tok[h, m]   = sum_{text rows i} exp(s_im - LSE_i),  s = scale q_i k_m (Eq. 8),
//   frame[h, t] = sum_{m in frame t} tok[h, m],
// with LSE the probe's saved row normaliser (Eq. 11). Text rows attend to
// every visual key of their video (dense causal), so every (text row, visual
// key) pair enters.
//
// One CTA per (128 visual keys of a video, KV group), 192 threads:
//   warp 4  TMA: the key tile K_g once, then Q_h of each text tile of the
//           video for the group's heads, into a 2-deep ring (128B swizzle)
//   warp 5  MMA: S^T = K_g Q_h^T (tcgen05, bf16 in, fp32 in TMEM; M = 128
//           keys, N = 128 text rows, 64 for a text tile of at most 64 rows)
//           into a double-buffered TMEM tile
//   warps 0-3  one thread per key (TMEM lane): adds exp2(s scale log2e -
//           LSE log2e) over the 128 text-row columns of its lane (LSE of the
//           step's text rows staged in shared memory), so no reduction
//           across threads is needed for the token map; after a head's last
//           text tile it writes tok[h, key] and the frame sums (shuffles, then
//           shared memory for N_v > 32).
// Every (head, key) has one writer and a fixed summation order. Every wait is
// bounded; on timeout the CTA records EVISEL_ETIMEOUT and drains its copies
// and MMAs. The key warps never leave their loop early (they meet at a named
// barrier every step); after a timeout they only skip the work.
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
constexpr int kBarKeys = 1;                      // named barrier of the 128 key threads

template <int D>
struct TeCfg {
  static constexpr int KB = D / 64;
  static constexpr int TILE_BYTES = kRows * D * 2;
  static constexpr int BLOCK = kRows * 128;
  static constexpr int QS = 2;
  static constexpr int OFF_K = 0;
  static constexpr int OFF_Q = TILE_BYTES;
  static constexpr int OFF_BAR = OFF_Q + QS * TILE_BYTES;
  static constexpr int B_KF = 0, B_QF = 1, B_QE = 1 + QS, B_SF = 1 + 2 * QS, B_SE = B_SF + 2, B_DRAIN = B_SE + 2;
  static constexpr int N_BARS = B_DRAIN + 1;
  static constexpr int OFF_LSE = OFF_BAR + N_BARS * 8;          // [2][128] fp32
  static constexpr int OFF_RED = OFF_LSE + 2 * kRows * 4;      // [4] fp32 per frame reduction
  static constexpr int OFF_MISC = OFF_RED + 4 * 4;
  static constexpr int SMEM_BYTES = OFF_MISC + 16 + 1024;
  static constexpr int TMEM_COLS = 256;
};

__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag) {
  const bool ok = ptx::mbar_wait(bar, parity, abort_flag, kWaitTimeoutNs);
  return __all_sync(0xffffffffu, ok);
}

__device__ __forceinline__ void record_failure(volatile int* abort_flag, int* status) {
  *abort_flag = 1;
  atomicExch(status, kStatusTimeout);
}

template <int D>
__global__ void __launch_bounds__(kThreads, 2) text_evidence_kernel(const __grid_constant__ TextEvidenceLaunch L) {
  using C = TeCfg<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t sbase = ptx::smem_addr(smem);
  auto bar = [&](int i) { return sbase + C::OFF_BAR + 8u * i; };
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + C::OFF_MISC);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::OFF_MISC + 4);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const EvChunk ch = L.chunks[blockIdx.x];
  const VideoInfo vi = L.videos[ch.video];
  const int g = blockIdx.y;                        // KV group
  const int gq = L.hq / L.hkv;
  const int n_tt = (vi.n_text + kRows - 1) / kRows;   // text tiles of the video
  const int n_steps = gq * n_tt;                   // step t: head g * gq + t / n_tt, text tile t % n_tt
  const int text0 = vi.vis_start + vi.n_vis;       // first text token

  if (threadIdx.x == 0) {
    for (int i = 0; i < C::N_BARS; ++i)
      ptx::mbar_init(bar(i), (i == C::B_SE || i == C::B_SE + 1) ? kRows : 1u);
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
    const uint64_t pol_q = ptx::l2_policy_evict_last();   // the video's text Q is read by every key tile
    const uint64_t pol_k = ptx::l2_policy_evict_first();  // a key tile is read once per KV group
    uint32_t leader = 0;
    int issued = 0;
    bool ok = true;
    if (n_steps > 0) {
      if (ptx::elect_one(leader)) {
        ptx::mbar_arrive_expect_tx(bar(C::B_KF), C::TILE_BYTES);
#pragma unroll
        for (int kb = 0; kb < C::KB; ++kb)
          ptx::tma_load_3d(sbase + C::OFF_K + kb * C::BLOCK, &L.tm_k, bar(C::B_KF), kb * 64, g,
                           vi.vis_start + ch.col0, pol_k);
      }
      __syncwarp();
    }
    for (int t = 0; ok && t < n_steps; ++t) {
      const int qs = t % C::QS;
      if (t >= C::QS && !warp_wait(bar(C::B_QE + qs), ((t - C::QS) / C::QS) & 1, abort_flag)) {
        ok = false;
        break;
      }
      const int h = g * gq + t / n_tt, tt = t % n_tt;
      if (ptx::elect_one(leader)) {
        ptx::mbar_arrive_expect_tx(bar(C::B_QF + qs), C::TILE_BYTES);
#pragma unroll
        for (int kb = 0; kb < C::KB; ++kb)
          ptx::tma_load_3d(sbase + C::OFF_Q + qs * C::TILE_BYTES + kb * C::BLOCK, &L.tm_q, bar(C::B_QF + qs),
                           kb * 64, h, text0 + tt * kRows, pol_q);
      }
      __syncwarp();
      ++issued;
    }
    if (!ok && lane == 0) record_failure(abort_flag, L.status);
    const volatile int never = 0;
    if (n_steps > 0) ptx::mbar_wait(bar(C::B_KF), 0, &never, kWaitTimeoutNs);
    for (int s = 0; s < C::QS && s < issued; ++s)
      ptx::mbar_wait(bar(C::B_QF + s), ((issued - 1 - s) / C::QS) & 1, &never, kWaitTimeoutNs);
  } else if (warp == kWarpMma) {
    constexpr uint32_t kIdesc = ptx::idesc_bf16_f32(kRows, kRows, false, false);
    // A text tile with at most 64 rows (the last, ragged tile of a video)
    // takes an N = 64 MMA; the key threads read only those columns.
    constexpr uint32_t kIdescHalf = ptx::idesc_bf16_f32(kRows, 64, false, false);
    uint32_t leader = 0;
    int first_leader = -1;
    bool same = true, issued = false, ok = true;
    if (n_steps > 0 && !warp_wait(bar(C::B_KF), 0, abort_flag)) ok = false;
    for (int t = 0; ok && t < n_steps; ++t) {
      const int b = t % 2;
      if (!warp_wait(bar(C::B_QF + t % C::QS), (t / C::QS) & 1, abort_flag) ||
          (t >= 2 && !warp_wait(bar(C::B_SE + b), ((t - 2) / 2) & 1, abort_flag))) {
        ok = false;
        break;
      }
      ptx::tc_fence_after();
      const bool me = ptx::elect_one(leader);
      if (first_leader < 0) first_leader = static_cast<int>(leader);
      same = same && static_cast<int>(leader) == first_leader;
      const uint32_t idesc = vi.n_text - (t % n_tt) * kRows <= 64 ? kIdescHalf : kIdesc;
      if (me && same) {
        const uint32_t kbase = sbase + C::OFF_K;
        const uint32_t qbase = sbase + C::OFF_Q + (t % C::QS) * C::TILE_BYTES;
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint64_t a = ptx::sdesc_sw128(kbase + (kk / 4) * C::BLOCK + (kk % 4) * 32, 16, 1024);
          const uint64_t bd = ptx::sdesc_sw128(qbase + (kk / 4) * C::BLOCK + (kk % 4) * 32, 16, 1024);
          ptx::mma_ss(tmem + b * kRows, a, bd, idesc, kk > 0 ? 1u : 0u);
        }
        ptx::mma_commit(bar(C::B_SF + b));
        ptx::mma_commit(bar(C::B_QE + t % C::QS));
      }
      __syncwarp();
      issued = true;
      ok = same;
      if (!ok) break;
    }
    if (!ok) {
      if (lane == 0) record_failure(abort_flag, L.status);
      if (issued && lane == first_leader) {
        const volatile int never = 0;
        ptx::mma_commit(bar(C::B_DRAIN));
        ptx::mbar_wait(bar(C::B_DRAIN), 0, &never, kWaitTimeoutNs);
      }
    }
    __syncwarp();
  } else {
    // Key threads: thread k = key ch.col0 + k of the video = TMEM lane k.
    const int key = threadIdx.x;
    const int npf = L.tokens_per_frame;
    const bool key_ok = ch.col0 + key < vi.n_vis;
    const uint32_t tbase = tmem + (static_cast<uint32_t>(warp * 32) << 16);
    float* lse_s = reinterpret_cast<float*>(smem + C::OFF_LSE);
    float* red = reinterpret_cast<float*>(smem + C::OFF_RED);
    bool ok = true;
    for (int hh = 0; hh < gq; ++hh) {
      const int h = g * gq + hh;
      float acc = 0.f;
      for (int tt = 0; tt < n_tt; ++tt) {
        const int t = hh * n_tt + tt, b = t % 2;
        // The step's text-row LSEs (log2 units; +inf past the video's text rows: those columns add 0).
        const int row = tt * kRows + key;
        lse_s[b * kRows + key] =
            row < vi.n_text ? __ldg(L.lse + static_cast<int64_t>(h) * L.n_tok + text0 + row) * 1.4426950408889634f
                            : INFINITY;
        ptx::bar_sync(kBarKeys, kRows);
        ok = ok && warp_wait(bar(C::B_SF + b), (t / 2) & 1, abort_flag);
        if (ok) {
          ptx::tc_fence_after();
          const float* lrow = lse_s + b * kRows;
          const int valid = vi.n_text - tt * kRows;   // text rows in this tile; columns past them add 0
#pragma unroll
          for (int c0 = 0; c0 < kRows; c0 += 64) {
            if (c0 >= valid) break;                    // a 64-column half of padding rows only
            uint32_t r0[32], r1[32];
            ptx::tmem_ld32(tbase + b * kRows + c0, r0);
            ptx::tmem_ld32(tbase + b * kRows + c0 + 32, r1);
            ptx::tmem_wait_ld();
            float a0 = 0.f, a1 = 0.f;
#pragma unroll
            for (int e = 0; e < 32; ++e) {
              a0 += ptx::ex2(__uint_as_float(r0[e]) * L.scale_log2 - lrow[c0 + e]);
              a1 += ptx::ex2(__uint_as_float(r1[e]) * L.scale_log2 - lrow[c0 + 32 + e]);
            }
            acc += a0 + a1;
          }
          ptx::tc_fence_before();
        }
        ptx::mbar_arrive(bar(C::B_SE + b));
      }
      // Token map and frame sums of head h (a video without text rows writes 0).
      float* tok = L.tok + static_cast<int64_t>(h) * L.total_vis + vi.vis_off + ch.col0;
      if (ok && key_ok) tok[key] = L.accumulate ? tok[key] + acc : acc;
      float f = key_ok ? acc : 0.f;
      const int w = npf < 32 ? npf : 32;
      for (int off = w / 2; off > 0; off >>= 1) f += __shfl_xor_sync(0xffffffffu, f, off);
      if (npf > 32) {
        if (lane == 0) red[warp] = f;
        ptx::bar_sync(kBarKeys, kRows);
        if (key % npf == 0) {
          float s = 0.f;
          for (int ww = warp; ww < warp + npf / 32; ++ww) s += red[ww];
          f = s;
        }
        ptx::bar_sync(kBarKeys, kRows);
      }
      if (ok && key_ok && key % npf == 0) {
        float* fr = L.frame + static_cast<int64_t>(h) * L.total_frames + vi.frame_off + (ch.col0 + key) / npf;
        *fr = L.accumulate ? *fr + f : f;
      }
    }
    if (!ok && key == 0) record_failure(abort_flag, L.status);
  }
  ptx::tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc<C::TMEM_COLS>(tmem);
  }
}

template <int D>
cudaError_t launch_d(const TextEvidenceLaunch& L, cudaStream_t stream) {
  using C = TeCfg<D>;
  auto kern = text_evidence_kernel<D>;
  static PerDeviceAttr smem_once;
  cudaError_t e = raise_smem_limit(smem_once, reinterpret_cast<const void*>(kern), C::SMEM_BYTES);
  if (e != cudaSuccess) return e;
  dim3 grid(L.n_chunks, L.hkv);
  kern<<<grid, kThreads, C::SMEM_BYTES, stream>>>(L);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_text_evidence(const TextEvidenceLaunch& L, cudaStream_t stream) {
  if (L.n_chunks == 0) return cudaSuccess;
  if (L.head_dim == 128) return launch_d<128>(L, stream);
  if (L.head_dim == 64) return launch_d<64>(L, stream);
  return cudaErrorInvalidValue;
}

}  // namespace evisel
