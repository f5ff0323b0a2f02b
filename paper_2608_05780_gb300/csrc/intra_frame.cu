// Intra-frame cue A_if (Sec. 3.2, "Evidence Decomposition"): for every frame
// the head-averaged token-level causal attention among its N_v visual tokens,
//   A_if[t, i, j] = (1 / Hq) sum_h exp(s^h_ij - LSE^h_i),  j <= i  (0 above),
// re-formed from the probe's saved LSE (the row's full softmax normaliser,
// Eq. 11) and recomputed logits s = q k^T scale (Eq. 8). A frame's keys are
// the row's own frame, which every mask keeps (the diagonal tile), so the
// mask enters only through the LSE.
//
// Work unit: one 128-row block of a video's visual rows, all query heads.
// A persistent grid (one CTA per SM) walks the blocks b = blockIdx.x,
// blockIdx.x + gridDim.x, ...; the load and MMA pipelines run on across
// block boundaries, so only the first block of a CTA pays the pipeline fill.
//   warp 4  TMA: Q_h per (block, head) into a 4-deep ring, K_g per
//           (block, KV group) into a 2-deep ring (128B swizzle, no multicast)
//   warp 5  MMA: S = Q_h K_g^T (tcgen05, bf16 in, fp32 in TMEM) into a
//           double-buffered TMEM S; one elected lane issues, the warp walks
//           the steps on warp-uniform values
//   warps 0-3  one thread per row (TMEM lane): reads the 32-column chunks of
//           its frame's window of S that hold a key of some row of its warp,
//           adds exp2(s scale log2e - LSE log2e) for every column, and at the
//           end of the block stores sum / Hq for its frame keys j <= i (the
//           other columns, masked keys, are dropped there).
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
  static constexpr int QS = 4;                   // Q ring stages
  static constexpr int KS = 2;                   // K ring stages
  static constexpr int OFF_Q = 0;
  static constexpr int OFF_K = OFF_Q + QS * TILE_BYTES;
  static constexpr int OFF_BAR = OFF_K + KS * TILE_BYTES;
  static constexpr int B_QF = 0, B_QE = QS, B_KF = 2 * QS, B_KE = 2 * QS + KS, B_SF = 2 * QS + 2 * KS,
                       B_SE = B_SF + 2, B_DRAIN = B_SE + 2;
  static constexpr int N_BARS = B_DRAIN + 1;
  static constexpr int OFF_STAGE = OFF_BAR + N_BARS * 8;   // per warp a 32 x 33 fp32 transpose tile
  static constexpr int STAGE_PITCH = 33;
  static constexpr int OFF_MISC = OFF_STAGE + 4 * 32 * STAGE_PITCH * 4;
  static constexpr int SMEM_BYTES = OFF_MISC + 16 + 1024;
  static constexpr int TMEM_COLS = 256;          // S double buffer
  static_assert(SMEM_BYTES <= 232448, "shared memory budget");
};

// Global block index -> (video, block within the video). A CTA visits its
// blocks in increasing order, so the cursor only moves forward.
struct BlockCursor {
  int v = 0;
  int first = 0;   // global index of video v's first block
  __device__ __forceinline__ bool seek(const IntraFrameLaunch& L, int b, VideoInfo& vi, int& rb) {
    for (; v < L.n_videos; ++v) {
      vi = L.videos[v];
      const int nb = (vi.n_vis + kRows - 1) / kRows;
      if (b < first + nb) {
        rb = b - first;
        return true;
      }
      first += nb;
    }
    return false;
  }
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
__device__ __forceinline__ void producer(const IntraFrameLaunch& L, uint32_t sbase, volatile int* abort_flag) {
  using C = IfCfg<D>;
  auto bar = [&](int i) { return sbase + C::OFF_BAR + 8u * i; };
  const int gq = L.hq / L.hkv;
  const uint64_t pol_q = ptx::l2_policy_evict_first();
  const uint64_t pol_k = ptx::l2_policy_evict_last();
  uint32_t leader = 0;
  int t = 0, nk = 0;   // Q tiles and K tiles issued so far
  bool ok = true;
  BlockCursor cur;
  for (int blk = blockIdx.x; ok && blk < L.total_blocks; blk += gridDim.x) {
    VideoInfo vi;
    int rb = 0;
    if (!cur.seek(L, blk, vi, rb)) break;
    const int row0 = vi.vis_start + rb * kRows;
    for (int h = 0; h < L.hq; ++h, ++t) {
      if (h % gq == 0) {   // first head of a KV group: its K tile into stage nk % KS
        const int ks = nk % C::KS;
        if (nk >= C::KS && !warp_wait(bar(C::B_KE + ks), ((nk - C::KS) / C::KS) & 1, abort_flag)) {
          ok = false;
          break;
        }
        if (ptx::elect_one(leader)) {
          ptx::mbar_arrive_expect_tx(bar(C::B_KF + ks), C::TILE_BYTES);
#pragma unroll
          for (int kb = 0; kb < C::KB; ++kb)
            ptx::tma_load_3d(sbase + C::OFF_K + ks * C::TILE_BYTES + kb * C::BLOCK, &L.tm_k, bar(C::B_KF + ks),
                             kb * 64, h / gq, row0, pol_k);
        }
        __syncwarp();
        ++nk;
      }
      const int qs = t % C::QS;
      if (t >= C::QS && !warp_wait(bar(C::B_QE + qs), ((t - C::QS) / C::QS) & 1, abort_flag)) {
        ok = false;
        break;
      }
      if (ptx::elect_one(leader)) {
        ptx::mbar_arrive_expect_tx(bar(C::B_QF + qs), C::TILE_BYTES);
#pragma unroll
        for (int kb = 0; kb < C::KB; ++kb)
          ptx::tma_load_3d(sbase + C::OFF_Q + qs * C::TILE_BYTES + kb * C::BLOCK, &L.tm_q, bar(C::B_QF + qs),
                           kb * 64, h, row0, pol_q);
      }
      __syncwarp();
    }
  }
  if (!ok && (threadIdx.x & 31) == 0) record_failure(abort_flag, L.status);
  // Drain: the last phase issued into each stage, so that no copy is in flight at exit.
  const volatile int never = 0;
  for (int s = 0; s < C::QS && s < t; ++s)
    ptx::mbar_wait(bar(C::B_QF + s), ((t - 1 - s) / C::QS) & 1, &never, kWaitTimeoutNs);
  for (int s = 0; s < C::KS && s < nk; ++s)
    ptx::mbar_wait(bar(C::B_KF + s), ((nk - 1 - s) / C::KS) & 1, &never, kWaitTimeoutNs);
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
  int t = 0, nk = 0, ks = 0;
  const int n_blk = L.total_blocks > static_cast<int>(blockIdx.x)
                        ? (L.total_blocks - static_cast<int>(blockIdx.x) + gridDim.x - 1) / gridDim.x
                        : 0;
  for (int i = 0; ok && i < n_blk; ++i) {
    for (int h = 0; h < L.hq; ++h, ++t) {
      const int b = t % 2;
      if (h % gq == 0) {
        ks = nk % C::KS;
        if (!warp_wait(bar(C::B_KF + ks), (nk / C::KS) & 1, abort_flag)) {
          ok = false;
          break;
        }
        ++nk;
      }
      // Q tile t landed; S buffer b was read by the rows (step t - 2).
      if (!warp_wait(bar(C::B_QF + t % C::QS), (t / C::QS) & 1, abort_flag) ||
          (t >= 2 && !warp_wait(bar(C::B_SE + b), ((t - 2) / 2) & 1, abort_flag))) {
        ok = false;
        break;
      }
      ptx::tc_fence_after();
      const bool me = ptx::elect_one(leader);
      if (first_leader < 0) first_leader = static_cast<int>(leader);
      same = same && static_cast<int>(leader) == first_leader;
      if (me && same) {
        const uint32_t qbase = sbase + C::OFF_Q + (t % C::QS) * C::TILE_BYTES;
        const uint32_t kbase = sbase + C::OFF_K + ks * C::TILE_BYTES;
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint64_t a = ptx::sdesc_sw128(qbase + (kk / 4) * C::BLOCK + (kk % 4) * 32, 16, 1024);
          const uint64_t bd = ptx::sdesc_sw128(kbase + (kk / 4) * C::BLOCK + (kk % 4) * 32, 16, 1024);
          ptx::mma_ss(tmem + b * kRows, a, bd, kIdesc, kk > 0 ? 1u : 0u);
        }
        ptx::mma_commit(bar(C::B_SF + b));
        ptx::mma_commit(bar(C::B_QE + t % C::QS));
        if (h % gq == gq - 1) ptx::mma_commit(bar(C::B_KE + ks));
      }
      __syncwarp();
      issued = true;
      ok = same;
      if (!ok) break;
    }
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
__device__ __forceinline__ void rows(const IntraFrameLaunch& L, uint32_t sbase, uint32_t tmem_base,
                                     volatile int* abort_flag, float* stage_all) {
  using C = IfCfg<D>;
  auto bar = [&](int i) { return sbase + C::OFF_BAR + 8u * i; };
  const int warp = threadIdx.x >> 5;
  const int row = threadIdx.x;                       // row within the block = TMEM lane
  const int npf = L.tokens_per_frame;
  const int col_base = ((32 * warp) / W) * W;        // the warp's window of key columns
  const int f0 = (row / npf) * npf;                  // first key of the row's frame (block-local)
  const uint32_t tmem = tmem_base + (static_cast<uint32_t>(warp * 32) << 16) + col_base;
  const float inv_h = 1.f / static_cast<float>(L.hq);
  float* stage = stage_all + warp * 32 * C::STAGE_PITCH;
  // 32-column chunks of the window that hold a key of some row of this warp
  // (warp-uniform): the chunk starts at or before the warp's last row and ends
  // at or after the first frame start among its rows.
  uint32_t need = 0;
  {
    const int first_f0 = ((32 * warp) / npf) * npf;
#pragma unroll
    for (int c = 0; c < W / 32; ++c)
      if (col_base + 32 * c <= 32 * warp + 31 && col_base + 32 * c + 31 >= first_f0) need |= 1u << c;
  }
  BlockCursor cur, nxt;
  VideoInfo vi;
  int rb = 0;
  bool have = static_cast<int>(blockIdx.x) < L.total_blocks && cur.seek(L, blockIdx.x, vi, rb);
  // LSE of (block, head): the value for the next step is loaded one step ahead.
  auto lse_at = [&](const VideoInfo& v, int r, int h) -> float {
    const int pos = r * kRows + row;
    return pos < v.n_vis ? __ldg(L.lse + static_cast<int64_t>(h) * L.n_tok + v.vis_start + pos) : 0.f;
  };
  float m_next = have ? lse_at(vi, rb, 0) : 0.f;
  int t = 0;
  bool ok = true;
  for (int blk = blockIdx.x; have; blk += gridDim.x) {
    VideoInfo vn;
    int rbn = 0;
    const bool more = blk + static_cast<int>(gridDim.x) < L.total_blocks &&
                      nxt.seek(L, blk + static_cast<int>(gridDim.x), vn, rbn);
    float acc[W];
#pragma unroll
    for (int c = 0; c < W; ++c) acc[c] = 0.f;
    for (int h = 0; h < L.hq; ++h, ++t) {
      const int b = t % 2;
      const float m = m_next * 1.4426950408889634f;
      if (h + 1 < L.hq) m_next = lse_at(vi, rb, h + 1);
      else if (more) m_next = lse_at(vn, rbn, 0);
      if (!warp_wait(bar(C::B_SF + b), (t / 2) & 1, abort_flag)) {
        ok = false;
        break;
      }
      ptx::tc_fence_after();
      // Up to two 32-column chunks in flight per wait (64 registers).
      constexpr int G = W / 32 < 2 ? W / 32 : 2;
#pragma unroll
      for (int c0 = 0; c0 < W / 32; c0 += G) {
        uint32_t r[G][32];
#pragma unroll
        for (int c = 0; c < G; ++c)
          if (need & (1u << (c0 + c))) ptx::tmem_ld32(tmem + b * kRows + 32 * (c0 + c), r[c]);
        ptx::tmem_wait_ld();
#pragma unroll
        for (int c = 0; c < G; ++c) {
          if (!(need & (1u << (c0 + c)))) continue;
#pragma unroll
          for (int e = 0; e < 32; ++e)
            acc[32 * (c0 + c) + e] += ptx::ex2(__uint_as_float(r[c][e]) * L.scale_log2 - m);
        }
      }
      ptx::tc_fence_before();
      ptx::mbar_arrive(bar(C::B_SE + b));
    }
    if (!ok) break;
    // Store: the warp's 32 rows are 32 consecutive rows of A_if (frames are
    // stored back to back), npf floats each. Each 32-column chunk of the
    // window goes through the warp's shared tile, so that the global stores
    // are whole 128-byte lines.
    {
      const int lane = threadIdx.x & 31;
      const int i = row - f0;                        // the row's index within its frame
      const int f0l = f0 - col_base;                 // the frame's first column in the window
      const int pos_w = rb * kRows + 32 * warp;      // visual position of the warp's first row
      const int n_rows = min(32, vi.n_vis - pos_w);  // rows of the warp inside the video
      float* dst = L.aif + (static_cast<int64_t>(vi.frame_off) * npf + pos_w) * npf;
#pragma unroll
      for (int c = 0; c < W / 32; ++c) {
        if (n_rows <= 0) continue;
        if (!(need & (1u << c))) {                   // warp-uniform: every key of the chunk is after every row's query
          if (!L.accumulate)
            for (int rr = 0; rr < n_rows; ++rr) dst[static_cast<int64_t>(rr) * npf + 32 * c + lane] = 0.f;
          continue;
        }
#pragma unroll
        for (int e = 0; e < 32; ++e) {
          const int j = 32 * c + e - f0l;
          stage[lane * C::STAGE_PITCH + e] = j <= i ? acc[32 * c + e] * inv_h : 0.f;   // keys after the query hold masked logits
        }
        __syncwarp();
        if (W > 32 || npf >= 32) {                   // window = frame: chunk c holds keys 32c .. 32c + 31 of every row
          for (int rr = 0; rr < n_rows; ++rr) {
            float* p = dst + static_cast<int64_t>(rr) * npf + 32 * c + lane;
            const float a = stage[rr * C::STAGE_PITCH + lane];
            *p = L.accumulate ? *p + a : a;
          }
        } else {                                     // npf < 32: the window holds 32 / npf frames
          for (int idx = lane; idx < n_rows * npf; idx += 32) {
            const int rr = idx / npf, j = idx - rr * npf;
            const float a = stage[rr * C::STAGE_PITCH + (rr / npf) * npf + j];
            dst[idx] = L.accumulate ? dst[idx] + a : a;
          }
        }
        __syncwarp();
      }
    }
    if (!more) break;
    vi = vn;
    rb = rbn;
  }
  if (!ok) record_failure(abort_flag, L.status);
}

template <int D, int W>
__global__ void __launch_bounds__(kThreads, 1) intra_frame_kernel(const __grid_constant__ IntraFrameLaunch L) {
  using C = IfCfg<D>;
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
    producer<D>(L, sbase, abort_flag);
  } else if (warp == kWarpMma) {
    mma_issuer<D>(L, sbase, tmem, abort_flag);
  } else {
    rows<D, W>(L, sbase, tmem, abort_flag, reinterpret_cast<float*>(smem + C::OFF_STAGE));
  }
  ptx::tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc<C::TMEM_COLS>(tmem);
  }
}

int sm_count() {
  static int cached[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) return 0;
  if (dev < 64 && cached[dev] > 0) return cached[dev];
  int n = 0;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
  if (dev < 64) cached[dev] = n;
  return n;
}

template <int D, int W>
cudaError_t launch_dw(const IntraFrameLaunch& L, cudaStream_t stream) {
  using C = IfCfg<D>;
  auto kern = intra_frame_kernel<D, W>;
  static PerDeviceAttr smem_once;
  cudaError_t e = raise_smem_limit(smem_once, reinterpret_cast<const void*>(kern), C::SMEM_BYTES);
  if (e != cudaSuccess) return e;
  const int n_sm = sm_count();
  if (n_sm <= 0) return cudaErrorInvalidDevice;
  const int grid = L.total_blocks < n_sm ? L.total_blocks : n_sm;
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
  if (L.n_videos == 0 || L.total_blocks == 0) return cudaSuccess;
  if (L.head_dim == 128) return launch_d<128>(L, stream);
  if (L.head_dim == 64) return launch_d<64>(L, stream);
  return cudaErrorInvalidValue;
}

}  // namespace evisel
