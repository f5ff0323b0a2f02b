// Top-p block retention of the sparse prefill (Appendix, "Detailed Sparse
// Prefilling", Eq. 6-9 and the retention rule after Eq. 9):
//   k_bar_j = mean of block j's keys (Eq. 7); for row i, H_i = the blocks of
//   its video that end before i; g_ij = q_i k_bar_j / sqrt(d) (Eq. 8);
//   p_ij = softmax over H_i (Eq. 9); S_i = the shortest prefix of H_i in
//   descending p (ties: lower block id) whose mass reaches tau_p.
// Output: per (head, row) a bit per block of the row's video: S_i and the
// row's own block (whose causal prefix the row always attends), as
// keep[h][word][row]; and per attention row tile the union over its rows and
// heads, as key-tile bits (a tile-level mask the attention kernel takes).
//
// kbar_kernel: one CTA per (block, KV head): the block's mean key in fp32,
//   stored as bf16 (the tensor cores' input type).
// topp_select_kernel: one CTA per (128-row tile of a video, KV group), 192
//   threads (warp 4 TMA, warp 5 MMA, warps 0-3 one row each). For each head of
//   the group, S = Q_h k_bar^T in chunks of 128 blocks (tcgen05, TMEM double
//   buffer), in four passes over the chunks:
//     0  the row's max and min logit over H_i and the softmax sum Z (online);
//     1  the mass per bin of 128 equal logit bins between max and min; the
//        bin b1 where the cumulative mass from the top reaches tau_p Z;
//     2  the same with 128 sub-bins of bin b1: sub-bin b2;
//     3  keep every block of a higher bin or sub-bin; inside sub-bin b2,
//        blocks in id order while the mass before them is below tau_p Z.
//   The blocks are ordered by logit as exactly as the sub-bin width
//   ((max - min) / 16384) resolves them; closer logits count as ties.
// topp_union_kernel: one thread per (row, head) ORs its bits, mapped to key
//   tiles, into its attention row tile's union.
// Every wait is bounded; a timeout records EVISEL_ETIMEOUT.
#include <cstdint>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "evisel_internal.h"
#include "sm103_ptx.cuh"

namespace evisel {
namespace {

constexpr int kRows = 128;
constexpr int kCols = 128;                       // blocks per chunk
constexpr int kBins = 128;
constexpr int kThreads = 192;
constexpr int kWarpProducer = 4;
constexpr int kWarpMma = 5;
constexpr int kPasses = 4;

template <int D>
struct TpCfg {
  static constexpr int KB = D / 64;
  static constexpr int TILE_BYTES = kRows * D * 2;   // 128 rows (Q) or 128 blocks (k_bar)
  static constexpr int BLOCK = kRows * 128;
  static constexpr int OFF_Q = 0;                     // 2 stages (one per head in flight)
  static constexpr int OFF_K = 2 * TILE_BYTES;        // 2 stages of k_bar chunks
  static constexpr int OFF_HIST = OFF_K + 2 * TILE_BYTES;   // [kBins][128] fp32
  static constexpr int OFF_BAR = OFF_HIST + kBins * kRows * 4;
  static constexpr int B_QF = 0, B_QE = 2, B_KF = 4, B_KE = 6, B_SF = 8, B_SE = 10, B_DRAIN = 12;
  static constexpr int N_BARS = 13;
  static constexpr int OFF_MISC = OFF_BAR + N_BARS * 8;
  static constexpr int SMEM_BYTES = OFF_MISC + 16 + 1024;
  static constexpr int TMEM_COLS = 256;
  static_assert(SMEM_BYTES <= 232448, "shared memory budget");
};

__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag) {
  const bool ok = ptx::mbar_wait(bar, parity, abort_flag, kWaitTimeoutNs);
  return __all_sync(0xffffffffu, ok);
}

__device__ __forceinline__ void record_failure(volatile int* abort_flag, int* status) {
  *abort_flag = 1;
  atomicExch(status, kStatusTimeout);
}

__global__ void __launch_bounds__(128) kbar_kernel(const __grid_constant__ ToppLaunch L) {
  // blockIdx.x: global block (video blocks back to back), blockIdx.y: KV head.
  const int gb = blockIdx.x, g = blockIdx.y;
  const ToppVideo* vp = L.vids;
  int v = 0;
  while (v + 1 < L.n_videos && vp[v + 1].blk_off <= gb) ++v;
  const ToppVideo vid = vp[v];
  const int j = gb - vid.blk_off;
  const int nvb = vid.n_vis / L.block;
  const int start = j < nvb ? j * L.block : vid.n_vis + (j - nvb) * L.block;
  const int len = j < nvb ? L.block : min(L.block, vid.n_vis + vid.n_text - start);
  const __nv_bfloat16* k = static_cast<const __nv_bfloat16*>(L.k);
  for (int e = threadIdx.x; e < L.head_dim; e += blockDim.x) {
    float s = 0.f;
    for (int t = 0; t < len; ++t)
      s += __bfloat162float(k[(static_cast<int64_t>(vid.start + start + t) * L.hkv + g) * L.head_dim + e]);
    static_cast<__nv_bfloat16*>(L.kbar)[(static_cast<int64_t>(gb) * L.hkv + g) * L.head_dim + e] =
        __float2bfloat16_rn(s / static_cast<float>(len));
  }
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1) topp_select_kernel(const __grid_constant__ ToppLaunch L) {
  using C = TpCfg<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t sbase = ptx::smem_addr(smem);
  auto bar = [&](int i) { return sbase + C::OFF_BAR + 8u * i; };
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + C::OFF_MISC);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::OFF_MISC + 4);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const ToppRowTile rt = L.tiles[blockIdx.x];
  const ToppVideo vid = L.vids[rt.video];
  const int g = blockIdx.y;
  const int gq = L.hq / L.hkv;
  const int nvb = vid.n_vis / L.block;
  // Blocks that end before the tile's last row: the chunk range of this tile.
  auto n_hist = [&](int pos_local) {
    return pos_local < vid.n_vis ? pos_local / L.block : nvb + (pos_local - vid.n_vis) / L.block;
  };
  const int nh_max = n_hist(rt.local0 + rt.q_len - 1);
  const int n_ch = (nh_max + kCols - 1) / kCols;
  const int n_steps = gq * kPasses * n_ch;       // step t: head t / (4 n_ch), pass (t / n_ch) % 4, chunk t % n_ch

  if (threadIdx.x == 0) {
    for (int i = 0; i < C::N_BARS; ++i) ptx::mbar_init(bar(i), (i == C::B_SE || i == C::B_SE + 1) ? kRows : 1u);
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
    const uint64_t pol = ptx::l2_policy_evict_last();
    uint32_t leader = 0;
    bool ok = true;
    int nq = 0, nk = 0;
    for (int t = 0; ok && t < n_steps; ++t) {
      const int hh = t / (kPasses * n_ch), ch = t % n_ch;
      if (t % (kPasses * n_ch) == 0) {           // the head's Q tile, once per head
        const int qs = nq % 2;
        if (nq >= 2 && !warp_wait(bar(C::B_QE + qs), ((nq - 2) / 2) & 1, abort_flag)) {
          ok = false;
          break;
        }
        if (ptx::elect_one(leader)) {
          ptx::mbar_arrive_expect_tx(bar(C::B_QF + qs), C::TILE_BYTES);
#pragma unroll
          for (int kb = 0; kb < C::KB; ++kb)
            ptx::tma_load_3d(sbase + C::OFF_Q + qs * C::TILE_BYTES + kb * C::BLOCK, &L.tm_q, bar(C::B_QF + qs),
                             kb * 64, g * gq + hh, rt.q_start, pol);
        }
        __syncwarp();
        ++nq;
      }
      const int ks = nk % 2;
      if (nk >= 2 && !warp_wait(bar(C::B_KE + ks), ((nk - 2) / 2) & 1, abort_flag)) {
        ok = false;
        break;
      }
      if (ptx::elect_one(leader)) {
        ptx::mbar_arrive_expect_tx(bar(C::B_KF + ks), C::TILE_BYTES);
#pragma unroll
        for (int kb = 0; kb < C::KB; ++kb)
          ptx::tma_load_3d(sbase + C::OFF_K + ks * C::TILE_BYTES + kb * C::BLOCK, &L.tm_kbar, bar(C::B_KF + ks),
                           kb * 64, g, vid.blk_off + ch * kCols, pol);
      }
      __syncwarp();
      ++nk;
    }
    if (!ok && lane == 0) record_failure(abort_flag, L.status);
    const volatile int never = 0;
    for (int s = 0; s < 2 && s < nq; ++s)
      ptx::mbar_wait(bar(C::B_QF + s), ((nq - 1 - s) / 2) & 1, &never, kWaitTimeoutNs);
    for (int s = 0; s < 2 && s < nk; ++s)
      ptx::mbar_wait(bar(C::B_KF + s), ((nk - 1 - s) / 2) & 1, &never, kWaitTimeoutNs);
  } else if (warp == kWarpMma) {
    constexpr uint32_t kIdesc = ptx::idesc_bf16_f32(kRows, kCols, false, false);
    uint32_t leader = 0;
    int first_leader = -1;
    bool same = true, issued = false, ok = true;
    int nq = 0;
    for (int t = 0; ok && t < n_steps; ++t) {
      const int b = t % 2;
      const bool head_start = t % (kPasses * n_ch) == 0;
      const bool head_end = t % (kPasses * n_ch) == kPasses * n_ch - 1;
      if (head_start) ++nq;
      const int qs = (nq - 1) % 2;
      if ((head_start && !warp_wait(bar(C::B_QF + qs), ((nq - 1) / 2) & 1, abort_flag)) ||
          !warp_wait(bar(C::B_KF + t % 2), (t / 2) & 1, abort_flag) ||
          (t >= 2 && !warp_wait(bar(C::B_SE + b), ((t - 2) / 2) & 1, abort_flag))) {
        ok = false;
        break;
      }
      ptx::tc_fence_after();
      const bool me = ptx::elect_one(leader);
      if (first_leader < 0) first_leader = static_cast<int>(leader);
      same = same && static_cast<int>(leader) == first_leader;
      if (me && same) {
        const uint32_t qbase = sbase + C::OFF_Q + qs * C::TILE_BYTES;
        const uint32_t kbase = sbase + C::OFF_K + (t % 2) * C::TILE_BYTES;
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint64_t a = ptx::sdesc_sw128(qbase + (kk / 4) * C::BLOCK + (kk % 4) * 32, 16, 1024);
          const uint64_t bd = ptx::sdesc_sw128(kbase + (kk / 4) * C::BLOCK + (kk % 4) * 32, 16, 1024);
          ptx::mma_ss(tmem + b * kCols, a, bd, kIdesc, kk > 0 ? 1u : 0u);
        }
        ptx::mma_commit(bar(C::B_SF + b));
        ptx::mma_commit(bar(C::B_KE + t % 2));
        if (head_end) ptx::mma_commit(bar(C::B_QE + qs));
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
    // Row threads: row = TMEM lane; the row's video-local position and |H_i|.
    const int row = threadIdx.x;
    const bool row_ok = row < rt.q_len;
    const int pos = rt.local0 + row;
    const int nh = row_ok ? n_hist(pos) : 0;
    const uint32_t tbase = tmem + (static_cast<uint32_t>(warp * 32) << 16);
    float* hist = reinterpret_cast<float*>(smem + C::OFF_HIST) + row;   // column of this thread: hist[bin * 128]
    const float sc = L.scale_log2;               // logits in log2 units
    bool ok = true;
    for (int hh = 0; hh < gq; ++hh) {
      const int h = g * gq + hh;
      float m = -INFINITY, gmin = INFINITY, z = 0.f;
      float w1 = 0.f, inv_w1 = 0.f, inv_w2 = 0.f, target = 0.f, above1 = 0.f, above2 = 0.f, tie = 0.f;
      int b1 = 0, b2 = 0;
      uint32_t* keep = L.keep + static_cast<int64_t>(h) * L.n_words * L.n_tok + rt.q_start + row;
      for (int pass = 0; pass < kPasses; ++pass) {
        if (pass == 1 || pass == 2) {
          for (int bi = 0; bi < kBins; ++bi) hist[bi * kRows] = 0.f;
        }
        for (int ch = 0; ch < n_ch; ++ch) {
          const int t = (hh * kPasses + pass) * n_ch + ch, b = t % 2;
          ok = ok && warp_wait(bar(C::B_SF + b), (t / 2) & 1, abort_flag);
          int run_bin = -1;                        // histogram passes: consecutive keys of one bin add in a register
          float run = 0.f;
          if (ok && __any_sync(0xffffffffu, nh > ch * kCols)) {   // warp-uniform: tcgen05.ld is collective
            ptx::tc_fence_after();
            // One compact loop per pass (uniform over the warp), 32 columns at a time.
#pragma unroll 1
            for (int c0 = 0; c0 < kCols; c0 += 32) {
              uint32_t r[32];
              ptx::tmem_ld32(tbase + b * kCols + c0, r);
              ptx::tmem_wait_ld();
              const int jn = nh - (ch * kCols + c0);         // columns e < jn are in H_i
              if (pass == 0) {
                float cmax = -INFINITY;
#pragma unroll
                for (int e = 0; e < 32; ++e) {
                  const float x = __uint_as_float(r[e]) * sc;
                  if (e < jn) {
                    cmax = fmaxf(cmax, x);
                    gmin = fminf(gmin, x);
                  }
                }
                if (cmax > m) {
                  z = (m == -INFINITY) ? 0.f : z * ptx::ex2(m - cmax);
                  m = cmax;
                }
                float zs = 0.f;
#pragma unroll
                for (int e = 0; e < 32; ++e)
                  if (e < jn) zs += ptx::ex2(__uint_as_float(r[e]) * sc - m);
                z += zs;
              } else if (pass == 1) {
#pragma unroll
                for (int e = 0; e < 32; ++e) {
                  if (e >= jn) break;
                  const float x = __uint_as_float(r[e]) * sc;
                  const int bin1 = min(kBins - 1, static_cast<int>((m - x) * inv_w1));
                  if (bin1 != run_bin) {
                    if (run_bin >= 0) hist[run_bin * kRows] += run;
                    run_bin = bin1;
                    run = 0.f;
                  }
                  run += ptx::ex2(x - m);
                }
              } else if (pass == 2) {
#pragma unroll
                for (int e = 0; e < 32; ++e) {
                  if (e >= jn) break;
                  const float x = __uint_as_float(r[e]) * sc;
                  const float u = m - x;
                  if (min(kBins - 1, static_cast<int>(u * inv_w1)) != b1) continue;
                  const int bin2 = min(kBins - 1, static_cast<int>((u - b1 * w1) * inv_w2));
                  if (bin2 != run_bin) {
                    if (run_bin >= 0) hist[run_bin * kRows] += run;
                    run_bin = bin2;
                    run = 0.f;
                  }
                  run += ptx::ex2(x - m);
                }
              } else {
                uint32_t word = 0u;
#pragma unroll
                for (int e = 0; e < 32; ++e) {
                  if (e >= jn) break;
                  const float x = __uint_as_float(r[e]) * sc;
                  const float u = m - x;
                  const int bin1 = min(kBins - 1, static_cast<int>(u * inv_w1));
                  bool kept = bin1 < b1;
                  if (bin1 == b1) {
                    const int bin2 = min(kBins - 1, static_cast<int>((u - b1 * w1) * inv_w2));
                    kept = bin2 < b2;
                    if (bin2 == b2) {                             // ties: lower ids first
                      kept = above2 + tie < target;
                      tie += ptx::ex2(x - m);
                    }
                  }
                  if (kept) word |= 1u << e;
                }
                const int w = ch * 4 + (c0 >> 5);
                if (row_ok && w < L.n_words) {
                  if (w == nh >> 5) word |= 1u << (nh & 31);     // the row's own block
                  keep[static_cast<int64_t>(w) * L.n_tok] = word;
                }
              }
            }
            ptx::tc_fence_before();
          } else if (pass == 3 && row_ok && ok) {
            // No column of this chunk is in H_i for the warp: zeros (and the own block).
            for (int wi = 0; wi < 4; ++wi) {
              const int w = ch * 4 + wi;
              if (w >= L.n_words) break;
              keep[static_cast<int64_t>(w) * L.n_tok] = w == nh >> 5 ? 1u << (nh & 31) : 0u;
            }
          }
          ptx::mbar_arrive(bar(C::B_SE + b));
          if (run_bin >= 0) hist[run_bin * kRows] += run;
        }
        // Between passes: the bin widths and the boundary (bin, mass above it).
        // A boundary is the first bin whose cumulative mass from the top reaches
        // the target; when rounding keeps the total below it (tau_p near 1), the
        // last non-empty bin, whose members are then all kept.
        if (pass == 0) {
          target = L.tau * z;
          w1 = fmaxf((m - gmin) / kBins, 1e-30f);
          inv_w1 = 1.f / w1;
          inv_w2 = static_cast<float>(kBins) * inv_w1;
        } else if (pass == 1 || pass == 2) {
          float acc = pass == 1 ? 0.f : above1, before_last = acc;
          int found = -1, last = 0;
          for (int bi = 0; bi < kBins; ++bi) {
            const float hb = hist[bi * kRows];
            if (hb > 0.f) {
              last = bi;
              before_last = acc;
            }
            if (acc + hb >= target) {
              found = bi;
              break;
            }
            acc += hb;
          }
          const int bb = found >= 0 ? found : last;
          const float ab = found >= 0 ? acc : before_last;
          if (pass == 1) {
            b1 = bb;
            above1 = ab;
          } else {
            b2 = bb;
            above2 = ab;
          }
        }
      }
      // The own block's word when it lies past the chunks of this tile.
      if (row_ok && ok && (nh >> 5) >= n_ch * 4 && (nh >> 5) < L.n_words)
        keep[static_cast<int64_t>(nh >> 5) * L.n_tok] = 1u << (nh & 31);
    }
    if (!ok && row == 0) record_failure(abort_flag, L.status);
  }
  ptx::tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc<C::TMEM_COLS>(tmem);
  }
}

__global__ void __launch_bounds__(128) topp_union_kernel(const __grid_constant__ ToppLaunch L) {
  // blockIdx.x: builder row tile, blockIdx.y: head; one thread per row. Word
  // by word of the union (32 key tiles = 32 * tile / block blocks), a thread
  // folds its blocks into tile bits, the warp ORs them, one lane stores.
  const ToppRowTile rt = L.tiles[blockIdx.x];
  if (rt.text) return;                           // the attention takes tile masks for visual rows only
  const ToppVideo vid = L.vids[rt.video];
  const int h = blockIdx.y, row = threadIdx.x;
  const int pos = rt.local0 + min(row, rt.q_len - 1);
  const bool row_ok = row < rt.q_len;
  const int bpt = L.tile / L.block;              // blocks per key tile: 1, 2, 4 or 8
  const int nvb = vid.n_vis / L.block;           // visual blocks (visual rows keep no text block)
  const int n_vt = (vid.n_vis + L.tile - 1) / L.tile;
  const uint32_t* keep = L.keep + static_cast<int64_t>(h) * L.n_words * L.n_tok + vid.start + pos;
  // Rows of one warp may belong to two attention row tiles (tile = 64): reduce per tile.
  const int my_tile = pos / L.tile;
  for (int tw = 0; tw * 32 < n_vt; ++tw) {
    uint32_t bits = 0u;
    if (row_ok) {
      for (int q = 0; q < bpt; ++q) {            // keep words tw * bpt + q: blocks of tiles 32 tw + (32 q .. 32 q + 31) / bpt
        const int w = tw * bpt + q;
        if (w >= L.n_words || w * 32 >= nvb) break;
        uint32_t x = keep[static_cast<int64_t>(w) * L.n_tok];
        if (w * 32 + 32 > nvb) x &= (1u << (nvb - w * 32)) - 1u;   // visual blocks only
        for (int k = 1; k < bpt; k <<= 1) x |= x >> k;             // a tile's OR in its lowest block bit
        for (int i = 0; i < 32 / bpt; ++i)
          if ((x >> (i * bpt)) & 1u) bits |= 1u << (q * (32 / bpt) + i);
      }
    }
    const int lane = threadIdx.x & 31;
    const int first_tile = __shfl_sync(0xffffffffu, my_tile, 0);
    const bool one_tile = __all_sync(0xffffffffu, my_tile == first_tile);
    if (one_tile) {
      const uint32_t wbits = __reduce_or_sync(0xffffffffu, bits);
      if (lane == 0 && wbits)
        atomicOr(L.tile_union + static_cast<int64_t>(vid.row_tile0 + my_tile) * L.n_tile_words + tw, wbits);
    } else if (bits) {
      atomicOr(L.tile_union + static_cast<int64_t>(vid.row_tile0 + my_tile) * L.n_tile_words + tw, bits);
    }
  }
}

template <int D>
cudaError_t launch_select(const ToppLaunch& L, cudaStream_t stream) {
  using C = TpCfg<D>;
  auto kern = topp_select_kernel<D>;
  static bool configured = false;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM_BYTES);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  dim3 grid(L.n_tiles, L.hkv);
  kern<<<grid, kThreads, C::SMEM_BYTES, stream>>>(L);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_topp(const ToppLaunch& L, cudaStream_t stream) {
  if (L.n_tiles == 0) return cudaSuccess;
  if (L.n_blocks_total > 0) {
    dim3 grid(L.n_blocks_total, L.hkv);
    kbar_kernel<<<grid, 128, 0, stream>>>(L);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  cudaError_t e = L.head_dim == 128 ? launch_select<128>(L, stream)
                : L.head_dim == 64  ? launch_select<64>(L, stream)
                                    : cudaErrorInvalidValue;
  if (e != cudaSuccess) return e;
  if (L.tile_union) {
    dim3 grid(L.n_tiles, L.hq);
    topp_union_kernel<<<grid, 128, 0, stream>>>(L);
    return cudaGetLastError();
  }
  return cudaSuccess;
}

}  // namespace evisel
