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
// topp_select_kernel: one CTA per (128-row tile of a video, KV group), 320
//   threads (warp 8 TMA, warp 9 MMA; warps 0-7 one row each, of head slot
//   warp / 4). The heads of the group go in pairs: S = Q_h k_bar^T for both
//   heads of a pair, in chunks of 128 blocks (tcgen05, both products from one
//   k_bar chunk, TMEM 2 buffers x 2 heads), in six passes over the chunks:
//     0     the row's max and min logit over H_i;
//     1..4  a radix select on the block's key q = floor((max - x) 2^14 / (max -
//           min)) (0 = the largest logit), digit by digit (3, 3, 4 and 4 bits,
//           top first): the mass per digit value of the blocks whose higher
//           digits equal the boundary's, in 8 or 16 register bins (the first
//           digit's bins together give the softmax sum Z); the boundary digit
//           is the one where the cumulative mass from the top reaches tau_p Z;
//     5     keep every block whose key is below the boundary key; at the
//           boundary key, blocks in id order while the mass before them is
//           below tau_p Z.
//   The blocks are ordered by logit as exactly as the key resolves them
//   ((max - min) / 16384); closer logits count as ties.
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
constexpr int kHeadSlots = 2;                    // heads in flight
constexpr int kRowWarps = 4 * kHeadSlots;        // warp w: rows 32 (w % 4) .. of head slot w / 4
constexpr int kWarpProducer = kRowWarps;
constexpr int kWarpMma = kRowWarps + 1;
constexpr int kThreads = 32 * (kRowWarps + 2);
constexpr int kQBits = 14;                       // key resolution: (max - min) / 2^14 over H_i
constexpr int kQMax = (1 << kQBits) - 1;
constexpr int kLevels = 4;                       // key digits of 3, 3, 4 and 4 bits
constexpr int kDigBins = 16;
constexpr int kPasses = kLevels + 2;             // stats, one pass per digit, bits

template <int D>
struct TpCfg {
  static constexpr int KB = D / 64;
  static constexpr int TILE_BYTES = kRows * D * 2;   // 128 rows (Q) or 128 blocks (k_bar)
  static constexpr int BLOCK = kRows * 128;
  static constexpr int OFF_Q = 0;                     // the pair's Q tiles (one stage)
  static constexpr int OFF_K = kHeadSlots * TILE_BYTES;   // 2 stages of k_bar chunks
  static constexpr int OFF_STASH = OFF_K + 2 * TILE_BYTES;   // [32][256] fp32: a group's u, per row thread
  static constexpr int OFF_BAR = OFF_STASH + 32 * kRows * kHeadSlots * 4;
  static constexpr int B_QF = 0, B_QE = 1, B_KF = 2, B_KE = 4, B_SF = 6, B_SE = 8, B_DRAIN = 10;
  static constexpr int N_BARS = 11;
  static constexpr int OFF_MISC = OFF_BAR + N_BARS * 8;
  static constexpr int SMEM_BYTES = OFF_MISC + 16 + 1024;
  static constexpr int TMEM_COLS = 2 * kHeadSlots * kCols;   // 2 buffers x 2 heads
  static_assert(SMEM_BYTES <= 232448, "shared memory budget");
};

// acc[K] += w for K = d, K < N (no bin for other d): a predicated add per
// bin with static register indices.
template <int K, int N>
__device__ __forceinline__ void bin_add(float (&acc)[kDigBins], int d, float w) {
  if constexpr (K < N) {
    asm("{\n\t.reg .pred p;\n\tsetp.eq.s32 p, %1, %2;\n\t@p add.rn.f32 %0, %0, %3;\n\t}"
        : "+f"(acc[K]) : "r"(d), "n"(K), "f"(w));
    bin_add<K + 1, N>(acc, d, w);
  }
}

// Digit lv of the key (top first): width and shift.
__host__ __device__ constexpr int digit_width(int lv) { return lv < 2 ? 3 : 4; }
__host__ __device__ constexpr int digit_shift(int lv) {
  return lv == 0 ? kQBits - 3 : lv == 1 ? kQBits - 6 : lv == 2 ? kQBits - 10 : 0;
}
static_assert(digit_shift(kLevels - 1) == 0 && digit_shift(2) == digit_width(3), "digits cover the key");

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
  const int n_pairs = (gq + kHeadSlots - 1) / kHeadSlots;
  const int per_pair = kPasses * n_ch;
  const int n_steps = n_pairs * per_pair;        // step t: pair t / per_pair, pass (t / n_ch) % kPasses, chunk t % n_ch

  if (threadIdx.x == 0) {
    for (int i = 0; i < C::N_BARS; ++i)
      ptx::mbar_init(bar(i), (i == C::B_SE || i == C::B_SE + 1) ? kRows * kHeadSlots : 1u);
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
    int nq = 0, nk = 0;                          // Q (per pair) and k_bar loads issued
    for (int t = 0; ok && t < n_steps; ++t) {
      const int pair = t / per_pair, ch = t % n_ch;
      if (t % per_pair == 0) {                   // the pair's Q tiles, once per pair
        if (pair >= 1 && !warp_wait(bar(C::B_QE), (pair - 1) & 1, abort_flag)) {
          ok = false;
          break;
        }
        const int nheads = min(kHeadSlots, gq - pair * kHeadSlots);
        if (ptx::elect_one(leader)) {
          ptx::mbar_arrive_expect_tx(bar(C::B_QF), nheads * C::TILE_BYTES);
          for (int sl = 0; sl < nheads; ++sl) {
#pragma unroll
            for (int kb = 0; kb < C::KB; ++kb)
              ptx::tma_load_3d(sbase + C::OFF_Q + sl * C::TILE_BYTES + kb * C::BLOCK, &L.tm_q, bar(C::B_QF),
                               kb * 64, g * gq + pair * kHeadSlots + sl, rt.q_start, pol);
          }
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
    // no copy in flight at exit: the last Q and k_bar loads have landed
    const volatile int never = 0;
    if (nq > 0) ptx::mbar_wait(bar(C::B_QF), (nq - 1) & 1, &never, kWaitTimeoutNs);
    for (int s = 0; s < 2 && s < nk; ++s)
      ptx::mbar_wait(bar(C::B_KF + s), ((nk - 1 - s) / 2) & 1, &never, kWaitTimeoutNs);
  } else if (warp == kWarpMma) {
    constexpr uint32_t kIdesc = ptx::idesc_bf16_f32(kRows, kCols, false, false);
    uint32_t leader = 0;
    int first_leader = -1;
    bool same = true, issued = false, ok = true;
    for (int t = 0; ok && t < n_steps; ++t) {
      const int b = t % 2, pair = t / per_pair;
      const bool pair_start = t % per_pair == 0;
      const bool pair_end = t % per_pair == per_pair - 1;
      if ((pair_start && !warp_wait(bar(C::B_QF), pair & 1, abort_flag)) ||
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
        const int nheads = min(kHeadSlots, gq - pair * kHeadSlots);
        const uint32_t kbase = sbase + C::OFF_K + (t % 2) * C::TILE_BYTES;
        for (int sl = 0; sl < nheads; ++sl) {
          const uint32_t qbase = sbase + C::OFF_Q + sl * C::TILE_BYTES;
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk) {
            const uint64_t a = ptx::sdesc_sw128(qbase + (kk / 4) * C::BLOCK + (kk % 4) * 32, 16, 1024);
            const uint64_t bd = ptx::sdesc_sw128(kbase + (kk / 4) * C::BLOCK + (kk % 4) * 32, 16, 1024);
            ptx::mma_ss(tmem + (b * kHeadSlots + sl) * kCols, a, bd, kIdesc, kk > 0 ? 1u : 0u);
          }
        }
        ptx::mma_commit(bar(C::B_SF + b));
        ptx::mma_commit(bar(C::B_KE + t % 2));
        if (pair_end) ptx::mma_commit(bar(C::B_QE));
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
    const int slot = warp / 4, row = threadIdx.x % kRows;
    const bool row_ok = row < rt.q_len;
    const int pos = rt.local0 + row;
    const int nh = row_ok ? n_hist(pos) : 0;
    const uint32_t tbase = tmem + (static_cast<uint32_t>((warp % 4) * 32) << 16) + slot * kCols;
    const float sc = L.scale_log2;               // logits in log2 units
    constexpr int kStash = kRows * kHeadSlots;   // this thread's column: stash[e * kStash]
    float* stash = reinterpret_cast<float*>(smem + C::OFF_STASH) + slot * kRows + row;
    bool ok = true;
    for (int pair = 0; pair < n_pairs; ++pair) {
      const int hh = pair * kHeadSlots + slot;
      const bool active = hh < gq;               // warp-uniform: an odd group leaves the last slot idle
      const int h = g * gq + min(hh, gq - 1);
      float m = -INFINITY, gmin = INFINITY, z = 0.f;
      float inv_r = 0.f, target = 0.f, above = 0.f, tie = 0.f;
      int wkey = 0;                              // the boundary's key digits found so far
      uint32_t* keep = L.keep + static_cast<int64_t>(h) * L.n_words * L.n_tok + rt.q_start + row;
      for (int pass = 0; pass < kPasses; ++pass) {
        const int lv = pass - 1;                 // digit of passes 1..kLevels
        const int width = digit_width(lv), dshift = digit_shift(lv);
        const int pshift = dshift + width;       // key >> pshift: the digits above this one
        // The window (keys with the boundary's higher digits) as bounds on v =
        // (max - x) 2^14 / (max - min): key = min(kQMax, floor(v)), so
        // key >> pshift == wkey iff lo <= v < hi (hi open at the top key).
        const float lo = static_cast<float>(wkey << pshift);
        const float hi = ((wkey + 1) << pshift) > kQMax ? INFINITY : static_cast<float>((wkey + 1) << pshift);
        float acc[kDigBins];
#pragma unroll
        for (int k = 0; k < kDigBins; ++k) acc[k] = 0.f;
        for (int ch = 0; ch < n_ch; ++ch) {
          const int t = (pair * kPasses + pass) * n_ch + ch, b = t % 2;
          ok = ok && warp_wait(bar(C::B_SF + b), (t / 2) & 1, abort_flag);
          if (ok && active && __any_sync(0xffffffffu, nh > ch * kCols)) {   // warp-uniform: tcgen05.ld is collective
            ptx::tc_fence_after();
            // One compact loop per pass (uniform over the warp), 32 columns at a
            // time. x, the key and the weight use non-contracted arithmetic so
            // that every pass sees the same values.
#pragma unroll 1
            for (int c0 = 0; c0 < kCols; c0 += 32) {
              uint32_t r[32];
              ptx::tmem_ld32(tbase + b * kHeadSlots * kCols + c0, r);
              ptx::tmem_wait_ld();
              const int jn = nh - (ch * kCols + c0);         // columns e < jn are in H_i
              if (pass == 0) {
                // The row's max and min over H_i (the softmax sum comes from the
                // first digit's bins, which every block of H_i falls in).
                float mx[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
                float mn[4] = {INFINITY, INFINITY, INFINITY, INFINITY};
#pragma unroll
                for (int e = 0; e < 32; ++e) {
                  const float x = __fmul_rn(__uint_as_float(r[e]), sc);
                  if (e < jn) {
                    mx[e & 3] = fmaxf(mx[e & 3], x);
                    mn[e & 3] = fminf(mn[e & 3], x);
                  }
                }
                m = fmaxf(m, fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])));
                gmin = fminf(gmin, fminf(fminf(mn[0], mn[1]), fminf(mn[2], mn[3])));
              } else if (lv == 0) {
                // The first digit (every column is in the window): no branches,
                // so that the columns' arithmetic overlaps.
#pragma unroll
                for (int e = 0; e < 32; ++e) {
                  const float u = __fsub_rn(m, __fmul_rn(__uint_as_float(r[e]), sc));
                  const float v = __fmul_rn(u, inv_r);
                  const int key = min(kQMax, __float2int_rz(v));
                  const int dig = (e < jn && v >= lo && v < hi) ? (key >> dshift) & ((1 << width) - 1) : -1;
                  bin_add<0, 8>(acc, dig, ptx::ex2(-u));
                }
              } else if (lv < kLevels) {
                // Later digits (a few percent of the columns): the window test stashes the
                // window's u; then each lane walks its own window columns in id
                // order and adds ex2(-u) to the digit's bin.
                uint32_t in_mask = 0u;
#pragma unroll
                for (int e = 0; e < 32; ++e) {
                  const float u = __fsub_rn(m, __fmul_rn(__uint_as_float(r[e]), sc));
                  const float v = __fmul_rn(u, inv_r);
                  if (e < jn && v >= lo && v < hi) {
                    in_mask |= 1u << e;
                    stash[e * kStash] = u;
                  }
                }
                while (in_mask != 0u) {
                  const int e = __ffs(in_mask) - 1;
                  in_mask &= in_mask - 1u;
                  const float u = stash[e * kStash];
                  const int key = min(kQMax, __float2int_rz(__fmul_rn(u, inv_r)));
                  bin_add<0, 16>(acc, (key >> dshift) & ((1 << width) - 1), ptx::ex2(-u));
                }
                __syncwarp();
              } else {
                // key < wkey iff v < wkey; key == wkey iff wkey <= v < wkey + 1 (open at the top key)
                const float k0 = static_cast<float>(wkey);
                const float k1 = wkey == kQMax ? INFINITY : static_cast<float>(wkey + 1);
                uint32_t word = 0u, at_mask = 0u;
#pragma unroll
                for (int e = 0; e < 32; ++e) {
                  const float u = __fsub_rn(m, __fmul_rn(__uint_as_float(r[e]), sc));
                  const float v = __fmul_rn(u, inv_r);
                  word |= (e < jn && v < k0) ? 1u << e : 0u;
                  if (e < jn && v >= k0 && v < k1) {
                    at_mask |= 1u << e;
                    stash[e * kStash] = u;
                  }
                }
                // the boundary key: lower ids first while the mass before them is below the target
                while (at_mask != 0u) {
                  const int e = __ffs(at_mask) - 1;
                  at_mask &= at_mask - 1u;
                  if (above + tie < target) word |= 1u << e;
                  tie += ptx::ex2(-stash[e * kStash]);
                }
                __syncwarp();
                const int w = ch * 4 + (c0 >> 5);
                if (row_ok && w < L.n_words) {
                  if (w == nh >> 5) word |= 1u << (nh & 31);     // the row's own block
                  keep[static_cast<int64_t>(w) * L.n_tok] = word;
                }
              }
            }
            ptx::tc_fence_before();
          } else if (pass == kPasses - 1 && row_ok && ok && active) {
            // No column of this chunk is in H_i for the warp: zeros (and the own block).
            for (int wi = 0; wi < 4; ++wi) {
              const int w = ch * 4 + wi;
              if (w >= L.n_words) break;
              keep[static_cast<int64_t>(w) * L.n_tok] = w == nh >> 5 ? 1u << (nh & 31) : 0u;
            }
          }
          ptx::mbar_arrive(bar(C::B_SE + b));
        }
        // Between passes: the key scale, then per digit the boundary value and
        // the mass above it. The boundary is the first digit value whose
        // cumulative mass from the top reaches the target; when rounding keeps
        // the total below it (tau_p near 1), the last non-empty one, whose
        // blocks are then all kept.
        if (pass == 0) {
          inv_r = static_cast<float>(kQMax + 1) / fmaxf(m - gmin, 1e-30f);
        } else if (lv < kLevels) {
          if (lv == 0) {
            // Z: the first digit's bins hold the weight of every block of H_i.
#pragma unroll
            for (int kb = 0; kb < 8; ++kb) z += acc[kb];
            target = L.tau * z;
          }
          float run = above, before_last = above;
          int found = -1, last = 0;
#pragma unroll
          for (int k = 0; k < kDigBins; ++k) {
            const float hb = acc[k];
            if (hb > 0.f) {
              last = k;
              before_last = run;
            }
            if (found < 0) {
              if (run + hb >= target) found = k;
              else run += hb;
            }
          }
          above = found >= 0 ? run : before_last;
          wkey = (wkey << width) | (found >= 0 ? found : last);
        }
      }
      // The own block's word when it lies past the chunks of this tile.
      if (row_ok && ok && active && (nh >> 5) >= n_ch * 4 && (nh >> 5) < L.n_words)
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
  static PerDeviceAttr smem_once;
  cudaError_t e = raise_smem_limit(smem_once, reinterpret_cast<const void*>(kern), C::SMEM_BYTES);
  if (e != cudaSuccess) return e;
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
