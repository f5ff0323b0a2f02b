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
//   k_bar chunk, TMEM 2 buffers x 2 heads), recomputed for every pass over the
//   chunks. A block's key is q = floor((max - x) 2^14 / (max - min)) over H_i
//   (0 = the largest logit); blocks are ordered by key, ties by id.
//   Fast path (every pair), four passes:
//     0     the row's max and min logit over H_i;
//     1, 2  two 3-bit digits of the boundary key: per digit value, the mass of
//           the blocks whose key lies below its top (a saturated difference of
//           floored keys times the weight, on the FMA pipe; the first pass also
//           sums Z); the boundary digit is the first whose mass reaches tau_p Z;
//     3     collect: blocks below the 6-bit window are kept, blocks in it are
//           listed per row (at most 32), blocks above it dropped.
//   The list (in id order) then gives the last 8 key bits the same way, in two
//   4-bit digits, and at the boundary key blocks are kept in id order while
//   the mass before them is below tau_p Z.
//   Radix path (the pairs where some row's window held more than 32 blocks),
//   after a CTA-wide decision: six passes, as the fast path's first two but a
//   radix select on the key, digit by digit (3, 3, 4 and 4 bits), the mass per
//   digit value in register bins; then every block whose key is below the
//   boundary key is kept and, at the boundary key, blocks in id order while the
//   mass before them is below tau_p Z.
// topp_union_kernel: per (visual row tile, 1,024 blocks) the OR of the rows'
//   bits over the heads, folded into key tiles, as its attention row tiles'
//   union words.
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
constexpr int kLevels = 4;                       // radix path: key digits of 3, 3, 4 and 4 bits
constexpr int kDigBins = 16;
constexpr int kRadixPasses = kLevels + 2;        // stats, one pass per digit, bits
constexpr int kFastPasses = 4;                   // stats, two 3-bit digits, collect
constexpr int kFastBins = 8;                     // digit values per fast digit pass
constexpr int kFastTops = kFastBins - 1;         // tops with a mass sum (the last digit's is not needed)
constexpr int kListCap = 32;                     // window blocks a row thread lists in the collect pass
constexpr float kMagic = 8388608.f;              // 2^23: v +rz 2^23 holds floor(v) in its mantissa

template <int D>
struct TpCfg {
  static constexpr int KB = D / 64;
  static constexpr int TILE_BYTES = kRows * D * 2;   // 128 rows (Q) or 128 blocks (k_bar)
  static constexpr int BLOCK = kRows * 128;
  static constexpr int OFF_Q = 0;                     // the pair's Q tiles (one stage)
  static constexpr int OFF_K = kHeadSlots * TILE_BYTES;   // 2 stages of k_bar chunks
  // [32][256] fp32 per row thread: the radix path's u of a 32-column group, or
  // the fast path's list of window blocks (u), with their ids in [32][256] int32.
  static constexpr int OFF_STASH = OFF_K + 2 * TILE_BYTES;
  static constexpr int OFF_LIST_ID = OFF_STASH + kListCap * kRows * kHeadSlots * 4;
  // [256][32] fp32: the collect pass's u of a 32-column group per row thread,
  // its 16-byte chunks XOR-swizzled by the thread's row % 8.
  static constexpr int OFF_GROUP_U = OFF_LIST_ID + kListCap * kRows * kHeadSlots * 4;
  static constexpr int OFF_BAR = OFF_GROUP_U + 32 * kRows * kHeadSlots * 4;
  static constexpr int B_QF = 0, B_QE = 1, B_KF = 2, B_KE = 4, B_SF = 6, B_SE = 8, B_DRAIN = 10, B_DEC = 11;
  static constexpr int N_BARS = 12;
  static constexpr int OFF_MISC = OFF_BAR + N_BARS * 8;   // TMEM address, abort flag, overflowed pairs
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

// Two fp32 fmas in one packed instruction: d_i = a_i b_i + c_i, each rounded
// to nearest (rn) or toward zero (rz) as the scalar fma would be.
__device__ __forceinline__ void fma2_rn(float& d0, float& d1, float a0, float a1, float b0, float b1, float c0,
                                        float c1) {
  asm("{\n\t.reg .b64 a, b, c;\n\tmov.b64 a, {%2, %3};\n\tmov.b64 b, {%4, %5};\n\tmov.b64 c, {%6, %7};\n\t"
      "fma.rn.f32x2 c, a, b, c;\n\tmov.b64 {%0, %1}, c;\n\t}"
      : "=f"(d0), "=f"(d1)
      : "f"(a0), "f"(a1), "f"(b0), "f"(b1), "f"(c0), "f"(c1));
}
__device__ __forceinline__ void fma2_rz(float& d0, float& d1, float a0, float a1, float b0, float b1, float c0,
                                        float c1) {
  asm("{\n\t.reg .b64 a, b, c;\n\tmov.b64 a, {%2, %3};\n\tmov.b64 b, {%4, %5};\n\tmov.b64 c, {%6, %7};\n\t"
      "fma.rz.f32x2 c, a, b, c;\n\tmov.b64 {%0, %1}, c;\n\t}"
      : "=f"(d0), "=f"(d1)
      : "f"(a0), "f"(a1), "f"(b0), "f"(b1), "f"(c0), "f"(c1));
}

// Cumulative masses of one digit pass: cm[k] += w for every digit top top[k]
// above the block's floored key f (both offset by 2^23, so top - f is an exact
// integer and its saturation the indicator), on the FMA pipe only, two sums
// per packed fma. With Z, the sum of every w rides along with the last top.
template <int N, bool kWithZ = false>
__device__ __forceinline__ void cum_add(float (&cm)[N], const float (&top)[N], float f, float w, float& z) {
  float ind[N];
#pragma unroll
  for (int k = 0; k < N; ++k) asm("sub.sat.f32 %0, %1, %2;" : "=f"(ind[k]) : "f"(top[k]), "f"(f));
#pragma unroll
  for (int k = 0; k + 1 < N; k += 2) fma2_rn(cm[k], cm[k + 1], ind[k], ind[k + 1], w, w, cm[k], cm[k + 1]);
  if constexpr (N % 2 == 1 && kWithZ) {
    fma2_rn(cm[N - 1], z, ind[N - 1], 1.f, w, w, cm[N - 1], z);
  } else {
    if constexpr (N % 2 == 1) cm[N - 1] = __fmaf_rn(w, ind[N - 1], cm[N - 1]);
    if constexpr (kWithZ) z = __fadd_rn(z, w);
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
  uint32_t* overflowed = reinterpret_cast<uint32_t*>(smem + C::OFF_MISC + 8);   // bit min(pair, 31)
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
  // Work: every pair on the fast path (kFastPasses passes over the n_ch chunks),
  // then, once every row warp has arrived on B_DEC, the pairs whose window
  // overflowed a row's list on the radix path (kRadixPasses passes). All roles
  // step through the same chunk sequence; step t uses S buffer t % 2.
  auto redo = [&](uint32_t mask, int pair) { return ((mask >> min(pair, 31)) & 1u) != 0u; };

  if (threadIdx.x == 0) {
    for (int i = 0; i < C::N_BARS; ++i)
      ptx::mbar_init(bar(i), (i == C::B_SE || i == C::B_SE + 1) ? kRows * kHeadSlots
                             : i == C::B_DEC                      ? kRowWarps
                                                                  : 1u);
    *abort_flag = 0;
    *overflowed = 0u;
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
    int nq = 0, nk = 0;                          // Q (per pair job) and k_bar loads issued
    auto job = [&](int pair, int passes) -> bool {
      if (n_ch == 0) return true;                // no block ends before the tile's rows: nothing to load
      if (nq >= 1 && !warp_wait(bar(C::B_QE), (nq - 1) & 1, abort_flag)) return false;
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
      for (int s = 0; s < passes * n_ch; ++s) {
        const int ch = s % n_ch, ks = nk % 2;
        if (nk >= 2 && !warp_wait(bar(C::B_KE + ks), ((nk - 2) / 2) & 1, abort_flag)) return false;
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
      return true;
    };
    bool ok = true;
    for (int pair = 0; ok && pair < n_pairs; ++pair) ok = job(pair, kFastPasses);
    uint32_t mask = 0u;
    if (ok) {
      ok = warp_wait(bar(C::B_DEC), 0, abort_flag);
      if (ok) mask = *reinterpret_cast<volatile uint32_t*>(overflowed);
    }
    for (int pair = 0; ok && pair < n_pairs; ++pair)
      if (redo(mask, pair)) ok = job(pair, kRadixPasses);
    if (!ok && lane == 0) record_failure(abort_flag, L.status);
    // no copy in flight at exit: the last Q and k_bar loads have landed
    const volatile int never = 0;
    if (nq > 0) ptx::mbar_wait(bar(C::B_QF), (nq - 1) & 1, &never, kWaitTimeoutNs);
    for (int s = 0; s < 2 && s < nk; ++s)
      ptx::mbar_wait(bar(C::B_KF + s), ((nk - 1 - s) / 2) & 1, &never, kWaitTimeoutNs);
  } else if (warp == kWarpMma) {
    constexpr uint32_t kIdesc = ptx::idesc_bf16_f32(kRows, kCols, false, false);
    uint32_t leader = 0;
    int first_leader = -1, nj = 0, t = 0;
    bool same = true, issued = false;
    auto job = [&](int pair, int passes) -> bool {
      if (n_ch == 0) return true;                // as the producer: no Q, no steps
      const int nheads = min(kHeadSlots, gq - pair * kHeadSlots);
      for (int s = 0; s < passes * n_ch; ++s, ++t) {
        const int b = t % 2;
        if ((s == 0 && !warp_wait(bar(C::B_QF), nj & 1, abort_flag)) ||
            !warp_wait(bar(C::B_KF + t % 2), (t / 2) & 1, abort_flag) ||
            (t >= 2 && !warp_wait(bar(C::B_SE + b), ((t - 2) / 2) & 1, abort_flag)))
          return false;
        ptx::tc_fence_after();
        const bool me = ptx::elect_one(leader);
        if (first_leader < 0) first_leader = static_cast<int>(leader);
        same = same && static_cast<int>(leader) == first_leader;
        if (me && same) {
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
          if (s == passes * n_ch - 1) ptx::mma_commit(bar(C::B_QE));
        }
        __syncwarp();
        issued = true;
        if (!same) return false;
      }
      ++nj;
      return true;
    };
    bool ok = true;
    for (int pair = 0; ok && pair < n_pairs; ++pair) ok = job(pair, kFastPasses);
    uint32_t mask = 0u;
    if (ok) {
      ok = warp_wait(bar(C::B_DEC), 0, abort_flag);
      if (ok) mask = *reinterpret_cast<volatile uint32_t*>(overflowed);
    }
    for (int pair = 0; ok && pair < n_pairs; ++pair)
      if (redo(mask, pair)) ok = job(pair, kRadixPasses);
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
    const float nsc = -sc;
    constexpr int kStash = kRows * kHeadSlots;   // this thread's column: stash[e * kStash]
    float* stash = reinterpret_cast<float*>(smem + C::OFF_STASH) + slot * kRows + row;
    int* list_id = reinterpret_cast<int*>(smem + C::OFF_LIST_ID) + slot * kRows + row;
    float4* group_u = reinterpret_cast<float4*>(smem + C::OFF_GROUP_U) + (slot * kRows + row) * 8;
    const int swz = row & 7;
    bool ok = true;
    int t = 0;                                   // chunk steps consumed

    // ---- fast path ----
    // Per pair: (0) the largest and smallest S over H_i; with m = max x
    // rounded up, u = m - x >= 0 for every block (one fma, exact sign) and the
    // floored key 2^23 + floor(u inv_r) is one fma rounded toward zero, with
    // inv_r = 2^14 / (max - min) in log2 units. (1, 2) two 3-bit digits of the
    // key, each from the cumulative masses below the tops of the window's
    // digit values (the first pass also sums Z); the boundary digit is the
    // first whose cumulative mass reaches tau_p Z; (3) collect: a block whose
    // key is below the window is kept, one in the window is listed (u, id), one
    // above it dropped. Then the list, ordered by u (ties: id order), is walked
    // from the mass below the window: a block is kept while the mass before it
    // is below tau_p Z. A row whose window holds more than kListCap blocks
    // flags the pair for the radix path.
    for (int pair = 0; pair < n_pairs; ++pair) {
      const int hh = pair * kHeadSlots + slot;
      const bool active = hh < gq;               // warp-uniform: an odd group leaves the last slot idle
      const int h = g * gq + min(hh, gq - 1);
      uint32_t* keep = L.keep + static_cast<int64_t>(h) * L.n_words * L.n_tok + rt.q_start + row;
      float smax = -INFINITY, smin = INFINITY, m = 0.f, inv_r = 0.f, z = 0.f, target = 0.f, above = 0.f;
      float lo = 0.f, hi = INFINITY;             // the window: keys lo .. hi - 1 (hi = +inf: up to the last key)
      int count = 0;                             // window blocks met by the collect pass
      for (int pass = 0; pass < kFastPasses; ++pass) {
        const float dstep = pass == 1 ? 2048.f : 256.f;   // keys per digit value
        float top[kFastTops], cm[kFastTops];
#pragma unroll
        for (int k = 0; k < kFastTops; ++k) {
          top[k] = kMagic + (lo + dstep * static_cast<float>(k + 1));
          cm[k] = 0.f;
        }
        for (int ch = 0; ch < n_ch; ++ch, ++t) {
          const int b = t % 2;
          ok = ok && warp_wait(bar(C::B_SF + b), (t / 2) & 1, abort_flag);
          if (ok && active && __any_sync(0xffffffffu, nh > ch * kCols)) {   // warp-uniform: tcgen05.ld is collective
            ptx::tc_fence_after();
#pragma unroll 1
            for (int c0 = 0; c0 < kCols; c0 += 32) {
              const int jn = nh - (ch * kCols + c0);         // columns e < jn are in H_i
              // past every row's H_i only the collect pass has words to write
              if (pass < kFastPasses - 1 && !__any_sync(0xffffffffu, jn > 0)) break;
              uint32_t r[32];
              ptx::tmem_ld32(tbase + b * kHeadSlots * kCols + c0, r);
              ptx::tmem_wait_ld();
              if (pass == 0) {
                float mx[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
                float mn[4] = {INFINITY, INFINITY, INFINITY, INFINITY};
#pragma unroll
                for (int e = 0; e < 32; ++e) {
                  if (e < jn) {
                    mx[e & 3] = fmaxf(mx[e & 3], __uint_as_float(r[e]));
                    mn[e & 3] = fminf(mn[e & 3], __uint_as_float(r[e]));
                  }
                }
                smax = fmaxf(smax, fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])));
                smin = fminf(smin, fminf(fminf(mn[0], mn[1]), fminf(mn[2], mn[3])));
              } else if (pass < kFastPasses - 1) {
                // u and the key by explicit roundings, so that every pass and
                // the list see the same values.
                // two columns per packed fma for u and the key
                const bool full = __all_sync(0xffffffffu, jn >= 32);
#pragma unroll
                for (int e = 0; e < 32; e += 2) {
                  float u0, u1, f0, f1;
                  fma2_rn(u0, u1, __uint_as_float(r[e]), __uint_as_float(r[e + 1]), nsc, nsc, m, m);
                  fma2_rz(f0, f1, u0, u1, inv_r, inv_r, kMagic, kMagic);
                  const float w0 = full || e < jn ? ptx::ex2(-u0) : 0.f;
                  const float w1 = full || e + 1 < jn ? ptx::ex2(-u1) : 0.f;
                  if (pass == 1) {
                    cum_add<kFastTops, true>(cm, top, f0, w0, z);
                    cum_add<kFastTops, true>(cm, top, f1, w1, z);
                  } else {
                    cum_add(cm, top, f0, w0, z);
                    cum_add(cm, top, f1, w1, z);
                  }
                }
              } else {
                // Kept (key < lo) and in-or-below-window (key < hi) as bit words
                // summed in fp32 from saturated indicators (exact: 16 bits a
                // half); u goes to the group scratch for the window's blocks.
                const float t_lo = kMagic + lo, t_hi = kMagic + hi;
                float k0 = 0.f, k1 = 0.f, h0 = 0.f, h1 = 0.f;
#pragma unroll
                for (int e4 = 0; e4 < 8; ++e4) {
                  float uu[4];
#pragma unroll
                  for (int i = 0; i < 4; i += 2) {
                    const int e = e4 * 4 + i;
                    float f[2];
                    fma2_rn(uu[i], uu[i + 1], __uint_as_float(r[e]), __uint_as_float(r[e + 1]), nsc, nsc, m, m);
                    fma2_rz(f[0], f[1], uu[i], uu[i + 1], inv_r, inv_r, kMagic, kMagic);
#pragma unroll
                    for (int j = 0; j < 2; ++j) {
                      float ik, ih;
                      asm("sub.sat.f32 %0, %1, %2;" : "=f"(ik) : "f"(t_lo), "f"(f[j]));
                      asm("sub.sat.f32 %0, %1, %2;" : "=f"(ih) : "f"(t_hi), "f"(f[j]));
                      const float pw = static_cast<float>(1u << ((e + j) & 15));
                      if (e < 16) fma2_rn(k0, h0, ik, ih, pw, pw, k0, h0);
                      else fma2_rn(k1, h1, ik, ih, pw, pw, k1, h1);
                    }
                  }
                  group_u[e4 ^ swz] = make_float4(uu[0], uu[1], uu[2], uu[3]);
                }
                const uint32_t valid = jn >= 32 ? 0xffffffffu : jn > 0 ? (1u << jn) - 1u : 0u;
                uint32_t word = (__float2uint_rz(k0) | (__float2uint_rz(k1) << 16)) & valid;
                uint32_t in_win = (__float2uint_rz(h0) | (__float2uint_rz(h1) << 16)) & valid & ~word;
                while (in_win != 0u) {
                  const int e = __ffs(in_win) - 1;
                  in_win &= in_win - 1u;
                  if (count < kListCap) {
                    stash[count * kStash] = reinterpret_cast<const float*>(group_u + ((e >> 2) ^ swz))[e & 3];
                    list_id[count * kStash] = ch * kCols + c0 + e;
                  }
                  ++count;
                }
                const int w = ch * 4 + (c0 >> 5);
                if (row_ok && w < L.n_words) {
                  if (w == nh >> 5) word |= 1u << (nh & 31);     // the row's own block
                  keep[static_cast<int64_t>(w) * L.n_tok] = word;
                }
              }
            }
            ptx::tc_fence_before();
          } else if (pass == kFastPasses - 1 && row_ok && ok && active) {
            // No column of this chunk is in H_i for the warp: zeros (and the own block).
            for (int wi = 0; wi < 4; ++wi) {
              const int w = ch * 4 + wi;
              if (w >= L.n_words) break;
              keep[static_cast<int64_t>(w) * L.n_tok] = w == nh >> 5 ? 1u << (nh & 31) : 0u;
            }
          }
          ptx::mbar_arrive(bar(C::B_SE + b));
        }
        if (pass == 0) {
          m = __fmul_ru(smax, sc);               // >= every x of H_i, so u >= 0
          inv_r = static_cast<float>(kQMax + 1) / fmaxf(__fmul_rn(__fsub_rn(smax, smin), sc), 1e-30f);
        } else if (pass < kFastPasses - 1) {
          if (pass == 1) target = L.tau * z;
          // the first digit value whose cumulative mass reaches the target; else
          // (the last digit holds it, or rounding keeps every sum below it) the last
          int d = kFastBins - 1;
#pragma unroll
          for (int k = kFastTops - 1; k >= 0; --k)
            if (cm[k] >= target) d = k;
          float below = above;                   // the mass below digit d
#pragma unroll
          for (int k = 0; k < kFastTops; ++k)
            if (k + 1 == d) below = cm[k];
          above = below;
          const float nlo = lo + dstep * static_cast<float>(d);
          hi = d + 1 < kFastBins ? lo + dstep * static_cast<float>(d + 1) : hi;
          lo = nlo;
        }
      }
      if (ok && active && row_ok && count > 0) {
        if (count > kListCap) {
          atomicOr(overflowed, 1u << min(pair, 31));
        } else {
          // The window's last 8 key bits from the list (in id order): two 4-bit
          // digits by cumulative masses, as the passes take theirs; then every
          // listed block below the boundary key is kept and, at it, blocks in id
          // order while the mass before them is below the target.
          const float base = above;              // the mass below the listed window
#pragma unroll 1
          for (int lev = 0; lev < 2; ++lev) {
            const float dstep = lev == 0 ? 16.f : 1.f;
            float top[15], cm[15];               // cm[k]: mass of the blocks with key below top[k]
#pragma unroll
            for (int k = 0; k < 15; ++k) {
              top[k] = kMagic + (lo + dstep * static_cast<float>(k + 1));
              cm[k] = base;
            }
            for (int i = 0; i < count; ++i) {
              const float u = stash[i * kStash];
              float unused = 0.f;
              cum_add(cm, top, __fmaf_rz(u, inv_r, kMagic), ptx::ex2(-u), unused);
            }
            int d = 15;
#pragma unroll
            for (int k = 14; k >= 0; --k)
              if (cm[k] >= target) d = k;
            float below = above;
#pragma unroll
            for (int k = 0; k < 15; ++k)
              if (k + 1 == d) below = cm[k];
            above = below;
            hi = d < 15 ? lo + dstep * static_cast<float>(d + 1) : hi;
            lo = lo + dstep * static_cast<float>(d);
          }
          const float t_lo = kMagic + lo, t_hi = kMagic + hi;   // the boundary key (up to the last at the top)
          float tie = 0.f;
          for (int i = 0; i < count; ++i) {
            const float u = stash[i * kStash];
            const float f = __fmaf_rz(u, inv_r, kMagic);
            bool kept = f < t_lo;
            if (f >= t_lo && f < t_hi) {
              kept = above + tie < target;
              tie = __fadd_rn(tie, ptx::ex2(-u));
            }
            if (kept) {
              const int id = list_id[i * kStash];
              atomicOr(keep + static_cast<int64_t>(id >> 5) * L.n_tok, 1u << (id & 31));
            }
          }
        }
      }
      __syncwarp();
      // The own block's word when it lies past the chunks of this tile.
      if (row_ok && ok && active && (nh >> 5) >= n_ch * 4 && (nh >> 5) < L.n_words)
        keep[static_cast<int64_t>(nh >> 5) * L.n_tok] = 1u << (nh & 31);
    }
    __syncwarp();
    if (lane == 0) ptx::mbar_arrive(bar(C::B_DEC));
    uint32_t mask = 0u;
    if (ok) {
      ok = warp_wait(bar(C::B_DEC), 0, abort_flag);
      if (ok) mask = *reinterpret_cast<volatile uint32_t*>(overflowed);
    }
    // ---- radix path, for the pairs some row flagged ----
    for (int pair = 0; ok && pair < n_pairs; ++pair) {
      if (!redo(mask, pair)) continue;
      const int hh = pair * kHeadSlots + slot;
      const bool active = hh < gq;               // warp-uniform: an odd group leaves the last slot idle
      const int h = g * gq + min(hh, gq - 1);
      float m = -INFINITY, gmin = INFINITY, z = 0.f;
      float inv_r = 0.f, target = 0.f, above = 0.f, tie = 0.f;
      int wkey = 0;                              // the boundary's key digits found so far
      uint32_t* keep = L.keep + static_cast<int64_t>(h) * L.n_words * L.n_tok + rt.q_start + row;
      for (int pass = 0; pass < kRadixPasses; ++pass) {
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
        for (int ch = 0; ch < n_ch; ++ch, ++t) {
          const int b = t % 2;
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
          } else if (pass == kRadixPasses - 1 && row_ok && ok && active) {
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

// Keeps bit 0 of every BPT-bit group of x (the group's OR after or_fold),
// packed into the low 32 / BPT bits.
template <int BPT>
__device__ __forceinline__ uint32_t or_fold(uint32_t x) {
#pragma unroll
  for (int k = 1; k < BPT; k <<= 1) x |= x >> k;
  return x;
}
template <int BPT>
__device__ __forceinline__ uint32_t compress(uint32_t x) {
  if constexpr (BPT == 1) {
    return x;
  } else if constexpr (BPT == 2) {
    x &= 0x55555555u;
    x = (x | (x >> 1)) & 0x33333333u;
    x = (x | (x >> 2)) & 0x0f0f0f0fu;
    x = (x | (x >> 4)) & 0x00ff00ffu;
    return (x | (x >> 8)) & 0x0000ffffu;
  } else if constexpr (BPT == 4) {
    x &= 0x11111111u;
    x = (x | (x >> 3)) & 0x03030303u;
    x = (x | (x >> 6)) & 0x000f000fu;
    return (x | (x >> 12)) & 0x000000ffu;
  } else {
    static_assert(BPT == 8, "blocks per key tile: 1, 2, 4 or 8");
    x &= 0x01010101u;
    x = (x | (x >> 7)) & 0x00030003u;
    return (x | (x >> 14)) & 0x0000000fu;
  }
}

constexpr int kUnionWords = 32;                  // keep words (1,024 blocks) per union CTA

// blockIdx.x: builder row tile (visual rows), blockIdx.y: a chunk of 32 keep
// words, i.e. 32 / BPT words of the union. A thread ORs its row's words over
// the heads (32 independent loads per head), masks them to the visual blocks,
// folds blocks into key tiles, the warps OR their rows (shuffles, then shared
// memory), and one thread stores each union word of each attention row tile
// the CTA covers (one writer per word: no atomics).
template <int BPT>
__global__ void __launch_bounds__(128) topp_union_kernel(const __grid_constant__ ToppLaunch L) {
  constexpr int kTileWords = kUnionWords / BPT;
  __shared__ uint32_t part[4][kTileWords];
  const ToppRowTile rt = L.tiles[blockIdx.x];
  if (rt.text) return;                           // the attention takes tile masks for visual rows only
  const ToppVideo vid = L.vids[rt.video];
  const int nvb = vid.n_vis / L.block;           // visual blocks (visual rows keep no text block)
  const int w0 = blockIdx.y * kUnionWords;
  if (w0 * 32 >= nvb) return;                    // uniform: no visual block in this chunk
  const int row = threadIdx.x, lane = row & 31, warp = row >> 5;
  const bool row_ok = row < rt.q_len;
  uint32_t acc[kUnionWords];
#pragma unroll
  for (int i = 0; i < kUnionWords; ++i) acc[i] = 0u;
  if (row_ok) {
    const uint32_t* kp = L.keep + static_cast<int64_t>(w0) * L.n_tok + rt.q_start + row;
    for (int h = 0; h < L.hq; ++h) {
      const uint32_t* kh = kp + static_cast<int64_t>(h) * L.n_words * L.n_tok;
#pragma unroll
      for (int i = 0; i < kUnionWords; ++i)
        if (w0 + i < L.n_words) acc[i] |= kh[static_cast<int64_t>(i) * L.n_tok];
    }
  }
  uint32_t tw[kTileWords];
#pragma unroll
  for (int j = 0; j < kTileWords; ++j) {
    uint32_t bits = 0u;
#pragma unroll
    for (int q = 0; q < BPT; ++q) {
      const int i = j * BPT + q, b0 = (w0 + i) * 32;   // blocks b0 .. b0 + 31
      uint32_t x = acc[i];
      if (b0 + 32 > nvb) x &= b0 < nvb ? (1u << (nvb - b0)) - 1u : 0u;
      bits |= compress<BPT>(or_fold<BPT>(x)) << (q * (32 / BPT));
    }
    tw[j] = __reduce_or_sync(0xffffffffu, bits);
  }
  // Attention row tiles: TILE = 128 is the CTA's rows; TILE = 64 gives warps
  // 0-1 and 2-3 a tile each (the builder's tiles start at multiples of 128).
  if (lane == 0) {
#pragma unroll
    for (int j = 0; j < kTileWords; ++j) part[warp][j] = tw[j];
  }
  __syncthreads();
  const int wpt = L.tile / 32;                   // warps per attention row tile
  const int n_at = (rt.q_len + L.tile - 1) / L.tile;
  const int t = threadIdx.x / kTileWords, j = threadIdx.x % kTileWords;
  if (t < n_at) {
    uint32_t bits = 0u;
    for (int ww = t * wpt; ww < (t + 1) * wpt; ++ww) bits |= part[ww][j];
    const int tile_word = w0 / BPT + j;
    if (tile_word < L.n_tile_words)
      L.tile_union[static_cast<int64_t>(vid.row_tile0 + rt.local0 / L.tile + t) * L.n_tile_words + tile_word] = bits;
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
    dim3 grid(L.n_tiles, (L.n_words + kUnionWords - 1) / kUnionWords);
    const int bpt = L.tile / L.block;
    if (bpt == 1) topp_union_kernel<1><<<grid, 128, 0, stream>>>(L);
    else if (bpt == 2) topp_union_kernel<2><<<grid, 128, 0, stream>>>(L);
    else if (bpt == 4) topp_union_kernel<4><<<grid, 128, 0, stream>>>(L);
    else if (bpt == 8) topp_union_kernel<8><<<grid, 128, 0, stream>>>(L);
    else return cudaErrorInvalidValue;
    return cudaGetLastError();
  }
  return cudaSuccess;
}

}  // namespace evisel
