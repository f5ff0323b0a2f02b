// Block-sparse, causal, grouped-query, varlen prefill attention for sm_103a
// (the paper's sparse probe, Sec. 3.2 Eq. 1, with exact token logits on every
// kept tile: Appendix Eq. 8 in token form and the row normalisation of Eq. 11).
//
// One CTA computes one work item: a query row tile against a list of kept kv
// tiles for two "slots" of query heads of one KV group. A slot is one 128-row
// MMA tile (one head for 128-token tiles, two heads for 64-token tiles); both
// slots use every K/V tile the CTA loads, and each slot's softmax runs while
// the tensor core works on the other slot.
//
// Warp roles (352 threads):
//   warps 0-3  softmax + epilogue of slot 0, one thread per query row (TMEM lane)
//   warps 4-7  softmax + epilogue of slot 1
//   warp 8     block set-up (mbarriers) and the loads of Q (both slots) and
//              K_0, before the block-wide barrier; then K_j into an NS-deep ring
//   warp 10    TMA: V_j into an NS-deep ring (apart from K, so that K tiles
//              run ahead of the V waits)
//   warp 9     MMA issuer; the warp walks the tiles together and one elected
//              lane issues, per kv tile j:
//                O0 += P0_j V_j,  S0_{j+1} = Q0 K_{j+1}^T,
//                O1 += P1_j V_j,  S1_{j+1} = Q1 K_{j+1}^T
// TMEM columns per slot: S (TILE) | O (D). P_j (bf16) is written over the
// first half of its own S_j columns and read from there by the P.V MMA; the
// slot's next S is issued after that P.V, and the tcgen05 MMAs of one thread
// execute in issue order. An item with one slot (the last heads of a KV group
// with an odd head count) uses the idle slot's S columns as a second S
// buffer: S_{j+1} is computed while the softmax works on S_j.
// Online softmax in fp32 (log2 domain) with lazy rescaling: the running max is
// only moved when it grows by more than 2^8, so O in TMEM is rescaled rarely.
// Text row tiles also spill their logits onto visual keys for the evidence
// pass. Every wait is bounded; on timeout the CTA records EVISEL_ETIMEOUT,
// drains its own async work and exits.
#include <cstdint>
#include <cuda_runtime.h>

#include "evisel_internal.h"
#include "sm103_ptx.cuh"

namespace evisel {
namespace {

static_assert(kSlots == 2, "the kernel runs two slots per work item");
constexpr int kThreads = 352;
constexpr int kWarpProducer = 8;   // Q, then the K ring
constexpr int kWarpMma = 9;
constexpr int kWarpVLoader = 10;   // the V ring
constexpr int kRows = 128;
constexpr float kRescaleThreshold = 8.0f;   // log2 units
constexpr float kLn2 = 0.69314718055994531f;

template <int TILE, int D, int NS>
struct Cfg {
  static constexpr int HP = kRows / TILE;        // query heads per slot
  static constexpr int KB = D / 64;              // 128-byte swizzle column blocks along d
  static constexpr int Q_BYTES = kRows * D * 2;  // one slot
  static constexpr int Q_BLOCK = kRows * 128;    // one column block of a slot's Q
  static constexpr int KV_BLOCK = TILE * 128;    // one column block of a K/V tile
  static constexpr int KV_BYTES = TILE * D * 2;
  static constexpr int OFF_Q = 0;                        // two slots
  static constexpr int OFF_K = OFF_Q + 2 * Q_BYTES;
  static constexpr int OFF_V = OFF_K + NS * KV_BYTES;
  static constexpr int OFF_BAR = OFF_V + NS * KV_BYTES;
  // barrier indices
  static constexpr int B_Q = 0;
  static constexpr int B_KF = 1;             // NS: K tile landed
  static constexpr int B_KE = B_KF + NS;     // NS: K tile consumed by both S MMAs
  static constexpr int B_VF = B_KE + NS;     // NS: V tile landed
  static constexpr int B_VE = B_VF + NS;     // NS: V tile consumed by both P.V MMAs
  static constexpr int B_SF = B_VE + NS;     // 2 (per slot): S_j computed
  static constexpr int B_PF = B_SF + 2;      // 2 (per slot): P_j written (128 arrivals)
  static constexpr int B_OF = B_PF + 2;      // 2 (per slot): O complete
  static constexpr int B_DRAIN = B_OF + 2;
  static constexpr int N_BARS = B_DRAIN + 1;
  static constexpr int OFF_MISC = OFF_BAR + N_BARS * 8;
  static constexpr int SMEM_USED = OFF_MISC + 16;
  // TMEM columns (32-bit): slot s occupies [s * SLOT_COLS, (s + 1) * SLOT_COLS)
  static constexpr int SLOT_COLS = TILE + D;
  static constexpr int COL_S = 0;
  static constexpr int COL_O = TILE;
  static constexpr int TMEM_COLS = (2 * SLOT_COLS <= 256) ? 256 : 512;
  // Dynamic smem requested: enough to keep TMEM demand per SM within 512 columns.
  static constexpr int SMEM_MIN = TMEM_COLS == 512 ? 117 * 1024 : 78 * 1024;
  static constexpr int SMEM_BYTES = (SMEM_USED + 1024 > SMEM_MIN) ? SMEM_USED + 1024 : SMEM_MIN;
  static_assert(SMEM_USED + 1024 <= 232448, "shared memory budget");
  static_assert((OFF_K % 1024) == 0 && (OFF_V % 1024) == 0 && (KV_BYTES % 1024) == 0, "1 KB aligned tiles");
  static_assert(2 * SLOT_COLS <= 512, "TMEM budget");
};

__device__ __forceinline__ void record_failure(volatile int* abort_flag, int* status, int code) {
  *abort_flag = 1;
  atomicExch(status, code);
}

// Bounded wait whose outcome is uniform across the warp, so that the warp stays
// converged for the warp-collective tcgen05 operations that follow.
__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag) {
  const bool ok = ptx::mbar_wait(bar, parity, abort_flag, kWaitTimeoutNs);
  return __all_sync(0xffffffffu, ok);
}

// Heads of the item's KV group from its first head on.
__device__ __forceinline__ int heads_left(const ProbeLaunch& L, int head) {
  const int gq = L.hq / L.hkv;
  return gq - head % gq;
}

// Block set-up by the K loader's first lane, before the block-wide barrier:
// the mbarriers and the abort flag, then the loads that the first S MMAs
// wait for (Q of both slots and K tile 0), so that their latency overlaps the
// TMEM allocation and the barrier instead of following them.
template <int TILE, int D, int NS>
__device__ __forceinline__ void setup_and_first_loads(const ProbeLaunch& L, const WorkItem& it, uint32_t sbase,
                                                      volatile int* abort_flag) {
  using C = Cfg<TILE, D, NS>;
  auto bar = [&](int i) { return sbase + C::OFF_BAR + 8u * i; };
  for (int i = 0; i < C::N_BARS; ++i) {
    const bool softmax_arrive = (i == C::B_PF || i == C::B_PF + 1);
    ptx::mbar_init(bar(i), softmax_arrive ? kRows : 1u);
  }
  *abort_flag = 0;
  ptx::fence_mbar_init();
  ptx::tma_prefetch_desc(&L.tm_q);
  ptx::tma_prefetch_desc(&L.tm_k);
  ptx::tma_prefetch_desc(&L.tm_v);
  const int left = heads_left(L, it.head);
  const int nslots = left > C::HP ? 2 : 1;
  const uint64_t pol_q = ptx::l2_policy_evict_first();
  ptx::mbar_arrive_expect_tx(bar(C::B_Q), nslots * C::Q_BYTES);
  for (int slot = 0; slot < nslots; ++slot) {
#pragma unroll
    for (int hp = 0; hp < C::HP; ++hp) {
      // A head past the group's end loads the first head again; its rows are never stored.
      const int h = slot * C::HP + hp < left ? it.head + slot * C::HP + hp : it.head;
#pragma unroll
      for (int kb = 0; kb < C::KB; ++kb)
        ptx::tma_load_3d(sbase + C::OFF_Q + slot * C::Q_BYTES + kb * C::Q_BLOCK + hp * TILE * 128, &L.tm_q,
                         bar(C::B_Q), kb * 64, h, it.q_start, pol_q);
    }
  }
  if (it.kv_count > 0) {
    const int g = it.head / (L.hq / L.hkv);
    ptx::mbar_arrive_expect_tx(bar(C::B_KF), C::KV_BYTES);
#pragma unroll
    for (int kb = 0; kb < C::KB; ++kb)
      ptx::tma_load_3d(sbase + C::OFF_K + kb * C::KV_BLOCK, &L.tm_k, bar(C::B_KF), kb * 64, g,
                       L.kv[it.kv_begin].start, ptx::l2_policy_evict_last());
  }
}

// One TMA warp per ring, so that K tiles run ahead of the V waits. Q and K
// tile 0 were sent by setup_and_first_loads; the K warp goes on from K tile 1.
template <int TILE, int D, int NS, bool IS_V>
__device__ __forceinline__ void producer(const ProbeLaunch& L, const WorkItem& it, uint32_t sbase_in,
                                         volatile int* abort_flag) {
  using C = Cfg<TILE, D, NS>;
  const uint32_t sbase = __shfl_sync(0xffffffffu, sbase_in, 0);
  auto bar = [&](int i) { return sbase + C::OFF_BAR + 8u * i; };
  const int head0 = __shfl_sync(0xffffffffu, it.head, 0);
  const int n = __shfl_sync(0xffffffffu, it.kv_count, 0);
  const int kv_begin = __shfl_sync(0xffffffffu, it.kv_begin, 0);
  const int g = head0 / (L.hq / L.hkv);
  const uint64_t pol_kv = ptx::l2_policy_evict_last();
  uint32_t leader = 0;

  const CUtensorMap* map = IS_V ? &L.tm_v : &L.tm_k;
  const int off = IS_V ? C::OFF_V : C::OFF_K;
  const int b_full = IS_V ? C::B_VF : C::B_KF;
  const int b_empty = IS_V ? C::B_VE : C::B_KE;
  const int first = (IS_V || n == 0) ? 0 : 1;   // K tile 0 went out with the set-up
  int issued = first;
  for (int j = first; j < n; ++j) {
    const int s = j % NS;
    const int u = j / NS;
    const int kv_start = __shfl_sync(0xffffffffu, L.kv[kv_begin + j].start, 0);
    if (u > 0 && !warp_wait(bar(b_empty + s), (u - 1) & 1, abort_flag)) {
      if ((threadIdx.x & 31) == leader) record_failure(abort_flag, L.status, kStatusTimeout);
      break;
    }
    if (ptx::elect_one(leader)) {
      ptx::mbar_arrive_expect_tx(bar(b_full + s), C::KV_BYTES);
#pragma unroll
      for (int kb = 0; kb < C::KB; ++kb)
        ptx::tma_load_3d(sbase + off + s * C::KV_BYTES + kb * C::KV_BLOCK, map, bar(b_full + s), kb * 64, g, kv_start,
                         pol_kv);
    }
    __syncwarp();
    issued = j + 1;
  }
  {
    // Drain: every load issued here completes on its own; wait for the last
    // phase issued into each stage (and for Q) so that no copy is in flight
    // when the CTA exits, whether or not another warp gave up.
    const volatile int never = 0;
    if (!IS_V) ptx::mbar_wait(bar(C::B_Q), 0, &never, kWaitTimeoutNs);
    for (int s = 0; s < NS && s < issued; ++s) {
      const int last = ((issued - 1 - s) / NS) * NS + s;
      ptx::mbar_wait(bar(b_full + s), (last / NS) & 1, &never, kWaitTimeoutNs);
    }
  }
}

// The whole warp walks the tiles on warp-uniform values; one elected lane
// issues every MMA and commit. tcgen05.commit tracks the MMAs of the thread
// that issues it, so the lane must not change: elect.sync picks the same lane
// of a converged warp, and a change is treated as a failure.
template <int TILE, int D, int NS>
__device__ __forceinline__ void mma_issuer(const ProbeLaunch& L, const WorkItem& it, uint32_t sbase_in,
                                           uint32_t tmem_in, volatile int* abort_flag) {
  using C = Cfg<TILE, D, NS>;
  const uint32_t sbase = __shfl_sync(0xffffffffu, sbase_in, 0);
  const uint32_t tmem = __shfl_sync(0xffffffffu, tmem_in, 0);
  const int n = __shfl_sync(0xffffffffu, it.kv_count, 0);
  const bool two = heads_left(L, __shfl_sync(0xffffffffu, it.head, 0)) > C::HP;
  auto bar = [&](int i) { return sbase + C::OFF_BAR + 8u * i; };
  constexpr uint32_t kIdescS = ptx::idesc_bf16_f32(kRows, TILE, false, false);
  constexpr uint32_t kIdescO = ptx::idesc_bf16_f32(kRows, D, false, true);
  uint32_t leader = 0;
  int first_leader = -1;
  bool same_leader = true;
  auto elect = [&]() -> bool {
    const bool me = ptx::elect_one(leader);
    if (first_leader < 0) first_leader = static_cast<int>(leader);
    same_leader = same_leader && static_cast<int>(leader) == first_leader;
    return me && same_leader;
  };
  // Descriptors of every operand buffer, built once; a k-step adds its byte
  // offset / 16 to the address field (the lowest bits; smem offsets < 256 KB
  // never carry out of it).
  const uint64_t dq0 = ptx::sdesc_sw128(sbase + C::OFF_Q, 16, 1024);
  const uint64_t dq1 = ptx::sdesc_sw128(sbase + C::OFF_Q + C::Q_BYTES, 16, 1024);
  const uint64_t dk0 = ptx::sdesc_sw128(sbase + C::OFF_K, 16, 1024);
  const uint64_t dk1 = ptx::sdesc_sw128(sbase + C::OFF_K + C::KV_BYTES, 16, 1024);
  const uint64_t dv0 = ptx::sdesc_sw128(sbase + C::OFF_V, C::KV_BLOCK, 1024);
  const uint64_t dv1 = ptx::sdesc_sw128(sbase + C::OFF_V + C::KV_BYTES, C::KV_BLOCK, 1024);
  static_assert(NS == 2, "two ring stages");
  // S[buf] = Q_slot K_j^T (buf: whose S columns receive it)
  auto mma_s = [&](int slot, int j, int buf) {
    const uint64_t qd = slot ? dq1 : dq0;
    const uint64_t kd = (j & 1) ? dk1 : dk0;
    const uint32_t d_tmem = tmem + buf * C::SLOT_COLS + C::COL_S;
#pragma unroll
    for (int kk = 0; kk < D / 16; ++kk) {
      const uint64_t a = qd + static_cast<uint64_t>(((kk / 4) * C::Q_BLOCK + (kk % 4) * 32) >> 4);
      const uint64_t bd = kd + static_cast<uint64_t>(((kk / 4) * C::KV_BLOCK + (kk % 4) * 32) >> 4);
      ptx::mma_ss(d_tmem, a, bd, kIdescS, kk > 0 ? 1u : 0u);
    }
  };
  // O_slot += P V_j, P from the first TILE/2 columns of S[buf].
  auto mma_pv = [&](int slot, int j, int buf) {
    const uint64_t vd = (j & 1) ? dv1 : dv0;
    const uint32_t d_tmem = tmem + slot * C::SLOT_COLS + C::COL_O;
    const uint32_t p_tmem = tmem + buf * C::SLOT_COLS + C::COL_S;
#pragma unroll
    for (int kk = 0; kk < TILE / 16; ++kk) {
      const uint64_t bd = vd + static_cast<uint64_t>((kk * 16 * 128) >> 4);
      ptx::mma_ts(d_tmem, p_tmem + kk * 8, bd, kIdescO, (j > 0 || kk > 0) ? 1u : 0u);
    }
  };

  bool issued = false;
  bool ok = warp_wait(bar(C::B_Q), 0, abort_flag) && warp_wait(bar(C::B_KF), 0, abort_flag);
  if (!two) {
    // One slot: the second slot's S columns double-buffer S, so S_{j+1} is
    // ready while the softmax works on S_j. Tile j uses buffer b = j & 1
    // (barriers SF[b] / PF[b], phase j >> 1); S_{j+2} reuses b after P_j.V.
    if (ok) {
      ptx::tc_fence_after();
      if (elect()) {
        mma_s(0, 0, 0);
        ptx::mma_commit(bar(C::B_SF));
        ptx::mma_commit(bar(C::B_KE));
      }
      __syncwarp();
      issued = true;
      ok = same_leader;
    }
    if (ok && n > 1) {
      if (!warp_wait(bar(C::B_KF + 1 % NS), (1 / NS) & 1, abort_flag)) {
        ok = false;
      } else {
        if (elect()) {
          mma_s(0, 1, 1);
          ptx::mma_commit(bar(C::B_SF + 1));
          ptx::mma_commit(bar(C::B_KE + 1 % NS));
        }
        __syncwarp();
        ok = same_leader;
      }
    }
    for (int j = 0; ok && j < n; ++j) {
      const int b = j & 1;
      const int s = j % NS;
      const int s2 = (j + 2) % NS;
      const bool more = j + 2 < n;
      if ((more && !warp_wait(bar(C::B_KF + s2), ((j + 2) / NS) & 1, abort_flag)) ||
          !warp_wait(bar(C::B_VF + s), (j / NS) & 1, abort_flag) ||
          !warp_wait(bar(C::B_PF + b), (j >> 1) & 1, abort_flag)) {
        ok = false;
        break;
      }
      ptx::tc_fence_after();
      if (elect()) {
        mma_pv(0, j, b);
        if (j + 1 == n) ptx::mma_commit(bar(C::B_OF));
        ptx::mma_commit(bar(C::B_VE + s));
        if (more) {
          mma_s(0, j + 2, b);
          ptx::mma_commit(bar(C::B_SF + b));
          ptx::mma_commit(bar(C::B_KE + s2));
        }
      }
      __syncwarp();
      ok = same_leader;
    }
  } else {
    if (ok) {
      ptx::tc_fence_after();
      if (elect()) {
        mma_s(0, 0, 0);
        ptx::mma_commit(bar(C::B_SF));
        mma_s(1, 0, 1);
        ptx::mma_commit(bar(C::B_SF + 1));
        ptx::mma_commit(bar(C::B_KE));
      }
      __syncwarp();
      issued = true;
      ok = same_leader;
    }
    for (int j = 0; ok && j < n; ++j) {
      const int s = j % NS;
      const int s1 = (j + 1) % NS;
      const bool more = j + 1 < n;
      // The K/V tiles landed long ago in steady state: test them before P0 so
      // that P0's arrival starts P0.V and the next S0 at once.
      if ((more && !warp_wait(bar(C::B_KF + s1), ((j + 1) / NS) & 1, abort_flag)) ||
          !warp_wait(bar(C::B_VF + s), (j / NS) & 1, abort_flag) || !warp_wait(bar(C::B_PF), j & 1, abort_flag)) {
        ok = false;
        break;
      }
      ptx::tc_fence_after();
      // slot 0: P.V of tile j, then S of tile j + 1
      if (elect()) {
        mma_pv(0, j, 0);
        if (!more) ptx::mma_commit(bar(C::B_OF));
        if (more) {
          mma_s(0, j + 1, 0);
          ptx::mma_commit(bar(C::B_SF));
        }
      }
      __syncwarp();
      // slot 1: P.V of tile j, then S of tile j + 1
      if (!warp_wait(bar(C::B_PF + 1), j & 1, abort_flag)) {
        ok = false;
        break;
      }
      ptx::tc_fence_after();
      if (elect()) {
        mma_pv(1, j, 1);
        if (!more) ptx::mma_commit(bar(C::B_OF + 1));
        ptx::mma_commit(bar(C::B_VE + s));
        if (more) {
          mma_s(1, j + 1, 1);
          ptx::mma_commit(bar(C::B_SF + 1));
          ptx::mma_commit(bar(C::B_KE + s1));
        }
      }
      __syncwarp();
      ok = same_leader;
    }
  }
  const int lane = threadIdx.x & 31;
  if (!ok) {
    if (lane == 0) record_failure(abort_flag, L.status, kStatusTimeout);
    // Wait for every MMA the issuing lane started before TMEM is released.
    if (issued && lane == first_leader) {
      const volatile int never = 0;
      ptx::mma_commit(bar(C::B_DRAIN));
      ptx::mbar_wait(bar(C::B_DRAIN), 0, &never, kWaitTimeoutNs);
    }
  }
  __syncwarp();
}

template <int TILE, int D, int NS, int FSW, int EMB>
__device__ __forceinline__ void softmax_epilogue(const ProbeLaunch& L, const WorkItem& it, int slot, uint32_t sbase,
                                                 uint32_t tmem_base, volatile int* abort_flag) {
  using C = Cfg<TILE, D, NS>;
  auto bar = [&](int i) { return sbase + C::OFF_BAR + 8u * i; };
  const int left = heads_left(L, it.head);
  if (slot * C::HP >= left) return;            // the item has one slot only
  const int warp = (threadIdx.x >> 5) & 3;
  const int row = threadIdx.x & 127;           // TMEM lane
  const int hp = row / TILE;
  const int row_local = row % TILE;
  const bool head_ok = slot * C::HP + hp < left;
  const int head = it.head + slot * C::HP + hp;
  const bool row_ok = head_ok && row_local < it.q_len;
  const int qpos = it.q_start + row_local;
  const uint32_t lane_base = static_cast<uint32_t>(warp * 32) << 16;
  const uint32_t tmem = tmem_base + lane_base + slot * C::SLOT_COLS;
  const bool spill_rows = it.text_row0 >= 0 && row_ok && L.spill != nullptr;   // no spill: evidence recomputed
  // With one slot, S alternates between both slots' S columns (see the MMA issuer).
  const bool two = left > C::HP;

  float* spill_row = nullptr;
  int vis_start = 0;
  if (it.text_row0 >= 0) {
    const VideoInfo vi = L.videos[it.video];
    vis_start = vi.vis_start;
    // Spill [hq, text_pitch / 32, n_vis, 32]: a warp's 32 rows are one row
    // block, and for one key they are 128 contiguous bytes.
    if (row_ok) {
      const int r = it.text_row0 + row_local;
      spill_row = L.spill + vi.spill_off + static_cast<int64_t>(head) * vi.n_vis * vi.text_pitch +
                  static_cast<int64_t>(r >> 5) * vi.n_vis * 32 + (r & 31);
    }
  }

  // Cross-frame partials (visual rows, when enabled): per kept kv tile and
  // key frame f, m + log2(sum of the frame's P) in log2 units, so that the
  // frame's share of the row's softmax is exp2(value - LSE log2 e).
  // FSW = the key span of one partial, min(N_v, 64), in the instantiation that
  // keeps them (0: not kept), so that the span ends are compile-time positions
  // and the plain probe is unchanged.
  float* fs_row = nullptr;
  if constexpr (FSW > 0) {
    if (it.text_row0 < 0 && row_ok)
      fs_row = L.fspill + (static_cast<int64_t>(head) * L.fs_nnz + it.kv_begin) * (TILE / FSW) * TILE + row_local;
  }

  // Per-row block masks (EMB = their block size; 0: none): the row's bit per
  // block of its video (top-p retention and the own block), applied to the
  // keys of every kv tile before the max, the spill and P.
  [[maybe_unused]] const uint32_t* em_row = nullptr;
  [[maybe_unused]] int em_vis_start = 0, em_n_vis = 0;
  if constexpr (EMB > 0) {
    const VideoInfo evi = L.videos[it.video];
    em_vis_start = evi.vis_start;
    em_n_vis = evi.n_vis;
    if (row_ok) em_row = L.keep + static_cast<int64_t>(head) * L.keep_words * L.n_tok + qpos;
  }

  float m_used = -INFINITY;   // running max, log2 units
  float l_sum = 0.f;
  bool ok = true;
  const uint64_t scale2 = ptx::f2(L.scale_log2, L.scale_log2);

  // With per-row masks (EMB) the kv tiles are read two tiles ahead and the
  // row's mask word one tile ahead, so that no global load waits between an
  // S-ready wait and the softmax that follows it. Without them the tile is
  // read before its S-ready wait, which covers the load.
  auto load_kv = [&](int jj) { return jj < it.kv_count ? L.kv[it.kv_begin + jj] : KvTile{0, 0, 0, 0}; };
  [[maybe_unused]] auto mask_word = [&](const KvTile& t) -> uint32_t {
    uint32_t w = 0xffffffffu;   // bit q: the tile's q-th block is attended
    if constexpr (EMB > 0) {
      if (em_row) {
        const int blk0 = t.visual ? (t.start - em_vis_start) / EMB
                                  : em_n_vis / EMB + (t.start - em_vis_start - em_n_vis) / EMB;
        w = em_row[static_cast<int64_t>(blk0 >> 5) * L.n_tok] >> (blk0 & 31);
      }
    }
    return w;
  };
  [[maybe_unused]] KvTile kv_next{0, 0, 0, 0}, kv_after{0, 0, 0, 0};
  [[maybe_unused]] uint32_t em_next = 0xffffffffu;
  if constexpr (EMB > 0) {
    kv_next = load_kv(0);
    kv_after = load_kv(1);
    if (it.kv_count > 0) em_next = mask_word(kv_next);
  }

  for (int j = 0; j < it.kv_count; ++j) {
    KvTile kv;
    [[maybe_unused]] uint32_t em_bits = 0xffffffffu;
    if constexpr (EMB > 0) {
      kv = kv_next;
      em_bits = em_next;
      kv_next = kv_after;
      if (j + 1 < it.kv_count) em_next = mask_word(kv_next);   // kv_next was read a tile ago
      kv_after = load_kv(j + 2);
    } else {
      kv = L.kv[it.kv_begin + j];
    }
    const int b = two ? slot : (j & 1);
    const uint32_t par = two ? (j & 1) : ((j >> 1) & 1);
    const uint32_t tS = tmem_base + lane_base + b * C::SLOT_COLS + C::COL_S;
    const uint32_t bar_pf = bar(C::B_PF + b);
    if (!warp_wait(bar(C::B_SF + b), par, abort_flag)) { ok = false; break; }
    ptx::tc_fence_after();
    // Keys past the tile's end (ragged tile) or above the diagonal are masked.
    int limit = TILE;
    if (kv.diag || kv.len < TILE) {
      limit = kv.len;
      if (kv.diag) limit = min(limit, qpos - kv.start + 1);
    }
    const bool spill = spill_rows && kv.visual;
    float* spill_dst = spill ? spill_row + static_cast<int64_t>(kv.start - vis_start) * 32 : nullptr;
    auto apply_em = [&](float* sv, int h) {
      if constexpr (EMB > 0) {
        if ((em_bits & ((1u << (TILE / EMB)) - 1u)) != (1u << (TILE / EMB)) - 1u) {
#pragma unroll
          for (int c = 0; c < 64; ++c)
            if (!((em_bits >> ((h * 64 + c) / EMB)) & 1u)) sv[c] = -INFINITY;
        }
      }
    };

    // Pass 1: row max (and the text rows' logit spill), 64 columns at a time.
    float m4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
    for (int h = 0; h < TILE / 64; ++h) {
      float s[64];
      {
        uint32_t r0[32], r1[32];
        ptx::tmem_ld32(tS + h * 64, r0);
        ptx::tmem_ld32(tS + h * 64 + 32, r1);
        ptx::tmem_wait_ld();
#pragma unroll
        for (int e = 0; e < 32; ++e) {
          s[e] = __uint_as_float(r0[e]);
          s[32 + e] = __uint_as_float(r1[e]);
        }
      }
      apply_em(s, h);
      if (spill) {
        float* dst = spill_dst + h * 64 * 32;
#pragma unroll
        for (int c = 0; c < 64; ++c)
          if (h * 64 + c < kv.len) __stcs(dst + c * 32, s[c] * L.scale);
      }
      if (limit < TILE) {
#pragma unroll
        for (int c = 0; c < 64; ++c) s[c] = h * 64 + c < limit ? s[c] : -INFINITY;
      }
#pragma unroll
      for (int c = 0; c < 64; c += 8) {
        m4[0] = ptx::max3(m4[0], s[c], s[c + 1]);
        m4[1] = ptx::max3(m4[1], s[c + 2], s[c + 3]);
        m4[2] = ptx::max3(m4[2], s[c + 4], s[c + 5]);
        m4[3] = ptx::max3(m4[3], s[c + 6], s[c + 7]);
      }
    }
    const float mx = fmaxf(fmaxf(m4[0], m4[1]), fmaxf(m4[2], m4[3]));
    const float m_tile = mx * L.scale_log2;
    const bool need = m_tile > m_used + kRescaleThreshold;
    float alpha = 1.f;
    if (need) {
      alpha = ptx::ex2(m_used - m_tile);
      l_sum *= alpha;
      m_used = m_tile;
    }
    const float m_safe = (m_used == -INFINITY) ? 0.f : m_used;

    // Lazy rescale of the O accumulator (only rows whose max moved by > 2^8).
    // With two slots S_j was issued after P_{j-1}.V, so that MMA has
    // completed; with one slot it is waited for (its V-empty barrier).
    if (j > 0 && __any_sync(0xffffffffu, need)) {
      if (!two && !warp_wait(bar(C::B_VE + (j - 1) % NS), ((j - 1) / NS) & 1, abort_flag)) {
        ok = false;
        break;
      }
      ptx::tc_fence_after();
#pragma unroll
      for (int c = 0; c < D / 32; ++c) {
        uint32_t r[32];
        ptx::tmem_ld32(tmem + C::COL_O + c * 32, r);
        ptx::tmem_wait_ld();
#pragma unroll
        for (int e = 0; e < 32; ++e) r[e] = __float_as_uint(__uint_as_float(r[e]) * alpha);
        ptx::tmem_st32(tmem + C::COL_O + c * 32, r);
      }
    }

    // Pass 2: P = 2^(s * scale * log2 e - m) in packed pairs, written as bf16
    // over the first half of S (columns of a 64-wide chunk are read before
    // the chunk's P is stored, and P of chunk h lands below chunk h + 1).
    const uint64_t negm2 = ptx::f2(-m_safe, -m_safe);
    uint64_t l2[4] = {0, 0, 0, 0};
    [[maybe_unused]] float l_tile = 0.f;
    [[maybe_unused]] float* fs_tile = nullptr;
    if constexpr (FSW > 0) {
      if (fs_row) fs_tile = fs_row + static_cast<int64_t>(j) * (TILE / FSW) * TILE;
    }
#pragma unroll
    for (int h = 0; h < TILE / 64; ++h) {
      float s[64];
      {
        uint32_t r0[32], r1[32];
        ptx::tmem_ld32(tS + h * 64, r0);
        ptx::tmem_ld32(tS + h * 64 + 32, r1);
        ptx::tmem_wait_ld();
#pragma unroll
        for (int e = 0; e < 32; ++e) {
          s[e] = __uint_as_float(r0[e]);
          s[32 + e] = __uint_as_float(r1[e]);
        }
      }
      apply_em(s, h);
      if (limit < TILE) {
#pragma unroll
        for (int c = 0; c < 64; ++c) s[c] = h * 64 + c < limit ? s[c] : -INFINITY;
      }
      uint32_t pk[32];
#pragma unroll
      for (int e = 0; e < 32; ++e) {
        float x0, x1;
        ptx::unf2(ptx::fma2(ptx::f2(s[2 * e], s[2 * e + 1]), scale2, negm2), x0, x1);
        const float p0 = ptx::ex2(x0);
        const float p1 = ptx::ex2(x1);
        l2[e & 3] = ptx::add2(l2[e & 3], ptx::f2(p0, p1));
        pk[e] = ptx::pack_bf16x2(p0, p1);
        if constexpr (FSW > 0) {
          if ((h * 64 + 2 * e + 2) % FSW == 0) {      // the last keys of span (h * 64 + 2e + 2) / FSW - 1
            float a0, a1, b0, b1, c0, c1, d0, d1;
            ptx::unf2(l2[0], a0, a1);
            ptx::unf2(l2[1], b0, b1);
            ptx::unf2(l2[2], c0, c1);
            ptx::unf2(l2[3], d0, d1);
            const float fsum = ((a0 + a1) + (b0 + b1)) + ((c0 + c1) + (d0 + d1));
            l_tile += fsum;
            l2[0] = l2[1] = l2[2] = l2[3] = 0;
            if (fs_tile)
              __stcs(fs_tile + ((h * 64 + 2 * e + 2) / FSW - 1) * TILE, fsum > 0.f ? m_safe + __log2f(fsum) : -INFINITY);
          }
        }
      }
      ptx::tmem_st32(tS + h * 32, pk);
    }
    if constexpr (FSW > 0) {
      l_sum += l_tile;
    } else {
      float a0, a1, b0, b1, c0, c1, d0, d1;
      ptx::unf2(l2[0], a0, a1);
      ptx::unf2(l2[1], b0, b1);
      ptx::unf2(l2[2], c0, c1);
      ptx::unf2(l2[3], d0, d1);
      l_sum += ((a0 + a1) + (b0 + b1)) + ((c0 + c1) + (d0 + d1));
    }
    ptx::tmem_wait_st();
    ptx::tc_fence_before();
    ptx::mbar_arrive(bar_pf);
  }

  ok = ok && warp_wait(bar(C::B_OF + slot), 0, abort_flag);
  if (!ok) record_failure(abort_flag, L.status, kStatusTimeout);
  ptx::tc_fence_after();

  const float inv_l = l_sum > 0.f ? 1.f / l_sum : 0.f;
  if (it.part < 0 && it.q_len == TILE) {
    // Every warp of the slot reaches the named barrier below, whether or not
    // one of them gave up on a wait, so that the barrier always completes;
    // the barrier then tells all 128 threads whether to store.
    // Full tile: the slot's O goes through its Q region of shared memory (no
    // MMA reads Q any more) in Q's swizzled layout, then out by TMA stores of
    // one 64-column block of one head each: whole 128-byte rows instead of 16
    // bytes per row and store.
    const uint32_t stage = sbase + C::OFF_Q + slot * C::Q_BYTES + hp * TILE * 128 + row_local * 128;
    if (ok) {
#pragma unroll
      for (int c = 0; c < D / 32; ++c) {
        uint32_t r[32];
        ptx::tmem_ld32(tmem + C::COL_O + c * 32, r);
        ptx::tmem_wait_ld();
#pragma unroll
        for (int q4 = 0; q4 < 4; ++q4) {
          uint4 w;
          w.x = ptx::pack_bf16x2(__uint_as_float(r[8 * q4 + 0]) * inv_l, __uint_as_float(r[8 * q4 + 1]) * inv_l);
          w.y = ptx::pack_bf16x2(__uint_as_float(r[8 * q4 + 2]) * inv_l, __uint_as_float(r[8 * q4 + 3]) * inv_l);
          w.z = ptx::pack_bf16x2(__uint_as_float(r[8 * q4 + 4]) * inv_l, __uint_as_float(r[8 * q4 + 5]) * inv_l);
          w.w = ptx::pack_bf16x2(__uint_as_float(r[8 * q4 + 6]) * inv_l, __uint_as_float(r[8 * q4 + 7]) * inv_l);
          // 16-byte chunk k of the row's 128-byte block kb sits at chunk k ^ (row & 7).
          const int kb = c / 2, k = (c % 2) * 4 + q4;
          const uint32_t addr = stage + kb * C::Q_BLOCK + ((k ^ (row_local & 7)) << 4);
          asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(w.x), "r"(w.y), "r"(w.z), "r"(w.w)
                       : "memory");
        }
      }
    }
    if (ok && row_ok) L.lse[static_cast<int64_t>(head) * L.n_tok + qpos] = (m_used + __log2f(l_sum)) * kLn2;
    ptx::fence_proxy_async_smem();
    const bool all_ok = ptx::bar_and(1 + slot, kRows, ok);
    if (all_ok && (threadIdx.x & 127) == 0) {
#pragma unroll
      for (int h = 0; h < C::HP; ++h) {
        if (slot * C::HP + h >= left) break;   // heads past the group's end are not stored
#pragma unroll
        for (int kb = 0; kb < C::KB; ++kb)
          ptx::tma_store_3d(&L.tm_o, sbase + C::OFF_Q + slot * C::Q_BYTES + kb * C::Q_BLOCK + h * TILE * 128, kb * 64,
                            it.head + slot * C::HP + h, it.q_start);
      }
      ptx::bulk_commit();
      ptx::bulk_wait_read();   // the shared memory source must outlive the copy
    }
  } else if (!ok) {
    return;
  } else if (it.part < 0) {
    uint4* dst = reinterpret_cast<uint4*>(static_cast<uint16_t*>(L.o) +
                                          (static_cast<int64_t>(qpos) * L.hq + head) * D);
#pragma unroll
    for (int c = 0; c < D / 32; ++c) {
      uint32_t r[32];
      ptx::tmem_ld32(tmem + C::COL_O + c * 32, r);
      ptx::tmem_wait_ld();
      if (row_ok) {
#pragma unroll
        for (int q4 = 0; q4 < 4; ++q4) {
          uint4 w;
          w.x = ptx::pack_bf16x2(__uint_as_float(r[8 * q4 + 0]) * inv_l, __uint_as_float(r[8 * q4 + 1]) * inv_l);
          w.y = ptx::pack_bf16x2(__uint_as_float(r[8 * q4 + 2]) * inv_l, __uint_as_float(r[8 * q4 + 3]) * inv_l);
          w.z = ptx::pack_bf16x2(__uint_as_float(r[8 * q4 + 4]) * inv_l, __uint_as_float(r[8 * q4 + 5]) * inv_l);
          w.w = ptx::pack_bf16x2(__uint_as_float(r[8 * q4 + 6]) * inv_l, __uint_as_float(r[8 * q4 + 7]) * inv_l);
          dst[c * 4 + q4] = w;
        }
      }
    }
    if (row_ok) L.lse[static_cast<int64_t>(head) * L.n_tok + qpos] = (m_used + __log2f(l_sum)) * kLn2;
  } else {
    const int64_t part = it.part + slot;
    float4* dst = reinterpret_cast<float4*>(L.part_o + (part * kRows + row) * D);
#pragma unroll
    for (int c = 0; c < D / 32; ++c) {
      uint32_t r[32];
      ptx::tmem_ld32(tmem + C::COL_O + c * 32, r);
      ptx::tmem_wait_ld();
#pragma unroll
      for (int q4 = 0; q4 < 8; ++q4)
        dst[c * 8 + q4] = make_float4(__uint_as_float(r[4 * q4]), __uint_as_float(r[4 * q4 + 1]),
                                      __uint_as_float(r[4 * q4 + 2]), __uint_as_float(r[4 * q4 + 3]));
    }
    L.part_ml[part * kRows + row] = make_float2(m_used, l_sum);
  }
}

template <int TILE, int D, int NS, int FSW, int EMB>
__global__ void __launch_bounds__(kThreads, 1) probe_attn_kernel(const __grid_constant__ ProbeLaunch L) {
  using C = Cfg<TILE, D, NS>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t sbase = ptx::smem_addr(smem);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + C::OFF_MISC);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::OFF_MISC + 4);
  const int warp = threadIdx.x >> 5;
  const WorkItem it = L.items[blockIdx.x];

  if (threadIdx.x == kWarpProducer * 32) setup_and_first_loads<TILE, D, NS>(L, it, sbase, abort_flag);
  if (warp == 0) {
    ptx::tmem_alloc<C::TMEM_COLS>(ptx::smem_addr(tmem_slot));
    ptx::tmem_relinquish();
  }
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == kWarpProducer) {
    producer<TILE, D, NS, false>(L, it, sbase, abort_flag);
  } else if (warp == kWarpVLoader) {
    producer<TILE, D, NS, true>(L, it, sbase, abort_flag);
  } else if (warp == kWarpMma) {
    mma_issuer<TILE, D, NS>(L, it, sbase, tmem, abort_flag);
  } else {
    softmax_epilogue<TILE, D, NS, FSW, EMB>(L, it, warp / 4, sbase, tmem, abort_flag);
  }
  ptx::tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc<C::TMEM_COLS>(tmem);
  }
}

template <int TILE, int D, int FSW, int EMB = 0>
cudaError_t launch_cfg(const ProbeLaunch& L, cudaStream_t stream) {
  constexpr int NS = 2;
  using C = Cfg<TILE, D, NS>;
  auto kern = probe_attn_kernel<TILE, D, NS, FSW, EMB>;
  static PerDeviceAttr smem_once;
  cudaError_t e = raise_smem_limit(smem_once, reinterpret_cast<const void*>(kern), C::SMEM_BYTES);
  if (e != cudaSuccess) return e;
  kern<<<L.n_items, kThreads, C::SMEM_BYTES, stream>>>(L);
  return cudaGetLastError();
}

// The plain probe (fsw = 0) or the one that keeps cross-frame partials over
// key spans of fsw tokens (16, 32 or 64).
template <int TILE, int D>
cudaError_t launch_fsw(const ProbeLaunch& L, int fsw, cudaStream_t stream) {
  if (L.keep) {                                  // per-row block masks (not with cross-frame partials)
    if (fsw != 0) return cudaErrorInvalidValue;
    switch (L.keep_block) {
      case 16: return launch_cfg<TILE, D, 0, 16>(L, stream);
      case 32: return launch_cfg<TILE, D, 0, 32>(L, stream);
      case 64: return launch_cfg<TILE, D, 0, 64>(L, stream);
      case 128:
        if constexpr (TILE == 128) return launch_cfg<TILE, D, 0, 128>(L, stream);
        return cudaErrorInvalidValue;
      default: return cudaErrorInvalidValue;
    }
  }
  switch (fsw) {
    case 0: return launch_cfg<TILE, D, 0>(L, stream);
    case 16: return launch_cfg<TILE, D, 16>(L, stream);
    case 32: return launch_cfg<TILE, D, 32>(L, stream);
    case 64: return launch_cfg<TILE, D, 64>(L, stream);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

cudaError_t launch_probe_attn(const ProbeLaunch& L, cudaStream_t stream) {
  if (L.n_items == 0) return cudaSuccess;
  const int fsw = L.fspill ? L.fs_span : 0;
  if (L.tile == 128 && L.head_dim == 128) return launch_fsw<128, 128>(L, fsw, stream);
  if (L.tile == 128 && L.head_dim == 64) return launch_fsw<128, 64>(L, fsw, stream);
  if (L.tile == 64 && L.head_dim == 128) return launch_fsw<64, 128>(L, fsw, stream);
  if (L.tile == 64 && L.head_dim == 64) return launch_fsw<64, 64>(L, fsw, stream);
  return cudaErrorInvalidValue;
}

}  // namespace evisel
