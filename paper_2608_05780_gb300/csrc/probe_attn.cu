// Block-sparse, causal, grouped-query, varlen prefill attention for sm_103a
// (the paper's sparse probe, Sec. 3.2 Eq. 1, with exact token logits on every
// kept tile: Appendix Eq. 8 in token form and the row normalisation of Eq. 11).
//
// One CTA computes one work item: a 128-row query tile (one head for 128-token
// tiles, two heads of one KV group for 64-token tiles) against a list of kept
// kv tiles. Warp roles:
//   warps 0-3  softmax + epilogue, one thread per query row (= TMEM lane)
//   warp 4     TMA producer: Q once, then K_j / V_j into an NS-deep smem ring
//   warp 5     MMA issuer (one thread): S_j = Q K_j^T into a double-buffered
//              TMEM S, O += P_j V_j with P_j read from TMEM (bf16)
// TMEM columns: S0 | S1 | P0 | P1 | O.
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

constexpr int kThreads = 192;
constexpr int kRows = 128;
constexpr float kRescaleThreshold = 8.0f;   // log2 units
constexpr float kLn2 = 0.69314718055994531f;

template <int TILE, int D, int NS>
struct Cfg {
  static constexpr int HP = kRows / TILE;        // query heads per CTA
  static constexpr int KB = D / 64;              // 128-byte swizzle column blocks along d
  static constexpr int Q_BYTES = kRows * D * 2;
  static constexpr int Q_BLOCK = kRows * 128;    // one column block of Q
  static constexpr int KV_BLOCK = TILE * 128;    // one column block of a K/V tile
  static constexpr int KV_BYTES = TILE * D * 2;
  static constexpr int OFF_Q = 0;
  static constexpr int OFF_K = OFF_Q + Q_BYTES;
  static constexpr int OFF_V = OFF_K + NS * KV_BYTES;
  static constexpr int OFF_BAR = OFF_V + NS * KV_BYTES;
  // barrier indices
  static constexpr int B_Q = 0;
  static constexpr int B_KF = 1;
  static constexpr int B_KE = B_KF + NS;
  static constexpr int B_VF = B_KE + NS;
  static constexpr int B_VE = B_VF + NS;
  static constexpr int B_SF = B_VE + NS;   // 2
  static constexpr int B_PF = B_SF + 2;    // 2
  static constexpr int B_PV = B_PF + 2;    // 2
  static constexpr int B_OF = B_PV + 2;
  static constexpr int B_DRAIN = B_OF + 1;
  static constexpr int N_BARS = B_DRAIN + 1;
  static constexpr int OFF_MISC = OFF_BAR + N_BARS * 8;
  static constexpr int SMEM_USED = OFF_MISC + 16;
  // TMEM columns (32-bit)
  static constexpr int COL_S0 = 0;
  static constexpr int COL_P0 = 2 * TILE;
  static constexpr int COL_O = 3 * TILE;
  static constexpr int TMEM_COLS = (3 * TILE + D <= 256) ? 256 : 512;
  // Dynamic smem requested: enough to keep TMEM demand per SM within 512 columns.
  static constexpr int SMEM_MIN = TMEM_COLS == 512 ? 117 * 1024 : 78 * 1024;
  static constexpr int SMEM_BYTES = (SMEM_USED + 1024 > SMEM_MIN) ? SMEM_USED + 1024 : SMEM_MIN;
  static_assert(SMEM_USED + 1024 <= 232448, "shared memory budget");
  static_assert((OFF_K % 1024) == 0 && (OFF_V % 1024) == 0 && (KV_BYTES % 1024) == 0, "1 KB aligned tiles");
};

__device__ __forceinline__ void record_failure(volatile int* abort_flag, int* status, int code) {
  *abort_flag = 1;
  atomicExch(status, code);
}

// Bounded wait whose outcome is uniform across the warp, so that the warp stays
// converged for the warp-collective tcgen05.ld / tcgen05.st that follow.
__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag) {
  const bool ok = ptx::mbar_wait(bar, parity, abort_flag, kWaitTimeoutNs);
  return __all_sync(0xffffffffu, ok);
}

template <int TILE, int D, int NS>
__device__ __forceinline__ void producer(const ProbeLaunch& L, const WorkItem& it, uint32_t sbase,
                                         volatile int* abort_flag) {
  using C = Cfg<TILE, D, NS>;
  auto bar = [&](int i) { return sbase + C::OFF_BAR + 8u * i; };
  const int gq = L.hq / L.hkv;
  const int g = it.head / gq;
  const bool second_ok = (C::HP == 1) || ((it.head + 1) < L.hq && (it.head + 1) / gq == g);
  const uint64_t pol_q = ptx::l2_policy_evict_first();
  const uint64_t pol_kv = ptx::l2_policy_evict_last();
  ptx::tma_prefetch_desc(&L.tm_q);
  ptx::tma_prefetch_desc(&L.tm_k);
  ptx::tma_prefetch_desc(&L.tm_v);

  ptx::mbar_arrive_expect_tx(bar(C::B_Q), C::Q_BYTES);
#pragma unroll
  for (int hp = 0; hp < C::HP; ++hp) {
    const int h = (hp == 0 || second_ok) ? it.head + hp : it.head;
#pragma unroll
    for (int kb = 0; kb < C::KB; ++kb)
      ptx::tma_load_3d(sbase + C::OFF_Q + kb * C::Q_BLOCK + hp * TILE * 128, &L.tm_q, bar(C::B_Q), kb * 64, h,
                       it.q_start, pol_q);
  }

  int k_issued = 0, v_issued = 0;
  for (int j = 0; j < it.kv_count; ++j) {
    const int s = j % NS;
    const int u = j / NS;
    const KvTile kv = L.kv[it.kv_begin + j];
    if (u > 0 && !ptx::mbar_wait(bar(C::B_KE + s), (u - 1) & 1, abort_flag, kWaitTimeoutNs)) {
      record_failure(abort_flag, L.status, kStatusTimeout);
      break;
    }
    ptx::mbar_arrive_expect_tx(bar(C::B_KF + s), C::KV_BYTES);
#pragma unroll
    for (int kb = 0; kb < C::KB; ++kb)
      ptx::tma_load_3d(sbase + C::OFF_K + s * C::KV_BYTES + kb * C::KV_BLOCK, &L.tm_k, bar(C::B_KF + s), kb * 64,
                       g, kv.start, pol_kv);
    k_issued = j + 1;
    if (u > 0 && !ptx::mbar_wait(bar(C::B_VE + s), (u - 1) & 1, abort_flag, kWaitTimeoutNs)) {
      record_failure(abort_flag, L.status, kStatusTimeout);
      break;
    }
    ptx::mbar_arrive_expect_tx(bar(C::B_VF + s), C::KV_BYTES);
#pragma unroll
    for (int kb = 0; kb < C::KB; ++kb)
      ptx::tma_load_3d(sbase + C::OFF_V + s * C::KV_BYTES + kb * C::KV_BLOCK, &L.tm_v, bar(C::B_VF + s), kb * 64,
                       g, kv.start, pol_kv);
    v_issued = j + 1;
  }
  {
    // Drain: every load issued here completes on its own; wait for the last
    // phase issued into each stage (and for Q) so that no copy is in flight
    // when the CTA exits, whether or not another warp gave up.
    const volatile int never = 0;
    ptx::mbar_wait(bar(C::B_Q), 0, &never, kWaitTimeoutNs);
    for (int s = 0; s < NS; ++s) {
      if (s < k_issued) {
        const int last = ((k_issued - 1 - s) / NS) * NS + s;
        ptx::mbar_wait(bar(C::B_KF + s), (last / NS) & 1, &never, kWaitTimeoutNs);
      }
      if (s < v_issued) {
        const int last = ((v_issued - 1 - s) / NS) * NS + s;
        ptx::mbar_wait(bar(C::B_VF + s), (last / NS) & 1, &never, kWaitTimeoutNs);
      }
    }
  }
}

template <int TILE, int D, int NS>
__device__ __forceinline__ void mma_issuer(const ProbeLaunch& L, const WorkItem& it, uint32_t sbase, uint32_t tmem,
                                           volatile int* abort_flag) {
  using C = Cfg<TILE, D, NS>;
  auto bar = [&](int i) { return sbase + C::OFF_BAR + 8u * i; };
  constexpr uint32_t kIdescS = ptx::idesc_bf16_f32(kRows, TILE, false, false);
  constexpr uint32_t kIdescO = ptx::idesc_bf16_f32(kRows, D, false, true);
  const int n = it.kv_count;
  bool ok = ptx::mbar_wait(bar(C::B_Q), 0, abort_flag, kWaitTimeoutNs);

  auto issue_s = [&](int j) -> bool {
    const int s = j % NS;
    const int b = j & 1;
    if (!ptx::mbar_wait(bar(C::B_KF + s), (j / NS) & 1, abort_flag, kWaitTimeoutNs)) return false;
    ptx::tc_fence_after();
    const uint32_t kbase = sbase + C::OFF_K + s * C::KV_BYTES;
#pragma unroll
    for (int kk = 0; kk < D / 16; ++kk) {
      const uint64_t a = ptx::sdesc_sw128(sbase + C::OFF_Q + (kk / 4) * C::Q_BLOCK + (kk % 4) * 32, 16, 1024);
      const uint64_t bd = ptx::sdesc_sw128(kbase + (kk / 4) * C::KV_BLOCK + (kk % 4) * 32, 16, 1024);
      ptx::mma_ss(tmem + C::COL_S0 + b * TILE, a, bd, kIdescS, kk > 0 ? 1u : 0u);
    }
    ptx::mma_commit(bar(C::B_SF + b));
    ptx::mma_commit(bar(C::B_KE + s));
    return true;
  };

  if (ok) {
    ptx::tc_fence_after();
    ok = issue_s(0);
  }
  for (int j = 0; ok && j < n; ++j) {
    if (j + 1 < n && !(ok = issue_s(j + 1))) break;
    const int s = j % NS;
    const int b = j & 1;
    if (!ptx::mbar_wait(bar(C::B_PF + b), (j >> 1) & 1, abort_flag, kWaitTimeoutNs) ||
        !ptx::mbar_wait(bar(C::B_VF + s), (j / NS) & 1, abort_flag, kWaitTimeoutNs)) {
      ok = false;
      break;
    }
    ptx::tc_fence_after();
    const uint32_t vbase = sbase + C::OFF_V + s * C::KV_BYTES;
#pragma unroll
    for (int kk = 0; kk < TILE / 16; ++kk) {
      const uint64_t bd = ptx::sdesc_sw128(vbase + kk * 16 * 128, C::KV_BLOCK, 1024);
      ptx::mma_ts(tmem + C::COL_O, tmem + C::COL_P0 + b * (TILE / 2) + kk * 8, bd, kIdescO,
                  (j > 0 || kk > 0) ? 1u : 0u);
    }
    ptx::mma_commit(bar(C::B_PV + b));
    ptx::mma_commit(bar(C::B_VE + s));
  }
  if (ok) {
    ptx::mma_commit(bar(C::B_OF));
  } else {
    record_failure(abort_flag, L.status, kStatusTimeout);
    // Wait for every MMA this thread issued before TMEM is released.
    const volatile int never = 0;
    ptx::mma_commit(bar(C::B_DRAIN));
    ptx::mbar_wait(bar(C::B_DRAIN), 0, &never, kWaitTimeoutNs);
  }
}

template <int TILE, int D, int NS>
__device__ __forceinline__ void softmax_epilogue(const ProbeLaunch& L, const WorkItem& it, uint32_t sbase,
                                                 uint32_t tmem, volatile int* abort_flag) {
  using C = Cfg<TILE, D, NS>;
  auto bar = [&](int i) { return sbase + C::OFF_BAR + 8u * i; };
  const int warp = threadIdx.x >> 5;
  const int row = threadIdx.x;                 // TMEM lane
  const int hp = row / TILE;
  const int row_local = row % TILE;
  const int gq = L.hq / L.hkv;
  const bool head_ok = (hp == 0) || ((it.head + 1) < L.hq && (it.head + 1) / gq == it.head / gq);
  const int head = it.head + hp;
  const bool row_ok = head_ok && row_local < it.q_len;
  const int qpos = it.q_start + row_local;
  const uint32_t lane_base = static_cast<uint32_t>(warp * 32) << 16;
  const bool spill_rows = it.text_row0 >= 0 && row_ok;

  float* spill_row = nullptr;
  int vis_start = 0;
  if (it.text_row0 >= 0) {
    const VideoInfo vi = L.videos[it.video];
    vis_start = vi.vis_start;
    if (row_ok)
      spill_row = L.spill + vi.spill_off +
                  (static_cast<int64_t>(head) * vi.n_text + it.text_row0 + row_local) * vi.vis_pitch;
  }

  float m_used = -INFINITY;   // running max, log2 units
  float l_sum = 0.f;
  bool ok = true;

  for (int j = 0; j < it.kv_count; ++j) {
    const int b = j & 1;
    const KvTile kv = L.kv[it.kv_begin + j];
    if (!warp_wait(bar(C::B_SF + b), (j >> 1) & 1, abort_flag)) { ok = false; break; }
    ptx::tc_fence_after();
    float s[TILE];
#pragma unroll
    for (int c = 0; c < TILE / 32; ++c) {
      uint32_t r[32];
      ptx::tmem_ld32(tmem + lane_base + C::COL_S0 + b * TILE + c * 32, r);
#pragma unroll
      for (int e = 0; e < 32; ++e) s[c * 32 + e] = __uint_as_float(r[e]);
    }
    ptx::tmem_wait_ld();

    // Text rows keep their natural-log logits onto visual keys for the evidence pass.
    if (spill_rows && kv.visual) {
      float* dst = spill_row + (kv.start - vis_start);
      const int n4 = (kv.len + 3) >> 2;
#pragma unroll
      for (int c4 = 0; c4 < TILE / 4; ++c4) {
        if (c4 < n4) {
          float4 w = make_float4(s[4 * c4] * L.scale, s[4 * c4 + 1] * L.scale, s[4 * c4 + 2] * L.scale,
                                 s[4 * c4 + 3] * L.scale);
          __stcs(reinterpret_cast<float4*>(dst) + c4, w);
        }
      }
    }

    if (kv.diag || kv.len < TILE) {
      int limit = kv.len;
      if (kv.diag) limit = min(limit, qpos - kv.start + 1);
#pragma unroll
      for (int c = 0; c < TILE; ++c) s[c] = c < limit ? s[c] : -INFINITY;
    }
    float m4[4] = {s[0], s[1], s[2], s[3]};
#pragma unroll
    for (int c = 4; c < TILE - 4; c += 8) {
      m4[0] = ptx::max3(m4[0], s[c], s[c + 1]);
      m4[1] = ptx::max3(m4[1], s[c + 2], s[c + 3]);
      m4[2] = ptx::max3(m4[2], s[c + 4], s[c + 5]);
      m4[3] = ptx::max3(m4[3], s[c + 6], s[c + 7]);
    }
    m4[0] = ptx::max3(m4[0], s[TILE - 4], s[TILE - 3]);
    m4[1] = ptx::max3(m4[1], s[TILE - 2], s[TILE - 1]);
    const float mx = ptx::max3(m4[0], m4[1], fmaxf(m4[2], m4[3]));
    const float m_tile = mx * L.scale_log2;
    const bool need = m_tile > m_used + kRescaleThreshold;
    float alpha = 1.f;
    if (need) {
      alpha = ptx::ex2(m_used - m_tile);
      l_sum *= alpha;
      m_used = m_tile;
    }
    const float m_safe = (m_used == -INFINITY) ? 0.f : m_used;

    // P buffer b was last read by PV_{j-2}.
    if (j >= 2 && !warp_wait(bar(C::B_PV + b), ((j - 2) >> 1) & 1, abort_flag)) {
      ok = false;
      break;
    }
    const uint64_t scale2 = ptx::f2(L.scale_log2, L.scale_log2);
    const uint64_t negm2 = ptx::f2(-m_safe, -m_safe);
    uint64_t l2[4] = {0, 0, 0, 0};
#pragma unroll
    for (int c = 0; c < TILE / 64; ++c) {
      uint32_t pk[32];
#pragma unroll
      for (int e = 0; e < 32; ++e) {
        float x0, x1;
        ptx::unf2(ptx::fma2(ptx::f2(s[c * 64 + 2 * e], s[c * 64 + 2 * e + 1]), scale2, negm2), x0, x1);
        const float p0 = ptx::ex2(x0);
        const float p1 = ptx::ex2(x1);
        l2[e & 3] = ptx::add2(l2[e & 3], ptx::f2(p0, p1));
        pk[e] = ptx::pack_bf16x2(p0, p1);
      }
      ptx::tmem_st32(tmem + lane_base + C::COL_P0 + b * (TILE / 2) + c * 32, pk);
    }
    {
      float a0, a1, b0, b1, c0, c1, d0, d1;
      ptx::unf2(l2[0], a0, a1);
      ptx::unf2(l2[1], b0, b1);
      ptx::unf2(l2[2], c0, c1);
      ptx::unf2(l2[3], d0, d1);
      l_sum += ((a0 + a1) + (b0 + b1)) + ((c0 + c1) + (d0 + d1));
    }

    // Lazy rescale of the O accumulator (only rows whose max moved by > 2^8).
    if (j > 0 && __any_sync(0xffffffffu, need)) {
      if (!warp_wait(bar(C::B_PV + ((j - 1) & 1)), ((j - 1) >> 1) & 1, abort_flag)) {
        ok = false;
        break;
      }
      ptx::tc_fence_after();
#pragma unroll
      for (int c = 0; c < D / 32; ++c) {
        uint32_t r[32];
        ptx::tmem_ld32(tmem + lane_base + C::COL_O + c * 32, r);
        ptx::tmem_wait_ld();
#pragma unroll
        for (int e = 0; e < 32; ++e) r[e] = __float_as_uint(__uint_as_float(r[e]) * alpha);
        ptx::tmem_st32(tmem + lane_base + C::COL_O + c * 32, r);
      }
    }
    ptx::tmem_wait_st();
    ptx::tc_fence_before();
    ptx::mbar_arrive(bar(C::B_PF + b));
  }

  if (!ok) {
    record_failure(abort_flag, L.status, kStatusTimeout);
    return;
  }
  if (!warp_wait(bar(C::B_OF), 0, abort_flag)) {
    record_failure(abort_flag, L.status, kStatusTimeout);
    return;
  }
  ptx::tc_fence_after();

  const float inv_l = l_sum > 0.f ? 1.f / l_sum : 0.f;
  if (it.part < 0) {
    uint4* dst = reinterpret_cast<uint4*>(static_cast<uint16_t*>(L.o) +
                                          (static_cast<int64_t>(qpos) * L.hq + head) * D);
#pragma unroll
    for (int c = 0; c < D / 32; ++c) {
      uint32_t r[32];
      ptx::tmem_ld32(tmem + lane_base + C::COL_O + c * 32, r);
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
    float4* dst = reinterpret_cast<float4*>(L.part_o + (static_cast<int64_t>(it.part) * kRows + row) * D);
#pragma unroll
    for (int c = 0; c < D / 32; ++c) {
      uint32_t r[32];
      ptx::tmem_ld32(tmem + lane_base + C::COL_O + c * 32, r);
      ptx::tmem_wait_ld();
#pragma unroll
      for (int q4 = 0; q4 < 8; ++q4)
        dst[c * 8 + q4] = make_float4(__uint_as_float(r[4 * q4]), __uint_as_float(r[4 * q4 + 1]),
                                      __uint_as_float(r[4 * q4 + 2]), __uint_as_float(r[4 * q4 + 3]));
    }
    L.part_ml[static_cast<int64_t>(it.part) * kRows + row] = make_float2(m_used, l_sum);
  }
}

template <int TILE, int D, int NS>
__global__ void __launch_bounds__(kThreads, 1) probe_attn_kernel(const __grid_constant__ ProbeLaunch L) {
  using C = Cfg<TILE, D, NS>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t sbase = ptx::smem_addr(smem);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + C::OFF_MISC);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::OFF_MISC + 4);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const WorkItem it = L.items[blockIdx.x];

  if (threadIdx.x == 0) {
    for (int i = 0; i < C::N_BARS; ++i) {
      const bool softmax_arrive = (i == C::B_PF || i == C::B_PF + 1);
      ptx::mbar_init(sbase + C::OFF_BAR + 8u * i, softmax_arrive ? kRows : 1u);
    }
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

  if (warp == 4) {
    if (lane == 0) producer<TILE, D, NS>(L, it, sbase, abort_flag);
  } else if (warp == 5) {
    if (lane == 0) mma_issuer<TILE, D, NS>(L, it, sbase, tmem, abort_flag);
  } else {
    softmax_epilogue<TILE, D, NS>(L, it, sbase, tmem, abort_flag);
  }
  ptx::tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc<C::TMEM_COLS>(tmem);
  }
}

template <int TILE, int D>
cudaError_t launch_cfg(const ProbeLaunch& L, cudaStream_t stream) {
  constexpr int NS = 2;
  using C = Cfg<TILE, D, NS>;
  auto kern = probe_attn_kernel<TILE, D, NS>;
  static bool configured = false;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM_BYTES);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  kern<<<L.n_items, kThreads, C::SMEM_BYTES, stream>>>(L);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_probe_attn(const ProbeLaunch& L, cudaStream_t stream) {
  if (L.n_items == 0) return cudaSuccess;
  if (L.tile == 128 && L.head_dim == 128) return launch_cfg<128, 128>(L, stream);
  if (L.tile == 128 && L.head_dim == 64) return launch_cfg<128, 64>(L, stream);
  if (L.tile == 64 && L.head_dim == 128) return launch_cfg<64, 128>(L, stream);
  if (L.tile == 64 && L.head_dim == 64) return launch_cfg<64, 64>(L, stream);
  return cudaErrorInvalidValue;
}

}  // namespace evisel
