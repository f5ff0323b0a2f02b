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
// cross_frame_pairs_kernel: one CTA per (visual row tile, 8 consecutive
// (kept tile, span) units): one thread per row, and a producer warp. For a
// head the 8 units are one contiguous run of 8 x TILE floats; the producer
// streams the heads' runs into a 4-stage shared-memory ring with 1-D bulk
// copies (cp.async.bulk, mbarrier completion): 8 CTAs of an SM hold 128 KB of
// loads in flight. A row thread sums its row's shares over the heads for the
// 8 units from the ring (LSE read four heads ahead), the CTA sums them over
// the N_v rows of each query frame (shuffles, then a shared-memory step for
// N_v > 32), and the first row of the frame adds the spans of each key frame
// and writes A_ff[a-1, b]. A frame pair
// (a, b) belongs to exactly one (row tile, kept tile), so every entry has one
// writer and a fixed summation order (deterministic).
// Unless it accumulates, the first CTA of each row tile also writes the
// zeros of its query frames' A_ff rows (entries of key frames the mask does
// not keep, and b >= a), so no clearing pass runs before it.
// e_ff_kernel: one CTA per (32 frames, video) forms E_ff from A_ff: the
// received attention by column sums (32 warps over the rows, coalesced), the
// given attention by row sums (a warp per frame); each lane keeps 16 loads in
// flight over four partial sums, and every partial is added in a fixed order.
#include <cstdint>
#include <cuda_runtime.h>

#include "evisel_internal.h"
#include "sm103_ptx.cuh"

namespace evisel {
namespace {

constexpr int kUnits = 8;                        // (kept tile, key span) units per CTA
constexpr int kStages = 4;                       // ring stages of kUnits x TILE floats
static_assert(kUnits % 2 == 0, "a key frame's spans (two at N_v = 128) stay in one CTA's units");
constexpr unsigned kFull = 0xffffffffu;
constexpr int kMaxKeptTiles = kCrossFrameMaxKept;   // kept tiles of a row tile that the clearing CTA stages

// 1-D bulk copy global -> shared, completion on an mbarrier (both addresses
// and the size multiples of 16 bytes).
__device__ __forceinline__ void bulk_load(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar,
                                          uint64_t policy) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;" ::"r"(
          dst),
      "l"(src), "r"(bytes), "r"(bar), "l"(policy)
      : "memory");
}

template <int TILE>
__global__ void __launch_bounds__(TILE + 32) cross_frame_pairs_kernel(const __grid_constant__ CrossFrameLaunch L) {
  extern __shared__ __align__(128) float ring[];  // [kStages][kUnits * TILE]
  __shared__ float red[TILE / 32][kUnits];
  __shared__ int kept[kMaxKeptTiles];
  __shared__ __align__(8) uint64_t bars[2 * kStages];   // full[s], then empty[s]
  __shared__ int abort_flag;
  const VisRow R = L.rows[blockIdx.x];
  const int fpt = L.fpt;                           // spans per kv tile: TILE / min(N_v, 64)
  const int u0 = blockIdx.y * kUnits;              // first unit: kept tile u0 / fpt, span u0 % fpt
  if (u0 >= R.kv_count * fpt) return;              // uniform over the CTA
  const int n_u = min(kUnits, R.kv_count * fpt - u0);
  const VideoInfo vi = L.videos[R.video];
  const int npf = L.tokens_per_frame, spf = L.spans_per_frame;
  const int T = vi.n_vis / npf;
  const int row = threadIdx.x, lane = row & 31, warp = row >> 5;
  const bool valid = row < R.q_len;
  const int a = (R.row_tile * TILE + row) / npf;   // the row's frame (video-local)
  const uint32_t bar0 = ptx::smem_addr(bars);
  auto full = [&](int st) { return bar0 + 8u * st; };
  auto empty = [&](int st) { return bar0 + 8u * (kStages + st); };
  if (threadIdx.x == 0) {
    for (int st = 0; st < kStages; ++st) {
      ptx::mbar_init(full(st), 1);
      ptx::mbar_init(empty(st), TILE / 32);
    }
    abort_flag = 0;
    ptx::fence_mbar_init();
  }
  __syncthreads();
  // Overwrite mode: the first CTA of each row tile writes the zeros of its
  // query frames' rows of A_ff, the entries no CTA writes (key frames of tiles
  // the mask does not keep, and b >= a), so the call needs no clearing pass.
  // The entries it writes and the ones the pairs below write are disjoint.
  if (!L.accumulate && blockIdx.y == 0 && R.kv_count <= kMaxKeptTiles) {
    for (int i = threadIdx.x; i < R.kv_count; i += blockDim.x)
      kept[i] = (L.kv[R.kv_begin + i].start - vi.vis_start) / TILE;
    __syncthreads();
    const int a0 = max(1, (R.row_tile * TILE) / npf);
    const int a1 = min(T, (R.row_tile * TILE + R.q_len) / npf);   // frames [a0, a1) of this row tile
    for (int a_ = a0; a_ < a1; ++a_) {
      float* arow = L.aff + L.aff_off[R.video] + static_cast<int64_t>(a_ - 1) * (T - 1);
      for (int b = threadIdx.x; b < T - 1; b += blockDim.x) {
        bool written = false;
        if (b < a_) {
          const int tb = b * npf / TILE;           // the key frame's tile: kept? (the list is sorted)
          int lo = 0, hi = R.kv_count;
          while (lo < hi) {
            const int mid = (lo + hi) >> 1;
            if (kept[mid] < tb) lo = mid + 1; else hi = mid;
          }
          written = lo < R.kv_count && kept[lo] == tb;
        }
        if (!written) arow[b] = 0.f;
      }
    }
  }
  // Units u0 .. u0 + 7 are consecutive spans of consecutive kept tiles: for a
  // head they are one contiguous run of n_u x TILE floats.
  if (warp == TILE / 32) {
    uint32_t leader = 0;
    if (ptx::elect_one(leader)) {
      const uint64_t pol = ptx::l2_policy_evict_first();
      const float* src = L.fspill + (static_cast<int64_t>(R.kv_begin) * fpt + u0) * TILE;
      const int64_t head_stride = static_cast<int64_t>(L.nnz) * fpt * TILE;
      const uint32_t bytes = static_cast<uint32_t>(n_u * TILE * 4);
      const uint32_t ring0 = ptx::smem_addr(ring);
      int h = 0;
      for (; h < L.hq; ++h) {
        const int st = h % kStages;
        if (h >= kStages && !ptx::mbar_wait(empty(st), (h / kStages - 1) & 1, &abort_flag, kWaitTimeoutNs)) {
          abort_flag = 1;
          atomicExch(L.status, kStatusTimeout);
          break;
        }
        ptx::mbar_arrive_expect_tx(full(st), bytes);
        bulk_load(ring0 + st * kUnits * TILE * 4, src + h * head_stride, bytes, full(st), pol);
      }
      // no copy in flight at exit: the last issued loads have landed
      const volatile int never = 0;
      for (int j = max(0, h - kStages); j < h; ++j)
        ptx::mbar_wait(full(j % kStages), (j / kStages) & 1, &never, kWaitTimeoutNs);
    }
    return;                                        // the sums below are the row threads'
  }
  float v[kUnits];
#pragma unroll
  for (int u = 0; u < kUnits; ++u) v[u] = 0.f;
  {
    const float* lse = L.lse + R.q_start + (valid ? row : 0);
    float mq[4];                                   // LSE of heads h .. h + 3, loaded four heads ahead
#pragma unroll
    for (int i = 0; i < 4; ++i) mq[i] = i < L.hq ? __ldg(lse + static_cast<int64_t>(i) * L.n_tok) : 0.f;
    bool ok = true;
    for (int h0 = 0; h0 < L.hq; h0 += 4) {
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int h = h0 + i;
        if (h < L.hq) {
          const float m = mq[i] * 1.4426950408889634f;
          mq[i] = h + 4 < L.hq ? __ldg(lse + static_cast<int64_t>(h + 4) * L.n_tok) : 0.f;
          const int st = h % kStages;
          // A warp that gives up releases no more stages: the producer stops
          // on the abort flag and waits only for the copies it has issued.
          const bool got =
              ok && __all_sync(kFull, ptx::mbar_wait(full(st), (h / kStages) & 1, &abort_flag, kWaitTimeoutNs));
          if (ok && !got) {
            ok = false;
            if (lane == 0) {
              abort_flag = 1;
              atomicExch(L.status, kStatusTimeout);
            }
          }
          if (got && valid) {
            const float* sr = ring + st * kUnits * TILE + row;
#pragma unroll
            for (int u = 0; u < kUnits; ++u)
              if (u < n_u) v[u] += ptx::ex2(sr[u * TILE] - m);
          }
          __syncwarp();
          if (got && lane == 0) ptx::mbar_arrive(empty(st));
        }
      }
    }
  }
  // Spans -> key frames (spf consecutive units), then sums over the N_v rows
  // of each query frame: shuffles inside a warp, shared memory across warps.
  const int w = npf < 32 ? npf : 32;
#pragma unroll
  for (int u = 0; u < kUnits; ++u) {
    float x = v[u];
    for (int off = w / 2; off > 0; off >>= 1) x += __shfl_xor_sync(kFull, x, off);
    v[u] = x;
  }
  if (npf > 32) {
    if (lane == 0) {
#pragma unroll
      for (int u = 0; u < kUnits; ++u) red[warp][u] = v[u];
    }
    ptx::bar_sync(1, TILE);                        // every row thread gets here (the producer warp has left)
    if (row % npf == 0) {
#pragma unroll
      for (int u = 0; u < kUnits; ++u) {
        float t = 0.f;
        for (int ww = warp; ww < warp + npf / 32; ++ww) t += red[ww][u];
        v[u] = t;
      }
    }
  }
  if (row % npf != 0 || a >= T) return;
  const float inv_norm = 1.f / static_cast<float>(npf * L.hq);
  float* aff = L.aff + L.aff_off[R.video] + static_cast<int64_t>(a - 1) * (T - 1);
  float fsum = 0.f;
#pragma unroll
  for (int u = 0; u < kUnits; ++u) {
    if (u >= n_u) break;
    fsum += v[u];
    const int uu = u0 + u;                         // unit within the row's list
    if ((uu % fpt + 1) % spf != 0) continue;       // the key frame has another span
    const int c_tile = (L.kv[R.kv_begin + uu / fpt].start - vi.vis_start) / TILE;
    const int b = (c_tile * fpt + uu % fpt) / spf; // key frame (video-local)
    if (b < a) {
      const float val = fsum * inv_norm;
      aff[b] = L.accumulate ? aff[b] + val : val;
    }
    fsum = 0.f;
  }
}

constexpr int kEffWarps = 32;

__global__ void __launch_bounds__(kEffWarps * 32) e_ff_kernel(const __grid_constant__ CrossFrameLaunch L) {
  __shared__ float part[kEffWarps][33];
  __shared__ float give[32];
  const VideoInfo vi = L.videos[blockIdx.y];
  const int T = vi.n_vis / L.tokens_per_frame;
  const int t0 = blockIdx.x * 32;
  if (t0 >= T) return;                             // uniform over the CTA
  const float* A = L.aff + L.aff_off[blockIdx.y];  // [(T-1), (T-1)]
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int t = t0 + lane;
  // Received: column t over the rows of frames a > t (row index a - 1 >= t).
  // Four partial sums, 16 loads in flight per lane, added in a fixed order.
  float recv = 0.f;
  if (t <= T - 2) {
    float r4[4] = {0.f, 0.f, 0.f, 0.f};
    int ra = t0 + warp;
    for (; ra + 15 * kEffWarps <= T - 2; ra += 16 * kEffWarps) {
      float x[16];
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        const int rr = ra + i * kEffWarps;
        x[i] = rr >= t ? A[static_cast<int64_t>(rr) * (T - 1) + t] : 0.f;
      }
#pragma unroll
      for (int i = 0; i < 16; ++i) r4[i & 3] += x[i];
    }
    for (; ra <= T - 2; ra += kEffWarps)
      if (ra >= t) r4[0] += A[static_cast<int64_t>(ra) * (T - 1) + t];
    recv = (r4[0] + r4[1]) + (r4[2] + r4[3]);
  }
  part[warp][lane] = recv;
  // Given: row t - 1 over the frames b < t, one warp per frame.
  {
    const int tg = t0 + warp;
    float g = 0.f;
    if (tg >= 1 && tg < T) {
      const float* row = A + static_cast<int64_t>(tg - 1) * (T - 1);
      float g4[4] = {0.f, 0.f, 0.f, 0.f};
      int b = lane;
      for (; b + 15 * 32 < tg; b += 16 * 32) {
        float x[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) x[i] = row[b + i * 32];
#pragma unroll
        for (int i = 0; i < 16; ++i) g4[i & 3] += x[i];
      }
      for (; b < tg; b += 32) g4[0] += row[b];
      g = (g4[0] + g4[1]) + (g4[2] + g4[3]);
    }
    for (int off = 16; off > 0; off >>= 1) g += __shfl_xor_sync(kFull, g, off);
    if (lane == 0) give[warp] = g;
  }
  __syncthreads();
  if (warp == 0 && t < T) {
    float r = 0.f;
#pragma unroll
    for (int w = 0; w < kEffWarps; ++w) r += part[w][lane];
    L.eff[vi.frame_off + t] = 0.5f * (give[lane] + r);
  }
}

template <int TILE>
cudaError_t launch_pairs(const CrossFrameLaunch& L, cudaStream_t stream) {
  constexpr int kRingBytes = kStages * kUnits * TILE * 4;
  static PerDeviceAttr smem_once;
  cudaError_t e = raise_smem_limit(smem_once, reinterpret_cast<const void*>(cross_frame_pairs_kernel<TILE>),
                                   kRingBytes);
  if (e != cudaSuccess) return e;
  dim3 grid(L.n_rows, (L.max_kv * L.fpt + kUnits - 1) / kUnits);
  cross_frame_pairs_kernel<TILE><<<grid, TILE + 32, kRingBytes, stream>>>(L);
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
    e_ff_kernel<<<grid, kEffWarps * 32, 0, stream>>>(L);
    return cudaGetLastError();
  }
  return cudaSuccess;
}

}  // namespace evisel
