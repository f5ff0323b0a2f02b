// Host-side planning rules shared by the two planners (evisel_capi.cpp and
// evisel_noalloc.cu), so that both entry points build the same work plan and
// give bit-identical results. Not part of the public ABI.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

namespace evisel {

// Length of the kv ranges that the text row tiles are split into (every
// planner uses it). Each work item pays a fixed cost (the Q and first K/V
// loads, the O epilogue, and for a split range the fp32 partials), so the
// ranges are long: half of one SM's share of the call's tile work (`work`: kv
// tiles summed over all work items of the call, unsplit), at most 64 tiles,
// never shorter than the longest visual row or 8. Longest-first scheduling
// starts them early, so they do not straggle.
inline int text_split_len(int max_visual, int64_t work) {
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
      sms < 1) {
    cudaGetLastError();
    sms = 148;
  }
  const int64_t share = work / sms / 2;
  const int floor_len = max_visual > 8 ? max_visual : 8;
  const int64_t len = share < 64 ? share : 64;
  return len > floor_len ? static_cast<int>(len) : floor_len;
}

}  // namespace evisel
