// Work split shared by the decode kernels: every head contributes its page
// units plus one owner unit; the list is cut into equal contiguous ranges, one
// per worker warp ("stream-K" at warp granularity).
#pragma once

#include "dmc_internal.cuh"

namespace dmc {

// Worker w owns units [range_start(w), range_start(w + 1)); when there are
// more workers than units some ranges are empty.
__device__ __forceinline__ long long range_start(int w, long long U, int nw) {
  return (long long)w * U / nw;
}

// Index of the (non-empty) worker whose unit range holds unit u.
__device__ __forceinline__ int worker_of_unit(long long u, long long U, int nw) {
  return (int)(((u + 1) * nw - 1) / U);
}

// Largest v in [0, n) with U[v] <= u (U ascending, U[0] = 0).
__device__ __forceinline__ int head_of_unit(const int* U, int n, int u) {
  int lo = 0, hi = n - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (U[mid] <= u) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// Exclusive prefix of units per (virtual) head into U[0..nvh], all threads:
// ceil(len / 32) page units, plus one owner unit per head when owner_units.
// Reads both slot-count buffers together with the parity word, so the prefix
// costs one round trip to memory.
static __device__ void scan_units(int* U, int* wsum, const int* ctl, const int* len_both, int nh,
                           int nvh, int Gv, int owner_units = 1) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int nthr = blockDim.x, nwarps = nthr >> 5;
  const int per = (nvh + nthr - 1) / nthr;
  const int i0 = min(tid * per, nvh), i1 = min(i0 + per, nvh);
  const int parity = *reinterpret_cast<const volatile int*>(ctl);
  int local = 0;
  for (int i = i0; i < i1; ++i) {
    const int l0 = len_both[i / Gv], l1 = len_both[nh + i / Gv];
    const int units = ceil_div(parity ? l1 : l0, kPage) + owner_units;
    U[i] = units;  // per-head count for now, prefixed below
    local += units;
  }
  int incl = local;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    int o = __shfl_up_sync(0xffffffffu, incl, off);
    if (lane >= off) incl += o;
  }
  if (lane == 31) wsum[warp] = incl;
  __syncthreads();
  if (tid == 0) {
    int run = 0;
    for (int w = 0; w < nwarps; ++w) { int t = wsum[w]; wsum[w] = run; run += t; }
    wsum[nwarps] = run;
  }
  __syncthreads();
  int run = wsum[warp] + incl - local;
  for (int i = i0; i < i1; ++i) {
    const int units = U[i];
    U[i] = run;
    run += units;
  }
  if (tid == 0) U[nvh] = wsum[nwarps];
  __syncthreads();
}

// scan_units by one warp, for a single kernel-visible head list (Gv = 1, one
// owner unit per head): the prefix of a later layer, built while the block's
// other warps still work.
static __device__ void scan_units_warp(int* U, const int* ctl, const int* len_both, int nh) {
  const int lane = threadIdx.x & 31;
  const int per = (nh + 31) / 32;
  const int i0 = min(lane * per, nh), i1 = min(i0 + per, nh);
  const int parity = *reinterpret_cast<const volatile int*>(ctl);
  int local = 0;
  for (int i = i0; i < i1; ++i) {
    const int units = ceil_div(parity ? len_both[nh + i] : len_both[i], kPage) + 1;
    U[i] = units;
    local += units;
  }
  int incl = local;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int o = __shfl_up_sync(0xffffffffu, incl, off);
    if (lane >= off) incl += o;
  }
  int run = incl - local;
  for (int i = i0; i < i1; ++i) {
    const int units = U[i];
    U[i] = run;
    run += units;
  }
  if (lane == 31) U[nh] = incl;
  __syncwarp();
}

}  // namespace dmc
