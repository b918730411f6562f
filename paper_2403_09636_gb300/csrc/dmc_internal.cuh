// Internal layout and device helpers shared by the DMC kernels (sm_103a).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "dmc.h"

namespace dmc {

constexpr int kPage = 32;              // slots per page (the paper's page size)
constexpr int kPrefillChunk = 128;     // prompt tokens per prefill block
constexpr int kMaxVirtualHeads = 16384;
constexpr int kMaxWindow = 32;         // longest window of the window-grouping approximation
constexpr int kDecodeWarpsPerBlock = 6;      // worker warps per block, CUDA-core decode kernel
constexpr int kDecodeWalkWarpsPerBlock = 8;  // the same, for a launch over several layers
constexpr int kGqaWarpsPerBlock = 4;         // worker warps per block, tensor-core decode kernel
// split-K partial states per layer a cache holds for the decode kernels: two
// per worker warp of the largest grid (CUDA-core kernel: 512 blocks x 8 warps;
// tensor-core kernel: 256 blocks x 4 warps, times the group's queries)
constexpr int kMaxWorkerStates = 8192;
constexpr int kGqaWorkerStates = 2048;

// Device-side view of one cache. Passed by value to every kernel.
struct Layout {
  int L, B, Hq, Hkv, G, D, esize;
  int NH;                  // B * Hkv heads per layer
  int MPH;                 // page-table width (pages per head)
  int max_slots;
  int64_t num_pages;
  int row_bytes;           // D * esize
  int page_bytes;          // 2 * kPage * row_bytes (K rows then V rows)
  char* pages;             // [num_pages][2][kPage][D]
  float* z;                // [num_pages][kPage]
  int* page_table;         // [L][NH][MPH]
  int* lengths;            // [L][2][NH]  double-buffered slot counts
  int* ctl;                // [L][4]: parity, finished-block counter
  int* counters;           // [L][NH * G] per (virtual) head combine counters
  char* pending;           // [L][NH][2][D]: grouped queries: new last rows awaiting the layer's end
  int* pending_at;         // [L][NH]: their slot (page * 32 + row), -1 = none
  float* pending_z;        // [L][NH]: their z
  unsigned long long* pool_top;
  unsigned int* error;
  float* partials;         // [partial_cap][D + 2]: split-K partial softmax states (m, l, acc)
  int partial_cap;
  long long partials_layer_stride;  // floats between layers' partial states (CUDA-core kernel;
                                    // 0: one region shared by all layers)
  unsigned char* opens;    // [max_prefill_tokens][Hkv]: token opens a slot
  int* plan;               // [Hkv][plan_stride]: first slot index per prompt chunk
  int plan_stride;
  int max_prefill_tokens;
  // window grouping (window > 0): the open segment's last tokens per head
  int window;              // 0 = exact DMC
  char* ring;              // [L][NH][window][2][D]: token p of the segment at entry p % window
  float* ring_w;           // [L][NH][window]: its omega
  int* seglen;             // [L][2][NH]: tokens of the open segment, double-buffered like lengths
};

__host__ __device__ inline int ceil_div(int a, int b) { return (a + b - 1) / b; }

// Launch shape of the decode kernel for one cache, fixed at create time.
struct DecodePlan {
  int grid;            // blocks of a launch over one layer
  int stages;          // shared-memory ring depth (quads per warp)
  int partial_states;  // split-K partial states one launch may write
  size_t smem;         // dynamic shared memory per block
  int grid_walk;       // blocks and shared memory of a CUDA-core launch over several
  size_t smem_walk;    // layers (its own warp count; grid_walk 0: the one-layer shape);
                       // the tensor-core kernel uses grid, smem
};

// ---------------------------------------------------------------- dtype helpers
template <typename T> struct Elt;
template <> struct Elt<float> {
  static __device__ __forceinline__ float to_f(float x) { return x; }
  static __device__ __forceinline__ float from_f(float x) { return x; }
};
template <> struct Elt<__nv_bfloat16> {
  static __device__ __forceinline__ float to_f(__nv_bfloat16 x) { return __bfloat162float(x); }
  static __device__ __forceinline__ __nv_bfloat16 from_f(float x) { return __float2bfloat16_rn(x); }
};

// Unpacks one 16-byte chunk into floats.
template <typename T> struct Chunk;
template <> struct Chunk<float> {
  static constexpr int N = 4;
  static __device__ __forceinline__ void unpack(const uint4& u, float* f) {
    f[0] = __uint_as_float(u.x); f[1] = __uint_as_float(u.y);
    f[2] = __uint_as_float(u.z); f[3] = __uint_as_float(u.w);
  }
  static __device__ __forceinline__ uint4 pack(const float* f) {
    return make_uint4(__float_as_uint(f[0]), __float_as_uint(f[1]), __float_as_uint(f[2]),
                      __float_as_uint(f[3]));
  }
};
template <> struct Chunk<__nv_bfloat16> {
  static constexpr int N = 8;
  // bf16 -> f32 is exact: the bf16 bits are the high half of the f32 bits.
  static __device__ __forceinline__ void unpack2(uint32_t w, float& lo, float& hi) {
    lo = __uint_as_float(w << 16);
    hi = __uint_as_float(w & 0xffff0000u);
  }
  static __device__ __forceinline__ void unpack(const uint4& u, float* f) {
    unpack2(u.x, f[0], f[1]); unpack2(u.y, f[2], f[3]);
    unpack2(u.z, f[4], f[5]); unpack2(u.w, f[6], f[7]);
  }
  static __device__ __forceinline__ uint32_t pack2(float lo, float hi) {
    __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&h);
  }
  static __device__ __forceinline__ uint4 pack(const float* f) {
    return make_uint4(pack2(f[0], f[1]), pack2(f[2], f[3]), pack2(f[4], f[5]), pack2(f[6], f[7]));
  }
};

__device__ __forceinline__ float sigmoidf_(float x) { return 1.0f / (1.0f + __expf(-x)); }

// ---------------------------------------------------------------- PTX: mbarrier, cp.async, mma
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile(
      "{\n\t.reg .b64 st;\n\t"
      "mbarrier.arrive.shared::cta.b64 st, [%0];\n\t}" ::"r"(bar)
      : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile(
      "{\n\t.reg .b64 st;\n\t"
      "mbarrier.arrive.expect_tx.shared::cta.b64 st, [%0], %1;\n\t}" ::"r"(bar),
      "r"(bytes)
      : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t));
  return t;
}

// Longest in-kernel wait before it gives up. Normal waits take microseconds;
// a build of a test kernel may shorten the limit.
#ifndef DMC_WAIT_LIMIT_NS
#define DMC_WAIT_LIMIT_NS 2000000000ull  // 2 s
#endif
constexpr uint64_t kWaitLimitNs = DMC_WAIT_LIMIT_NS;

// Waits for the phase with the given parity to complete. Gives up after
// kWaitLimitNs, sets DMC_FAULT_WAIT_TIMEOUT and returns false.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, unsigned int* err) {
#pragma unroll 1
  for (int i = 0; i < 128; ++i)
    if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
#pragma unroll 1
  while (true) {
    if (mbar_try_wait(bar, parity)) return true;
    if (globaltimer_ns() - t0 > kWaitLimitNs) {
      atomicOr(err, DMC_FAULT_WAIT_TIMEOUT);
      return false;
    }
  }
}

// cp.async (LDGSTS) of 16 bytes, L2 only, into this thread's shared memory.
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;" ::: "memory");
}
// Waits until at most N of this thread's committed cp.async groups are pending.
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// cp.async of 16 bytes that reads src only when `valid`; otherwise the 16
// shared bytes are zero-filled (src must still be a valid address).
__device__ __forceinline__ void cp_async16_zfill(uint32_t dst, const void* src, bool valid) {
  const uint32_t n = valid ? 16u : 0u;
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(n)
               : "memory");
}

// Four 8x8 b16 matrices from shared memory; lane i gives the row address of
// row i % 8 of matrix i / 8.
__device__ __forceinline__ void ldmatrix_x4(uint32_t addr, uint32_t& r0, uint32_t& r1,
                                            uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr)
               : "memory");
}
__device__ __forceinline__ void ldmatrix_x4_trans(uint32_t addr, uint32_t& r0, uint32_t& r1,
                                                  uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr)
               : "memory");
}

// D = A (16x16, row) * B (16x8, col) + D, bf16 inputs, fp32 accumulate.
__device__ __forceinline__ void mma_bf16_16816(float* d, uint32_t a0, uint32_t a1, uint32_t a2,
                                               uint32_t a3, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
      "{%8, %9}, {%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// Programmatic dependent launch: wait for the grid this one depends on (a
// no-op when launched without the attribute), then let the next grid start.
__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void griddep_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Named barrier over the first `threads` threads of the block.
__device__ __forceinline__ void named_sync(int id, int threads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(threads) : "memory");
}

}  // namespace dmc
