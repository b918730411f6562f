// Prompt-phase DMC attention on the fifth-generation tensor cores (tcgen05).
//
// At inference every prompt token attends over the cache as it stands right
// after that token's own update (Eq. attn-softmax; the training mask of
// Sec. 3.2 with binary alpha gives the same pattern): the slots closed before
// the token, plus the slot the token has just merged into or opened, whose
// value at that moment is the running omega-weighted mean of its segment so
// far (Eq. partial-accumulation). With len(i) the slot count after token i,
// query i therefore sees the final values of slots [0, len(i) - 1) and one
// "diagonal" state.
//
// One CTA of 8 warps per (128 query rows, KV head, sequence); a row is a
// (token, query head of the group) pair, token-major, so a group of G queries
// shares every K/V tile. The closed slots are read from the cache pages that
// the prefill scan has just written, in tiles of 128 slots:
//   S = Q K^T          tcgen05.mma kind::f16, M = N = 128, K = head_dim, into TMEM
//   softmax            two threads per row, each half of its columns:
//                      tcgen05.ld of S, the staircase mask (slot < len(i) - 1),
//                      online softmax in the log2 domain (the halves trade
//                      their maxima through shared memory), P rounded to bf16
//                      and stored over the thread's own S columns in TMEM
//   O += P V           tcgen05.mma with P read from TMEM and V as an MN-major B
//                      operand, into TMEM
// The diagonal state enters as one more tile built from the prompt's k, v rows
// of the token's 128-token chunk and the segment sums the prefill scan
// recorded at the chunk start ("carry"): its score is Q Kraw^T summed with the
// segment's weights, its value P_d Vraw (see the end of the kernel).
#include <math.h>

#include "dmc_internal.cuh"

namespace dmc {

constexpr int kPaRows = 128;     // query rows per tile (M)
constexpr int kPaSlots = 128;    // slots per K/V tile (N of S, K of P V)
constexpr int kPaThreads = 256;  // two threads per query row, each half of its columns
constexpr int kPaD = 128;        // head_dim handled by this kernel
constexpr int kPaTileBytes = kPaRows * kPaD * 2;  // 32 KB: [128 rows][256 B]
// dynamic shared memory: Q | K | V | misc, 104 KB: two CTAs per SM (P lives in TMEM)
constexpr int kPaQ = 0, kPaK = kPaTileBytes, kPaV = 2 * kPaTileBytes;
constexpr int kPaMisc = 3 * kPaTileBytes;
constexpr int kPaSmem = kPaMisc + 8192;

struct PrefillAttnArgs {
  Layout lay;
  int layer, first_seq, num_seqs;
  const char* q;   // [total_tokens][Hq][D]
  const char* k;   // [total_tokens][Hkv][D]
  const char* v;
  const int* cu;
  int total_tokens, max_seqlen;
  const float* carry;  // [chunk id][Hkv][2D + 1]
  char* out;           // [total_tokens][Hq][D]
};

// byte offset of 16-byte chunk j (0..15) of row r in a [128 rows][256 B] tile
// kept as two 128-byte column halves, 128B-swizzled (chunk ^ row % 8)
__device__ __forceinline__ uint32_t pa_swz(int r, int j) {
  return (uint32_t)((j >> 3) * (kPaRows * 128) + r * 128 + (((j & 7) ^ (r & 7)) << 4));
}

// tcgen05 shared-memory matrix descriptor: 128B swizzle, start address, leading
// and stride byte offsets (all in 16-byte units), descriptor version 1
__device__ __forceinline__ uint64_t pa_desc(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
  return (uint64_t)((saddr >> 4) & 0x3FFF) | ((uint64_t)((lbo >> 4) & 0x3FFF) << 16) |
         ((uint64_t)((sbo >> 4) & 0x3FFF) << 32) | ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}

// instruction descriptor, kind::f16: bf16 A and B, fp32 D, M = N = 128;
// b_mn selects an MN-major B operand
__device__ __forceinline__ uint32_t pa_idesc(bool b_mn) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((b_mn ? 1u : 0u) << 16) | ((128u >> 3) << 17) |
         ((128u >> 4) << 24);
}

__device__ __forceinline__ void pa_mma(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc,
                                       bool acc) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a), "l"(b), "r"(idesc), "r"(acc ? 1 : 0));
}

// the same with A (M x K, bf16 pairs packed in 32-bit columns) read from tensor memory
__device__ __forceinline__ void pa_mma_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b, uint32_t idesc,
                                          bool acc) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b), "r"(idesc), "r"(acc ? 1 : 0));
}

// 2^x by the SFU (ex2.approx, flushing subnormal results to zero)
__device__ __forceinline__ float pa_ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ void pa_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                   bar)
               : "memory");
}

// 32 consecutive fp32 columns of this thread's TMEM lane
__device__ __forceinline__ void pa_ld32(uint32_t taddr, float* f) {
  uint32_t v[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,"
      "%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]),
        "=r"(v[7]), "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]),
        "=r"(v[14]), "=r"(v[15]), "=r"(v[16]), "=r"(v[17]), "=r"(v[18]), "=r"(v[19]), "=r"(v[20]),
        "=r"(v[21]), "=r"(v[22]), "=r"(v[23]), "=r"(v[24]), "=r"(v[25]), "=r"(v[26]), "=r"(v[27]),
        "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 32; ++i) f[i] = __uint_as_float(v[i]);
}

__device__ __forceinline__ void pa_st32(uint32_t taddr, const float* f) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,"
      "%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
      "r"(__float_as_uint(f[0])), "r"(__float_as_uint(f[1])), "r"(__float_as_uint(f[2])),
      "r"(__float_as_uint(f[3])), "r"(__float_as_uint(f[4])), "r"(__float_as_uint(f[5])),
      "r"(__float_as_uint(f[6])), "r"(__float_as_uint(f[7])), "r"(__float_as_uint(f[8])),
      "r"(__float_as_uint(f[9])), "r"(__float_as_uint(f[10])), "r"(__float_as_uint(f[11])),
      "r"(__float_as_uint(f[12])), "r"(__float_as_uint(f[13])), "r"(__float_as_uint(f[14])),
      "r"(__float_as_uint(f[15])), "r"(__float_as_uint(f[16])), "r"(__float_as_uint(f[17])),
      "r"(__float_as_uint(f[18])), "r"(__float_as_uint(f[19])), "r"(__float_as_uint(f[20])),
      "r"(__float_as_uint(f[21])), "r"(__float_as_uint(f[22])), "r"(__float_as_uint(f[23])),
      "r"(__float_as_uint(f[24])), "r"(__float_as_uint(f[25])), "r"(__float_as_uint(f[26])),
      "r"(__float_as_uint(f[27])), "r"(__float_as_uint(f[28])), "r"(__float_as_uint(f[29])),
      "r"(__float_as_uint(f[30])), "r"(__float_as_uint(f[31]))
      : "memory");
}

__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void fence_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

template <int G>
__global__ void __launch_bounds__(kPaThreads, 2) dmc_prefill_attn_kernel(const PrefillAttnArgs a) {
  constexpr int D = kPaD;
  constexpr int ROW = D * 2;          // bytes per bf16 row
  constexpr int TT = kPaRows / G;     // tokens per tile
  constexpr int HALF = kPaSlots / 2;  // columns of S (and of O) per thread
  extern __shared__ __align__(1024) unsigned char smem[];
  const Layout& L = a.lay;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int tile = blockIdx.x, h = blockIdx.y, s = blockIdx.z;
  const int bh = (a.first_seq + s) * L.Hkv + h;

  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kPaMisc);  // [0] S done, [1] O done
  uint32_t* tslot = reinterpret_cast<uint32_t*>(smem + kPaMisc + 16);
  volatile int* s_abort = reinterpret_cast<volatile int*>(smem + kPaMisc + 32);  // a wait gave up
  int* s_len = reinterpret_cast<int*>(smem + kPaMisc + 64);            // [128] slots after token
  float* s_om = reinterpret_cast<float*>(smem + kPaMisc + 64 + 512);   // [128] omega
  float* s_rz = reinterpret_cast<float*>(smem + kPaMisc + 64 + 1024);  // [128] 1 / z after token
  float* s_x = reinterpret_cast<float*>(smem + kPaMisc + 64 + 1536);   // [2][128] row exchange
  float* s_y = reinterpret_cast<float*>(smem + kPaMisc + 64 + 2560);   // [2][128] row exchange
  unsigned char* s_op = smem + kPaMisc + 64 + 3584;                    // [128] token opens a slot
  int* s_wc = reinterpret_cast<int*>(smem + kPaMisc + 64 + 3712);      // [4] openings per warp
  int* s_wf = reinterpret_cast<int*>(smem + kPaMisc + 64 + 3728);      // [4] the warp has one
  float* s_wz = reinterpret_cast<float*>(smem + kPaMisc + 64 + 3744);  // [4] its last segment's omega sum
  int* s_wm = reinterpret_cast<int*>(smem + kPaMisc + 64 + 3760);      // [4] its last opening token
  int* s_seg = reinterpret_cast<int*>(smem + kPaMisc + 4096);          // [128] first token of the segment, or -1

  const int t0 = a.cu[s], t1 = a.cu[s + 1];
  if (!(t0 >= 0 && t0 <= t1 && t1 <= a.total_tokens && t1 - t0 <= a.max_seqlen)) return;
  const int tok0 = t0 + tile * TT;
  if (tok0 >= t1) return;
  const int tokN = min(tok0 + TT, t1);
  const int c = (tok0 - t0) / kPrefillChunk;
  const int a0 = t0 + c * kPrefillChunk;  // the chunk holding the tile
  const int cid = (t0 + c * kPrefillChunk) / kPrefillChunk + s;
  const int base = L.plan[(size_t)h * L.plan_stride + cid];  // slots before the chunk
  if (base < 0) return;  // the plan failed (capacity or pool); its fault bit is set
  const int parity = *reinterpret_cast<volatile int*>(&L.ctl[a.layer * 4]);
  const int len_final = L.lengths[((size_t)a.layer * 2 + parity) * L.NH + bh];
  const int* ptab = L.page_table + ((size_t)a.layer * L.NH + bh) * L.MPH;
  const __nv_bfloat16* qg = reinterpret_cast<const __nv_bfloat16*>(a.q);
  const float* carry = a.carry + ((size_t)cid * L.Hkv + h) * (2 * D + 1);

  // ---- Q and the first K/V tile start streaming before anything else. The
  // first tile is read up to min(128, len_final) slots: every slot the head
  // holds has been written, and the staircase mask hides those a row does not
  // see; tiles after the first are read up to the slots the tile's rows see.
  const uint32_t sQ = smem_u32(smem + kPaQ);
  for (int i = tid; i < kPaRows * 16; i += kPaThreads) {
    const int rr = i >> 4, j = i & 15;
    const int tt = tok0 + rr / G;
    const bool ok = tt < tokN;
    const char* src = a.q + (((size_t)(ok ? tt : tok0) * L.Hq + (size_t)h * G + rr % G) * ROW) + j * 16;
    cp_async16_zfill(sQ + pa_swz(rr, j), src, ok);
  }
  // K (which = 0) or V (which = 1) rows of slot tile jt, slots below hi
  auto load_tile = [&](int which, int jt, int hi) {
    const uint32_t dst = smem_u32(smem + (which ? kPaV : kPaK));
    for (int i = tid; i < kPaSlots * 16; i += kPaThreads) {
      const int rr = i >> 4, j = i & 15;
      const int slot = jt * kPaSlots + rr;
      const bool ok = slot < hi;
      const int page = ok ? ptab[slot / kPage] : 0;
      const char* src = L.pages + (size_t)page * L.page_bytes +
                        (size_t)(ok ? slot % kPage : 0) * ROW + (size_t)which * kPage * ROW + j * 16;
      cp_async16_zfill(dst + pa_swz(rr, j), src, ok);
    }
  };
  // copy groups, oldest first: Q + K0, V0, then per tile K(j + 1) and V(j + 1)
  load_tile(0, 0, min(kPaSlots, len_final));
  cp_async_commit();
  load_tile(1, 0, min(kPaSlots, len_final));
  cp_async_commit();

  // ---- per-token decisions, omega, slot counts and 1 / z of the chunk up to
  // the tile end. z after token i is the omega sum of i's segment so far: from
  // the segment's opening token, or from the carried sums when no token of the
  // chunk up to i opens a slot (a segmented prefix sum over the chunk).
  int incl = 0, seg = 0, lastop = -1;
  float zs = 0.f;
  if (tid < kPrefillChunk) {
    const int tau = a0 + tid;
    int op = 0;
    float om = 0.f;
    if (tau < tokN) {
      op = L.opens[(size_t)tau * L.Hkv + h];
      float y = 0.f;
#pragma unroll
      for (int g = 0; g < G; ++g)
        y += __bfloat162float(qg[((size_t)tau * L.Hq + (size_t)h * G + g) * D]);
      om = sigmoidf_(y / (float)G);  // omega = sigmoid(mean of the group's q[0])
    }
    s_op[tid] = (unsigned char)op;
    s_om[tid] = om;
    // within the warp for now: openings up to this token, and the omega sum
    // back to the last opening (seg: one was found)
    incl = op;
    seg = op;
    zs = om;
    lastop = op ? tid : -1;  // the last opening token up to this one
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int o = __shfl_up_sync(0xffffffffu, incl, off);
      const int so = __shfl_up_sync(0xffffffffu, seg, off);
      const float zo = __shfl_up_sync(0xffffffffu, zs, off);
      const int lo = __shfl_up_sync(0xffffffffu, lastop, off);
      if (lane >= off) {
        incl += o;
        if (!seg) zs += zo;
        seg |= so;
        lastop = max(lastop, lo);
      }
    }
    if (lane == 31) {
      s_wc[warp] = incl;
      s_wf[warp] = seg;
      s_wz[warp] = zs;
      s_wm[warp] = lastop;
    }
  }
  if (tid == 0) {
    mbar_init(smem_u32(&bars[0]), 1);
    mbar_init(smem_u32(&bars[1]), 1);
    fence_mbar_init();
    *s_abort = 0;
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(tslot)),
                 "r"(256));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  __syncthreads();
  if (tid < kPrefillChunk) {
    int add = base;
    for (int w = 0; w < warp; ++w) add += s_wc[w];
    s_len[tid] = incl + add;  // slot count after token a0 + tid
    for (int w = 0; w < warp; ++w) lastop = max(lastop, s_wm[w]);
    s_seg[tid] = lastop;
    if (!seg) {
      // the segment runs in from earlier warps, or from before the chunk
      bool found = false;
      for (int w = warp - 1; w >= 0 && !found; --w) {
        zs += s_wz[w];
        found = s_wf[w] != 0;
      }
      if (!found) zs += carry[2 * D];  // no opening in the chunk up to here
    }
    s_rz[tid] = 1.f / zs;
  }
  __syncthreads();

  // ---- thread (r, hf): query row r (token tok0 + r / G, query head h G + r % G),
  // columns [hf * 64, hf * 64 + 64) of its S and O rows
  const int r = tid & (kPaRows - 1), hf = tid >> 7;
  const int tau_r = tok0 + r / G;
  const bool row_ok = tau_r < tokN;
  const int nvis = row_ok ? s_len[tau_r - a0] - 1 : 0;  // closed slots this row sees
  const int nvis_max = s_len[tokN - 1 - a0] - 1;
  const int vis_hi = min(nvis_max, len_final);          // slots worth loading
  const int ntiles = (vis_hi + kPaSlots - 1) / kPaSlots;

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tslot;
  const uint32_t tS = tmem, tO = tmem + 128;
  const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;  // this warp's TMEM lanes
  const uint32_t col0 = hf * HALF;                                // this thread's first column
  const float qscale = 1.4426950408889634f / sqrtf((float)D);   // log2(e) / sqrt(d_h)

  // Waits for a tensor-core commit. A wait that gives up (mbar_wait sets the
  // fault bit) raises s_abort; later waits then return at once, and the block
  // leaves at the next point where every thread has passed a barrier after
  // the wait: no further MMA is issued, its copies drain, TMEM is freed.
  auto wait_bar = [&](int which, int ph) {
    if (*s_abort) return;
    if (!mbar_wait(smem_u32(&bars[which]), ph, L.error)) *s_abort = 1;
  };
  auto leave = [&]() {
    cp_async_wait<0>();
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
      tc_fence_after();
      asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(256));
    }
  };

  // Per slot tile j, with P kept in tensor memory so that the K buffer frees
  // as soon as S is computed:
  //   K(j) landed -> S = Q K^T -> K(j + 1) starts -> softmax, P (bf16) over
  //   this thread's own S columns -> V(j) landed -> O += P V -> V(j + 1) starts
  // The copy groups stay in step (one, possibly empty, per K and per V slot),
  // so "all but the newest group" always means the tile needed next.
  float m = -INFINITY, l = 0.f;  // l: this thread's half of the row sum
  for (int jt = 0; jt < ntiles; ++jt) {
    cp_async_wait<1>();  // Q and K(jt) have landed (this thread's copies)
    fence_async_smem();
    __syncthreads();
    if (*s_abort) break;  // uniform: every wait that could raise it is behind the barrier
    if (tid == 0) {
      tc_fence_after();
      const uint32_t kA = sQ, kB = smem_u32(smem + kPaK);
#pragma unroll
      for (int kk = 0; kk < D / 16; ++kk) {
        const uint32_t off = (kk >> 2) * (kPaRows * 128) + (kk & 3) * 32;
        pa_mma(tS, pa_desc(kA + off, 16, 1024), pa_desc(kB + off, 16, 1024), pa_idesc(false), kk > 0);
      }
      pa_commit(smem_u32(&bars[0]));
    }
    wait_bar(0, jt & 1);  // S is in TMEM and the K buffer is free
    tc_fence_after();
    if (jt + 1 < ntiles) load_tile(0, jt + 1, vis_hi);
    cp_async_commit();
    // ---- online softmax: this thread's half of the row. The running maximum m
    // moves only when a tile's row maximum exceeds it by more than 8 (P then
    // stays below 2^8; O and l are rescaled only on a move), in the log2 domain.
    const int vis_row = min(max(nvis - jt * kPaSlots, 0), kPaSlots);  // visible columns of the row
    const int vis_me = min(max(vis_row - (int)col0, 0), HALF);         // ... in this half
    const int vis_warp = __reduce_max_sync(0xffffffffu, vis_me);       // TMEM loads are warp-wide
    const bool full = __all_sync(0xffffffffu, vis_me == HALF);         // no mask in this warp
    float mx = -INFINITY;  // of the raw scores
    for (int c0 = 0; c0 < vis_warp; c0 += 32) {
      float f[32];
      pa_ld32(tS + lane_base + col0 + c0, f);
      if (full) {
#pragma unroll
        for (int i = 0; i < 32; ++i) mx = fmaxf(mx, f[i]);
      } else {
#pragma unroll
        for (int i = 0; i < 32; ++i)
          if (c0 + i < vis_me) mx = fmaxf(mx, f[i]);
      }
    }
    s_x[hf * kPaRows + r] = mx * qscale;  // qscale > 0
    __syncthreads();
    if (*s_abort) break;
    const float mt = fmaxf(mx * qscale, s_x[(hf ^ 1) * kPaRows + r]);  // the tile's row maximum
    const bool grow = mt > m + 8.f;  // false while the row has seen nothing
    const float mn = grow ? mt : m;
    const float nmn = -mn;
    float sum = 0.f;
    uint32_t pk[HALF / 2];  // P of this half, bf16 pairs
#pragma unroll
    for (int c0 = 0; c0 < HALF; c0 += 32) {
      float f[32];
      if (c0 < vis_warp) {
        pa_ld32(tS + lane_base + col0 + c0, f);
        if (full) {
#pragma unroll
          for (int i = 0; i < 32; ++i) f[i] = pa_ex2(fmaf(f[i], qscale, nmn));
        } else {
#pragma unroll
          for (int i = 0; i < 32; ++i) f[i] = (c0 + i < vis_me) ? pa_ex2(fmaf(f[i], qscale, nmn)) : 0.f;
        }
      } else {
#pragma unroll
        for (int i = 0; i < 32; ++i) f[i] = 0.f;
      }
#pragma unroll
      for (int i = 0; i < 32; ++i) sum += f[i];
#pragma unroll
      for (int i = 0; i < 16; ++i) pk[c0 / 2 + i] = Chunk<__nv_bfloat16>::pack2(f[2 * i], f[2 * i + 1]);
    }
    // P over the first half of this thread's own S columns: slots col0 + 2i,
    // col0 + 2i + 1 in column col0 + i (the other half's thread writes its own)
    {
      float pf[32];
#pragma unroll
      for (int i = 0; i < 32; ++i) pf[i] = __uint_as_float(pk[i]);
      pa_st32(tS + lane_base + col0, pf);
    }
    // a move of the maximum rescales l and this half of O (rows that saw
    // nothing yet hold zeros)
    const bool resc = grow && m != -INFINITY;
    const float corr = resc ? pa_ex2(m - mn) : 1.f;
    l = l * corr + sum;
    if (__any_sync(0xffffffffu, resc)) {
      for (int c0 = 0; c0 < HALF; c0 += 32) {
        float f[32];
        pa_ld32(tO + lane_base + col0 + c0, f);
#pragma unroll
        for (int i = 0; i < 32; ++i) f[i] *= corr;
        pa_st32(tO + lane_base + col0 + c0, f);
      }
    }
    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
    m = mn;
    cp_async_wait<1>();  // V(jt) has landed (K(jt + 1) may still be on its way)
    fence_async_smem();
    tc_fence_before();
    __syncthreads();
    if (tid == 0) {
      tc_fence_after();
      const uint32_t vB = smem_u32(smem + kPaV);
#pragma unroll
      for (int kk = 0; kk < kPaSlots / 16; ++kk) {
        // slots 16 kk ... from half kk / 4 of the row, 8 packed columns per step
        const uint32_t aT = tS + (uint32_t)((kk >> 2) * HALF + (kk & 3) * 8);
        pa_mma_ts(tO, aT, pa_desc(vB + kk * 2048, kPaRows * 128, 1024), pa_idesc(true), jt > 0 || kk > 0);
      }
      pa_commit(smem_u32(&bars[1]));
    }
    // P V done: O holds this tile, S (P) and the V buffer are free
    wait_bar(1, jt & 1);
    tc_fence_after();
    if (jt + 1 < ntiles) load_tile(1, jt + 1, vis_hi);
    cp_async_commit();
  }
  cp_async_wait<0>();
  tc_fence_after();
  __syncthreads();  // every MMA and copy of the loop is over: the K and V buffers are free
  if (*s_abort) {
    leave();
    return;
  }

  // ---- the diagonal state as one more tile. When token i of the chunk
  // attends, its own slot holds k~ = (c_k [no opening in the chunk up to i] +
  // sum over j = lo..i of omega_j k_j) / z_i, lo being its segment's first
  // token in the chunk (c_k: the carried sums), and v~ alike. Its score
  // q . k~ and its share of O come from the chunk's raw rows:
  // S_d = Q Kraw^T (with q[0] cleared: the gate is not a feature) summed with
  // the weights omega_j / z_i, then O += P_d Vraw with
  // P_d[j] = exp2(score - m) omega_j / z_i over the segment's columns.
  const int nrows = tokN - a0;
  if (tid < kPaRows) *reinterpret_cast<__nv_bfloat16*>(smem + kPaQ + pa_swz(tid, 0)) = __float2bfloat16_rn(0.f);
  {
    const uint32_t sK = smem_u32(smem + kPaK), sV = smem_u32(smem + kPaV);
    for (int i = tid; i < kPaRows * 16; i += kPaThreads) {
      const int rr = i >> 4, j = i & 15;
      const bool ok = rr < nrows;
      const size_t src = ((size_t)(a0 + (ok ? rr : 0)) * L.Hkv + h) * ROW + j * 16;
      cp_async16_zfill(sK + pa_swz(rr, j), a.k + src, ok);
      cp_async16_zfill(sV + pa_swz(rr, j), a.v + src, ok);
    }
    cp_async_commit();
    cp_async_wait<0>();
  }
  fence_async_smem();
  tc_fence_before();
  __syncthreads();
  if (tid == 0) {
    tc_fence_after();
    const uint32_t kB = smem_u32(smem + kPaK);
#pragma unroll
    for (int kk = 0; kk < D / 16; ++kk) {
      const uint32_t off = (kk >> 2) * (kPaRows * 128) + (kk & 3) * 32;
      pa_mma(tS, pa_desc(sQ + off, 16, 1024), pa_desc(kB + off, 16, 1024), pa_idesc(false), kk > 0);
    }
    pa_commit(smem_u32(&bars[0]));
  }
  const int ti = (row_ok ? r / G : 0) + (tok0 - a0);  // the row's token in the chunk
  const int sg = s_seg[ti];                            // its segment's first token, or -1
  const int lo = max(sg, 0);
  const float rz = s_rz[ti];
  float cdot = 0.f;  // q . c_k over this half's dims, when the segment runs in from before the chunk
  if (sg < 0) {
#pragma unroll
    for (int jj = 0; jj < 8; ++jj) {
      const int cj = hf * 8 + jj;
      float qf[8];
      Chunk<__nv_bfloat16>::unpack(*reinterpret_cast<const uint4*>(smem + kPaQ + pa_swz(r, cj)), qf);
#pragma unroll
      for (int e = 0; e < 8; ++e) cdot = fmaf(qf[e], carry[cj * 8 + e], cdot);
    }
  }
  wait_bar(0, ntiles & 1);  // S_d is in TMEM
  tc_fence_after();
  float wsum = 0.f;
#pragma unroll
  for (int c0 = 0; c0 < HALF; c0 += 32) {
    float f[32];
    pa_ld32(tS + lane_base + col0 + c0, f);
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      const int j = (int)col0 + c0 + i;
      if (j >= lo && j <= ti) wsum = fmaf(s_om[j], f[i], wsum);
    }
  }
  s_x[hf * kPaRows + r] = wsum + cdot;
  __syncthreads();
  if (*s_abort) {
    leave();
    return;
  }
  const float dsc = (s_x[r] + s_x[kPaRows + r]) * rz * qscale;  // the diagonal score (log2 units)
  {
    const bool grow = dsc > m + 8.f;
    const float mn = grow ? dsc : m;
    const bool resc = grow && m != -INFINITY;
    const float corr = resc ? pa_ex2(m - mn) : 1.f;
    l *= corr;
    if (__any_sync(0xffffffffu, resc)) {
      for (int c0 = 0; c0 < HALF; c0 += 32) {
        float f[32];
        pa_ld32(tO + lane_base + col0 + c0, f);
#pragma unroll
        for (int i = 0; i < 32; ++i) f[i] *= corr;
        pa_st32(tO + lane_base + col0 + c0, f);
      }
    }
    m = mn;
  }
  const float pd = pa_ex2(dsc - m);  // the diagonal's weight, below 2^8
  const float pw = pd * rz;
  {
    uint32_t pk[HALF / 2];
#pragma unroll
    for (int c0 = 0; c0 < HALF; c0 += 32) {
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        const int j = (int)col0 + c0 + 2 * i;
        const float p0 = (j >= lo && j <= ti) ? pw * s_om[j] : 0.f;
        const float p1 = (j + 1 >= lo && j + 1 <= ti) ? pw * s_om[j + 1] : 0.f;
        pk[c0 / 2 + i] = Chunk<__nv_bfloat16>::pack2(p0, p1);
      }
    }
    float pf[32];
#pragma unroll
    for (int i = 0; i < 32; ++i) pf[i] = __uint_as_float(pk[i]);
    pa_st32(tS + lane_base + col0, pf);
  }
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
  s_y[hf * kPaRows + r] = l + (hf == 0 ? pd : 0.f);  // the row sum, the diagonal counted once
  tc_fence_before();
  __syncthreads();
  if (tid == 0) {
    tc_fence_after();
    const uint32_t vB = smem_u32(smem + kPaV);
#pragma unroll
    for (int kk = 0; kk < kPaSlots / 16; ++kk) {
      const uint32_t aT = tS + (uint32_t)((kk >> 2) * HALF + (kk & 3) * 8);
      pa_mma_ts(tO, aT, pa_desc(vB + kk * 2048, kPaRows * 128, 1024), pa_idesc(true), ntiles > 0 || kk > 0);
    }
    pa_commit(smem_u32(&bars[1]));
  }
  wait_bar(1, ntiles & 1);
  tc_fence_after();
  const float inv = 1.f / (s_y[r] + s_y[kPaRows + r]);
  const float cw = (sg < 0) ? pw : 0.f;  // weight of the carried value sums
  char* orow = a.out + ((size_t)(row_ok ? tau_r : tok0) * L.Hq + (size_t)h * G + r % G) * ROW;
  for (int c0 = 0; c0 < HALF; c0 += 32) {
    float f[32];
    pa_ld32(tO + lane_base + col0 + c0, f);
    if (row_ok) {
#pragma unroll
      for (int q4 = 0; q4 < 4; ++q4) {
        const int cc = col0 + c0 + q4 * 8;
        float o[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) o[e] = fmaf(cw, carry[D + cc + e], f[q4 * 8 + e]) * inv;
        *reinterpret_cast<uint4*>(orow + cc * 2) = Chunk<__nv_bfloat16>::pack(o);
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(256));
  }
}

bool prefill_attn_supported(const Layout& L) {
  return L.esize == 2 && L.D == kPaD && (L.G == 1 || L.G == 2 || L.G == 4 || L.G == 8);
}

template <int G>
static cudaError_t launch_pa(const PrefillAttnArgs& a, cudaStream_t stream) {
  cudaError_t e = cudaFuncSetAttribute(dmc_prefill_attn_kernel<G>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, kPaSmem);
  if (e != cudaSuccess) return e;
  constexpr int TT = kPaRows / G;
  const int tiles = (a.max_seqlen + TT - 1) / TT;
  if (tiles == 0) return cudaSuccess;
  dmc_prefill_attn_kernel<G><<<dim3(tiles, a.lay.Hkv, a.num_seqs), kPaThreads, kPaSmem, stream>>>(a);
  return cudaGetLastError();
}

cudaError_t prefill_attn_launch(const Layout& L, int layer, int first_seq, int num_seqs,
                                const void* q, const void* k, const void* v, const int* cu,
                                int total_tokens, int max_seqlen, const float* carry, void* out,
                                cudaStream_t stream) {
  PrefillAttnArgs a;
  a.lay = L;
  a.layer = layer;
  a.first_seq = first_seq;
  a.num_seqs = num_seqs;
  a.q = static_cast<const char*>(q);
  a.k = static_cast<const char*>(k);
  a.v = static_cast<const char*>(v);
  a.cu = cu;
  a.total_tokens = total_tokens;
  a.max_seqlen = max_seqlen;
  a.carry = carry;
  a.out = static_cast<char*>(out);
  switch (L.G) {
    case 1: return launch_pa<1>(a, stream);
    case 2: return launch_pa<2>(a, stream);
    case 4: return launch_pa<4>(a, stream);
    case 8: return launch_pa<8>(a, stream);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace dmc
