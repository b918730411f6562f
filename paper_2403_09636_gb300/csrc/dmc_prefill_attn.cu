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
// two copies (by item parity) of a chunk's carried sums, 2D + 1 floats each
constexpr int kPaCarry = kPaMisc + 8192;
constexpr int kPaCarryBytes = 1040;
constexpr int kPaSmem = kPaCarry + 2 * kPaCarryBytes;  // two CTAs per SM

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
  int seq_base;        // this launch's first sequence within the call (chunk ids count sequences)
};

// Sequences per launch: the per-CTA table of work items before each sequence
// lives in shared memory.
constexpr int kPaMaxSeqs = 768;
static_assert(kPaMaxSeqs == 3 * kPaThreads, "three sequences per thread in the item prefix");

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

// cp.async of 4 bytes (through L1) into shared memory
__device__ __forceinline__ void pa_cp_async4(uint32_t dst, const void* src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(dst), "l"(src) : "memory");
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

// Persistent: each CTA takes query tiles (work items) from a counter in the
// layer's control words until none is left; the last CTA to finish resets the
// counter. Items run sequence by sequence and KV head by KV head, so the CTAs
// at work share a few heads' slot tiles in L2, and each head's tiles from the
// last (which see the most slots) to the first. TMEM, the mbarriers and their
// phases live across items, and an item's Q, first K/V tile and per-token
// inputs are requested while the item before it finishes: Q once the previous
// diagonal score no longer needs the Q buffer, the rest once its last P V is
// done.
template <int G>
__global__ void __launch_bounds__(kPaThreads, 2) dmc_prefill_attn_kernel(const PrefillAttnArgs a) {
  constexpr int D = kPaD;
  constexpr int ROW = D * 2;          // bytes per bf16 row
  constexpr int TT = kPaRows / G;     // tokens per tile
  constexpr int HALF = kPaSlots / 2;  // columns of S (and of O) per thread
  extern __shared__ __align__(1024) unsigned char smem[];
  const Layout& L = a.lay;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kPaMisc);  // [0] S done, [1] O done
  uint32_t* tslot = reinterpret_cast<uint32_t*>(smem + kPaMisc + 16);
  volatile int* s_abort = reinterpret_cast<volatile int*>(smem + kPaMisc + 32);  // a wait gave up
  volatile int* s_item = reinterpret_cast<volatile int*>(smem + kPaMisc + 40);   // [2] next item
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
  int* s_pref = reinterpret_cast<int*>(smem + kPaMisc + 4608);         // [num_seqs + 1] items before each sequence

  int* ctr = L.ctl + a.layer * 4 + 2;  // [0] the next work item, [1] CTAs done
  const int parity = *reinterpret_cast<volatile int*>(&L.ctl[a.layer * 4]);
  // ---- the work items: Hkv x ceil(len / TT) per valid sequence, their
  // exclusive prefix per sequence (3 sequences per thread, one block scan)
  {
    int cnt[3], sum = 0;
#pragma unroll
    for (int k = 0; k < 3; ++k) {
      const int sq = 3 * tid + k;
      cnt[k] = 0;
      if (sq < a.num_seqs) {
        const int t0 = a.cu[sq], t1 = a.cu[sq + 1];
        if (t0 >= 0 && t0 <= t1 && t1 <= a.total_tokens && t1 - t0 <= a.max_seqlen)
          cnt[k] = L.Hkv * ((t1 - t0 + TT - 1) / TT);
      }
      sum += cnt[k];
    }
    int incl = sum;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int o = __shfl_up_sync(0xffffffffu, incl, off);
      if (lane >= off) incl += o;
    }
    if (lane == 31) s_x[warp] = __int_as_float(incl);
    __syncthreads();
    int run = incl - sum;
    for (int w = 0; w < warp; ++w) run += __float_as_int(s_x[w]);
#pragma unroll
    for (int k = 0; k < 3; ++k) {
      const int sq = 3 * tid + k;
      if (sq < a.num_seqs) s_pref[sq] = run;
      run += cnt[k];
    }
    if (tid == kPaThreads - 1) s_pref[a.num_seqs] = run;  // the last thread's run is the total
    __syncthreads();
  }
  const int nitems = s_pref[a.num_seqs];
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
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tslot;
  const uint32_t tS = tmem, tO = tmem + 128;
  const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;  // this warp's TMEM lanes
  const int hf = tid >> 7;
  const uint32_t col0 = hf * HALF;                                // this thread's first column
  const float qscale = 1.4426950408889634f / sqrtf((float)D);   // log2(e) / sqrt(d_h)
  uint32_t ph[2] = {0u, 0u};  // phase parity of the next completion of each mbarrier

  // Waits for a tensor-core commit. A wait that gives up (mbar_wait sets the
  // fault bit) raises s_abort; later waits then return at once, and the CTA
  // leaves at the next point where every thread has passed a barrier after
  // the wait: no further MMA is issued, its copies drain, TMEM is freed.
  auto wait_bar = [&](int which) {
    if (!*s_abort && !mbar_wait(smem_u32(&bars[which]), ph[which], L.error)) *s_abort = 1;
    ph[which] ^= 1u;
  };

  const uint32_t sQ = smem_u32(smem + kPaQ);
  const __nv_bfloat16* qg = reinterpret_cast<const __nv_bfloat16*>(a.q);

  // One work item: the query tile `tile` (from the sequence's start) of KV
  // head h of sequence s; base < 0 marks an item with nothing to do (past the
  // last item, or the plan failed, whose fault bit is then set).
  struct Item {
    int s, h, tile, t0, t1, base, len_final;
  };
  auto item_of = [&](int item) -> Item {
    Item w;
    w.base = -1;
    w.s = w.h = w.tile = w.t0 = w.t1 = w.len_final = 0;
    if (item >= nitems) return w;
    int lo = 0, hi = a.num_seqs - 1;  // the sequence: last s with s_pref[s] <= item
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (s_pref[mid] <= item) lo = mid; else hi = mid - 1;
    }
    const int per_head = (s_pref[lo + 1] - s_pref[lo]) / L.Hkv;
    const int rem = item - s_pref[lo];
    w.s = lo;
    w.h = rem / per_head;
    w.tile = per_head - 1 - rem % per_head;
    w.t0 = a.cu[lo];
    w.t1 = a.cu[lo + 1];
    const int c = w.tile * TT / kPrefillChunk;
    const int cid = w.t0 / kPrefillChunk + c + a.seq_base + lo;
    w.base = L.plan[(size_t)w.h * L.plan_stride + cid];  // slots before the chunk
    w.len_final = L.lengths[((size_t)a.layer * 2 + parity) * L.NH + (a.first_seq + lo) * L.Hkv + w.h];
    return w;
  };
  // Q of an item (not committed: it forms a copy group with the item's staged
  // carried sums)
  auto issue_q = [&](const Item& w) {
    const int tok0 = w.t0 + w.tile * TT, tokN = min(tok0 + TT, w.t1);
    for (int i = tid; i < kPaRows * 16; i += kPaThreads) {
      const int rr = i >> 4, j = i & 15;
      const int tt = tok0 + rr / G;
      const bool ok = tt < tokN;
      const char* src = a.q + (((size_t)(ok ? tt : tok0) * L.Hq + (size_t)w.h * G + rr % G) * ROW) + j * 16;
      cp_async16_zfill(sQ + pa_swz(rr, j), src, ok);
    }
  };
  // K (which = 0) or V (which = 1) rows of slot tile jt, slots below hi;
  // page(p) gives the page id of the head's page p
  // Slot tile jt of a head into the K (which = 0) or V buffer, slots past hi
  // zero-filled; pg[q] is the page of the tile's slots [32 q, 32 q + 32). A
  // thread copies 16 bytes of rows tid / 16 + 16 k, k = 0..7, which lie in
  // page k / 2 of the tile (tid / 16 < 16), so the page ids are read by
  // compile-time index.
  static_assert(kPaThreads == 256 && kPaSlots == 4 * kPage, "row k of a thread lies in page k / 2");
  auto load_tile_pg = [&](const int* pg, int which, int jt, int hi) {
    // row r + 16 k: page k / 2, row r + 16 (k & 1) of it, at pa_swz(r, j) + 16 k
    // rows of 128 bytes in shared memory (r + 16 k and r have the same swizzle)
    const int r = tid >> 4, j = tid & 15;
    const uint32_t dst = smem_u32(smem + (which ? kPaV : kPaK)) + pa_swz(r, j);
    const size_t off = (size_t)r * ROW + (size_t)which * kPage * ROW + j * 16;
    const int lim = hi - jt * kPaSlots - r;  // row r + 16 k is a slot below hi iff 16 k < lim
    const char* pb[kPaSlots / kPage];
#pragma unroll
    for (int q = 0; q < kPaSlots / kPage; ++q) pb[q] = L.pages + (size_t)pg[q] * L.page_bytes + off;
#pragma unroll
    for (int k = 0; k < kPaSlots * 16 / kPaThreads; ++k) {
      const bool ok = 16 * k < lim;
      cp_async16_zfill(dst + k * 16 * 128, ok ? pb[k >> 1] + (k & 1) * 16 * ROW : L.pages, ok);
    }
  };
  // the page ids of slot tile jt of a head (those holding slots below hi)
  auto tile_pages = [&](const int* pt, int jt, int hi, int* pg) {
#pragma unroll
    for (int q = 0; q < kPaSlots / kPage; ++q) {
      const int p = jt * (kPaSlots / kPage) + q;
      pg[q] = p * kPage < hi ? pt[p] : 0;
    }
  };
  auto ptab_of = [&](const Item& w) {
    return L.page_table + ((size_t)a.layer * L.NH + (a.first_seq + w.s) * L.Hkv + w.h) * L.MPH;
  };
  // The first K/V tile, up to min(128, len_final) slots: every slot the head
  // holds has been written, and the staircase mask hides those a row does not
  // see. Copy groups, oldest first: Q (+ carry), K0, V0, then per
  // tile K(j + 1), V(j + 1).
  auto issue_kv0 = [&](const Item& w) {
    int pg[kPaSlots / kPage];
    tile_pages(ptab_of(w), 0, min(kPaSlots, w.len_final), pg);
    load_tile_pg(pg, 0, 0, min(kPaSlots, w.len_final));
    cp_async_commit();
    load_tile_pg(pg, 1, 0, min(kPaSlots, w.len_final));
    cp_async_commit();
  };
  // an item's carried sums, into copy `par` of the carry buffer (requested with
  // its Q, the two form one copy group)
  auto issue_carry = [&](const Item& w, int par) {
    const int cid = w.t0 / kPrefillChunk + w.tile * TT / kPrefillChunk + a.seq_base + w.s;
    const float* carry_g = a.carry + ((size_t)cid * L.Hkv + w.h) * (2 * D + 1);
    const uint32_t dc = smem_u32(smem + kPaCarry + par * kPaCarryBytes);
    for (int i = tid; i < 2 * D + 1; i += kPaThreads) pa_cp_async4(dc + 4 * i, carry_g + i);
  };
  // the per-token inputs of an item's chunk (its decision bytes and the
  // group's q[0]) for thread tid < 128, into registers
  int m_op = 0;
  uint32_t m_q0[(G + 1) / 2];
  auto load_meta = [&](const Item& w) {
    const int tok0 = w.t0 + w.tile * TT, tokN = min(tok0 + TT, w.t1);
    const int tau = w.t0 + (w.tile * TT / kPrefillChunk) * kPrefillChunk + tid;
    m_op = 0;
#pragma unroll
    for (int g = 0; g < (G + 1) / 2; ++g) m_q0[g] = 0u;
    if (tid < kPrefillChunk && tau < tokN) {
      m_op = L.opens[(size_t)tau * L.Hkv + w.h];
      const unsigned short* qs = reinterpret_cast<const unsigned short*>(qg) +
                                 ((size_t)tau * L.Hq + (size_t)w.h * G) * D;
#pragma unroll
      for (int g = 0; g < G; ++g) m_q0[g / 2] |= (uint32_t)qs[(size_t)g * D] << (16 * (g & 1));
    }
  };

  if (tid == 0) s_item[0] = atomicAdd(&ctr[0], 1);
  __syncthreads();
  int item = s_item[0];
  Item cur = item_of(item);
  if (cur.base >= 0) {
    issue_q(cur);
    issue_carry(cur, 0);
    cp_async_commit();
    issue_kv0(cur);
    load_meta(cur);
  }

  for (int it = 0;; ++it) {
    if (item >= nitems || *s_abort) break;
    if (tid == 0) s_item[(it + 1) & 1] = atomicAdd(&ctr[0], 1);  // read after the next barrier
    if (cur.base < 0) {
      // the plan failed for this item: nothing was requested for it
      __syncthreads();
      item = s_item[(it + 1) & 1];
      cur = item_of(item);
      if (cur.base >= 0) {
        issue_q(cur);
        issue_carry(cur, (it + 1) & 1);
        cp_async_commit();
        issue_kv0(cur);
        load_meta(cur);
      }
      continue;
    }
    const int s = cur.s, h = cur.h, t0 = cur.t0, t1 = cur.t1, base = cur.base, len_final = cur.len_final;
    const int bh = (a.first_seq + s) * L.Hkv + h;
    const int tok0 = t0 + cur.tile * TT;
    const int tokN = min(tok0 + TT, t1);
    const int c = (tok0 - t0) / kPrefillChunk;
    const int a0 = t0 + c * kPrefillChunk;  // the chunk holding the tile
    const int* ptab = L.page_table + ((size_t)a.layer * L.NH + bh) * L.MPH;
    // the chunk's carried sums came with this item's Q (copy groups, oldest
    // first: Q + carry, K0, V0; this
    // thread's copies of the first have landed here, and the first barrier
    // below makes all of them visible); the carry is kept by item parity,
    // since a thread may start this item while another still reads the
    // previous item's carry in its epilogue
    cp_async_wait<2>();
    const float* carry = reinterpret_cast<const float*>(smem + kPaCarry + (it & 1) * kPaCarryBytes);

    // ---- per-token decisions, omega, slot counts and 1 / z of the chunk up to
    // the tile end. z after token i is the omega sum of i's segment so far: from
    // the segment's opening token, or from the carried sums when no token of the
    // chunk up to i opens a slot (a segmented prefix sum over the chunk).
    int incl = 0, seg = 0, lastop = -1;
    float zs = 0.f;
    if (tid < kPrefillChunk) {
      const int tau = a0 + tid;
      const int op = m_op;  // requested with the item's Q
      float om = 0.f;
      if (tau < tokN) {
        float y = 0.f;
  #pragma unroll
        for (int g = 0; g < G; ++g)
          y += __uint_as_float(((m_q0[g / 2] >> (16 * (g & 1))) & 0xffffu) << 16);
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
    __syncthreads();
    const int item_next = s_item[(it + 1) & 1];
    const Item nxt = item_of(item_next);  // its loads are long done when its inputs are requested
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
  
  
    // Per slot tile j, with P kept in tensor memory so that the K buffer frees
    // as soon as S is computed:
    //   K(j) landed -> S = Q K^T -> K(j + 1) starts -> softmax, P (bf16) over
    //   this thread's own S columns -> V(j) landed -> O += P V -> V(j + 1) starts
    // The copy groups stay in step (one, possibly empty, per K and per V slot),
    // so "all but the newest group" always means the tile needed next.
    float m = -INFINITY, l = 0.f;  // l: this thread's half of the row sum
    for (int jt = 0; jt < ntiles; ++jt) {
      // the next tile's page ids, requested now so that its copies need not
      // wait for them
      int pgn[kPaSlots / kPage];
      tile_pages(ptab, jt + 1, jt + 1 < ntiles ? vis_hi : 0, pgn);
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
      wait_bar(0);  // S is in TMEM and the K buffer is free
      tc_fence_after();
      if (jt + 1 < ntiles) load_tile_pg(pgn, 0, jt + 1, vis_hi);
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
      wait_bar(1);
      tc_fence_after();
      if (jt + 1 < ntiles) load_tile_pg(pgn, 1, jt + 1, vis_hi);
      cp_async_commit();
    }
    cp_async_wait<0>();
    tc_fence_after();
    __syncthreads();  // every MMA and copy of the loop is over: the K and V buffers are free
    if (*s_abort) break;
  
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
    wait_bar(0);  // S_d is in TMEM
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
    if (*s_abort) break;
    if (nxt.base >= 0) {
      // S_d is done and every q . c_k read: the Q buffer is free, and the
      // other carry copy (the previous item's) is no longer read
      issue_q(nxt);
      issue_carry(nxt, (it + 1) & 1);
      cp_async_commit();
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
    wait_bar(1);
    tc_fence_after();
    if (nxt.base >= 0) {  // the last P V is done: the K and V buffers are free
      issue_kv0(nxt);
      load_meta(nxt);
    }
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
    tc_fence_before();  // this item's TMEM loads are done before the next item's MMAs
    item = item_next;
    cur = nxt;
  }
  cp_async_wait<0>();
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(256));
  }
  if (tid == 0) {  // the last CTA out resets the work counter for the next call
    __threadfence();
    if (atomicAdd(&ctr[1], 1) == (int)gridDim.x - 1) {
      ctr[0] = 0;
      ctr[1] = 0;
      __threadfence();
    }
  }
}

bool prefill_attn_supported(const Layout& L) {
  return L.esize == 2 && L.D == kPaD && (L.G == 1 || L.G == 2 || L.G == 4 || L.G == 8);
}

template <int G>
static cudaError_t launch_pa(PrefillAttnArgs a, cudaStream_t stream) {
  cudaError_t e = cudaFuncSetAttribute(dmc_prefill_attn_kernel<G>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, kPaSmem);

  int dev = 0, sms = 0;
  if (e == cudaSuccess) e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return e;
  constexpr int TT = kPaRows / G;
  const long long tiles = (a.max_seqlen + TT - 1) / TT;
  const int num_seqs = a.num_seqs, first_seq = a.first_seq;
  const int* cu = a.cu;
  // at most kPaMaxSeqs sequences per launch (the work-item table)
  for (int s0 = 0; s0 < num_seqs; s0 += kPaMaxSeqs) {
    a.seq_base = s0;
    a.num_seqs = min(kPaMaxSeqs, num_seqs - s0);
    a.first_seq = first_seq + s0;
    a.cu = cu + s0;
    const long long items = tiles * a.lay.Hkv * a.num_seqs;  // an upper bound
    if (items == 0) continue;
    // two CTAs per SM: their shared memory (2 x 111 KB) and TMEM (2 x 256
    // columns) fit; a CTA that found no SM slot would only start after the
    // others and find the work counter empty
    const long long resident = 2LL * sms;
    const int grid = (int)(items < resident ? items : resident);
    dmc_prefill_attn_kernel<G><<<grid, kPaThreads, kPaSmem, stream>>>(a);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
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
