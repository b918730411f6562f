// Prompt-phase DMC compression (Algorithm 1 over a prompt, without attention).
//
// With binary alpha, Eq. partial-accumulation makes every slot the
// omega-weighted mean of one segment of consecutive tokens: a segment opens at
// a token with alpha = 0 (k[0] < 0) or at the first token of an empty head, and
// runs up to the next opening token; z of the slot is the segment's summed
// omega. Two kernels, no host synchronisation:
//
//  plan: one block per (sequence, KV head). Reads k[t, h, 0] of the prompt,
//        records which tokens open a slot (one byte per token and head), counts
//        openings per 128-token chunk, takes pages for the head's new slots from
//        the pool (one atomic per head), and stores each chunk's first slot index.
//  scan: one block per (128-token chunk, KV head, sequence). The block owns the
//        segments that open inside its chunk (and chunk 0 also owns the tokens
//        that continue the head's existing last slot); a segment that runs past
//        the chunk end is followed to its end. Lanes split a row into 16-byte
//        pieces and accumulate sum(omega k), sum(omega v), sum(omega) in fp32;
//        the slot is the quotient, rounded once to the cache dtype. Exact
//        compression walks the chunk's tokens in row groups (see the kernel);
//        window grouping gives each segment to one warp. When asked for
//        (prompt attention), the block also records, at every chunk start a
//        segment runs across, the segment's sums up to that point (the
//        "carry"), so that each chunk can rebuild the running state of its
//        tokens without reading back to the segment's start.
//  ring: window grouping only, after the scan: stores each head's open
//        segment's last W - 1 tokens and its length.
#include "dmc_internal.cuh"

namespace dmc {

constexpr int kPlanThreads = 256;
constexpr int kScanThreads = 128;

struct PrefillArgs {
  Layout lay;
  int layer, first_seq, num_seqs;
  const char* q;
  long long q_tok, q_head;  // element strides of the queries' first components
  const char* k;
  const char* v;
  const int* cu;
  int total_tokens, max_seqlen;
  float* carry;  // [chunk id][Hkv][2D + 1] (sum w k, sum w v, sum w), or null
};

__device__ __forceinline__ bool seq_bounds(const PrefillArgs& a, int s, int& t0, int& t1) {
  t0 = a.cu[s];
  t1 = a.cu[s + 1];
  return t0 >= 0 && t0 <= t1 && t1 <= a.total_tokens && (t1 - t0) <= a.max_seqlen;
}

__device__ __forceinline__ int chunk_id(int t0, int c, int s) { return (t0 + c * kPrefillChunk) / kPrefillChunk + s; }

template <typename T, int D>
__global__ void __launch_bounds__(kPlanThreads) dmc_prefill_plan_kernel(const PrefillArgs a) {
  extern __shared__ int cnt[];  // [ceil(max_seqlen / 128)]
  __shared__ int s_fail, s_first_page, s_nan, s_wsum[kPlanThreads / 32 + 1];
  const Layout& L = a.lay;
  const int s = blockIdx.x, h = blockIdx.y;
  const int bh = (a.first_seq + s) * L.Hkv + h;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  griddep_launch_dependents();  // the scan may start its copies of k and v
  const int parity = *reinterpret_cast<volatile int*>(&L.ctl[a.layer * 4]);
  int* len = L.lengths + ((size_t)a.layer * 2 + parity) * L.NH;
  int t0, t1;
  if (!seq_bounds(a, s, t0, t1)) {
    if (tid == 0) atomicOr(L.error, DMC_FAULT_BAD_SEQLENS);
    return;
  }
  const int ntok = t1 - t0;
  const int nch = ceil_div(ntok, kPrefillChunk);
  const int len_old = len[bh];
  for (int c = tid; c < nch; c += kPlanThreads) cnt[c] = 0;
  if (tid == 0) { s_fail = 0; s_nan = 0; }
  __syncthreads();
  const T* kk = reinterpret_cast<const T*>(a.k);
  for (int base = 0; base < ntok; base += kPlanThreads) {
    const int i = base + tid;
    bool opens = false;
    if (i < ntok) {
      const size_t t = (size_t)(t0 + i);
      const float x = Elt<T>::to_f(kk[(t * L.Hkv + h) * D]);
      if (x != x) s_nan = 1;
      // alpha = round(sigmoid(k[0])) = [k[0] >= 0]; alpha = 0 opens a slot,
      // and so does the first token of an empty head.
      opens = !(x >= 0.f) || (i == 0 && len_old == 0);
      L.opens[t * L.Hkv + h] = opens ? 1 : 0;
    }
    const unsigned bal = __ballot_sync(0xffffffffu, opens);
    if (lane == 0 && base + warp * 32 < ntok) atomicAdd(&cnt[(base + warp * 32) / kPrefillChunk], __popc(bal));
  }
  __syncthreads();
  // exclusive scan of the chunk counts (nch <= max_seqlen / 128 + 1)
  const int per = ceil_div(nch, kPlanThreads);
  const int c0 = min(tid * per, nch), c1 = min(c0 + per, nch);
  int local = 0;
  for (int c = c0; c < c1; ++c) local += cnt[c];
  int incl = local;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int o = __shfl_up_sync(0xffffffffu, incl, off);
    if (lane >= off) incl += o;
  }
  if (lane == 31) s_wsum[warp] = incl;
  __syncthreads();
  if (tid == 0) {
    int run = 0;
    for (int w = 0; w < kPlanThreads / 32; ++w) { const int t = s_wsum[w]; s_wsum[w] = run; run += t; }
    s_wsum[kPlanThreads / 32] = run;
  }
  __syncthreads();
  const int new_slots = s_wsum[kPlanThreads / 32];
  const int len_new = len_old + new_slots;
  const int old_pages = ceil_div(len_old, kPage), new_pages = ceil_div(len_new, kPage);
  const int need = new_pages - old_pages;
  if (tid == 0) {
    int fail = 0, first = 0;
    if (len_new > L.max_slots) {
      atomicOr(L.error, DMC_FAULT_SLOT_CAPACITY);
      fail = 1;
    } else if (need > 0) {
      const unsigned long long f = atomicAdd(L.pool_top, (unsigned long long)need);
      if (f + (unsigned long long)need > (unsigned long long)L.num_pages) {
        atomicOr(L.error, DMC_FAULT_PAGES_EXHAUSTED);
        fail = 1;
      } else {
        first = (int)f;
      }
    }
    if (s_nan) atomicOr(L.error, DMC_FAULT_NAN_GATE);
    s_fail = fail;
    s_first_page = first;
  }
  __syncthreads();
  const int fail = s_fail;
  int run = s_wsum[warp] + incl - local;
  for (int c = c0; c < c1; ++c) {
    L.plan[(size_t)h * L.plan_stride + chunk_id(t0, c, s)] = fail ? -1 : len_old + run;
    run += cnt[c];
  }
  if (!fail) {
    int* pt = L.page_table + ((size_t)a.layer * L.NH + bh) * L.MPH;
    for (int i = tid; i < need; i += kPlanThreads) pt[old_pages + i] = s_first_page + i;
    if (tid == 0) len[bh] = len_new;
  }
}

// Carry slot of the chunk of sequence s that starts at token cs (t0 = the
// sequence's first token).
__device__ __forceinline__ float* carry_at(const PrefillArgs& a, int t0, int cs, int s, int h, int D) {
  return a.carry + ((size_t)chunk_id(t0, (cs - t0) / kPrefillChunk, s) * a.lay.Hkv + h) * (2 * D + 1);
}

// Window grouping: one warp sums segment [tb, te) into `slot`, counting only
// its last W tokens; the head's open segment keeps its last W - 1 tokens in
// the ring (token p of the segment at entry p % W) and its length in seglen,
// and a prompt that continues it (merge_old) takes the continued segment's
// tokens still inside the window from there.
template <typename T, int D>
__device__ __noinline__ void scan_window_segment(const PrefillArgs& a, int h, int bh, int tb,
                                                 int te, int slot, bool merge_old) {
  using CK = Chunk<T>;
  constexpr int ROW = D * (int)sizeof(T);
  constexpr int LPR = ROW / 16;  // lanes per row
  constexpr int RPI = 32 / LPR;  // rows per warp iteration
  constexpr int EPC = CK::N;
  const Layout& L = a.lay;
  const int lane = threadIdx.x & 31, sub = lane / LPR, lr = lane % LPR;
  const T* qq = reinterpret_cast<const T*>(a.q);
  float ak[EPC], av[EPC], zs = 0.f;
#pragma unroll
  for (int e = 0; e < EPC; ++e) { ak[e] = 0.f; av[e] = 0.f; }
  const int page = L.page_table[((size_t)a.layer * L.NH + bh) * L.MPH + slot / kPage];
  char* kdst = L.pages + (size_t)page * L.page_bytes + (size_t)(slot % kPage) * ROW + lr * 16;
  char* vdst = kdst + (size_t)kPage * ROW;
  float* zp = L.z + (size_t)page * kPage + slot % kPage;
  const int W = L.window;
  const int parity = *reinterpret_cast<const volatile int*>(&L.ctl[a.layer * 4]);
  const char* ring = L.ring + ((size_t)a.layer * L.NH + bh) * W * 2 * ROW;
  const float* ring_w = L.ring_w + ((size_t)a.layer * L.NH + bh) * W;
  if (merge_old && sub == 0) {
    // the continued segment's tokens still inside the window, from the ring
    const int n_old = L.seglen[((size_t)a.layer * 2 + parity) * L.NH + bh];
    const int m = min(n_old, max(0, W - (te - tb)));
    for (int e = 0; e < m; ++e) {
      const int pos = (n_old - 1 - e) % W;
      float ko[EPC], vo[EPC];
      CK::unpack(*reinterpret_cast<const uint4*>(ring + (size_t)pos * 2 * ROW + lr * 16), ko);
      CK::unpack(*reinterpret_cast<const uint4*>(ring + (size_t)pos * 2 * ROW + ROW + lr * 16), vo);
      const float w = ring_w[pos];
#pragma unroll
      for (int e2 = 0; e2 < EPC; ++e2) {
        ak[e2] = fmaf(w, ko[e2], ak[e2]);
        av[e2] = fmaf(w, vo[e2], av[e2]);
      }
      if (lr == 0) zs += w;
    }
  }
  const size_t hrow = (size_t)L.Hkv * ROW;
  const char* kb = a.k + (size_t)h * ROW + lr * 16;
  const char* vb = a.v + (size_t)h * ROW + lr * 16;
#pragma unroll 2
  for (int t = max(tb, te - W) + sub; t < te; t += RPI) {  // the segment's last W tokens
    const uint4 kr = __ldg(reinterpret_cast<const uint4*>(kb + (size_t)t * hrow));
    const uint4 vr = __ldg(reinterpret_cast<const uint4*>(vb + (size_t)t * hrow));
    float y = 0.f;
    for (int g = 0; g < L.G; ++g)
      y += Elt<T>::to_f(qq[(size_t)t * a.q_tok + (size_t)(h * L.G + g) * a.q_head]);
    const float w = sigmoidf_(y / (float)L.G);  // omega = sigmoid(q[0]) (group mean for GQA)
    float kf[EPC], vf[EPC];
    CK::unpack(kr, kf);
    CK::unpack(vr, vf);
    if (lr == 0) kf[0] = 0.f;  // k[0] <- 0 (Algorithm 1)
#pragma unroll
    for (int e = 0; e < EPC; ++e) {
      ak[e] = fmaf(w, kf[e], ak[e]);
      av[e] = fmaf(w, vf[e], av[e]);
    }
    zs += w;
  }
#pragma unroll
  for (int off = LPR; off < 32; off <<= 1) {
#pragma unroll
    for (int e = 0; e < EPC; ++e) {
      ak[e] += __shfl_xor_sync(0xffffffffu, ak[e], off);
      av[e] += __shfl_xor_sync(0xffffffffu, av[e], off);
    }
    zs += __shfl_xor_sync(0xffffffffu, zs, off);
  }
  // the lr == 0 lane holds z; every lane needs it for the quotient
  zs = __shfl_sync(0xffffffffu, zs, lane - lr);
  if (sub != 0) return;
  const float iz = 1.f / zs;
  float kn[EPC], vn[EPC];
#pragma unroll
  for (int e = 0; e < EPC; ++e) {
    kn[e] = ak[e] * iz;
    vn[e] = av[e] * iz;
  }
  if (lr == 0) kn[0] = 0.f;
  *reinterpret_cast<uint4*>(kdst) = CK::pack(kn);
  *reinterpret_cast<uint4*>(vdst) = CK::pack(vn);
  if (lr == 0) *zp = zs;
}

// Window grouping: the head's open segment [tb, te = end of the prompt), which
// had n_old tokens before this prompt, leaves its last W - 1 tokens (k with
// k[0] cleared, v, omega) in the ring and its length in seglen. One warp.
template <typename T, int D>
__device__ __forceinline__ void fill_ring(const PrefillArgs& a, int h, int bh, int tb, int te,
                                          int n_old) {
  constexpr int ROW = D * (int)sizeof(T);
  constexpr int LPR = ROW / 16;
  constexpr int RPI = 32 / LPR;
  const Layout& L = a.lay;
  const int W = L.window;
  const int lane = threadIdx.x & 31, sub = lane / LPR, lr = lane % LPR;
  const int parity = *reinterpret_cast<const volatile int*>(&L.ctl[a.layer * 4]);
  char* ring = L.ring + ((size_t)a.layer * L.NH + bh) * W * 2 * ROW;
  float* ring_w = L.ring_w + ((size_t)a.layer * L.NH + bh) * W;
  const T* qq = reinterpret_cast<const T*>(a.q);
  const size_t hrow = (size_t)L.Hkv * ROW;
  for (int t = max(tb, te - (W - 1)) + sub; t < te; t += RPI) {
    const int pos = (n_old + t - tb) % W;
    uint4 kr = __ldg(reinterpret_cast<const uint4*>(a.k + (size_t)t * hrow + (size_t)h * ROW + lr * 16));
    const uint4 vr = __ldg(reinterpret_cast<const uint4*>(a.v + (size_t)t * hrow + (size_t)h * ROW + lr * 16));
    if (lr == 0) {
      // k[0] <- 0: the first element of this lane's piece
      if (sizeof(T) == 2) kr.x &= 0xffff0000u;
      else kr.x = 0u;
    }
    *reinterpret_cast<uint4*>(ring + (size_t)pos * 2 * ROW + lr * 16) = kr;
    *reinterpret_cast<uint4*>(ring + (size_t)pos * 2 * ROW + ROW + lr * 16) = vr;
    if (lr == 0) {
      float y = 0.f;
      for (int g = 0; g < L.G; ++g)
        y += Elt<T>::to_f(qq[(size_t)t * a.q_tok + (size_t)(h * L.G + g) * a.q_head]);
      ring_w[pos] = sigmoidf_(y / (float)L.G);
    }
  }
  if (lane == 0) L.seglen[((size_t)a.layer * 2 + parity) * L.NH + bh] = n_old + (te - tb);
}

// Exact compression (no window). The chunk's tokens are split evenly among
// row groups of LPR lanes (a lane holds one 16-byte piece of a row); each group
// walks its tokens in order and closes a slot at every opening token. A lane
// streams its pieces of the group's rows through a private ring in shared
// memory (16-byte async copies, kRing rows ahead, issued before anything else
// the block needs), so the copies overlap the block's setup and the walk. What
// a group sums before its first opening is handed, through shared memory, to
// the group that holds the open segment before it. The chunk's last segment is
// followed past the chunk end up to the next opening token (recording the carry
// at each chunk start it runs across), and chunk 0 also finishes the segment
// that continues the head's existing last slot.
constexpr int kRing = 8;        // rows in a lane's ring
constexpr int kRingBatch = 4;   // rows per async-copy group
constexpr size_t kScanRingBytes = (size_t)kRing * 2 * kScanThreads * 16;

template <typename T, int D>
__global__ void __launch_bounds__(kScanThreads, 6) dmc_prefill_scan_kernel(const PrefillArgs a) {
  using CK = Chunk<T>;
  constexpr int ROW = D * (int)sizeof(T);
  constexpr int LPR = ROW / 16;               // lanes per row
  constexpr int NG = kScanThreads / LPR;      // row groups
  constexpr int TPG = kPrefillChunk / NG;     // tokens per group
  constexpr int NB = (TPG + kRingBatch - 1) / kRingBatch;
  constexpr int EPC = CK::N;
  constexpr int kMaxPages = kPrefillChunk / kPage + 2;
  constexpr int HS = 2 * D + 1;               // floats of one group's head sums
  static_assert(kScanThreads == kPrefillChunk, "one thread per chunk token");
  static_assert(TPG <= 32 && 32 % TPG == 0, "a group's tokens sit in one ballot word");
  static_assert(kRing == 2 * kRingBatch, "two copy groups in flight");
  static_assert((size_t)NG * HS * sizeof(float) <= kScanRingBytes, "heads fit the ring");
  __shared__ __align__(16) unsigned char ring[kScanRingBytes];  // [kRing][K, V][thread] 16 B
  __shared__ float s_w[kPrefillChunk];
  __shared__ unsigned s_bal[kPrefillChunk / 32], s_nbal[kPrefillChunk / 32];
  __shared__ int s_page[kMaxPages];
  __shared__ int s_next;
  const Layout& L = a.lay;
  const int c = blockIdx.x, h = blockIdx.y, s = blockIdx.z;
  const int bh = (a.first_seq + s) * L.Hkv + h;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int g = tid / LPR, lr = tid % LPR;
  int t0, t1;
  // every block waits for the plan before it ends, so that the scan never
  // completes ahead of the plan it was launched after
  if (!seq_bounds(a, s, t0, t1) || t0 + c * kPrefillChunk >= t1) {
    griddep_wait();
    return;
  }
  const int a0 = t0 + c * kPrefillChunk;
  const int a1 = min(a0 + kPrefillChunk, t1);
  const int g0 = a0 + g * TPG, g1 = min(g0 + TPG, a1);  // the group's tokens
  const size_t hrow = (size_t)L.Hkv * ROW;
  const char* kb = a.k + (size_t)h * ROW + lr * 16;
  const char* vb = a.v + (size_t)h * ROW + lr * 16;
  const uint32_t rbase = smem_u32(ring) + tid * 16;
  auto rk = [&](int pos) { return rbase + (uint32_t)(pos * 2) * kScanThreads * 16; };
  auto issue = [&](int b) {  // copy group b: the group's rows g0 + 4b ... (always committed)
#pragma unroll
    for (int u = 0; u < kRingBatch; ++u) {
      const int t = g0 + b * kRingBatch + u;
      if (b < NB && t < g1) {
        const uint32_t dk = rk((b % 2) * kRingBatch + u);
        cp_async16(dk, kb + (size_t)t * hrow);
        cp_async16(dk + kScanThreads * 16, vb + (size_t)t * hrow);
      }
    }
    cp_async_commit();
  };
  issue(0);
  issue(1);
  // launched as a programmatic dependent of the plan: what follows reads its
  // outputs (the copies above read only the prompt)
  griddep_wait();

  const int base = L.plan[(size_t)h * L.plan_stride + chunk_id(t0, c, s)];
  const unsigned char* op = L.opens + h;
  const size_t ostride = (size_t)L.Hkv;
  const T* qq = reinterpret_cast<const T*>(a.q);
  auto omega = [&](int t) {  // omega = sigmoid(q[0]) (group mean for GQA)
    float y = 0.f;
    for (int gq = 0; gq < L.G; ++gq)
      y += Elt<T>::to_f(qq[(size_t)t * a.q_tok + (size_t)(h * L.G + gq) * a.q_head]);
    return sigmoidf_(y / (float)L.G);
  };
  // pages of the slots the block may write, [base - 1, base + 128): at most
  // kMaxPages entries, all inside the head's row since the plan fitted the slots
  const int pfirst = max(base - 1, 0) / kPage;
  if (base >= 0 && tid < kMaxPages && pfirst + tid < L.MPH)
    s_page[tid] = L.page_table[((size_t)a.layer * L.NH + bh) * L.MPH + pfirst + tid];
  // one thread per token: does it open a slot, and its omega; the same for the
  // next 128 tokens' openings (the first of them ends the chunk's last segment)
  {
    const int t = a0 + tid, tn = a1 + tid;
    const bool f = t < a1 && op[(size_t)t * ostride];
    const bool fn = tn < t1 && op[(size_t)tn * ostride];
    s_w[tid] = t < a1 ? omega(t) : 0.f;
    const unsigned bal = __ballot_sync(0xffffffffu, f), nbal = __ballot_sync(0xffffffffu, fn);
    if (lane == 0) { s_bal[warp] = bal; s_nbal[warp] = nbal; }
  }
  __syncthreads();
  int nstart = 0, first = -1, next = -1;
#pragma unroll
  for (int w = 0; w < kPrefillChunk / 32; ++w) {
    const unsigned b = s_bal[w], nb = s_nbal[w];
    if (first < 0 && b) first = w * 32 + __ffs(b) - 1;
    if (next < 0 && nb) next = a1 + w * 32 + __ffs(nb) - 1;
    nstart += __popc(b);
  }
  const bool pre = (c == 0) && !(s_bal[0] & 1u);  // continues the existing last slot
  if (base < 0 || (nstart == 0 && !pre)) {
    // the plan failed, or every token belongs to an earlier chunk's segment
    cp_async_wait<0>();
    return;
  }
  if (next < 0) {  // no opening in the next 128 tokens: search on (uniform)
    if (tid == 0) s_next = t1;
    __syncthreads();
    for (int b0 = a1 + kPrefillChunk; b0 < t1; b0 += kScanThreads) {
      const int tt = b0 + tid;
      const bool gq = tt < t1 && op[(size_t)tt * ostride];
      if (gq) atomicMin(&s_next, tt);
      if (__syncthreads_or(gq)) break;
    }
    next = s_next;
  }

  float ak[EPC], av[EPC], zs = 0.f;
  auto reset = [&]() {
#pragma unroll
    for (int e = 0; e < EPC; ++e) { ak[e] = 0.f; av[e] = 0.f; }
    zs = 0.f;
  };
  auto add_row = [&](const uint4& kr, const uint4& vr, float w) {
    float kf[EPC], vf[EPC];
    CK::unpack(kr, kf);
    CK::unpack(vr, vf);
    if (lr == 0) kf[0] = 0.f;  // k[0] <- 0 (Algorithm 1)
#pragma unroll
    for (int e = 0; e < EPC; ++e) {
      ak[e] = fmaf(w, kf[e], ak[e]);
      av[e] = fmaf(w, vf[e], av[e]);
    }
    zs += w;
  };
  auto slot_ptr = [&](int slot) {
    const int page = s_page[slot / kPage - pfirst];
    return L.pages + (size_t)page * L.page_bytes + (size_t)(slot % kPage) * ROW + lr * 16;
  };
  auto write_slot = [&](int slot) {  // the slot = the segment's omega-weighted mean
    char* kdst = slot_ptr(slot);
    const float iz = 1.f / zs;
    float kn[EPC], vn[EPC];
#pragma unroll
    for (int e = 0; e < EPC; ++e) {
      kn[e] = ak[e] * iz;
      vn[e] = av[e] * iz;
    }
    if (lr == 0) kn[0] = 0.f;
    *reinterpret_cast<uint4*>(kdst) = CK::pack(kn);
    *reinterpret_cast<uint4*>(kdst + (size_t)kPage * ROW) = CK::pack(vn);
    if (lr == 0) L.z[(size_t)s_page[slot / kPage - pfirst] * kPage + slot % kPage] = zs;
  };
  auto group_bits = [&](int gg) {  // the opening tokens of group gg's range
    const unsigned b = s_bal[(gg * TPG) >> 5] >> ((gg * TPG) & 31);
    return TPG == 32 ? b : (b & ((1u << TPG) - 1u));
  };

  // walk: tokens [max(g0, wb), g1), wb = the first token the block owns (the
  // token loop stays rolled: one copy of the slot write keeps the code small)
  const int wb = pre ? a0 : a0 + first;
  const unsigned gbits = group_bits(g);
  int slot = base - 1;  // the slot of the segment being summed
  {
    const int wi = (g * TPG) >> 5;
    for (int w = 0; w < wi; ++w) slot += __popc(s_bal[w]);
    slot += __popc(s_bal[wi] & ((1u << ((g * TPG) & 31)) - 1u));
  }
  float hk[EPC], hv[EPC], hz = 0.f;  // the sums before the group's first opening
  bool open = false;                 // summing a segment that opened in this group
  reset();
  for (int b = 0; b < NB; ++b) {
    cp_async_wait<1>();  // copy group b has landed
#pragma unroll 1
    for (int u = 0; u < kRingBatch; ++u) {
      const int t = g0 + b * kRingBatch + u;
      if (t >= wb && t < g1) {
        if ((gbits >> (t - g0)) & 1u) {  // t opens a slot: the segment before it ends
          if (open) {
            write_slot(slot);
          } else {
#pragma unroll
            for (int e = 0; e < EPC; ++e) { hk[e] = ak[e]; hv[e] = av[e]; }
            hz = zs;
          }
          reset();
          open = true;
          ++slot;
        }
        const uint32_t sk = rk((b % 2) * kRingBatch + u);
        uint4 kr, vr;
        asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
                     : "=r"(kr.x), "=r"(kr.y), "=r"(kr.z), "=r"(kr.w) : "r"(sk) : "memory");
        asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
                     : "=r"(vr.x), "=r"(vr.y), "=r"(vr.z), "=r"(vr.w)
                     : "r"(sk + kScanThreads * 16) : "memory");
        add_row(kr, vr, s_w[t - a0]);
      }
    }
    issue(b + 2);  // into the ring rows just read
  }
  if (!open) {  // no opening in the range: all of it joins an earlier segment
#pragma unroll
    for (int e = 0; e < EPC; ++e) { hk[e] = ak[e]; hv[e] = av[e]; }
    hz = zs;
  }
  // the heads replace the ring (every copy has landed: the last groups are empty)
  cp_async_wait<0>();
  __syncthreads();
  float* heads = reinterpret_cast<float*>(ring);
#pragma unroll
  for (int e = 0; e < EPC; ++e) {
    heads[g * HS + lr * EPC + e] = hk[e];
    heads[g * HS + D + lr * EPC + e] = hv[e];
  }
  if (lr == 0) heads[g * HS + 2 * D] = hz;
  __syncthreads();

  const bool carry = a.carry != nullptr;
  auto put_carry = [&](int cs) {  // the sums so far, as the carry of the chunk at cs
    float* cp = carry_at(a, t0, cs, s, h, D);
#pragma unroll
    for (int e = 0; e < EPC; ++e) {
      cp[lr * EPC + e] = ak[e];
      cp[D + lr * EPC + e] = av[e];
    }
    if (lr == 0) cp[2 * D] = zs;
  };
  // adds the heads of the groups after gg up to the first with an opening; if
  // none has one, the segment is the chunk's last and runs on to `next`
  auto finish = [&](int gg) {
    for (++gg; gg < NG; ++gg) {
      const float* hp = heads + gg * HS;
#pragma unroll
      for (int e = 0; e < EPC; ++e) {
        ak[e] += hp[lr * EPC + e];
        av[e] += hp[D + lr * EPC + e];
      }
      zs += hp[2 * D];
      if (group_bits(gg)) return;
    }
    for (int pb = a1; pb < next; pb += kPrefillChunk) {
      if (carry) put_carry(pb);  // the segment runs across the chunk starting at pb
      const int pe = min(next, pb + kPrefillChunk);
      for (int tb = pb; tb < pe; tb += 2) {
        uint4 kr[2], vr[2];
        float w[2];
#pragma unroll
        for (int u = 0; u < 2; ++u) {
          if (tb + u < pe) {
            kr[u] = __ldg(reinterpret_cast<const uint4*>(kb + (size_t)(tb + u) * hrow));
            vr[u] = __ldg(reinterpret_cast<const uint4*>(vb + (size_t)(tb + u) * hrow));
            w[u] = omega(tb + u);
          }
        }
#pragma unroll
        for (int u = 0; u < 2; ++u)
          if (tb + u < pe) add_row(kr[u], vr[u], w[u]);
      }
    }
  };
  // job 0: the group's open segment (its sums are in the registers); job 1
  // (group 0 of chunk 0 only): the segment that continues the head's last slot
  const int jobs_end = (pre && g == 0) ? 2 : 1;
  for (int job = open ? 0 : 1; job < jobs_end; ++job) {
    int from = g;
    if (job == 1) {
      // the old slot's K z_old, V z_old and z_old start the sums
      slot = base - 1;
      from = -1;
      const char* kold = slot_ptr(slot);
      float ko[EPC], vo[EPC];
      CK::unpack(*reinterpret_cast<const uint4*>(kold), ko);
      CK::unpack(*reinterpret_cast<const uint4*>(kold + (size_t)kPage * ROW), vo);
      const float zo = L.z[(size_t)s_page[slot / kPage - pfirst] * kPage + slot % kPage];
#pragma unroll
      for (int e = 0; e < EPC; ++e) {
        ak[e] = ko[e] * zo;
        av[e] = vo[e] * zo;
      }
      zs = zo;
      if (carry) put_carry(t0);  // the state the prompt's first token continues
    }
    finish(from);
    write_slot(slot);
  }
}

// Window grouping: one warp per segment (the slot counts only the segment's
// last W tokens, and a continued segment's old tokens come from the ring).
template <typename T, int D>
__global__ void __launch_bounds__(kScanThreads) dmc_prefill_scan_window_kernel(const PrefillArgs a) {
  __shared__ int starts[kPrefillChunk];
  __shared__ int s_wcnt[kScanThreads / 32];
  __shared__ int s_next;
  const Layout& L = a.lay;
  const int c = blockIdx.x, h = blockIdx.y, s = blockIdx.z;
  const int bh = (a.first_seq + s) * L.Hkv + h;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  int t0, t1;
  if (!seq_bounds(a, s, t0, t1)) return;
  const int a0 = t0 + c * kPrefillChunk;
  if (a0 >= t1) return;
  const int a1 = min(a0 + kPrefillChunk, t1);
  const int base = L.plan[(size_t)h * L.plan_stride + chunk_id(t0, c, s)];
  if (base < 0) return;
  const unsigned char* op = L.opens + h;
  const size_t ostride = (size_t)L.Hkv;

  // positions of the tokens of [a0, a1) that open a slot, in order
  static_assert(kScanThreads == kPrefillChunk, "one thread per chunk token");
  const int t = a0 + tid;
  const bool f = (t < a1) && op[(size_t)t * ostride];
  const unsigned bal = __ballot_sync(0xffffffffu, f);
  if (lane == 0) s_wcnt[warp] = __popc(bal);
  if (tid == 0) s_next = t1;
  __syncthreads();
  int before = __popc(bal & ((1u << lane) - 1u));
  for (int w = 0; w < warp; ++w) before += s_wcnt[w];
  int nstart = 0;
  for (int w = 0; w < kScanThreads / 32; ++w) nstart += s_wcnt[w];
  if (f) starts[before] = t;
  // the first opening token at or after a1 ends the chunk's last segment
  for (int b0 = a1; b0 < t1; b0 += kScanThreads) {
    const int tt = b0 + tid;
    const bool g = tt < t1 && op[(size_t)tt * ostride];
    if (g) atomicMin(&s_next, tt);
    if (__syncthreads_or(g)) break;
  }
  __syncthreads();
  const int next = s_next;
  const bool pre = (c == 0) && !op[(size_t)t0 * ostride];  // continues the existing last slot
  const int items = nstart + (pre ? 1 : 0);
  for (int it = warp; it < items; it += kScanThreads / 32) {
    if (pre && it == 0) {
      const int te = nstart > 0 ? starts[0] : next;
      scan_window_segment<T, D>(a, h, bh, t0, te, base - 1, true);
    } else {
      const int j = it - (pre ? 1 : 0);
      const int tb = starts[j];
      const int te = (j + 1 < nstart) ? starts[j + 1] : next;
      scan_window_segment<T, D>(a, h, bh, tb, te, base + j, false);
    }
  }
}

// Window grouping: after the scan (which read the old window of continued
// segments), one block per (sequence, KV head) finds the head's open segment
// (from the prompt's last opening token, or the whole prompt if it continued
// the old one) and stores its last W - 1 tokens and its length.
template <typename T, int D>
__global__ void __launch_bounds__(kPlanThreads) dmc_prefill_ring_kernel(const PrefillArgs a) {
  __shared__ int s_last;
  const Layout& L = a.lay;
  const int s = blockIdx.x, h = blockIdx.y;
  const int bh = (a.first_seq + s) * L.Hkv + h;
  const int tid = threadIdx.x;
  int t0, t1;
  if (!seq_bounds(a, s, t0, t1) || t1 == t0) return;
  if (L.plan[(size_t)h * L.plan_stride + chunk_id(t0, 0, s)] < 0) return;  // the plan failed
  if (tid == 0) s_last = -1;
  __syncthreads();
  for (int b = t1 - kPlanThreads; b + kPlanThreads > t0; b -= kPlanThreads) {
    const int t = b + tid;
    if (t >= t0 && L.opens[(size_t)t * L.Hkv + h]) atomicMax(&s_last, t);
    if (__syncthreads_or(s_last >= 0)) break;
  }
  const int last = s_last;
  if (tid >= 32) return;
  const int parity = *reinterpret_cast<const volatile int*>(&L.ctl[a.layer * 4]);
  const int n_old = last >= 0 ? 0 : L.seglen[((size_t)a.layer * 2 + parity) * L.NH + bh];
  fill_ring<T, D>(a, h, bh, last >= 0 ? last : t0, t1, n_old);
}

template <typename T, int D>
static cudaError_t launch_prefill(const PrefillArgs& a, cudaStream_t stream) {
  const int max_chunks = ceil_div(a.max_seqlen, kPrefillChunk);
  const size_t plan_smem = (size_t)max(max_chunks, 1) * sizeof(int);
  if (plan_smem > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(dmc_prefill_plan_kernel<T, D>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)plan_smem);
    if (e != cudaSuccess) return e;
  }
  dmc_prefill_plan_kernel<T, D><<<dim3(a.num_seqs, a.lay.Hkv), kPlanThreads, plan_smem, stream>>>(a);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  if (max_chunks > 0) {
    const dim3 grid(max_chunks, a.lay.Hkv, a.num_seqs);
    if (a.lay.window > 0) {
      dmc_prefill_scan_window_kernel<T, D><<<grid, kScanThreads, 0, stream>>>(a);
    } else {
      cudaLaunchConfig_t cfg = {};
      cfg.gridDim = grid;
      cfg.blockDim = dim3(kScanThreads);
      cfg.stream = stream;
      cudaLaunchAttribute attr[1];
      attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
      attr[0].val.programmaticStreamSerializationAllowed = 1;
      cfg.attrs = attr;
      cfg.numAttrs = 1;
      e = cudaLaunchKernelEx(&cfg, dmc_prefill_scan_kernel<T, D>, a);
      if (e != cudaSuccess) return e;
    }
    e = cudaGetLastError();
  }
  if (e == cudaSuccess && a.lay.window > 0) {
    dmc_prefill_ring_kernel<T, D><<<dim3(a.num_seqs, a.lay.Hkv), kPlanThreads, 0, stream>>>(a);
    e = cudaGetLastError();
  }
  return e;
}

cudaError_t prefill_launch(const Layout& L, int layer, int first_seq, int num_seqs, const void* q,
                           long long q_tok, long long q_head, const void* k, const void* v,
                           const int* cu, int total_tokens, int max_seqlen, float* carry,
                           cudaStream_t stream) {
  PrefillArgs a;
  a.lay = L;
  a.layer = layer;
  a.first_seq = first_seq;
  a.num_seqs = num_seqs;
  a.q = static_cast<const char*>(q);
  a.q_tok = q_tok;
  a.q_head = q_head;
  a.k = static_cast<const char*>(k);
  a.v = static_cast<const char*>(v);
  a.cu = cu;
  a.total_tokens = total_tokens;
  a.max_seqlen = max_seqlen;
  a.carry = carry;
  if (L.esize == 4 && L.D == 64) return launch_prefill<float, 64>(a, stream);
  if (L.esize == 4 && L.D == 128) return launch_prefill<float, 128>(a, stream);
  if (L.esize == 2 && L.D == 64) return launch_prefill<__nv_bfloat16, 64>(a, stream);
  if (L.esize == 2 && L.D == 128) return launch_prefill<__nv_bfloat16, 128>(a, stream);
  return cudaErrorInvalidValue;
}

}  // namespace dmc
