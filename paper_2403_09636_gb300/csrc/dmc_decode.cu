// Fused DMC decode step: Algorithm 1 on the new token of every KV head plus
// single-query softmax attention over each head's updated, variable-length,
// paged cache (Eq. attn-softmax over the compressed slots, Sec. 3.1).
//
// Work split ("stream-K" over slot pages): every head h contributes
// ceil(len_old(h) / 32) page units plus one "owner" unit that holds the token
// being merged or appended. All units of a layer form one list; block b takes
// the contiguous range [b*U/nb, (b+1)*U/nb), so every block streams the same
// number of pages whatever the spread of head lengths. A head cut by a range
// boundary is finished by whichever of its blocks arrives last (a counter, no
// waiting): it merges the blocks' partial softmax states in a fixed order.
//
// Inside a block one producer warp walks the range and issues TMA bulk copies
// (cp.async.bulk) of each page's K rows and V rows into a ring of shared
// memory stages; 8 consumer warps read them. A 32-slot page maps one slot row
// onto each 8-lane group; a lane holds 16 bytes of the row per 128-byte chunk.
// The slot that Algorithm 1 changes (the merged last slot, or the new one) is
// never read from the page: the owner unit computes it in registers from the
// old row, z and the new k, v, stores it rounded to the cache dtype, and
// scores that rounded value, so every block of the layer reads only slots this
// launch does not write.
//
// Slot counts are double-buffered per layer: this launch reads buffer `parity`
// and writes the other; the last block to finish flips the parity. That keeps
// the unit list consistent while owners publish new lengths, and stays correct
// when the launch is replayed from a CUDA graph.
#include <math.h>

#include <mutex>

#include "dmc_internal.cuh"

namespace dmc {

constexpr int kConsumerWarps = 8;
constexpr int kConsumers = kConsumerWarps * 32;
constexpr int kDecodeThreads = kConsumers + 32;
constexpr int kStages = 4;
constexpr int kMaxDecodeBlocks = 1024;

enum : int { kFlagAcc = 1, kFlagNaN = 2 };

struct StageHdr {
  int len_old;
  int rows;      // fixed slot rows in this stage
  int flags;     // kFlagAcc: owner unit merges into the last slot
  int tgt_page;  // owner: page of the slot being written, -1 = allocate one
  float omega;
  int pad[11];
};
static_assert(sizeof(StageHdr) == 64, "header is 64 bytes");

struct DecodeArgs {
  Layout lay;
  int layer;
  int Gv;  // virtual heads per KV head: 1, or G when each query head of a group runs alone
  const char* q;
  const char* k;
  const char* v;
  char* out;
};

template <typename T, int D>
struct DecodeGeom {
  static constexpr int ROW = D * (int)sizeof(T);
  static constexpr int NCH = ROW / 128;      // 16-byte chunks per lane of an 8-lane group
  static constexpr int EPC = Chunk<T>::N;    // elements per chunk
  static constexpr int EPL = NCH * EPC;      // elements of a row held by one lane
  static constexpr int OFF_Q = 64;
  static constexpr int OFF_KIN = OFF_Q + ROW;
  static constexpr int OFF_VIN = OFF_KIN + ROW;
  static constexpr int OFF_KOLD = OFF_VIN + ROW;
  static constexpr int OFF_VOLD = OFF_KOLD + ROW;
  static constexpr int OFF_Z = OFF_VOLD + ROW;
  static constexpr int OFF_K = ((OFF_Z + kPage * 4) + 127) / 128 * 128;
  static constexpr int OFF_V = OFF_K + kPage * ROW;
  static constexpr int STAGE = OFF_V + kPage * ROW;
  static constexpr int RING = kStages * STAGE;
  static constexpr int OFF_BARS = RING;                       // full[S], empty[S]
  static constexpr int OFF_RED = OFF_BARS + 2 * kStages * 8;  // [warps][D + 2] floats
  static constexpr int OFF_MISC = OFF_RED + kConsumerWarps * (D + 2) * 4;  // 16 ints
  static constexpr int OFF_U = OFF_MISC + 64;                 // [NVH + 1] ints
  static size_t smem_bytes(int nvh) { return (size_t)OFF_U + (size_t)(nvh + 1) * 4; }
};

// Block b owns units [range_start(b), range_start(b + 1)); when there are more
// blocks than units some ranges are empty.
__device__ __forceinline__ long long range_start(int b, long long U, int nb) {
  return (long long)b * U / nb;
}

// Index of the (non-empty) block whose unit range holds unit u.
__device__ __forceinline__ int block_of_unit(long long u, long long U, int nb) {
  return (int)(((u + 1) * nb - 1) / U);
}

// Exclusive prefix of units per virtual head into U[0..nvh], all threads.
__device__ void scan_units(int* U, int* wsum, const int* len_cur, int nvh, int Gv) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int nthr = blockDim.x, nwarps = nthr >> 5;
  const int per = (nvh + nthr - 1) / nthr;
  const int i0 = min(tid * per, nvh), i1 = min(i0 + per, nvh);
  int local = 0;
  for (int i = i0; i < i1; ++i) local += ceil_div(len_cur[i / Gv], kPage) + 1;
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
    U[i] = run;
    run += ceil_div(len_cur[i / Gv], kPage) + 1;
  }
  if (tid == 0) U[nvh] = wsum[nwarps];
  __syncthreads();
}

template <typename T, int D>
__device__ __forceinline__ void merge_state(float& m, float& l, float* acc, float m2, float l2,
                                            const float* acc2) {
  constexpr int EPL = DecodeGeom<T, D>::EPL;
  const float mn = fmaxf(m, m2);
  const float c1 = (m == -INFINITY) ? 0.f : exp2f(m - mn);
  const float c2 = (m2 == -INFINITY) ? 0.f : exp2f(m2 - mn);
  l = l * c1 + l2 * c2;
#pragma unroll
  for (int i = 0; i < EPL; ++i) acc[i] = acc[i] * c1 + acc2[i] * c2;
  m = mn;
}

template <typename T, int D>
__global__ void __launch_bounds__(kDecodeThreads, 2)
dmc_decode_kernel(const DecodeArgs a) {
  using G_ = DecodeGeom<T, D>;
  using CK = Chunk<T>;
  constexpr int ROW = G_::ROW, NCH = G_::NCH, EPC = G_::EPC, EPL = G_::EPL;
  extern __shared__ __align__(128) unsigned char smem[];

  const Layout& L = a.lay;
  const int Gv = a.Gv;
  const int NVH = L.NH * Gv;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int nb = gridDim.x, bid = blockIdx.x;
  int* ctl = L.ctl + a.layer * 4;
  const int parity = *reinterpret_cast<volatile int*>(&ctl[0]);
  const int* len_cur = L.lengths + ((size_t)a.layer * 2 + parity) * L.NH;
  int* len_nxt = L.lengths + ((size_t)a.layer * 2 + (parity ^ 1)) * L.NH;
  int* ptab = L.page_table + (size_t)a.layer * L.NH * L.MPH;

  const uint32_t bars = smem_u32(smem + G_::OFF_BARS);
  auto full_bar = [&](int s) { return bars + 8u * s; };
  auto empty_bar = [&](int s) { return bars + 8u * (kStages + s); };
  float* red = reinterpret_cast<float*>(smem + G_::OFF_RED);
  volatile int* misc = reinterpret_cast<volatile int*>(smem + G_::OFF_MISC);
  int* U = reinterpret_cast<int*>(smem + G_::OFF_U);

  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), kConsumerWarps);
    }
    fence_mbar_init();
    misc[0] = 0;  // abort
    misc[1] = 0;  // combine
  }
  scan_units(U, reinterpret_cast<int*>(smem + G_::OFF_MISC) + 4, len_cur, NVH, Gv);

  const long long Utot = U[NVH];
  const int u0 = (int)((long long)bid * Utot / nb);
  const int u1 = (int)((long long)(bid + 1) * Utot / nb);

  if (u0 < u1 && warp == kConsumerWarps) {
    // ------------------------------------------------------------ producer warp
    int vh = 0;
    {  // largest vh with U[vh] <= u0
      int lo = 0, hi = NVH - 1;
      while (lo < hi) {
        int mid = (lo + hi + 1) >> 1;
        if (U[mid] <= u0) lo = mid; else hi = mid - 1;
      }
      vh = lo;
    }
    int bh = 0, len_old = 0, acc = 0, lfixed = 0, win_base = -1, win = 0;
    float omega = 0.f;
    bool nan_gate = false;
    const int* pt_row = ptab;
    int it = 0;
    for (int u = u0; u < u1; ++u, ++it) {
      while (U[vh + 1] <= u) ++vh;
      const int hu0 = U[vh], nU = U[vh + 1] - hu0, j = u - hu0;
      const bool first = (u == u0) || (j == 0);
      if (first) {
        bh = vh / Gv;
        const int b = bh / L.Hkv, h = bh % L.Hkv;
        len_old = len_cur[bh];
        const float x = Elt<T>::to_f(reinterpret_cast<const T*>(a.k)[(size_t)bh * D]);
        nan_gate = (x != x);
        acc = (x >= 0.f && len_old > 0) ? 1 : 0;  // alpha = round(sigmoid(k[0])) = [k[0] >= 0]
        lfixed = len_old - acc;                     // slots no unit of this launch writes
        float q0 = 0.f;
        if (lane < L.G)
          q0 = Elt<T>::to_f(
              reinterpret_cast<const T*>(a.q)[((size_t)b * L.Hq + (size_t)h * L.G + lane) * D]);
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) q0 += __shfl_xor_sync(0xffffffffu, q0, off);
        omega = sigmoidf_(q0 / (float)L.G);  // omega = sigmoid(mean of the group's q[0])
        pt_row = ptab + (size_t)bh * L.MPH;
        win_base = -1;
      }
      const bool owner = (j == nU - 1);
      const int rows = owner ? 0 : max(0, min(kPage, lfixed - j * kPage));
      int page = 0;
      if (rows > 0) {
        const int wb = j >> 5;
        if (wb != win_base) {
          const int idx = wb * 32 + lane;
          win = idx < L.MPH ? pt_row[idx] : 0;
          win_base = wb;
        }
        page = __shfl_sync(0xffffffffu, win, j & 31);
      }
      int old_page = -1, tgt = -1;
      if (owner) {
        if (acc) {
          old_page = pt_row[(len_old - 1) / kPage];
          tgt = old_page;
        } else if (len_old % kPage != 0) {
          tgt = pt_row[len_old / kPage];
        }
      }
      const int st = it % kStages;
      const uint32_t ph = (uint32_t)(it / kStages) & 1u;
      if (lane == 0) {
        bool ok = misc[0] == 0 && mbar_wait(empty_bar(st), ph ^ 1u, L.error);
        if (!ok) {
          misc[0] = 1;
        } else {
          unsigned char* stage = smem + (size_t)st * G_::STAGE;
          StageHdr* hdr = reinterpret_cast<StageHdr*>(stage);
          hdr->len_old = len_old;
          hdr->rows = rows;
          hdr->flags = (owner && acc ? kFlagAcc : 0) | (nan_gate ? kFlagNaN : 0);
          hdr->tgt_page = tgt;
          hdr->omega = omega;
          uint32_t bytes = 0;
          if (first) bytes += ROW;
          if (rows) bytes += 2u * rows * ROW;
          if (owner) bytes += 2u * ROW + (acc ? 2u * ROW + kPage * 4u : 0u);
          const uint32_t fb = full_bar(st);
          if (bytes == 0) {
            mbar_arrive(fb);
          } else {
            mbar_arrive_expect_tx(fb, bytes);
            const uint32_t sbase = smem_u32(stage);
            if (first) {
              const int b = bh / L.Hkv, h = bh % L.Hkv, g = vh % Gv;
              bulk_g2s(sbase + G_::OFF_Q,
                       a.q + ((size_t)b * L.Hq + (size_t)h * L.G + g) * ROW, ROW, fb);
            }
            if (rows) {
              const char* pg = L.pages + (size_t)page * L.page_bytes;
              bulk_g2s(sbase + G_::OFF_K, pg, rows * ROW, fb);
              bulk_g2s(sbase + G_::OFF_V, pg + kPage * ROW, rows * ROW, fb);
            }
            if (owner) {
              bulk_g2s(sbase + G_::OFF_KIN, a.k + (size_t)bh * ROW, ROW, fb);
              bulk_g2s(sbase + G_::OFF_VIN, a.v + (size_t)bh * ROW, ROW, fb);
              if (acc) {
                const int r = (len_old - 1) % kPage;
                const char* pg = L.pages + (size_t)old_page * L.page_bytes;
                bulk_g2s(sbase + G_::OFF_KOLD, pg + (size_t)r * ROW, ROW, fb);
                bulk_g2s(sbase + G_::OFF_VOLD, pg + (size_t)(kPage + r) * ROW, ROW, fb);
                bulk_g2s(sbase + G_::OFF_Z, L.z + (size_t)old_page * kPage, kPage * 4, fb);
              }
            }
          }
        }
      }
      __syncwarp();
      if (misc[0]) break;
    }
    if (lane == 0 && misc[0]) {
      // Aborted: let every copy already issued land before the block exits.
      for (int k = max(0, it - kStages); k < it; ++k)
        mbar_wait(full_bar(k % kStages), (uint32_t)(k / kStages) & 1u, L.error);
    }
  } else if (u0 < u1) {
    // ------------------------------------------------------------ consumer warps
    const int grp = warp * 4 + (lane >> 3);  // slot row of a page handled by this 8-lane group
    const int l8 = lane & 7;
    const float qscale = 1.4426950408889634f / sqrtf((float)D);  // log2(e) / sqrt(d_h)
    float qf[EPL];
    float m = -INFINITY, lsum = 0.f, acc[EPL];
#pragma unroll
    for (int i = 0; i < EPL; ++i) { acc[i] = 0.f; qf[i] = 0.f; }
    int vh = 0;
    {
      int lo = 0, hi = NVH - 1;
      while (lo < hi) {
        int mid = (lo + hi + 1) >> 1;
        if (U[mid] <= u0) lo = mid; else hi = mid - 1;
      }
      vh = lo;
    }
    int it = 0;
    for (int u = u0; u < u1; ++u, ++it) {
      while (U[vh + 1] <= u) ++vh;
      const int hu0 = U[vh], nU = U[vh + 1] - hu0, j = u - hu0;
      const bool first = (u == u0) || (j == 0);
      const bool owner = (j == nU - 1);
      const bool seg_end = owner || (u == u1 - 1);
      const int st = it % kStages;
      const uint32_t ph = (uint32_t)(it / kStages) & 1u;
      const unsigned char* stage = smem + (size_t)st * G_::STAGE;
      bool have = misc[0] == 0 && mbar_wait(full_bar(st), ph, L.error);
      if (!have) misc[0] = 1;
      have = __shfl_sync(0xffffffffu, have ? 1 : 0, 0) != 0;
      if (have) {
        const StageHdr hdr = *reinterpret_cast<const StageHdr*>(stage);
        if (first) {
#pragma unroll
          for (int c = 0; c < NCH; ++c) {
            float f[EPC];
            CK::unpack(*reinterpret_cast<const uint4*>(stage + G_::OFF_Q + c * 128 + l8 * 16), f);
#pragma unroll
            for (int e = 0; e < EPC; ++e) qf[c * EPC + e] = f[e] * qscale;
          }
          if (l8 == 0) qf[0] = 0.f;  // q[0] is the importance gate, not a feature
        }
        {
          // Every lane scores a row (rows past hdr.rows hold stale data and
          // are discarded) so the shuffles run with the whole warp.
          const bool active = grp < hdr.rows;
          const unsigned char* krow = stage + G_::OFF_K + grp * ROW;
          const unsigned char* vrow = stage + G_::OFF_V + grp * ROW;
          float s = 0.f;
#pragma unroll
          for (int c = 0; c < NCH; ++c) {
            float f[EPC];
            CK::unpack(*reinterpret_cast<const uint4*>(krow + c * 128 + l8 * 16), f);
#pragma unroll
            for (int e = 0; e < EPC; ++e) s = fmaf(qf[c * EPC + e], f[e], s);
          }
          s += __shfl_xor_sync(0xffffffffu, s, 1);
          s += __shfl_xor_sync(0xffffffffu, s, 2);
          s += __shfl_xor_sync(0xffffffffu, s, 4);
          if (active) {
            const float mn = fmaxf(m, s);
            const float corr = exp2f(m - mn);
            const float p = exp2f(s - mn);
            lsum = fmaf(lsum, corr, p);
#pragma unroll
            for (int c = 0; c < NCH; ++c) {
              float f[EPC];
              CK::unpack(*reinterpret_cast<const uint4*>(vrow + c * 128 + l8 * 16), f);
#pragma unroll
              for (int e = 0; e < EPC; ++e)
                acc[c * EPC + e] = fmaf(acc[c * EPC + e], corr, p * f[e]);
            }
            m = mn;
          }
        }
        if (owner && warp == 0 && lane < 8) {
          // Algorithm 1 on the new token, in fp32, result rounded to the cache dtype.
          const int bh = vh / Gv;
          const bool accumulate = (hdr.flags & kFlagAcc) != 0;
          const float w = hdr.omega;
          const int len_old = hdr.len_old;
          float zold = 0.f, znew = w;
          if (accumulate) {
            zold = reinterpret_cast<const float*>(stage + G_::OFF_Z)[(len_old - 1) % kPage];
            znew = zold + w;
          }
          uint4 nk[NCH], nv[NCH];
          float kr[EPL], vr[EPL];
#pragma unroll
          for (int c = 0; c < NCH; ++c) {
            float kin[EPC], vin[EPC];
            CK::unpack(*reinterpret_cast<const uint4*>(stage + G_::OFF_KIN + c * 128 + l8 * 16), kin);
            CK::unpack(*reinterpret_cast<const uint4*>(stage + G_::OFF_VIN + c * 128 + l8 * 16), vin);
            if (c == 0 && l8 == 0) kin[0] = 0.f;  // k[0] <- 0 (Algorithm 1)
            float kn[EPC], vn[EPC];
            if (accumulate) {
              float ko[EPC], vo[EPC];
              CK::unpack(*reinterpret_cast<const uint4*>(stage + G_::OFF_KOLD + c * 128 + l8 * 16), ko);
              CK::unpack(*reinterpret_cast<const uint4*>(stage + G_::OFF_VOLD + c * 128 + l8 * 16), vo);
#pragma unroll
              for (int e = 0; e < EPC; ++e) {
                kn[e] = (ko[e] * zold + kin[e] * w) / znew;
                vn[e] = (vo[e] * zold + vin[e] * w) / znew;
              }
            } else {
#pragma unroll
              for (int e = 0; e < EPC; ++e) { kn[e] = kin[e]; vn[e] = vin[e]; }
            }
            nk[c] = CK::pack(kn);
            nv[c] = CK::pack(vn);
            CK::unpack(nk[c], kr + c * EPC);  // the stored (rounded) values
            CK::unpack(nv[c], vr + c * EPC);
          }
          if (vh % Gv == 0) {  // one writer per KV head
            const int slot = accumulate ? len_old - 1 : len_old;
            bool ok = slot < L.max_slots;
            if (!ok && l8 == 0) atomicOr(L.error, DMC_FAULT_SLOT_CAPACITY);
            int page = hdr.tgt_page;
            if (ok && page < 0) {
              if (l8 == 0) {
                const unsigned long long id = atomicAdd(L.pool_top, 1ull);
                if (id >= (unsigned long long)L.num_pages) {
                  atomicOr(L.error, DMC_FAULT_PAGES_EXHAUSTED);
                  page = -1;
                } else {
                  page = (int)id;
                  ptab[(size_t)bh * L.MPH + slot / kPage] = page;
                }
              }
              page = __shfl_sync(0xffu, page, 0, 8);
            }
            ok = ok && page >= 0;
            if (ok) {
              char* dst = L.pages + (size_t)page * L.page_bytes + (size_t)(slot % kPage) * ROW;
#pragma unroll
              for (int c = 0; c < NCH; ++c) {
                *reinterpret_cast<uint4*>(dst + c * 128 + l8 * 16) = nk[c];
                *reinterpret_cast<uint4*>(dst + (size_t)kPage * ROW + c * 128 + l8 * 16) = nv[c];
              }
            }
            if (l8 == 0) {
              if (ok) L.z[(size_t)page * kPage + slot % kPage] = znew;
              len_nxt[bh] = ok ? slot + 1 : len_old;
              if (hdr.flags & kFlagNaN) atomicOr(L.error, DMC_FAULT_NAN_GATE);
            }
          }
          float s = 0.f;
#pragma unroll
          for (int i = 0; i < EPL; ++i) s = fmaf(qf[i], kr[i], s);
          s += __shfl_xor_sync(0xffu, s, 1);
          s += __shfl_xor_sync(0xffu, s, 2);
          s += __shfl_xor_sync(0xffu, s, 4);
          const float mn = fmaxf(m, s);
          const float corr = exp2f(m - mn);
          const float p = exp2f(s - mn);
          lsum = fmaf(lsum, corr, p);
#pragma unroll
          for (int i = 0; i < EPL; ++i) acc[i] = fmaf(acc[i], corr, p * vr[i]);
          m = mn;
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(empty_bar(st));

      if (seg_end) {
        // ---- merge the 32 groups' softmax states, then emit or hand off
#pragma unroll
        for (int off = 8; off < 32; off <<= 1) {
          const float m2 = __shfl_xor_sync(0xffffffffu, m, off);
          const float l2 = __shfl_xor_sync(0xffffffffu, lsum, off);
          float a2[EPL];
#pragma unroll
          for (int i = 0; i < EPL; ++i) a2[i] = __shfl_xor_sync(0xffffffffu, acc[i], off);
          merge_state<T, D>(m, lsum, acc, m2, l2, a2);
        }
        float* rw = red + warp * (D + 2);
        if (lane == 0) { rw[0] = m; rw[1] = lsum; }
        if (lane < 8) {
#pragma unroll
          for (int c = 0; c < NCH; ++c)
#pragma unroll
            for (int e = 0; e < EPC; ++e)
              rw[2 + (c * 128 + l8 * 16) / (int)sizeof(T) + e] = acc[c * EPC + e];
        }
        named_sync(1, kConsumers);
        // block-level state for dimension tid (tid < D)
        float M = -INFINITY;
#pragma unroll
        for (int w = 0; w < kConsumerWarps; ++w) M = fmaxf(M, red[w * (D + 2)]);
        float Ls = 0.f, O = 0.f;
#pragma unroll
        for (int w = 0; w < kConsumerWarps; ++w) {
          const float mw = red[w * (D + 2)];
          const float cw = (mw == -INFINITY) ? 0.f : exp2f(mw - M);
          Ls = fmaf(red[w * (D + 2) + 1], cw, Ls);
          if (tid < D) O = fmaf(red[w * (D + 2) + 2 + tid], cw, O);
        }
        const int bh = vh / Gv, g = vh % Gv;
        const int b = bh / L.Hkv, h = bh % L.Hkv;
        const size_t orow = ((size_t)b * L.Hq + (size_t)h * L.G + g) * D;
        const bool whole = (hu0 >= u0) && owner;
        if (whole) {
          if (tid < D) reinterpret_cast<T*>(a.out)[orow + tid] = Elt<T>::from_f(O / Ls);
        } else {
          const int slot = 2 * bid + (hu0 <= u0 ? 0 : 1);
          float* pp = L.partials + (size_t)slot * (D + 2);
          if (tid == 0) { pp[0] = M; pp[1] = Ls; }
          if (tid < D) pp[2 + tid] = O;
          __threadfence();
          named_sync(1, kConsumers);
          const long long hend = U[vh + 1];
          const int bf = block_of_unit(hu0, Utot, nb);
          const int bl = block_of_unit(hend - 1, Utot, nb);
          if (tid == 0) {
            // contributors: the blocks of [bf, bl] with a non-empty unit range
            int ncontrib = 0;
            for (int cb = bf; cb <= bl; ++cb)
              ncontrib += range_start(cb, Utot, nb) < range_start(cb + 1, Utot, nb);
            int* cnt = L.counters + (size_t)a.layer * L.NH * L.G + vh;
            const int old = atomicAdd(cnt, 1);
            const int last = (old == ncontrib - 1);
            if (last) *cnt = 0;
            misc[1] = last;
          }
          named_sync(1, kConsumers);
          if (misc[1]) {
            __threadfence();
            float Mc = -INFINITY;
            for (int cb = bf; cb <= bl; ++cb) {
              const long long cstart = range_start(cb, Utot, nb);
              if (cstart == range_start(cb + 1, Utot, nb)) continue;
              const int cs = 2 * cb + (hu0 <= cstart ? 0 : 1);
              Mc = fmaxf(Mc, __ldcg(L.partials + (size_t)cs * (D + 2)));
            }
            float Lc = 0.f, Oc = 0.f;
            for (int cb = bf; cb <= bl; ++cb) {
              const long long cstart = range_start(cb, Utot, nb);
              if (cstart == range_start(cb + 1, Utot, nb)) continue;
              const int cs = 2 * cb + (hu0 <= cstart ? 0 : 1);
              const float* cp = L.partials + (size_t)cs * (D + 2);
              const float mc = __ldcg(cp);
              const float cw = (mc == -INFINITY) ? 0.f : exp2f(mc - Mc);
              Lc = fmaf(__ldcg(cp + 1), cw, Lc);
              if (tid < D) Oc = fmaf(__ldcg(cp + 2 + tid), cw, Oc);
            }
            if (tid < D) reinterpret_cast<T*>(a.out)[orow + tid] = Elt<T>::from_f(Oc / Lc);
          }
        }
        named_sync(1, kConsumers);  // `red` and misc[1] are reused by the next head
        m = -INFINITY;
        lsum = 0.f;
#pragma unroll
        for (int i = 0; i < EPL; ++i) acc[i] = 0.f;
      }
    }
  }

  __syncthreads();
  if (tid == 0) {
    __threadfence();
    const int old = atomicAdd(&ctl[1], 1);
    if (old == nb - 1) {  // last block of the launch: publish the new slot counts
      ctl[1] = 0;
      ctl[0] = parity ^ 1;
      __threadfence();
    }
  }
}

template <typename T, int D>
static cudaError_t setup_decode(int nvh, int* grid, size_t* smem) {
  using G_ = DecodeGeom<T, D>;
  *smem = G_::smem_bytes(nvh);
  cudaError_t e = cudaFuncSetAttribute(dmc_decode_kernel<T, D>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)*smem);
  if (e != cudaSuccess) return e;
  int occ = 0, dev = 0, sms = 0;
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, dmc_decode_kernel<T, D>,
                                                    kDecodeThreads, *smem);
  if (e != cudaSuccess) return e;
  if (occ < 1) return cudaErrorInvalidConfiguration;
  e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return e;
  *grid = min(sms * occ, kMaxDecodeBlocks);
  return cudaSuccess;
}

cudaError_t decode_setup(const Layout& L, int Gv, int* grid, size_t* smem) {
  const int nvh = L.NH * Gv;
  cudaError_t e = cudaErrorInvalidValue;
  if (L.esize == 4 && L.D == 64) e = setup_decode<float, 64>(nvh, grid, smem);
  if (L.esize == 4 && L.D == 128) e = setup_decode<float, 128>(nvh, grid, smem);
  if (L.esize == 2 && L.D == 64) e = setup_decode<__nv_bfloat16, 64>(nvh, grid, smem);
  if (L.esize == 2 && L.D == 128) e = setup_decode<__nv_bfloat16, 128>(nvh, grid, smem);
  // no more blocks than the most units a layer can have
  const long long max_units = (long long)nvh * (L.MPH + 1);
  if (e == cudaSuccess && max_units < *grid) *grid = (int)max_units;
  return e;
}

cudaError_t decode_launch(const Layout& L, int layer, int Gv, int grid, size_t smem,
                          const void* q, const void* k, const void* v, void* out,
                          cudaStream_t stream) {
  DecodeArgs a;
  a.lay = L;
  a.layer = layer;
  a.Gv = Gv;
  a.q = static_cast<const char*>(q);
  a.k = static_cast<const char*>(k);
  a.v = static_cast<const char*>(v);
  a.out = static_cast<char*>(out);
  if (L.esize == 4 && L.D == 64)
    dmc_decode_kernel<float, 64><<<grid, kDecodeThreads, smem, stream>>>(a);
  else if (L.esize == 4 && L.D == 128)
    dmc_decode_kernel<float, 128><<<grid, kDecodeThreads, smem, stream>>>(a);
  else if (L.esize == 2 && L.D == 64)
    dmc_decode_kernel<__nv_bfloat16, 64><<<grid, kDecodeThreads, smem, stream>>>(a);
  else if (L.esize == 2 && L.D == 128)
    dmc_decode_kernel<__nv_bfloat16, 128><<<grid, kDecodeThreads, smem, stream>>>(a);
  else
    return cudaErrorInvalidValue;
  return cudaGetLastError();
}

// ---------------------------------------------------------------- static scratch
// Scratch of dmc_decode_step_static_scratch: room for the split-K partial
// softmax states of one launch (2 per block, head_dim <= 128, grid <= 1024
// blocks), 1.04 MB. Every GPU that loads the library holds it until exit.
constexpr size_t kStaticPartialFloats = (size_t)2 * kMaxDecodeBlocks * (128 + 2);
static __device__ __align__(256) float g_decode_static_partials[kStaticPartialFloats];

// Host code must not pass g_decode_static_partials itself to a kernel (on the
// host it only names a stand-in). This looks up its device address once per
// device, with that device current, and remembers it.
cudaError_t decode_static_partials(int device, float** ptr, size_t* floats) {
  constexpr int kMaxDevices = 64;
  static std::mutex mu;
  static float* addr[kMaxDevices] = {};
  if (device < 0 || device >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(mu);
  if (addr[device] == nullptr) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_decode_static_partials);
    if (e != cudaSuccess) return e;
    addr[device] = static_cast<float*>(p);
  }
  *ptr = addr[device];
  *floats = kStaticPartialFloats;
  return cudaSuccess;
}

}  // namespace dmc
