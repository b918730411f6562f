// DMC decode step for grouped-query attention on tensor cores (bf16).
//
// The paper combines DMC with the 8x grouped-query attention of Llama 2 70B
// (one decision and one compressed cache per KV head, shared by the G query
// heads of its group). Here one warp handles all G <= 8 queries of a KV head,
// so every slot page is read once for the whole group and the scores and the
// value sums become small matrix products on the tensor cores
// (mma.sync m16n8k16, bf16 in, fp32 accumulate):
//
//   S  = Q K^T     M = 16 query rows (the G queries, the rest zero),
//                  N = 8 slots, K = 16 dims;
//   O^T += V^T P^T M = 16 dims, N = 8 queries, K = 16 slots.
//
// The score fragment (row = query, cols = 2 slots) is exactly the B operand
// layout of the second product, so P never leaves registers and the output
// accumulator O^T has no padded rows. K and V move in tiles of 16 slots (half
// a page): each lane cp.asyncs 16-byte chunks into a per-warp ring in shared
// memory, chunks XOR-swizzled by row so that ldmatrix (and ldmatrix.trans for
// V) reads without bank conflicts; rows past the head's length are
// zero-filled. The softmax is online in the log2 domain, per query row.
//
// Work split, owner update, split-head combine, double-buffered slot counts,
// programmatic dependent launch and the walk over several layers in one launch
// follow the MHA kernel (dmc_decode.cu): units are a head's pages plus one
// owner unit, split evenly over all warps; the owner applies Algorithm 1 once
// per KV head, and the new row enters the attention as a one-row tile; a head
// cut between warps is merged by the last warp to finish it, in worker order.
#include <math.h>

#include "dmc_internal.cuh"
#include "dmc_split.cuh"

namespace dmc {

constexpr int kGWarps = kGqaWarpsPerBlock;  // workers per block
constexpr int kGThreads = kGWarps * 32;
constexpr int kGRing = 4;     // tiles per warp ring (kGRing - 1 in flight)
constexpr int kTile = 16;     // slots per tile
constexpr int kGWindow = 64;  // page units per warp window
constexpr int kGMaxBlocks = 256;
constexpr int kGMaxQueries = 8;
constexpr int kGHeadWindow = 32;  // KV heads whose gates a warp holds in its lanes
static_assert(kGMaxBlocks * kGWarps * 2 <= kGqaWorkerStates, "partials hold two states per worker");

enum : int { kGFlagAcc = 1, kGFlagNaN = 2 };

struct GqaArgs {
  Layout lay;
  int layer0, nlayers;  // layers [layer0, layer0 + nlayers), walked in order
  const char* q;        // layer layer0 + i at q + i * q_ls bytes: [B][Hq][D]
  const char* k;        // at k + i * kv_ls: [B][Hkv][D]
  const char* v;
  char* out;            // at out + i * q_ls: [B][Hq][D]
  long long q_ls, kv_ls;
};

template <int D>
struct GqaGeom {
  static constexpr int ROW = D * 2;               // bf16 row bytes
  static constexpr int CPR = ROW / 16;            // 16-byte chunks per row
  static constexpr int KT = D / 16;               // k-steps of S = m-tiles of O^T
  static constexpr int TILE = 2 * kTile * ROW;    // 16 K rows then 16 V rows
  static constexpr int WRING = kGRing * TILE;
  static constexpr int WWIN = 2 * kGWindow * 4;   // page ids, rows to copy
  static constexpr int WARP_BYTES = WRING + WWIN;
  static constexpr int MISC = 64;
  // two unit prefixes (by layer parity)
  static size_t smem_bytes(int nh) {
    return (size_t)kGWarps * WARP_BYTES + MISC + (size_t)2 * (nh + 1) * 4;
  }
};

// Byte offset of 16-byte chunk c of a row inside a 16-row block; the chunk
// index is XOR-ed with the row so that 8 consecutive rows hit 8 bank groups.
__device__ __forceinline__ uint32_t swz(int row, int c, int row_bytes) {
  return (uint32_t)(row * row_bytes + ((c ^ (row & 7)) << 4));
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&h);
}

// kWin: the cache uses the window-grouping approximation (L.window > 0)
template <int D, bool kWin>
__global__ void __launch_bounds__(kGThreads, 1) dmc_decode_gqa_kernel(const GqaArgs a) {
  using G_ = GqaGeom<D>;
  constexpr int ROW = G_::ROW, CPR = G_::CPR, KT = G_::KT;
  using CK = Chunk<__nv_bfloat16>;
  extern __shared__ __align__(128) unsigned char smem[];

  const Layout& L = a.lay;
  const int G = L.G;
  const int NH = L.NH;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, t = lane & 3;  // mma fragment row / column pair
  unsigned char* ring = smem + (size_t)warp * G_::WARP_BYTES;
  int* wpid = reinterpret_cast<int*>(ring + G_::WRING);
  int* wrws = wpid + kGWindow;
  int* misc = reinterpret_cast<int*>(smem + (size_t)kGWarps * G_::WARP_BYTES);
  int* Ubuf = misc + G_::MISC / 4;  // the unit prefixes of layers li (buffer li & 1)
  volatile int* s_done = misc + 8;  // [2]: warps of the block done with the layer in buffer b
  volatile int* s_tag = misc + 10;  // [2]: 1 + the index li of the layer whose prefix buffer b holds

  // Walking several layers, a warp goes on to the next layer as soon as its own
  // part of the current one is done: the block builds the first two layers'
  // unit prefixes here, and the last of its warps to leave layer li builds
  // layer li + 2's into the buffer it frees.
  scan_units(Ubuf, misc, L.ctl + a.layer0 * 4, L.lengths + (size_t)a.layer0 * 2 * NH, NH, NH, 1);
  if (a.nlayers > 1)
    scan_units(Ubuf + NH + 1, misc, L.ctl + (a.layer0 + 1) * 4,
               L.lengths + (size_t)(a.layer0 + 1) * 2 * NH, NH, NH, 1);
  if (tid == 0) {
    s_done[0] = s_done[1] = 0;
    s_tag[0] = 1;
    s_tag[1] = 2;
  }
  __syncthreads();

  for (int li = 0; li < a.nlayers; ++li) {
  const int layer = a.layer0 + li;
  const char* qL = a.q + (size_t)li * a.q_ls;
  const char* kL = a.k + (size_t)li * a.kv_ls;
  const char* vL = a.v + (size_t)li * a.kv_ls;
  char* outL = a.out + (size_t)li * a.q_ls;
  int* ctl = L.ctl + layer * 4;
  const int parity = *reinterpret_cast<volatile int*>(&ctl[0]);
  const int* len_cur = L.lengths + ((size_t)layer * 2 + parity) * NH;
  int* len_nxt = L.lengths + ((size_t)layer * 2 + (parity ^ 1)) * NH;
  int* ptab = L.page_table + (size_t)layer * NH * L.MPH;
  float* partials = L.partials + (size_t)layer * L.partials_layer_stride;
  const int ub = li & 1;
  int* U = Ubuf + ub * (NH + 1);

  // ---------------------------------------------------------------- prologue
  bool have_units = true;
  if (li > 0) {
    // this layer's unit prefix (built by the block's last warp to leave layer
    // li - 2); a warp that gives up waiting does no work in the layer
    const uint64_t w0 = globaltimer_ns();
    while (s_tag[ub] != li + 1) {
      __nanosleep(32);
      if (globaltimer_ns() - w0 > kWaitLimitNs) {
        if (lane == 0) atomicOr(L.error, DMC_FAULT_WAIT_TIMEOUT);
        have_units = false;
        break;
      }
    }
    have_units = __all_sync(0xffffffffu, have_units);
    __threadfence_block();  // the prefix is read after its tag
  }
  const long long Utot = have_units ? U[NH] : 0;
  const int NW = gridDim.x * kGWarps;
  const int wid = blockIdx.x * kGWarps + warp;
  const int u0 = have_units ? (int)range_start(wid, Utot, NW) : 0;
  const int u1 = have_units ? (int)range_start(wid + 1, Utot, NW) : 0;
  const int n = u1 - u0;
  const uint32_t ring_s = smem_u32(ring);

  // page window: page id and rows to copy of units [pb, pb + kGWindow)
  int pb = u0;
  auto load_window = [&](int first) {
    pb = first;
    __syncwarp();
    for (int i = lane; i < kGWindow; i += 32) {
      const int u = first + i;
      int pid = 0, rws = 0;
      if (u < u1) {
        const int hv = head_of_unit(U, NH, u);
        const int j = u - U[hv];
        if (j < U[hv + 1] - U[hv] - 1) {
          pid = ptab[(size_t)hv * L.MPH + j];
          rws = min(kPage, len_cur[hv] - j * kPage);
        }
      }
      wpid[i] = pid;
      wrws[i] = rws;
    }
    __syncwarp();
  };

  // issue cursor: tile it of unit u0 + ik; an owner unit reserves one tile
  int ik = 0, it = 0, itn = -1, islot = 0;
  auto issue_next = [&]() {
    while (ik < n) {
      const int iu = u0 + ik;
      if (iu - pb >= kGWindow) load_window(iu);
      if (itn < 0) {
        const int rws = wrws[iu - pb];
        itn = rws > 0 ? ceil_div(rws, kTile) : 1;
      }
      if (it < itn) break;
      ++ik;
      it = 0;
      itn = -1;
    }
    if (ik < n) {
      const int iu = u0 + ik;
      const int rws = wrws[iu - pb];
      if (rws > 0) {
        const char* pg = L.pages + (size_t)wpid[iu - pb] * L.page_bytes;
        const uint32_t dst = ring_s + islot * G_::TILE;
#pragma unroll
        for (int i = 0; i < 2 * kTile * CPR / 32; ++i) {
          const int x = lane + 32 * i;
          const int which = x / (kTile * CPR);  // 0: K, 1: V
          const int rem = x % (kTile * CPR);
          const int r = rem / CPR, c = rem % CPR;
          const int row = it * kTile + r;
          const bool valid = row < rws;
          const char* src = pg + (size_t)which * kPage * ROW + (size_t)(valid ? row : 0) * ROW + c * 16;
          cp_async16_zfill(dst + which * kTile * ROW + swz(r, c, ROW), src, valid);
        }
      }
      ++it;
    }
    cp_async_commit();  // one group per call, possibly empty, on every lane
    islot = (islot + 1 == kGRing) ? 0 : islot + 1;
  };

  if (n > 0) {
    load_window(u0);
    for (int s = 0; s < kGRing - 1; ++s) issue_next();
  }

  // q, k, v and the slots this launch writes are touched only after this point
  if (li == 0) {
    griddep_wait();
    griddep_launch_dependents();
  }

  if (n > 0) {
    // lane i holds the gates of KV head hb + i
    int hb = 0, t_len = 0, t_flags = 0;
    float t_omega = 0.f;
    auto load_heads = [&](int first) {
      hb = first;
      const int hv = first + lane;
      t_len = 0;
      t_flags = 0;
      t_omega = 0.f;
      if (hv < NH && U[hv] < u1) {
        const int b = hv / L.Hkv, h = hv % L.Hkv;
        const int len = len_cur[hv];
        const float x = __bfloat162float(reinterpret_cast<const __nv_bfloat16*>(kL)[(size_t)hv * D]);
        float qs = 0.f;
        for (int gg = 0; gg < G; ++gg)
          qs += __bfloat162float(reinterpret_cast<const __nv_bfloat16*>(
              qL)[((size_t)b * L.Hq + (size_t)h * G + gg) * D]);
        t_len = len;
        // alpha = round(sigmoid(k[0])) = [k[0] >= 0]; an empty head always appends
        t_flags = ((x >= 0.f && len > 0) ? kGFlagAcc : 0) | ((x != x) ? kGFlagNaN : 0);
        t_omega = sigmoidf_(qs / (float)G);  // omega = sigmoid(mean of the group's q[0])
      }
    };
    int vh = head_of_unit(U, NH, u0);
    load_heads(vh);

    // A fragments of the group's queries: row g = query g (zero for g >= G),
    // q[0] removed. qa[kk][0]: dims kk*16 + 2t, +1; qa[kk][1]: dims + 8.
    auto load_q = [&](int hv, uint32_t (*qa)[2]) {
      const int b = hv / L.Hkv, h = hv % L.Hkv;
      const uint32_t* qrow = reinterpret_cast<const uint32_t*>(
          qL + ((size_t)b * L.Hq + (size_t)h * G + (g < G ? g : 0)) * ROW);
#pragma unroll
      for (int kk = 0; kk < KT; ++kk) {
        qa[kk][0] = g < G ? __ldg(qrow + kk * 8 + t) : 0u;
        qa[kk][1] = g < G ? __ldg(qrow + kk * 8 + 4 + t) : 0u;
      }
    };
    uint32_t qa[KT][2], qn[KT][2];
    load_q(vh, qn);

    const float qscale = 1.4426950408889634f / sqrtf((float)D);  // log2(e) / sqrt(d_h)
    float o[KT][4];
    float m = -INFINITY, lsum = 0.f;
#pragma unroll
    for (int mt = 0; mt < KT; ++mt) o[mt][0] = o[mt][1] = o[mt][2] = o[mt][3] = 0.f;
    int len_old = 0, flags = 0, cslot = 0;
    float omega = 0.f;

    // one tile of 16 slots, the first `valid` of them attended
    auto do_tile = [&](uint32_t tile, int valid) {
      float sc[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
      const int mi = lane >> 3, r = lane & 7;
      const int srow = (mi >> 1) * 8 + r;
#pragma unroll
      for (int kk = 0; kk < KT; ++kk) {
        uint32_t b00, b01, b10, b11;
        ldmatrix_x4(tile + swz(srow, kk * 2 + (mi & 1), ROW), b00, b01, b10, b11);
        mma_bf16_16816(sc[0], qa[kk][0], 0u, qa[kk][1], 0u, b00, b01);
        mma_bf16_16816(sc[1], qa[kk][0], 0u, qa[kk][1], 0u, b10, b11);
      }
      // scores of query g at slots 2t, 2t + 1, 8 + 2t, 9 + 2t
      float s[4] = {sc[0][0] * qscale, sc[0][1] * qscale, sc[1][0] * qscale, sc[1][1] * qscale};
      if (2 * t >= valid) s[0] = -INFINITY;
      if (2 * t + 1 >= valid) s[1] = -INFINITY;
      if (8 + 2 * t >= valid) s[2] = -INFINITY;
      if (9 + 2 * t >= valid) s[3] = -INFINITY;
      float mx = fmaxf(fmaxf(s[0], s[1]), fmaxf(s[2], s[3]));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
      const float mn = fmaxf(m, mx);
      const float corr = (m == -INFINITY) ? 0.f : exp2f(m - mn);
      float p[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) p[i] = (s[i] == -INFINITY) ? 0.f : exp2f(s[i] - mn);
      float ps = (p[0] + p[1]) + (p[2] + p[3]);
      ps += __shfl_xor_sync(0xffffffffu, ps, 1);
      ps += __shfl_xor_sync(0xffffffffu, ps, 2);
      lsum = lsum * corr + ps;
      m = mn;
      // output columns of this lane are queries 2t and 2t + 1
      const float c_lo = __shfl_sync(0xffffffffu, corr, 8 * t);
      const float c_hi = __shfl_sync(0xffffffffu, corr, 8 * t + 4);
      const uint32_t pb0 = pack_bf16x2(p[0], p[1]), pb1 = pack_bf16x2(p[2], p[3]);
      const uint32_t vtile = tile + kTile * ROW;
#pragma unroll
      for (int mt = 0; mt < KT; ++mt) {
        o[mt][0] *= c_lo;
        o[mt][1] *= c_hi;
        o[mt][2] *= c_lo;
        o[mt][3] *= c_hi;
        uint32_t a0, a1, a2, a3;
        ldmatrix_x4_trans(vtile + swz(srow, mt * 2 + (mi & 1), ROW), a0, a1, a2, a3);
        mma_bf16_16816(o[mt], a0, a1, a2, a3, pb0, pb1);
      }
    };

    for (int k = 0; k < n; ++k) {
      const int u = u0 + k;
      while (U[vh + 1] <= u) ++vh;
      const int hu0 = U[vh], hend = U[vh + 1], nU = hend - hu0, j = u - hu0;
      const bool owner = (j == nU - 1);
      if (k == 0 || j == 0) {
        if (vh - hb >= kGHeadWindow) load_heads(vh);
        const int src = vh - hb;
        len_old = __shfl_sync(0xffffffffu, t_len, src);
        flags = __shfl_sync(0xffffffffu, t_flags, src);
        omega = __shfl_sync(0xffffffffu, t_omega, src);
#pragma unroll
        for (int kk = 0; kk < KT; ++kk) {
          qa[kk][0] = qn[kk][0];
          qa[kk][1] = qn[kk][1];
        }
        if (t == 0) qa[0][0] &= 0xffff0000u;  // q[0] (low half of dims 0, 1) is the gate
        if (hend < u1) load_q(vh + 1, qn);    // the next head's queries, ahead of use
      }
      const int accum = flags & kGFlagAcc;
      if (!owner) {
        const int rows_copied = min(kPage, len_old - j * kPage);
        const int rows = min(kPage, len_old - accum - j * kPage);  // the merged slot is excluded
        const int ntl = ceil_div(rows_copied, kTile);
        for (int tl = 0; tl < ntl; ++tl) {
          issue_next();
          cp_async_wait<kGRing - 1>();
          __syncwarp();  // every lane's copies of this tile have landed
          do_tile(ring_s + cslot * G_::TILE, max(0, min(kTile, rows - tl * kTile)));
          cslot = (cslot + 1 == kGRing) ? 0 : cslot + 1;
        }
      } else {
        // Algorithm 1 on the KV head's new token, once for the group: lanes
        // 0..CPR-1 build the key row, lanes CPR..2*CPR-1 the value row, 8
        // dims each, in fp32, rounded to bf16.
        const bool is_v = lane >= CPR;
        const int c = is_v ? lane - CPR : lane;
        const bool act = lane < 2 * CPR;
        // When this warp has just streamed the head's last page (unit u - 1),
        // the old last row is in the tile it consumed last: read it before
        // the issue below reuses that ring slot. The issue window may still
        // hold that page's id.
        const bool ring_row = !kWin && accum && k > 0 && j > 0;
        uint4 oraw = make_uint4(0, 0, 0, 0);
        if (ring_row && act) {
          const int ps = (cslot == 0 ? kGRing : cslot) - 1;
          oraw = *reinterpret_cast<const uint4*>(smem + (ring_s - smem_u32(smem)) + ps * G_::TILE +
                                                 (is_v ? kTile * ROW : 0) + swz((len_old - 1) % kTile, c, ROW));
        }
        issue_next();
        cp_async_wait<kGRing - 1>();
        __syncwarp();  // the reserved tile's slot is free
        const uint32_t tile = ring_s + cslot * G_::TILE;
        cslot = (cslot + 1 == kGRing) ? 0 : cslot + 1;
        int tgt = -1;
        if (accum || len_old % kPage != 0) {
          const int up = u - 1;
          tgt = (k > 0 && j > 0 && up >= pb && up - pb < kGWindow)
                    ? wpid[up - pb]
                    : ptab[(size_t)vh * L.MPH + (len_old - 1) / kPage];
        }
        // window grouping: the slot is the mean of the segment's last W tokens,
        // the W - 1 before this one being in the head's ring
        const int W = kWin ? L.window : 0;
        const int Wm = kWin ? L.window : 1;
        int n_old = 0, nwin = 0;  // tokens before this one, of them in the window
        const char* ring = nullptr;
        const float* ring_w = nullptr;
        float zold = 0.f, znew = omega;
        if (W > 0) {
          ring = L.ring + ((size_t)layer * NH + vh) * W * 2 * ROW;
          ring_w = L.ring_w + ((size_t)layer * NH + vh) * W;
          if (accum) {
            n_old = L.seglen[((size_t)layer * 2 + parity) * NH + vh];
            nwin = min(n_old, W - 1);
            for (int e = 0; e < nwin; ++e) znew += ring_w[(n_old - 1 - e) % Wm];
          }
        } else if (accum) {
          zold = L.z[(size_t)tgt * kPage + (len_old - 1) % kPage];
          znew = zold + omega;
        }
        uint4 nrow = make_uint4(0, 0, 0, 0);
        if (act) {
          float in[8], nw[8];
          const char* src_in = (is_v ? vL : kL) + (size_t)vh * ROW + c * 16;
          CK::unpack(__ldg(reinterpret_cast<const uint4*>(src_in)), in);
          if (!is_v && c == 0) in[0] = 0.f;  // k[0] <- 0 (Algorithm 1)
          if (W > 0) {
#pragma unroll
            for (int e = 0; e < 8; ++e) nw[e] = in[e] * omega;
            for (int e2 = 0; e2 < nwin; ++e2) {
              const int pos = (n_old - 1 - e2) % Wm;
              float old[8];
              CK::unpack(*reinterpret_cast<const uint4*>(ring + (size_t)pos * 2 * ROW + (is_v ? ROW : 0) + c * 16), old);
              const float w = ring_w[pos];
#pragma unroll
              for (int e = 0; e < 8; ++e) nw[e] = fmaf(w, old[e], nw[e]);
            }
#pragma unroll
            for (int e = 0; e < 8; ++e) nw[e] /= znew;
            // the new token joins the ring at entry n_old % W
            char* re = L.ring + ((size_t)layer * NH + vh) * W * 2 * ROW + (size_t)(n_old % Wm) * 2 * ROW;
            *reinterpret_cast<uint4*>(re + (is_v ? ROW : 0) + c * 16) = CK::pack(in);
          } else if (accum) {
            float old[8];
            if (ring_row) {
              CK::unpack(oraw, old);
            } else {
              const char* orow = L.pages + (size_t)tgt * L.page_bytes +
                                 (size_t)(is_v ? kPage : 0) * ROW + (size_t)((len_old - 1) % kPage) * ROW;
              CK::unpack(*reinterpret_cast<const uint4*>(orow + c * 16), old);
            }
#pragma unroll
            for (int e = 0; e < 8; ++e) nw[e] = (old[e] * zold + in[e] * omega) / znew;
          } else {
#pragma unroll
            for (int e = 0; e < 8; ++e) nw[e] = in[e];
          }
          nrow = CK::pack(nw);
        }
        const int slot = accum ? len_old - 1 : len_old;
        bool ok = slot < L.max_slots;
        int page = tgt;
        if (ok && page < 0) {
          if (lane == 0) {
            const unsigned long long id = atomicAdd(L.pool_top, 1ull);
            if (id >= (unsigned long long)L.num_pages) {
              atomicOr(L.error, DMC_FAULT_PAGES_EXHAUSTED);
              page = -1;
            } else {
              page = (int)id;
              ptab[(size_t)vh * L.MPH + slot / kPage] = page;
            }
          }
          page = __shfl_sync(0xffffffffu, page, 0);
        }
        ok = ok && page >= 0;
        if (lane == 0) {
          if (slot >= L.max_slots) atomicOr(L.error, DMC_FAULT_SLOT_CAPACITY);
          if (ok) L.z[(size_t)page * kPage + slot % kPage] = znew;
          len_nxt[vh] = ok ? slot + 1 : len_old;
          if (W > 0) {
            L.ring_w[((size_t)layer * NH + vh) * W + n_old % Wm] = omega;
            L.seglen[((size_t)layer * 2 + (parity ^ 1)) * NH + vh] = n_old + 1;
          }
          if (flags & kGFlagNaN) atomicOr(L.error, DMC_FAULT_NAN_GATE);
        }
        if (ok && act) {
          char* dst = L.pages + (size_t)page * L.page_bytes + (size_t)(is_v ? kPage : 0) * ROW +
                      (size_t)(slot % kPage) * ROW;
          *reinterpret_cast<uint4*>(dst + c * 16) = nrow;
        }
        // the new row is row 0 of a one-row tile; the other value rows are
        // zero so that their zero weights give exact zeros
        unsigned char* tp = smem + (tile - smem_u32(smem));
        for (int x = lane; x < kTile * CPR; x += 32) {
          const int r = x / CPR, cc = x % CPR;
          *reinterpret_cast<uint4*>(tp + kTile * ROW + swz(r, cc, ROW)) = make_uint4(0, 0, 0, 0);
        }
        __syncwarp();
        if (act) *reinterpret_cast<uint4*>(tp + (is_v ? kTile * ROW : 0) + swz(0, c, ROW)) = nrow;
        __syncwarp();
        do_tile(tile, 1);
      }

      if (owner || k == n - 1) {
        // ---- this warp's part of the head is done
        const int b = vh / L.Hkv, h = vh % L.Hkv;
        __nv_bfloat16* ob = reinterpret_cast<__nv_bfloat16*>(outL) + ((size_t)b * L.Hq + (size_t)h * G) * D;
        const int q_lo = 2 * t, q_hi = 2 * t + 1;
        if (hu0 >= u0 && owner) {
          // the whole head was in this warp
          const float l_lo = __shfl_sync(0xffffffffu, lsum, 8 * t);
          const float l_hi = __shfl_sync(0xffffffffu, lsum, 8 * t + 4);
#pragma unroll
          for (int mt = 0; mt < KT; ++mt) {
            const int d0 = mt * 16 + g;
            if (q_lo < G) {
              ob[(size_t)q_lo * D + d0] = __float2bfloat16_rn(o[mt][0] / l_lo);
              ob[(size_t)q_lo * D + d0 + 8] = __float2bfloat16_rn(o[mt][2] / l_lo);
            }
            if (q_hi < G) {
              ob[(size_t)q_hi * D + d0] = __float2bfloat16_rn(o[mt][1] / l_hi);
              ob[(size_t)q_hi * D + d0 + 8] = __float2bfloat16_rn(o[mt][3] / l_hi);
            }
          }
        } else {
          // publish this warp's partial states (one per query); the last
          // contributor combines
          const int ps = 2 * wid + (hu0 <= u0 ? 0 : 1);
          float* pp = partials + (size_t)ps * G * (D + 2);
          if (t == 0 && g < G) {
            pp[(size_t)g * (D + 2)] = m;
            pp[(size_t)g * (D + 2) + 1] = lsum;
          }
#pragma unroll
          for (int mt = 0; mt < KT; ++mt) {
            const int d0 = mt * 16 + g;
            if (q_lo < G) {
              pp[(size_t)q_lo * (D + 2) + 2 + d0] = o[mt][0];
              pp[(size_t)q_lo * (D + 2) + 2 + d0 + 8] = o[mt][2];
            }
            if (q_hi < G) {
              pp[(size_t)q_hi * (D + 2) + 2 + d0] = o[mt][1];
              pp[(size_t)q_hi * (D + 2) + 2 + d0 + 8] = o[mt][3];
            }
          }
          __threadfence();
          __syncwarp();
          const int wf = worker_of_unit(hu0, Utot, NW);
          const int wl = worker_of_unit(hend - 1, Utot, NW);
          const bool dense = Utot >= NW;
          int last = 0;
          if (lane == 0) {
            int ncontrib = wl - wf + 1;
            if (!dense) {
              ncontrib = 0;
              for (int cw = wf; cw <= wl; ++cw)
                ncontrib += range_start(cw, Utot, NW) < range_start(cw + 1, Utot, NW);
            }
            int* cnt = L.counters + (size_t)layer * NH * G + vh;
            const int old = atomicAdd(cnt, 1);
            last = (old == ncontrib - 1);
            if (last) *cnt = 0;
          }
          last = __shfl_sync(0xffffffffu, last, 0);
          if (last) {
            __threadfence();
            // lane: query g, a quarter of the dims
            constexpr int DPQ = D / 4;
            const int qq = g, d_lo = t * DPQ;
            float Mc = -INFINITY;
            for (int cw = wf; cw <= wl; ++cw) {
              const long long cs0 = range_start(cw, Utot, NW);
              if (cs0 == range_start(cw + 1, Utot, NW)) continue;
              const int cs = 2 * cw + (hu0 <= cs0 ? 0 : 1);
              if (qq < G) Mc = fmaxf(Mc, __ldcg(partials + ((size_t)cs * G + qq) * (D + 2)));
            }
            float Lc = 0.f, Oc[DPQ];
#pragma unroll
            for (int i = 0; i < DPQ; ++i) Oc[i] = 0.f;
            for (int cw = wf; cw <= wl; ++cw) {
              const long long cs0 = range_start(cw, Utot, NW);
              if (cs0 == range_start(cw + 1, Utot, NW)) continue;
              const int cs = 2 * cw + (hu0 <= cs0 ? 0 : 1);
              if (qq < G) {
                const float* cp = partials + ((size_t)cs * G + qq) * (D + 2);
                const float mc = __ldcg(cp);
                const float cwt = (mc == -INFINITY) ? 0.f : exp2f(mc - Mc);
                Lc = fmaf(__ldcg(cp + 1), cwt, Lc);
#pragma unroll
                for (int i = 0; i < DPQ; ++i) Oc[i] = fmaf(__ldcg(cp + 2 + d_lo + i), cwt, Oc[i]);
              }
            }
            if (qq < G) {
              const float inv = 1.f / Lc;
#pragma unroll
              for (int i = 0; i < DPQ; ++i)
                ob[(size_t)qq * D + d_lo + i] = __float2bfloat16_rn(Oc[i] * inv);
            }
          }
        }
        m = -INFINITY;
        lsum = 0.f;
#pragma unroll
        for (int mt = 0; mt < KT; ++mt) o[mt][0] = o[mt][1] = o[mt][2] = o[mt][3] = 0.f;
      }
    }
  }
  cp_async_wait<0>();

  // this warp is done with the layer: the grid's last warp out publishes the
  // new slot counts; the block's last warp out builds the prefix of layer
  // li + 2 into the buffer the layer used
  __syncwarp();
  int last_in_block = 0;
  if (lane == 0) {
    __threadfence();
    const int old = atomicAdd(&ctl[1], 1);
    if (old == (int)gridDim.x * kGWarps - 1) {
      ctl[1] = 0;
      ctl[0] = parity ^ 1;
      __threadfence();
    }
    last_in_block = atomicAdd(const_cast<int*>(&s_done[ub]), 1) == kGWarps - 1;
  }
  last_in_block = __shfl_sync(0xffffffffu, last_in_block, 0);
  if (last_in_block) {
    __threadfence_block();  // every warp's reads of the buffer came before its count
    if (li + 2 < a.nlayers)
      scan_units_warp(U, L.ctl + (layer + 2) * 4, L.lengths + (size_t)(layer + 2) * 2 * NH, NH);
    if (lane == 0) {
      s_done[ub] = 0;
      __threadfence_block();
      s_tag[ub] = li + 3;
    }
  }
  }  // layers
}

template <int D>
static cudaError_t setup_gqa(const Layout& L, DecodePlan* plan) {
  using G_ = GqaGeom<D>;
  int dev = 0, sms = 0, optin = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  if (e != cudaSuccess) return e;
  plan->stages = kGRing;
  plan->smem = G_::smem_bytes(L.NH);
  if (plan->smem > (size_t)optin) return cudaErrorInvalidConfiguration;
  e = cudaFuncSetAttribute(dmc_decode_gqa_kernel<D, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)plan->smem);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(dmc_decode_gqa_kernel<D, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)plan->smem);
  if (e != cudaSuccess) return e;
  int occ = 0, occw = 0;
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, dmc_decode_gqa_kernel<D, false>, kGThreads,
                                                    plan->smem);
  if (e == cudaSuccess)
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occw, dmc_decode_gqa_kernel<D, true>, kGThreads,
                                                      plan->smem);
  occ = min(occ, occw);
  if (e != cudaSuccess) return e;
  if (occ < 1) return cudaErrorInvalidConfiguration;
  plan->grid = min(sms * occ, kGMaxBlocks);
  const long long max_units = (long long)L.NH * (L.MPH + 1);
  const long long max_blocks = (max_units + kGWarps - 1) / kGWarps;
  if (max_blocks < plan->grid) plan->grid = (int)max_blocks;
  plan->partial_states = 2 * plan->grid * kGWarps * L.G;
  plan->grid_walk = plan->grid;  // one launch shape whatever the layers
  plan->smem_walk = plan->smem;
  if (plan->partial_states > L.partial_cap) return cudaErrorInvalidConfiguration;
  return cudaSuccess;
}

bool gqa_supported(const Layout& L) {
  return L.esize == 2 && L.G >= 2 && L.G <= kGMaxQueries && (L.D == 64 || L.D == 128);
}

cudaError_t gqa_setup(const Layout& L, DecodePlan* plan) {
  if (L.D == 64) return setup_gqa<64>(L, plan);
  if (L.D == 128) return setup_gqa<128>(L, plan);
  return cudaErrorInvalidValue;
}

cudaError_t gqa_launch(const Layout& L, int layer0, int nlayers, const DecodePlan& plan, bool pdl,
                       const void* q, const void* k, const void* v, void* out, cudaStream_t stream) {
  GqaArgs a;
  a.lay = L;
  a.layer0 = layer0;
  a.nlayers = nlayers;
  a.q_ls = (long long)L.B * L.Hq * L.row_bytes;
  a.kv_ls = (long long)L.B * L.Hkv * L.row_bytes;
  a.q = static_cast<const char*>(q);
  a.k = static_cast<const char*>(k);
  a.v = static_cast<const char*>(v);
  a.out = static_cast<char*>(out);
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(plan.grid);
  cfg.blockDim = dim3(kGThreads);
  cfg.dynamicSmemBytes = plan.smem;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  cudaError_t e = cudaErrorInvalidValue;
  const bool win = L.window > 0;
  if (L.D == 64) e = win ? cudaLaunchKernelEx(&cfg, dmc_decode_gqa_kernel<64, true>, a)
                         : cudaLaunchKernelEx(&cfg, dmc_decode_gqa_kernel<64, false>, a);
  if (L.D == 128) e = win ? cudaLaunchKernelEx(&cfg, dmc_decode_gqa_kernel<128, true>, a)
                          : cudaLaunchKernelEx(&cfg, dmc_decode_gqa_kernel<128, false>, a);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace dmc
