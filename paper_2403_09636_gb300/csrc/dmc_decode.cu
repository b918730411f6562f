// Fused DMC decode step: Algorithm 1 on the new token of every KV head plus
// single-query softmax attention over each head's updated, variable-length,
// paged cache (Eq. attn-softmax over the compressed slots, Sec. 3.1).
//
// Work split: every head h contributes ceil(len_old(h) / 32) page units plus
// one "owner" unit that carries the token being merged or appended. All units
// of a layer form one list, split into equal contiguous ranges over every warp
// of the grid ("stream-K" at warp granularity), so each warp streams the same
// number of pages whatever the spread of head lengths. Warps are independent
// workers: there is no barrier between them after the prologue.
//
// A warp streams its pages in "quads" of 4 slot rows, one row per 8-lane
// group, 16 bytes per lane per 128-byte chunk of a row. Each lane copies its
// own chunks of K and V with cp.async into a private ring of kRing quads in
// shared memory and later reads back exactly the bytes it copied, so the ring
// needs no synchronisation; kRing - 1 quads are in flight per warp. A head cut
// by range boundaries is finished by whichever of its warps arrives last
// (a counter, no waiting), which merges the partial softmax states in worker
// order, so results are deterministic.
//
// The slot that Algorithm 1 changes (the merged last slot, or the new one) is
// never read from the page: the owner unit computes it in registers from the
// old row, z and the new k, v, stores it rounded to the cache dtype and scores
// that rounded value, so no warp reads a slot the launch writes.
//
// Slot counts are double-buffered per layer: this launch reads buffer
// `parity` and writes the other; the last block to finish flips the parity, so
// the unit list stays consistent while owners publish new lengths, and a
// replayed CUDA graph stays correct.
//
// Programmatic dependent launch: everything before griddep_wait() reads only
// this layer's cache state (lengths, page table, pages), never q, k, v or
// anything a preceding kernel of another layer writes, so it may overlap the
// tail of the previous kernel on the stream. The host does not use the
// attribute when the previous decode launch of the cache was for the same
// layer.
#include <math.h>

#include <mutex>

#include "dmc_internal.cuh"
#include "dmc_split.cuh"

namespace dmc {

// Worker warps per block: a launch over one layer ends with a tail (its last
// heads finish while other warps idle), which fewer, longer warp ranges make
// shorter; a launch over several layers pays the tail once, and streams faster
// with more warps in flight.
constexpr int kWarpsOne = kDecodeWarpsPerBlock;
constexpr int kWarpsWalk = kDecodeWalkWarpsPerBlock;
constexpr int kRing = 5;        // quads per warp ring (kRing - 1 in flight)
constexpr int kWindow = 64;     // page units per warp window (page id + rows to copy)
constexpr int kHeadWindow = 32; // heads whose gates a warp holds in its lanes
constexpr int kMaxDecodeBlocks = 512;
constexpr int kMaxWorkers = kMaxDecodeBlocks * (kWarpsOne > kWarpsWalk ? kWarpsOne : kWarpsWalk);
static_assert(kMaxWorkers * 2 <= kMaxWorkerStates, "partials hold two states per worker");

enum : int { kFlagAcc = 1, kFlagNaN = 2 };

struct DecodeArgs {
  Layout lay;
  int layer0, nlayers;  // layers [layer0, layer0 + nlayers), walked in order
  int Gv;  // virtual heads per KV head: 1, or G when each query head of a group runs alone
  const char* q;  // layer layer0 + i at q + i * q_ls bytes: [B][Hq][D]
  const char* k;  // at k + i * kv_ls: [B][Hkv][D]
  const char* v;
  char* out;      // at out + i * q_ls: [B][Hq][D]
  long long q_ls, kv_ls;
};

template <typename T, int D>
struct DecodeGeom {
  static constexpr int ROW = D * (int)sizeof(T);
  static constexpr int NCH = ROW / 128;    // 16-byte chunks per lane of an 8-lane group
  static constexpr int EPC = Chunk<T>::N;  // elements per chunk
  static constexpr int EPL = NCH * EPC;    // elements of a row held by one lane
  // ring slot of one warp: [2 * NCH chunks][32 lanes][16 bytes], K chunks first
  static constexpr int WSLOT = 2 * NCH * 32 * 16;
  static constexpr int WRING = kRing * WSLOT;
  static constexpr int WWIN = 2 * kWindow * 4;  // page ids, rows to copy
  static constexpr int WARP_BYTES = WRING + WWIN;
  static constexpr int MISC = 64;
  static size_t smem_bytes(int nvh, int warps) {
    return (size_t)warps * WARP_BYTES + MISC + (size_t)(nvh + 1) * 4;
  }
};

template <int EPL>
__device__ __forceinline__ void merge_state(float& m, float& l, float* acc, float m2, float l2,
                                            const float* acc2) {
  const float mn = fmaxf(m, m2);
  const float c1 = (m == -INFINITY) ? 0.f : exp2f(m - mn);
  const float c2 = (m2 == -INFINITY) ? 0.f : exp2f(m2 - mn);
  l = l * c1 + l2 * c2;
#pragma unroll
  for (int i = 0; i < EPL; ++i) acc[i] = acc[i] * c1 + acc2[i] * c2;
  m = mn;
}

// Floats per split-K partial state: m, l, two pad words, then the D
// accumulator floats, so the accumulator is 16-byte aligned.
template <int D>
constexpr int kPartialStride = D + 4;

// The last contributor of a split head merges the nc partial states of workers
// wf..wf+nc-1 in worker order and writes the head's output row. Lane
// (cg = lane / 8, dg = lane % 8) sums contributors cg, cg + 4, ... over dims
// [dg * D / 8, (dg + 1) * D / 8), eight contributors' loads in flight per
// batch; the four contributor groups are then added with shuffles.
template <typename T, int D>
__device__ __noinline__ void combine_partials(const float* partials, int wf, int first_off,
                                                 int nc, int lane, T* orow) {
  constexpr int PS = kPartialStride<D>;
  constexpr int V4 = D / 32;  // float4 per lane per contributor
  const int cg = lane >> 3, dg = lane & 7;
  auto slot = [&](int i) { return 2 * (wf + i) + (i == 0 ? first_off : 0); };
  float2 ml0 = make_float2(-INFINITY, 0.f);
  if (lane < nc) ml0 = __ldcg(reinterpret_cast<const float2*>(partials + (size_t)slot(lane) * PS));
  float Mc = ml0.x;
  for (int i = lane + 32; i < nc; i += 32) Mc = fmaxf(Mc, __ldcg(partials + (size_t)slot(i) * PS));
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) Mc = fmaxf(Mc, __shfl_xor_sync(0xffffffffu, Mc, off));
  float Lc = 0.f;
  float4 o[V4];
#pragma unroll
  for (int k = 0; k < V4; ++k) o[k] = make_float4(0.f, 0.f, 0.f, 0.f);
  for (int i0 = 0; i0 < nc; i0 += 32) {
    const int i = i0 + lane;
    float2 ml = ml0;
    if (i0 > 0)
      ml = i < nc ? __ldcg(reinterpret_cast<const float2*>(partials + (size_t)slot(i) * PS))
                  : make_float2(-INFINITY, 0.f);
    const float w = (i < nc && ml.x != -INFINITY) ? exp2f(ml.x - Mc) : 0.f;
    Lc = fmaf(ml.y, w, Lc);
    const int n32 = min(32, nc - i0);
    for (int c0 = 0; c0 < n32; c0 += 8) {
      float4 v[2][V4];
      float wv[2];
#pragma unroll
      for (int r = 0; r < 2; ++r) {
        const int c = c0 + 4 * r + cg;  // < 32
        wv[r] = __shfl_sync(0xffffffffu, w, c);
        if (c < n32) {
          const float4* p = reinterpret_cast<const float4*>(partials + (size_t)slot(i0 + c) * PS + 4) + dg * V4;
#pragma unroll
          for (int k = 0; k < V4; ++k) v[r][k] = __ldcg(p + k);
        } else {
          wv[r] = 0.f;
#pragma unroll
          for (int k = 0; k < V4; ++k) v[r][k] = make_float4(0.f, 0.f, 0.f, 0.f);
        }
      }
#pragma unroll
      for (int r = 0; r < 2; ++r)
#pragma unroll
        for (int k = 0; k < V4; ++k) {
          o[k].x = fmaf(v[r][k].x, wv[r], o[k].x);
          o[k].y = fmaf(v[r][k].y, wv[r], o[k].y);
          o[k].z = fmaf(v[r][k].z, wv[r], o[k].z);
          o[k].w = fmaf(v[r][k].w, wv[r], o[k].w);
        }
    }
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) Lc += __shfl_xor_sync(0xffffffffu, Lc, off);
#pragma unroll
  for (int k = 0; k < V4; ++k)
#pragma unroll
    for (int off = 8; off < 32; off <<= 1) {
      o[k].x += __shfl_xor_sync(0xffffffffu, o[k].x, off);
      o[k].y += __shfl_xor_sync(0xffffffffu, o[k].y, off);
      o[k].z += __shfl_xor_sync(0xffffffffu, o[k].z, off);
      o[k].w += __shfl_xor_sync(0xffffffffu, o[k].w, off);
    }
  if (cg == 0) {
    const float inv = 1.f / Lc;
    float f[4 * V4];
#pragma unroll
    for (int k = 0; k < V4; ++k) {
      f[4 * k] = o[k].x * inv;
      f[4 * k + 1] = o[k].y * inv;
      f[4 * k + 2] = o[k].z * inv;
      f[4 * k + 3] = o[k].w * inv;
    }
    constexpr int EPC = Chunk<T>::N;
    char* dst = reinterpret_cast<char*>(orow) + (size_t)dg * (D / 8) * sizeof(T);
#pragma unroll
    for (int c = 0; c < 4 * V4 / EPC; ++c)
      *reinterpret_cast<uint4*>(dst + c * 16) = Chunk<T>::pack(f + c * EPC);
  }
}

// kWin: the cache uses the window-grouping approximation (L.window > 0);
// NWARP: worker warps per block
template <typename T, int D, bool kWin, int NWARP>
__global__ void __launch_bounds__(NWARP * 32, 2)
dmc_decode_kernel(const DecodeArgs a) {
  using G_ = DecodeGeom<T, D>;
  using CK = Chunk<T>;
  constexpr int ROW = G_::ROW, NCH = G_::NCH, EPC = G_::EPC, EPL = G_::EPL;
  constexpr int PSTRIDE = kPartialStride<D>;
  extern __shared__ __align__(128) unsigned char smem[];

  const Layout& L = a.lay;
  const int Gv = a.Gv;
  const int NVH = L.NH * Gv;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  unsigned char* ring = smem + (size_t)warp * G_::WARP_BYTES;
  int* wpid = reinterpret_cast<int*>(ring + G_::WRING);
  int* wrws = wpid + kWindow;
  int* misc = reinterpret_cast<int*>(smem + (size_t)NWARP * G_::WARP_BYTES);
  int* U = misc + G_::MISC / 4;

  for (int li = 0; li < a.nlayers; ++li) {
  const int layer = a.layer0 + li;
  const char* qL = a.q + (size_t)li * a.q_ls;
  const char* kL = a.k + (size_t)li * a.kv_ls;
  const char* vL = a.v + (size_t)li * a.kv_ls;
  char* outL = a.out + (size_t)li * a.q_ls;
  int* ctl = L.ctl + layer * 4;
  const int parity = *reinterpret_cast<volatile int*>(&ctl[0]);
  const int* len_cur = L.lengths + ((size_t)layer * 2 + parity) * L.NH;
  int* len_nxt = L.lengths + ((size_t)layer * 2 + (parity ^ 1)) * L.NH;
  int* ptab = L.page_table + (size_t)layer * L.NH * L.MPH;
  float* partials = L.partials + (size_t)layer * L.partials_layer_stride;
  char* pending = L.pending + (size_t)layer * L.NH * 2 * ROW;
  int* pending_at = L.pending_at + (size_t)layer * L.NH;
  float* pending_z = L.pending_z + (size_t)layer * L.NH;

  if (li > 0) __syncthreads();  // every warp is done with the previous layer's U and window
  // ---------------------------------------------------------------- prologue
  scan_units(U, misc, ctl, L.lengths + (size_t)layer * 2 * L.NH, L.NH, NVH, Gv);
  const long long Utot = U[NVH];
  const int NW = gridDim.x * NWARP;
  const int wid = blockIdx.x * NWARP + warp;
  const int u0 = (int)range_start(wid, Utot, NW);
  const int u1 = (int)range_start(wid + 1, Utot, NW);
  const int grp = lane >> 3, l8 = lane & 7;
  const uint32_t ring_s = smem_u32(ring);

  const int n = u1 - u0;

  // page window: page id and rows to copy of units [pb, pb + kWindow)
  int pb = u0;
  auto load_window = [&](int first) {
    pb = first;
    __syncwarp();
    for (int i = lane; i < kWindow; i += 32) {
      const int u = first + i;
      int pid = 0, rws = 0;
      if (u < u1) {
        const int hv = head_of_unit(U, NVH, u);
        const int j = u - U[hv];
        if (j < U[hv + 1] - U[hv] - 1) {
          const int bh = hv / Gv;
          pid = ptab[(size_t)bh * L.MPH + j];
          rws = min(kPage, len_cur[bh] - j * kPage);
        }
      }
      wpid[i] = pid;
      wrws[i] = rws;
    }
    __syncwarp();
  };

  // issue cursor: unit u0 + ik, quad iq of that unit
  int ik = 0, iq = 0, inq = -1, islot = 0;
  auto issue_next = [&]() {
    while (ik < n) {
      const int iu = u0 + ik;
      if (iu - pb >= kWindow) load_window(iu);
      if (inq < 0) inq = (wrws[iu - pb] + 3) >> 2;
      if (iq < inq) break;
      ++ik;
      iq = 0;
      inq = -1;
    }
    if (ik < n) {
      const int iu = u0 + ik;
      const int row = iq * 4 + grp;
      if (row < wrws[iu - pb]) {
        const char* src = L.pages + (size_t)wpid[iu - pb] * L.page_bytes + (size_t)row * ROW + l8 * 16;
        const uint32_t dst = ring_s + islot * G_::WSLOT + lane * 16;
#pragma unroll
        for (int c = 0; c < NCH; ++c) {
          cp_async16(dst + c * 512, src + c * 128);
          cp_async16(dst + (NCH + c) * 512, src + (size_t)kPage * ROW + c * 128);
        }
      }
      ++iq;
    }
    cp_async_commit();  // one group per call, possibly empty, on every lane
    islot = (islot + 1 == kRing) ? 0 : islot + 1;
  };

  if (u0 < u1) {
    load_window(u0);
    for (int s = 0; s < kRing - 1; ++s) issue_next();
  }

  // q, k, v and the slots this launch writes are touched only after this point
  if (li == 0) {
    griddep_wait();
    griddep_launch_dependents();
  }

  if (u0 < u1) {
    // lane i holds the gates of head hb + i
    int hb = 0, t_len = 0, t_flags = 0;
    float t_omega = 0.f;
    auto load_heads = [&](int first) {
      hb = first;
      const int hv = first + lane;
      t_len = 0;
      t_flags = 0;
      t_omega = 0.f;
      if (hv < NVH && U[hv] < u1) {
        const int bh = hv / Gv, b = bh / L.Hkv, h = bh % L.Hkv;
        const int len = len_cur[bh];
        const float x = Elt<T>::to_f(reinterpret_cast<const T*>(kL)[(size_t)bh * D]);
        float qs = 0.f;
        for (int g = 0; g < L.G; ++g)
          qs += Elt<T>::to_f(
              reinterpret_cast<const T*>(qL)[((size_t)b * L.Hq + (size_t)h * L.G + g) * D]);
        t_len = len;
        // alpha = round(sigmoid(k[0])) = [k[0] >= 0]; an empty head always appends
        t_flags = ((x >= 0.f && len > 0) ? kFlagAcc : 0) | ((x != x) ? kFlagNaN : 0);
        t_omega = sigmoidf_(qs / (float)L.G);  // omega = sigmoid(mean of the group's q[0])
      }
    };
    int vh = head_of_unit(U, NVH, u0);
    load_heads(vh);
    // the query row of the next head, loaded ahead of its use
    auto q_ptr = [&](int hv) {
      const int bh = hv / Gv, b = bh / L.Hkv, h = bh % L.Hkv, g = hv % Gv;
      return qL + ((size_t)b * L.Hq + (size_t)h * L.G + g) * ROW + l8 * 16;
    };
    uint4 qraw[NCH];
#pragma unroll
    for (int c = 0; c < NCH; ++c) qraw[c] = __ldg(reinterpret_cast<const uint4*>(q_ptr(vh) + c * 128));

    const float qscale = 1.4426950408889634f / sqrtf((float)D);  // log2(e) / sqrt(d_h)
    float qf[EPL], acc[EPL];
    float m = -INFINITY, lsum = 0.f;
#pragma unroll
    for (int i = 0; i < EPL; ++i) { acc[i] = 0.f; qf[i] = 0.f; }
    int len_old = 0, flags = 0, cslot = 0;
    float omega = 0.f;

    for (int k = 0; k < n; ++k) {
      const int u = u0 + k;
      while (U[vh + 1] <= u) ++vh;
      const int hu0 = U[vh], hend = U[vh + 1], nU = hend - hu0, j = u - hu0;
      const bool owner = (j == nU - 1);
      const int bh = vh / Gv;
      if (k == 0 || j == 0) {
        if (vh - hb >= kHeadWindow) load_heads(vh);
        const int src = vh - hb;
        len_old = __shfl_sync(0xffffffffu, t_len, src);
        flags = __shfl_sync(0xffffffffu, t_flags, src);
        omega = __shfl_sync(0xffffffffu, t_omega, src);
#pragma unroll
        for (int c = 0; c < NCH; ++c) {
          float f[EPC];
          CK::unpack(qraw[c], f);
#pragma unroll
          for (int e = 0; e < EPC; ++e) qf[c * EPC + e] = f[e] * qscale;
        }
        if (l8 == 0) qf[0] = 0.f;  // q[0] is the importance gate, not a feature
        // prefetch the query of the head that follows in this range
        const int next = hend < u1 ? vh + 1 : -1;
        if (next >= 0) {
#pragma unroll
          for (int c = 0; c < NCH; ++c)
            qraw[c] = __ldg(reinterpret_cast<const uint4*>(q_ptr(next) + c * 128));
        }
      }
      const int accum = flags & kFlagAcc;
      if (!owner) {
        const int rows_copied = min(kPage, len_old - j * kPage);
        const int rows = min(kPage, len_old - accum - j * kPage);  // the merged slot is excluded
        const int nq = (rows_copied + 3) >> 2;
        for (int qd = 0; qd < nq; ++qd) {
          issue_next();
          cp_async_wait<kRing - 1>();  // this lane's copies of quad qd have landed
          const unsigned char* sl = ring + cslot * G_::WSLOT + lane * 16;
          cslot = (cslot + 1 == kRing) ? 0 : cslot + 1;
          float s0 = 0.f, s1 = 0.f;
#pragma unroll
          for (int c = 0; c < NCH; ++c) {
            float f[EPC];
            CK::unpack(*reinterpret_cast<const uint4*>(sl + c * 512), f);
#pragma unroll
            for (int e = 0; e < EPC; e += 2) {
              s0 = fmaf(qf[c * EPC + e], f[e], s0);
              s1 = fmaf(qf[c * EPC + e + 1], f[e + 1], s1);
            }
          }
          float s = s0 + s1;
          s += __shfl_xor_sync(0xffffffffu, s, 1);
          s += __shfl_xor_sync(0xffffffffu, s, 2);
          s += __shfl_xor_sync(0xffffffffu, s, 4);
          if (qd * 4 + grp < rows) {
            const float mn = fmaxf(m, s);
            const float corr = exp2f(m - mn);
            const float p = exp2f(s - mn);
            lsum = fmaf(lsum, corr, p);
#pragma unroll
            for (int c = 0; c < NCH; ++c) {
              float f[EPC];
              CK::unpack(*reinterpret_cast<const uint4*>(sl + (NCH + c) * 512), f);
#pragma unroll
              for (int e = 0; e < EPC; ++e)
                acc[c * EPC + e] = fmaf(acc[c * EPC + e], corr, p * f[e]);
            }
            m = mn;
          }
        }
      } else {
        // Window grouping: the merge averages the open segment's window with
        // the new token. The four row groups read the window's rows (entries
        // grp, grp + 4, ... back from the newest) and add their sums.
        constexpr int WR = kWin ? EPL : 1;
        float rk[WR], rv[WR], rz = 0.f;
        int n_old = 0, nwin = 0;  // tokens before this one, of them in the window
        if constexpr (kWin) {
#pragma unroll
          for (int i = 0; i < EPL; ++i) { rk[i] = 0.f; rv[i] = 0.f; }
          const int W = L.window;
          if (accum) {
            n_old = L.seglen[((size_t)layer * 2 + parity) * L.NH + bh];
            nwin = min(n_old, W - 1);
            const char* ring = L.ring + ((size_t)layer * L.NH + bh) * W * 2 * ROW;
            const float* ring_w = L.ring_w + ((size_t)layer * L.NH + bh) * W;
            for (int e = grp; e < nwin; e += 4) {
              const int pos = (n_old - 1 - e) % W;
              const float w = ring_w[pos];
              rz += w;
#pragma unroll
              for (int c = 0; c < NCH; ++c) {
                float ko[EPC], vo[EPC];
                CK::unpack(*reinterpret_cast<const uint4*>(ring + (size_t)pos * 2 * ROW + c * 128 + l8 * 16), ko);
                CK::unpack(*reinterpret_cast<const uint4*>(ring + (size_t)pos * 2 * ROW + ROW + c * 128 + l8 * 16), vo);
#pragma unroll
                for (int q = 0; q < EPC; ++q) {
                  rk[c * EPC + q] = fmaf(w, ko[q], rk[c * EPC + q]);
                  rv[c * EPC + q] = fmaf(w, vo[q], rv[c * EPC + q]);
                }
              }
            }
          }
#pragma unroll
          for (int off = 8; off < 32; off <<= 1) {
#pragma unroll
            for (int i = 0; i < EPL; ++i) {
              rk[i] += __shfl_xor_sync(0xffffffffu, rk[i], off);
              rv[i] += __shfl_xor_sync(0xffffffffu, rv[i], off);
            }
            rz += __shfl_xor_sync(0xffffffffu, rz, off);
          }
        }
        // When this warp has just streamed the head's last page (unit u - 1),
        // its last quad holds the old last row in the ring, in the lanes of row
        // group (len_old - 1) % 4, and the issue window may still hold that
        // page's id: that group then applies the update without a round trip
        // for either.
        const bool ring_row = !kWin && accum && k > 0 && j > 0;
        const int og = ring_row ? ((len_old - 1) & 3) : 0;
        const unsigned gmask = 0xffu << (8 * og);
        if (grp == og) {
        // Algorithm 1 on the new token, in fp32, result rounded to the cache dtype.
        int tgt = -1;
        if (accum || len_old % kPage != 0) {
          const int up = u - 1;
          tgt = (k > 0 && j > 0 && up >= pb && up - pb < kWindow)
                    ? wpid[up - pb]
                    : ptab[(size_t)bh * L.MPH + (len_old - 1) / kPage];
        }
        const unsigned char* rrow =
            ring + (size_t)((cslot == 0 ? kRing : cslot) - 1) * G_::WSLOT + lane * 16;
        float zold = 0.f, znew = omega;
        const char* orow = nullptr;
        // window grouping: the slot is the mean of the segment's last W
        // tokens, the W - 1 before this one being in the head's ring
        const int W = kWin ? L.window : 0;
        const int Wm = kWin ? L.window : 1;  // the ring's modulus (only used when W > 0)
        if (W > 0) {
          znew = omega + rz;
        } else if (accum) {
          orow = L.pages + (size_t)tgt * L.page_bytes + (size_t)((len_old - 1) % kPage) * ROW;
          zold = L.z[(size_t)tgt * kPage + (len_old - 1) % kPage];
          znew = zold + omega;
        }
        uint4 nk[NCH], nv[NCH];
        float s = 0.f;
#pragma unroll
        for (int c = 0; c < NCH; ++c) {
          float kin[EPC], vin[EPC];
          CK::unpack(__ldg(reinterpret_cast<const uint4*>(kL + (size_t)bh * ROW + c * 128 + l8 * 16)), kin);
          CK::unpack(__ldg(reinterpret_cast<const uint4*>(vL + (size_t)bh * ROW + c * 128 + l8 * 16)), vin);
          if (c == 0 && l8 == 0) kin[0] = 0.f;  // k[0] <- 0 (Algorithm 1)
          float kn[EPC], vn[EPC];
          if (W > 0) {
#pragma unroll
            for (int e = 0; e < EPC; ++e) {
              kn[e] = fmaf(kin[e], omega, rk[(c * EPC + e) % WR]) / znew;
              vn[e] = fmaf(vin[e], omega, rv[(c * EPC + e) % WR]) / znew;
            }
            if (vh % Gv == 0) {
              // the new token joins the ring at entry n_old % W (no reader of
              // this launch looks there)
              char* re = L.ring + ((size_t)layer * L.NH + bh) * W * 2 * ROW + (size_t)(n_old % Wm) * 2 * ROW;
              *reinterpret_cast<uint4*>(re + c * 128 + l8 * 16) = CK::pack(kin);
              *reinterpret_cast<uint4*>(re + ROW + c * 128 + l8 * 16) = CK::pack(vin);
            }
          } else if (accum) {
            float ko[EPC], vo[EPC];
            if (ring_row) {
              CK::unpack(*reinterpret_cast<const uint4*>(rrow + c * 512), ko);
              CK::unpack(*reinterpret_cast<const uint4*>(rrow + (NCH + c) * 512), vo);
            } else {
              CK::unpack(*reinterpret_cast<const uint4*>(orow + c * 128 + l8 * 16), ko);
              CK::unpack(*reinterpret_cast<const uint4*>(orow + (size_t)kPage * ROW + c * 128 + l8 * 16), vo);
            }
#pragma unroll
            for (int e = 0; e < EPC; ++e) {
              kn[e] = (ko[e] * zold + kin[e] * omega) / znew;
              vn[e] = (vo[e] * zold + vin[e] * omega) / znew;
            }
          } else {
#pragma unroll
            for (int e = 0; e < EPC; ++e) { kn[e] = kin[e]; vn[e] = vin[e]; }
          }
          nk[c] = CK::pack(kn);
          nv[c] = CK::pack(vn);
          float kr[EPC];
          CK::unpack(nk[c], kr);  // score the stored (rounded) key
#pragma unroll
          for (int e = 0; e < EPC; ++e) s = fmaf(qf[c * EPC + e], kr[e], s);
        }
        if (vh % Gv == 0) {  // one writer per KV head
          const int slot = accum ? len_old - 1 : len_old;
          bool ok = slot < L.max_slots;
          if (!ok && l8 == 0) atomicOr(L.error, DMC_FAULT_SLOT_CAPACITY);
          int page = tgt;
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
            page = __shfl_sync(gmask, page, 0, 8);
          }
          ok = ok && page >= 0;
          // With grouped queries the other virtual heads of this KV head may
          // still read the old last row and z in this launch: the new row waits
          // in the pending buffer until the launch's last block writes it.
          char* dst = Gv > 1 ? pending + (size_t)bh * 2 * ROW
                             : L.pages + (size_t)page * L.page_bytes + (size_t)(slot % kPage) * ROW;
          const size_t vstride = Gv > 1 ? (size_t)ROW : (size_t)kPage * ROW;
          if (ok) {
#pragma unroll
            for (int c = 0; c < NCH; ++c) {
              *reinterpret_cast<uint4*>(dst + c * 128 + l8 * 16) = nk[c];
              *reinterpret_cast<uint4*>(dst + vstride + c * 128 + l8 * 16) = nv[c];
            }
          }
          if (l8 == 0) {
            if (Gv > 1) {
              pending_at[bh] = ok ? page * kPage + slot % kPage : -1;
              pending_z[bh] = znew;
            } else if (ok) {
              L.z[(size_t)page * kPage + slot % kPage] = znew;
            }
            len_nxt[bh] = ok ? slot + 1 : len_old;
            if (W > 0) {
              L.ring_w[((size_t)layer * L.NH + bh) * W + n_old % Wm] = omega;
              L.seglen[((size_t)layer * 2 + (parity ^ 1)) * L.NH + bh] = n_old + 1;
            }
            if (flags & kFlagNaN) atomicOr(L.error, DMC_FAULT_NAN_GATE);
          }
        }
        s += __shfl_xor_sync(gmask, s, 1);
        s += __shfl_xor_sync(gmask, s, 2);
        s += __shfl_xor_sync(gmask, s, 4);
        const float mn = fmaxf(m, s);
        const float corr = exp2f(m - mn);
        const float p = exp2f(s - mn);
        lsum = fmaf(lsum, corr, p);
#pragma unroll
        for (int c = 0; c < NCH; ++c) {
          float vr[EPC];
          CK::unpack(nv[c], vr);
#pragma unroll
          for (int e = 0; e < EPC; ++e) acc[c * EPC + e] = fmaf(acc[c * EPC + e], corr, p * vr[e]);
        }
        m = mn;
        }
      }

      if (owner || k == n - 1) {
        // ---- this warp's part of the head is done: merge its 4 groups
#pragma unroll
        for (int off = 8; off < 32; off <<= 1) {
          const float m2 = __shfl_xor_sync(0xffffffffu, m, off);
          const float l2 = __shfl_xor_sync(0xffffffffu, lsum, off);
          float a2[EPL];
#pragma unroll
          for (int i = 0; i < EPL; ++i) a2[i] = __shfl_xor_sync(0xffffffffu, acc[i], off);
          merge_state<EPL>(m, lsum, acc, m2, l2, a2);
        }
        const int b = bh / L.Hkv, h = bh % L.Hkv, g = vh % Gv;
        T* orow = reinterpret_cast<T*>(outL) + ((size_t)b * L.Hq + (size_t)h * L.G + g) * D;
        if (hu0 >= u0 && hend <= u1) {
          // the whole head was in this warp
          if (lane < 8) {
            const float inv = 1.f / lsum;
#pragma unroll
            for (int c = 0; c < NCH; ++c) {
              float o[EPC];
#pragma unroll
              for (int e = 0; e < EPC; ++e) o[e] = acc[c * EPC + e] * inv;
              if constexpr (sizeof(T) == 2) {
                *reinterpret_cast<uint4*>(orow + (c * 128 + l8 * 16) / 2) = CK::pack(o);
              } else {
                *reinterpret_cast<uint4*>(orow + (c * 128 + l8 * 16) / 4) = CK::pack(o);
              }
            }
          }
        } else {
          // publish this warp's partial state; the last contributor combines
          const int ps = 2 * wid + (hu0 <= u0 ? 0 : 1);
          float* pp = partials + (size_t)ps * PSTRIDE;
          if (lane == 0) *reinterpret_cast<float2*>(pp) = make_float2(m, lsum);
          // lanes of group g write float4 number g, g + 4, ... of their dims
#pragma unroll
          for (int v = 0; v < EPL / 4; ++v) {
            if ((v & 3) == grp) {
              const int c = v / (EPC / 4), e = (v % (EPC / 4)) * 4;
              *reinterpret_cast<float4*>(pp + 4 + (c * 128 + l8 * 16) / (int)sizeof(T) + e) =
                  make_float4(acc[c * EPC + e], acc[c * EPC + e + 1], acc[c * EPC + e + 2],
                              acc[c * EPC + e + 3]);
            }
          }
          __threadfence();  // the partial is visible before the counter moves
          __syncwarp();
          const int wf = worker_of_unit(hu0, Utot, NW);
          const int wl = worker_of_unit(hend - 1, Utot, NW);
          // With at least one unit per worker every worker in [wf, wl] holds
          // part of the head; otherwise some ranges in it are empty.
          const bool dense = Utot >= NW;
          int last = 0;
          if (lane == 0) {
            int ncontrib = wl - wf + 1;
            if (!dense) {
              ncontrib = 0;
              for (int cw = wf; cw <= wl; ++cw)
                ncontrib += range_start(cw, Utot, NW) < range_start(cw + 1, Utot, NW);
            }
            int* cnt = L.counters + (size_t)layer * L.NH * L.G + vh;
            const int old = atomicAdd(cnt, 1);
            last = (old == ncontrib - 1);
            if (last) *cnt = 0;
          }
          last = __shfl_sync(0xffffffffu, last, 0);
          if (last) {
            __threadfence();  // every contributor's partial is visible to this lane
            if (dense) {
              // worker wf + i wrote state 2 (wf + i) + 1 if the head starts
              // inside its range (only possible for i = 0), else 2 (wf + i)
              const int first_off = (hu0 > range_start(wf, Utot, NW)) ? 1 : 0;
              combine_partials<T, D>(partials, wf, first_off, wl - wf + 1, lane, orow);
            } else {
              // fewer units than workers (tiny caches): one unit per non-empty
              // range, so each contributor wrote state 2 cw of its range
              float Mc = -INFINITY, Lc = 0.f;
              for (int cw = wf; cw <= wl; ++cw) {
                if (range_start(cw, Utot, NW) == range_start(cw + 1, Utot, NW)) continue;
                Mc = fmaxf(Mc, __ldcg(partials + (size_t)(2 * cw) * PSTRIDE));
              }
              constexpr int DPL = D / 32;  // output dims per lane
              float Oc[DPL];
#pragma unroll
              for (int i = 0; i < DPL; ++i) Oc[i] = 0.f;
              for (int cw = wf; cw <= wl; ++cw) {
                if (range_start(cw, Utot, NW) == range_start(cw + 1, Utot, NW)) continue;
                const float* cp = partials + (size_t)(2 * cw) * PSTRIDE;
                const float mc = __ldcg(cp);
                const float cwt = (mc == -INFINITY) ? 0.f : exp2f(mc - Mc);
                Lc = fmaf(__ldcg(cp + 1), cwt, Lc);
#pragma unroll
                for (int i = 0; i < DPL; ++i) Oc[i] = fmaf(__ldcg(cp + 4 + lane * DPL + i), cwt, Oc[i]);
              }
              const float inv = 1.f / Lc;
#pragma unroll
              for (int i = 0; i < DPL; ++i) orow[lane * DPL + i] = Elt<T>::from_f(Oc[i] * inv);
            }
          }
        }
        m = -INFINITY;
        lsum = 0.f;
#pragma unroll
        for (int i = 0; i < EPL; ++i) acc[i] = 0.f;
      }
    }
  }
  cp_async_wait<0>();

  __syncthreads();
  if (tid == 0) {
    __threadfence();
    misc[0] = atomicAdd(&ctl[1], 1) == (int)gridDim.x - 1;
  }
  __syncthreads();
  if (misc[0]) {
    // last block of the launch: every owner has finished
    if (Gv > 1) {
      __threadfence();
      for (int bh = tid; bh < L.NH; bh += NWARP * 32) {
        const int at = pending_at[bh];
        if (at < 0) continue;
        char* dst = L.pages + (size_t)(at / kPage) * L.page_bytes + (size_t)(at % kPage) * ROW;
        const char* src = pending + (size_t)bh * 2 * ROW;
        for (int i = 0; i < ROW; i += 16) {
          *reinterpret_cast<uint4*>(dst + i) = *reinterpret_cast<const uint4*>(src + i);
          *reinterpret_cast<uint4*>(dst + (size_t)kPage * ROW + i) =
              *reinterpret_cast<const uint4*>(src + ROW + i);
        }
        L.z[at] = pending_z[bh];
      }
      __syncthreads();
    }
    if (tid == 0) {  // publish the new slot counts
      __threadfence();
      ctl[1] = 0;
      ctl[0] = parity ^ 1;
      __threadfence();
    }
  }
  }  // layers
}

// Shared memory and blocks per SM of one warp count (both window variants).
template <typename T, int D, int NWARP>
static cudaError_t setup_warps(int nvh, int optin, size_t* smem, int* occ) {
  *smem = DecodeGeom<T, D>::smem_bytes(nvh, NWARP);
  if (*smem > (size_t)optin) return cudaErrorInvalidConfiguration;
  cudaError_t e = cudaFuncSetAttribute(dmc_decode_kernel<T, D, false, NWARP>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)*smem);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(dmc_decode_kernel<T, D, true, NWARP>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, (int)*smem);
  int o = 0, ow = 0;
  if (e == cudaSuccess)
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&o, dmc_decode_kernel<T, D, false, NWARP>, NWARP * 32,
                                                      *smem);
  if (e == cudaSuccess)
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&ow, dmc_decode_kernel<T, D, true, NWARP>, NWARP * 32,
                                                      *smem);
  if (e != cudaSuccess) return e;
  *occ = min(o, ow);
  return *occ < 1 ? cudaErrorInvalidConfiguration : cudaSuccess;
}

template <typename T, int D>
static cudaError_t setup_decode(int nvh, DecodePlan* plan) {
  int dev = 0, sms = 0, optin = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  if (e != cudaSuccess) return e;
  plan->stages = kRing;
  int occ = 0, occw = 0;
  e = setup_warps<T, D, kWarpsOne>(nvh, optin, &plan->smem, &occ);
  if (e != cudaSuccess) return e;
  plan->grid = min(sms * occ, kMaxDecodeBlocks);
  // a launch over several layers takes the one-layer shape when its own does
  // not fit (wide rows with many heads)
  e = setup_warps<T, D, kWarpsWalk>(nvh, optin, &plan->smem_walk, &occw);
  plan->grid_walk = e == cudaSuccess ? min(sms * occw, kMaxDecodeBlocks) : 0;
  if (e == cudaErrorInvalidConfiguration) e = cudaSuccess;
  return e;
}

cudaError_t decode_setup(const Layout& L, int Gv, DecodePlan* plan) {
  const int nvh = L.NH * Gv;
  cudaError_t e = cudaErrorInvalidValue;
  if (L.esize == 4 && L.D == 64) e = setup_decode<float, 64>(nvh, plan);
  if (L.esize == 4 && L.D == 128) e = setup_decode<float, 128>(nvh, plan);
  if (L.esize == 2 && L.D == 64) e = setup_decode<__nv_bfloat16, 64>(nvh, plan);
  if (L.esize == 2 && L.D == 128) e = setup_decode<__nv_bfloat16, 128>(nvh, plan);
  if (e != cudaSuccess) return e;
  // no more warps than the most units a layer can have
  const long long max_units = (long long)nvh * (L.MPH + 1);
  plan->grid = (int)std::min<long long>(plan->grid, (max_units + kWarpsOne - 1) / kWarpsOne);
  plan->grid_walk = (int)std::min<long long>(plan->grid_walk, (max_units + kWarpsWalk - 1) / kWarpsWalk);
  plan->partial_states = 2 * max(plan->grid * kWarpsOne, plan->grid_walk * kWarpsWalk);
  if (plan->partial_states > L.partial_cap) return cudaErrorInvalidConfiguration;
  return cudaSuccess;
}

template <typename T, int D, int NWARP>
static cudaError_t launch_warps(const DecodeArgs& a, int grid, size_t smem, bool pdl, cudaStream_t stream) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(NWARP * 32);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  if (a.lay.window > 0) return cudaLaunchKernelEx(&cfg, dmc_decode_kernel<T, D, true, NWARP>, a);
  return cudaLaunchKernelEx(&cfg, dmc_decode_kernel<T, D, false, NWARP>, a);
}

template <typename T, int D>
static cudaError_t launch_decode(const DecodeArgs& a, const DecodePlan& plan, bool pdl,
                                 cudaStream_t stream) {
  if (a.nlayers > 1 && plan.grid_walk > 0)
    return launch_warps<T, D, kWarpsWalk>(a, plan.grid_walk, plan.smem_walk, pdl, stream);
  return launch_warps<T, D, kWarpsOne>(a, plan.grid, plan.smem, pdl, stream);
}

cudaError_t decode_launch(const Layout& L, int layer0, int nlayers, int Gv, const DecodePlan& plan,
                          bool pdl, const void* q, const void* k, const void* v, void* out,
                          cudaStream_t stream) {
  DecodeArgs a;
  a.lay = L;
  a.layer0 = layer0;
  a.nlayers = nlayers;
  a.q_ls = (long long)L.B * L.Hq * L.row_bytes;
  a.kv_ls = (long long)L.B * L.Hkv * L.row_bytes;
  a.Gv = Gv;
  a.q = static_cast<const char*>(q);
  a.k = static_cast<const char*>(k);
  a.v = static_cast<const char*>(v);
  a.out = static_cast<char*>(out);
  cudaError_t e = cudaErrorInvalidValue;
  if (L.esize == 4 && L.D == 64) e = launch_decode<float, 64>(a, plan, pdl, stream);
  else if (L.esize == 4 && L.D == 128) e = launch_decode<float, 128>(a, plan, pdl, stream);
  else if (L.esize == 2 && L.D == 64) e = launch_decode<__nv_bfloat16, 64>(a, plan, pdl, stream);
  else if (L.esize == 2 && L.D == 128) e = launch_decode<__nv_bfloat16, 128>(a, plan, pdl, stream);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

// ---------------------------------------------------------------- static scratch
// Scratch of dmc_decode_step_static_scratch: the split-K partial softmax states
// of one launch, 8 MiB. That holds two states of head_dim + 4 floats for each
// of the MHA kernel's 4096 worker warps at most, and the tensor-core kernel's
// two states per query of a group of 8 (head_dim + 2 floats each) for up to
// 252 blocks of 4 warps (a GB300 runs 152). Every GPU that loads the library
// holds it until exit.
constexpr size_t kStaticPartialFloats = (size_t)2 << 20;
static_assert(kStaticPartialFloats >= (size_t)2 * kMaxWorkers * kPartialStride<128>,
              "the static scratch holds every MHA decode grid");
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
