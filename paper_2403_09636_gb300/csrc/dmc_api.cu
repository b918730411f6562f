// Host side of the C ABI declared in include/dmc.h: config validation, the
// layout of a cache inside the caller's arena, and the small utility kernels
// (lengths copy, head export). The hot kernels live in dmc_decode.cu and
// dmc_prefill.cu.
#include <string.h>

#include <new>

#include "dmc_internal.cuh"

namespace dmc {
cudaError_t decode_setup(const Layout& L, int Gv, DecodePlan* plan);
cudaError_t decode_launch(const Layout& L, int layer0, int nlayers, int Gv, const DecodePlan& plan,
                          bool pdl, const void* q, const void* k, const void* v, void* out,
                          cudaStream_t stream);
cudaError_t prefill_launch(const Layout& L, int layer, int first_seq, int num_seqs, const void* q,
                           long long q_tok, long long q_head, const void* k, const void* v,
                           const int* cu, int total_tokens, int max_seqlen, float* carry,
                           cudaStream_t stream);
bool prefill_attn_supported(const Layout& L);
cudaError_t prefill_attn_launch(const Layout& L, int layer, int first_seq, int num_seqs,
                                const void* q, const void* k, const void* v, const int* cu,
                                int total_tokens, int max_seqlen, const float* carry, void* out,
                                cudaStream_t stream);
cudaError_t decode_static_partials(int device, float** ptr, size_t* floats);
bool gqa_supported(const Layout& L);
cudaError_t gqa_setup(const Layout& L, DecodePlan* plan);
cudaError_t gqa_launch(const Layout& L, int layer0, int nlayers, const DecodePlan& plan, bool pdl, const void* q,
                       const void* k, const void* v, void* out, cudaStream_t stream);
// Split-K partial states a cache's arena holds: two per worker warp of the
// decode grid (at most 512 blocks x 6 warps), times the group size for the
// tensor-core kernel, which keeps one per query.
inline size_t partial_states_cap(bool cuda_core, int G) {
  return cuda_core ? (size_t)kMaxWorkerStates : (size_t)kGqaWorkerStates * G;
}
}  // namespace dmc

using dmc::Layout;

struct dmc_cache {
  dmc_cache_config cfg;
  Layout lay;
  int device;
  int Gv;
  bool gqa;  // grouped queries on the tensor-core kernel (one worker per KV head)
  dmc::DecodePlan plan;
  int last_decode_lo, last_decode_hi;  // layers [lo, hi) of the latest kernel if it was a decode, else empty
  char* meta;  // lengths, ctl, counters, pool top, error: cleared by create / reset
  size_t meta_bytes;
  float* carry;  // segment sums at prompt chunk starts (prompt attention)
};

namespace {

constexpr size_t kAlign = 256;

size_t align_up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }

bool valid_config(const dmc_cache_config* c) {
  if (!c) return false;
  if (c->num_layers < 1 || c->batch < 1 || c->num_kv_heads < 1 || c->num_q_heads < 1) return false;
  if (c->num_q_heads % c->num_kv_heads != 0) return false;
  const int G = c->num_q_heads / c->num_kv_heads;
  if (G > 32) return false;
  if (c->head_dim != 64 && c->head_dim != 128) return false;
  if (c->dtype != DMC_F32 && c->dtype != DMC_BF16) return false;
  if (c->page_size != dmc::kPage) return false;
  if (c->max_slots_per_head < 1 || c->num_pages < 1 || c->num_pages > (int64_t)INT32_MAX) return false;
  if (c->max_prefill_tokens < 0 || c->window < 0 || c->window > dmc::kMaxWindow) return false;
  const int64_t nh = (int64_t)c->batch * c->num_kv_heads;
  if (nh * G > dmc::kMaxVirtualHeads) return false;
  return true;
}

// Byte offsets of every region; returns the total size.
struct Offsets {
  size_t pages, z, ptab, meta, lengths, ctl, counters, pool_top, error, meta_end, partials,
      pending, pending_at, pending_z, opens, plan, carry, ring, ring_w, seglen, total;
  int MPH, plan_stride;
};

Offsets offsets(const dmc_cache_config* c) {
  Offsets o;
  const int esize = c->dtype == DMC_F32 ? 4 : 2;
  const size_t row = (size_t)c->head_dim * esize;
  const size_t page_bytes = 2 * dmc::kPage * row;
  const int NH = c->batch * c->num_kv_heads;
  const int G = c->num_q_heads / c->num_kv_heads;
  o.MPH = dmc::ceil_div(c->max_slots_per_head, dmc::kPage);
  o.plan_stride = c->max_prefill_tokens / dmc::kPrefillChunk + c->batch + 2;
  size_t at = 0;
  o.pages = at; at = align_up(at + (size_t)c->num_pages * page_bytes);
  o.z = at; at = align_up(at + (size_t)c->num_pages * dmc::kPage * 4);
  o.ptab = at; at = align_up(at + (size_t)c->num_layers * NH * o.MPH * 4);
  o.meta = at;
  o.lengths = at; at = align_up(at + (size_t)c->num_layers * 2 * NH * 4);
  o.ctl = at; at = align_up(at + (size_t)c->num_layers * 4 * 4);
  o.counters = at; at = align_up(at + (size_t)c->num_layers * NH * G * 4);
  o.seglen = at; at = align_up(at + (c->window > 0 ? (size_t)c->num_layers * 2 * NH * 4 : 0));
  o.pool_top = at; at = align_up(at + 8);
  o.error = at; at = align_up(at + 4);
  o.meta_end = at;
  // Both decode kernels (the CUDA-core one for every cache but grouped bf16
  // queries of 2 to 8 per KV head, which run on the tensor-core kernel) keep
  // their split-K states per layer, and the CUDA-core one its pending rows: one
  // launch may walk several layers whose blocks run at their own pace.
  const bool cuda_core = !(c->dtype == DMC_BF16 && G >= 2 && G <= 8);
  o.partials = at;
  at = align_up(at + (size_t)c->num_layers * dmc::partial_states_cap(cuda_core, G) * (c->head_dim + 4) * 4);
  const size_t pend = (cuda_core && G > 1) ? (size_t)c->num_layers * NH : 0;
  o.pending = at; at = align_up(at + pend * 2 * row);
  o.pending_at = at; at = align_up(at + pend * 4);
  o.pending_z = at; at = align_up(at + pend * 4);
  o.opens = at; at = align_up(at + (size_t)c->max_prefill_tokens * c->num_kv_heads);
  o.plan = at; at = align_up(at + (size_t)c->num_kv_heads * o.plan_stride * 4);
  o.carry = at; at = align_up(at + (size_t)o.plan_stride * c->num_kv_heads * (2 * c->head_dim + 1) * 4);
  o.ring = at; at = align_up(at + (size_t)c->num_layers * NH * c->window * 2 * row);
  o.ring_w = at; at = align_up(at + (size_t)c->num_layers * NH * c->window * 4);
  o.total = at;
  return o;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

dmc_status cuda_status(cudaError_t e) { return e == cudaSuccess ? DMC_OK : DMC_ERR_CUDA; }

__global__ void lengths_copy_kernel(const Layout L, int layer, int* out) {
  const int parity = *reinterpret_cast<volatile int*>(&L.ctl[layer * 4]);
  const int* src = L.lengths + ((size_t)layer * 2 + parity) * L.NH;
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < L.NH; i += gridDim.x * blockDim.x)
    out[i] = src[i];
}

// One block per exported head; copies min(len, cap) slots as 16-byte pieces.
__global__ void export_kernel(const Layout L, int layer, const int* ids, int cap, char* kout,
                              char* vout, float* zout, int* lout) {
  const int i = blockIdx.x;
  const int bh = ids[i];
  const int parity = *reinterpret_cast<volatile int*>(&L.ctl[layer * 4]);
  if (bh < 0 || bh >= L.NH) {
    if (threadIdx.x == 0) lout[i] = -1;
    return;
  }
  const int len = L.lengths[((size_t)layer * 2 + parity) * L.NH + bh];
  if (threadIdx.x == 0) lout[i] = len;
  const int n = min(len, cap);
  const int pieces = L.row_bytes / 16;
  const int* pt = L.page_table + ((size_t)layer * L.NH + bh) * L.MPH;
  for (int x = threadIdx.x; x < n * pieces; x += blockDim.x) {
    const int s = x / pieces, p = x % pieces;
    const char* src = L.pages + (size_t)pt[s / dmc::kPage] * L.page_bytes +
                      (size_t)(s % dmc::kPage) * L.row_bytes + p * 16;
    const size_t dst = ((size_t)i * cap + s) * L.row_bytes + p * 16;
    *reinterpret_cast<uint4*>(kout + dst) = *reinterpret_cast<const uint4*>(src);
    *reinterpret_cast<uint4*>(vout + dst) =
        *reinterpret_cast<const uint4*>(src + (size_t)dmc::kPage * L.row_bytes);
  }
  for (int s = threadIdx.x; s < n; s += blockDim.x)
    zout[(size_t)i * cap + s] = L.z[(size_t)pt[s / dmc::kPage] * dmc::kPage + s % dmc::kPage];
}

}  // namespace

extern "C" {

size_t dmc_cache_required_bytes(const dmc_cache_config* cfg) {
  if (!valid_config(cfg)) return 0;
  return offsets(cfg).total;
}

dmc_status dmc_cache_create(const dmc_cache_config* cfg, void* arena_dev, size_t arena_bytes,
                            cudaStream_t stream, dmc_cache_t* out) {
  if (!out) return DMC_ERR_INVALID_ARG;
  *out = nullptr;
  if (!valid_config(cfg) || !arena_dev) return DMC_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(arena_dev) & (kAlign - 1)) != 0) return DMC_ERR_INVALID_ARG;
  const Offsets o = offsets(cfg);
  if (arena_bytes < o.total) return DMC_ERR_ARENA_TOO_SMALL;
  dmc_cache* c = new (std::nothrow) dmc_cache();
  if (!c) return DMC_ERR_INVALID_ARG;
  c->cfg = *cfg;
  char* base = static_cast<char*>(arena_dev);
  Layout& L = c->lay;
  L.L = cfg->num_layers;
  L.B = cfg->batch;
  L.Hq = cfg->num_q_heads;
  L.Hkv = cfg->num_kv_heads;
  L.G = cfg->num_q_heads / cfg->num_kv_heads;
  L.D = cfg->head_dim;
  L.esize = cfg->dtype == DMC_F32 ? 4 : 2;
  L.NH = cfg->batch * cfg->num_kv_heads;
  L.MPH = o.MPH;
  L.max_slots = cfg->max_slots_per_head;
  L.num_pages = cfg->num_pages;
  L.row_bytes = L.D * L.esize;
  L.page_bytes = 2 * dmc::kPage * L.row_bytes;
  L.pages = base + o.pages;
  L.z = reinterpret_cast<float*>(base + o.z);
  L.page_table = reinterpret_cast<int*>(base + o.ptab);
  L.lengths = reinterpret_cast<int*>(base + o.lengths);
  L.ctl = reinterpret_cast<int*>(base + o.ctl);
  L.counters = reinterpret_cast<int*>(base + o.counters);
  L.pending = base + o.pending;
  L.pending_at = reinterpret_cast<int*>(base + o.pending_at);
  L.pending_z = reinterpret_cast<float*>(base + o.pending_z);
  L.pool_top = reinterpret_cast<unsigned long long*>(base + o.pool_top);
  L.error = reinterpret_cast<unsigned int*>(base + o.error);
  L.partials = reinterpret_cast<float*>(base + o.partials);
  const bool cuda_core = !(cfg->dtype == DMC_BF16 && L.G >= 2 && L.G <= 8);
  L.partial_cap = (int)dmc::partial_states_cap(cuda_core, L.G);
  L.partials_layer_stride = (long long)L.partial_cap * (L.D + 4);
  L.opens = reinterpret_cast<unsigned char*>(base + o.opens);
  L.plan = reinterpret_cast<int*>(base + o.plan);
  L.plan_stride = o.plan_stride;
  c->carry = reinterpret_cast<float*>(base + o.carry);
  L.window = cfg->window;
  L.ring = cfg->window > 0 ? base + o.ring : nullptr;
  L.ring_w = cfg->window > 0 ? reinterpret_cast<float*>(base + o.ring_w) : nullptr;
  L.seglen = cfg->window > 0 ? reinterpret_cast<int*>(base + o.seglen) : nullptr;
  L.max_prefill_tokens = cfg->max_prefill_tokens;
  c->meta = base + o.meta;
  c->meta_bytes = o.meta_end - o.meta;
  // Grouped queries in bf16 (2 to 8 per KV head) run on the tensor-core kernel,
  // one unit list entry per KV head; otherwise every query head is its own
  // entry of the CUDA-core kernel (G = 1 for MHA).
  c->gqa = dmc::gqa_supported(L);
  c->Gv = c->gqa ? 1 : L.G;
  c->last_decode_lo = c->last_decode_hi = 0;
  cudaError_t e = cudaGetDevice(&c->device);
  if (e == cudaSuccess) e = c->gqa ? dmc::gqa_setup(L, &c->plan) : dmc::decode_setup(L, c->Gv, &c->plan);
  if (e == cudaSuccess) e = cudaMemsetAsync(c->meta, 0, c->meta_bytes, stream);
  if (e != cudaSuccess) {
    delete c;
    return DMC_ERR_CUDA;
  }
  *out = c;
  return DMC_OK;
}

// A decode launch may overlap the tail of the kernel before it on the stream
// (programmatic dependent launch) only if that kernel was this cache's decode
// of other layers: its prologue reads the first layer's slot counts, page table
// and pages, which this cache's prefill and decode of that layer write.
bool use_pdl(dmc_cache* c, int layer0, int nlayers) {
  const bool pdl = c->last_decode_hi > c->last_decode_lo &&
                   (layer0 < c->last_decode_lo || layer0 >= c->last_decode_hi);
  c->last_decode_lo = layer0;
  c->last_decode_hi = layer0 + nlayers;
  return pdl;
}
void no_pdl_next(dmc_cache* c) { c->last_decode_lo = c->last_decode_hi = 0; }

dmc_status dmc_cache_destroy(dmc_cache_t cache) {
  delete cache;
  return DMC_OK;
}

dmc_status dmc_cache_reset(dmc_cache_t c, cudaStream_t stream) {
  if (!c) return DMC_ERR_INVALID_ARG;
  no_pdl_next(c);
  return cuda_status(cudaMemsetAsync(c->meta, 0, c->meta_bytes, stream));
}

dmc_status dmc_prefill_compress(dmc_cache_t c, int32_t layer, int32_t first_seq, int32_t num_seqs,
                                const void* q_dev, int64_t q_token_stride, int64_t q_head_stride,
                                const void* k_dev, const void* v_dev, const int32_t* cu_seqlens_dev,
                                int32_t total_tokens, int32_t max_seqlen, cudaStream_t stream) {
  if (!c) return DMC_ERR_INVALID_ARG;
  const Layout& L = c->lay;
  if (layer < 0 || layer >= L.L || first_seq < 0 || num_seqs < 0 || first_seq + num_seqs > L.B)
    return DMC_ERR_INVALID_ARG;
  if (total_tokens < 0 || total_tokens > L.max_prefill_tokens || max_seqlen < 0 ||
      max_seqlen > total_tokens)
    return DMC_ERR_INVALID_ARG;
  if (num_seqs == 0 || total_tokens == 0) return DMC_OK;
  if (!q_dev || !k_dev || !v_dev || !cu_seqlens_dev || !aligned16(k_dev) || !aligned16(v_dev))
    return DMC_ERR_INVALID_ARG;
  if (q_token_stride < 0 || q_head_stride < 0) return DMC_ERR_INVALID_ARG;
  no_pdl_next(c);
  return cuda_status(dmc::prefill_launch(L, layer, first_seq, num_seqs, q_dev, q_token_stride,
                                         q_head_stride, k_dev, v_dev, cu_seqlens_dev, total_tokens,
                                         max_seqlen, nullptr, stream));
}

dmc_status dmc_prefill_attention(dmc_cache_t c, int32_t layer, int32_t first_seq,
                                 int32_t num_seqs, const void* q_dev, const void* k_dev,
                                 const void* v_dev, const int32_t* cu_seqlens_dev,
                                 int32_t total_tokens, int32_t max_seqlen, void* out_dev,
                                 cudaStream_t stream) {
  if (!c) return DMC_ERR_INVALID_ARG;
  const Layout& L = c->lay;
  if (!dmc::prefill_attn_supported(L) || L.window != 0) return DMC_ERR_INVALID_ARG;
  if (layer < 0 || layer >= L.L || first_seq < 0 || num_seqs < 0 || first_seq + num_seqs > L.B)
    return DMC_ERR_INVALID_ARG;
  if (total_tokens < 0 || total_tokens > L.max_prefill_tokens || max_seqlen < 0 ||
      max_seqlen > total_tokens)
    return DMC_ERR_INVALID_ARG;
  if (num_seqs == 0 || total_tokens == 0) return DMC_OK;
  if (!q_dev || !k_dev || !v_dev || !cu_seqlens_dev || !out_dev || !aligned16(q_dev) ||
      !aligned16(k_dev) || !aligned16(v_dev) || !aligned16(out_dev))
    return DMC_ERR_INVALID_ARG;
  no_pdl_next(c);
  const long long q_tok = (long long)L.Hq * L.D, q_head = L.D;
  cudaError_t e = dmc::prefill_launch(L, layer, first_seq, num_seqs, q_dev, q_tok, q_head, k_dev,
                                      v_dev, cu_seqlens_dev, total_tokens, max_seqlen, c->carry,
                                      stream);
  if (e != cudaSuccess) return DMC_ERR_CUDA;
  return cuda_status(dmc::prefill_attn_launch(L, layer, first_seq, num_seqs, q_dev, k_dev, v_dev,
                                              cu_seqlens_dev, total_tokens, max_seqlen, c->carry,
                                              out_dev, stream));
}

dmc_status dmc_decode_step(dmc_cache_t c, int32_t layer, const void* q_dev, const void* k_dev,
                           const void* v_dev, void* out_dev, cudaStream_t stream) {
  if (!c) return DMC_ERR_INVALID_ARG;
  const Layout& L = c->lay;
  if (layer < 0 || layer >= L.L) return DMC_ERR_INVALID_ARG;
  if (!aligned16(q_dev) || !aligned16(k_dev) || !aligned16(v_dev) || !aligned16(out_dev) ||
      !q_dev || !k_dev || !v_dev || !out_dev)
    return DMC_ERR_INVALID_ARG;
  const bool pdl = use_pdl(c, layer, 1);
  if (c->gqa)
    return cuda_status(dmc::gqa_launch(L, layer, 1, c->plan, pdl, q_dev, k_dev, v_dev, out_dev, stream));
  return cuda_status(dmc::decode_launch(L, layer, 1, c->Gv, c->plan, pdl, q_dev, k_dev, v_dev,
                                        out_dev, stream));
}

dmc_status dmc_decode_step_layers(dmc_cache_t c, int32_t first_layer, int32_t num_layers,
                                  const void* q_dev, const void* k_dev, const void* v_dev,
                                  void* out_dev, cudaStream_t stream) {
  if (!c) return DMC_ERR_INVALID_ARG;
  const Layout& L = c->lay;
  if (first_layer < 0 || num_layers < 0 || first_layer + num_layers > L.L) return DMC_ERR_INVALID_ARG;
  if (num_layers == 0) return DMC_OK;
  if (!aligned16(q_dev) || !aligned16(k_dev) || !aligned16(v_dev) || !aligned16(out_dev) ||
      !q_dev || !k_dev || !v_dev || !out_dev)
    return DMC_ERR_INVALID_ARG;
  const bool pdl = use_pdl(c, first_layer, num_layers);
  if (c->gqa)
    return cuda_status(dmc::gqa_launch(L, first_layer, num_layers, c->plan, pdl, q_dev, k_dev, v_dev,
                                       out_dev, stream));
  return cuda_status(dmc::decode_launch(L, first_layer, num_layers, c->Gv, c->plan, pdl, q_dev,
                                        k_dev, v_dev, out_dev, stream));
}

dmc_status dmc_decode_step_static_scratch(dmc_cache_t c, int32_t layer, const void* q_dev,
                                          const void* k_dev, const void* v_dev, void* out_dev,
                                          cudaStream_t stream) {
  if (!c) return DMC_ERR_INVALID_ARG;
  const Layout& L = c->lay;
  if (layer < 0 || layer >= L.L) return DMC_ERR_INVALID_ARG;
  if (!aligned16(q_dev) || !aligned16(k_dev) || !aligned16(v_dev) || !aligned16(out_dev) ||
      !q_dev || !k_dev || !v_dev || !out_dev)
    return DMC_ERR_INVALID_ARG;
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return DMC_ERR_CUDA;
  if (dev != c->device) return DMC_ERR_INVALID_ARG;
  float* scratch = nullptr;
  size_t floats = 0;
  e = dmc::decode_static_partials(dev, &scratch, &floats);
  if (e != cudaSuccess) return DMC_ERR_CUDA;
  // One launch writes two partial states per worker warp: of head_dim + 4
  // floats for the CUDA-core kernel (6 warps per block), and one per query
  // of the group, of head_dim + 2 floats, for the tensor-core kernel (4 warps
  // per block). A grid that needs more than the array holds is cut to fit;
  // the work split follows the grid, so results differ from dmc_decode_step's
  // only by the order of the split-K sums.
  const size_t state_floats = (size_t)L.D + (c->gqa ? 2 : 4);
  const size_t per_block = (size_t)2 * (c->gqa ? dmc::kGqaWarpsPerBlock : dmc::kDecodeWarpsPerBlock) *
                           (c->gqa ? L.G : 1);
  const size_t fit_blocks = floats / state_floats / per_block;
  if (fit_blocks < 1) return DMC_ERR_INVALID_ARG;
  dmc::DecodePlan plan = c->plan;
  if ((size_t)plan.grid > fit_blocks) plan.grid = (int)fit_blocks;
  plan.partial_states = (int)(per_block * plan.grid);
  Layout ls = L;
  ls.partials = scratch;
  ls.partial_cap = (int)(floats / state_floats);
  ls.partials_layer_stride = 0;  // one layer per launch here
  const bool pdl = use_pdl(c, layer, 1);
  if (c->gqa)
    return cuda_status(dmc::gqa_launch(ls, layer, 1, plan, pdl, q_dev, k_dev, v_dev, out_dev, stream));
  return cuda_status(dmc::decode_launch(ls, layer, 1, c->Gv, plan, pdl, q_dev, k_dev, v_dev,
                                        out_dev, stream));
}

dmc_status dmc_cache_lengths(dmc_cache_t c, int32_t layer, int32_t* out_dev, cudaStream_t stream) {
  if (!c || !out_dev || layer < 0 || layer >= c->lay.L) return DMC_ERR_INVALID_ARG;
  const int threads = 256, blocks = dmc::ceil_div(c->lay.NH, threads);
  lengths_copy_kernel<<<blocks, threads, 0, stream>>>(c->lay, layer, out_dev);
  return cuda_status(cudaGetLastError());
}

dmc_status dmc_cache_export_heads(dmc_cache_t c, int32_t layer, int32_t n,
                                  const int32_t* head_ids_dev, int32_t cap, void* k_out_dev,
                                  void* v_out_dev, float* z_out_dev, int32_t* len_out_dev,
                                  cudaStream_t stream) {
  if (!c || layer < 0 || layer >= c->lay.L || n < 0 || cap < 0) return DMC_ERR_INVALID_ARG;
  if (n == 0) return DMC_OK;
  if (!head_ids_dev || !k_out_dev || !v_out_dev || !z_out_dev || !len_out_dev ||
      !aligned16(k_out_dev) || !aligned16(v_out_dev))
    return DMC_ERR_INVALID_ARG;
  export_kernel<<<n, 256, 0, stream>>>(c->lay, layer, head_ids_dev, cap,
                                       static_cast<char*>(k_out_dev),
                                       static_cast<char*>(v_out_dev), z_out_dev, len_out_dev);
  return cuda_status(cudaGetLastError());
}

dmc_status dmc_cache_status(dmc_cache_t c, cudaStream_t stream, uint32_t* bits,
                            int64_t* pages_used) {
  if (!c) return DMC_ERR_INVALID_ARG;
  uint32_t b = 0;
  unsigned long long top = 0;
  cudaError_t e = cudaStreamSynchronize(stream);
  if (e == cudaSuccess) e = cudaMemcpy(&b, c->lay.error, 4, cudaMemcpyDeviceToHost);
  if (e == cudaSuccess) e = cudaMemcpy(&top, c->lay.pool_top, 8, cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return DMC_ERR_CUDA;
  if (bits) *bits = b;
  if (pages_used) *pages_used = (int64_t)top;
  if (b & DMC_FAULT_PAGES_EXHAUSTED) return DMC_ERR_PAGES_EXHAUSTED;
  if (b) return DMC_ERR_DEVICE_FAULT;
  return DMC_OK;
}

const char* dmc_status_string(dmc_status s) {
  switch (s) {
    case DMC_OK: return "ok";
    case DMC_ERR_INVALID_ARG: return "invalid argument";
    case DMC_ERR_ARENA_TOO_SMALL: return "arena too small";
    case DMC_ERR_PAGES_EXHAUSTED: return "page pool exhausted";
    case DMC_ERR_CUDA: return "CUDA runtime error";
    case DMC_ERR_DEVICE_FAULT: return "device fault";
  }
  return "unknown status";
}

}  // extern "C"
