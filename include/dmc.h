/*
 * dmc.h -- C ABI of the Dynamic Memory Compression hot path on one GPU (sm_103a).
 *
 * Dynamic Memory Compression (Nawrot et al., "Dynamic Memory Compression:
 * Retrofitting LLMs for Accelerated Inference", ICML 2024, arXiv 2403.09636)
 * keeps, per layer and per KV head, a variable-length cache of slots. For
 * every new token t (Eq. reuse, Algorithm 1):
 *   alpha_t = round(sigmoid(k_t[0]))  -> computed here as k_t[0] >= 0
 *   omega_t = sigmoid(q_t[0])         (grouped queries: of the group's mean q[0])
 *   k_t[0] = q_t[0] = 0
 *   alpha_t = 1: the last slot becomes the omega-weighted running mean,
 *                K_l <- (K_l z + k_t omega)/(z + omega), V_l likewise, z += omega
 *   alpha_t = 0: (k_t, v_t) open a new slot with z = omega
 * and the token's queries attend (Eq. attn-softmax, scale 1/sqrt(d_h)) over the
 * updated slots of their KV head. The first token of an empty head always opens
 * a slot (initial conditions of Eq. partial-accumulation).
 *
 * Conventions for every call below:
 *  - Pointers named *_dev are device pointers; all tensors are row-major and
 *    contiguous unless a stride is given, in the cache's dtype (float or
 *    bfloat16), and 16-byte aligned. The caller owns every buffer, including the
 *    arena that holds the cache; the library allocates no device memory.
 *  - Calls are asynchronous on the given stream and return launch-time status.
 *    All calls on one cache must be ordered on the GPU (one stream, or explicit
 *    events): they share the cache's scratch space.
 *  - Faults found on the device (page pool exhausted, a head over its slot
 *    capacity, a NaN gate, inconsistent cu_seqlens, a wait that timed out) set
 *    sticky bits that dmc_cache_status reports; the kernels skip the faulty
 *    write and never trap. Results after a fault are unspecified.
 *  - Inputs are const: the library never writes q[0] or k[0] of caller buffers.
 */
#ifndef DMC_H_
#define DMC_H_

#include <stddef.h>
#include <stdint.h>

#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  DMC_OK = 0,
  DMC_ERR_INVALID_ARG = 1,      /* bad config, pointer, alignment or size */
  DMC_ERR_ARENA_TOO_SMALL = 2,  /* arena_bytes < dmc_cache_required_bytes */
  DMC_ERR_PAGES_EXHAUSTED = 3,  /* sticky: the page pool ran out */
  DMC_ERR_CUDA = 4,             /* a CUDA runtime call failed */
  DMC_ERR_DEVICE_FAULT = 5      /* sticky: another device fault bit is set */
} dmc_status;

typedef enum { DMC_F32 = 0, DMC_BF16 = 1 } dmc_dtype;

/* Sticky device fault bits returned by dmc_cache_status. */
#define DMC_FAULT_PAGES_EXHAUSTED 0x1u  /* no free page for a new slot */
#define DMC_FAULT_SLOT_CAPACITY 0x2u    /* a head would exceed max_slots_per_head */
#define DMC_FAULT_NAN_GATE 0x4u         /* k[0] was NaN (treated as append) */
#define DMC_FAULT_BAD_SEQLENS 0x8u      /* cu_seqlens not monotone / out of range */
#define DMC_FAULT_WAIT_TIMEOUT 0x10u    /* an in-kernel wait gave up (kernel returned) */

/* Shape of one cache. Storage is paged (the paper stores its variable-length
 * heads with PagedAttention, 32 slots per page, pages allocated on demand per
 * head; Sec. 3.3 "Storing a variable-length KV cache" and the throughput
 * section). One page holds 32 key rows then 32 value rows of head_dim
 * elements, plus 32 fp32 z values kept beside the pool. */
typedef struct {
  int32_t num_layers;
  int32_t batch;               /* sequences */
  int32_t num_q_heads;         /* query heads per layer */
  int32_t num_kv_heads;        /* KV heads per layer; num_q_heads % num_kv_heads == 0 */
  int32_t head_dim;            /* 64 or 128 */
  int32_t dtype;               /* dmc_dtype of slots, q, k, v and outputs */
  int32_t page_size;           /* slots per page; must be 32 */
  int32_t max_slots_per_head;  /* slot capacity of one head (page-table width) */
  int64_t num_pages;           /* pages in the pool shared by all layers and heads */
  int32_t max_prefill_tokens;  /* largest total_tokens of one dmc_prefill_compress */
  int32_t window;              /* 0: DMC as in Algorithm 1. w in [1, 32]: the window-
                                  grouping approximation (Sec. 3.3): a slot is the
                                  omega-weighted mean of the last min(segment length,
                                  w) tokens of its segment; each head then keeps its
                                  open segment's last tokens (the window cache). */
} dmc_cache_config;

typedef struct dmc_cache* dmc_cache_t;

/* Bytes of device memory a cache with this config needs (0 if invalid). */
size_t dmc_cache_required_bytes(const dmc_cache_config* cfg);

/* Lays the cache out inside the caller's device arena (256-byte aligned,
 * arena_bytes >= dmc_cache_required_bytes) and clears its lengths on `stream`.
 * The arena must stay allocated until dmc_cache_destroy. The handle remembers
 * the current device; later calls must run with that device current. */
dmc_status dmc_cache_create(const dmc_cache_config* cfg, void* arena_dev, size_t arena_bytes,
                            cudaStream_t stream, dmc_cache_t* out);

/* Frees the host-side handle (the arena stays the caller's). NULL is a no-op. */
dmc_status dmc_cache_destroy(dmc_cache_t cache);

/* Empties every head of every layer, returns all pages to the pool and clears
 * the fault bits (asynchronous on `stream`). */
dmc_status dmc_cache_reset(dmc_cache_t cache, cudaStream_t stream);

/* Prompt-phase compression (the paper notes Algorithm 1's savings apply to the
 * prompt too, Sec. 3.3 "Window grouping approximation"): runs Algorithm 1 over
 * the prompt tokens of `num_seqs` sequences [first_seq, first_seq + num_seqs)
 * of one layer, without attention. Computed in closed form: with binary alpha,
 * Eq. partial-accumulation makes every slot the omega-weighted mean of one
 * segment of tokens (a segment opens at a token with alpha = 0 or at the first
 * token of an empty head), z = the segment's summed omega. A head that already
 * holds slots continues its last segment, exactly as token-by-token decoding.
 *   q_dev: element (t, j) of the queries' first components is read at
 *          q_dev[t * q_token_stride + j * q_head_stride] (elements; only q[.,0]
 *          is used, so a packed [total_tokens, num_q_heads] array works);
 *   k_dev, v_dev: [total_tokens, num_kv_heads, head_dim], sequences packed;
 *   cu_seqlens_dev: int32 [num_seqs + 1], cu_seqlens[0] = 0,
 *          cu_seqlens[num_seqs] = total_tokens;
 *   max_seqlen: an upper bound of every cu_seqlens[i+1] - cu_seqlens[i].
 * total_tokens <= max_prefill_tokens. Reads each k/v row once. */
dmc_status dmc_prefill_compress(dmc_cache_t cache, int32_t layer, int32_t first_seq,
                                int32_t num_seqs, const void* q_dev, int64_t q_token_stride,
                                int64_t q_head_stride, const void* k_dev, const void* v_dev,
                                const int32_t* cu_seqlens_dev, int32_t total_tokens,
                                int32_t max_seqlen, cudaStream_t stream);

/* dmc_prefill_compress plus the attention output of every prompt token.
 * At inference a prompt token attends over the cache as it stands right after
 * its own update (Eq. attn-softmax over the compressed slots; the training
 * mask of Sec. 3.2 with binary alpha gives the same pattern): the final values
 * of the slots closed before it, and the slot it has just merged into or
 * opened, whose value at that moment is the running omega-weighted mean of its
 * segment (Eq. partial-accumulation). The cache afterwards is exactly as after
 * dmc_prefill_compress of the same prompt; a head that already holds slots
 * continues its last segment, so splitting a prompt over calls gives the same
 * outputs. The score is q[1:]^T k[1:] / sqrt(head_dim) (q[0] and k[0] are the
 * gates). Runs on the tcgen05 tensor cores: bf16 caches with head_dim 128 and
 * 1, 2, 4 or 8 query heads per KV head, exact compression (window = 0); other
 * caches return DMC_ERR_INVALID_ARG.
 *   q_dev:   [total_tokens, num_q_heads, head_dim], packed (q[., ., 0] also
 *            gives omega, as in dmc_prefill_compress);
 *   k_dev, v_dev: [total_tokens, num_kv_heads, head_dim], sequences packed;
 *   cu_seqlens_dev, total_tokens, max_seqlen: as in dmc_prefill_compress;
 *   out_dev: [total_tokens, num_q_heads, head_dim] (written, bf16).
 * All device pointers 16-byte aligned. Asynchronous on `stream`; device faults
 * (capacity, pool, bad cu_seqlens, a wait that gave up) set the sticky bits
 * read by dmc_cache_status. */
dmc_status dmc_prefill_attention(dmc_cache_t cache, int32_t layer, int32_t first_seq,
                                 int32_t num_seqs, const void* q_dev, const void* k_dev,
                                 const void* v_dev, const int32_t* cu_seqlens_dev,
                                 int32_t total_tokens, int32_t max_seqlen, void* out_dev,
                                 cudaStream_t stream);

/* One decode step of one layer for all `batch` sequences: Algorithm 1 on the
 * new token of every KV head (append or accumulate, fused), then every query
 * head attends over its KV head's updated slots (split across thread blocks
 * by slot ranges, merged with an online softmax).
 *   q_dev:   [batch, num_q_heads, head_dim]
 *   k_dev, v_dev: [batch, num_kv_heads, head_dim]
 *   out_dev: [batch, num_q_heads, head_dim] (written)
 */
dmc_status dmc_decode_step(dmc_cache_t cache, int32_t layer, const void* q_dev,
                           const void* k_dev, const void* v_dev, void* out_dev,
                           cudaStream_t stream);

/* dmc_decode_step for the layers [first_layer, first_layer + num_layers) in
 * one launch, when the inputs of all of them are ready (the step of each layer
 * reads only that layer's cache and inputs, Algorithm 1 and Eq. attn-softmax
 * per KV head, so the layers are independent). Same slots and lengths for
 * every layer as calling dmc_decode_step on the layers in order, and the same
 * outputs up to the order of the split-K sums: the CUDA-core kernel runs more
 * warps per block over several layers than over one, so a head may be split
 * over other warps (outputs are bit-identical when neither grid splits a head,
 * and always for the tensor-core kernel). What it saves is one launch and one
 * kernel start-up and tail per layer, which dominate small caches.
 *   q_dev:   [num_layers, batch, num_q_heads, head_dim]
 *   k_dev, v_dev: [num_layers, batch, num_kv_heads, head_dim]
 *   out_dev: [num_layers, batch, num_q_heads, head_dim] (written)
 * Both decode kernels (the CUDA-core one and the tensor-core one for grouped
 * bf16 queries of 2 to 8 per KV head) walk the layers in one launch.
 * num_layers = 0 is a no-op. */
dmc_status dmc_decode_step_layers(dmc_cache_t cache, int32_t first_layer, int32_t num_layers,
                                  const void* q_dev, const void* k_dev, const void* v_dev,
                                  void* out_dev, cudaStream_t stream);

/* dmc_decode_step with its scratch in the library's own static device memory.
 * The paper has no counterpart; this exists for callers that cannot allocate
 * device memory of their own: a plugin or custom operator that a host
 * framework hands only its input and output buffers (the framework owns every
 * allocation), or a latency-critical loop that must not pay cudaMalloc's
 * implicit device synchronisation. Same arguments and semantics as
 * dmc_decode_step; it allocates nothing and calls no allocating routine.
 * The scratch is the split-K partial softmax states of one launch, kept in a
 * file-scope __device__ array of 8 MiB (2,097,152 floats) that every GPU
 * loading the library holds until the process exits. One launch needs
 *   2 * grid * 6 states of head_dim + 4 floats   (CUDA-core kernel: MHA, fp32,
 *                                                 groups above 8), or
 *   2 * grid * 4 * G states of head_dim + 2 floats (tensor-core kernel: bf16
 *                                                 groups of 2 to 8 queries),
 * grid being the cache's decode grid (at most one or two blocks per SM). Every
 * MHA grid fits; a tensor-core grid of group 8 and head_dim 128 fits up to 252
 * blocks (a GB300 runs 152). A grid that does not fit is cut to the blocks
 * that do: the work split follows the grid, so the results then differ from
 * dmc_decode_step's only by the rounding of the split-K sums; when it fits,
 * they are bit-identical. Nothing in the array needs to start at zero: each
 * launch writes every state before reading it. The first call on a device
 * looks up the array's device address on that device (which must be current
 * and be the cache's device) and keeps it for the life of the process, so the
 * device must not be reset (cudaDeviceReset) after that call, and the first
 * call should come before any stream capture. All calls share the one array,
 * so calls whose launches overlap on the GPU (any caches, any streams) race
 * and must be ordered by the caller. */
dmc_status dmc_decode_step_static_scratch(dmc_cache_t cache, int32_t layer, const void* q_dev,
                                          const void* k_dev, const void* v_dev, void* out_dev,
                                          cudaStream_t stream);

/* Copies the slot count of every head of `layer`, int32 [batch, num_kv_heads],
 * into out_dev (asynchronous). */
dmc_status dmc_cache_lengths(dmc_cache_t cache, int32_t layer, int32_t* out_dev,
                             cudaStream_t stream);

/* Copies the slots of n heads (head_ids_dev[i] = seq * num_kv_heads + kv_head)
 * of `layer` into dense buffers (asynchronous; for tests and inspection):
 *   k_out_dev, v_out_dev: [n, cap, head_dim] in the cache dtype;
 *   z_out_dev: float [n, cap]; len_out_dev: int32 [n] (the full length, even
 *   when it exceeds cap; only min(len, cap) slots are copied). */
dmc_status dmc_cache_export_heads(dmc_cache_t cache, int32_t layer, int32_t n,
                                  const int32_t* head_ids_dev, int32_t cap, void* k_out_dev,
                                  void* v_out_dev, float* z_out_dev, int32_t* len_out_dev,
                                  cudaStream_t stream);

/* Synchronizes `stream`, then reads the sticky fault bits (into *bits if not
 * NULL) and the number of pool pages handed out so far (into *pages_used if
 * not NULL). Returns DMC_OK, DMC_ERR_PAGES_EXHAUSTED or DMC_ERR_DEVICE_FAULT. */
dmc_status dmc_cache_status(dmc_cache_t cache, cudaStream_t stream, uint32_t* bits,
                            int64_t* pages_used);

/* Static description of a status code. */
const char* dmc_status_string(dmc_status status);

#ifdef __cplusplus
}
#endif

#endif /* DMC_H_ */
