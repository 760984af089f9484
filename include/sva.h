/*
 * sva.h -- streaming video attention: policy-indexed chunk-causal attention
 * over a (chunk, level)-indexed KV cache, with a fused 3D-RoPE + cache
 * scatter, for one GB300 GPU (sm_103a).
 *
 * Method: "Rethinking Streaming Video Diffusion Model: Context, Execution,
 * and Training", Section 3.  A *node* (b, j) is chunk b of the video at
 * denoising level j in {0..K} (j = K pure noise, j = 0 clean; Section 3.1).
 * A context policy phi picks, for every history offset r in
 * {1..min(W, b-1)}, the level of chunk b-r the node reads (Eq. 2-3); the
 * node's queries then attend over its own chunk (bidirectionally) plus the
 * cached keys/values of those states, everything else masked with -inf
 * (Eq. 4).  Several nodes of one pipeline round (Eq. 6) are processed by one
 * launch, which is how progressive history is executed (Section 3.3).
 * Around that: the input projection producing q, k, v (sva_qkv_project), the
 * RoPE + cache write (sva_rope_kv_write), a block-sparse form of the token
 * mask of Eq. 4 (sva_attend_nodes_sparse) and its token-level form on the
 * own chunk and on the history (sva_attend_nodes_masked).
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * - Every device buffer is owned by the caller: the cache buffer handed to
 *   sva_cache_create and every Q/K/V/O/LSE tensor.  The library owns only
 *   the opaque sva_cache object (host slot table and cached TMA
 *   descriptors), freed by sva_destroy.  The library never allocates device
 *   memory.
 * - Tensors are dense, row-major, bf16 unless stated, 16-byte aligned.
 *   Token-major activations are [n_nodes][T][H][d] with T = F*Hp*Wp tokens
 *   per chunk, token u = (f*Hp + h)*Wp + w.
 * - Calls that take a stream validate on the host, enqueue on that stream and
 *   return; nothing is launched when validation fails.  Device-side errors
 *   (a bounded wait inside a kernel that timed out) are reported later by
 *   sva_poll_device_status.
 * - On failure a call returns a non-zero sva_status and sets a thread-local
 *   message readable with sva_last_error().
 * - One cache is used from one host thread and one stream at a time.
 */
#ifndef SVA_H_
#define SVA_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  SVA_OK = 0,
  SVA_ERR_INVALID_ARGUMENT = 1, /* null/misaligned pointer, bad size, bad id */
  SVA_ERR_NOT_RESIDENT = 2,     /* a (seq, chunk, level) state is not in the cache */
  SVA_ERR_CAUSALITY = 3,        /* a context state is not in the node's past (Eq. 4) */
  SVA_ERR_CAPACITY = 4,         /* too many nodes/contexts/slots, position beyond the table */
  SVA_ERR_UNSUPPORTED = 5,      /* geometry the kernels do not implement */
  SVA_ERR_CUDA = 6,             /* a CUDA runtime/driver call failed */
  SVA_ERR_DEVICE_TIMEOUT = 7,   /* a kernel's bounded wait expired */
  SVA_ERR_UNAVAILABLE = 8       /* a selected level not yet reached by the pipeline (Eq. 7) */
} sva_status;

/* Context policies, Eq. 3 (Section 3.2). */
enum {
  SVA_POLICY_CLEAN = 0, /* phi(j, r) = 0 */
  SVA_POLICY_SAME = 1,  /* phi(j, r) = j */
  SVA_POLICY_PROG = 2   /* phi(j, r) = max(j - r, 0) */
};

/* Visibility inside a node's own chunk (Eq. 4, Section 3.2: attention within
 * the current chunk "may be bidirectional"). */
enum {
  SVA_WITHIN_BIDIRECTIONAL = 0, /* every own-chunk key visible to every query */
  SVA_WITHIN_FRAME_CAUSAL = 1   /* a query of latent frame f sees own-chunk keys of frames <= f */
};

#define SVA_MAX_CTX 16   /* history states one node may read */
#define SVA_MAX_NODES 64 /* nodes in one sva_rope_kv_write / sva_attend_nodes call */

typedef struct sva_cache sva_cache;
typedef struct CUstream_st* sva_stream; /* a cudaStream_t; NULL = legacy default stream */

/* Geometry of the chunks and of the KV cache.
 *   num_heads   H, 1..128
 *   head_dim    d, 64 or 128
 *   frames      F latent frames per chunk; grid_h x grid_w patches per frame
 *               (T = F*grid_h*grid_w tokens per chunk, 1..65536)
 *   num_slots   number of (chunk, level) states the cache holds at once
 *   rope_pairs  head-dimension pairs rotated by the t, h and w positions;
 *               they must sum to d/2 (3D RoPE reading: the paper does not name
 *               a positional encoding)
 *   max_frames  absolute latent-frame positions covered by the RoPE table:
 *               every written chunk b needs F*b + F - 1 < max_frames
 *   rope_theta  RoPE base (10000 in the usual convention)              */
typedef struct {
  int32_t num_heads;
  int32_t head_dim;
  int32_t frames;
  int32_t grid_h;
  int32_t grid_w;
  int32_t num_slots;
  int32_t rope_pairs[3];
  int32_t max_frames;
  double rope_theta;
} sva_geometry;

/* One denoising node of a launch (Section 3.1-3.3).
 *   seq          independent video stream the node belongs to (stream
 *                batching); contexts must come from the same seq
 *   chunk, level the node (b, j)
 *   own_slot     cache slot bound to (seq, chunk, level); written by
 *                sva_rope_kv_write, always visible to the node itself
 *   within       SVA_WITHIN_BIDIRECTIONAL or SVA_WITHIN_FRAME_CAUSAL; the
 *                history states are always wholly visible
 *   n_ctx        number of history states read, 0..SVA_MAX_CTX
 *   ctx_slot     their cache slots (e.g. from sva_select_context +
 *                sva_cache_lookup), each of a chunk < `chunk`
 *   ctx_visible  Eq. 4 at state granularity: 1 = mask 0 on that state's
 *                tokens, 0 = mask -inf (the state is skipped)           */
typedef struct {
  int32_t seq;
  int32_t chunk;
  int32_t level;
  int32_t own_slot;
  int32_t within;
  int32_t n_ctx;
  int32_t ctx_slot[SVA_MAX_CTX];
  uint8_t ctx_visible[SVA_MAX_CTX];
} sva_node;

/* Bytes of device memory the cache needs for `g`: the slot pool
 * [num_slots][2 (K, V)][H][Tpad][d] bf16 with Tpad = T rounded up to 128,
 * the RoPE cos/sin tables (the patch-row and patch-column ones also stored
 * pair-major) and a status word.  0 if `g` is invalid. */
size_t sva_cache_bytes(const sva_geometry* g);

/* Creates a cache over the caller's device buffer `dev_buf` (at least
 * sva_cache_bytes(g) bytes, 256-byte aligned, on the current device).
 * Zeroes the pad rows and the status word, uploads the RoPE tables, and
 * builds the TMA descriptor of the slot pool.  Synchronous.  The buffer must
 * outlive the cache.  Errors: INVALID_ARGUMENT, UNSUPPORTED, CUDA. */
sva_status sva_cache_create(const sva_geometry* g, void* dev_buf, size_t bytes, sva_cache** out);

/* Binds a free slot to state (seq, chunk, level) (the KV cache of
 * Section 3.2, indexed by chunk and level).  The slot is not resident until
 * sva_rope_kv_write has written it.  Errors: INVALID_ARGUMENT (level < 0 or
 * the state is already bound), CAPACITY (no free slot). */
sva_status sva_cache_bind(sva_cache* c, int32_t seq, int32_t chunk, int32_t level, int32_t* slot);

/* Slot bound to (seq, chunk, level).  Errors: NOT_RESIDENT if unbound. */
sva_status sva_cache_lookup(const sva_cache* c, int32_t seq, int32_t chunk, int32_t level,
                            int32_t* slot);

/* Frees the slot of (seq, chunk, level) (rolling window).  Host-side only:
 * the caller must not release a slot that a queued kernel still reads.
 * Errors: NOT_RESIDENT if unbound. */
sva_status sva_cache_release(sva_cache* c, int32_t seq, int32_t chunk, int32_t level);

/* Eq. 2-3 (Section 3.2) with the full offset window R = {1..min(W, b-1)}:
 * writes (chunk - r, phi(level, r)) for r = 1.. into chunks/levels, in order
 * of increasing r, and their number into *n.  Chunks are numbered from 1 as
 * in the paper.  Errors: INVALID_ARGUMENT (unknown policy, K < 1,
 * level outside 0..K, W < 0, null pointers), CAPACITY (cap too small). */
sva_status sva_select_context(int32_t policy, int32_t K, int32_t W, int32_t chunk, int32_t level,
                              int32_t cap, int32_t* chunks, int32_t* levels, int32_t* n);

/* Eq. 6 (Section 3.3): the states [x_n^K, x_{n-1}^{K-1}, ..., x_{n-K+1}^1]
 * active at the start of round n of a pipeline over chunks 1..B, chunks
 * outside 1..B left out.  Writes them (levels K down to 1) and their number.
 * Errors: INVALID_ARGUMENT, CAPACITY (cap < number of states). */
sva_status sva_pipeline_round(int32_t K, int32_t B, int32_t round, int32_t cap, int32_t* chunks,
                              int32_t* levels, int32_t* count);

/* Eq. 7 (Section 3.3): checks that every state (chunks[i], levels[i]) a node
 * (chunk, level) of a K-level pipeline reads has been reached, i.e.
 * levels[i] >= max(level - r, 0) with r = chunk - chunks[i] >= 1.
 * Returns OK, UNAVAILABLE (first violation named in sva_last_error), or
 * INVALID_ARGUMENT / CAUSALITY for malformed lists. */
sva_status sva_check_pipeline(int32_t K, int32_t level, int32_t chunk, int32_t n,
                              const int32_t* chunks, const int32_t* levels);

/* Applies 3D RoPE to each node's new keys (and, if q_inout is not NULL, to
 * its queries, in place) at the node's absolute positions (F*chunk + f, h, w)
 * and scatters K' and the unrotated V into the node's own slot (the cache
 * write that makes the node's features available to later reads and to
 * in-round progressive reads, Section 3.3).  Marks the own slots resident.
 *   k_new, v_new, q_inout: [n_nodes][T][H][d] bf16, node i = nodes[i].
 * Stream-ordered.  Errors: INVALID_ARGUMENT (null/misaligned pointer,
 * unbound or mismatched own_slot, duplicate own_slot), CAPACITY
 * (n_nodes > SVA_MAX_NODES, position beyond max_frames), CUDA. */
sva_status sva_rope_kv_write(sva_cache* c, const sva_node* nodes, int32_t n_nodes,
                             const void* k_new, const void* v_new, void* q_inout, sva_stream s);

/* sva_rope_kv_write with an RMS normalisation of each token's key (and query)
 * vector in front of the rotation, fused in the same pass (reading: the paper
 * names no normalisation; Wan-style DiTs normalise q and k this way before
 * RoPE).  For a token's K row x of H*d elements:
 *   x' = x * gamma_k / sqrt(mean(x^2) + eps),
 * then RoPE; likewise Q with gamma_q; V is copied unchanged.  fp32 arithmetic,
 * one bf16 rounding of the rotated result.
 *   gamma_k, gamma_q: fp32 [H*d] device vectors, 16-byte aligned (gamma_q may
 *   be NULL when q_inout is NULL); eps > 0.
 * Errors: as sva_rope_kv_write, plus INVALID_ARGUMENT for bad gammas or eps. */
sva_status sva_rope_kv_write_qknorm(sva_cache* c, const sva_node* nodes, int32_t n_nodes,
                                    const void* k_new, const void* v_new, void* q_inout,
                                    const float* gamma_k, const float* gamma_q, float eps,
                                    sva_stream s);

/* The linear projection in front of the attention layer, producing the
 * token-major inputs of sva_rope_kv_write (the paper's denoiser is a DiT
 * whose attention layers take q, k, v from the token features; Section 3.2
 * reads K and V from them; the layer itself is not spelled out):
 *   [q | k | v] = x W^T + b,  q, k, v each [rows][H*d] = [rows][H][d],
 * with H, d from the cache's geometry.  bf16 operands, fp32 accumulation on
 * the tensor cores, bias added in fp32, one bf16 rounding per output.
 *   x       [rows][in_features] bf16 (e.g. rows = n_nodes * T token features)
 *   weight  [3*H*d][in_features] bf16, out_features x in_features: q's output
 *           rows first, then k's, then v's
 *   bias    [3*H*d] fp32, or NULL
 *   q, k, v [rows][H*d] bf16 outputs
 * in_features a positive multiple of 8; H*d a multiple of 128; every pointer
 * 16-byte aligned and in device memory of the cache's device (a host or
 * another GPU's pointer is rejected with INVALID_ARGUMENT before anything is
 * launched).  Runs on pairs of CTAs (clusters of two) with two-SM MMAs;
 * each CTA loads its own operand tiles from this GPU's memory (no copy
 * writes more than one CTA).  Stream-ordered; a device timeout is
 * reported by sva_poll_device_status.  Errors: INVALID_ARGUMENT,
 * UNSUPPORTED (H*d), CUDA. */
sva_status sva_qkv_project(sva_cache* c, const void* x, int32_t rows, int32_t in_features,
                           const void* weight, const float* bias, void* q, void* k, void* v,
                           sva_stream s);

/* sva_qkv_project with the RoPE + cache write of sva_rope_kv_write fused into
 * its epilogue (no normalisation), for the token rows of n_nodes nodes:
 * rows = n_nodes * T, node i's tokens at rows [i*T, (i+1)*T) of x.
 *   [q | k | v] = x W^T + b        (fp32 accumulators, bias added in fp32)
 * then q and k of each token are rotated by the 3D RoPE at its absolute
 * position (F*chunk + f, h, w) in fp32 and rounded to bf16 once; Q' goes to
 * q_out and K' with the unrotated V into each node's own slot, which is
 * marked resident.  The result equals sva_qkv_project followed by
 * sva_rope_kv_write up to the intermediate bf16 rounding of q and k, which
 * this call does not make.
 *   nodes   as for sva_rope_kv_write (own_slot bound to (seq, chunk, level),
 *           distinct own slots, n_nodes <= SVA_MAX_NODES)
 *   x       [n_nodes*T][in_features] bf16; weight, bias as sva_qkv_project
 *   q_out   [n_nodes][T][H][d] bf16
 * Stream-ordered.  Errors: those of sva_qkv_project and sva_rope_kv_write. */
sva_status sva_qkv_project_rope(sva_cache* c, const sva_node* nodes, int32_t n_nodes,
                                const void* x, int32_t in_features, const void* weight,
                                const float* bias, void* q_out, sva_stream s);

/* Policy-indexed chunk-causal attention (Eq. 4) for a batch of nodes:
 *   out[i][u][h] = sum_v softmax_v(scale * q[i][u][h] . k_v + M(u, v)) v_v
 * over the keys of node i's own slot and its visible context slots; M is 0
 * on those and -inf elsewhere; attention inside the own chunk is
 * bidirectional.
 *   q    [n_nodes][T][H][d] bf16 (already rotated)
 *   out  [n_nodes][T][H][d] bf16
 *   lse  [n_nodes][H][T] fp32 natural-log sum-exp of the masked logits, or NULL
 *   scale  logit scale, e.g. 1/sqrt(d); finite and > 0
 * Every referenced slot must be resident; contexts must be of the same seq
 * and an earlier chunk, with no slot repeated.  Stream-ordered after the
 * sva_rope_kv_write that filled the slots.  Errors: INVALID_ARGUMENT,
 * NOT_RESIDENT, CAUSALITY, CAPACITY, CUDA. */
sva_status sva_attend_nodes(sva_cache* c, const sva_node* nodes, int32_t n_nodes, const void* q,
                            void* out, float* lse, float scale, sva_stream s);

/* sva_attend_nodes with query-dependent block-sparse access: the token-level
 * mask M of Eq. 4 (Section 3.2), which may give every query its own subset of
 * the causal history, taken at the granularity of 128-query x 128-key tiles.
 *   tile_mask  device array of 32-bit words [n_nodes][nt][words_per_row],
 *              nt = ceil(T / 128) (query tiles of a node = key tiles of a
 *              state).  Bit k (word k / 32, bit k % 32) of row (node i, query
 *              tile qt) set: queries [128 qt, 128 qt + 128) of node i may
 *              attend key tile k % nt (keys [128 (k % nt), ...)) of the node's
 *              key state k / nt, where state 0 is the own slot and state
 *              1 + j is nodes[i].ctx_slot[j].  4-byte aligned; read by the
 *              kernel on `s`, so it must stay valid until that completes.
 *   words_per_row >= ceil((1 + n_ctx) * nt / 32) for every node, and
 *              (1 + n_ctx) * nt <= 4096.
 * The tile mask adds to every other mask: keys of hidden context slots, of
 * later frames under SVA_WITHIN_FRAME_CAUSAL and the padding stay masked
 * whatever the bit.  Key tiles that no query tile of a work unit (a pair of
 * query tiles) may attend are neither loaded nor multiplied, so the cost
 * falls with the density.  A query that sees no key gets O = 0 and LSE =
 * -inf.  Split plans are chosen as for the dense mask.  Errors: as
 * sva_attend_nodes, plus INVALID_ARGUMENT for a NULL or misaligned mask or a
 * short row and CAPACITY beyond 4096 key tiles per node. */
sva_status sva_attend_nodes_sparse(sva_cache* c, const sva_node* nodes, int32_t n_nodes,
                                   const void* q, void* out, float* lse, float scale,
                                   const uint32_t* tile_mask, int32_t words_per_row,
                                   sva_stream s);

/* The masks of sva_attend_nodes_masked, both optional (NULL: no such mask). */
typedef struct {
  /* Block-sparse access, as the tile_mask / words_per_row of
   * sva_attend_nodes_sparse. */
  const uint32_t* tile_mask;
  int32_t tile_words;
  /* Token-level visibility inside each node's own chunk: device array of
   * 32-bit words [n_nodes][T][own_words]; bit v (word v / 32, bit v % 32) of
   * row (node i, query token u) set means query u of node i may attend key
   * token v of its own chunk.  own_words >= ceil(T / 32); 4-byte aligned. */
  const uint32_t* own_mask;
  int32_t own_words;
  /* Token-level visibility of the history: device array of 32-bit words
   * [n_nodes][T][hist_states][hist_words]; bit v of row (node i, query token
   * u, context j) set means query u of node i may attend key token v of the
   * state in nodes[i].ctx_slot[j].  hist_states >= n_ctx of every node (and
   * >= 1), hist_words >= ceil(T / 32); 4-byte aligned. */
  const uint32_t* hist_mask;
  int32_t hist_states;
  int32_t hist_words;
} sva_attn_mask;

/* sva_attend_nodes with the general token-level mask M of Eq. 4 (Section
 * 3.2) inside the own chunk and on the history, and/or query-dependent
 * block-sparse access to the history: M(u, v) = -inf where the own-chunk or
 * history bit of (u, v) or the tile bit of (u's query tile, v's key tile) is
 * clear, on top of every other mask (hidden context slots, the within-chunk
 * mode, padding).  The frame-causal
 * mode is the own mask with bit v set iff v's latent frame is not after u's.
 * Queries that see no key get O = 0 and LSE = -inf.  Both masks are read by
 * the kernel on `s` and must stay valid until it completes.  Errors: as
 * sva_attend_nodes_sparse, plus INVALID_ARGUMENT for a misaligned token mask,
 * a short row or too few history states; a NULL mask pointer or three NULL
 * masks is plain sva_attend_nodes. */
sva_status sva_attend_nodes_masked(sva_cache* c, const sva_node* nodes, int32_t n_nodes,
                                   const void* q, void* out, float* lse, float scale,
                                   const sva_attn_mask* mask, sva_stream s);

/* Bytes of the optional split workspace of a cache (0 if c is NULL).  With
 * a workspace attached, sva_attend_nodes may divide each (node, head,
 * query-tile pair) work unit into up to 4 contiguous key ranges computed by
 * separate CTAs and merged on the device (the softmax of Eq. 4 recombined
 * from per-range maxima and sums), which fills the GPU when a launch has
 * too few work units; results agree with the unsplit computation to
 * rounding. */
size_t sva_attend_workspace_bytes(const sva_cache* c);

/* Attaches a caller-owned device buffer of at least
 * sva_attend_workspace_bytes(c) bytes (256-byte aligned, on the cache's
 * device) as the split workspace, or detaches it when dev_buf is NULL.
 * Zeroes the buffer's counters (synchronous).  The buffer must outlive its
 * use; launches on one cache that overlap on the GPU must not share it.
 * Errors: INVALID_ARGUMENT, CUDA. */
sva_status sva_cache_set_workspace(sva_cache* c, void* dev_buf, size_t bytes);

/* sva_attend_nodes for callers that may not allocate device memory at all:
 * for example a plugin that its host framework hands only input and output
 * buffers, with every other byte of device memory budgeted by that
 * framework, or a serving loop that forbids cudaMalloc because it can block
 * and synchronise the device.  Such a caller cannot provide the split
 * workspace of sva_cache_set_workspace.  This entry point takes the same
 * arguments, runs the same checks and chooses the same key-range split plan
 * as sva_attend_nodes with a workspace attached, so its results are bitwise
 * the same, but it keeps its key-range partials and arrival counters in a
 * scratch array that the library declares in device memory itself (32 MiB,
 * held by every GPU that loads the library until the process exits).  It
 * allocates nothing and calls no allocating routine.  Launches whose split
 * plan needs more than 32 MiB of scratch (counters plus 133 KB per split
 * item at head_dim 128) are rejected with SVA_ERR_CAPACITY and launch
 * nothing; launches that need no split use no scratch and are never
 * rejected for size.
 * Each call clears the array's counters on `s` before its kernel; the
 * partials left by one call are overwritten by the next.  All calls on a
 * device share the one array, so calls whose kernels can overlap on the
 * GPU (different streams without ordering between them) race and must not
 * be issued.  The first call on a device looks up the array's device
 * address (cudaGetSymbolAddress); make that first call before any stream
 * capture.  The paper has no counterpart of this entry point.
 * Errors: as sva_attend_nodes, plus CAPACITY for a plan that does not fit. */
sva_status sva_attend_nodes_noalloc(sva_cache* c, const sva_node* nodes, int32_t n_nodes,
                                    const void* q, void* out, float* lse, float scale,
                                    sva_stream s);

/* Synchronizes `s`, then reads and clears the device status word: returns
 * DEVICE_TIMEOUT if a kernel gave up a bounded wait since the last poll,
 * CUDA if the stream reported an error, else OK. */
sva_status sva_poll_device_status(sva_cache* c, sva_stream s);

/* Test hook for failure detection; no GPU fault is involved.  mode 1 makes
 * the next sva_attend_nodes launch on `c` withhold one of its V-tile copies,
 * so the kernel's bounded wait on that copy expires after timeout_s; every
 * CTA then records SVA_ERR_DEVICE_TIMEOUT in the status word, waits for its
 * own copies and MMAs in flight, frees its tensor memory and exits, and
 * sva_poll_device_status reports the timeout.  Needs nodes of >= 2 key
 * tiles.  mode 0 clears the hook.  timeout_s (1 ms .. 60 s) also becomes the
 * bounded-wait limit of this cache's later launches (default 1 s).
 * Errors: INVALID_ARGUMENT. */
sva_status sva_debug_inject(sva_cache* c, int32_t mode, double timeout_s);

/* Frees the cache object (not the caller's device buffer). */
sva_status sva_destroy(sva_cache* c);

/* Thread-local message describing the last failure ("" if none). */
const char* sva_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* SVA_H_ */
