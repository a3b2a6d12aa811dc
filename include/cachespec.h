/*
 * cachespec.h -- C ABI of libcachespec.so: the draft-and-verify step of
 * speculative sampling on one GB300 (sm_103a).
 *
 * The paper's cache-miss branch (Sec. 3.4) runs the target LLM with the small
 * model as speculative drafter: the drafter proposes k tokens, the target
 * scores the k+1 positions in one pass, and the standard speculative-sampling
 * rule of the works the paper cites (Sec. 2, Sec. 3.4, App. A.4) accepts,
 * corrects or extends the draft.  This library implements the two
 * data-parallel operations of that step:
 *
 *   cs_verify_attention -- the KV-bound core of the target's verify pass:
 *                          multi-query GQA attention of the k+1 positions
 *                          over each request's paged KV cache, causal among
 *                          the drafted tokens;
 *   cs_spec_accept      -- the acceptance step: temperature softmax of target
 *                          and draft logits, accept test, residual / bonus
 *                          draw by inverse CDF, and its greedy variant;
 *   cs_sample           -- the drafter's per-position sampling step (the same
 *                          temperature softmax and inverse-CDF draw);
 *   cs_kv_append,
 *   cs_kv_commit        -- the paged KV cache around the verify pass: append
 *                          the verify positions' K/V rows, then keep the
 *                          accepted prefix;
 *   cs_route            -- the front end's batched semantic routing: cosine
 *                          scores against group centroids, arg max, threshold;
 *   cs_tree_verify_attention,
 *   cs_tree_accept,
 *   cs_kv_commit_tree   -- token-tree verification, the multi-candidate
 *                          variant of the step among those Sec. 2 cites: a
 *                          tree of drafted candidates is scored in one pass
 *                          (each node sees the prefix and its ancestors), one
 *                          root-to-node path is accepted, and its K/V rows
 *                          are moved next to the root.
 *
 * Conventions for every entry point
 *   - All tensor arguments are DEVICE pointers owned by the caller, dense
 *     row-major in the layouts stated below.  The library never allocates,
 *     frees or synchronises (except the status reads cs_read_device_status
 *     and cs_verify_attention_noalloc_status, which say so).
 *   - Calls are asynchronous on `stream` (a cudaStream_t; NULL is the legacy
 *     default stream) and return once the work is enqueued.
 *   - Arguments are checked on the host before anything is enqueued; a bad
 *     argument returns an error code and enqueues nothing.  Values that live
 *     in device memory (context lengths, page ids, token ids) cannot be
 *     checked on the host; their out-of-range behaviour is defined per call.
 *   - On any status other than CS_OK, cs_last_error() returns a message for
 *     the calling thread.
 */
#ifndef CACHESPEC_H
#define CACHESPEC_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaStream_t. */
typedef struct CUstream_st* cs_stream_t;

typedef enum {
    CS_OK = 0,
    CS_ERR_INVALID_ARG = 1,   /* a dimension, pointer, alignment or scalar is invalid */
    CS_ERR_UNSUPPORTED = 2,   /* valid, but outside what these kernels implement */
    CS_ERR_CUDA = 3,          /* the CUDA runtime or driver reported an error */
    CS_ERR_WORKSPACE = 4      /* workspace missing or smaller than the query says */
} cs_status;

typedef enum { CS_F32 = 0, CS_BF16 = 1 } cs_dtype;

/* Geometry of one verify-attention call. */
typedef struct {
    int32_t batch;              /* B >= 0 requests (0: nothing to do) */
    int32_t n_q_heads;          /* Hq > 0 query heads */
    int32_t n_kv_heads;         /* Hkv > 0 KV heads, Hq % Hkv == 0; G = Hq / Hkv */
    int32_t head_dim;           /* D; this library implements D == 128 */
    int32_t page_size;          /* ps tokens per page: 8, 16, 32, 64, 128 or 256 */
    int32_t max_pages_per_seq;  /* columns of page_table (> 0) */
    int32_t num_pages;          /* P pages in the pool (> 0) */
    float sm_scale;             /* softmax scale; <= 0 selects 1/sqrt(D) */
} cs_attn_dims;

/* Geometry of one acceptance call. */
typedef struct {
    int32_t batch;              /* B >= 0 requests (0: nothing to do) */
    int32_t vocab;              /* V > 0 */
    int32_t logit_dtype;        /* cs_dtype of target and draft logits */
} cs_accept_dims;

/* Geometry of one routing call. */
typedef struct {
    int32_t batch;              /* B >= 0 requests */
    int32_t n_groups;           /* N >= 0 groups (0: every request misses) */
    int32_t dim;                /* embedding width, a multiple of 64 up to CS_MAX_ROUTE_DIM */
} cs_route_dims;
#define CS_MAX_ROUTE_DIM 384

/* ABI version of this header (bumped on any incompatible change). */
#define CS_ABI_VERSION 1
int32_t cs_abi_version(void);

/* Message describing the last non-OK status returned on this thread. */
const char* cs_last_error(void);

/*
 * Verify attention (the target's attention over the k+1 verify positions,
 * Sec. 3.4's verify pass).
 *
 * For every request b, query head h and draft row i in [0, k]:
 *     out[b,i,h,:] = softmax_j( sm_scale * q[b,i,h,:] . K_j ) V_j
 * over the keys j = 0 .. L_b-(k+1)+i of KV head h / G: each drafted
 * position sees the whole prefix and the drafts before it.  Key j of
 * request b is slot j % ps of page page_table[b][j / ps].
 *
 *   q          bf16 [B, k+1, Hq, D]
 *   k_pages    bf16 [P, Hkv, ps, D]   16-byte aligned
 *   v_pages    bf16 [P, Hkv, ps, D]   16-byte aligned
 *   page_table int32 [B, max_pages_per_seq]; entries past the last page of a
 *              request are never read
 *   ctx_lens   int32 [B]; L_b counts the k+1 verify positions
 *   n_draft    k in [1, 16]; (k+1)*G must not exceed 144
 *   out        bf16 [B, k+1, Hq, D] (must not alias the inputs)
 *   workspace  device scratch of at least
 *              cs_verify_attention_workspace_bytes(dims, k) bytes, 256-byte
 *              aligned, ZERO-FILLED before its first use; every call that
 *              completes leaves it ready for the next call.  Calls that share
 *              a workspace must be ordered (same stream or events).  May be
 *              NULL when the query returns 0.
 *
 * Defined behaviour for device-resident values: L_b is clamped to
 * [0, max_pages_per_seq*ps]; a row with no admissible key
 * (L_b-(k+1)+i < 0) outputs zeros; a page id outside [0, P) reads as zeros.
 * Pool slots past L_b may hold any bits (including NaN); they never reach
 * the output.  Arithmetic: S = q.K in bf16 with fp32 accumulation, the
 * softmax in fp32, and the P.V product on bf16 V as stored, with P taken as
 * the sum of two bf16 terms (hi = bf16(P), lo = bf16(P - hi): ~16
 * significant bits) and fp32 accumulation.  P is formed scaled by 2^-64 (the
 * row sum carries the same factor), so that no partial sum of P.V overflows
 * fp32: every finite bf16 V, up to bf16's largest value, gives a finite
 * output within the stated tolerance.
 *
 * Returns CS_ERR_INVALID_ARG (null pointer, misalignment, bad dimension, NaN
 * scale, n_draft out of range), CS_ERR_UNSUPPORTED (D != 128, page size,
 * (k+1)*G > 144), CS_ERR_WORKSPACE, or CS_ERR_CUDA (launch failure).
 */
size_t cs_verify_attention_workspace_bytes(const cs_attn_dims* dims, int32_t n_draft);
cs_status cs_verify_attention(const cs_attn_dims* dims, const void* q, const void* k_pages,
                              const void* v_pages, const int32_t* page_table,
                              const int32_t* ctx_lens, int32_t n_draft, void* out,
                              void* workspace, size_t workspace_bytes, cs_stream_t stream);

/*
 * Speculative acceptance (the accept / correct / extend rule of the
 * speculative sampling the paper's drafter follows, Sec. 3.4; temperature 0
 * is the greedy mode of the paper's App. B runs).
 *
 * Temperature T > 0, for each request b:
 *   p_i = softmax(target[b,i,:] / T) for i in [0, k];
 *   q_i = softmax(draft[b,i,:] / T)  for i in [0, k);
 *   position i accepts x_i = draft_tokens[b,i] iff u_i < p_i(x_i) / q_i(x_i);
 *   a = the first rejected position, or k if none is rejected;
 *   if a < k the emitted token is drawn from max(0, p_a - q_a) normalised,
 *   else (the bonus token) from p_k, in both cases as the smallest token id
 *   whose running mass (ascending ids) exceeds u_k times the total.
 * Temperature 0 (greedy): g_i = argmax target[b,i,:] (lowest id on ties);
 *   position i accepts iff x_i == g_i; the emitted token is g_a.
 *
 *   target_logits  [B, k+1, V] fp32 or bf16 (dims->logit_dtype), element-aligned
 *   draft_logits   [B, k,   V] same dtype; may be NULL when temperature == 0
 *   draft_tokens   int32 [B, k]; an id outside [0, V) is rejected at its position
 *   uniforms       fp32 [B, k+1] in [0, 1): u_0..u_{k-1} for the accept tests,
 *                  u_k for the single final draw
 *   n_draft        k in [1, 16]
 *   temperature    T >= 0 and finite
 *   out_tokens     int32 [B, k+1]: x_0..x_{a-1}, the emitted token, then -1
 *   out_n_accepted int32 [B]: a
 *   workspace      device scratch of at least cs_spec_accept_workspace_bytes(dims, k)
 *                  bytes, 256-byte aligned, any initial contents: every call
 *                  writes each scratch word it later reads (one pair per row
 *                  segment of the statistics pass).  Calls that share a
 *                  workspace must be ordered (same stream or events).
 *
 * A logit of -inf marks a masked token (probability zero); NaN and +inf are
 * not allowed, and every row needs a finite entry.  The result is a
 * deterministic function of the inputs.
 *
 * Returns CS_ERR_INVALID_ARG (null pointer, misalignment, bad dimension,
 * bad temperature, n_draft out of range), CS_ERR_UNSUPPORTED (vocab above
 * CS_MAX_VOCAB), CS_ERR_WORKSPACE (missing or too small) or CS_ERR_CUDA.
 */
#define CS_MAX_VOCAB (1 << 22)
size_t cs_spec_accept_workspace_bytes(const cs_accept_dims* dims, int32_t n_draft);
cs_status cs_spec_accept(const cs_accept_dims* dims, const void* target_logits,
                         const void* draft_logits, const int32_t* draft_tokens,
                         const float* uniforms, int32_t n_draft, float temperature,
                         int32_t* out_tokens, int32_t* out_n_accepted, void* workspace,
                         size_t workspace_bytes, cs_stream_t stream);

/*
 * Allocation-free verify attention.  The paper has no counterpart: this entry
 * point serves callers of this library that cannot allocate device memory
 * themselves -- code running inside a host framework that owns every device
 * allocation, serving loops that allow no allocation after start-up
 * (cudaMalloc can stall the whole device), or bindings without a device
 * allocator.
 *
 * Same arguments, layouts, results and error codes as cs_verify_attention,
 * without the workspace: the scratch is a fixed array of
 * CS_NOALLOC_SCRATCH_BYTES compiled into this library, which every GPU that
 * loads the library holds until the process exits.  The call never runs
 * cudaMalloc, cudaFree or any other allocating routine.
 *   - A problem that needs more scratch than that (see
 *     cs_verify_attention_workspace_bytes) returns CS_ERR_UNSUPPORTED with a
 *     message giving both sizes; use cs_verify_attention then.
 *   - The first call on each device looks up the array's device address with
 *     cudaGetSymbolAddress (with that device current) and caches it; make
 *     that first call before any stream capture begins.
 *   - Each call clears the part of the scratch that must start at zero (an
 *     asynchronous memset on `stream`), so a failed call does not affect the
 *     next one.
 *   - Every call on a device shares the one array: calls whose kernels may
 *     overlap on the GPU (different streams, or host threads using different
 *     streams) race on it.  Order them on one stream or with events.
 */
#define CS_NOALLOC_SCRATCH_BYTES (32u << 20)
cs_status cs_verify_attention_noalloc(const cs_attn_dims* dims, const void* q, const void* k_pages,
                                      const void* v_pages, const int32_t* page_table,
                                      const int32_t* ctx_lens, int32_t n_draft, void* out,
                                      cs_stream_t stream);

/*
 * Device status word of the allocation-free entry point on the current
 * device (the counterpart of cs_read_device_status, whose workspace the
 * caller of cs_verify_attention_noalloc does not have): 0, or the CS_DEVICE_*
 * bits of the latest cs_verify_attention_noalloc call enqueued before it on
 * `stream` (each call clears the word first, so a bit names that call's
 * failure: its output is invalid).  Copies 4 bytes to the host and
 * SYNCHRONISES `stream`; allocates nothing.  The paper has no counterpart.
 * CS_ERR_INVALID_ARG for a NULL status_out, CS_ERR_CUDA on a copy failure.
 */
cs_status cs_verify_attention_noalloc_status(int32_t* status_out, cs_stream_t stream);

/*
 * Paged KV cache around the verify pass (Sec. 3.4's draft-and-verify step).
 *
 * cs_kv_append writes the K and V rows of the n_new newest positions of
 * every request into its pages before verify attention (n_new = k+1: the
 * last committed token and the k drafts).  ctx_lens[b] = L_b already counts
 * them (clamped to [0, max_pages_per_seq*page_size], as in
 * cs_verify_attention), so row i of request b, KV head h lands at key
 * position L_b - n_new + i: slot (L_b - n_new + i) % ps of page
 * page_table[b][(L_b - n_new + i) / ps].  A row whose position is negative
 * or whose page id lies outside [0, num_pages) is not written.
 *
 *   dims        the pool geometry (head_dim 128; n_q_heads and sm_scale unused)
 *   new_k/new_v bf16 [B, n_new, Hkv, 128], 16-byte aligned
 *   k_pages/v_pages bf16 [P, Hkv, ps, 128], 16-byte aligned, updated in place
 *   page_table  int32 [B, max_pages_per_seq]; ctx_lens int32 [B]
 *   n_new       in [1, 4096]
 * Requests must not share the page slots they write (the writes would race).
 *
 * cs_kv_commit shortens every context after the acceptance step to the rows
 * that stay valid: the prefix, the last committed token and the accepted
 * drafts, ctx_lens[b] <- max(0, ctx_lens[b] - n_draft + n_accepted[b]).
 * The emitted token (residual or bonus draw) has no row yet: it is the first
 * input of the next step.  Pages past the new length are not released.
 *
 * Both return CS_ERR_INVALID_ARG (null pointer, misalignment, bad dimension
 * or count), CS_ERR_UNSUPPORTED (head_dim != 128) or CS_ERR_CUDA.
 */
cs_status cs_kv_append(const cs_attn_dims* dims, const void* new_k, const void* new_v, void* k_pages,
                       void* v_pages, const int32_t* page_table, const int32_t* ctx_lens, int32_t n_new,
                       cs_stream_t stream);
cs_status cs_kv_commit(int32_t batch, int32_t* ctx_lens, const int32_t* n_accepted, int32_t n_draft,
                       cs_stream_t stream);

/*
 * Batched semantic routing (the paper's front end, Sec. 3.1): the score of
 * request b against group i is the cosine similarity of their embeddings,
 *     S(b, i) = (e_b . c_i) / (|e_b| |c_i|)   (0 when either norm is 0);
 * out_best[b] = argmax_i S(b, i) (the lowest i on ties; -1 when N == 0),
 * out_score[b] = that score (-inf when N == 0), and
 * out_group[b] = out_best[b] when out_score[b] >= tau, else -1 (the request
 * goes to the cache-miss branch).
 *
 *   emb        bf16 [B, dim], 16-byte aligned
 *   centroids  bf16 [N, dim], 16-byte aligned (may be NULL when N == 0)
 *   inv_norms  fp32 [N]: 1/|c_i| (0 for a zero row), as written by
 *              cs_route_norms for the same centroids (may be NULL when N == 0)
 *   tau        the matching threshold, finite
 *   out_*      int32 / fp32 [B]
 *   workspace  at least cs_route_workspace_bytes(dims) bytes, 256-byte
 *              aligned, any initial contents; calls sharing one must be
 *              ordered.  Its first 4 bytes are the device status word
 *              (cs_read_device_status); zero-fill the workspace before its
 *              first use.
 * The scores are fp32 sums of exact bf16 products: they differ from exact
 * cosines by at most ~dim * 2^-24 relative.
 *
 * cs_route_norms writes inv_norms for N centroids (run it whenever the
 * centroids change).
 *
 * Return CS_ERR_INVALID_ARG (null pointer, misalignment, bad count or
 * threshold), CS_ERR_UNSUPPORTED (dim not a multiple of 64 in
 * [64, CS_MAX_ROUTE_DIM]), CS_ERR_WORKSPACE or CS_ERR_CUDA.
 */
size_t cs_route_workspace_bytes(const cs_route_dims* dims);
cs_status cs_route_norms(int32_t n_groups, int32_t dim, const void* centroids, float* inv_norms,
                         cs_stream_t stream);
cs_status cs_route(const cs_route_dims* dims, const void* emb, const void* centroids,
                   const float* inv_norms, float tau, int32_t* out_group, int32_t* out_best,
                   float* out_score, void* workspace, size_t workspace_bytes, cs_stream_t stream);

/*
 * Draft-side sampling (the drafter's step before the verify pass: it
 * proposes x_i ~ q_i one position at a time, Sec. 3.4), with the same
 * conventions as the final draw of cs_spec_accept.
 *
 * For every request b:
 *   T > 0: out_tokens[b] = the smallest token id whose running mass of
 *          softmax(logits[b,:] / T) (ascending ids) exceeds uniforms[b]
 *          times the total (if rounding leaves none, the largest id of
 *          positive weight);
 *   T == 0: out_tokens[b] = argmax logits[b,:] (lowest id on ties).
 *
 *   logits       [B, V] fp32 or bf16 (dims->logit_dtype), element-aligned
 *   uniforms     fp32 [B] in [0, 1) (read only when T > 0)
 *   temperature  T >= 0 and finite
 *   out_tokens   int32 [B]
 *   workspace    device scratch of at least cs_sample_workspace_bytes(dims)
 *                bytes, 256-byte aligned, any initial contents; calls that
 *                share one must be ordered.
 *
 * A logit of -inf marks a masked token; every row needs a finite entry.
 * Returns CS_ERR_INVALID_ARG, CS_ERR_UNSUPPORTED (vocab above CS_MAX_VOCAB),
 * CS_ERR_WORKSPACE or CS_ERR_CUDA.
 */
size_t cs_sample_workspace_bytes(const cs_accept_dims* dims);
cs_status cs_sample(const cs_accept_dims* dims, const void* logits, const float* uniforms,
                    float temperature, int32_t* out_tokens, void* workspace,
                    size_t workspace_bytes, cs_stream_t stream);

/*
 * Token-tree verification (the tree-structured, multi-candidate variants of
 * speculative decoding that Sec. 2 cites beside the chain of Sec. 3.4).
 *
 * A request's tree has n nodes in topological order, described by
 * parents int32 [B, n]: node 0 is the root (the last committed token; its
 * entry is ignored), node c >= 1 is a drafted token whose parent must lie in
 * [0, c).  A node whose parent does not is detached: it sees only the prefix
 * and itself, and the walk never reaches it.  Node m's K/V rows sit at key
 * position L_b - n + m (ctx_lens counts the n tree positions, as for the
 * chain; cs_kv_append with n_new = n writes them).
 *
 * cs_tree_verify_attention: for every node i, query head h,
 *     out[b,i,h,:] = softmax_j( sm_scale * q[b,i,h,:] . K_j ) V_j
 * over the prefix keys j < L_b - n and the tree keys L_b - n + m for every
 * ancestor m of i and i itself.  Arguments, layouts (q and out are
 * [B, n, Hq, D]), workspace rules and defined behaviour as for
 * cs_verify_attention, with n_nodes in [1, 64] in place of n_draft + 1.
 * Trees with n * G > 144 query rows per KV head are processed as row blocks
 * of at most 144 rows, each reading that head's keys again.
 *
 * cs_tree_accept: the walk of multi-candidate speculative sampling.  At the
 * current node u (the root first) the running distribution r starts as
 * p_u = softmax(target[b,u,:] / T); the children of u are tested in
 * ascending index against q_u = softmax(draft[b,u,:] / T), the distribution
 * they were drafted from: child c with token x is accepted iff
 * u_{c-1} < r(x) / q_u(x); a rejection replaces r by max(0, r - q_u)
 * normalised (if that has no positive mass the remaining children are
 * skipped and r is p_u again).  An accepted child is emitted and becomes u;
 * when no child is accepted (or u is a leaf) one token is drawn from r by
 * the inverse CDF of cs_spec_accept at u_{n-1}, and the walk ends.  When the
 * children of every node are independent draws from its q_u, the emitted
 * tokens follow the target distribution.  A chain (parents[c] = c - 1) is
 * the rule of cs_spec_accept with k = n - 1.  T == 0: at node u the first
 * child whose token is argmax target[b,u,:] (lowest id on ties) is accepted,
 * else that argmax is emitted.
 *
 *   target_logits  [B, n, V] fp32 or bf16; row u is node u's next-token
 *                  distribution
 *   draft_logits   [B, n, V] same dtype; row u is the distribution u's
 *                  children were drafted from (rows of leaves are not read);
 *                  may be NULL when temperature == 0
 *   node_tokens    int32 [B, n]: the token of each node (entry 0 unused); an
 *                  id outside [0, V) is never accepted
 *   uniforms       fp32 [B, n] in [0, 1): u_{c-1} tests node c, u_{n-1} is
 *                  the draw
 *   out_tokens     int32 [B, n]: the accepted tokens in walk order, the
 *                  emitted token, then -1
 *   out_path       int32 [B, n]: the accepted nodes in walk order, then -1
 *   out_n_accepted int32 [B]: the number of accepted nodes a
 *   workspace      at least cs_tree_accept_workspace_bytes(dims, n) bytes,
 *                  256-byte aligned, any initial contents; calls sharing one
 *                  must be ordered.
 * Logit conventions as for cs_spec_accept.
 *
 * cs_kv_commit_tree: after the walk, moves the K and V rows of the accepted
 * nodes path[0..a) (out_path, out_n_accepted) to the positions right after
 * the root, L_b - n + 1 + i, and sets ctx_lens[b] = L_b - n + 1 + a (L_b
 * clamped to [0, max_pages_per_seq * ps], a to [0, n-1]).  Rows whose page
 * id lies outside [0, num_pages) are not moved.  The emitted token has no
 * row yet: it is the first input of the next step.
 *
 * Return CS_ERR_INVALID_ARG (null pointer, misalignment, bad dimension,
 * n_nodes outside [1, 64], bad temperature), CS_ERR_UNSUPPORTED (as for the
 * chain calls), CS_ERR_WORKSPACE or CS_ERR_CUDA.
 */
#define CS_MAX_TREE_NODES 64
size_t cs_tree_verify_attention_workspace_bytes(const cs_attn_dims* dims, int32_t n_nodes);
cs_status cs_tree_verify_attention(const cs_attn_dims* dims, const void* q, const void* k_pages,
                                   const void* v_pages, const int32_t* page_table, const int32_t* ctx_lens,
                                   const int32_t* parents, int32_t n_nodes, void* out, void* workspace,
                                   size_t workspace_bytes, cs_stream_t stream);
size_t cs_tree_accept_workspace_bytes(const cs_accept_dims* dims, int32_t n_nodes);
cs_status cs_tree_accept(const cs_accept_dims* dims, const void* target_logits, const void* draft_logits,
                         const int32_t* parents, const int32_t* node_tokens, const float* uniforms,
                         int32_t n_nodes, float temperature, int32_t* out_tokens, int32_t* out_path,
                         int32_t* out_n_accepted, void* workspace, size_t workspace_bytes, cs_stream_t stream);
cs_status cs_kv_commit_tree(const cs_attn_dims* dims, void* k_pages, void* v_pages, const int32_t* page_table,
                            int32_t* ctx_lens, const int32_t* path, const int32_t* n_accepted, int32_t n_nodes,
                            cs_stream_t stream);

/*
 * Device status word of a verify-attention workspace: 0 when every call that
 * used it finished normally; otherwise a bit set of CS_DEVICE_* flags (a
 * bounded wait inside a kernel gave up, so that call's output is invalid).
 * Copies 4 bytes to the host and SYNCHRONISES `stream`.  The word is sticky
 * until the caller zero-fills the workspace again.
 */
#define CS_DEVICE_WAIT_TIMEOUT 1
cs_status cs_read_device_status(const void* workspace, int32_t* status_out, cs_stream_t stream);

/*
 * Failure-detection self-test.  Enqueues one kernel whose single thread runs
 * the bounded mbarrier wait that every wait of the attention kernels uses, on
 * a barrier that nothing completes.  After about one second the wait gives up
 * and the thread sets CS_DEVICE_WAIT_TIMEOUT in the status word, the first 4
 * bytes of `workspace` (a device buffer of at least 4 bytes, 4-byte aligned,
 * owned by the caller; nothing else in it is touched).  Read the word with
 * cs_read_device_status.  No fault, trap or hang: the context stays usable.
 * CS_ERR_INVALID_ARG for a NULL or misaligned workspace.
 */
cs_status cs_selftest_wait_timeout(void* workspace, cs_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* CACHESPEC_H */
