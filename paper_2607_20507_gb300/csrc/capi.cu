// capi.cu -- the extern "C" surface of libcachespec.so (see include/cachespec.h):
// host-side argument checks, the workspace queries and dispatch to the
// kernel launchers.  Nothing here allocates, frees or synchronises device
// memory except cs_read_device_status, which is documented to synchronise.
#include <math.h>
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include "cs_internal.h"

namespace cs {

namespace {
thread_local char g_err[512] = "";
int g_sms[64] = {0};

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

bool pow2_page(int ps) {
    return ps == 8 || ps == 16 || ps == 32 || ps == 64 || ps == 128 || ps == 256;
}

// Geometry checks shared by the chain and tree attention calls.
cs_status check_attn_geometry(const cs_attn_dims* d) {
    if (!d) return fail(CS_ERR_INVALID_ARG, "dims is NULL");
    if (d->batch < 0) return fail(CS_ERR_INVALID_ARG, "batch %d < 0", d->batch);
    if (d->n_q_heads <= 0 || d->n_kv_heads <= 0)
        return fail(CS_ERR_INVALID_ARG, "head counts must be positive (Hq=%d, Hkv=%d)", d->n_q_heads,
                    d->n_kv_heads);
    if (d->n_q_heads % d->n_kv_heads != 0)
        return fail(CS_ERR_INVALID_ARG, "Hq=%d is not a multiple of Hkv=%d", d->n_q_heads,
                    d->n_kv_heads);
    if (d->head_dim <= 0) return fail(CS_ERR_INVALID_ARG, "head_dim %d <= 0", d->head_dim);
    if (d->page_size <= 0) return fail(CS_ERR_INVALID_ARG, "page_size %d <= 0", d->page_size);
    if (d->max_pages_per_seq <= 0)
        return fail(CS_ERR_INVALID_ARG, "max_pages_per_seq %d <= 0", d->max_pages_per_seq);
    if (d->num_pages <= 0) return fail(CS_ERR_INVALID_ARG, "num_pages %d <= 0", d->num_pages);
    if (isnan(d->sm_scale) || isinf(d->sm_scale))
        return fail(CS_ERR_INVALID_ARG, "sm_scale is not finite");
    if (d->head_dim != 128) return fail(CS_ERR_UNSUPPORTED, "head_dim %d (this library implements 128)", d->head_dim);
    if (!pow2_page(d->page_size))
        return fail(CS_ERR_UNSUPPORTED, "page_size %d (supported: 8..256, powers of two)", d->page_size);
    if ((long long)d->max_pages_per_seq * d->page_size > (1LL << 30))
        return fail(CS_ERR_INVALID_ARG, "max_pages_per_seq * page_size exceeds 2^30 keys");
    return CS_OK;
}

cs_status check_attn(const cs_attn_dims* d, int32_t n_draft) {
    if (!d) return fail(CS_ERR_INVALID_ARG, "dims is NULL");
    if (n_draft < 1 || n_draft > 16) return fail(CS_ERR_INVALID_ARG, "n_draft %d not in [1, 16]", n_draft);
    const cs_status st = check_attn_geometry(d);
    if (st != CS_OK) return st;
    const long long rows = (long long)(n_draft + 1) * (d->n_q_heads / d->n_kv_heads);
    if (rows > 144) return fail(CS_ERR_UNSUPPORTED, "(k+1)*G = %lld query rows per KV head (max 144)", rows);
    return CS_OK;
}

cs_status check_tree_attn(const cs_attn_dims* d, int32_t n_nodes) {
    if (!d) return fail(CS_ERR_INVALID_ARG, "dims is NULL");
    if (n_nodes < 1 || n_nodes > CS_MAX_TREE_NODES)
        return fail(CS_ERR_INVALID_ARG, "n_nodes %d not in [1, %d]", n_nodes, CS_MAX_TREE_NODES);
    return check_attn_geometry(d);
}

// Pointer checks shared by the chain and tree attention calls.
cs_status check_attn_pointers(const void* q, const void* k_pages, const void* v_pages, const int32_t* page_table,
                              const int32_t* ctx_lens, const void* out) {
    if (!q || !k_pages || !v_pages || !page_table || !ctx_lens || !out)
        return fail(CS_ERR_INVALID_ARG, "a tensor pointer is NULL");
    if (!aligned(k_pages, 16) || !aligned(v_pages, 16))
        return fail(CS_ERR_INVALID_ARG, "k_pages and v_pages must be 16-byte aligned");
    if (!aligned(q, 4) || !aligned(out, 8))
        return fail(CS_ERR_INVALID_ARG, "q must be 4-byte and out 8-byte aligned");
    if (!aligned(page_table, 4) || !aligned(ctx_lens, 4))
        return fail(CS_ERR_INVALID_ARG, "page_table and ctx_lens must be 4-byte aligned");
    return CS_OK;
}

cs_status check_accept(const cs_accept_dims* d, int32_t n_draft, float temperature) {
    if (!d) return fail(CS_ERR_INVALID_ARG, "dims is NULL");
    if (d->batch < 0) return fail(CS_ERR_INVALID_ARG, "batch %d < 0", d->batch);
    if (d->vocab <= 0) return fail(CS_ERR_INVALID_ARG, "vocab %d <= 0", d->vocab);
    if (d->logit_dtype != CS_F32 && d->logit_dtype != CS_BF16)
        return fail(CS_ERR_INVALID_ARG, "logit_dtype %d is neither CS_F32 nor CS_BF16", d->logit_dtype);
    if (n_draft < 1 || n_draft > 16) return fail(CS_ERR_INVALID_ARG, "n_draft %d not in [1, 16]", n_draft);
    if (!(temperature >= 0.f) || isinf(temperature))
        return fail(CS_ERR_INVALID_ARG, "temperature must be finite and >= 0");
    if ((long long)d->batch * (n_draft + 1) * (long long)d->vocab > (1LL << 46))
        return fail(CS_ERR_INVALID_ARG, "logit tensor too large");
    if (d->vocab > CS_MAX_VOCAB)
        return fail(CS_ERR_UNSUPPORTED, "vocab %d (this library implements up to %d)", d->vocab, CS_MAX_VOCAB);
    return CS_OK;
}
cs_status check_route(const cs_route_dims* d) {
    if (!d) return fail(CS_ERR_INVALID_ARG, "dims is NULL");
    if (d->batch < 0 || d->n_groups < 0) return fail(CS_ERR_INVALID_ARG, "batch and n_groups must be >= 0");
    if (d->dim <= 0 || d->dim % 64 != 0 || d->dim > CS_MAX_ROUTE_DIM)
        return fail(CS_ERR_UNSUPPORTED, "dim %d (supported: multiples of 64 up to %d)", d->dim, CS_MAX_ROUTE_DIM);
    if ((d->batch + 127) / 128 > 65535) return fail(CS_ERR_UNSUPPORTED, "batch %d too large for one call", d->batch);
    return CS_OK;
}

cs_status check_sample(const cs_accept_dims* d, float temperature) {
    if (!d) return fail(CS_ERR_INVALID_ARG, "dims is NULL");
    if (d->batch < 0) return fail(CS_ERR_INVALID_ARG, "batch %d < 0", d->batch);
    if (d->vocab <= 0) return fail(CS_ERR_INVALID_ARG, "vocab %d <= 0", d->vocab);
    if (d->logit_dtype != CS_F32 && d->logit_dtype != CS_BF16)
        return fail(CS_ERR_INVALID_ARG, "logit_dtype %d is neither CS_F32 nor CS_BF16", d->logit_dtype);
    if (!(temperature >= 0.f) || isinf(temperature))
        return fail(CS_ERR_INVALID_ARG, "temperature must be finite and >= 0");
    if ((long long)d->batch * (long long)d->vocab > (1LL << 46))
        return fail(CS_ERR_INVALID_ARG, "logit tensor too large");
    if (d->vocab > CS_MAX_VOCAB)
        return fail(CS_ERR_UNSUPPORTED, "vocab %d (this library implements up to %d)", d->vocab, CS_MAX_VOCAB);
    return CS_OK;
}
}  // namespace

cs_status fail(cs_status st, const char* fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, sizeof g_err, fmt, ap);
    va_end(ap);
    return st;
}

cs_status cuda_fail(cudaError_t e, const char* what) {
    return fail(CS_ERR_CUDA, "%s: %s (%s)", what, cudaGetErrorString(e), cudaGetErrorName(e));
}

int current_sm_count() {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 148;
    if (!g_sms[dev]) {
        int n = 0;
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
            n = 148;
        g_sms[dev] = n;
    }
    return g_sms[dev];
}

}  // namespace cs

using namespace cs;

extern "C" {

int32_t cs_abi_version(void) { return CS_ABI_VERSION; }

const char* cs_last_error(void) { return g_err; }

size_t cs_verify_attention_workspace_bytes(const cs_attn_dims* dims, int32_t n_draft) {
    if (check_attn(dims, n_draft) != CS_OK) return 0;
    return plan_verify_attention(*dims, n_draft, current_sm_count()).bytes;
}

cs_status cs_verify_attention(const cs_attn_dims* dims, const void* q, const void* k_pages,
                              const void* v_pages, const int32_t* page_table,
                              const int32_t* ctx_lens, int32_t n_draft, void* out,
                              void* workspace, size_t workspace_bytes, cs_stream_t stream) {
    cs_status st = check_attn(dims, n_draft);
    if (st != CS_OK) return st;
    if (dims->batch == 0) return CS_OK;
    st = check_attn_pointers(q, k_pages, v_pages, page_table, ctx_lens, out);
    if (st != CS_OK) return st;
    const AttnPlan plan = plan_verify_attention(*dims, n_draft, current_sm_count());
    if (!workspace || workspace_bytes < plan.bytes)
        return fail(CS_ERR_WORKSPACE, "workspace of %zu bytes given, %zu needed", workspace_bytes,
                    plan.bytes);
    if (!aligned(workspace, 256)) return fail(CS_ERR_INVALID_ARG, "workspace must be 256-byte aligned");
    return launch_verify_attention(*dims, plan, q, k_pages, v_pages, page_table, ctx_lens, nullptr, out,
                                   workspace, reinterpret_cast<cudaStream_t>(stream));
}

size_t cs_tree_verify_attention_workspace_bytes(const cs_attn_dims* dims, int32_t n_nodes) {
    if (check_tree_attn(dims, n_nodes) != CS_OK) return 0;
    return plan_tree_attention(*dims, n_nodes, current_sm_count()).bytes;
}

cs_status cs_tree_verify_attention(const cs_attn_dims* dims, const void* q, const void* k_pages,
                                   const void* v_pages, const int32_t* page_table, const int32_t* ctx_lens,
                                   const int32_t* parents, int32_t n_nodes, void* out, void* workspace,
                                   size_t workspace_bytes, cs_stream_t stream) {
    cs_status st = check_tree_attn(dims, n_nodes);
    if (st != CS_OK) return st;
    if (dims->batch == 0) return CS_OK;
    st = check_attn_pointers(q, k_pages, v_pages, page_table, ctx_lens, out);
    if (st != CS_OK) return st;
    if (!parents) return fail(CS_ERR_INVALID_ARG, "parents is NULL");
    if (!aligned(parents, 4)) return fail(CS_ERR_INVALID_ARG, "parents must be 4-byte aligned");
    const AttnPlan plan = plan_tree_attention(*dims, n_nodes, current_sm_count());
    if (!workspace || workspace_bytes < plan.bytes)
        return fail(CS_ERR_WORKSPACE, "workspace of %zu bytes given, %zu needed", workspace_bytes, plan.bytes);
    if (!aligned(workspace, 256)) return fail(CS_ERR_INVALID_ARG, "workspace must be 256-byte aligned");
    return launch_verify_attention(*dims, plan, q, k_pages, v_pages, page_table, ctx_lens, parents, out,
                                   workspace, reinterpret_cast<cudaStream_t>(stream));
}

size_t cs_tree_accept_workspace_bytes(const cs_accept_dims* dims, int32_t n_nodes) {
    if (check_sample(dims, 1.0f) != CS_OK || n_nodes < 1 || n_nodes > CS_MAX_TREE_NODES) return 0;
    return tree_accept_workspace_bytes(*dims, n_nodes);
}

cs_status cs_tree_accept(const cs_accept_dims* dims, const void* target_logits, const void* draft_logits,
                         const int32_t* parents, const int32_t* node_tokens, const float* uniforms,
                         int32_t n_nodes, float temperature, int32_t* out_tokens, int32_t* out_path,
                         int32_t* out_n_accepted, void* workspace, size_t workspace_bytes, cs_stream_t stream) {
    cs_status st = check_sample(dims, temperature);
    if (st != CS_OK) return st;
    if (n_nodes < 1 || n_nodes > CS_MAX_TREE_NODES)
        return fail(CS_ERR_INVALID_ARG, "n_nodes %d not in [1, %d]", n_nodes, CS_MAX_TREE_NODES);
    if ((long long)dims->batch * n_nodes * (long long)dims->vocab > (1LL << 46))
        return fail(CS_ERR_INVALID_ARG, "logit tensor too large");
    if (dims->batch == 0) return CS_OK;
    if (!target_logits || !parents || !node_tokens || !uniforms || !out_tokens || !out_path || !out_n_accepted)
        return fail(CS_ERR_INVALID_ARG, "a tensor pointer is NULL");
    if (temperature > 0.f && !draft_logits)
        return fail(CS_ERR_INVALID_ARG, "draft_logits is NULL with temperature > 0");
    const size_t esz = dims->logit_dtype == CS_F32 ? 4 : 2;
    if (!aligned(target_logits, esz) || (draft_logits && !aligned(draft_logits, esz)))
        return fail(CS_ERR_INVALID_ARG, "logit pointers must be aligned to their element size");
    if (!aligned(parents, 4) || !aligned(node_tokens, 4) || !aligned(uniforms, 4) || !aligned(out_tokens, 4) ||
        !aligned(out_path, 4) || !aligned(out_n_accepted, 4))
        return fail(CS_ERR_INVALID_ARG, "int32/fp32 pointers must be 4-byte aligned");
    const size_t need = tree_accept_workspace_bytes(*dims, n_nodes);
    if (!workspace || workspace_bytes < need)
        return fail(CS_ERR_WORKSPACE, "workspace of %zu bytes given, %zu needed", workspace_bytes, need);
    if (!aligned(workspace, 256)) return fail(CS_ERR_INVALID_ARG, "workspace must be 256-byte aligned");
    return launch_tree_accept(*dims, target_logits, temperature > 0.f ? draft_logits : nullptr, parents, node_tokens,
                              uniforms, n_nodes, temperature, out_tokens, out_path, out_n_accepted, workspace,
                              reinterpret_cast<cudaStream_t>(stream));
}

cs_status cs_kv_commit_tree(const cs_attn_dims* dims, void* k_pages, void* v_pages, const int32_t* page_table,
                            int32_t* ctx_lens, const int32_t* path, const int32_t* n_accepted, int32_t n_nodes,
                            cs_stream_t stream) {
    if (!dims) return fail(CS_ERR_INVALID_ARG, "dims is NULL");
    const cs_attn_dims* d = dims;
    if (d->batch < 0) return fail(CS_ERR_INVALID_ARG, "batch %d < 0", d->batch);
    if (d->n_kv_heads <= 0 || d->page_size <= 0 || d->max_pages_per_seq <= 0 || d->num_pages <= 0)
        return fail(CS_ERR_INVALID_ARG, "n_kv_heads, page_size, max_pages_per_seq and num_pages must be positive");
    if (d->head_dim != 128) return fail(CS_ERR_UNSUPPORTED, "head_dim %d (this library implements 128)", d->head_dim);
    if (n_nodes < 1 || n_nodes > CS_MAX_TREE_NODES)
        return fail(CS_ERR_INVALID_ARG, "n_nodes %d not in [1, %d]", n_nodes, CS_MAX_TREE_NODES);
    if ((long long)d->max_pages_per_seq * d->page_size > (1LL << 30))
        return fail(CS_ERR_INVALID_ARG, "max_pages_per_seq * page_size exceeds 2^30 keys");
    if (d->batch == 0) return CS_OK;
    if (!k_pages || !v_pages || !page_table || !ctx_lens || !path || !n_accepted)
        return fail(CS_ERR_INVALID_ARG, "a tensor pointer is NULL");
    if (!aligned(k_pages, 16) || !aligned(v_pages, 16))
        return fail(CS_ERR_INVALID_ARG, "page pools must be 16-byte aligned");
    if (!aligned(page_table, 4) || !aligned(ctx_lens, 4) || !aligned(path, 4) || !aligned(n_accepted, 4))
        return fail(CS_ERR_INVALID_ARG, "int32 pointers must be 4-byte aligned");
    return launch_kv_commit_tree(*d, k_pages, v_pages, page_table, ctx_lens, path, n_accepted, n_nodes,
                                 reinterpret_cast<cudaStream_t>(stream));
}

size_t cs_spec_accept_workspace_bytes(const cs_accept_dims* dims, int32_t n_draft) {
    if (check_accept(dims, n_draft, 1.0f) != CS_OK) return 0;
    return accept_workspace_bytes_any(*dims, n_draft);
}

cs_status cs_spec_accept(const cs_accept_dims* dims, const void* target_logits,
                         const void* draft_logits, const int32_t* draft_tokens,
                         const float* uniforms, int32_t n_draft, float temperature,
                         int32_t* out_tokens, int32_t* out_n_accepted, void* workspace,
                         size_t workspace_bytes, cs_stream_t stream) {
    cs_status st = check_accept(dims, n_draft, temperature);
    if (st != CS_OK) return st;
    if (dims->batch == 0) return CS_OK;
    if (!target_logits || !draft_tokens || !uniforms || !out_tokens || !out_n_accepted)
        return fail(CS_ERR_INVALID_ARG, "a tensor pointer is NULL");
    if (temperature > 0.f && !draft_logits)
        return fail(CS_ERR_INVALID_ARG, "draft_logits is NULL with temperature > 0");
    const size_t esz = dims->logit_dtype == CS_F32 ? 4 : 2;
    if (!aligned(target_logits, esz) || (draft_logits && !aligned(draft_logits, esz)))
        return fail(CS_ERR_INVALID_ARG, "logit pointers must be aligned to their element size");
    if (!aligned(draft_tokens, 4) || !aligned(uniforms, 4) || !aligned(out_tokens, 4) ||
        !aligned(out_n_accepted, 4))
        return fail(CS_ERR_INVALID_ARG, "int32/fp32 pointers must be 4-byte aligned");
    const size_t need = accept_workspace_bytes(*dims, n_draft, temperature);
    if (!workspace || workspace_bytes < need)
        return fail(CS_ERR_WORKSPACE, "workspace of %zu bytes given, %zu needed", workspace_bytes, need);
    if (!aligned(workspace, 256)) return fail(CS_ERR_INVALID_ARG, "workspace must be 256-byte aligned");
    return launch_spec_accept(*dims, target_logits, temperature > 0.f ? draft_logits : nullptr,
                              draft_tokens, uniforms, n_draft, temperature, out_tokens,
                              out_n_accepted, workspace, reinterpret_cast<cudaStream_t>(stream));
}

cs_status cs_kv_append(const cs_attn_dims* dims, const void* new_k, const void* new_v, void* k_pages,
                       void* v_pages, const int32_t* page_table, const int32_t* ctx_lens, int32_t n_new,
                       cs_stream_t stream) {
    if (!dims) return fail(CS_ERR_INVALID_ARG, "dims is NULL");
    const cs_attn_dims* d = dims;
    if (d->batch < 0) return fail(CS_ERR_INVALID_ARG, "batch %d < 0", d->batch);
    if (d->n_kv_heads <= 0 || d->page_size <= 0 || d->max_pages_per_seq <= 0 || d->num_pages <= 0)
        return fail(CS_ERR_INVALID_ARG, "n_kv_heads, page_size, max_pages_per_seq and num_pages must be positive");
    if (d->head_dim != 128) return fail(CS_ERR_UNSUPPORTED, "head_dim %d (this library implements 128)", d->head_dim);
    if (n_new < 1 || n_new > 4096) return fail(CS_ERR_INVALID_ARG, "n_new %d not in [1, 4096]", n_new);
    if ((long long)d->max_pages_per_seq * d->page_size > (1LL << 30))
        return fail(CS_ERR_INVALID_ARG, "max_pages_per_seq * page_size exceeds 2^30 keys");
    if (d->batch == 0) return CS_OK;
    if (!new_k || !new_v || !k_pages || !v_pages || !page_table || !ctx_lens)
        return fail(CS_ERR_INVALID_ARG, "a tensor pointer is NULL");
    if (!aligned(new_k, 16) || !aligned(new_v, 16) || !aligned(k_pages, 16) || !aligned(v_pages, 16))
        return fail(CS_ERR_INVALID_ARG, "new rows and page pools must be 16-byte aligned");
    if (!aligned(page_table, 4) || !aligned(ctx_lens, 4))
        return fail(CS_ERR_INVALID_ARG, "page_table and ctx_lens must be 4-byte aligned");
    return launch_kv_append(*d, new_k, new_v, k_pages, v_pages, page_table, ctx_lens, n_new,
                            reinterpret_cast<cudaStream_t>(stream));
}

cs_status cs_kv_commit(int32_t batch, int32_t* ctx_lens, const int32_t* n_accepted, int32_t n_draft,
                       cs_stream_t stream) {
    if (batch < 0) return fail(CS_ERR_INVALID_ARG, "batch %d < 0", batch);
    if (n_draft < 0 || n_draft > 16) return fail(CS_ERR_INVALID_ARG, "n_draft %d not in [0, 16]", n_draft);
    if (batch == 0) return CS_OK;
    if (!ctx_lens || !n_accepted) return fail(CS_ERR_INVALID_ARG, "a tensor pointer is NULL");
    if (!aligned(ctx_lens, 4) || !aligned(n_accepted, 4))
        return fail(CS_ERR_INVALID_ARG, "ctx_lens and n_accepted must be 4-byte aligned");
    return launch_kv_commit(ctx_lens, n_accepted, batch, n_draft, reinterpret_cast<cudaStream_t>(stream));
}

size_t cs_route_workspace_bytes(const cs_route_dims* dims) {
    if (check_route(dims) != CS_OK) return 0;
    return plan_route(*dims, current_sm_count()).bytes;
}

cs_status cs_route_norms(int32_t n_groups, int32_t dim, const void* centroids, float* inv_norms,
                         cs_stream_t stream) {
    if (n_groups < 0) return fail(CS_ERR_INVALID_ARG, "n_groups %d < 0", n_groups);
    if (dim <= 0 || dim % 64 != 0 || dim > CS_MAX_ROUTE_DIM)
        return fail(CS_ERR_UNSUPPORTED, "dim %d (supported: multiples of 64 up to %d)", dim, CS_MAX_ROUTE_DIM);
    if (n_groups == 0) return CS_OK;
    if (!centroids || !inv_norms) return fail(CS_ERR_INVALID_ARG, "a tensor pointer is NULL");
    if (!aligned(centroids, 16) || !aligned(inv_norms, 4))
        return fail(CS_ERR_INVALID_ARG, "centroids must be 16-byte and inv_norms 4-byte aligned");
    return launch_route_norms(n_groups, dim, centroids, inv_norms, reinterpret_cast<cudaStream_t>(stream));
}

cs_status cs_route(const cs_route_dims* dims, const void* emb, const void* centroids, const float* inv_norms,
                   float tau, int32_t* out_group, int32_t* out_best, float* out_score, void* workspace,
                   size_t workspace_bytes, cs_stream_t stream) {
    cs_status st = check_route(dims);
    if (st != CS_OK) return st;
    if (isnan(tau) || isinf(tau)) return fail(CS_ERR_INVALID_ARG, "tau is not finite");
    if (dims->batch == 0) return CS_OK;
    if (!emb || !out_group || !out_best || !out_score) return fail(CS_ERR_INVALID_ARG, "a tensor pointer is NULL");
    if (dims->n_groups > 0 && (!centroids || !inv_norms))
        return fail(CS_ERR_INVALID_ARG, "centroids and inv_norms are NULL with n_groups > 0");
    if (!aligned(emb, 16) || (centroids && !aligned(centroids, 16)))
        return fail(CS_ERR_INVALID_ARG, "emb and centroids must be 16-byte aligned");
    if ((inv_norms && !aligned(inv_norms, 4)) || !aligned(out_group, 4) || !aligned(out_best, 4) ||
        !aligned(out_score, 4))
        return fail(CS_ERR_INVALID_ARG, "int32/fp32 pointers must be 4-byte aligned");
    const RoutePlan pl = plan_route(*dims, current_sm_count());
    if (!workspace || workspace_bytes < pl.bytes)
        return fail(CS_ERR_WORKSPACE, "workspace of %zu bytes given, %zu needed", workspace_bytes, pl.bytes);
    if (!aligned(workspace, 256)) return fail(CS_ERR_INVALID_ARG, "workspace must be 256-byte aligned");
    return launch_route(*dims, pl, emb, centroids, inv_norms, tau, out_group, out_best, out_score, workspace,
                        reinterpret_cast<cudaStream_t>(stream));
}

size_t cs_sample_workspace_bytes(const cs_accept_dims* dims) {
    if (check_sample(dims, 1.0f) != CS_OK) return 0;
    return accept_workspace_bytes_any(*dims, 0);
}

cs_status cs_sample(const cs_accept_dims* dims, const void* logits, const float* uniforms,
                    float temperature, int32_t* out_tokens, void* workspace, size_t workspace_bytes,
                    cs_stream_t stream) {
    cs_status st = check_sample(dims, temperature);
    if (st != CS_OK) return st;
    if (dims->batch == 0) return CS_OK;
    if (!logits || !uniforms || !out_tokens) return fail(CS_ERR_INVALID_ARG, "a tensor pointer is NULL");
    const size_t esz = dims->logit_dtype == CS_F32 ? 4 : 2;
    if (!aligned(logits, esz)) return fail(CS_ERR_INVALID_ARG, "logits must be aligned to their element size");
    if (!aligned(uniforms, 4) || !aligned(out_tokens, 4))
        return fail(CS_ERR_INVALID_ARG, "int32/fp32 pointers must be 4-byte aligned");
    const size_t need = accept_workspace_bytes(*dims, 0, temperature);
    if (!workspace || workspace_bytes < need)
        return fail(CS_ERR_WORKSPACE, "workspace of %zu bytes given, %zu needed", workspace_bytes, need);
    if (!aligned(workspace, 256)) return fail(CS_ERR_INVALID_ARG, "workspace must be 256-byte aligned");
    // the acceptance path with no drafted positions: every request decides
    // a = 0 and draws its token from p_0 (or takes its argmax when T == 0)
    return launch_spec_accept(*dims, logits, nullptr, nullptr, uniforms, 0, temperature, out_tokens,
                              nullptr, workspace, reinterpret_cast<cudaStream_t>(stream));
}

cs_status cs_selftest_wait_timeout(void* workspace, cs_stream_t stream) {
    if (!workspace) return fail(CS_ERR_INVALID_ARG, "workspace is NULL");
    if (!aligned(workspace, 4)) return fail(CS_ERR_INVALID_ARG, "workspace must be 4-byte aligned");
    const cudaError_t e = launch_wait_selftest(static_cast<int*>(workspace), reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "wait self-test launch");
    return CS_OK;
}

cs_status cs_read_device_status(const void* workspace, int32_t* status_out, cs_stream_t stream) {
    if (!workspace || !status_out) return fail(CS_ERR_INVALID_ARG, "NULL argument");
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    cudaError_t e = cudaMemcpyAsync(status_out, workspace, sizeof(int32_t), cudaMemcpyDeviceToHost, s);
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpyAsync(status)");
    e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
    return CS_OK;
}

}  // extern "C"
