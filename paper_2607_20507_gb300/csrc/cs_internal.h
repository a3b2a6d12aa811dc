// cs_internal.h -- host-side interface between the C ABI (capi.cu) and the
// kernel launchers.  Not installed; the public surface is include/cachespec.h.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "cachespec.h"

namespace cs {

// Records a printf-style message for cs_last_error() and returns `st`.
cs_status fail(cs_status st, const char* fmt, ...);
cs_status cuda_fail(cudaError_t e, const char* what);

// Streaming multiprocessors of the current device (cached per device).
int current_sm_count();

// ------------------------------------------------------------- attention
struct AttnPlan {
    int group;        // G = Hq / Hkv
    int rows;         // k + 1 (chain) or the tree's node count
    bool tree;        // tree mask (parents given) instead of the causal chain
    int n_rows_all;   // rows * G query rows per KV head
    int n_rb;         // row blocks per KV head (each one span of the schedule)
    int n_rows;       // query rows per row block (n_rows_all when n_rb == 1)
    int row_warps;    // ceil(n_rows / 16) warps of query rows
    int split;        // consumer groups sharing each tile's keys (1 or 2)
    bool tc;          // the tcgen05 kernel (33..128 rows, one row block)
    int grid;         // persistent CTAs (resident capacity of the device)
    size_t off_part_o, off_part_ml, off_part_span, bytes;   // workspace layout (status word at 0)
};
AttnPlan plan_verify_attention(const cs_attn_dims& d, int n_draft, int sm_count);
AttnPlan plan_tree_attention(const cs_attn_dims& d, int n_nodes, int sm_count);

// parents: NULL for the causal chain, the [B, rows] parent array for a tree
// (must match plan.tree)
// The failure-detection self-test (cs_selftest_wait_timeout).
cudaError_t launch_wait_selftest(int* status, cudaStream_t stream);

cs_status launch_verify_attention(const cs_attn_dims& d, const AttnPlan& plan, const void* q,
                                  const void* k_pages, const void* v_pages,
                                  const int32_t* page_table, const int32_t* ctx_lens,
                                  const int32_t* parents, void* out, void* workspace,
                                  cudaStream_t stream);

// ------------------------------------------------------------ acceptance
size_t accept_workspace_bytes(const cs_accept_dims& d, int n_draft, float temperature);
// The larger of the sampling and greedy requirements.
size_t accept_workspace_bytes_any(const cs_accept_dims& d, int n_draft);
cs_status launch_spec_accept(const cs_accept_dims& d, const void* target, const void* draft,
                             const int32_t* tokens, const float* uniforms, int n_draft,
                             float temperature, int32_t* out_tokens, int32_t* out_n,
                             void* workspace, cudaStream_t stream);

// token trees: target and draft rows [B, n, V], parents / tokens /
// uniforms [B, n]; outputs tokens and path [B, n], accepted count [B]
size_t tree_accept_workspace_bytes(const cs_accept_dims& d, int n_nodes);
cs_status launch_tree_accept(const cs_accept_dims& d, const void* target, const void* draft,
                             const int32_t* parents, const int32_t* tokens, const float* uniforms, int n_nodes,
                             float temperature, int32_t* out_tokens, int32_t* out_path, int32_t* out_n,
                             void* workspace, cudaStream_t stream);

// ------------------------------------------------------------- KV cache
cs_status launch_kv_append(const cs_attn_dims& d, const void* new_k, const void* new_v, void* k_pages,
                           void* v_pages, const int32_t* page_table, const int32_t* ctx_lens, int n_new,
                           cudaStream_t stream);
cs_status launch_kv_commit(int32_t* ctx_lens, const int32_t* n_accepted, int batch, int n_draft,
                           cudaStream_t stream);
cs_status launch_kv_commit_tree(const cs_attn_dims& d, void* k_pages, void* v_pages, const int32_t* page_table,
                                int32_t* ctx_lens, const int32_t* path, const int32_t* n_accepted, int n_nodes,
                                cudaStream_t stream);

// -------------------------------------------------------------- routing
constexpr int kMaxRouteDim = CS_MAX_ROUTE_DIM;
struct RoutePlan {
    int m_tiles, n_tiles;   // 128-request and 128-group tiles
    long long items;        // m_tiles * n_tiles (request tile, group tile) pairs
    int grid;               // persistent CTAs, each an equal contiguous item range
    int seg_slots;          // partial slots per request tile
    size_t bytes;           // workspace: status word (256 B), then [m_tiles, seg_slots, 128] partials
};
RoutePlan plan_route(const cs_route_dims& d, int sm_count);
cs_status launch_route(const cs_route_dims& d, const RoutePlan& pl, const void* emb, const void* centroids,
                       const float* inv_norms, float tau, int32_t* out_group, int32_t* out_best,
                       float* out_score, void* workspace, cudaStream_t stream);
cs_status launch_route_norms(int n_groups, int dim, const void* centroids, float* inv_norms, cudaStream_t stream);

}  // namespace cs
