// kv_cache.cu -- the paged KV cache around the verify pass: appending the
// K/V rows of the k+1 verify positions before verify attention, and
// committing the accepted prefix after the acceptance step (the target's
// draft-and-verify step, Sec. 3.4; the positions follow the convention of
// cs_verify_attention: ctx_lens counts the k+1 verify positions).
//
// Append: one thread moves 16 bytes; 16 threads move one 256-byte row of one
// head (D = 128 bf16), so every load of the new rows and every store into a
// page slot is a contiguous 256-byte segment.  Commit is one thread per
// request.
//
// Tree commit (after a token-tree acceptance): the accepted nodes' rows move,
// in walk order, to the positions right after the root.  Node path[i] sat at
// L - n + path[i] >= L - n + 1 + i, so with the rows taken in ascending i no
// source is an earlier destination; the 16 threads of a (request, head,
// K or V) group each own one 16-byte column and copy it row after row, so a
// destination that overwrites an earlier source is written by the thread
// that already read that source.
#include "cs_device.cuh"
#include "cs_internal.h"

namespace cs {
namespace {

constexpr int kAppendThreads = 256;
constexpr int kRowThreads = 16;   // 16 x 16 B = one 128-dim bf16 row

struct AppendParams {
    const uint4* new_k;        // [B, n_new, Hkv, D]
    const uint4* new_v;
    uint4* k_pages;            // [P, Hkv, ps, D]
    uint4* v_pages;
    const int32_t* page_table; // [B, max_pages]
    const int32_t* ctx_lens;   // [B]
    long long rows;            // B * n_new * Hkv
    int n_new, Hkv, ps, max_pages, P;
};

__global__ void __launch_bounds__(kAppendThreads) kv_append_kernel(const AppendParams p) {
    const long long t = (long long)blockIdx.x * kAppendThreads + threadIdx.x;
    const long long r = t / kRowThreads;   // (b, i, h) row of the new K/V
    const int c = (int)(t % kRowThreads);
    if (r >= p.rows) return;
    const int h = (int)(r % p.Hkv);
    const long long bi = r / p.Hkv;
    const int i = (int)(bi % p.n_new);
    const int b = (int)(bi / p.n_new);
    int L = __ldg(p.ctx_lens + b);
    L = max(0, min(L, p.max_pages * p.ps));
    const int pos = L - p.n_new + i;          // key position of verify row i
    if (pos < 0) return;                      // the context cannot hold this row
    const int page = __ldg(p.page_table + (size_t)b * p.max_pages + pos / p.ps);
    if (page < 0 || page >= p.P) return;      // no such page: nothing is written
    const size_t dst = (((size_t)page * p.Hkv + h) * p.ps + pos % p.ps) * kRowThreads + c;
    const size_t src = (size_t)r * kRowThreads + c;
    p.k_pages[dst] = __ldg(p.new_k + src);
    p.v_pages[dst] = __ldg(p.new_v + src);
}

__global__ void kv_commit_kernel(int32_t* ctx_lens, const int32_t* n_accepted, int batch, int n_draft) {
    const int b = blockIdx.x * blockDim.x + threadIdx.x;
    if (b >= batch) return;
    // rows kept: the prefix, the verify input token and the accepted drafts
    const int L = ctx_lens[b] - n_draft + __ldg(n_accepted + b);
    ctx_lens[b] = L > 0 ? L : 0;
}

constexpr int kTreeCommitThreads = 256;

struct TreeCommitParams {
    uint4* k_pages;            // [P, Hkv, ps, D]
    uint4* v_pages;
    const int32_t* page_table; // [B, max_pages]
    const int32_t* ctx_lens;   // [B]
    const int32_t* path;       // [B, n]
    const int32_t* n_accepted; // [B]
    long long groups;          // B * Hkv * 2 (K and V)
    int n, Hkv, ps, max_pages, P;
};

__global__ void __launch_bounds__(kTreeCommitThreads) kv_commit_tree_kernel(const TreeCommitParams p) {
    const long long t = (long long)blockIdx.x * kTreeCommitThreads + threadIdx.x;
    const long long g = t / kRowThreads;
    const int c = (int)(t % kRowThreads);
    if (g >= p.groups) return;
    const int kv = (int)(g & 1);
    const int h = (int)((g >> 1) % p.Hkv);
    const int b = (int)((g >> 1) / p.Hkv);
    int L = __ldg(p.ctx_lens + b);
    L = max(0, min(L, p.max_pages * p.ps));
    const int a = max(0, min(__ldg(p.n_accepted + b), p.n - 1));
    const int base = L - p.n;
    uint4* pool = kv ? p.v_pages : p.k_pages;
    const int32_t* table = p.page_table + (size_t)b * p.max_pages;
    for (int i = 0; i < a; ++i) {
        const int node = __ldg(p.path + (size_t)b * p.n + i);
        if (node < 1 || node >= p.n) continue;
        const int src = base + node, dst = base + 1 + i;
        if (src == dst || dst < 0) continue;
        const int sp = __ldg(table + src / p.ps), dp = __ldg(table + dst / p.ps);
        if (sp < 0 || sp >= p.P || dp < 0 || dp >= p.P) continue;
        const uint4 v = pool[(((size_t)sp * p.Hkv + h) * p.ps + src % p.ps) * kRowThreads + c];
        pool[(((size_t)dp * p.Hkv + h) * p.ps + dst % p.ps) * kRowThreads + c] = v;
    }
}

// The kept length after a tree commit: the prefix, the root and the a
// accepted nodes (a clamped to [0, n-1], L to the page capacity).
__global__ void kv_commit_tree_len_kernel(int32_t* ctx_lens, const int32_t* n_accepted, int batch, int n,
                                          int cap) {
    const int b = blockIdx.x * blockDim.x + threadIdx.x;
    if (b >= batch) return;
    const int L = max(0, min(ctx_lens[b], cap));
    const int a = max(0, min(__ldg(n_accepted + b), n - 1));
    ctx_lens[b] = max(0, L - n + 1 + a);
}

}  // namespace

cs_status launch_kv_commit_tree(const cs_attn_dims& d, void* k_pages, void* v_pages, const int32_t* page_table,
                                int32_t* ctx_lens, const int32_t* path, const int32_t* n_accepted, int n_nodes,
                                cudaStream_t stream) {
    TreeCommitParams p{};
    p.k_pages = static_cast<uint4*>(k_pages);
    p.v_pages = static_cast<uint4*>(v_pages);
    p.page_table = page_table;
    p.ctx_lens = ctx_lens;
    p.path = path;
    p.n_accepted = n_accepted;
    p.groups = (long long)d.batch * d.n_kv_heads * 2;
    p.n = n_nodes;
    p.Hkv = d.n_kv_heads;
    p.ps = d.page_size;
    p.max_pages = d.max_pages_per_seq;
    p.P = d.num_pages;
    const long long blocks = (p.groups * kRowThreads + kTreeCommitThreads - 1) / kTreeCommitThreads;
    if (blocks > 0x7fffffffLL) return fail(CS_ERR_UNSUPPORTED, "too many rows to commit in one call");
    kv_commit_tree_kernel<<<(unsigned)blocks, kTreeCommitThreads, 0, stream>>>(p);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_fail(e, "kv_commit_tree_kernel launch");
    kv_commit_tree_len_kernel<<<(d.batch + 255) / 256, 256, 0, stream>>>(ctx_lens, n_accepted, d.batch, n_nodes,
                                                                        d.max_pages_per_seq * d.page_size);
    e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_fail(e, "kv_commit_tree_len_kernel launch");
    return CS_OK;
}

cs_status launch_kv_append(const cs_attn_dims& d, const void* new_k, const void* new_v, void* k_pages,
                           void* v_pages, const int32_t* page_table, const int32_t* ctx_lens, int n_new,
                           cudaStream_t stream) {
    AppendParams p{};
    p.new_k = static_cast<const uint4*>(new_k);
    p.new_v = static_cast<const uint4*>(new_v);
    p.k_pages = static_cast<uint4*>(k_pages);
    p.v_pages = static_cast<uint4*>(v_pages);
    p.page_table = page_table;
    p.ctx_lens = ctx_lens;
    p.rows = (long long)d.batch * n_new * d.n_kv_heads;
    p.n_new = n_new;
    p.Hkv = d.n_kv_heads;
    p.ps = d.page_size;
    p.max_pages = d.max_pages_per_seq;
    p.P = d.num_pages;
    const long long threads = p.rows * kRowThreads;
    const long long blocks = (threads + kAppendThreads - 1) / kAppendThreads;
    if (blocks > 0x7fffffffLL) return fail(CS_ERR_UNSUPPORTED, "too many rows to append in one call");
    kv_append_kernel<<<(unsigned)blocks, kAppendThreads, 0, stream>>>(p);
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_fail(e, "kv_append_kernel launch");
    return CS_OK;
}

cs_status launch_kv_commit(int32_t* ctx_lens, const int32_t* n_accepted, int batch, int n_draft,
                           cudaStream_t stream) {
    kv_commit_kernel<<<(batch + 255) / 256, 256, 0, stream>>>(ctx_lens, n_accepted, batch, n_draft);
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_fail(e, "kv_commit_kernel launch");
    return CS_OK;
}

}  // namespace cs
