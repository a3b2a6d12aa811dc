// verify_attention.cu -- multi-query GQA verify attention over a paged KV
// cache (the KV-bound core of the target's verify pass in the paper's
// draft-and-verify step, Sec. 3.4).
//
// Schedule (persistent, balanced).  The work is the flattened sequence of
// 64-key tiles of every (request b, KV head h) span, requests in order, heads
// in order, tiles in key order; span (b, h) has T_b = ceil(L_b / 64) tiles.
// The grid holds exactly as many CTAs as are resident at once; each span also
// costs a few work units for its start, and CTA c takes the tiles of units
// [cU/G, (c+1)U/G) (tiles_before below), so the CTAs' work evens out.  A span
// that lies inside one CTA's range is finished there and written in bf16;
// a span cut by range boundaries leaves one partial per piece -- the piece's
// own normalised output and its (m, l) -- (each CTA writes at most two: its
// first and its last piece), and a second small kernel merges the pieces of
// every cut span with log-sum-exp weights, all spans in parallel.
//
// Token trees (the multi-candidate verification variant) use the same
// kernel with a different mask: node i of a request's tree sees every prefix
// key and the rows of its own ancestors, found from the parent array by
// pointer doubling at the start of each span.  A tree whose (nodes x G)
// query rows exceed what one CTA holds is cut into row blocks, each its own
// span ("virtual head") over the same keys.
//
// With few query rows (at most 32 per KV head) every 64-key tile is split
// between two consumer warp groups, each running its own online softmax over
// 32 of the keys; the two states of a row are folded in shared memory when a
// span piece ends.  Twice the warps then hide the latency of the mma.sync
// chains, which otherwise pace the tile rate.
//
// Per CTA: one producer warp streams the K and V tiles of its range through
// TMA into a 3-stage shared-memory ring guarded by mbarriers, without
// draining between spans.  One 5-D tensor map covers each page pool as
// (64 dims, keys, 2 dim halves, heads, pages): a box is both 128-byte halves
// of up to 64 keys of one page and head, landing as [half][key][64 dims]
// with the 128-byte swizzle, so a 16-token page is one 4 KB copy.  The page
// ids of the next 32 / pieces tiles come from one warp-wide load issued a
// batch ahead, and the page table is prefetched into L2 at launch.
// Consumer warps own 16 of the (k+1)*G query rows of the current span each
// (draft row i = r / G, query head h*G + r % G), so every K/V byte staged in
// shared memory serves all rows; they run S = Q K^T and O += P V on bf16
// tensor cores (mma.sync m16n8k16, fp32 accumulate) with an fp32 online
// softmax in the log2 domain.  V is used as stored; P enters the product as
// the sum of two bf16 terms (hi + lo, ~16 significant bits: bf16 P alone
// rounds the weights coarsely enough to exceed 2e-3 + 1e-2|o| on rows whose
// terms cancel), and it is formed as P * 2^-64, a factor the row sum carries
// too, so that no partial sum of P.V can overflow fp32 for any finite bf16 V.
#include <math.h>
#include <stdio.h>

#include <type_traits>

#include <cudaTypedefs.h>

#include "cs_device.cuh"
#include "cs_internal.h"

namespace cs {
namespace {

constexpr int kD = 128;                       // head dim implemented
constexpr int kTileT = 64;                    // keys per pipeline tile
constexpr int kTensorTileBytes = kTileT * 256; // 64 keys x 128 dims x 2 B
constexpr int kStageBytes = 2 * kTensorTileBytes;   // K + V
constexpr int kStages = 3;
constexpr int kMaxRowWarps = 9;               // 144 query rows
constexpr int kMaxSplitRowWarps = 2;          // key-split consumers: up to 32 query rows
constexpr int kMaxBatchPerLaunch = 1024;      // requests whose schedule one launch holds
constexpr int kMaxGrid = 512;                 // persistent CTAs at most (slot list size)
constexpr int kMinTilesPerCta = 8;            // 256 KB of K/V per CTA before a span is cut
constexpr int kBarrierBytes = 128;
constexpr int kSmemBytes = kStages * kStageBytes + kBarrierBytes +
                           (kMaxBatchPerLaunch + 1) * 8 /*prefix*/ + kMaxBatchPerLaunch * 4 /*L*/ +
                           1024 /*alignment slack*/;

struct AttnParams {
    const __nv_bfloat16* q;      // [B, R, Hq, D]
    __nv_bfloat16* out;          // [B, R, Hq, D]
    const int32_t* page_table;   // [B, max_pages]
    const int32_t* ctx_lens;     // [B]
    const int32_t* parents;      // [B, R] tree parents (tree kernel only)
    float* part_o;               // [2 * grid, n_rows, D]
    float2* part_ml;             // [2 * grid, n_rows]  (m in log2 units, l)
    int* part_span;              // [2 * grid] span (b * n_vh + h) of each partial slot, -1 if unused
    int* status;
    int Hq, Hkv, G, R, n_rows, ps, box_t, max_pages, row_warps;
    int n_rb;                    // row blocks per KV head (n_rows rows each)
    int n_vh;                    // Hkv * n_rb spans per request ("virtual heads")
    int n_rows_all;              // R * G query rows per KV head
    int tc_stages, tc_vstages;   // tcgen05 kernel: K and V ring depths
    int tc_q_half;               // tcgen05 kernel: bytes between query dim halves
    int b_base, n_batch;         // requests [b_base, b_base + n_batch) in this launch
    int span_x;                  // work units charged to each span's start (see tiles_before)
    float scale_log2;            // sm_scale * log2(e)
};

__device__ __forceinline__ void flag_timeout(int* status) {
    atomicOr(status, CS_DEVICE_WAIT_TIMEOUT);
}

__device__ __forceinline__ int tiles_of(int L) { return max(1, (L + kTileT - 1) / kTileT); }

// The CTA whose range holds work unit v (ranges start at floor(c*U/G)).
__device__ __forceinline__ int owner_of(long long v, long long U, int G) {
    return (int)(((v + 1) * G + U - 1) / U) - 1;
}

// The work split.  Every span (request, KV head or row block) costs its T
// tiles plus X units for starting it (query rows, epilogue: a CTA's time
// grows with the span pieces it holds).  In the sequence of work units --
// each span's X start units, then its T tiles -- CTA c of G takes units
// [floor(c U / G), floor((c+1) U / G)) of U = W + X * n_vh * B, i.e. the
// tiles whose unit index falls there.  tiles_before(v) counts the tiles
// whose unit index is below v; request b's units start at
// prefix[b] + X * n_vh * b (prefix: its first tile).
__device__ __forceinline__ long long tiles_before(long long v, const long long* prefix, const int* lens,
                                                  int n_batch, int n_vh, int X) {
    if (v <= 0) return 0;
    int lo = 0, hi = n_batch - 1;   // largest b whose units start at or below v
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (prefix[mid] + (long long)X * n_vh * mid <= v) lo = mid;
        else hi = mid - 1;
    }
    const int T = tiles_of(lens[lo]);
    const long long local = v - (prefix[lo] + (long long)X * n_vh * lo);
    const int S = T + X;
    // local < (n_vh + 1) * S: one 32-bit division whenever that fits
    const long long h = local <= 0x7fffffffLL ? (long long)((unsigned)local / (unsigned)S) : local / S;
    if (h >= n_vh) return prefix[lo] + (long long)n_vh * T;   // past the last unit
    const long long tv = local - h * S;
    return prefix[lo] + h * T + (tv > X ? tv - X : 0);
}

// floor(c * U / G) for the unit range of CTA c
__device__ __forceinline__ long long unit_start(int c, long long U, int G) {
    const long long n = (long long)c * U;
    return n <= 0xffffffffLL ? (long long)((unsigned)n / (unsigned)G) : n / G;
}

// Position of flat tile f in the schedule: request (launch-local), head, tile.
struct Cursor {
    int b, h, t, T;
};

__device__ __forceinline__ Cursor locate(long long f, const long long* prefix, const int* lens,
                                         int n_batch, int n_vh) {
    int lo = 0, hi = n_batch - 1;   // largest b with prefix[b] <= f
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (prefix[mid] <= f) lo = mid;
        else hi = mid - 1;
    }
    Cursor c;
    c.b = lo;
    c.T = tiles_of(lens[lo]);
    const long long local = f - prefix[lo];
    c.h = (int)(local / c.T);
    c.t = (int)(local % c.T);
    return c;
}

__device__ __forceinline__ void advance(Cursor& c, const int* lens, int n_batch, int n_vh) {
    if (++c.t < c.T) return;
    c.t = 0;
    if (++c.h < n_vh) return;
    c.h = 0;
    if (++c.b < n_batch) c.T = tiles_of(lens[c.b]);
}

// Ancestor-or-self bit masks of tree nodes `lane` and `lane + 32` (n <= 64
// nodes; a parent outside [0, c) detaches node c).  Pointer doubling: after
// round r a node's mask holds its ancestors closer than 2^(r+1) levels and
// its jump points 2^(r+1) levels up, so six rounds cover any depth < 64.
__device__ __forceinline__ void tree_ancestor_masks(const int32_t* par, int n, int lane, uint64_t& m0,
                                                    uint64_t& m1) {
    const int c0 = lane, c1 = lane + 32;
    int j0 = -1, j1 = -1;
    if (c0 > 0 && c0 < n) {
        const int q = __ldg(par + c0);
        j0 = (q >= 0 && q < c0) ? q : -1;
    }
    if (c1 < n) {
        const int q = __ldg(par + c1);
        j1 = (q >= 0 && q < c1) ? q : -1;
    }
    m0 = c0 < n ? (1ull << c0) : 0ull;
    m1 = c1 < n ? (1ull << c1) : 0ull;
#pragma unroll
    for (int r = 0; r < 6; ++r) {
        const int s0 = j0 & 31, s1 = j1 & 31;
        const uint64_t a0 = __shfl_sync(0xffffffffu, m0, s0), a1 = __shfl_sync(0xffffffffu, m1, s0);
        const int ja0 = __shfl_sync(0xffffffffu, j0, s0), ja1 = __shfl_sync(0xffffffffu, j1, s0);
        const uint64_t b0 = __shfl_sync(0xffffffffu, m0, s1), b1 = __shfl_sync(0xffffffffu, m1, s1);
        const int jb0 = __shfl_sync(0xffffffffu, j0, s1), jb1 = __shfl_sync(0xffffffffu, j1, s1);
        if (j0 >= 0) {
            m0 |= j0 >= 32 ? a1 : a0;
            j0 = j0 >= 32 ? ja1 : ja0;
        }
        if (j1 >= 0) {
            m1 |= j1 >= 32 ? b1 : b0;
            j1 = j1 >= 32 ? jb1 : jb0;
        }
    }
}

// kSplit: consumer warp groups that share each tile (1, or 2 when the query
// rows fit two row warps: each group takes 32 of the tile's 64 keys)
template <bool kTree, int kBoxT, int kSplit>
__global__ void __launch_bounds__(kSplit == 1 ? (kMaxRowWarps + 1) * 32 : (2 * kMaxSplitRowWarps + 1) * 32,
                                  kSplit == 1 ? 1 : 2)
verify_attention_kernel(const __grid_constant__ CUtensorMap tmap_k,
                        const __grid_constant__ CUtensorMap tmap_v, const AttnParams p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + kStages * kStageBytes);
    uint64_t* empty = full + kStages;
    uint64_t* fold_a = empty + kStages;   // key-split: every consumer is done with the stage
    uint64_t* fold_b = fold_a + 1;        // key-split: the second group's state is in the stage
    long long* s_prefix = reinterpret_cast<long long*>(smem + kStages * kStageBytes + kBarrierBytes);
    int* s_len = reinterpret_cast<int*>(s_prefix + kMaxBatchPerLaunch + 1);
    __shared__ long long s_wtot[kMaxRowWarps + 1];
    __shared__ long long s_carry;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nw = p.row_warps;
    const int nb = p.n_batch;
    // the page table of this launch into L2, spread over the CTAs, while the
    // schedule is computed (the producer's first lookups then hit L2)
    if (warp == kSplit * nw) {
        const char* tab = reinterpret_cast<const char*>(p.page_table + (size_t)p.b_base * p.max_pages);
        const long long lines = ((long long)nb * p.max_pages * 4 + 127) / 128;
        for (long long i = (long long)blockIdx.x * 32 + lane; i < lines; i += (long long)gridDim.x * 32)
            asm volatile("prefetch.global.L2 [%0];" ::"l"(tab + i * 128));
    }

    // ---- schedule: exclusive prefix of tiles per request (x heads), clamped L
    if (threadIdx.x == 0) {
        s_carry = 0;
        for (int i = 0; i < kStages; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], kSplit * nw);
        }
        mbar_init(fold_a, kSplit * nw);
        mbar_init(fold_b, nw);
        fence_barrier_init();
    }
    // launched as a programmatic dependent of the kernel before it: the
    // prologue above overlaps that kernel, every input is read below.  The
    // merge kernel (this kernel's dependent) may then start and work out its
    // schedule while this one runs.
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    __syncthreads();
    const int l_cap = p.max_pages * p.ps;
    for (int base = 0; base < nb; base += blockDim.x) {
        const int bl = base + threadIdx.x;
        long long v = 0;
        if (bl < nb) {
            int L = __ldg(p.ctx_lens + p.b_base + bl);
            L = max(0, min(L, l_cap));
            s_len[bl] = L;
            v = (long long)tiles_of(L) * p.n_vh;
        }
        long long inc = v;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const long long y = __shfl_up_sync(0xffffffffu, inc, off);
            if (lane >= off) inc += y;
        }
        if (lane == 31) s_wtot[warp] = inc;
        __syncthreads();
        long long before = s_carry;
        for (int w = 0; w < warp; ++w) before += s_wtot[w];
        if (bl < nb) s_prefix[bl] = before + inc - v;
        __syncthreads();
        if (threadIdx.x == blockDim.x - 1) s_carry = before + inc;
        __syncthreads();
    }
    if (threadIdx.x == 0) s_prefix[nb] = s_carry;
    __syncthreads();

    const long long W = s_prefix[nb];
    // at least kMinTilesPerCta tiles per CTA: small problems use fewer CTAs
    // rather than cutting every span into one-tile pieces
    const long long g_need = (W + kMinTilesPerCta - 1) / kMinTilesPerCta;
    const int Gc = (int)(g_need < (long long)gridDim.x ? (g_need > 0 ? g_need : 1) : gridDim.x);
    const int cta = blockIdx.x;
    // this CTA's two partial slots start unused (thread 0 -- row warp 0,
    // lane 0 -- is also the one that records a partial's span below)
    if (threadIdx.x == 0) {
        p.part_span[2 * cta] = -1;
        p.part_span[2 * cta + 1] = -1;
    }
    if (cta >= Gc) return;
    const long long U = W + (long long)p.span_x * p.n_vh * nb;
    const long long f0 = tiles_before(unit_start(cta, U, Gc), s_prefix, s_len, nb, p.n_vh, p.span_x);
    const long long f1 = tiles_before(unit_start(cta + 1, U, Gc), s_prefix, s_len, nb, p.n_vh, p.span_x);
    if (f0 >= f1) return;
    const int n_tiles = (int)(f1 - f0);
    const uint32_t smem_base = smem_u32(smem);

    if (warp == kSplit * nw) {
        // ------------------------------------------------------ producer
        // The whole warp produces: the next tile is issued once its stage is
        // free (lane pc owns page piece pc; the page ids of 32/pieces tiles
        // come from one warp-wide load issued a batch ahead).
        if (lane == 0) {
            tma_prefetch_desc(&tmap_k);
            tma_prefetch_desc(&tmap_v);
        }
        constexpr int pieces = kTileT / kBoxT;
        constexpr uint32_t piece_bytes = (uint32_t)kBoxT * 256u;   // both dim halves of kBoxT keys
        constexpr int per_batch = 32 / pieces;   // tiles whose page ids one warp-wide load covers
        // lane l: the page of piece l % pieces of tile j0 + l / pieces
        auto batch_pages = [&](int j0) -> int {
            const int jj = j0 + lane / pieces;
            if (jj >= n_tiles) return -1;
            const Cursor cc = locate(f0 + jj, s_prefix, s_len, nb, p.n_vh);
            const int tok = cc.t * kTileT + (lane % pieces) * kBoxT;
            if (tok >= s_len[cc.b]) return -1;
            return __ldg(p.page_table + (size_t)(p.b_base + cc.b) * p.max_pages + tok / p.ps);
        };
        Cursor cur = locate(f0, s_prefix, s_len, nb, p.n_vh);
        int pg_cur = batch_pages(0);
        int pg_next = per_batch < n_tiles ? batch_pages(per_batch) : -1;
        int jt = 0;   // next tile to issue
        uint32_t polls = 0;
        uint64_t t_idle = 0;
        while (jt < n_tiles) {
            bool progress = false;
            if (jt < n_tiles) {
                const int st = jt % kStages;
                int go = 1;
                if (lane == 0 && jt >= kStages) go = mbar_test_wait(&empty[st], (uint32_t)(jt / kStages - 1) & 1);
                if (__shfl_sync(0xffffffffu, go, 0)) {
                    const int jb = jt % per_batch;
                    if (jt > 0 && jb == 0) {
                        pg_cur = pg_next;
                        pg_next = jt + per_batch < n_tiles ? batch_pages(jt + per_batch) : -1;
                    }
                    const int page = __shfl_sync(0xffffffffu, pg_cur, jb * pieces + lane % pieces);
                    const int L = s_len[cur.b];
                    const int ts = cur.t * kTileT;
                    const int h_cur = cur.h / p.n_rb;   // the KV head of this span
                    advance(cur, s_len, nb, p.n_vh);
                    int valid = 0;
                    for (int pc = 0; pc < pieces; ++pc)
                        if (ts + pc * kBoxT < L) ++valid;
                    if (lane == 0) mbar_arrive_expect_tx(&full[st], (uint32_t)valid * piece_bytes * 2u);
                    __syncwarp();
                    if (lane < valid) {
                        const uint32_t kdst = smem_base + st * kStageBytes + (uint32_t)lane * piece_bytes;
                        const uint32_t vdst = kdst + kTensorTileBytes;
                        const int slot = (ts + lane * kBoxT) % p.ps;
                        tma_load_5d(kdst, &tmap_k, &full[st], 0, slot, 0, h_cur, page);
                        tma_load_5d(vdst, &tmap_v, &full[st], 0, slot, 0, h_cur, page);
                    }
                    ++jt;
                    progress = true;
                }
            }
            if (progress) {
                polls = 0;
            } else if ((++polls & 255u) == 0) {
                const uint64_t now = global_timer_ns();
                if (polls == 256) t_idle = now;
                else if (now - t_idle > 1000000000ull) {   // about one second without progress
                    if (lane == 0) flag_timeout(p.status);
                    break;
                }
            }
        }
        return;
    }

    // ---------------------------------------------------------- consumers
    // 128-byte row of (key, dim half) in a K or V tile: pieces of box_t keys,
    // each [half][key][64 dims]
    auto key_row = [](int key, int half) { return key + (key & ~(kBoxT - 1)) + half * kBoxT; };
    constexpr int kNT = 8 / kSplit;        // 8-key n-tiles of a warp's share of a tile
    const int kh = kSplit == 1 ? 0 : warp / nw;   // key share: keys [kh*64/kSplit, (kh+1)*64/kSplit) of a tile
    const int rw = warp - kh * nw;         // row warp: query rows [16 rw, 16 rw + 16)
    const int g = lane >> 2, tq = lane & 3;
    const int row0 = rw * 16 + g, row1 = row0 + 8;
    const int lm = lane >> 3, lr = lane & 7;   // ldmatrix: matrix index, row within it
    const float c = p.scale_log2;

    Cursor cur = locate(f0, s_prefix, s_len, nb, p.n_vh);
    int seg_t0 = cur.t;
    bool first_seg = true;
    int folds = 0;

    uint32_t qa[8][4];
    float o[16][4];
    float m_raw[2], l[2];
    int lim0 = 0, lim1 = 0;              // chain: exclusive key limit of each row
    uint64_t anc0 = ~0ull, anc1 = ~0ull;   // tree: ancestor-or-self mask of each row's node
    int tree_base = 0, span_L = 0;       // tree: key position of node 0, context length
    int head = 0, grow0 = 0, grow1 = 0;  // KV head and global query rows of the span

    auto begin_span = [&](const Cursor& cc) {
        const int bg = p.b_base + cc.b;
        head = cc.h / p.n_rb;
        const int rbase = (cc.h - head * p.n_rb) * p.n_rows;
        grow0 = row0 < p.n_rows ? rbase + row0 : p.n_rows_all;
        grow1 = row1 < p.n_rows ? rbase + row1 : p.n_rows_all;
        if (grow0 > p.n_rows_all) grow0 = p.n_rows_all;
        if (grow1 > p.n_rows_all) grow1 = p.n_rows_all;
#pragma unroll
        for (int k = 0; k < 2; ++k) {
            const int r = k ? grow1 : grow0;
            const __nv_bfloat16* qr = nullptr;
            if (r < p.n_rows_all) {
                const int i = r / p.G, gi = r % p.G;
                qr = p.q + (((size_t)bg * p.R + i) * p.Hq + (size_t)head * p.G + gi) * kD;
            }
#pragma unroll
            for (int kk = 0; kk < 8; ++kk) {
                const int col = kk * 16 + tq * 2;
                qa[kk][k] = qr ? __ldg(reinterpret_cast<const uint32_t*>(qr + col)) : 0u;
                qa[kk][2 + k] = qr ? __ldg(reinterpret_cast<const uint32_t*>(qr + col + 8)) : 0u;
            }
        }
#pragma unroll
        for (int i = 0; i < 16; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
        m_raw[0] = m_raw[1] = kNegInf;
        l[0] = l[1] = 0.f;
        const int L = s_len[cc.b];
        if (kTree) {
            uint64_t ma, mb;
            tree_ancestor_masks(p.parents + (size_t)bg * p.R, p.R, lane, ma, mb);
            const int i0 = grow0 / p.G, i1 = grow1 / p.G;
            const uint64_t x0 = __shfl_sync(0xffffffffu, ma, i0 & 31), y0 = __shfl_sync(0xffffffffu, mb, i0 & 31);
            const uint64_t x1 = __shfl_sync(0xffffffffu, ma, i1 & 31), y1 = __shfl_sync(0xffffffffu, mb, i1 & 31);
            anc0 = grow0 < p.n_rows_all ? (i0 >= 32 ? y0 : x0) : ~0ull;
            anc1 = grow1 < p.n_rows_all ? (i1 >= 32 ? y1 : x1) : ~0ull;
            tree_base = L - p.R;
            span_L = L;
        } else {
            // exclusive key limit of each of this thread's two rows
            lim0 = grow0 < p.n_rows_all ? L - p.R + 1 + grow0 / p.G : L;
            lim1 = grow1 < p.n_rows_all ? L - p.R + 1 + grow1 / p.G : L;
        }
    };
    begin_span(cur);

    for (int j = 0; j < n_tiles; ++j) {
        const int st = j % kStages;
        const uint32_t use = (uint32_t)(j / kStages);
        if (!mbar_wait_bounded(&full[st], use & 1)) {
            flag_timeout(p.status);
            break;
        }
        const int L = s_len[cur.b];
        const int ts = cur.t * kTileT;
        if (ts + kTileT > L) {
            // keys past L_b (pages not loaded, or slots past the context) may
            // hold any bits: zero their V rows so that P = 0 cannot meet NaN
            const int first = max(0, L - ts);
            uint8_t* vrow = smem + st * kStageBytes + kTensorTileBytes;
            for (int idx = lane; idx < (kTileT - first) * 16; idx += 32) {
                const int r = first + (idx >> 4), ch = idx & 15;
                *reinterpret_cast<uint4*>(vrow + key_row(r, ch >> 3) * 128 + (ch & 7) * 16) =
                    make_uint4(0, 0, 0, 0);
            }
            __syncwarp();
        }
        const uint32_t kb = smem_base + st * kStageBytes;
        const uint32_t vb = kb + kTensorTileBytes;
        // ---- S = Q K^T over this warp's keys: kNT n-tiles of 8 keys
        float sc[kNT][4];
#pragma unroll
        for (int i = 0; i < kNT; ++i) sc[i][0] = sc[i][1] = sc[i][2] = sc[i][3] = 0.f;
        const int key0 = kh * (kTileT / kSplit);
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
#pragma unroll
            for (int np = 0; np < kNT / 2; ++np) {
                const int key = key0 + (2 * np + (lm >> 1)) * 8 + lr;
                const int ch = (kk & 3) * 2 + (lm & 1);
                uint32_t b0, b1, b2, b3;
                ldsm_x4(kb + key_row(key, kk >> 2) * 128 + ((ch ^ (key & 7)) << 4), b0, b1, b2, b3);
                mma_bf16_16816(sc[2 * np], qa[kk], b0, b1);
                mma_bf16_16816(sc[2 * np + 1], qa[kk], b2, b3);
            }
        }
        // ---- causal-verify mask (and the context end)
        if (kTree) {
            // tree: a key in the tree region is visible iff its node is an
            // ancestor (or the node itself); keys past L_b never are
            if (ts + kTileT > tree_base) {
                // visibility of the tile's 64 keys as one word per row: the
                // prefix part, the row's ancestors shifted to the tile, and
                // nothing at or past L_b
                const int d = ts - tree_base;   // tree node of the tile's first key
                const uint64_t pre = d >= 0 ? 0ull : (d <= -64 ? ~0ull : (1ull << -d) - 1ull);
                const uint64_t live = span_L - ts >= 64 ? ~0ull : (1ull << max(span_L - ts, 0)) - 1ull;
                const uint64_t t0 = d >= 64 ? 0ull : (d >= 0 ? anc0 >> d : (d <= -64 ? 0ull : anc0 << -d));
                const uint64_t t1 = d >= 64 ? 0ull : (d >= 0 ? anc1 >> d : (d <= -64 ? 0ull : anc1 << -d));
                const uint64_t v0 = ((pre | t0) & live) >> (key0 + tq * 2), v1 = ((pre | t1) & live) >> (key0 + tq * 2);
#pragma unroll
                for (int nt = 0; nt < kNT; ++nt) {
#pragma unroll
                    for (int e = 0; e < 2; ++e) {
                        if (!((v0 >> (nt * 8 + e)) & 1ull)) sc[nt][e] = kNegInf;
                        if (!((v1 >> (nt * 8 + e)) & 1ull)) sc[nt][2 + e] = kNegInf;
                    }
                }
            }
        } else if (ts + kTileT > min(lim0, lim1)) {
#pragma unroll
            for (int nt = 0; nt < kNT; ++nt) {
#pragma unroll
                for (int e = 0; e < 2; ++e) {
                    const int key = ts + key0 + nt * 8 + tq * 2 + e;
                    if (key >= lim0) sc[nt][e] = kNegInf;
                    if (key >= lim1) sc[nt][2 + e] = kNegInf;
                }
            }
        }
        // ---- online softmax (log2 domain)
#pragma unroll
        for (int rh = 0; rh < 2; ++rh) {
            float mx = kNegInf;
#pragma unroll
            for (int nt = 0; nt < kNT; ++nt) mx = fmaxf(mx, fmaxf(sc[nt][2 * rh], sc[nt][2 * rh + 1]));
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
            const float m_new = fmaxf(m_raw[rh], mx);
            const float m_use = m_new == kNegInf ? 0.f : m_new;
            const float alpha = ex2((m_raw[rh] - m_use) * c);
            m_raw[rh] = m_new;
            const float neg = -m_use * c - kPShift;   // P * 2^-64 (the row sum carries the same factor)
            float rs = 0.f;
#pragma unroll
            for (int nt = 0; nt < kNT; ++nt) {
                const float p0 = ex2(fmaf(sc[nt][2 * rh], c, neg));
                const float p1 = ex2(fmaf(sc[nt][2 * rh + 1], c, neg));
                sc[nt][2 * rh] = p0;
                sc[nt][2 * rh + 1] = p1;
                rs += p0 + p1;
            }
            l[rh] = l[rh] * alpha + rs;
#pragma unroll
            for (int dn = 0; dn < 16; ++dn) {
                o[dn][2 * rh] *= alpha;
                o[dn][2 * rh + 1] *= alpha;
            }
        }
        // ---- O += P V over this warp's keys: k-steps of 16 keys.  P as the sum
        // of two bf16 terms (hi + lo) against V as stored (bf16)
#pragma unroll
        for (int kk = 0; kk < kNT / 2; ++kk) {
            uint32_t ah[4], al[4];
            split_bf16x2(sc[2 * kk][0], sc[2 * kk][1], ah[0], al[0]);
            split_bf16x2(sc[2 * kk][2], sc[2 * kk][3], ah[1], al[1]);
            split_bf16x2(sc[2 * kk + 1][0], sc[2 * kk + 1][1], ah[2], al[2]);
            split_bf16x2(sc[2 * kk + 1][2], sc[2 * kk + 1][3], ah[3], al[3]);
            const int key = key0 + kk * 16 + (lm & 1) * 8 + lr;
#pragma unroll
            for (int dp = 0; dp < 8; ++dp) {
                const int dblk = 2 * dp + (lm >> 1);
                const int ch = dblk & 7;
                uint32_t b0, b1, b2, b3;
                ldsm_x4_trans(vb + key_row(key, dblk >> 3) * 128 + ((ch ^ (key & 7)) << 4), b0, b1, b2, b3);
                mma_bf16_16816(o[2 * dp], ah, b0, b1);
                mma_bf16_16816(o[2 * dp + 1], ah, b2, b3);
                mma_bf16_16816(o[2 * dp], al, b0, b1);
                mma_bf16_16816(o[2 * dp + 1], al, b2, b3);
            }
        }
        const bool piece_end = !(j + 1 < n_tiles && cur.t + 1 < cur.T);
        if (kSplit > 1 && piece_end) {
            // fold the two key shares of every row: once every consumer is
            // done with this stage (fold_a), the second group leaves its
            // (O, m, l) in it (fold_b) and the first group folds them into
            // its own.  Both waits are bounded.
            const uint32_t ph = (uint32_t)(folds++ & 1);
            float* scr = reinterpret_cast<float*>(smem + st * kStageBytes) + rw * (64 * 32 + 4 * 32);
            __syncwarp();
            if (lane == 0) mbar_arrive(fold_a);
            if (kh == 1) {
                if (!mbar_wait_bounded(fold_a, ph)) {
                    flag_timeout(p.status);
                    break;
                }
#pragma unroll
                for (int i = 0; i < 16; ++i)
                    reinterpret_cast<float4*>(scr)[i * 32 + lane] = make_float4(o[i][0], o[i][1], o[i][2], o[i][3]);
                reinterpret_cast<float4*>(scr + 64 * 32)[lane] = make_float4(m_raw[0], m_raw[1], l[0], l[1]);
                __syncwarp();
                if (lane == 0) mbar_arrive(fold_b);
            } else {
                if (!mbar_wait_bounded(fold_b, ph)) {
                    flag_timeout(p.status);
                    break;
                }
                const float4 ml = reinterpret_cast<const float4*>(scr + 64 * 32)[lane];
                const float mo[2] = {ml.x, ml.y}, lo[2] = {ml.z, ml.w};
                float a_s[2], a_o[2];
#pragma unroll
                for (int rh = 0; rh < 2; ++rh) {
                    const float mn = fmaxf(m_raw[rh], mo[rh]);
                    const float mu = mn == kNegInf ? 0.f : mn;
                    a_s[rh] = ex2((m_raw[rh] - mu) * c);
                    a_o[rh] = ex2((mo[rh] - mu) * c);
                    l[rh] = l[rh] * a_s[rh] + lo[rh] * a_o[rh];
                    m_raw[rh] = mn;
                }
#pragma unroll
                for (int i = 0; i < 16; ++i) {
                    const float4 v = reinterpret_cast<const float4*>(scr)[i * 32 + lane];
                    o[i][0] = o[i][0] * a_s[0] + v.x * a_o[0];
                    o[i][1] = o[i][1] * a_s[0] + v.y * a_o[0];
                    o[i][2] = o[i][2] * a_s[1] + v.z * a_o[1];
                    o[i][3] = o[i][3] * a_s[1] + v.w * a_o[1];
                }
            }
        }
        // generic-proxy writes (zeroed rows, the fold's scratch) must be
        // ordered before the next TMA write into this stage
        if (ts + kTileT > L || (kSplit > 1 && piece_end))
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        __syncwarp();
        if (lane == 0) mbar_arrive(&empty[st]);

        if (!piece_end) {
            advance(cur, s_len, nb, p.n_vh);
            continue;
        }

        // ---------------------------------------------- end of a piece of span
        const int bg = p.b_base + cur.b;
        if (kSplit > 1 && kh == 1) {   // folded into the first group's state
            if (j + 1 < n_tiles) {
                advance(cur, s_len, nb, p.n_vh);
                seg_t0 = cur.t;
                first_seg = false;
                begin_span(cur);
            }
            continue;
        }
        const bool complete = seg_t0 == 0 && cur.t + 1 == cur.T;
        float lt[2];
#pragma unroll
        for (int rh = 0; rh < 2; ++rh) {
            lt[rh] = l[rh];
            lt[rh] += __shfl_xor_sync(0xffffffffu, lt[rh], 1);
            lt[rh] += __shfl_xor_sync(0xffffffffu, lt[rh], 2);
        }
        if (complete) {
#pragma unroll
            for (int rh = 0; rh < 2; ++rh) {
                const int grow = rh ? grow1 : grow0;
                if (grow >= p.n_rows_all) continue;
                const float inv = lt[rh] > 0.f ? 1.f / lt[rh] : 0.f;
                const int i = grow / p.G, gi = grow % p.G;
                __nv_bfloat16* dst =
                    p.out + (((size_t)bg * p.R + i) * p.Hq + (size_t)head * p.G + gi) * kD + tq * 2;
#pragma unroll
                for (int dn = 0; dn < 16; ++dn)
                    *reinterpret_cast<uint32_t*>(dst + dn * 8) =
                        pack_bf16x2(o[dn][2 * rh] * inv, o[dn][2 * rh + 1] * inv);
            }
        } else {
            const size_t slot = 2 * (size_t)cta + (first_seg ? 0 : 1);
#pragma unroll
            for (int rh = 0; rh < 2; ++rh) {
                const int row = rh ? row1 : row0;
                if (row >= p.n_rows || (rh ? grow1 : grow0) >= p.n_rows_all) continue;
                // the piece's own normalised output and (m, l): the merge takes
                // a convex combination, which no V value can overflow
                const float inv = lt[rh] > 0.f ? 1.f / lt[rh] : 0.f;
                float* dst = p.part_o + (slot * p.n_rows + row) * kD + tq * 2;
#pragma unroll
                for (int dn = 0; dn < 16; ++dn)
                    *reinterpret_cast<float2*>(dst + dn * 8) = make_float2(o[dn][2 * rh] * inv, o[dn][2 * rh + 1] * inv);
                if (tq == 0)
                    p.part_ml[slot * p.n_rows + row] =
                        make_float2(m_raw[rh] == kNegInf ? kNegInf : m_raw[rh] * c, lt[rh]);
            }
            if (threadIdx.x == 0) p.part_span[slot] = cur.b * p.n_vh + cur.h;
        }
        if (j + 1 < n_tiles) {
            advance(cur, s_len, nb, p.n_vh);
            seg_t0 = cur.t;
            first_seg = false;
            begin_span(cur);
        }
    }
}

// ---------------------------------------------------------------------------
// Merge of split spans.  Each piece of a cut span left its own normalised
// output o_q and (m_q, l_q); the span's output is sum_q w_q o_q with
// w_q = l_q 2^(m_q - M) / sum_r l_r 2^(m_r - M), a convex combination (no
// value can overflow).  One warp per query row (lanes across the pieces for
// the weights, across the 128 dims for the sum).
// Two ways to find a span's pieces, the launch taking the one with the
// smaller grid:
//  * per span: every CTA recomputes the main kernel's work split from the
//    context lengths (cheap for few requests, and done while the main
//    kernel runs) and finds the CTAs that cut its span; a span with a single
//    piece was written whole and is skipped;
//  * per main-kernel CTA: the main kernels record the span of each partial
//    slot (-1 when unused):
// slot 2c holds CTA c's first piece, 2c + 1 its last one when that is a
// different piece.  In slot order a cut span's pieces are consecutive,
// unused slots aside, and at most one cut span starts in each CTA: its last
// piece, or -- one piece only -- that piece, unless the previous CTA's last
// piece belongs to the same span.  Merge CTA (c, y) reads the slot list
// around CTA c once into shared memory, gathers the pieces of the span that
// starts in CTA c (if any) and merges rows 8y .. 8y + 7 of it.  Six merge
// CTAs fit an SM, so the whole grid is resident at once in the usual case.
// ---------------------------------------------------------------------------
constexpr int kMergeThreads = 256;
constexpr int kMergeRows = kMergeThreads / 32;   // query rows per merge CTA
constexpr int kMergePerSm = 6;                   // merge CTAs resident per SM (registers capped to fit)
constexpr int kMergePieces = 8;                  // pieces of a row merged in one round trip (per-span form)
constexpr int kMergePiecesCut = 4;               // the same for the register-capped per-CTA form
constexpr int kMergeWin = 64;                    // slots read ahead of CTA c's first slot

// the convex combination of one row's pieces (slots[0..n_p)), by one warp.
// Up to kPieces pieces (the usual case) take one round trip: every
// piece's (m, l) and this lane's four output columns of every piece are
// requested together; more pieces go through the general loop.
template <int kPieces>
__device__ __forceinline__ void merge_row(const AttnParams& p, const int* slots, int n_p, int bl, int h, int row,
                                          int lane) {
    const int bg = p.b_base + bl;
    const int head = h / p.n_rb, rbase = (h - head * p.n_rb) * p.n_rows;
    if (row >= p.n_rows || rbase + row >= p.n_rows_all) return;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    if (n_p <= kPieces) {
        float4 v[kPieces];
        float2 ml = make_float2(kNegInf, 0.f);   // lane q < n_p: piece q
        if (lane < n_p) ml = __ldcg(&p.part_ml[(size_t)slots[lane] * p.n_rows + row]);
#pragma unroll
        for (int j = 0; j < kPieces; ++j) {
            v[j] = make_float4(0.f, 0.f, 0.f, 0.f);
            if (j < n_p)
                v[j] = __ldcg(reinterpret_cast<const float4*>(p.part_o + ((size_t)slots[j] * p.n_rows + row) * kD +
                                                              lane * 4));
        }
        float M = ml.x;
#pragma unroll
        for (int off = 4; off > 0; off >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, off));
        M = __shfl_sync(0xffffffffu, M, 0);
        float wq = (M == kNegInf || ml.x == kNegInf) ? 0.f : ml.y * ex2(ml.x - M);
        float lsum = wq;
#pragma unroll
        for (int off = 4; off > 0; off >>= 1) lsum += __shfl_xor_sync(0xffffffffu, lsum, off);
        lsum = __shfl_sync(0xffffffffu, lsum, 0);
        const float inv = lsum > 0.f ? 1.f / lsum : 0.f;
        wq *= inv;
#pragma unroll
        for (int j = 0; j < kPieces; ++j) {
            const float wgt = __shfl_sync(0xffffffffu, wq, j);
            if (j < n_p) {
                acc.x = fmaf(wgt, v[j].x, acc.x);
                acc.y = fmaf(wgt, v[j].y, acc.y);
                acc.z = fmaf(wgt, v[j].z, acc.z);
                acc.w = fmaf(wgt, v[j].w, acc.w);
            }
        }
    } else {
        float M = kNegInf;
        for (int q = lane; q < n_p; q += 32) M = fmaxf(M, __ldcg(&p.part_ml[(size_t)slots[q] * p.n_rows + row]).x);
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, off));
        float lsum = 0.f;
        if (M != kNegInf)
            for (int q = lane; q < n_p; q += 32) {
                const float2 ml = __ldcg(&p.part_ml[(size_t)slots[q] * p.n_rows + row]);
                if (ml.x != kNegInf) lsum = fmaf(ml.y, ex2(ml.x - M), lsum);
            }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) lsum += __shfl_xor_sync(0xffffffffu, lsum, off);
        const float inv = lsum > 0.f ? 1.f / lsum : 0.f;
        for (int q0 = 0; q0 < n_p && inv > 0.f; q0 += 32) {
            float wq = 0.f;   // the weight of piece q0 + lane
            if (q0 + lane < n_p) {
                const float2 ml = __ldcg(&p.part_ml[(size_t)slots[q0 + lane] * p.n_rows + row]);
                wq = ml.x == kNegInf ? 0.f : ml.y * ex2(ml.x - M) * inv;
            }
            const int nq = min(32, n_p - q0);
            for (int qq = 0; qq < nq; qq += kPieces) {
                float4 v[kPieces];
                float wgt[kPieces];
#pragma unroll
                for (int j = 0; j < kPieces; ++j) {
                    const bool ok = qq + j < nq;
                    wgt[j] = __shfl_sync(0xffffffffu, wq, (qq + j) & 31);
                    const size_t sl = (size_t)slots[q0 + (ok ? qq + j : 0)];
                    v[j] = ok ? __ldcg(reinterpret_cast<const float4*>(p.part_o + (sl * p.n_rows + row) * kD + lane * 4))
                              : make_float4(0.f, 0.f, 0.f, 0.f);
                    if (!ok) wgt[j] = 0.f;
                }
#pragma unroll
                for (int j = 0; j < kPieces; ++j) {
                    acc.x = fmaf(wgt[j], v[j].x, acc.x);
                    acc.y = fmaf(wgt[j], v[j].y, acc.y);
                    acc.z = fmaf(wgt[j], v[j].z, acc.z);
                    acc.w = fmaf(wgt[j], v[j].w, acc.w);
                }
            }
        }
    }
    const int i = (rbase + row) / p.G, gi = (rbase + row) % p.G;
    __nv_bfloat16* dst = p.out + (((size_t)bg * p.R + i) * p.Hq + (size_t)head * p.G + gi) * kD + lane * 4;
    uint2 pk;
    pk.x = pack_bf16x2(acc.x, acc.y);
    pk.y = pack_bf16x2(acc.z, acc.w);
    *reinterpret_cast<uint2*>(dst) = pk;
}

// grid (span h, request bl, 8-row chunk)
__global__ void __launch_bounds__(kMergeThreads)
verify_attention_merge_span_kernel(const AttnParams p, int grid_main) {
    __shared__ long long s_red[2][kMergeThreads / 32];
    __shared__ int s_slots[2 * kMaxGrid];
    __shared__ int s_np;
    const int h = blockIdx.x, bl = blockIdx.y;
    const int nb = p.n_batch;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int l_cap = p.max_pages * p.ps;

    // tiles before request bl, and in total (x spans)
    long long before = 0, total = 0;
    for (int b = threadIdx.x; b < nb; b += kMergeThreads) {
        int L = __ldg(p.ctx_lens + p.b_base + b);
        L = max(0, min(L, l_cap));
        const long long v = (long long)tiles_of(L) * p.n_vh;
        total += v;
        if (b < bl) before += v;
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
        before += __shfl_xor_sync(0xffffffffu, before, off);
        total += __shfl_xor_sync(0xffffffffu, total, off);
    }
    if (lane == 0) {
        s_red[0][warp] = before;
        s_red[1][warp] = total;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        long long bf = 0, W = 0;
        for (int w = 0; w < kMergeThreads / 32; ++w) {
            bf += s_red[0][w];
            W += s_red[1][w];
        }
        int L = __ldg(p.ctx_lens + p.b_base + bl);
        L = max(0, min(L, l_cap));
        const int T = tiles_of(L);
        const long long g_need = (W + kMinTilesPerCta - 1) / kMinTilesPerCta;
        const int Gc = (int)(g_need < (long long)grid_main ? (g_need > 0 ? g_need : 1) : grid_main);
        // in work units (tiles_before): the span's start units begin at vs,
        // its tiles at vs + X; the CTA whose unit range holds its first tile
        // holds it as its first piece unless that range starts before vs
        // (unit vs - 1 is the previous span's last tile); every later owner
        // holds it as its first piece
        const int X = p.span_x;
        const long long U = W + (long long)X * p.n_vh * nb;
        const long long vs = bf + (long long)X * p.n_vh * bl + (long long)h * (T + X);
        const int c_first = owner_of(vs + X, U, Gc);
        const int c_last = owner_of(vs + X + T - 1, U, Gc);
        int n_p = 0;
        for (int cc = c_first; cc <= c_last && n_p < 2 * kMaxGrid; ++cc)
            s_slots[n_p++] = 2 * cc + ((cc == c_first && (long long)cc * U / Gc < vs) ? 1 : 0);
        s_np = n_p;
    }
    __syncthreads();
    const int n_p = s_np;
    // everything above depends only on the context lengths; the pieces are
    // the main kernel's output.  Every CTA waits, even one with nothing to
    // merge, so that this grid never completes before the main kernel (a
    // programmatic dependent of this kernel may rely on that), then lets the
    // next kernel of the stream start.
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    if (n_p <= 1) return;   // written whole by the main kernel
    merge_row<kMergePieces>(p, s_slots, n_p, bl, h, blockIdx.z * kMergeRows + warp, lane);
}

// grid (main-kernel CTA c, 8-row chunk)
__global__ void __launch_bounds__(kMergeThreads, kMergePerSm)
verify_attention_merge_cut_kernel(const AttnParams p, int n_slots) {
    __shared__ int s_win[2 + kMergeWin];   // slots 2c-2 .. 2c+kMergeWin-1
    __shared__ int s_slots[2 * kMaxGrid];
    __shared__ int s_np, s_span;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // the slot list is the main kernel's output.  Every CTA waits, even one
    // with nothing to merge, so that this grid never completes before the
    // main kernel (a programmatic dependent of this kernel may rely on that),
    // then lets the next kernel of the stream start.
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    const int c = blockIdx.x, w0 = 2 * c - 2;
    if (threadIdx.x < 2 + kMergeWin) {
        const int r = w0 + (int)threadIdx.x;
        s_win[threadIdx.x] = r >= 0 && r < n_slots ? __ldcg(&p.part_span[r]) : -1;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        auto span_at = [&](int r) {
            return r < 0 || r >= n_slots ? -1 : (r - w0 < 2 + kMergeWin ? s_win[r - w0] : __ldcg(&p.part_span[r]));
        };
        const int first = span_at(2 * c), last = span_at(2 * c + 1);
        // the cut span that starts in CTA c, and its first slot
        int id = -1, r0 = -1;
        if (last >= 0) {
            id = last;
            r0 = 2 * c + 1;
        } else if (first >= 0) {
            const int prev = c > 0 ? (span_at(2 * c - 1) >= 0 ? span_at(2 * c - 1) : span_at(2 * c - 2)) : -1;
            if (prev != first) {
                id = first;
                r0 = 2 * c;
            }
        }
        int n_p = 0;
        if (id >= 0) {
            s_slots[n_p++] = r0;
            // the following CTAs' first pieces, while the span goes on
            for (int cc = c + 1; 2 * cc < n_slots && n_p < 2 * kMaxGrid; ++cc) {
                if (span_at(2 * cc) != id) break;
                s_slots[n_p++] = 2 * cc;
                if (span_at(2 * cc + 1) >= 0) break;   // CTA cc has a later piece: the span ends here
            }
        }
        s_np = n_p;
        s_span = id;
    }
    __syncthreads();
    const int n_p = s_np, id = s_span;
    if (n_p <= 1) return;   // no cut span starts here (a single piece cannot occur)
    merge_row<kMergePiecesCut>(p, s_slots, n_p, id / p.n_vh, id % p.n_vh, blockIdx.y * kMergeRows + warp, lane);
}

#include "verify_attention_tc.cuh"

PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    if (!fn) {
        void* ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
    }
    return fn;
}

// halves: dim halves per box (2: [half][keys][64 dims] per page piece; 1: one
// half per box, for tiles laid out [half][64 keys][64 dims])
cs_status encode_pool_map(CUtensorMap* map, const void* pool, const cs_attn_dims& d, int box_t, int halves = 2) {
    auto enc = tensor_map_encoder();
    if (!enc) return fail(CS_ERR_CUDA, "cuTensorMapEncodeTiled is not available from the driver");
    // (64 dims, keys, 2 dim halves, heads, pages): one box holds both halves
    // of box_t keys, half-major, so it lands as [half][key][64 dims]
    const cuuint64_t dims[5] = {64, (cuuint64_t)d.page_size, 2, (cuuint64_t)d.n_kv_heads,
                                (cuuint64_t)d.num_pages};
    const cuuint64_t row = (cuuint64_t)d.head_dim * 2;
    const cuuint64_t strides[4] = {row, 128, row * d.page_size, row * d.page_size * d.n_kv_heads};
    const cuuint32_t box[5] = {64, (cuuint32_t)box_t, (cuuint32_t)halves, 1, 1};
    const cuuint32_t estr[5] = {1, 1, 1, 1, 1};
    const CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, const_cast<void*>(pool), dims,
                           strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                           CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                           CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(CS_ERR_CUDA, "cuTensorMapEncodeTiled failed (CUresult %d)", (int)r);
    return CS_OK;
}

// The query rows of one KV head of one request (or of one row block of
// them) as one box per dim half: q [B, R, Hq, D] seen as (D, Hq, R, B), box
// (64, G, box_rows, 1), landing as [draft row][group head][64 dims] = query
// row i*G + g of the block.  A block that runs past row R reads zeros there.
cs_status encode_q_map(CUtensorMap* map, const void* q, const cs_attn_dims& d, int rows, int box_rows) {
    auto enc = tensor_map_encoder();
    if (!enc) return fail(CS_ERR_CUDA, "cuTensorMapEncodeTiled is not available from the driver");
    const int G = d.n_q_heads / d.n_kv_heads;
    const cuuint64_t dims[4] = {(cuuint64_t)d.head_dim, (cuuint64_t)d.n_q_heads, (cuuint64_t)rows, (cuuint64_t)d.batch};
    const cuuint64_t row = (cuuint64_t)d.head_dim * 2;
    const cuuint64_t strides[3] = {row, row * d.n_q_heads, row * d.n_q_heads * rows};
    const cuuint32_t box[4] = {64, (cuuint32_t)G, (cuuint32_t)box_rows, 1};
    const cuuint32_t estr[4] = {1, 1, 1, 1};
    const CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(q), dims, strides, box, estr,
                           CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                           CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(CS_ERR_CUDA, "cuTensorMapEncodeTiled (q) failed (CUresult %d)", (int)r);
    return CS_OK;
}

// CTAs per SM of the tcgen05 kernel (1 when its shared memory fits; cached).
int tc_resident_per_sm() {
    static int cache[64] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
        cudaGetLastError();
        return 0;
    }
    if (!cache[dev]) {
        int n = 0;
        if (cudaFuncSetAttribute(verify_attention_tc_kernel<false, 16>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 tc_smem_bytes(kTcRows)) != cudaSuccess ||
            cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, verify_attention_tc_kernel<false, 16>, kTcThreads,
                                                          tc_smem_bytes(kTcRows)) != cudaSuccess)
            n = 0;
        cudaGetLastError();
        cache[dev] = n + 1;
    }
    return cache[dev] - 1;
}

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// A launch that may start while the kernel before it in the stream runs
// (the kernel waits with griddepcontrol.wait before it reads its inputs).
template <typename... Args, typename... Params>
cudaError_t launch_dependent(void (*kern)(Params...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                             Args... args) {
    cudaLaunchAttribute attr;
    attr.id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr.val.programmaticStreamSerializationAllowed = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cfg.attrs = &attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, args...);
}

// The split merge as a programmatic dependent of the main kernel: it may
// start early and waits (griddepcontrol.wait) before it reads the partials.
// The form with the smaller grid: per span (spans x 8-row chunks; few
// requests) or per main-kernel CTA (main grid x 8-row chunks).
cudaError_t launch_merge(const AttnParams& p, const AttnPlan& pl, cudaStream_t stream) {
    cudaLaunchAttribute attr;
    attr.id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr.val.programmaticStreamSerializationAllowed = 1;
    cudaLaunchConfig_t cfg = {};
    const unsigned chunks = (unsigned)((pl.n_rows + kMergeRows - 1) / kMergeRows);
    cfg.blockDim = dim3(kMergeThreads, 1, 1);
    cfg.stream = stream;
    cfg.attrs = &attr;
    cfg.numAttrs = 1;
    if ((long long)p.n_vh * p.n_batch <= (long long)pl.grid) {
        cfg.gridDim = dim3(p.n_vh, p.n_batch, chunks);
        return cudaLaunchKernelEx(&cfg, verify_attention_merge_span_kernel, p, (int)pl.grid);
    }
    cfg.gridDim = dim3((unsigned)pl.grid, chunks, 1);
    return cudaLaunchKernelEx(&cfg, verify_attention_merge_cut_kernel, p, 2 * (int)pl.grid);
}

// Resident CTAs per SM of the kernel at a given block size (cached per device).
template <bool kTree, int kSplit>
int resident_per_sm(int threads) {
    // every box size instantiates the same code shape; the 16-key one stands for all
    static int cache[64][kMaxRowWarps + 2] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
        cudaGetLastError();
        return 1;
    }
    const int key = threads / 32;
    if (key <= 0 || key > kMaxRowWarps + 1) return 1;
    if (!cache[dev][key]) {
        int n = 0;
        if (cudaFuncSetAttribute(verify_attention_kernel<kTree, 16, kSplit>,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes) != cudaSuccess ||
            cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, verify_attention_kernel<kTree, 16, kSplit>, threads,
                                                          kSmemBytes) != cudaSuccess ||
            n <= 0) {
            cudaGetLastError();
            n = 1;
        }
        cache[dev][key] = n;
    }
    return cache[dev][key];
}

}  // namespace

// Workspace layout of a plan: the status word (256 B), then the split
// partials (m, l) [2 grid, rows], O [2 grid, rows, D] and the span of each
// partial slot [2 grid].
void attn_layout(AttnPlan& pl) {
    size_t off = 256;
    pl.off_part_ml = off;
    off = align_up(off + sizeof(float) * 2 * (size_t)2 * pl.grid * pl.n_rows, 256);
    pl.off_part_o = off;
    off = align_up(off + sizeof(float) * kD * (size_t)2 * pl.grid * pl.n_rows, 256);
    pl.off_part_span = off;
    off = align_up(off + sizeof(int) * (size_t)2 * pl.grid, 256);
    pl.bytes = off;
}

// allow_tc: whether the tcgen05 form may be chosen (the mma.sync form's own
// plan otherwise)
AttnPlan plan_attention(const cs_attn_dims& d, int rows, bool tree, int sm_count, bool allow_tc = true) {
    AttnPlan pl{};
    pl.group = d.n_q_heads / d.n_kv_heads;
    pl.rows = rows;
    pl.tree = tree;
    pl.n_rows_all = pl.rows * pl.group;
    // query rows of one span: all of them, or equal row blocks of a multiple
    // of 16 rows when they do not fit one CTA
    const int cap = kMaxRowWarps * 16;
    pl.n_rb = (pl.n_rows_all + cap - 1) / cap;
    pl.n_rows = pl.n_rb == 1 ? pl.n_rows_all : ((pl.n_rows_all + pl.n_rb - 1) / pl.n_rb + 15) / 16 * 16;
    pl.row_warps = (pl.n_rows + 15) / 16;
    // few rows: two consumer groups share each tile's keys
    pl.split = pl.row_warps <= kMaxSplitRowWarps ? 2 : 1;
    // more than 32 rows on pages of 16+ tokens: the tcgen05 kernel (up to 32
    // rows the key-split mma.sync form streams faster), in one block of up
    // to 128 rows or -- trees -- in row blocks of whole nodes of at most 128
    // rows each, every block its own span (its keys are then read once per
    // block)
    int tc_rb = 1, tc_rows = pl.n_rows_all;
    while (tree && tc_rows > kTcRows && tc_rb < rows) {
        ++tc_rb;
        tc_rows = ((rows + tc_rb - 1) / tc_rb) * pl.group;
    }
    pl.tc = allow_tc && tc_rows > kTcMinRows && tc_rows <= kTcRows && d.page_size >= 16 && rows <= 256 &&
            pl.group <= 256 &&
            tc_resident_per_sm() >= 1;
    if (pl.tc) {
        pl.n_rb = tc_rb;
        pl.n_rows = tc_rows;
        pl.row_warps = (pl.n_rows + 15) / 16;
        pl.split = 1;
        pl.grid = (sm_count > 0 ? sm_count : 148) * tc_resident_per_sm();
        if (pl.grid > kMaxGrid) pl.grid = kMaxGrid;
    } else {
        // persistent grid: exactly the CTAs that are resident at once
        const int threads = (pl.split * pl.row_warps + 1) * 32;
        const int res = pl.split == 2 ? (tree ? resident_per_sm<true, 2>(threads) : resident_per_sm<false, 2>(threads))
                                      : (tree ? resident_per_sm<true, 1>(threads) : resident_per_sm<false, 1>(threads));
        pl.grid = (sm_count > 0 ? sm_count : 148) * res;
        if (pl.grid > kMaxGrid) pl.grid = kMaxGrid;
    }
    attn_layout(pl);
    if (pl.tc) {
        // a query buffer TMA cannot read falls back to the mma.sync form on
        // the same workspace (its grid capped at this one): room for both
        AttnPlan alt = plan_attention(d, rows, tree, sm_count, false);
        if (alt.grid > pl.grid) alt.grid = pl.grid;
        attn_layout(alt);
        if (alt.bytes > pl.bytes) pl.bytes = alt.bytes;
    }
    return pl;
}

AttnPlan plan_verify_attention(const cs_attn_dims& d, int n_draft, int sm_count) {
    return plan_attention(d, n_draft + 1, false, sm_count);
}

AttnPlan plan_tree_attention(const cs_attn_dims& d, int n_nodes, int sm_count) {
    return plan_attention(d, n_nodes, true, sm_count);
}

cs_status launch_verify_attention(const cs_attn_dims& d, const AttnPlan& pl, const void* q,
                                  const void* k_pages, const void* v_pages,
                                  const int32_t* page_table, const int32_t* ctx_lens,
                                  const int32_t* parents, void* out, void* workspace,
                                  cudaStream_t stream) {
    if (pl.tree != (parents != nullptr))
        return fail(CS_ERR_INVALID_ARG, "tree plan and parent array do not match");
    const int box_t = d.page_size < kTileT ? d.page_size : kTileT;
    CUtensorMap tk, tv;
    cs_status st = encode_pool_map(&tk, k_pages, d, box_t);
    if (st != CS_OK) return st;
    st = encode_pool_map(&tv, v_pages, d, box_t);
    if (st != CS_OK) return st;

    uint8_t* ws = static_cast<uint8_t*>(workspace);
    AttnParams p{};
    p.q = static_cast<const __nv_bfloat16*>(q);
    p.out = static_cast<__nv_bfloat16*>(out);
    p.page_table = page_table;
    p.ctx_lens = ctx_lens;
    p.parents = parents;
    p.status = reinterpret_cast<int*>(ws);
    p.part_ml = reinterpret_cast<float2*>(ws + pl.off_part_ml);
    p.part_o = reinterpret_cast<float*>(ws + pl.off_part_o);
    p.part_span = reinterpret_cast<int*>(ws + pl.off_part_span);
    p.Hq = d.n_q_heads;
    p.Hkv = d.n_kv_heads;
    p.G = pl.group;
    p.R = pl.rows;
    p.n_rows = pl.n_rows;
    p.ps = d.page_size;
    p.box_t = box_t;
    p.max_pages = d.max_pages_per_seq;
    p.row_warps = pl.row_warps;
    p.n_rb = pl.n_rb;
    p.n_vh = d.n_kv_heads * pl.n_rb;
    p.n_rows_all = pl.n_rows_all;
    // a span piece's own cost in tile units (clock stamps: ~1 tile's time at
    // 35 rows, ~2.7 at 72 in the tcgen05 form)
    p.span_x = pl.tc ? (pl.n_rows + 12) / 24 : 1;
    if (p.span_x < 1) p.span_x = 1;
    const float scale = d.sm_scale > 0.f ? d.sm_scale : 1.0f / sqrtf((float)d.head_dim);
    p.scale_log2 = scale * 1.4426950408889634f;

    if (pl.tc && (reinterpret_cast<uintptr_t>(q) & 15) != 0) {
        // the query rows come in by TMA, which needs a 16-byte aligned base:
        // run the mma.sync form on the same workspace (its grid capped at
        // the plan's, so the partial slots fit)
        AttnPlan alt = plan_attention(d, pl.rows, pl.tree, 0, false);
        if (alt.grid > pl.grid) alt.grid = pl.grid;
        attn_layout(alt);   // fits: the tcgen05 plan's size covers this layout
        return launch_verify_attention(d, alt, q, k_pages, v_pages, page_table, ctx_lens, parents, out, workspace,
                                       stream);
    }
    if (pl.tc) {
        CUtensorMap tq;
        st = encode_q_map(&tq, q, d, pl.rows, pl.n_rows / pl.group);
        if (st != CS_OK) return st;
        // one box per page piece with both dim halves, as for the other form

        using TcKern = void (*)(const CUtensorMap, const CUtensorMap, const CUtensorMap, const AttnParams);
        static const TcKern tc_kerns[2][3] = {
            {verify_attention_tc_kernel<false, 16>, verify_attention_tc_kernel<false, 32>,
             verify_attention_tc_kernel<false, 64>},
            {verify_attention_tc_kernel<true, 16>, verify_attention_tc_kernel<true, 32>,
             verify_attention_tc_kernel<true, 64>}};
        const int ti = box_t == 16 ? 0 : box_t == 32 ? 1 : 2;
        const TcKern tk_fn = tc_kerns[pl.tree][ti];
        p.tc_stages = tc_k_stages(pl.n_rows);
        p.tc_vstages = tc_v_stages(pl.n_rows);
        p.tc_q_half = tc_q_half_bytes(pl.n_rows);
        const int smem_bytes = tc_smem_bytes(pl.n_rows);
        cudaError_t e = cudaFuncSetAttribute(tk_fn, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes);
        if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute(verify_attention_tc_kernel)");
        for (int b0 = 0; b0 < d.batch; b0 += kMaxBatchPerLaunch) {
            p.b_base = b0;
            p.n_batch = d.batch - b0 < kMaxBatchPerLaunch ? d.batch - b0 : kMaxBatchPerLaunch;
            e = launch_dependent(tk_fn, dim3(pl.grid), dim3(kTcThreads), (size_t)smem_bytes, stream, tk, tv, tq, p);
            if (e != cudaSuccess) return cuda_fail(e, "verify_attention_tc_kernel launch");
            e = launch_merge(p, pl, stream);
            if (e != cudaSuccess) return cuda_fail(e, "verify_attention_merge_kernel launch");
        }
        return CS_OK;
    }
    // kernels by (key split, tree, box size 8/16/32/64 keys)
    using Kern = void (*)(const CUtensorMap, const CUtensorMap, const AttnParams);
    static const Kern kerns[2][2][4] = {
        {{verify_attention_kernel<false, 8, 1>, verify_attention_kernel<false, 16, 1>,
          verify_attention_kernel<false, 32, 1>, verify_attention_kernel<false, 64, 1>},
         {verify_attention_kernel<true, 8, 1>, verify_attention_kernel<true, 16, 1>,
          verify_attention_kernel<true, 32, 1>, verify_attention_kernel<true, 64, 1>}},
        {{verify_attention_kernel<false, 8, 2>, verify_attention_kernel<false, 16, 2>,
          verify_attention_kernel<false, 32, 2>, verify_attention_kernel<false, 64, 2>},
         {verify_attention_kernel<true, 8, 2>, verify_attention_kernel<true, 16, 2>,
          verify_attention_kernel<true, 32, 2>, verify_attention_kernel<true, 64, 2>}}};
    const int bi = box_t == 8 ? 0 : box_t == 16 ? 1 : box_t == 32 ? 2 : 3;
    const int si = pl.split == 2 ? 1 : 0;
    const Kern kern = kerns[si][pl.tree][bi];
    cudaError_t e = cudaSuccess;
    {
        static bool attr_done[2][2][4][64] = {};
        int dev = 0;
        e = cudaGetDevice(&dev);
        if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
        if (dev < 0 || dev >= 64 || !attr_done[si][pl.tree][bi][dev]) {
            e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
            if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute(verify_attention_kernel)");
            if (dev >= 0 && dev < 64) attr_done[si][pl.tree][bi][dev] = true;
        }
    }
    const dim3 block((pl.split * pl.row_warps + 1) * 32);
    for (int b0 = 0; b0 < d.batch; b0 += kMaxBatchPerLaunch) {
        p.b_base = b0;
        p.n_batch = d.batch - b0 < kMaxBatchPerLaunch ? d.batch - b0 : kMaxBatchPerLaunch;
        e = launch_dependent(kern, dim3(pl.grid), block, (size_t)kSmemBytes, stream, tk, tv, p);
        if (e != cudaSuccess) return cuda_fail(e, "verify_attention_kernel launch");
        e = launch_merge(p, pl, stream);
        if (e != cudaSuccess) return cuda_fail(e, "verify_attention_merge_kernel launch");
    }
    return CS_OK;
}

}  // namespace cs
