// spec_accept.cu -- the acceptance step of speculative sampling (the rule
// the paper's drafter follows, Sec. 3.4): temperature softmax statistics of
// target and draft rows, the min(1, p/q) accept test, the residual
// max(0, p - q) or bonus draw by inverse CDF, and the greedy variant.
//
// Two kernels per call, no atomics, no spin-waits and no scratch that has to
// start at a known value:
//   1. accept_stats_kernel streams every row of every request (target rows
//      0..k, then draft rows 0..k-1; target rows only when greedy) once.  The
//      rows are cut into 4 KB items and the flattened item sequence is split
//      into one contiguous, equal range per warp of a grid that fills the
//      device, so every SM reads the same number of bytes.  A warp keeps the
//      next item in flight while it reduces the current one and writes one
//      partial per row segment of its range: (max, sum 2^((z-max)c)) -- one
//      exponential per logit -- or, greedy, (max, lowest id of the max).
//      The partials of a row sit side by side in the order of the row, and
//      the warp that holds a row's last item records how many there are.
//   2. accept_draw_kernel runs one thread-block cluster per request and is
//      launched as a programmatic dependent of kernel 1: it loads its inputs
//      while kernel 1 finishes.  Every CTA folds the partials of the
//      request's rows in the same fixed order (so all of them hold
//      bit-identical statistics), runs the accept tests
//      (one lane per position, the first rejection found by a ballot) and
//      computes the draw mass of its slice of the vocabulary for the deciding
//      row pair.  The CTAs swap their masses through distributed shared
//      memory, fold them in rank order, and the CTA whose cell holds u_k * Z
//      finds the token within its slice.
//   Greedy mode replaces kernel 2 by accept_greedy_kernel (one warp per
//   request: argmax agreement).
// Token trees (multi-candidate verification) reuse kernel 1 over the target
// rows of every node and the draft rows of the nodes that have children
// (a leaf's draft row is not read), and walk the tree in tree_draw_kernel
// (one cluster per request): the children of the current node are tested in
// turn, each rejection turning the running distribution into the residual
// max(p - kappa q, 0) / Z, whose mass Z takes one cluster-wide pass over the
// row pair; the walk ends with the draw of section 2 at that kappa.  The
// greedy walk is tree_greedy_kernel.
// No probability is written to memory; the scratch holds the row-segment
// pairs and one count per row.
#include <limits.h>
#include <math.h>

#include "cs_device.cuh"
#include "cs_internal.h"

namespace cs {
namespace {

constexpr int kThreads = 256;                  // kernel 1 and the greedy kernel
constexpr int kWarps = kThreads / 32;
constexpr int kDrawThreads = 512;              // kernel 2
constexpr int kDrawWarps = kDrawThreads / 32;
constexpr int kVecs = 8;                       // kernel 1: 16-byte vectors per lane per item
constexpr int kItemBytes = 32 * kVecs * 16;    // 4 KB of one row
constexpr int kRunVecs = 2;                    // kernel 2: 16-byte vectors per thread per row per pass
constexpr int kMaxRows = 33;                   // 2k+1 rows of a request, k <= 16
constexpr int kRowsPerDrawWarp = (kMaxRows + kDrawWarps - 1) / kDrawWarps;
constexpr int kMaxPasses = 128;                // passes of one CTA over its vocabulary slice
constexpr int kMaxCluster = 16;
constexpr int kMaxTreeNodes = 64;

struct AcceptParams {
    const void* target;       // [B, n_t, V]: chain n_t = k+1, tree n_t = nodes
    const void* draft;        // [B, d_rows, V]: chain d_rows = k, tree d_rows = nodes
    const int32_t* tokens;    // chain [B, k]; tree [B, n_t] (node tokens)
    const float* uniforms;    // chain [B, k+1]; tree [B, n_t]
    int32_t* out_tokens;      // chain [B, k+1]; tree [B, n_t]
    int32_t* out_n;           // [B], or null (the sampler)
    const int32_t* parents;   // tree [B, n_t] (null for the chain)
    int32_t* out_path;        // tree [B, n_t]: accepted nodes in walk order
    int B, V, k;
    int n_t, d_rows;          // target rows and draft rows per request
    int R;                    // rows per request streamed by kernel 1: n_t + d_rows, or n_t (greedy)
    int I;                    // 4 KB items per row
    long long N;              // B * R * I items in all
    int W;                    // busy warps of kernel 1 (warp w owns items [w*N/W, (w+1)*N/W)), W <= N
    int J;                    // partial slots per row (row segments a row can have)
    int slice;                // kernel 2: logits of the vocabulary per CTA of a cluster
    int b_base;               // kernel 2: first request of this launch
    float c_hi, c_lo;         // log2(e) / T as a float pair
    float2* part;             // [B*R, J] row-segment partials, in row order
    int* cnt;                 // [B*R] segments of each row
};

// ------------------------------------------------------------ small helpers
__device__ __forceinline__ uint4 ld_stream(const void* p) {
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}

__device__ __forceinline__ float to_f(float v) { return v; }
__device__ __forceinline__ float to_f(__nv_bfloat16 v) { return __bfloat162float(v); }

template <typename T>
__device__ __forceinline__ bool aligned16(const T* p) {
    return (reinterpret_cast<uintptr_t>(p) & 15u) == 0;
}

template <typename T>
union Vec16 {
    uint4 q;
    T t[16 / sizeof(T)];
};

// 16 bytes of row[start ..]; entries at or past `end` read as -inf.  `stream`
// bypasses L1 (kernel 1 touches every byte once).
template <typename T, bool kStream>
__device__ __forceinline__ uint4 load16(const T* row, int start, int end, bool vec) {
    constexpr int kPer = 16 / (int)sizeof(T);
    if (vec && start + kPer <= end)
        return kStream ? ld_stream(row + start) : __ldg(reinterpret_cast<const uint4*>(row + start));
    Vec16<T> v;
#pragma unroll
    for (int e = 0; e < kPer; ++e) v.t[e] = start + e < end ? row[start + e] : (T)kNegInf;
    return v.q;
}

// A pair (m, s) stands for sum_v 2^((z_v - m) c); empty is (-inf, 0).
__device__ __forceinline__ void fold(float& m, float& s, float m2, float s2, float c_hi, float c_lo) {
    const float M = fmaxf(m, m2);
    if (M == kNegInf) return;
    const float a = m == kNegInf ? 0.f : s * ex2_scaled(m - M, c_hi, c_lo);
    const float b = m2 == kNegInf ? 0.f : s2 * ex2_scaled(m2 - M, c_hi, c_lo);
    s = a + b;
    m = M;
}

// (max, id) with the lowest id on ties; the id travels as int bits.
__device__ __forceinline__ void argmax_fold(float2& acc, float2 o) {
    if (o.x > acc.x || (o.x == acc.x && __float_as_int(o.y) < __float_as_int(acc.y))) acc = o;
}

// Unnormalised weight of one logit, 2^((z - m) c), with the same single-term
// exponent the statistics summed (so that the weights of a row add up to its
// normaliser S).  m is finite, so -inf weighs 2^-inf = 0.
__device__ __forceinline__ float weight(float z, float m, float c_hi) { return ex2((z - m) * c_hi); }

__device__ __forceinline__ float warp_incl_scan(float x, int lane) {
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
        const float y = __shfl_up_sync(0xffffffffu, x, off);
        if (lane >= off) x += y;
    }
    return x;
}

__device__ __forceinline__ int warp_max_int(int x) {
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) x = max(x, __shfl_xor_sync(0xffffffffu, x, off));
    return x;
}

// Folds the (m, s) pairs of the 32 lanes: the maximum first, then one
// rescale per lane and a butterfly sum.  Every lane ends with the same pair.
__device__ __forceinline__ float2 warp_fold_sum(float m, float s, float c_hi, float c_lo) {
    float M = m;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, off));
    float t = m == kNegInf ? 0.f : s * ex2_scaled(m - M, c_hi, c_lo);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) t += __shfl_xor_sync(0xffffffffu, t, off);
    return make_float2(M, t);
}

// (max, lowest id of the max) over the 32 lanes, in every lane.
__device__ __forceinline__ float2 warp_fold_argmax(float2 acc) {
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
        float2 o;
        o.x = __shfl_xor_sync(0xffffffffu, acc.x, off);
        o.y = __shfl_xor_sync(0xffffffffu, acc.y, off);
        argmax_fold(acc, o);
    }
    return acc;
}

// Row r of request b: target rows 0 .. n_t-1, then draft rows.
template <typename T>
__device__ __forceinline__ const T* row_ptr(const AcceptParams& p, int b, int r) {
    const int V = p.V, nt = p.n_t;
    return r < nt ? static_cast<const T*>(p.target) + ((size_t)b * nt + r) * V
                  : static_cast<const T*>(p.draft) + ((size_t)b * p.d_rows + (r - nt)) * V;
}

// Bit u set iff tree node u of the parent array `par` (n <= 64 nodes) has a
// child; every lane of the warp returns the same mask.
__device__ __forceinline__ uint64_t tree_child_mask(const int32_t* par, int n, int lane) {
    uint64_t m = 0;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const int c = lane + 32 * h;
        if (c > 0 && c < n) {
            const int q = __ldg(par + c);
            if (q >= 0 && q < c) m |= 1ull << q;
        }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) m |= __shfl_xor_sync(0xffffffffu, m, off);
    return m;
}

// x / d for x >= 0, d > 0: one 32-bit division whenever both fit (every
// realistic problem), the 64-bit routine otherwise.
__device__ __forceinline__ long long div_nn(long long x, long long d) {
    if ((unsigned long long)x <= 0xffffffffull && (unsigned long long)d <= 0xffffffffull)
        return (long long)((unsigned)x / (unsigned)d);
    return x / d;
}

// First item of warp w's range (kernel 1's balanced split).
__device__ __forceinline__ long long range_lo(const AcceptParams& p, long long w) {
    return div_nn(w * p.N, p.W);
}

// Programmatic dependent launch: each kernel may start while the one before
// it runs; it waits here before reading what that kernel wrote (a no-op
// when it was launched without the attribute).
__device__ __forceinline__ void wait_prior_grid() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void allow_dependent_launch() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// ------------------------------------------------------------ kernel 1
// Largest of the 8 * kVecs logits of one lane's item (bf16: packed maxima,
// one instruction per pair).
__device__ __forceinline__ float item_max(const uint4 (&v)[kVecs], __nv_bfloat16) {
    __nv_bfloat162 a = *reinterpret_cast<const __nv_bfloat162*>(&v[0].x);
    __nv_bfloat162 b = *reinterpret_cast<const __nv_bfloat162*>(&v[0].y);
    __nv_bfloat162 c = *reinterpret_cast<const __nv_bfloat162*>(&v[0].z);
    __nv_bfloat162 d = *reinterpret_cast<const __nv_bfloat162*>(&v[0].w);
#pragma unroll
    for (int u = 1; u < kVecs; ++u) {
        a = __hmax2(a, *reinterpret_cast<const __nv_bfloat162*>(&v[u].x));
        b = __hmax2(b, *reinterpret_cast<const __nv_bfloat162*>(&v[u].y));
        c = __hmax2(c, *reinterpret_cast<const __nv_bfloat162*>(&v[u].z));
        d = __hmax2(d, *reinterpret_cast<const __nv_bfloat162*>(&v[u].w));
    }
    a = __hmax2(__hmax2(a, b), __hmax2(c, d));
    return fmaxf(__low2float(a), __high2float(a));
}

__device__ __forceinline__ float item_max(const uint4 (&v)[kVecs], float) {
    float a = kNegInf, b = kNegInf;
#pragma unroll
    for (int u = 0; u < kVecs; ++u) {
        a = fmaxf(a, fmaxf(__uint_as_float(v[u].x), __uint_as_float(v[u].y)));
        b = fmaxf(b, fmaxf(__uint_as_float(v[u].z), __uint_as_float(v[u].w)));
    }
    return fmaxf(a, b);
}

// The logits of a 32-bit word: two bf16 (low half first) or one fp32.
__device__ __forceinline__ float word_lo(uint32_t x, __nv_bfloat16) { return __uint_as_float(x << 16); }
__device__ __forceinline__ float word_hi(uint32_t x, __nv_bfloat16) { return __uint_as_float(x & 0xffff0000u); }

// sum over one lane's item of 2^((z - m) c_hi), four independent partial sums.
template <typename T>
__device__ __forceinline__ float item_sum(const uint4 (&v)[kVecs], float m, float c_hi) {
    float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
#pragma unroll
    for (int u = 0; u < kVecs; ++u) {
        const uint32_t w[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
        if constexpr (sizeof(T) == 2) {
            s0 += ex2((word_lo(w[0], T()) - m) * c_hi);
            s1 += ex2((word_hi(w[0], T()) - m) * c_hi);
            s2 += ex2((word_lo(w[1], T()) - m) * c_hi);
            s3 += ex2((word_hi(w[1], T()) - m) * c_hi);
            s0 += ex2((word_lo(w[2], T()) - m) * c_hi);
            s1 += ex2((word_hi(w[2], T()) - m) * c_hi);
            s2 += ex2((word_lo(w[3], T()) - m) * c_hi);
            s3 += ex2((word_hi(w[3], T()) - m) * c_hi);
        } else {
            s0 += ex2((__uint_as_float(w[0]) - m) * c_hi);
            s1 += ex2((__uint_as_float(w[1]) - m) * c_hi);
            s2 += ex2((__uint_as_float(w[2]) - m) * c_hi);
            s3 += ex2((__uint_as_float(w[3]) - m) * c_hi);
        }
    }
    return (s0 + s1) + (s2 + s3);
}

template <typename T, bool kGreedy>
__global__ void __launch_bounds__(kThreads, 2) accept_stats_kernel(const AcceptParams p) {
    constexpr int kPer = 16 / (int)sizeof(T);
    constexpr int kItem = kItemBytes / (int)sizeof(T);
    const int lane = threadIdx.x & 31;
    const long long w = (long long)blockIdx.x * kWarps + (threadIdx.x >> 5);
    // launched as a programmatic dependent of the kernel before it: its
    // inputs are read only past this wait, and the second kernel (which
    // reads some inputs before its own wait) only starts after it
    wait_prior_grid();
    allow_dependent_launch();
    if (w >= p.W) return;
    const long long lo = range_lo(p, w), hi = range_lo(p, w + 1);
    const int I = p.I, V = p.V, R = p.R;
    // tree: the draft row of a node without children is never used; its
    // items are skipped (read as -inf).  The child mask is cached per request.
    long long kids_b = -1;
    uint64_t kids = 0;
    auto unused_row = [&](long long row) -> bool {
        if (kGreedy || !p.parents) return false;
        const int r = (int)(row % R);
        if (r < p.n_t) return false;
        const long long b = row / R;
        if (b != kids_b) {
            kids = tree_child_mask(p.parents + (size_t)b * p.n_t, p.n_t, lane);
            kids_b = b;
        }
        return !((kids >> (r - p.n_t)) & 1ull);
    };

    // One item into registers: lane l holds vectors u*32 + l; entries past
    // the row's end read as -inf.
    auto load = [&](long long row, int item, uint4 (&v)[kVecs]) {
        if (unused_row(row)) {
            Vec16<T> ninf;
#pragma unroll
            for (int e = 0; e < 16 / (int)sizeof(T); ++e) ninf.t[e] = (T)kNegInf;
#pragma unroll
            for (int u = 0; u < kVecs; ++u) v[u] = ninf.q;
            return;
        }
        const T* rp = row_ptr<T>(p, (int)(row / R), (int)(row % R));
        const int e0 = item * kItem, e1 = min(V, e0 + kItem);
        if (aligned16(rp) && e1 - e0 == kItem) {
#pragma unroll
            for (int u = 0; u < kVecs; ++u) v[u] = ld_stream(rp + e0 + (u * 32 + lane) * kPer);
        } else {
            const bool vec = aligned16(rp);
#pragma unroll
            for (int u = 0; u < kVecs; ++u) v[u] = load16<T, true>(rp, e0 + (u * 32 + lane) * kPer, e1, vec);
        }
    };

    long long row = div_nn(lo, I);
    int item = (int)(lo - row * I);
    uint4 cur[kVecs], nxt[kVecs];
    load(row, item, cur);
    float m = kNegInf, s = 0.f;            // sampling: lane's running (max, sum)
    int id = INT_MAX;                      // greedy: lane's lowest id of the max (m)
    for (long long f = lo; f < hi; ++f) {
        long long nrow = row;
        int nitem = item + 1;
        if (nitem == I) {
            nrow = row + 1;
            nitem = 0;
        }
        if (f + 1 < hi) load(nrow, nitem, nxt);
        if (kGreedy) {
            const int base = item * kItem;
#pragma unroll
            for (int u = 0; u < kVecs; ++u) {   // ascending ids: strict > keeps the lowest
                Vec16<T> v;
                v.q = cur[u];
#pragma unroll
                for (int e = 0; e < kPer; ++e) {
                    const float z = to_f(v.t[e]);
                    if (z > m) {
                        m = z;
                        id = base + (u * 32 + lane) * kPer + e;
                    }
                }
            }
        } else {
            const float mi = item_max(cur, T());
            if (mi > m) {
                s = m == kNegInf ? 0.f : s * ex2_scaled(m - mi, p.c_hi, p.c_lo);
                m = mi;
            }
            if (m != kNegInf) s += item_sum<T>(cur, m, p.c_hi);
        }
        if (nitem == 0 || f + 1 == hi) {
            // the row segment ends: fold the lanes and publish the pair in
            // slot w - (owner of the row's first item) of the row
            const float2 acc = kGreedy ? warp_fold_argmax(make_float2(m, __int_as_float(id)))
                                       : warp_fold_sum(m, s, p.c_hi, p.c_lo);
            if (lane == 0) {
                const long long first_owner = div_nn((row * I + 1) * p.W - 1, p.N);
                const int j = (int)(w - first_owner);
                p.part[row * p.J + j] = acc;
                if (nitem == 0) p.cnt[row] = j + 1;   // this warp holds the row's last item
            }
            m = kNegInf;
            s = 0.f;
            id = INT_MAX;
        }
        row = nrow;
        item = nitem;
#pragma unroll
        for (int u = 0; u < kVecs; ++u) cur[u] = nxt[u];
    }
}

// ------------------------------------------------- row statistics (kernel 2)
// Row g's partials are part[g*J .. g*J + cnt[g]), in the order of the row.
// Lane l folds slots l, l+32, ... in order, then the lanes are folded; the
// result is the same in every lane and in every CTA that folds row g.
// The rows of one call are folded kBatch at a time, with the loads of a
// whole batch in flight together.
template <bool kGreedy, int kBatch>
__device__ __forceinline__ void fold_rows(const AcceptParams& p, int b, int first_row, int row_step,
                                          int n_rows, int lane, float2* s_stat) {
    const float2 empty = make_float2(kNegInf, kGreedy ? __int_as_float(INT_MAX) : 0.f);
    for (int r0 = first_row; r0 < n_rows; r0 += kBatch * row_step) {
        float2 pre[kBatch];
        int n[kBatch];
#pragma unroll
        for (int j = 0; j < kBatch; ++j) {
            const int r = r0 + j * row_step;
            pre[j] = empty;
            n[j] = 0;
            if (r < n_rows) {
                const long long g = (long long)b * p.R + r;
                n[j] = __ldcg(p.cnt + g);
                if (lane < p.J) pre[j] = __ldcg(p.part + g * p.J + lane);
            }
        }
#pragma unroll
        for (int j = 0; j < kBatch; ++j) {
            const int r = r0 + j * row_step;
            if (r >= n_rows) break;
            const long long g = (long long)b * p.R + r;
            float2 f = lane < n[j] ? pre[j] : empty;
            for (int l = lane + 32; l < n[j]; l += 32) {
                const float2 o = __ldcg(p.part + g * p.J + l);
                if (kGreedy) argmax_fold(f, o);
                else fold(f.x, f.y, o.x, o.y, p.c_hi, p.c_lo);
            }
            f = kGreedy ? warp_fold_argmax(f) : warp_fold_sum(f.x, f.y, p.c_hi, p.c_lo);
            if (lane == 0) s_stat[r] = f;
        }
    }
}

// ------------------------------------------------------------ accept test
// p(x) / q(x) of a drafted token: zt, zd are its target and draft logits,
// st, sd the rows' statistics; 0 for an invalid token or p(x) == 0, +inf
// when q(x) == 0.
__device__ __forceinline__ float accept_ratio(bool valid, float zt, float zd, float2 st, float2 sd,
                                              float c_hi, float c_lo) {
    if (!valid || zt == kNegInf) return 0.f;
    if (zd == kNegInf) return __int_as_float(0x7f800000);
    // log2 p(x)/q(x) = ((zt - mt) - (zd - md)) c + log2 Sd - log2 St, carried
    // as an unevaluated float pair
    const float dz = (zt - st.x) - (zd - sd.x);
    const float A = dz * c_hi;
    float E = fmaf(dz, c_lo, fmaf(dz, c_hi, -A));
    const float Bl = lg2(sd.y) - lg2(st.y);
    const float H = A + Bl;
    const float bb = H - A;
    E += (A - (H - bb)) + (Bl - bb);
    return ex2(H) * fmaf(E, kLn2, 1.f);
}

// Whether position i rejects: u_i < p_i(x_i) / q_i(x_i) fails.
__device__ __forceinline__ bool rejects(bool valid, float zt, float zd, float2 st, float2 sd, float u,
                                        float c_hi, float c_lo) {
    return !(u < accept_ratio(valid, zt, zd, st, sd, c_hi, c_lo));
}

// ------------------------------------------------------------ cluster PTX
__device__ __forceinline__ uint32_t cluster_rank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}

__device__ __forceinline__ uint32_t cluster_size() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_nctarank;" : "=r"(r));
    return r;
}

__device__ __forceinline__ void cluster_arrive() {
    asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
}

__device__ __forceinline__ void cluster_wait() {
    asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// Reads a float2 at the same shared-memory offset in CTA `rank` of the cluster.
__device__ __forceinline__ float2 ld_cluster_f2(const float2* local, uint32_t rank) {
    uint32_t remote;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(smem_u32(local)), "r"(rank));
    float2 v;
    asm volatile("ld.shared::cluster.v2.f32 {%0, %1}, [%2];" : "=f"(v.x), "=f"(v.y) : "r"(remote) : "memory");
    return v;
}

// ------------------------------------------------------------ draw weights
// Weights of thread-run [start, start + kRun) of the draw row pair (entries at
// or past `end` weigh zero): max(p - q, 0), or p alone when !residual.
template <typename T>
// The draw weights are p and max(p - q, 0) scaled by S_t (the inverse CDF
// does not depend on a common factor): 2^((zt - mt)c) and
// max(2^((zt - mt)c) - rho 2^((zd - md)c), 0) with rho = S_t / S_d.
struct DrawRow {
    const T* rt;
    const T* rd;
    float mt, md, rho, c_hi;
    bool at, ad;
};

template <typename T, bool kResidual>
__device__ __forceinline__ void run_weights(const DrawRow<T>& d, int start, int end,
                                            float (&w)[kRunVecs * 16 / sizeof(T)]) {
    constexpr int kPer = 16 / (int)sizeof(T);
    uint4 vt[kRunVecs], vd[kRunVecs];
    if (d.at && (!kResidual || d.ad) && start + kRunVecs * kPer <= end) {
#pragma unroll
        for (int u = 0; u < kRunVecs; ++u) {
            vt[u] = __ldg(reinterpret_cast<const uint4*>(d.rt + start + u * kPer));
            if (kResidual) vd[u] = __ldg(reinterpret_cast<const uint4*>(d.rd + start + u * kPer));
        }
    } else {
#pragma unroll
        for (int u = 0; u < kRunVecs; ++u) {
            vt[u] = load16<T, false>(d.rt, start + u * kPer, end, d.at);
            if (kResidual) vd[u] = load16<T, false>(d.rd, start + u * kPer, end, d.ad);
        }
    }
#pragma unroll
    for (int u = 0; u < kRunVecs; ++u) {
        Vec16<T> a, b;
        a.q = vt[u];
        if (kResidual) b.q = vd[u];
#pragma unroll
        for (int e = 0; e < kPer; ++e) {
            const float pt = weight(to_f(a.t[e]), d.mt, d.c_hi);
            if (kResidual) w[u * kPer + e] = fmaxf(fmaf(-d.rho, weight(to_f(b.t[e]), d.md, d.c_hi), pt), 0.f);
            else w[u * kPer + e] = pt;
        }
    }
}

// One pass of a CTA over logits [pass_start, pass_start + kDrawThreads*kRun):
// every thread's weights, its inclusive scan position and the pass total.
// The warp totals are folded in warp order, so the pass total and every
// thread's prefix are the same numbers whenever the pass is recomputed.
struct PassScan {
    float incl;    // mass of the pass up to and including this thread's run
    float excl;    // incl less the thread's own run (the start of its walk)
    float own;     // mass of this thread's run
    float total;   // mass of the pass
    int last;      // largest id of the pass with positive weight, -1 if none
};

template <typename T, bool kResidual>
__device__ __forceinline__ PassScan pass_scan_t(const DrawRow<T>& d, int pass_start, int end,
                                              float (&w)[kRunVecs * 16 / sizeof(T)], float (&s_wsum)[kDrawWarps],
                                              int (&s_wlast)[kDrawWarps]) {
    constexpr int kRun = kRunVecs * 16 / (int)sizeof(T);
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    const int start = pass_start + tid * kRun;
    run_weights<T, kResidual>(d, start, end, w);
    float ls = 0.f;
    int lp = -1;
#pragma unroll
    for (int e = 0; e < kRun; ++e) {
        ls += w[e];
        if (w[e] > 0.f) lp = start + e;
    }
    const float incl = warp_incl_scan(ls, lane);
    lp = warp_max_int(lp);
    if (lane == 31) s_wsum[wid] = incl;
    if (lane == 0) s_wlast[wid] = lp;
    __syncthreads();
    PassScan r;
    float off = 0.f, tot = 0.f;
    int last = -1;
#pragma unroll
    for (int j = 0; j < kDrawWarps; ++j) {
        if (j == wid) off = tot;
        tot += s_wsum[j];
        last = max(last, s_wlast[j]);
    }
    __syncthreads();   // s_wsum / s_wlast are reused by the next pass
    // the last thread's incl is the pass total bit for bit (same additions)
    r.incl = off + incl;
    r.excl = r.incl - ls;
    r.own = ls;
    r.total = tot;
    r.last = last;
    return r;
}

template <typename T>
__device__ __forceinline__ PassScan pass_scan(const DrawRow<T>& d, bool residual, int pass_start, int end,
                                              float (&w)[kRunVecs * 16 / sizeof(T)], float (&s_wsum)[kDrawWarps],
                                              int (&s_wlast)[kDrawWarps]) {
    return residual ? pass_scan_t<T, true>(d, pass_start, end, w, s_wsum, s_wlast)
                    : pass_scan_t<T, false>(d, pass_start, end, w, s_wsum, s_wlast);
}

// Per-warp pass totals of a slice (one block-wide buffer per kernel).
__device__ __forceinline__ float* draw_warp_pass_totals() {
    __shared__ float s_wpass[kDrawWarps * kMaxPasses];
    return s_wpass;
}

struct SliceMass {
    float mass;   // the slice's mass: the pass totals added in pass order
    int last;     // largest id of the slice with positive weight, -1 if none
};

// All n_pass passes of this CTA's slice [c0, c1), streamed without a block
// barrier per pass: each warp folds its runs with the warp scan of pass_scan
// and leaves its total for the pass; one barrier at the end, then every pass
// total is the warp totals added in warp order, bit for bit the total that
// pass_scan computes when the pass is walked again.  s_pass[ps] receives
// them.
template <typename T, bool kResidual>
__device__ __forceinline__ SliceMass slice_passes_t(const DrawRow<T>& d, int c0, int c1, int n_pass, float* s_pass,
                                                    int (&s_wlast)[kDrawWarps]) {
    constexpr int kRun = kRunVecs * 16 / (int)sizeof(T);
    constexpr int kPass = kDrawThreads * kRun;
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    float* s_wpass = draw_warp_pass_totals();
    float w[kRun];
    int last = -1;
    for (int ps = 0; ps < n_pass; ++ps) {
        const int nx = c0 + (ps + 1) * kPass + tid * kRun;
        if (ps + 1 < n_pass && (tid & 3) == 0 && nx < c1) {
            // the next pass into L1 while this one is reduced (a 128-byte
            // line holds the runs of four threads); only addresses inside the
            // slice are touched
            asm volatile("prefetch.global.L1 [%0];" ::"l"(d.rt + nx));
            if (kResidual) asm volatile("prefetch.global.L1 [%0];" ::"l"(d.rd + nx));
        }
        const int start = c0 + ps * kPass + tid * kRun;
        run_weights<T, kResidual>(d, start, c1, w);
        float ls = 0.f;
#pragma unroll
        for (int e = 0; e < kRun; ++e) {
            ls += w[e];
            if (w[e] > 0.f) last = start + e;
        }
        const float incl = warp_incl_scan(ls, lane);
        if (lane == 31) s_wpass[wid * kMaxPasses + ps] = incl;
    }
    last = warp_max_int(last);
    if (lane == 0) s_wlast[wid] = last;
    __syncthreads();
    if (tid < n_pass) {
        float tot = 0.f;
#pragma unroll
        for (int j = 0; j < kDrawWarps; ++j) tot += s_wpass[j * kMaxPasses + tid];
        s_pass[tid] = tot;
    }
    SliceMass r{0.f, -1};
#pragma unroll
    for (int j = 0; j < kDrawWarps; ++j) r.last = max(r.last, s_wlast[j]);
    __syncthreads();
    for (int ps = 0; ps < n_pass; ++ps) r.mass += s_pass[ps];
    __syncthreads();   // s_wlast / s_pass stay unchanged until every thread has read them
    return r;
}

template <typename T>
__device__ __forceinline__ SliceMass slice_passes(const DrawRow<T>& d, bool residual, int c0, int c1, int n_pass,
                                                  float* s_pass, int (&s_wlast)[kDrawWarps]) {
    return residual ? slice_passes_t<T, true>(d, c0, c1, n_pass, s_pass, s_wlast)
                    : slice_passes_t<T, false>(d, c0, c1, n_pass, s_pass, s_wlast);
}

// ------------------------------------------------------------ the draw
// Inverse-CDF draw of one token from the weights of row pair d -- p, or
// max(p - rho q, 0) when `residual` (rho as folded into d) -- over the
// vocabulary slices of the cluster: this CTA owns [c0, c1) in n_pass passes.
// Round 0 sums the slice masses and swaps them through distributed shared
// memory; a residual without positive mass falls back to p in round 1.  On
// return `writer` is the thread of this CTA that stores `token` (-1: another
// CTA does).  Exchange slots alternate with the round counter xr, so one
// cluster barrier per round keeps a slot from being rewritten while a peer
// may still read it.
template <typename T>
__device__ __forceinline__ void cluster_draw(const DrawRow<T>& d, bool residual, float uk, int c0, int c1,
                                             int n_pass, uint32_t rank, uint32_t n_ranks, float* s_pass,
                                             float (&s_wsum)[kDrawWarps], int (&s_wlast)[kDrawWarps],
                                             int (&s_first)[kDrawWarps], float2* s_x, int& xr, int& token,
                                             int& writer) {
    constexpr int kPer = 16 / (int)sizeof(T);
    constexpr int kRun = kRunVecs * kPer;
    constexpr int kPass = kDrawThreads * kRun;
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    float w[kRun];
    token = 0;
    writer = -1;
    for (int round = 0; round < 2; ++round) {
        // one pass: scanned at once, its weights and prefixes kept for the
        // walk; several: streamed, and the owning pass walked again
        PassScan kept{0.f, 0.f, 0.f, 0.f, -1};
        SliceMass sm{0.f, -1};
        if (n_pass == 1) {
            kept = pass_scan<T>(d, residual, c0, c1, w, s_wsum, s_wlast);
            if (tid == 0) s_pass[0] = kept.total;
            sm.mass = kept.total;
            sm.last = kept.last;
        } else {
            sm = slice_passes<T>(d, residual, c0, c1, n_pass, s_pass, s_wlast);
        }
        const float mass = sm.mass;
        const int last = sm.last;
        const int slot = xr & 1;
        ++xr;
        if (tid == 0) s_x[slot] = make_float2(mass, __int_as_float(last));
        cluster_arrive();
        cluster_wait();
        // every CTA folds the masses of ranks 0..n-1 in the same order
        float2 x = make_float2(0.f, __int_as_float(-1));
        if (lane < (int)n_ranks) x = ld_cluster_f2(&s_x[slot], lane);
        const float incl = warp_incl_scan(x.x, lane);
        const float Z = __shfl_sync(0xffffffffu, incl, 31);
        if (!(Z > 0.f) && residual && round == 0) {
            // no positive residual (p == q up to rounding): draw from p instead
            residual = false;
            continue;
        }
        const float t = uk * Z;
        const float before = incl - x.x;
        const unsigned own = __ballot_sync(0xffffffffu, lane < (int)n_ranks && x.x > 0.f && incl > t);
        if (!own) {
            // u_k * Z at or past the total through rounding: the last positive weight
            const int lp = warp_max_int(__float_as_int(x.y));
            token = lp >= 0 ? lp : 0;
            if (rank == 0) writer = 0;
            break;
        }
        const int owner = __ffs(own) - 1;
        if ((int)rank != owner) break;
        float tt = t - __shfl_sync(0xffffffffu, before, owner);   // position within this slice
        // the pass that holds the cell, in the order the mass was summed
        int pj = -1;
        float cum = 0.f;
        for (int ps = 0; ps < n_pass; ++ps) {
            const float m = s_pass[ps];
            if (m > 0.f && cum + m > tt) {
                pj = ps;
                break;
            }
            cum += m;
        }
        if (pj < 0) {   // rounding: the slice's last positive weight
            token = last;
            writer = 0;
            break;
        }
        tt -= cum;
        // walked again, the pass's scan reproduces its total bit for bit
        const PassScan sc = n_pass == 1 ? kept : pass_scan<T>(d, residual, c0 + pj * kPass, c1, w, s_wsum, s_wlast);
        // the first run with positive mass whose prefix passes tt (a run of
        // zero weights can come first through rounding; it never owns the draw)
        const unsigned cross = __ballot_sync(0xffffffffu, sc.own > 0.f && sc.incl > tt);
        if (lane == 0) s_first[wid] = cross ? wid * 32 + __ffs(cross) - 1 : INT_MAX;
        __syncthreads();
        int first = INT_MAX;
#pragma unroll
        for (int j = 0; j < kDrawWarps; ++j) first = min(first, s_first[j]);
        if (first == INT_MAX) {   // rounding: the pass's last positive weight
            token = sc.last;
            writer = 0;
            break;
        }
        if (tid == first) {
            const int start = c0 + pj * kPass + tid * kRun;
            float c = sc.excl;
            int pick = -1, lastp = -1;
#pragma unroll
            for (int e = 0; e < kRun; ++e) {
                c += w[e];
                if (w[e] > 0.f) {   // only a token with positive weight can be drawn
                    lastp = start + e;
                    if (pick < 0 && c > tt) pick = start + e;
                }
            }
            token = pick >= 0 ? pick : lastp;   // the run has a positive weight
        }
        writer = first;
        break;
    }}

// ------------------------------------------------------------ kernel 2
template <typename T>
__global__ void __launch_bounds__(kDrawThreads, 2) accept_draw_kernel(const AcceptParams p) {
    constexpr int kPer = 16 / (int)sizeof(T);
    constexpr int kRun = kRunVecs * kPer;
    constexpr int kPass = kDrawThreads * kRun;
    __shared__ float2 s_stat[kMaxRows];
    __shared__ float s_pass[kMaxPasses];
    __shared__ float s_wsum[kDrawWarps];
    __shared__ int s_wlast[kDrawWarps];
    __shared__ int s_first[kDrawWarps];
    __shared__ int s_a;
    __shared__ float2 s_x[2];   // (slice mass, last positive id) per exchange round

    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    const uint32_t rank = cluster_rank(), n_ranks = cluster_size();
    const int b = p.b_base + blockIdx.y;
    const int k = p.k, V = p.V;

    // ---- the accept-test inputs of lane i < k of warp 0, loaded first
    bool valid = false;
    float zt = 0.f, zd = 0.f, ui = 1.f;
    int xi = -1;
    if (wid == 0 && lane < k) {
        xi = __ldg(p.tokens + (size_t)b * k + lane);
        ui = __ldg(p.uniforms + (size_t)b * (k + 1) + lane);
        valid = xi >= 0 && xi < V;
        if (valid) {
            zt = to_f(row_ptr<T>(p, b, lane)[xi]);
            zd = to_f(row_ptr<T>(p, b, k + 1 + lane)[xi]);
        }
    }
    const float uk = __ldg(p.uniforms + (size_t)b * (k + 1) + k);

    // ---- row statistics of the request (kernel 1's output), then the tests
    wait_prior_grid();
    allow_dependent_launch();   // the next call's first kernel may start
    fold_rows<false, kRowsPerDrawWarp>(p, b, wid, kDrawWarps, p.R, lane, s_stat);
    __syncthreads();
    if (wid == 0) {
        bool rej = false;
        if (lane < k) rej = rejects(valid, zt, zd, s_stat[lane], s_stat[k + 1 + lane], ui, p.c_hi, p.c_lo);
        const unsigned m = __ballot_sync(0xffffffffu, rej);
        if (lane == 0) s_a = m ? __ffs(m) - 1 : k;
    }
    __syncthreads();
    const int a = s_a;

    // ---- the draw: this CTA's slice [c0, c1) of row pair a
    const int c0 = min(V, (int)rank * p.slice), c1 = min(V, c0 + p.slice);
    const int n_pass = (c1 - c0 + kPass - 1) / kPass;
    DrawRow<T> d;
    d.rt = row_ptr<T>(p, b, a);
    d.rd = a < k ? row_ptr<T>(p, b, k + 1 + a) : d.rt;
    // a row without a finite entry (outside the contract) weighs zero everywhere
    const float2 st = s_stat[a], sd = a < k ? s_stat[k + 1 + a] : make_float2(0.f, 0.f);
    d.mt = st.x == kNegInf ? 0.f : st.x;
    d.md = sd.x == kNegInf ? 0.f : sd.x;
    d.rho = sd.y > 0.f ? st.y / sd.y : 0.f;
    d.c_hi = p.c_hi;
    d.at = aligned16(d.rt);
    d.ad = aligned16(d.rd);

    if (n_pass > 1) {
        // several passes: ask L2 for the whole slice of the row pair now, so
        // that the passes below find it there instead of waiting on DRAM
        const char* bt = reinterpret_cast<const char*>(d.rt + c0);
        const char* bd = reinterpret_cast<const char*>(d.rd + c0);
        const int bytes = (c1 - c0) * (int)sizeof(T);
        for (int off = tid * 128; off < bytes; off += kDrawThreads * 128) {
            asm volatile("prefetch.global.L2 [%0];" ::"l"(bt + off));
            if (a < k) asm volatile("prefetch.global.L2 [%0];" ::"l"(bd + off));
        }
    }
    int token = 0;
    int writer = -1;   // the thread of this CTA that writes the emitted token
    int xr = 0;
    cluster_draw<T>(d, a < k, uk, c0, c1, n_pass, rank, n_ranks, s_pass, s_wsum, s_wlast, s_first, s_x, xr,
                    token, writer);
    if (tid == writer) p.out_tokens[(size_t)b * (k + 1) + a] = token >= 0 ? token : 0;
    if (rank == 0 && tid <= k && tid != a) {
        const int32_t x = tid < a ? __ldg(p.tokens + (size_t)b * k + tid) : -1;
        p.out_tokens[(size_t)b * (k + 1) + tid] = x;
    }
    if (rank == 0 && tid == 0 && p.out_n) p.out_n[b] = a;
    // no CTA leaves while another may still read its exchange slots
    cluster_arrive();
    cluster_wait();
}

// ------------------------------------------------------------ greedy
template <typename T>
__global__ void __launch_bounds__(kThreads) accept_greedy_kernel(const AcceptParams p) {
    __shared__ float2 s_stat[kWarps][kMaxRows];
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    const int b = blockIdx.x * kWarps + wid;
    const int k = p.k;
    wait_prior_grid();
    allow_dependent_launch();   // the next call's first kernel may start
    if (b >= p.B) return;
    fold_rows<true, 4>(p, b, 0, 1, k + 1, lane, s_stat[wid]);
    __syncwarp();
    int g = 0, x = -1;
    if (lane <= k) {
        g = __float_as_int(s_stat[wid][lane].y);
        if (g == INT_MAX) g = 0;   // a row with no finite entry
    }
    if (lane < k) x = __ldg(p.tokens + (size_t)b * k + lane);
    const unsigned miss = __ballot_sync(0xffffffffu, lane < k && x != g);
    const int a = miss ? __ffs(miss) - 1 : k;
    const int emit = __shfl_sync(0xffffffffu, g, a);
    if (lane <= k) p.out_tokens[(size_t)b * (k + 1) + lane] = lane < a ? x : (lane == a ? emit : -1);
    if (lane == 0 && p.out_n) p.out_n[b] = a;
}

// ------------------------------------------------------------ token trees
// Cluster-wide mass of the draw weights of row pair d (p scaled by S_t, or
// max(p - kappa q, 0) scaled by S_t when `residual`): every CTA sums its
// slice, the slice masses are swapped through distributed shared memory and
// folded in rank order, so every CTA holds the same total.
template <typename T>
__device__ __forceinline__ float cluster_mass(const DrawRow<T>& d, bool residual, int c0, int c1, int n_pass,
                                              uint32_t n_ranks, float (&s_wsum)[kDrawWarps],
                                              int (&s_wlast)[kDrawWarps], float2* s_x, int& xr) {
    __shared__ float s_tpass[kMaxPasses];
    const float mass = slice_passes<T>(d, residual, c0, c1, n_pass, s_tpass, s_wlast).mass;
    (void)s_wsum;
    const int slot = xr & 1;
    ++xr;
    if (threadIdx.x == 0) s_x[slot] = make_float2(mass, 0.f);
    cluster_arrive();
    cluster_wait();
    const int lane = threadIdx.x & 31;
    float2 x = make_float2(0.f, 0.f);
    if (lane < (int)n_ranks) x = ld_cluster_f2(&s_x[slot], lane);
    return __shfl_sync(0xffffffffu, warp_incl_scan(x.x, lane), 31);
}

// One cluster per request walks its tree (multi-candidate speculative
// sampling).  At node u the running distribution is r = max(p_u - kappa q_u,
// 0) / Z (kappa = 0, Z = 1: r = p_u); child c with token x is accepted iff
// u_{c-1} < r(x) / q_u(x) = max(p(x)/q(x) - kappa, 0) / Z.  A rejection
// makes r the residual max(0, r - q_u) normalised, which is the same form
// with kappa + Z in place of kappa; its mass is one cluster pass over the
// row pair, needed only when another sibling is still to be tested (the
// draw sums its own weights).  A residual without positive mass ends the
// tests and the draw falls back to p_u.
template <typename T>
__global__ void __launch_bounds__(kDrawThreads, 2) tree_draw_kernel(const AcceptParams p) {
    constexpr int kPer = 16 / (int)sizeof(T);
    constexpr int kRun = kRunVecs * kPer;
    constexpr int kPass = kDrawThreads * kRun;
    __shared__ float2 s_stat[2 * kMaxTreeNodes];
    __shared__ float2 s_z[kMaxTreeNodes];      // target / draft logit of node c's token in its parent's rows
    __shared__ int s_par[kMaxTreeNodes];
    __shared__ int s_tok[kMaxTreeNodes];
    __shared__ float s_u[kMaxTreeNodes];
    __shared__ unsigned long long s_kids[kMaxTreeNodes];
    __shared__ int s_path[kMaxTreeNodes];
    __shared__ float s_pass[kMaxPasses];
    __shared__ float s_wsum[kDrawWarps];
    __shared__ int s_wlast[kDrawWarps];
    __shared__ int s_first[kDrawWarps];
    __shared__ float2 s_x[2];

    const int tid = threadIdx.x, lane = tid & 31;
    const uint32_t rank = cluster_rank(), n_ranks = cluster_size();
    const int b = p.b_base + blockIdx.y;
    const int n = p.n_t, V = p.V;

    // ---- the tree and every accept-test input, loaded before the statistics
    for (int c = tid; c < n; c += kDrawThreads) {
        int par = -1;
        if (c > 0) {
            const int q = __ldg(p.parents + (size_t)b * n + c);
            par = (q >= 0 && q < c) ? q : -1;
        }
        const int x = __ldg(p.tokens + (size_t)b * n + c);
        s_par[c] = par;
        s_tok[c] = x;
        s_u[c] = __ldg(p.uniforms + (size_t)b * n + c);
        float2 z = make_float2(kNegInf, 0.f);    // an invalid token tests as ratio 0
        if (par >= 0 && x >= 0 && x < V)
            z = make_float2(to_f(row_ptr<T>(p, b, par)[x]), to_f(row_ptr<T>(p, b, n + par)[x]));
        s_z[c] = z;
    }
    __syncthreads();
    for (int u = tid; u < n; u += kDrawThreads) {
        unsigned long long m = 0;
        for (int c = u + 1; c < n; ++c)
            if (s_par[c] == u) m |= 1ull << c;
        s_kids[u] = m;
    }
    wait_prior_grid();
    allow_dependent_launch();   // the next call's first kernel may start
    fold_rows<false, 8>(p, b, tid >> 5, kDrawWarps, p.R, lane, s_stat);
    __syncthreads();

    // ---- the walk: every thread takes the same decisions from shared data
    const int c0 = min(V, (int)rank * p.slice), c1 = min(V, c0 + p.slice);
    const int n_pass = (c1 - c0 + kPass - 1) / kPass;
    int node = 0, depth = 0, xr = 0;
    float kappa = 0.f;
    DrawRow<T> d;
    d.c_hi = p.c_hi;
    for (;;) {
        const float2 st = s_stat[node], sd = s_stat[n + node];
        d.rt = row_ptr<T>(p, b, node);
        d.rd = row_ptr<T>(p, b, n + node);
        d.mt = st.x == kNegInf ? 0.f : st.x;
        d.md = sd.x == kNegInf ? 0.f : sd.x;
        d.at = aligned16(d.rt);
        d.ad = aligned16(d.rd);
        const float rho1 = sd.y > 0.f ? st.y / sd.y : 0.f;
        unsigned long long kids = s_kids[node];
        float kap = 0.f, Z = 1.f;
        int next = -1;
        while (kids) {
            const int c = __ffsll((long long)kids) - 1;
            kids &= kids - 1;
            const float2 z = s_z[c];
            float ratio = accept_ratio(z.x != kNegInf, z.x, z.y, st, sd, p.c_hi, p.c_lo);
            if (kap > 0.f) ratio = fmaxf(ratio - kap, 0.f) / Z;
            if (s_u[c - 1] < ratio) {
                next = c;
                break;
            }
            kap += Z;               // the residual of this rejection
            if (!kids) break;       // no sibling left: the draw sums its own weights
            d.rho = kap * rho1;
            Z = cluster_mass<T>(d, true, c0, c1, n_pass, n_ranks, s_wsum, s_wlast, s_x, xr) / st.y;
            if (!(Z > 0.f)) {       // no positive residual (p == kappa q up to rounding): draw from p
                kap = 0.f;
                break;
            }
        }
        if (next < 0) {
            kappa = kap;
            break;
        }
        if (tid == 0) s_path[depth] = next;
        ++depth;
        node = next;
    }

    // ---- the draw at the final node
    d.rho = kappa * (s_stat[n + node].y > 0.f ? s_stat[node].y / s_stat[n + node].y : 0.f);
    if (!(kappa > 0.f)) d.rd = d.rt;
    if (n_pass > 1) {
        const char* bt = reinterpret_cast<const char*>(d.rt + c0);
        const char* bd = reinterpret_cast<const char*>(d.rd + c0);
        const int bytes = (c1 - c0) * (int)sizeof(T);
        for (int off = tid * 128; off < bytes; off += kDrawThreads * 128) {
            asm volatile("prefetch.global.L2 [%0];" ::"l"(bt + off));
            if (kappa > 0.f) asm volatile("prefetch.global.L2 [%0];" ::"l"(bd + off));
        }
    }
    int token = 0, writer = -1;
    cluster_draw<T>(d, kappa > 0.f, s_u[n - 1], c0, c1, n_pass, rank, n_ranks, s_pass, s_wsum, s_wlast, s_first,
                    s_x, xr, token, writer);
    __syncthreads();
    int32_t* out = p.out_tokens + (size_t)b * n;
    if (tid == writer) out[depth] = token >= 0 ? token : 0;
    if (rank == 0) {
        for (int i = tid; i < n; i += kDrawThreads) {
            if (i < depth) {
                out[i] = s_tok[s_path[i]];
                p.out_path[(size_t)b * n + i] = s_path[i];
            } else {
                if (i > depth) out[i] = -1;
                p.out_path[(size_t)b * n + i] = -1;
            }
        }
        if (tid == 0) p.out_n[b] = depth;
    }
    // no CTA leaves while another may still read its exchange slots
    cluster_arrive();
    cluster_wait();
}

// Greedy tree walk, one warp per request: at node u the first child whose
// token is the arg max of u's target row is accepted, else that arg max is
// emitted.
template <typename T>
__global__ void __launch_bounds__(kThreads) tree_greedy_kernel(const AcceptParams p) {
    __shared__ float2 s_stat[kWarps][kMaxTreeNodes];
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    const int b = blockIdx.x * kWarps + wid;
    if (b >= p.B) return;
    const int n = p.n_t;
    int par[2], tok[2];
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const int c = lane + 32 * h;
        par[h] = -1;
        tok[h] = -1;
        if (c < n) {
            tok[h] = __ldg(p.tokens + (size_t)b * n + c);
            if (c > 0) {
                const int q = __ldg(p.parents + (size_t)b * n + c);
                par[h] = (q >= 0 && q < c) ? q : -1;
            }
        }
    }
    wait_prior_grid();
    allow_dependent_launch();   // the next call's first kernel may start
    fold_rows<true, 4>(p, b, 0, 1, n, lane, s_stat[wid]);
    __syncwarp();
    int32_t* out = p.out_tokens + (size_t)b * n;
    int32_t* path = p.out_path + (size_t)b * n;
    int node = 0, depth = 0, g = 0;
    for (;;) {
        g = __float_as_int(s_stat[wid][node].y);
        if (g == INT_MAX) g = 0;   // a row with no finite entry
        const unsigned m0 = __ballot_sync(0xffffffffu, par[0] == node && tok[0] == g);
        const unsigned m1 = __ballot_sync(0xffffffffu, par[1] == node && tok[1] == g);
        if (!m0 && !m1) break;
        const int next = m0 ? __ffs(m0) - 1 : 32 + __ffs(m1) - 1;
        if (lane == 0) {
            out[depth] = g;
            path[depth] = next;
        }
        ++depth;
        node = next;
    }
    for (int i = lane; i < n; i += 32) {
        if (i == depth) out[i] = g;
        else if (i > depth) out[i] = -1;
        if (i >= depth) path[i] = -1;
    }
    if (lane == 0) p.out_n[b] = depth;
}

// ------------------------------------------------------------------- host
// Resident CTAs of `kern` on the current device (cached per device and slot).
template <typename K>
int resident_ctas(K kern, int slot, int threads, int smem) {
    static int cache[64][8] = {};
    int dev = 0;
    cudaGetDevice(&dev);
    int occ = (dev >= 0 && dev < 64) ? cache[dev][slot] : 0;
    if (!occ) {
        if (smem > 48 * 1024) cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, kern, threads, smem) != cudaSuccess || occ <= 0)
            occ = 2;
        cudaGetLastError();
        if (dev >= 0 && dev < 64) cache[dev][slot] = occ;
    }
    return occ * current_sm_count();
}

int g_max_cluster[64] = {0};

// The largest cluster (16, non-portable, or 8) the device schedules for the
// draw kernel.
int max_cluster_size() {
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev < 0 || dev >= 64) return 8;
    if (g_max_cluster[dev]) return g_max_cluster[dev];
    int best = 8;
    void (*kerns[4])(const AcceptParams) = {accept_draw_kernel<__nv_bfloat16>, accept_draw_kernel<float>,
                                            tree_draw_kernel<__nv_bfloat16>, tree_draw_kernel<float>};
    bool attrs_ok = true;
    for (auto k : kerns)
        attrs_ok = attrs_ok && cudaFuncSetAttribute(k, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) == cudaSuccess;
    if (attrs_ok) {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(kMaxCluster, 1, 1);
        cfg.blockDim = dim3(kDrawThreads, 1, 1);
        cudaLaunchAttribute attr;
        attr.id = cudaLaunchAttributeClusterDimension;
        attr.val.clusterDim.x = kMaxCluster;
        attr.val.clusterDim.y = 1;
        attr.val.clusterDim.z = 1;
        cfg.attrs = &attr;
        cfg.numAttrs = 1;
        bool all = true;
        for (auto k : kerns) {
            int n = 0;
            all = all && cudaOccupancyMaxActiveClusters(&n, k, &cfg) == cudaSuccess && n > 0;
        }
        if (all) best = kMaxCluster;
    }
    cudaGetLastError();
    g_max_cluster[dev] = best;
    return best;
}

struct AcceptPlan {
    int R, I, W, J, grid1;
    long long N;
    int cluster, slice;
    size_t off_cnt, bytes;
};

template <typename T, bool G>
int stats_resident() {
    const int slot = (G ? 1 : 0) + (sizeof(T) == 4 ? 2 : 0);
    return resident_ctas(accept_stats_kernel<T, G>, slot, kThreads, 0);
}

// n_t target rows and d_rows draft rows per request (chain: k+1 and k;
// tree: the node count twice).
AcceptPlan plan_accept_rows(const cs_accept_dims& d, int n_t, int d_rows, bool greedy, bool with_cluster) {
    const bool f32 = d.logit_dtype == CS_F32;
    AcceptPlan P{};
    P.R = greedy ? n_t : n_t + d_rows;
    const int item = kItemBytes / (f32 ? 4 : 2);
    P.I = (d.vocab + item - 1) / item;
    P.N = (long long)d.batch * P.R * P.I;
    const int resident = f32 ? (greedy ? stats_resident<float, true>() : stats_resident<float, false>())
                             : (greedy ? stats_resident<__nv_bfloat16, true>()
                                       : stats_resident<__nv_bfloat16, false>());
    long long g = (P.N + kWarps - 1) / kWarps;
    if (g > resident) g = resident;
    P.grid1 = (int)(g > 0 ? g : 1);
    // every busy warp owns at least one item, so a row's segments come from
    // consecutive warps
    const long long warps = (long long)P.grid1 * kWarps;
    P.W = (int)(warps < P.N ? warps : (P.N > 0 ? P.N : 1));
    // a row meets at most (I-1)/q + 2 ranges of q >= 1 items, and at most I
    const long long q = P.N / P.W > 0 ? P.N / P.W : 1;
    const long long J = (P.I - 1) / q + 2;
    P.J = (int)(J < P.I ? J : P.I);
    const size_t rows = (size_t)d.batch * P.R;
    P.off_cnt = (rows * P.J * sizeof(float2) + 255) / 256 * 256;
    P.bytes = P.off_cnt + (rows * sizeof(int) + 255) / 256 * 256;
    if (!greedy && with_cluster) {
        // All clusters in one wave (two CTAs per SM), no CTA with an empty
        // slice, at most kMaxPasses passes per CTA.
        const int pass = kDrawThreads * kRunVecs * (f32 ? 4 : 8);
        const int sms = current_sm_count();
        int c = 2 * sms / (d.batch > 0 ? d.batch : 1);
        const int by_vocab = (d.vocab + pass - 1) / pass;
        if (c > by_vocab) c = by_vocab;
        const int cmax = max_cluster_size();
        if (c > cmax) c = cmax;
        const int need = (int)(((long long)d.vocab + (long long)kMaxPasses * pass - 1) / ((long long)kMaxPasses * pass));
        if (c < need) c = need;
        if (c < 1) c = 1;
        P.cluster = c;
        const int per = (d.vocab + c - 1) / c;
        P.slice = (per + 7) / 8 * 8;
    }
    return P;
}

AcceptPlan plan_accept(const cs_accept_dims& d, int n_draft, bool greedy, bool with_cluster) {
    return plan_accept_rows(d, n_draft + 1, n_draft, greedy, with_cluster);
}

template <typename T, bool G>
cs_status launch_typed(AcceptParams p, const AcceptPlan& P, bool tree, cudaStream_t stream) {
    // both kernels are programmatic dependents of the kernel before them:
    // each may start early and waits (griddepcontrol.wait) before it reads
    // what that kernel wrote
    cudaLaunchAttribute attrs[2];
    attrs[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attrs[0].val.programmaticStreamSerializationAllowed = 1;
    cudaError_t e;
    {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3((unsigned)P.grid1, 1, 1);
        cfg.blockDim = dim3(kThreads, 1, 1);
        cfg.stream = stream;
        cfg.attrs = attrs;
        cfg.numAttrs = 1;
        e = cudaLaunchKernelEx(&cfg, accept_stats_kernel<T, G>, p);
        if (e != cudaSuccess) return cuda_fail(e, "accept_stats_kernel launch");
    }
    if (G) {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3((p.B + kWarps - 1) / kWarps, 1, 1);
        cfg.blockDim = dim3(kThreads, 1, 1);
        cfg.stream = stream;
        cfg.attrs = attrs;
        cfg.numAttrs = 1;
        e = cudaLaunchKernelEx(&cfg, tree ? tree_greedy_kernel<T> : accept_greedy_kernel<T>, p);
        if (e != cudaSuccess) return cuda_fail(e, "greedy acceptance kernel launch");
        return CS_OK;
    }
    auto kern = tree ? tree_draw_kernel<T> : accept_draw_kernel<T>;
    if (P.cluster > 8) {
        e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
        if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute(non-portable cluster)");
    }
    attrs[1].id = cudaLaunchAttributeClusterDimension;
    attrs[1].val.clusterDim.x = P.cluster;
    attrs[1].val.clusterDim.y = 1;
    attrs[1].val.clusterDim.z = 1;
    for (int b0 = 0; b0 < p.B; b0 += 65535) {
        p.b_base = b0;
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(P.cluster, p.B - b0 < 65535 ? p.B - b0 : 65535, 1);
        cfg.blockDim = dim3(kDrawThreads, 1, 1);
        cfg.stream = stream;
        cfg.attrs = attrs;
        cfg.numAttrs = 2;
        e = cudaLaunchKernelEx(&cfg, kern, p);
        if (e != cudaSuccess) return cuda_fail(e, "acceptance draw kernel launch");
    }
    return CS_OK;
}

}  // namespace

size_t accept_workspace_bytes(const cs_accept_dims& d, int n_draft, float temperature) {
    if (temperature == 0.f) return plan_accept(d, n_draft, true, false).bytes;
    return plan_accept(d, n_draft, false, false).bytes;
}

size_t accept_workspace_bytes_any(const cs_accept_dims& d, int n_draft) {
    const size_t a = plan_accept(d, n_draft, true, false).bytes;
    const size_t b = plan_accept(d, n_draft, false, false).bytes;
    return a > b ? a : b;
}

cs_status launch_spec_accept(const cs_accept_dims& d, const void* target, const void* draft,
                             const int32_t* tokens, const float* uniforms, int n_draft,
                             float temperature, int32_t* out_tokens, int32_t* out_n,
                             void* workspace, cudaStream_t stream) {
    const bool greedy = temperature == 0.f;
    const AcceptPlan P = plan_accept(d, n_draft, greedy, true);
    AcceptParams p{};
    p.target = target;
    p.draft = draft;
    p.tokens = tokens;
    p.uniforms = uniforms;
    p.out_tokens = out_tokens;
    p.out_n = out_n;
    p.B = d.batch;
    p.V = d.vocab;
    p.k = n_draft;
    p.n_t = n_draft + 1;
    p.d_rows = n_draft;
    p.R = P.R;
    p.I = P.I;
    p.N = P.N;
    p.W = P.W;
    p.J = P.J;
    p.slice = P.slice;
    const double c = temperature > 0.f ? 1.4426950408889634 / (double)temperature : 0.0;
    p.c_hi = (float)c;
    p.c_lo = (float)(c - (double)p.c_hi);
    p.part = static_cast<float2*>(workspace);
    p.cnt = reinterpret_cast<int*>(static_cast<uint8_t*>(workspace) + P.off_cnt);
    if (d.logit_dtype == CS_F32)
        return greedy ? launch_typed<float, true>(p, P, false, stream) : launch_typed<float, false>(p, P, false, stream);
    return greedy ? launch_typed<__nv_bfloat16, true>(p, P, false, stream)
                  : launch_typed<__nv_bfloat16, false>(p, P, false, stream);
}

size_t tree_accept_workspace_bytes(const cs_accept_dims& d, int n_nodes) {
    const size_t a = plan_accept_rows(d, n_nodes, n_nodes, true, false).bytes;
    const size_t b = plan_accept_rows(d, n_nodes, n_nodes, false, false).bytes;
    return a > b ? a : b;
}

cs_status launch_tree_accept(const cs_accept_dims& d, const void* target, const void* draft,
                             const int32_t* parents, const int32_t* tokens, const float* uniforms, int n_nodes,
                             float temperature, int32_t* out_tokens, int32_t* out_path, int32_t* out_n,
                             void* workspace, cudaStream_t stream) {
    const bool greedy = temperature == 0.f;
    const AcceptPlan P = plan_accept_rows(d, n_nodes, n_nodes, greedy, true);
    AcceptParams p{};
    p.target = target;
    p.draft = draft;
    p.tokens = tokens;
    p.uniforms = uniforms;
    p.out_tokens = out_tokens;
    p.out_n = out_n;
    p.parents = parents;
    p.out_path = out_path;
    p.B = d.batch;
    p.V = d.vocab;
    p.k = n_nodes - 1;
    p.n_t = n_nodes;
    p.d_rows = n_nodes;
    p.R = P.R;
    p.I = P.I;
    p.N = P.N;
    p.W = P.W;
    p.J = P.J;
    p.slice = P.slice;
    const double c = temperature > 0.f ? 1.4426950408889634 / (double)temperature : 0.0;
    p.c_hi = (float)c;
    p.c_lo = (float)(c - (double)p.c_hi);
    p.part = static_cast<float2*>(workspace);
    p.cnt = reinterpret_cast<int*>(static_cast<uint8_t*>(workspace) + P.off_cnt);
    if (d.logit_dtype == CS_F32)
        return greedy ? launch_typed<float, true>(p, P, true, stream) : launch_typed<float, false>(p, P, true, stream);
    return greedy ? launch_typed<__nv_bfloat16, true>(p, P, true, stream)
                  : launch_typed<__nv_bfloat16, false>(p, P, true, stream);
}

}  // namespace cs
