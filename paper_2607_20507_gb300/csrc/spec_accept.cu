// spec_accept.cu -- the acceptance step of speculative sampling (the rule
// the paper's drafter follows, Sec. 3.4): temperature softmax statistics of
// target and draft rows, the min(1, p/q) accept test, the residual
// max(0, p - q) or bonus draw by inverse CDF, and the greedy variant.
//
// Design.  One thread-block cluster per request; CTA r of the cluster owns a
// contiguous slice of the vocabulary.  Positions are handled in order:
//   1. each CTA streams its slice of target row i (and draft row i) once
//      with 128-bit loads, keeping a running (max, sum 2^((z-max)c)) per
//      thread (one exponential per logit), then reduces it with warp
//      shuffles and shared memory;
//   2. the CTAs swap their partial statistics through distributed shared
//      memory and fold them in rank order, so every CTA holds bit-identical
//      row statistics and takes the same accept decision;
//   3. the first rejection ends the loop: rows after it cannot change the
//      result and are never read.
// The draw re-reads the slice of the deciding row pair (just read, so served
// by L2): a block prefix scan over the slice gives each CTA its mass, the
// cluster folds the masses in rank order, and the CTA whose cell contains
// u*Z scans again to find the token.  No probability is written to memory.
#include <cooperative_groups.h>
#include <limits.h>
#include <math.h>

#include "cs_device.cuh"
#include "cs_internal.h"

namespace cg = cooperative_groups;

namespace cs {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kGroup = 8;     // consecutive logits a thread takes per step (one 16-byte bf16 vector)
constexpr int kBatch = 2;     // groups per row in flight per thread

struct AcceptParams {
    const void* target;       // [B, k+1, V]
    const void* draft;        // [B, k, V]
    const int32_t* tokens;    // [B, k]
    const float* uniforms;    // [B, k+1]
    int32_t* out_tokens;      // [B, k+1]
    int32_t* out_n;           // [B]
    int V, k, chunk;
    int b_base;               // first request of this launch (grids hold <= 65535 requests)
    float c_hi, c_lo;         // log2(e) / T as a float pair
};

// ------------------------------------------------------------ logit loads
__device__ __forceinline__ uint4 ld_stream(const void* p) {
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}

__device__ __forceinline__ float to_f(float v) { return v; }
__device__ __forceinline__ float to_f(__nv_bfloat16 v) { return __bfloat162float(v); }

// Eight consecutive logits row[start .. start+8) as fp32; entries at or past
// `end` read as -inf.  `vec` says the row base is 16-byte aligned.
__device__ __forceinline__ void load8(const __nv_bfloat16* row, int start, int end, bool vec,
                                      float (&v)[kGroup]) {
    if (vec && start + kGroup <= end) {
        const uint4 u = ld_stream(row + start);
        const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            v[2 * e] = bf16_bits_to_float(w[e] & 0xffffu);
            v[2 * e + 1] = bf16_bits_to_float(w[e] >> 16);
        }
    } else {
#pragma unroll
        for (int e = 0; e < kGroup; ++e)
            v[e] = start + e < end ? __bfloat162float(row[start + e]) : kNegInf;
    }
}

__device__ __forceinline__ void load8(const float* row, int start, int end, bool vec,
                                      float (&v)[kGroup]) {
    if (vec && start + kGroup <= end) {
        const uint4 a = ld_stream(row + start), b = ld_stream(row + start + 4);
        v[0] = __uint_as_float(a.x); v[1] = __uint_as_float(a.y);
        v[2] = __uint_as_float(a.z); v[3] = __uint_as_float(a.w);
        v[4] = __uint_as_float(b.x); v[5] = __uint_as_float(b.y);
        v[6] = __uint_as_float(b.z); v[7] = __uint_as_float(b.w);
    } else {
#pragma unroll
        for (int e = 0; e < kGroup; ++e) v[e] = start + e < end ? row[start + e] : kNegInf;
    }
}

template <typename T>
__device__ __forceinline__ bool aligned16(const T* p) {
    return (reinterpret_cast<uintptr_t>(p) & 15u) == 0;
}

// ------------------------------------------------------- (max, sum) algebra
// A pair (m, s) stands for sum_v 2^((z_v - m) c); empty is (-inf, 0).
__device__ __forceinline__ void fold(float& m, float& s, float m2, float s2, float c_hi, float c_lo) {
    const float M = fmaxf(m, m2);
    if (M == kNegInf) return;
    const float a = m == kNegInf ? 0.f : s * ex2_scaled(m - M, c_hi, c_lo);
    const float b = m2 == kNegInf ? 0.f : s2 * ex2_scaled(m2 - M, c_hi, c_lo);
    s = a + b;
    m = M;
}

template <int N>
__device__ __forceinline__ void running_update(float& m, float& s, const float (&v)[N][kGroup],
                                               float c) {
    float bm = kNegInf;
#pragma unroll
    for (int u = 0; u < N; ++u)
#pragma unroll
        for (int e = 0; e < kGroup; ++e) bm = fmaxf(bm, v[u][e]);
    if (bm > m) {
        s = m == kNegInf ? 0.f : s * ex2((m - bm) * c);
        m = bm;
    }
    if (m == kNegInf) return;
#pragma unroll
    for (int u = 0; u < N; ++u)
#pragma unroll
        for (int e = 0; e < kGroup; ++e) s += ex2((v[u][e] - m) * c);
}

// Per-thread statistics of this CTA's slice [c0, c1) of one or two rows.
template <typename T>
__device__ __forceinline__ void slice_stats(const T* rt, const T* rd, bool two, int c0, int c1,
                                            float c, float (&m)[2], float (&s)[2]) {
    m[0] = m[1] = kNegInf;
    s[0] = s[1] = 0.f;
    const int ng = c1 > c0 ? (c1 - c0 + kGroup - 1) / kGroup : 0;
    const bool vt = aligned16(rt), vd = two && aligned16(rd);
    for (int g0 = threadIdx.x; g0 < ng; g0 += kThreads * kBatch) {
        float at[kBatch][kGroup], ad[kBatch][kGroup];
#pragma unroll
        for (int u = 0; u < kBatch; ++u) {
            const int gi = g0 + u * kThreads;
            if (gi < ng) {
                load8(rt, c0 + gi * kGroup, c1, vt, at[u]);
                if (two) load8(rd, c0 + gi * kGroup, c1, vd, ad[u]);
            } else {
#pragma unroll
                for (int e = 0; e < kGroup; ++e) at[u][e] = ad[u][e] = kNegInf;
            }
        }
        running_update(m[0], s[0], at, c);
        if (two) running_update(m[1], s[1], ad, c);
    }
}

// Block reduction of per-thread (m, s) pairs for two rows, in a fixed order
// (xor butterflies within each warp, then across the warp results in warp 0).
// Thread 0 ends with the CTA's pairs.
__device__ __forceinline__ void block_fold2(float (&m)[2], float (&s)[2], float c_hi, float c_lo,
                                            float (*red)[4]) {
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
#pragma unroll
        for (int r = 0; r < 2; ++r) {
            const float m2 = __shfl_xor_sync(0xffffffffu, m[r], off);
            const float s2 = __shfl_xor_sync(0xffffffffu, s[r], off);
            fold(m[r], s[r], m2, s2, c_hi, c_lo);
        }
    }
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) {
        red[warp][0] = m[0];
        red[warp][1] = s[0];
        red[warp][2] = m[1];
        red[warp][3] = s[1];
    }
    __syncthreads();
    if (warp == 0) {
        const bool have = lane < kWarps;
        m[0] = have ? red[lane][0] : kNegInf;
        s[0] = have ? red[lane][1] : 0.f;
        m[1] = have ? red[lane][2] : kNegInf;
        s[1] = have ? red[lane][3] : 0.f;
#pragma unroll
        for (int off = kWarps / 2; off > 0; off >>= 1) {
#pragma unroll
            for (int r = 0; r < 2; ++r) {
                const float m2 = __shfl_xor_sync(0xffffffffu, m[r], off);
                const float s2 = __shfl_xor_sync(0xffffffffu, s[r], off);
                fold(m[r], s[r], m2, s2, c_hi, c_lo);
            }
        }
    }
}

// Cluster fold of the CTAs' (m, s) pairs for two rows: lane r of warp 0
// reads rank r's pairs from distributed shared memory, then an xor butterfly
// in a fixed order.  Every CTA folds the same values in the same order, so
// lane 0 of every CTA holds bit-identical results.  Warp 0 only.
__device__ __forceinline__ void cluster_fold2(cg::cluster_group& cl, const float* mine, int n_ranks,
                                              float c_hi, float c_lo, float (&M)[2], float (&S)[2]) {
    const int lane = threadIdx.x & 31;
    M[0] = M[1] = kNegInf;
    S[0] = S[1] = 0.f;
    if (lane < n_ranks) {
        const float4 v = *reinterpret_cast<const float4*>(cl.map_shared_rank(mine, lane));
        M[0] = v.x;
        S[0] = v.y;
        M[1] = v.z;
        S[1] = v.w;
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
#pragma unroll
        for (int r = 0; r < 2; ++r) {
            const float m2 = __shfl_xor_sync(0xffffffffu, M[r], off);
            const float s2 = __shfl_xor_sync(0xffffffffu, S[r], off);
            fold(M[r], S[r], m2, s2, c_hi, c_lo);
        }
    }
}

// Block-wide inclusive scan of one float per thread (fixed order).  Returns
// the inclusive prefix; `excl` gets the exclusive one, `total` the block sum.
__device__ __forceinline__ float block_scan(float x, float& excl, float& total, float* wsum) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    float inc = x;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
        const float y = __shfl_up_sync(0xffffffffu, inc, off);
        if (lane >= off) inc += y;
    }
    if (lane == 31) wsum[warp] = inc;
    __syncthreads();
    if (warp == 0) {
        float w = lane < kWarps ? wsum[lane] : 0.f;
        float wi = w;
#pragma unroll
        for (int off = 1; off < kWarps; off <<= 1) {
            const float y = __shfl_up_sync(0xffffffffu, wi, off);
            if (lane >= off) wi += y;
        }
        if (lane < kWarps) wsum[kWarps + lane] = wi - w;   // exclusive warp prefix
        if (lane == kWarps - 1) wsum[2 * kWarps] = wi;     // block total
    }
    __syncthreads();
    const float wp = wsum[kWarps + warp];
    const float incl = wp + inc;
    const float up = __shfl_up_sync(0xffffffffu, incl, 1);
    excl = lane == 0 ? wp : up;
    total = wsum[2 * kWarps];
    __syncthreads();   // wsum is reused by the next call
    return incl;
}

// Probability-scale weight of one logit: 2^((z - m) c) / S, zero for -inf.
__device__ __forceinline__ float weight(float z, float m, float inv_s, float c_hi, float c_lo) {
    return z == kNegInf ? 0.f : ex2_scaled(z - m, c_hi, c_lo) * inv_s;
}

struct DrawRow {
    float mt, inv_st, md, inv_sd;
    int residual;   // 1: max(0, p - q); 0: p only
};

// Scans this CTA's slice of the draw distribution in ascending token order.
// Without `search` it returns the slice mass.  With `search` it returns the
// first token whose running mass (starting from `base`) exceeds `t`, or the
// slice's last token of positive weight when rounding leaves none; -1 if the
// slice has no positive weight.
template <typename T>
__device__ float draw_scan(const T* rt, const T* rd, int c0, int c1, const DrawRow& w, float c_hi,
                           float c_lo, bool search, float base, float t, int* s_found,
                           float* wsum) {
    const int ng = c1 > c0 ? (c1 - c0 + kGroup - 1) / kGroup : 0;
    const bool vt = aligned16(rt), vd = w.residual && aligned16(rd);
    float run = base;
    int last_pos = -1;
    if (search && threadIdx.x == 0) *s_found = INT_MAX;
    __syncthreads();
    for (int g0 = 0; g0 < ng; g0 += kThreads) {
        const int gi = g0 + threadIdx.x;
        float r[kGroup];
        if (gi < ng) {
            float zt[kGroup], zd[kGroup];
            load8(rt, c0 + gi * kGroup, c1, vt, zt);
            if (w.residual) load8(rd, c0 + gi * kGroup, c1, vd, zd);
#pragma unroll
            for (int e = 0; e < kGroup; ++e) {
                const float pt = weight(zt[e], w.mt, w.inv_st, c_hi, c_lo);
                const float qd = w.residual ? weight(zd[e], w.md, w.inv_sd, c_hi, c_lo) : 0.f;
                r[e] = fmaxf(pt - qd, 0.f);
                if (r[e] > 0.f) last_pos = c0 + gi * kGroup + e;
            }
        } else {
#pragma unroll
            for (int e = 0; e < kGroup; ++e) r[e] = 0.f;
        }
        float sj = 0.f;
#pragma unroll
        for (int e = 0; e < kGroup; ++e) sj += r[e];
        float excl, total;
        const float incl = block_scan(sj, excl, total, wsum);
        if (search) {
            const bool cross = run + incl > t;
            if (cross) atomicMin(s_found, threadIdx.x);
            __syncthreads();
            const int owner = *s_found;
            if (owner != INT_MAX) {
                // the owner thread walks its eight weights; the result goes back
                // through s_found as a token id (>= 0) offset below INT_MIN/2
                __syncthreads();
                if (threadIdx.x == owner) {
                    float cum = run + excl;
                    int pick = -1, lastp = -1;
#pragma unroll
                    for (int e = 0; e < kGroup; ++e) {
                        cum += r[e];
                        if (r[e] > 0.f) lastp = c0 + gi * kGroup + e;
                        if (pick < 0 && cum > t) pick = c0 + gi * kGroup + e;
                    }
                    *s_found = INT_MIN + 1 + (pick >= 0 ? pick : lastp);
                }
                __syncthreads();
                const int res = *s_found - (INT_MIN + 1);
                __syncthreads();
                return (float)res;
            }
        }
        run += total;
    }
    if (!search) return run;
    // no crossing inside the slice: its last token of positive weight
    if (threadIdx.x == 0) *s_found = -1;
    __syncthreads();
    if (last_pos >= 0) atomicMax(s_found, last_pos);
    __syncthreads();
    const int res = *s_found;
    __syncthreads();
    return (float)res;
}

// ------------------------------------------------------------------ kernel
template <typename T, bool kGreedy>
__global__ void __launch_bounds__(kThreads) spec_accept_kernel(const AcceptParams p) {
    cg::cluster_group cl = cg::this_cluster();
    const int n_ranks = (int)cl.num_blocks();
    const int rank = (int)cl.block_rank();
    const int b = blockIdx.y + p.b_base;
    const int V = p.V, k = p.k;
    const int c0 = min(V, rank * p.chunk), c1 = min(V, c0 + p.chunk);
    const T* tgt = static_cast<const T*>(p.target) + (size_t)b * (k + 1) * V;
    const T* drf = kGreedy ? nullptr : static_cast<const T*>(p.draft) + (size_t)b * k * V;
    const int32_t* x = p.tokens + (size_t)b * k;
    const float* u = p.uniforms + (size_t)b * (k + 1);
    const float c_hi = p.c_hi, c_lo = p.c_lo;

    __shared__ __align__(16) float xch[2][4];   // this CTA's contribution to the current exchange
    __shared__ float red[kWarps][4];
    __shared__ float wsum[2 * kWarps + 1];
    __shared__ float bc[8];              // values broadcast by thread 0
    __shared__ int bci[4];
    __shared__ int s_found;
    int epoch = 0;

    if (kGreedy) {
        int a = k, emit = 0;
        for (int i = 0; i <= k; ++i) {
            const T* row = tgt + (size_t)i * V;
            const bool vec = aligned16(row);
            const int x_i = (threadIdx.x == 0 && i < k) ? __ldg(x + i) : -1;
            float best = kNegInf;
            int bi = INT_MAX;
            const int ng = c1 > c0 ? (c1 - c0 + kGroup - 1) / kGroup : 0;
            for (int g0 = threadIdx.x; g0 < ng; g0 += kThreads * kBatch) {
                float v[kBatch][kGroup];
#pragma unroll
                for (int uu = 0; uu < kBatch; ++uu) {
                    const int gi = g0 + uu * kThreads;
                    if (gi < ng) load8(row, c0 + gi * kGroup, c1, vec, v[uu]);
                }
#pragma unroll
                for (int uu = 0; uu < kBatch; ++uu) {
                    const int gi = g0 + uu * kThreads;
                    if (gi >= ng) continue;
#pragma unroll
                    for (int e = 0; e < kGroup; ++e)
                        if (v[uu][e] > best) {   // ascending ids: strict > keeps the lowest
                            best = v[uu][e];
                            bi = c0 + gi * kGroup + e;
                        }
                }
            }
            // block argmax, lowest id on ties
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) {
                const float b2 = __shfl_xor_sync(0xffffffffu, best, off);
                const int i2 = __shfl_xor_sync(0xffffffffu, bi, off);
                if (b2 > best || (b2 == best && i2 < bi)) {
                    best = b2;
                    bi = i2;
                }
            }
            if ((threadIdx.x & 31) == 0) {
                red[threadIdx.x >> 5][0] = best;
                red[threadIdx.x >> 5][1] = __int_as_float(bi);
            }
            __syncthreads();
            if (threadIdx.x < 32) {
                const int lane = threadIdx.x;
                best = lane < kWarps ? red[lane][0] : kNegInf;
                bi = lane < kWarps ? __float_as_int(red[lane][1]) : INT_MAX;
#pragma unroll
                for (int off = kWarps / 2; off > 0; off >>= 1) {
                    const float b2 = __shfl_xor_sync(0xffffffffu, best, off);
                    const int i2 = __shfl_xor_sync(0xffffffffu, bi, off);
                    if (b2 > best || (b2 == best && i2 < bi)) {
                        best = b2;
                        bi = i2;
                    }
                }
                if (lane == 0) {
                    xch[epoch & 1][0] = best;
                    xch[epoch & 1][1] = __int_as_float(bi);
                }
            }
            cl.sync();
            if (threadIdx.x < 32) {
                const int lane = threadIdx.x;
                float gb = kNegInf;
                int gidx = INT_MAX;
                if (lane < n_ranks) {
                    const float* rx = cl.map_shared_rank(&xch[epoch & 1][0], lane);
                    gb = rx[0];
                    gidx = __float_as_int(rx[1]);
                }
#pragma unroll
                for (int off = 16; off > 0; off >>= 1) {
                    const float b2 = __shfl_xor_sync(0xffffffffu, gb, off);
                    const int i2 = __shfl_xor_sync(0xffffffffu, gidx, off);
                    if (b2 > gb || (b2 == gb && i2 < gidx)) {
                        gb = b2;
                        gidx = i2;
                    }
                }
                if (lane == 0) {
                    if (gidx == INT_MAX) gidx = 0;   // a row with no finite entry
                    bci[0] = gidx;
                    bci[1] = (i == k || x_i != gidx) ? 1 : 0;
                }
            }
            __syncthreads();
            ++epoch;
            if (bci[1]) {
                a = i;
                emit = bci[0];
                break;
            }
            __syncthreads();
        }
        if (rank == 0 && threadIdx.x == 0) {
            int32_t* out = p.out_tokens + (size_t)b * (k + 1);
            for (int j = 0; j < a; ++j) out[j] = __ldg(x + j);
            out[a] = emit;
            for (int j = a + 1; j <= k; ++j) out[j] = -1;
            p.out_n[b] = a;
        }
        cl.sync();
        return;
    }

    // ----------------------------------------------------------- T > 0
    float mt = 0.f, St = 1.f, md = 0.f, Sd = 1.f;
    int a = k;
    for (int i = 0; i <= k; ++i) {
        const bool two = i < k;
        // thread 0 fetches what the accept test needs while the slice streams
        int xi = -1;
        float zt_x = 0.f, zd_x = 0.f, ui = 0.f;
        if (threadIdx.x == 0 && two) {
            xi = __ldg(x + i);
            ui = __ldg(u + i);
            if (xi >= 0 && xi < V) {
                zt_x = to_f(tgt[(size_t)i * V + xi]);
                zd_x = to_f(drf[(size_t)i * V + xi]);
            }
        }
        float m[2], s[2];
        slice_stats(tgt + (size_t)i * V, two ? drf + (size_t)i * V : tgt, two, c0, c1, c_hi, m, s);
        block_fold2(m, s, c_hi, c_lo, red);
        if (threadIdx.x == 0) {
            xch[epoch & 1][0] = m[0];
            xch[epoch & 1][1] = s[0];
            xch[epoch & 1][2] = m[1];
            xch[epoch & 1][3] = s[1];
        }
        cl.sync();
        if (threadIdx.x < 32) {
            float M[2], S[2];
            cluster_fold2(cl, &xch[epoch & 1][0], n_ranks, c_hi, c_lo, M, S);
            if (threadIdx.x == 0) {
                bc[0] = M[0];
                bc[1] = S[0];
                bc[2] = M[1];
                bc[3] = S[1];
                int reject = 0;
                if (two) {
                    if (xi < 0 || xi >= V || zt_x == kNegInf) {
                        reject = 1;
                    } else {
                        // log2 p(x)/q(x) = ((zt - mt) - (zd - md)) c + log2 Sd - log2 St,
                        // carried as an unevaluated float pair
                        const float dz = (zt_x - M[0]) - (zd_x - M[1]);
                        const float A = dz * c_hi;
                        float E = fmaf(dz, c_lo, fmaf(dz, c_hi, -A));
                        const float Bl = lg2(S[1]) - lg2(S[0]);
                        const float H = A + Bl;
                        const float bb = H - A;
                        E += (A - (H - bb)) + (Bl - bb);
                        const float ratio = ex2(H) * fmaf(E, kLn2, 1.f);
                        reject = !(ui < ratio);
                    }
                }
                bci[0] = reject;
            }
        }
        __syncthreads();
        ++epoch;
        mt = bc[0];
        St = bc[1];
        md = bc[2];
        Sd = bc[3];
        const int reject = bci[0];
        __syncthreads();
        if (i == k) break;
        if (reject) {
            a = i;
            break;
        }
    }

    // ------------------------------------------------------------ the draw
    const T* rt = tgt + (size_t)a * V;
    const T* rd = a < k ? drf + (size_t)a * V : tgt;
    DrawRow w{mt, 1.f / St, md, 1.f / Sd, a < k ? 1 : 0};
    int token = -1, owner = -1;
    for (int attempt = 0; attempt < 2; ++attempt) {
        const float mass = draw_scan(rt, rd, c0, c1, w, c_hi, c_lo, false, 0.f, 0.f, &s_found, wsum);
        if (threadIdx.x == 0) xch[epoch & 1][0] = mass;
        cl.sync();
        if (threadIdx.x < 32) {
            // lane r holds rank r's mass; an inclusive scan in a fixed order
            // gives every CTA the same cumulative masses
            const int lane = threadIdx.x;
            const float Mr = lane < n_ranks ? *cl.map_shared_rank(&xch[epoch & 1][0], lane) : 0.f;
            float incl = Mr;
#pragma unroll
            for (int off = 1; off < 32; off <<= 1) {
                const float y = __shfl_up_sync(0xffffffffu, incl, off);
                if (lane >= off) incl += y;
            }
            const float Z = __shfl_sync(0xffffffffu, incl, 31);
            const float excl = incl - Mr;   // only used as the owner's base (see below)
            const float up = __shfl_up_sync(0xffffffffu, incl, 1);
            const float base_l = lane == 0 ? 0.f : up;
            (void)excl;
            int retry = 0, own = -1;
            float base = 0.f, t = 0.f;
            if (!(Z > 0.f)) {
                retry = 1;   // p == q up to rounding: fall back to p of the same row
            } else {
                t = __ldg(u + k) * Z;
                const unsigned cross = __ballot_sync(0xffffffffu, lane < n_ranks && Mr > 0.f && incl > t);
                const unsigned pos = __ballot_sync(0xffffffffu, lane < n_ranks && Mr > 0.f);
                if (cross) {
                    own = __ffs(cross) - 1;
                    base = __shfl_sync(0xffffffffu, base_l, own);
                } else {   // u*Z at or past the total through rounding
                    own = 31 - __clz(pos);
                    base = 0.f;
                    t = __int_as_float(0x7f800000);
                }
            }
            if (lane == 0) {
                bci[0] = retry;
                bci[1] = own;
                bc[4] = base;
                bc[5] = t;
            }
        }
        __syncthreads();
        ++epoch;
        const int retry = bci[0];
        owner = bci[1];
        const float base = bc[4], t = bc[5];
        __syncthreads();
        if (retry && attempt == 0 && w.residual) {
            w.residual = 0;
            continue;
        }
        if (owner == rank) {
            token = (int)draw_scan(rt, rd, c0, c1, w, c_hi, c_lo, true, base, t, &s_found, wsum);
        }
        break;
    }
    if (threadIdx.x == 0) {
        int32_t* out = p.out_tokens + (size_t)b * (k + 1);
        if (owner == rank) out[a] = token >= 0 ? token : c0;
        if (rank == 0) {
            for (int j = 0; j < a; ++j) out[j] = __ldg(x + j);
            for (int j = a + 1; j <= k; ++j) out[j] = -1;
            p.out_n[b] = a;
            if (owner < 0) out[a] = 0;   // no positive weight anywhere (not a distribution)
        }
    }
    cl.sync();   // shared memory of every rank stays alive until all reads are done
}

int g_max_cluster[64] = {0};

int max_cluster_size(int dev) {
    if (dev < 0 || dev >= 64) return 8;
    if (g_max_cluster[dev]) return g_max_cluster[dev];
    int best = 8;
    auto kern = spec_accept_kernel<__nv_bfloat16, false>;
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) == cudaSuccess) {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(16, 1, 1);
        cfg.blockDim = dim3(kThreads, 1, 1);
        cudaLaunchAttribute attr;
        attr.id = cudaLaunchAttributeClusterDimension;
        attr.val.clusterDim.x = 16;
        attr.val.clusterDim.y = 1;
        attr.val.clusterDim.z = 1;
        cfg.attrs = &attr;
        cfg.numAttrs = 1;
        int n = 0;
        if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) == cudaSuccess && n > 0) best = 16;
    }
    cudaGetLastError();
    g_max_cluster[dev] = best;
    return best;
}

template <typename T, bool G>
cs_status launch_typed(AcceptParams p, int cluster, int batch, cudaStream_t stream) {
    auto kern = spec_accept_kernel<T, G>;
    if (cluster > 8) {
        static bool done[64] = {};
        int dev = 0;
        cudaGetDevice(&dev);
        if (dev < 0 || dev >= 64 || !done[dev]) {
            const cudaError_t e =
                cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
            if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute(non-portable cluster)");
            if (dev >= 0 && dev < 64) done[dev] = true;
        }
    }
    for (int b0 = 0; b0 < batch; b0 += 65535) {
        p.b_base = b0;
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(cluster, batch - b0 < 65535 ? batch - b0 : 65535, 1);
        cfg.blockDim = dim3(kThreads, 1, 1);
        cfg.dynamicSmemBytes = 0;
        cfg.stream = stream;
        cudaLaunchAttribute attr;
        attr.id = cudaLaunchAttributeClusterDimension;
        attr.val.clusterDim.x = cluster;
        attr.val.clusterDim.y = 1;
        attr.val.clusterDim.z = 1;
        cfg.attrs = &attr;
        cfg.numAttrs = 1;
        const cudaError_t e = cudaLaunchKernelEx(&cfg, kern, p);
        if (e != cudaSuccess) return cuda_fail(e, "spec_accept_kernel launch");
    }
    return CS_OK;
}

}  // namespace

cs_status launch_spec_accept(const cs_accept_dims& d, const void* target, const void* draft,
                             const int32_t* tokens, const float* uniforms, int n_draft,
                             float temperature, int32_t* out_tokens, int32_t* out_n,
                             cudaStream_t stream) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    const int sms = current_sm_count();
    // Enough CTAs to cover the SMs several times over, at least ~2K logits per
    // CTA, at most the largest cluster the device schedules.
    const int want = (4 * sms + d.batch - 1) / d.batch;
    int cluster = 1;
    while (cluster < want && cluster < 16) cluster <<= 1;
    int by_vocab = 1;
    while (by_vocab * 2 <= d.vocab / 2048 && by_vocab < 16) by_vocab <<= 1;
    if (cluster > by_vocab) cluster = by_vocab;
    const int cmax = max_cluster_size(dev);
    if (cluster > cmax) cluster = cmax;

    AcceptParams p{};
    p.target = target;
    p.draft = draft;
    p.tokens = tokens;
    p.uniforms = uniforms;
    p.out_tokens = out_tokens;
    p.out_n = out_n;
    p.V = d.vocab;
    p.k = n_draft;
    const int per = (d.vocab + cluster - 1) / cluster;
    p.chunk = (per + kGroup - 1) / kGroup * kGroup;
    const double c = temperature > 0.f ? 1.4426950408889634 / (double)temperature : 0.0;
    p.c_hi = (float)c;
    p.c_lo = (float)(c - (double)p.c_hi);
    const bool greedy = temperature == 0.f;
    if (d.logit_dtype == CS_F32)
        return greedy ? launch_typed<float, true>(p, cluster, d.batch, stream)
                      : launch_typed<float, false>(p, cluster, d.batch, stream);
    return greedy ? launch_typed<__nv_bfloat16, true>(p, cluster, d.batch, stream)
                  : launch_typed<__nv_bfloat16, false>(p, cluster, d.batch, stream);
}

}  // namespace cs
