// route.cu -- batched semantic routing of the paper's front end (Sec. 3.1):
// the score of request x against group G_i is the cosine similarity of its
// embedding with the group's centroid, the request goes to the best group
// i* = argmax_i S (lowest i on ties), or to the cache-miss branch when
// S(x, G_i*) < tau.
//
// The scores are one GEMM, E C^T, with the arg max fused into its epilogue
// (the B x N score matrix never reaches memory):
//   route_gemm_kernel: a CTA owns 128 requests (MMA M) and a contiguous range
//     of 128-group tiles.  Warp 0 loads the CTA's embedding rows once (one TMA
//     box per 64-dim chunk, 128-byte swizzle, kept in shared memory) and
//     streams the centroid chunks through a 6-slot TMA ring; warp 1 issues
//     tcgen05.mma from one thread (M = 128, N = 128, K = 16 per instruction,
//     fp32 accumulators in tensor memory, two buffers); warps 4-7 take one
//     row each per thread, scale each dot product by the centroid's inverse
//     norm and keep the running maximum and its lowest index.
//   route_merge_kernel: one warp per request folds the CTAs' partials (score
//     first, then lower index), applies the request's own inverse norm and
//     the threshold.
//   route_norms_kernel: inverse L2 norms of the centroids (the group index
//     changes slowly, so this runs when it changes, not per batch).
#include <cudaTypedefs.h>

#include "cs_device.cuh"
#include "cs_internal.h"

namespace cs {
namespace {

constexpr int kRM = 128;                  // requests per tile (MMA M)
constexpr int kRN = 128;                  // groups per tile (MMA N)
constexpr int kKC = 64;                   // dims per chunk: one 128-byte swizzle row
constexpr int kChunkBytes = kRM * 128;    // 128 rows x 64 dims x 2 B
constexpr int kMaxSlots = 12;             // centroid-chunk ring, at most
constexpr int kRThreads = 256;            // warp 0 TMA, warp 1 MMA, warp 2 TMEM, warps 4-7 epilogue
constexpr int kRTmemCols = 2 * kRN;
constexpr int kRBarBytes = 256;
constexpr int kRStaticSmem = 2 * kRN * 4 + 64;   // inverse-norm double buffer, TMEM address
constexpr int kRSmemLimit = 232448;              // opt-in shared memory per block on sm_103a

__host__ __device__ constexpr int route_slots(int n_chunks) {
    return (kRSmemLimit - kRStaticSmem - 1024 - kRBarBytes - n_chunks * kChunkBytes) / kChunkBytes < kMaxSlots
               ? (kRSmemLimit - kRStaticSmem - 1024 - kRBarBytes - n_chunks * kChunkBytes) / kChunkBytes
               : kMaxSlots;
}
__host__ __device__ constexpr int route_smem_bytes(int n_chunks) {
    return 1024 + n_chunks * kChunkBytes + route_slots(n_chunks) * kChunkBytes + kRBarBytes;
}
static_assert(route_slots(kMaxRouteDim / kKC) >= 6, "ring too shallow for the widest embedding");

struct RouteParams {
    int B, N, d, n_chunks, n_tiles, slots, grid, seg_slots;
    long long items;              // m_tiles * n_tiles work items, split evenly over the grid
    const float* inv_norm_c;      // [N]
    float2* part;                 // [m_tiles, seg_slots, 128]: (max of dot * inv_norm_c, index as int bits)
    int* status;
};

// The CTA whose item range holds item x: ranges are [c*I/G, (c+1)*I/G).
__host__ __device__ __forceinline__ int route_owner(long long x, long long items, int grid) {
    return (int)(((x + 1) * grid + items - 1) / items) - 1;
}

__host__ __device__ constexpr uint32_t route_idesc() {
    // kind::f16: bf16 A and B (both K-major), fp32 D, M = 128, N = 128
    return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(kRN >> 3) << 17) | ((uint32_t)(kRM >> 4) << 24);
}

__device__ __forceinline__ uint64_t sw128_desc(uint32_t addr) {
    // 128-byte swizzle, K-major: 8-row groups 1024 bytes apart
    return (uint64_t)((addr >> 4) & 0x3FFF) | ((uint64_t)1 << 16) | ((uint64_t)(1024 >> 4) << 32) |
           (1ull << 46) | (2ull << 61);
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, uint64_t* bar, int c0, int c1) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(smem_u32(bar))
        : "memory");
}

__device__ __forceinline__ bool mbar_test(uint64_t* bar, uint32_t parity) {
    uint32_t done;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}\n"
        : "=r"(done)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return done != 0;
}

// Spins (no suspend) on the phase; about one second at most, then records
// the timeout in the status word and returns false.
__device__ __forceinline__ bool wait_bar(uint64_t* bar, uint32_t parity, int* status) {
    if (mbar_test(bar, parity)) return true;
    const uint64_t t0 = global_timer_ns();
    for (uint32_t it = 0; it < (1u << 28); ++it) {
        if (mbar_test(bar, parity)) return true;
        if ((it & 1023u) == 1023u && global_timer_ns() - t0 > 1000000000ull) break;
    }
    atomicOr(status, CS_DEVICE_WAIT_TIMEOUT);
    return false;
}

__device__ __forceinline__ void umma_commit(uint64_t* bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(bar))
                 : "memory");
}

__device__ __forceinline__ void epi_bar_sync() { asm volatile("bar.sync 1, 128;" ::: "memory"); }

// Persistent: CTA c owns the work items [c*I/G, (c+1)*I/G) of the m-major
// sequence (request tile m, group tile t).  The request tile stays resident
// in shared memory while t advances and is reloaded when m changes.
__global__ void __launch_bounds__(kRThreads, 1)
route_gemm_kernel(const __grid_constant__ CUtensorMap tmap_e, const __grid_constant__ CUtensorMap tmap_c,
                  const RouteParams p) {
    extern __shared__ uint8_t smem_raw[];
    __shared__ __align__(16) float s_inv[2 * kRN];
    __shared__ uint32_t s_tmem;
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int slots = p.slots;
    uint8_t* sa = smem;                                   // [n_chunks][128 rows][128 B]
    uint8_t* sb = smem + p.n_chunks * kChunkBytes;        // [slots][128 groups][128 B]
    uint64_t* bars = reinterpret_cast<uint64_t*>(sb + slots * kChunkBytes);
    uint64_t* a_full = bars;
    uint64_t* a_free = bars + 1;
    uint64_t* d_full = bars + 2;             // [2]
    uint64_t* d_free = bars + 4;             // [2]
    uint64_t* mma_done = bars + 6;
    uint64_t* full = bars + 7;               // [slots]
    uint64_t* empty = full + kMaxSlots;      // [slots]

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const long long it0 = (long long)blockIdx.x * p.items / p.grid;
    const long long it1 = (long long)(blockIdx.x + 1) * p.items / p.grid;
    const int nt = (int)(it1 - it0);
    if (warp == 2) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&s_tmem)),
                     "n"(kRTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    if (threadIdx.x == 0) {
        mbar_init(a_full, 1);
        mbar_init(a_free, 1);
        for (int i = 0; i < 2; ++i) {
            mbar_init(&d_full[i], 1);
            mbar_init(&d_free[i], 4);
        }
        mbar_init(mma_done, 1);
        for (int i = 0; i < slots; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], 1);
        }
        fence_barrier_init();
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tmem = s_tmem;

    if (warp == 0 && lane == 0) {
        // ---------------------------------------------------------- TMA
        tma_prefetch_desc(&tmap_e);
        tma_prefetch_desc(&tmap_c);
        int s = 0, cur_m = -1;
        uint32_t use = 0, a_loads = 0;
        bool ok = true;
        for (long long it = it0; it < it1 && ok; ++it) {
            const int m = (int)(it / p.n_tiles), t = (int)(it - (long long)m * p.n_tiles);
            if (m != cur_m) {
                if (a_loads > 0 && !wait_bar(a_free, (a_loads - 1) & 1, p.status)) break;
                mbar_arrive_expect_tx(a_full, (uint32_t)(p.n_chunks * kChunkBytes));
                for (int kc = 0; kc < p.n_chunks; ++kc)
                    tma_load_2d(smem_u32(sa + kc * kChunkBytes), &tmap_e, a_full, kc * kKC, m * kRM);
                ++a_loads;
                cur_m = m;
            }
            for (int kc = 0; kc < p.n_chunks; ++kc) {
                if (use > 0 && !wait_bar(&empty[s], (use - 1) & 1, p.status)) {
                    ok = false;
                    break;
                }
                mbar_arrive_expect_tx(&full[s], (uint32_t)kChunkBytes);
                tma_load_2d(smem_u32(sb + s * kChunkBytes), &tmap_c, &full[s], kc * kKC, t * kRN);
                if (++s == slots) {
                    s = 0;
                    ++use;
                }
            }
        }
        // no copy in flight at exit: the last fill of every slot and the last
        // request tile have landed
        const long long total = (long long)nt * p.n_chunks;
        for (long long f = total > slots ? total - slots : 0; f < total; ++f)
            if (!mbar_wait_bounded(&full[f % slots], (uint32_t)(f / slots) & 1))
                atomicOr(p.status, CS_DEVICE_WAIT_TIMEOUT);
        if (a_loads > 0 && !mbar_wait_bounded(a_full, (a_loads - 1) & 1)) atomicOr(p.status, CS_DEVICE_WAIT_TIMEOUT);
    } else if (warp == 1 && lane == 0) {
        // ---------------------------------------------------------- MMA
        int s = 0, cur_m = -1;
        uint32_t use = 0, a_loads = 0;
        bool ok = true;
        for (int tl = 0; tl < nt && ok; ++tl) {
            const int m = (int)((it0 + tl) / p.n_tiles);
            if (m != cur_m) {
                if (a_loads > 0) umma_commit(a_free);   // the previous request tile may be overwritten
                if (!wait_bar(a_full, a_loads & 1, p.status)) break;
                ++a_loads;
                cur_m = m;
            }
            const int db = tl & 1;
            if (tl >= 2 && !wait_bar(&d_free[db], (uint32_t)((tl >> 1) - 1) & 1, p.status)) break;
            for (int kc = 0; kc < p.n_chunks; ++kc) {
                if (!wait_bar(&full[s], use & 1, p.status)) {
                    ok = false;
                    break;
                }
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                const uint32_t a0 = smem_u32(sa + kc * kChunkBytes), b0 = smem_u32(sb + s * kChunkBytes);
#pragma unroll
                for (int ks = 0; ks < kKC / 16; ++ks) {
                    const uint32_t acc = (kc > 0 || ks > 0) ? 1u : 0u;
                    asm volatile(
                        "{\n\t.reg .pred q;\n\tsetp.ne.b32 q, %4, 0;\n\t"
                        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, q;\n\t}\n" ::"r"(tmem + db * kRN),
                        "l"(sw128_desc(a0 + ks * 32)), "l"(sw128_desc(b0 + ks * 32)), "r"(route_idesc()), "r"(acc)
                        : "memory");
                }
                umma_commit(&empty[s]);
                if (++s == slots) {
                    s = 0;
                    ++use;
                }
            }
            if (ok) umma_commit(&d_full[db]);
        }
        umma_commit(mma_done);
        if (!mbar_wait_bounded(mma_done, 0)) atomicOr(p.status, CS_DEVICE_WAIT_TIMEOUT);
    } else if (warp >= 4) {
        // ------------------------------------------------------ epilogue
        const int sub = warp & 3;
        const int row = sub * 32 + lane;
        const uint32_t t_lane = tmem + ((uint32_t)(sub * 32) << 16);
        const float kNaN = __int_as_float(0x7fffffff);   // excluded by fmaxf and by ==
        auto inv_of = [&](long long it) {
            const int t = (int)(it % p.n_tiles);
            const int j = t * kRN + row;
            return j < p.N ? __ldg(p.inv_norm_c + j) : kNaN;
        };
        auto flush = [&](int m, float best, int idx) {
            const int b = m * kRM + row;
            if (b < p.B) {
                const int slot = blockIdx.x - route_owner((long long)m * p.n_tiles, p.items, p.grid);
                p.part[((size_t)m * p.seg_slots + slot) * kRM + row] = make_float2(best, __int_as_float(idx));
            }
        };
        float inv_next = nt > 0 ? inv_of(it0) : 0.f;
        float best = kNegInf;
        int idx = -1, cur_m = nt > 0 ? (int)(it0 / p.n_tiles) : -1;
        bool dead = false;
        for (int tl = 0; tl < nt; ++tl) {
            const long long it = it0 + tl;
            const int m = (int)(it / p.n_tiles), t = (int)(it - (long long)m * p.n_tiles);
            if (m != cur_m) {
                flush(cur_m, best, idx);
                best = kNegInf;
                idx = -1;
                cur_m = m;
            }
            const int db = tl & 1;
            s_inv[db * kRN + row] = inv_next;
            epi_bar_sync();
            if (tl + 1 < nt) inv_next = inv_of(it + 1);
            // after a timed-out wait the warp keeps taking part in the named
            // barrier (every epilogue warp passes it nt times) but skips the rest
            int ok = 0;
            if (lane == 0 && !dead) ok = wait_bar(&d_full[db], (uint32_t)(tl >> 1) & 1, p.status) ? 1 : 0;
            ok = __shfl_sync(0xffffffffu, ok, 0);
            if (!ok) {
                dead = true;
                continue;
            }
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
#pragma unroll 1
            for (int c0 = 0; c0 < kRN; c0 += 32) {
                uint32_t r[32];
                asm volatile(
                    "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
                    "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
                    : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
                      "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
                      "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]),
                      "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]),
                      "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
                    : "r"(t_lane + db * kRN + c0));
                asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
                const float4* sv = reinterpret_cast<const float4*>(s_inv + db * kRN + c0);
                float sc[32];
                float mx = kNegInf;
#pragma unroll
                for (int q4 = 0; q4 < 8; ++q4) {
                    const float4 v = sv[q4];
                    sc[4 * q4 + 0] = __uint_as_float(r[4 * q4 + 0]) * v.x;
                    sc[4 * q4 + 1] = __uint_as_float(r[4 * q4 + 1]) * v.y;
                    sc[4 * q4 + 2] = __uint_as_float(r[4 * q4 + 2]) * v.z;
                    sc[4 * q4 + 3] = __uint_as_float(r[4 * q4 + 3]) * v.w;
                    mx = fmaxf(mx, fmaxf(fmaxf(sc[4 * q4], sc[4 * q4 + 1]), fmaxf(sc[4 * q4 + 2], sc[4 * q4 + 3])));
                }
                // ascending group ids and a strict > across chunks keep the
                // lowest id of the maximum; inside the chunk, its first hit
                if (mx > best) {
                    int e0 = 31;
#pragma unroll
                    for (int e = 31; e >= 0; --e)
                        if (sc[e] == mx) e0 = e;
                    best = mx;
                    idx = t * kRN + c0 + e0;
                }
            }
            asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
            __syncwarp();
            if (lane == 0) mbar_arrive(&d_free[db]);
        }
        if (cur_m >= 0) flush(cur_m, best, idx);
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    if (warp == 2)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "n"(kRTmemCols) : "memory");
}

// One warp per request: fold the partials of the CTAs that covered its
// request tile (higher score, then lower index), scale by the request's own
// inverse norm, apply the threshold.
__global__ void __launch_bounds__(256) route_merge_kernel(const __nv_bfloat16* emb, const float2* part, int B, int d,
                                                           int n_tiles, long long items, int grid, int seg_slots,
                                                           float tau, int32_t* out_group, int32_t* out_best,
                                                           float* out_score) {
    const int b = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
    if (b >= B) return;
    float ss = 0.f;
    for (int k = lane; k < d; k += 32) {
        const float e = __bfloat162float(emb[(size_t)b * d + k]);
        ss = fmaf(e, e, ss);
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, off);
    float best = kNegInf;
    int idx = -1;
    if (n_tiles > 0) {
        const int m = b / kRM;
        const int n_seg = route_owner((long long)(m + 1) * n_tiles - 1, items, grid) -
                          route_owner((long long)m * n_tiles, items, grid) + 1;
        for (int j = lane; j < n_seg; j += 32) {
            const float2 v = part[((size_t)m * seg_slots + j) * kRM + (b % kRM)];
            const int vi = __float_as_int(v.y);
            if (vi >= 0 && (idx < 0 || v.x > best || (v.x == best && vi < idx))) {
                best = v.x;
                idx = vi;
            }
        }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
        const float ob = __shfl_xor_sync(0xffffffffu, best, off);
        const int oi = __shfl_xor_sync(0xffffffffu, idx, off);
        if (oi >= 0 && (idx < 0 || ob > best || (ob == best && oi < idx))) {
            best = ob;
            idx = oi;
        }
    }
    if (lane == 0) {
        const float inv_e = ss > 0.f ? rsqrtf(ss) : 0.f;
        const float score = idx >= 0 ? best * inv_e : kNegInf;
        out_best[b] = idx;
        out_score[b] = score;
        out_group[b] = (idx >= 0 && score >= tau) ? idx : -1;
    }
}

// One warp per centroid: 1 / |c_i| (0 for a zero vector).
__global__ void __launch_bounds__(256) route_norms_kernel(const __nv_bfloat16* c, int N, int d, float* inv_norm) {
    const int i = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
    if (i >= N) return;
    float ss = 0.f;
    for (int k = lane; k < d; k += 32) {
        const float x = __bfloat162float(c[(size_t)i * d + k]);
        ss = fmaf(x, x, ss);
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, off);
    if (lane == 0) inv_norm[i] = ss > 0.f ? rsqrtf(ss) : 0.f;
}

PFN_cuTensorMapEncodeTiled_v12000 route_encoder() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    if (!fn) {
        void* ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
    }
    return fn;
}

// [rows, d] bf16 row-major as (d, rows); box {64, 128}, 128-byte swizzle.
cs_status encode_rows_map(CUtensorMap* map, const void* base, int rows, int d) {
    auto enc = route_encoder();
    if (!enc) return fail(CS_ERR_CUDA, "cuTensorMapEncodeTiled is not available from the driver");
    const cuuint64_t dims[2] = {(cuuint64_t)d, (cuuint64_t)(rows > 0 ? rows : 1)};
    const cuuint64_t strides[1] = {(cuuint64_t)d * 2};
    const cuuint32_t box[2] = {kKC, kRM};
    const cuuint32_t estr[2] = {1, 1};
    const CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
                           estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                           CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(CS_ERR_CUDA, "cuTensorMapEncodeTiled(route) failed (CUresult %d)", (int)r);
    return CS_OK;
}

}  // namespace

RoutePlan plan_route(const cs_route_dims& d, int sm_count) {
    RoutePlan pl{};
    pl.m_tiles = (d.batch + kRM - 1) / kRM;
    pl.n_tiles = (d.n_groups + kRN - 1) / kRN;
    pl.items = (long long)pl.m_tiles * pl.n_tiles;
    const int sms = sm_count > 0 ? sm_count : 148;
    pl.grid = (int)(pl.items < sms ? pl.items : sms);
    // CTAs covering one request tile: its n_tiles items meet at most
    // floor((n_tiles - 1) * G / I) + 2 of the G ranges
    pl.seg_slots = pl.items > 0 ? (int)(((long long)(pl.n_tiles - 1) * pl.grid) / pl.items) + 2 : 0;
    pl.bytes = 256 + ((size_t)pl.m_tiles * pl.seg_slots * kRM * sizeof(float2) + 255) / 256 * 256;
    return pl;
}

cs_status launch_route(const cs_route_dims& d, const RoutePlan& pl, const void* emb, const void* centroids,
                       const float* inv_norms, float tau, int32_t* out_group, int32_t* out_best,
                       float* out_score, void* workspace, cudaStream_t stream) {
    uint8_t* ws = static_cast<uint8_t*>(workspace);
    cudaError_t e;
    if (pl.grid > 0) {
        CUtensorMap te, tc;
        cs_status st = encode_rows_map(&te, emb, d.batch, d.dim);
        if (st != CS_OK) return st;
        st = encode_rows_map(&tc, centroids, d.n_groups, d.dim);
        if (st != CS_OK) return st;
        const int n_chunks = d.dim / kKC;
        const int smem = route_smem_bytes(n_chunks);
        static int attr_smem[64] = {};
        int dev = 0;
        cudaGetDevice(&dev);
        if (dev < 0 || dev >= 64 || attr_smem[dev] < smem) {
            e = cudaFuncSetAttribute(route_gemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
            if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute(route_gemm_kernel)");
            if (dev >= 0 && dev < 64) attr_smem[dev] = smem;
        }
        RouteParams p{};
        p.B = d.batch;
        p.N = d.n_groups;
        p.d = d.dim;
        p.n_chunks = n_chunks;
        p.n_tiles = pl.n_tiles;
        p.slots = route_slots(n_chunks);
        p.grid = pl.grid;
        p.seg_slots = pl.seg_slots;
        p.items = pl.items;
        p.inv_norm_c = inv_norms;
        p.status = reinterpret_cast<int*>(ws);
        p.part = reinterpret_cast<float2*>(ws + 256);
        route_gemm_kernel<<<pl.grid, kRThreads, smem, stream>>>(te, tc, p);
        e = cudaGetLastError();
        if (e != cudaSuccess) return cuda_fail(e, "route_gemm_kernel launch");
    }
    route_merge_kernel<<<(d.batch + 7) / 8, 256, 0, stream>>>(
        static_cast<const __nv_bfloat16*>(emb), reinterpret_cast<const float2*>(ws + 256), d.batch, d.dim,
        pl.n_tiles, pl.items, pl.grid, pl.seg_slots, tau, out_group, out_best, out_score);
    e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_fail(e, "route_merge_kernel launch");
    return CS_OK;
}

cs_status launch_route_norms(int n_groups, int dim, const void* centroids, float* inv_norms, cudaStream_t stream) {
    route_norms_kernel<<<(n_groups + 7) / 8, 256, 0, stream>>>(static_cast<const __nv_bfloat16*>(centroids),
                                                               n_groups, dim, inv_norms);
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_fail(e, "route_norms_kernel launch");
    return CS_OK;
}

}  // namespace cs
