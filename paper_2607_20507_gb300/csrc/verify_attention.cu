// verify_attention.cu -- multi-query GQA verify attention over a paged KV
// cache (the KV-bound core of the target's verify pass in the paper's
// draft-and-verify step, Sec. 3.4).
//
// Work decomposition (flash-decoding style split-KV):
//   one CTA = (request b, KV head h, split s) over keys [s*C, min((s+1)*C, L_b)).
//   The (k+1)*G query rows that read KV head h (draft row i = r / G, query
//   head h*G + r % G) are packed into one tile, 16 rows per consumer warp, so
//   every K/V byte staged in shared memory serves all of them.
// Pipeline: one producer warp streams 64-token K and V tiles of the pages
//   through TMA (128-byte swizzle) into a 3-stage shared-memory ring guarded
//   by mbarriers; consumer warps run S = Q K^T and O += P V on bf16 tensor
//   cores (mma.sync m16n8k16, fp32 accumulate) with an fp32 online softmax in
//   the log2 domain.
// Splits: a request whose context needs one split writes bf16 output
//   directly; otherwise every split writes (O, m, l) partials to the
//   workspace and the last CTA to finish (an atomic ticket that wraps back
//   to zero, no spin-wait) merges them with log-sum-exp weights.
#include <math.h>
#include <stdio.h>

#include <cudaTypedefs.h>

#include "cs_device.cuh"
#include "cs_internal.h"

namespace cs {
namespace {

constexpr int kD = 128;                       // head dim implemented
constexpr int kTileT = 64;                    // keys per pipeline tile
constexpr int kHalfBytes = kTileT * 128;      // 64 keys x 64 dims x 2 B (one swizzle half)
constexpr int kTensorTileBytes = 2 * kHalfBytes;
constexpr int kStageBytes = 2 * kTensorTileBytes;   // K + V
constexpr int kStages = 3;
constexpr int kMaxRowWarps = 9;               // 144 query rows
constexpr int kSmemBytes = kStages * kStageBytes + 1024 /*align*/ + 128 /*barriers*/;

struct AttnParams {
    const __nv_bfloat16* q;      // [B, R, Hq, D]
    __nv_bfloat16* out;          // [B, R, Hq, D]
    const int32_t* page_table;   // [B, max_pages]
    const int32_t* ctx_lens;     // [B]
    float* part_o;               // [B, Hkv, ns_max, n_rows, D]
    float2* part_ml;             // [B, Hkv, ns_max, n_rows]  (m in log2 units, l)
    unsigned int* tickets;       // [B, Hkv]
    int* status;
    int Hq, Hkv, G, R, n_rows, ps, box_t, max_pages, chunk, ns_max, row_warps;
    int b_base;                  // first request of this launch (grids hold <= 65535 requests)
    float scale_log2;            // sm_scale * log2(e)
};

__device__ __forceinline__ void flag_timeout(int* status) {
    atomicOr(status, CS_DEVICE_WAIT_TIMEOUT);
}

__global__ void __launch_bounds__((kMaxRowWarps + 1) * 32, 1)
verify_attention_kernel(const __grid_constant__ CUtensorMap tmap_k,
                        const __grid_constant__ CUtensorMap tmap_v, const AttnParams p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + kStages * kStageBytes);
    uint64_t* empty = full + kStages;
    __shared__ int s_last;
    __shared__ int s_abort;

    const int split = blockIdx.x, h = blockIdx.y, b = blockIdx.z + p.b_base;
    int L = __ldg(p.ctx_lens + b);
    L = max(0, min(L, p.max_pages * p.ps));
    const int ns = max(1, (L + p.chunk - 1) / p.chunk);
    if (split >= ns) return;
    const int t_begin = split * p.chunk;
    const int t_end = min(L, t_begin + p.chunk);
    const int n_tiles = t_end > t_begin ? (t_end - t_begin + kTileT - 1) / kTileT : 0;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nw = p.row_warps;

    if (threadIdx.x == 0) {
        for (int i = 0; i < kStages; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], nw);
        }
        s_abort = 0;
        fence_barrier_init();
    }
    __syncthreads();

    const uint32_t smem_base = smem_u32(smem);

    if (warp == nw) {
        // ------------------------------------------------------ producer
        if (lane == 0 && n_tiles > 0) {
            tma_prefetch_desc(&tmap_k);
            tma_prefetch_desc(&tmap_v);
            const int pieces = kTileT / p.box_t;
            const uint32_t piece_bytes = (uint32_t)p.box_t * 128u;
            const int32_t* table = p.page_table + (size_t)b * p.max_pages;
            for (int t = 0; t < n_tiles; ++t) {
                const int st = t % kStages;
                const uint32_t use = (uint32_t)(t / kStages);
                if (t >= kStages && !mbar_wait_bounded(&empty[st], (use - 1) & 1)) {
                    flag_timeout(p.status);
                    s_abort = 1;
                    break;
                }
                const int ts = t_begin + t * kTileT;
                int valid = 0;
                for (int pc = 0; pc < pieces; ++pc)
                    if (ts + pc * p.box_t < t_end) ++valid;
                mbar_arrive_expect_tx(&full[st], (uint32_t)valid * piece_bytes * 4u);
                const uint32_t kdst = smem_base + st * kStageBytes;
                const uint32_t vdst = kdst + kTensorTileBytes;
                for (int pc = 0; pc < valid; ++pc) {
                    const int tok = ts + pc * p.box_t;
                    const int page = __ldg(table + tok / p.ps);
                    const int slot = tok % p.ps;
                    const uint32_t off = (uint32_t)pc * piece_bytes;
#pragma unroll
                    for (int hh = 0; hh < 2; ++hh) {
                        tma_load_4d(kdst + hh * kHalfBytes + off, &tmap_k, &full[st], hh * 64, slot,
                                    h, page);
                        tma_load_4d(vdst + hh * kHalfBytes + off, &tmap_v, &full[st], hh * 64, slot,
                                    h, page);
                    }
                }
            }
        }
    } else {
        // ------------------------------------------------------ consumers
        const int g = lane >> 2, tq = lane & 3;
        const int row0 = warp * 16 + g, row1 = row0 + 8;
        // Q fragments (A operand, 16 rows x 128 dims) straight from global memory.
        uint32_t qa[8][4];
        {
            const __nv_bfloat16* qr[2] = {nullptr, nullptr};
            const int rr[2] = {row0, row1};
#pragma unroll
            for (int k = 0; k < 2; ++k) {
                if (rr[k] < p.n_rows) {
                    const int i = rr[k] / p.G, gi = rr[k] % p.G;
                    qr[k] = p.q + (((size_t)b * p.R + i) * p.Hq + (size_t)h * p.G + gi) * kD;
                }
            }
#pragma unroll
            for (int kk = 0; kk < 8; ++kk) {
                const int c = kk * 16 + tq * 2;
                qa[kk][0] = qr[0] ? __ldg(reinterpret_cast<const uint32_t*>(qr[0] + c)) : 0u;
                qa[kk][1] = qr[1] ? __ldg(reinterpret_cast<const uint32_t*>(qr[1] + c)) : 0u;
                qa[kk][2] = qr[0] ? __ldg(reinterpret_cast<const uint32_t*>(qr[0] + c + 8)) : 0u;
                qa[kk][3] = qr[1] ? __ldg(reinterpret_cast<const uint32_t*>(qr[1] + c + 8)) : 0u;
            }
        }
        // exclusive key limit of each of this thread's two rows
        const int lim0 = row0 < p.n_rows ? min(t_end, L - p.R + 1 + row0 / p.G) : t_end;
        const int lim1 = row1 < p.n_rows ? min(t_end, L - p.R + 1 + row1 / p.G) : t_end;
        const int lim_min = min(lim0, lim1);
        const float c = p.scale_log2;

        float o[16][4];
#pragma unroll
        for (int i = 0; i < 16; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
        float m_raw[2] = {kNegInf, kNegInf};
        float l[2] = {0.f, 0.f};

        // per-lane ldmatrix address pieces: matrix index and row within it
        const int lm = lane >> 3, lr = lane & 7;

        for (int t = 0; t < n_tiles; ++t) {
            const int st = t % kStages;
            const uint32_t use = (uint32_t)(t / kStages);
            if (!mbar_wait_bounded(&full[st], use & 1)) {
                flag_timeout(p.status);
                s_abort = 1;
                break;
            }
            const int ts = t_begin + t * kTileT;
            const uint32_t kb = smem_base + st * kStageBytes;
            const uint32_t vb = kb + kTensorTileBytes;
            if (ts + kTileT > t_end) {
                // keys past the split (pages not loaded, or slots past L_b) may
                // hold any bits: zero their V rows so that P = 0 cannot meet NaN
                const int first = t_end - ts;
                uint8_t* vrow = smem + st * kStageBytes + kTensorTileBytes;
                for (int idx = lane; idx < (kTileT - first) * 16; idx += 32) {
                    const int r = first + (idx >> 4), ch = idx & 15;
                    *reinterpret_cast<uint4*>(vrow + (ch >> 3) * kHalfBytes + r * 128 +
                                              (ch & 7) * 16) = make_uint4(0, 0, 0, 0);
                }
                __syncwarp();
            }

            // ---- S = Q K^T over 64 keys: 8 n-tiles of 8 keys
            float sc[8][4];
#pragma unroll
            for (int i = 0; i < 8; ++i) sc[i][0] = sc[i][1] = sc[i][2] = sc[i][3] = 0.f;
#pragma unroll
            for (int kk = 0; kk < 8; ++kk) {
                const uint32_t half = kb + (kk >> 2) * kHalfBytes;
#pragma unroll
                for (int np = 0; np < 4; ++np) {
                    const int key = (2 * np + (lm >> 1)) * 8 + lr;
                    const int ch = (kk & 3) * 2 + (lm & 1);
                    uint32_t b0, b1, b2, b3;
                    ldsm_x4(half + key * 128 + ((ch ^ (key & 7)) << 4), b0, b1, b2, b3);
                    mma_bf16_16816(sc[2 * np], qa[kk], b0, b1);
                    mma_bf16_16816(sc[2 * np + 1], qa[kk], b2, b3);
                }
            }
            // ---- causal-verify mask and split end
            if (ts + kTileT > lim_min) {
#pragma unroll
                for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
                    for (int e = 0; e < 2; ++e) {
                        const int key = ts + nt * 8 + tq * 2 + e;
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
                for (int nt = 0; nt < 8; ++nt) mx = fmaxf(mx, fmaxf(sc[nt][2 * rh], sc[nt][2 * rh + 1]));
                mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
                mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
                const float m_new = fmaxf(m_raw[rh], mx);
                const float m_use = m_new == kNegInf ? 0.f : m_new;
                const float alpha = ex2((m_raw[rh] - m_use) * c);
                m_raw[rh] = m_new;
                const float neg = -m_use * c;
                float rs = 0.f;
#pragma unroll
                for (int nt = 0; nt < 8; ++nt) {
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
            // ---- O += P V over the 64 keys: 4 k-steps of 16 keys
#pragma unroll
            for (int kk = 0; kk < 4; ++kk) {
                uint32_t a[4];
                a[0] = pack_bf16x2(sc[2 * kk][0], sc[2 * kk][1]);
                a[1] = pack_bf16x2(sc[2 * kk][2], sc[2 * kk][3]);
                a[2] = pack_bf16x2(sc[2 * kk + 1][0], sc[2 * kk + 1][1]);
                a[3] = pack_bf16x2(sc[2 * kk + 1][2], sc[2 * kk + 1][3]);
                const int key = kk * 16 + (lm & 1) * 8 + lr;
#pragma unroll
                for (int dp = 0; dp < 8; ++dp) {
                    const int dblk = 2 * dp + (lm >> 1);
                    const int ch = dblk & 7;
                    uint32_t b0, b1, b2, b3;
                    ldsm_x4_trans(vb + (dblk >> 3) * kHalfBytes + key * 128 + ((ch ^ (key & 7)) << 4),
                                  b0, b1, b2, b3);
                    mma_bf16_16816(o[2 * dp], a, b0, b1);
                    mma_bf16_16816(o[2 * dp + 1], a, b2, b3);
                }
            }
            // generic-proxy writes (the zeroed rows) must be ordered before the
            // next TMA write into this stage
            if (ts + kTileT > t_end) asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            __syncwarp();
            if (lane == 0) mbar_arrive(&empty[st]);
        }

        // ---- epilogue of this warp's 16 rows
        if (!s_abort) {
#pragma unroll
            for (int rh = 0; rh < 2; ++rh) {
                float lt = l[rh];
                lt += __shfl_xor_sync(0xffffffffu, lt, 1);
                lt += __shfl_xor_sync(0xffffffffu, lt, 2);
                const int row = rh ? row1 : row0;
                if (row >= p.n_rows) continue;
                if (ns == 1) {
                    const float inv = lt > 0.f ? 1.f / lt : 0.f;
                    const int i = row / p.G, gi = row % p.G;
                    __nv_bfloat16* dst =
                        p.out + (((size_t)b * p.R + i) * p.Hq + (size_t)h * p.G + gi) * kD + tq * 2;
#pragma unroll
                    for (int dn = 0; dn < 16; ++dn)
                        *reinterpret_cast<uint32_t*>(dst + dn * 8) =
                            pack_bf16x2(o[dn][2 * rh] * inv, o[dn][2 * rh + 1] * inv);
                } else {
                    const size_t slot = ((size_t)b * p.Hkv + h) * p.ns_max + split;
                    float* dst = p.part_o + (slot * p.n_rows + row) * kD + tq * 2;
#pragma unroll
                    for (int dn = 0; dn < 16; ++dn)
                        *reinterpret_cast<float2*>(dst + dn * 8) =
                            make_float2(o[dn][2 * rh], o[dn][2 * rh + 1]);
                    if (tq == 0)
                        p.part_ml[slot * p.n_rows + row] =
                            make_float2(m_raw[rh] == kNegInf ? kNegInf : m_raw[rh] * c, lt);
                }
            }
        }
    }

    if (ns == 1) return;

    // ---------------------------------------------- last split merges
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) {
        int last = 0;
        if (!s_abort) {
            const unsigned int prev = atomicInc(p.tickets + (size_t)b * p.Hkv + h, (unsigned)(ns - 1));
            last = prev == (unsigned)(ns - 1);
        }
        s_last = last;
    }
    __syncthreads();
    if (!s_last) return;
    __threadfence();

    const size_t slot0 = ((size_t)b * p.Hkv + h) * p.ns_max;
    for (int e = threadIdx.x; e < p.n_rows * (kD / 4); e += blockDim.x) {
        const int row = e / (kD / 4), d4 = (e % (kD / 4)) * 4;
        float M = kNegInf;
        for (int s = 0; s < ns; ++s) M = fmaxf(M, __ldcg(&p.part_ml[(slot0 + s) * p.n_rows + row]).x);
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
        float lsum = 0.f;
        if (M != kNegInf) {
            for (int s = 0; s < ns; ++s) {
                const float2 ml = __ldcg(&p.part_ml[(slot0 + s) * p.n_rows + row]);
                const float w = ex2(ml.x - M);
                if (w == 0.f) continue;
                const float4 v = __ldcg(reinterpret_cast<const float4*>(
                    p.part_o + ((slot0 + s) * p.n_rows + row) * kD + d4));
                lsum = fmaf(w, ml.y, lsum);
                acc.x = fmaf(w, v.x, acc.x);
                acc.y = fmaf(w, v.y, acc.y);
                acc.z = fmaf(w, v.z, acc.z);
                acc.w = fmaf(w, v.w, acc.w);
            }
        }
        const float inv = lsum > 0.f ? 1.f / lsum : 0.f;
        const int i = row / p.G, gi = row % p.G;
        __nv_bfloat16* dst = p.out + (((size_t)b * p.R + i) * p.Hq + (size_t)h * p.G + gi) * kD + d4;
        uint2 pk;
        pk.x = pack_bf16x2(acc.x * inv, acc.y * inv);
        pk.y = pack_bf16x2(acc.z * inv, acc.w * inv);
        *reinterpret_cast<uint2*>(dst) = pk;
    }
}

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

cs_status encode_pool_map(CUtensorMap* map, const void* pool, const cs_attn_dims& d, int box_t) {
    auto enc = tensor_map_encoder();
    if (!enc) return fail(CS_ERR_CUDA, "cuTensorMapEncodeTiled is not available from the driver");
    const cuuint64_t dims[4] = {(cuuint64_t)d.head_dim, (cuuint64_t)d.page_size,
                                (cuuint64_t)d.n_kv_heads, (cuuint64_t)d.num_pages};
    const cuuint64_t row = (cuuint64_t)d.head_dim * 2;
    const cuuint64_t strides[3] = {row, row * d.page_size, row * d.page_size * d.n_kv_heads};
    const cuuint32_t box[4] = {64, (cuuint32_t)box_t, 1, 1};
    const cuuint32_t estr[4] = {1, 1, 1, 1};
    const CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(pool), dims,
                           strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                           CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                           CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(CS_ERR_CUDA, "cuTensorMapEncodeTiled failed (CUresult %d)", (int)r);
    return CS_OK;
}

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

}  // namespace

AttnPlan plan_verify_attention(const cs_attn_dims& d, int n_draft, int sm_count) {
    AttnPlan pl{};
    pl.group = d.n_q_heads / d.n_kv_heads;
    pl.rows = n_draft + 1;
    pl.n_rows = pl.rows * pl.group;
    pl.row_warps = (pl.n_rows + 15) / 16;
    const long long l_cap = (long long)d.max_pages_per_seq * d.page_size;
    // Aim for about four CTAs per SM slot (two resident per SM) over the
    // expected half-full contexts; one split never exceeds 4096 keys so that
    // a long request cannot leave a long tail, and is at least one tile.
    const long long target_units = 8LL * (sm_count > 0 ? sm_count : 148);
    long long want = ((long long)d.batch * d.n_kv_heads * (l_cap / 2) + target_units - 1) / target_units;
    want = (want + kTileT - 1) / kTileT * kTileT;
    if (want < kTileT) want = kTileT;
    if (want > 4096) want = 4096;
    pl.chunk = (int)want;
    pl.ns_max = (int)((l_cap + pl.chunk - 1) / pl.chunk);
    if (pl.ns_max < 1) pl.ns_max = 1;
    size_t off = 256;   // status word lives at offset 0
    if (pl.ns_max > 1) {
        pl.off_tickets = off;
        off = align_up(off + sizeof(unsigned int) * (size_t)d.batch * d.n_kv_heads, 256);
        pl.off_part_ml = off;
        off = align_up(off + sizeof(float) * 2 * (size_t)d.batch * d.n_kv_heads * pl.ns_max * pl.n_rows, 256);
        pl.off_part_o = off;
        off = align_up(off + sizeof(float) * kD * (size_t)d.batch * d.n_kv_heads * pl.ns_max * pl.n_rows, 256);
    }
    pl.bytes = off;
    return pl;
}

cs_status launch_verify_attention(const cs_attn_dims& d, const AttnPlan& pl, const void* q,
                                  const void* k_pages, const void* v_pages,
                                  const int32_t* page_table, const int32_t* ctx_lens, void* out,
                                  void* workspace, cudaStream_t stream) {
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
    p.status = reinterpret_cast<int*>(ws);
    p.tickets = pl.ns_max > 1 ? reinterpret_cast<unsigned int*>(ws + pl.off_tickets) : nullptr;
    p.part_ml = pl.ns_max > 1 ? reinterpret_cast<float2*>(ws + pl.off_part_ml) : nullptr;
    p.part_o = pl.ns_max > 1 ? reinterpret_cast<float*>(ws + pl.off_part_o) : nullptr;
    p.Hq = d.n_q_heads;
    p.Hkv = d.n_kv_heads;
    p.G = pl.group;
    p.R = pl.rows;
    p.n_rows = pl.n_rows;
    p.ps = d.page_size;
    p.box_t = box_t;
    p.max_pages = d.max_pages_per_seq;
    p.chunk = pl.chunk;
    p.ns_max = pl.ns_max;
    p.row_warps = pl.row_warps;
    const float scale = d.sm_scale > 0.f ? d.sm_scale : 1.0f / sqrtf((float)d.head_dim);
    p.scale_log2 = scale * 1.4426950408889634f;

    static bool attr_set = false;
    if (!attr_set) {
        cudaError_t e = cudaFuncSetAttribute(verify_attention_kernel,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
        if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute(verify_attention_kernel)");
        attr_set = true;
    }
    const dim3 block((pl.row_warps + 1) * 32);
    for (int b0 = 0; b0 < d.batch; b0 += 65535) {
        p.b_base = b0;
        const dim3 grid(pl.ns_max, d.n_kv_heads, d.batch - b0 < 65535 ? d.batch - b0 : 65535);
        verify_attention_kernel<<<grid, block, kSmemBytes, stream>>>(tk, tv, p);
        const cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return cuda_fail(e, "verify_attention_kernel launch");
    }
    return CS_OK;
}

}  // namespace cs
