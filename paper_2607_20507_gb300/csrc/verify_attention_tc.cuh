// verify_attention_tc.cuh -- the tcgen05 form of the verify-attention kernel
// (included by verify_attention.cu inside its anonymous namespace, so that it
// shares the schedule, the parameter block, the tensor maps and the merge).
//
// Used for 33..128 query rows per KV head, where the mma.sync consumers of
// the other form run out of tensor throughput (up to 32 rows the key-split
// mma.sync form streams faster than this one with its M = 128 padding).  A
// token tree with more rows comes in row blocks of whole nodes, at most 128
// rows each; each block is a span of its own (reading the request's keys
// again) whose query box starts at the block's first node.
// Same persistent schedule (contiguous ranges of equal work, spans, two partial
// slots per CTA, merge kernel), one CTA per SM, twelve warps.  Each SMSP
// (warp % 4) runs one role warp and up to two softmax warps; the live
// softmax warps fill SMSPs 0 and 1 first, so the two producers sit on SMSPs
// 2 and 3, where they share the issue slots with the fewest softmax warps
// (with them on SMSPs 0 and 1 the kernel ran 7-15% slower):
//   warp 2  K producer: the span's query rows (one 4-D box per dim half into
//           one buffer, refilled once the previous span's rows have been
//           copied into tensor memory; each half as many 128-byte rows as
//           the span has: the MMA's 128-row window runs on into whatever
//           follows, which only feeds padded rows) and the K tiles of the
//           range through the K ring, one box per page piece with both dim
//           halves (contiguous 256-byte rows: a per-half box of 128-byte rows
//           kept the SM's copy engine saturated at two thirds of the
//           bandwidth), so a tile lands as [piece][dim half][keys][128 B],
//           128-byte swizzle;
//           beside each stage it leaves whether the tile opens or closes a
//           piece;
//   warp 3  V producer: the V tiles through the V ring, the same way.  The
//           two rings share the 16 KB stages that shared memory holds beside
//           the query buffer (a third for K, which is released as soon as
//           its QK is done; the rest for V, held until its PV is done), so
//           each side runs ahead as far as its own consumer allows;
//   warp 0  QK issuer (the whole warp waits, one elected lane issues): at
//           a piece's start the query rows from shared into tensor memory
//           (tcgen05.cp, one buffer per span parity), then per tile
//           S_t = Q K_t^T into tensor memory (M = 128 padded rows, per page
//           piece N = its keys, Q from tensor memory, K a K-major
//           shared-memory operand, 8 steps of 16 dims) as soon as K_t has
//           landed and one of four S buffers is free -- up to four tiles
//           ahead of the softmax.  It also allocates the tensor memory (512
//           columns: four S/P buffers of 64, O in 128, two query buffers of
//           64);
//   warp 1  PV issuer: O += P_t V_t (N = 128 dims, 8 steps of 16 keys: 4
//           with P_hi, 4 with P_lo) as soon as the softmax releases P_t and
//           V_t has landed, with P read from tensor memory and V, as stored
//           in bf16, an MN-major operand (per 16 keys, the rows of one page
//           piece) whose two dim halves lie one piece half apart; in a span's
//           last tile it first zeroes the V rows past L_b (their slots may
//           hold any bits);
//   warps 4-11 softmax and epilogue, one warp per 16 tensor-memory lanes
//           (query rows; warp 4+q lanes 32q..32q+15, warp 8+q lanes
//           32q+16..32q+31; a warp whose lanes hold no query row idles):
//           threads t and t+16 share the row of lane t % 16 and take keys
//           0..31 and 32..63 of every tile (16-lane tensor-memory access),
//           so a row's maximum and sum meet in one shuffle.  Mask, running
//           max, exp2, row sum, P written back over S as two bf16 terms, hi
//           and lo (bf16 P alone can exceed the output tolerance on rows
//           whose terms cancel), formed as P * 2^-64 so that no partial sum
//           of P.V overflows fp32 for any finite bf16 V; pairs of keys in
//           packed fp32 arithmetic.  O is rescaled in tensor memory only
//           when the running max grows by more than 2^8 (the stale max keeps
//           every P below 256); at a span piece's end the row is normalised
//           and written (bf16) or left as a partial, dims 0..63 by thread t
//           and 64..127 by thread t+16.
// Every mbarrier wait is bounded; a wait that gives up sets the status word
// and a shared flag that ends every warp's loop.

constexpr int kTcMaxK = 6;                         // K ring depth, at most
constexpr int kTcMaxV = 10;                        // V ring depth, at most
constexpr int kTcThreads = 384;                    // 12 warps: 4 roles, 8 softmax (three warps per SMSP)
constexpr int kTcKWarp = 2;                        // the K producer (and the query rows)
constexpr int kTcVWarp = 3;                        // the V producer
constexpr int kTcQkWarp = 0;                       // the QK issuer (and tensor-memory allocator)
constexpr int kTcPvWarp = 1;                       // the PV issuer
constexpr int kTcRows = 128;                       // MMA M: query rows, padded
constexpr int kTcMinRows = 32;                     // fewer query rows take the key-split mma.sync form
constexpr int kTcSBuf = 4;                         // S/P buffers in tensor memory
constexpr int kTcOCol = kTcSBuf * 64;              // first column of O
constexpr int kTcQCol = kTcOCol + 128;             // first column of the two query buffers (64 each)
constexpr int kTcTmemCols = 512;                   // S/P [0, 256) in four buffers, O [256, 384), Q [384, 512)
constexpr int kTcBarBytes = 512;
constexpr int kTcFixedSmem = kTcBarBytes + (kMaxBatchPerLaunch + 1) * 8 + kMaxBatchPerLaunch * 4 + 1024;
constexpr int kTcSmemLimit = 232448 - 2560;        // opt-in shared memory per block, less the static part

// Bytes between the two dim halves of a span's query rows (1024-aligned).
__host__ __device__ constexpr int tc_q_half_bytes(int rows) { return (rows * 128 + 1023) / 1024 * 1024; }
// 16 KB tile stages (one K or one V tile each) that fit beside the query
// buffer of `rows` rows, split between the K ring (a third: K is released
// as soon as its QK is done) and the V ring (the rest: V waits for the
// softmax).
__host__ __device__ constexpr int tc_tile_stages(int rows) {
    return (kTcSmemLimit - kTcFixedSmem - 2 * tc_q_half_bytes(rows)) / kTensorTileBytes;
}
__host__ __device__ constexpr int tc_k_stages(int rows) {
    return (tc_tile_stages(rows) + 1) / 3 < 2 ? 2
           : (tc_tile_stages(rows) + 1) / 3 > kTcMaxK ? kTcMaxK : (tc_tile_stages(rows) + 1) / 3;
}
__host__ __device__ constexpr int tc_v_stages(int rows) {
    return tc_tile_stages(rows) - tc_k_stages(rows) > kTcMaxV ? kTcMaxV : tc_tile_stages(rows) - tc_k_stages(rows);
}
__host__ __device__ constexpr int tc_smem_bytes(int rows) {
    return 2 * tc_q_half_bytes(rows) + (tc_k_stages(rows) + tc_v_stages(rows)) * kTensorTileBytes + kTcFixedSmem;
}
static_assert(tc_k_stages(kTcRows) >= 2 && tc_v_stages(kTcRows) >= 4, "rings too shallow for 128 query rows");
static_assert((2 * kTcMaxK + 2 * kTcMaxV + 4 + 3 * kTcSBuf + 1) * 8 <= kTcBarBytes, "barrier block too small");
constexpr float kTcRescale = 8.f;                  // log2 growth of the max that forces a rescale of O

__device__ __forceinline__ uint64_t tc_sw128_desc(uint32_t addr) {
    // K-major, 128-byte swizzle: 8-row groups 1024 bytes apart (leading offset unused)
    return (uint64_t)((addr >> 4) & 0x3FFF) | ((uint64_t)1 << 16) | ((uint64_t)(1024 >> 4) << 32) | (1ull << 46) |
           (2ull << 61);
}

// MN-major, 128-byte swizzle, for a V page piece [dim half][keys][128 B]:
// 8-key groups 1024 bytes apart (stride), the two 64-dim halves
// `half_bytes` apart (leading offset)
__device__ __forceinline__ uint64_t tc_mn_desc(uint32_t addr, uint32_t half_bytes) {
    return (uint64_t)((addr >> 4) & 0x3FFF) | ((uint64_t)(half_bytes >> 4) << 16) |
           ((uint64_t)(1024 >> 4) << 32) | (1ull << 46) | (2ull << 61);
}

// kind::f16 instruction descriptor: fp32 D, M = 128, N = n, A and B both
// bf16 (f16 = false) or both fp16; b_mn: B is MN-major (its N index contiguous)
__host__ __device__ constexpr uint32_t tc_idesc(int n, bool b_mn, bool f16) {
    return (1u << 4) | (f16 ? 0u : (1u << 7) | (1u << 10)) | (b_mn ? (1u << 16) : 0u) | ((uint32_t)(n >> 3) << 17) |
           ((uint32_t)(kTcRows >> 4) << 24);
}

// One lane of the (converged) warp, the same one every time: the lowest.
__device__ __forceinline__ bool elect_one() {
    uint32_t r;
    asm volatile(
        "{\n\t.reg .pred P;\n\telect.sync _|P, 0xffffffff;\n\tselp.u32 %0, 1, 0, P;\n\t}\n"
        : "=r"(r));
    return r != 0;
}

// 128 rows x 32 bytes of a K-major shared-memory operand (the same
// descriptor the MMA would read it through) into 128 lanes x 8 columns of
// tensor memory, laid out as an A operand from tensor memory.  Executes in
// issue order with the MMAs of the same thread that follow it.
__device__ __forceinline__ void tc_cp_128x256b(uint32_t taddr, uint64_t sdesc) {
    asm volatile("tcgen05.cp.cta_group::1.128x256b [%0], %1;" ::"r"(taddr), "l"(sdesc) : "memory");
}

__device__ __forceinline__ void tc_commit(uint64_t* bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(bar))
                 : "memory");
}

__device__ __forceinline__ void tc_mma_ss(uint32_t d, uint64_t a, uint64_t b, uint32_t idesc, uint32_t acc) {
    asm volatile(
        "{\n\t.reg .pred q;\n\tsetp.ne.b32 q, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, q;\n\t}\n" ::"r"(d),
        "l"(a), "l"(b), "r"(idesc), "r"(acc)
        : "memory");
}

__device__ __forceinline__ void tc_mma_ts(uint32_t d, uint32_t a_tmem, uint64_t b, uint32_t idesc, uint32_t acc) {
    asm volatile(
        "{\n\t.reg .pred q;\n\tsetp.ne.b32 q, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, q;\n\t}\n" ::"r"(d),
        "r"(a_tmem), "l"(b), "r"(idesc), "r"(acc)
        : "memory");
}

__device__ __forceinline__ void tc_ld32(uint32_t addr, float (&v)[32]) {
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(addr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

__device__ __forceinline__ void tc_st32(uint32_t addr, const uint32_t (&r)[32]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
        "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(addr),
        "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]),
        "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]), "r"(r[17]),
        "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]),
        "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
        : "memory");
}

__device__ __forceinline__ void tc_st16(uint32_t addr, const uint32_t (&r)[16]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(
            addr),
        "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]),
        "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
        : "memory");
}

// 16 lanes x 32 columns, twice: threads 0..15 read lanes base..base+15 at
// columns col..col+31, threads 16..31 the same lanes at col + split..  (each
// thread one lane, 32 consecutive columns)
template <int kSplitOff>
__device__ __forceinline__ void tc_ld16x2_32(uint32_t addr, float (&v)[32]) {
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.16x32bx2.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32], %33;"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(addr), "n"(kSplitOff));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

template <int kSplitOff>
__device__ __forceinline__ void tc_st16x2_32(uint32_t addr, const uint32_t (&r)[32]) {
    asm volatile(
        "tcgen05.st.sync.aligned.16x32bx2.x32.b32 [%0], %1, {%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
        "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32,%33};" ::"r"(addr),
        "n"(kSplitOff), "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
        "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]),
        "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]),
        "r"(r[26]), "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
        : "memory");
}

template <int kSplitOff>
__device__ __forceinline__ void tc_st16x2_16(uint32_t addr, const uint32_t (&r)[16]) {
    asm volatile(
        "tcgen05.st.sync.aligned.16x32bx2.x16.b32 [%0], %1, {%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
        "%17};" ::"r"(addr),
        "n"(kSplitOff), "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
        "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
        : "memory");
}

// Packed fp32 pairs (one instruction for both lanes of a pair)
__device__ __forceinline__ uint64_t f2_pack(float a, float b) {
    uint64_t r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(a), "f"(b));
    return r;
}
__device__ __forceinline__ void f2_unpack(uint64_t v, float& a, float& b) {
    asm("mov.b64 {%0, %1}, %2;" : "=f"(a), "=f"(b) : "l"(v));
}
__device__ __forceinline__ uint64_t f2_fma(uint64_t a, uint64_t b, uint64_t c) {
    uint64_t d;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
    return d;
}
__device__ __forceinline__ uint64_t f2_add(uint64_t a, uint64_t b) {
    uint64_t d;
    asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
    return d;
}
__device__ __forceinline__ uint64_t f2_sub(uint64_t a, uint64_t b) {
    uint64_t d;
    asm("sub.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
    return d;
}
__device__ __forceinline__ float fmax3(float a, float b, float c) {
    float d;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
    return d;
}

__device__ __forceinline__ void tc_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// Bounded wait that also gives up at once when another warp already has.
__device__ __forceinline__ bool tc_wait(uint64_t* bar, uint32_t parity, volatile int* dead, int* status) {
    if (mbar_test_wait(bar, parity)) return true;
    if (*dead) return false;
    if (mbar_wait_bounded(bar, parity)) return true;
    *dead = 1;
    atomicOr(status, CS_DEVICE_WAIT_TIMEOUT);
    return false;
}


template <bool kTree, int kBoxT>
__global__ void __launch_bounds__(kTcThreads, 1)
verify_attention_tc_kernel(const __grid_constant__ CUtensorMap tmap_k, const __grid_constant__ CUtensorMap tmap_v,
                           const __grid_constant__ CUtensorMap tmap_q, const AttnParams p) {
    constexpr int kPieces = kTileT / kBoxT;
    constexpr uint32_t kPieceBytes = (uint32_t)kBoxT * 256u;   // bytes of one page piece of K (or of V)
    constexpr uint32_t kPieceHalf = (uint32_t)kBoxT * 128u;    // one dim half of a page piece
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int SK = p.tc_stages, SV = p.tc_vstages;          // K and V ring depths
    const int qh = p.tc_q_half;                             // bytes between the dim halves of a span's rows
    uint8_t* sq = smem;                                     // [2 halves][rows][128 B]: one span's query rows
    uint8_t* sk = smem + 2 * qh;                            // [K stage][half][64 keys][128 B]
    uint8_t* sv = sk + SK * kTensorTileBytes;               // [V stage][half][64 keys][128 B]
    uint64_t* bars = reinterpret_cast<uint64_t*>(sv + SV * kTensorTileBytes);
    uint64_t* kfull = bars;                                 // [SK] K tile landed
    uint64_t* kempty = kfull + kTcMaxK;                     // [SK] K tile consumed (QK done)
    uint64_t* vfull = kempty + kTcMaxK;                     // [SV] V tile landed
    uint64_t* vempty = vfull + kTcMaxV;                     // [SV] V tile consumed (PV done)
    uint64_t* q_full = vempty + kTcMaxV;                    // a span's query rows landed in shared memory
    uint64_t* q_cp = q_full + 1;                            // ... and were copied into tensor memory
    uint64_t* q_free = q_cp + 1;                            // [2] last QK of a span done (tensor-memory buffer)
    uint64_t* s_full = q_free + 2;                          // [kTcSBuf] S_t in tensor memory
    uint64_t* p_full = s_full + kTcSBuf;                    // [kTcSBuf] P_t written (count: live softmax warps)
    uint64_t* o_ready = p_full + kTcSBuf;                   // [kTcSBuf] PV_t done (S buffer free again)
    uint64_t* o_free = o_ready + kTcSBuf;                   // O read out by the epilogue (count: live softmax warps)
    long long* s_prefix = reinterpret_cast<long long*>(reinterpret_cast<uint8_t*>(bars) + kTcBarBytes);
    int* s_len = reinterpret_cast<int*>(s_prefix + kMaxBatchPerLaunch + 1);
    __shared__ long long s_wtot[kTcThreads / 32];
    __shared__ long long s_carry;
    __shared__ uint32_t s_tmem;
    __shared__ volatile int s_dead;
    __shared__ int s_keys[kTcMaxV];   // keys of the tile in each V stage (V rows past are zeroed)
    __shared__ int s_info[kTcMaxK];   // per K stage, bit 0: the tile opens a span piece, bit 1: ends one

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nb = p.n_batch;
    // softmax warps with a live query row: 16-lane group g (lanes 16g..16g+15)
    // belongs to warp 4 + g / 2 + 4 (g % 2); groups past the span's rows idle
    const int n_live = min(8, ((kTree ? p.n_rows : p.n_rows_all) + 15) / 16);

    if (warp == kTcKWarp) {
        // the page table of this launch into L2 while the schedule is computed
        const char* tab = reinterpret_cast<const char*>(p.page_table + (size_t)p.b_base * p.max_pages);
        const long long lines = ((long long)nb * p.max_pages * 4 + 127) / 128;
        for (long long i = (long long)blockIdx.x * 32 + lane; i < lines; i += (long long)gridDim.x * 32)
            asm volatile("prefetch.global.L2 [%0];" ::"l"(tab + i * 128));
    }
    if (warp == kTcQkWarp) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&s_tmem)),
                     "n"(kTcTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    if (threadIdx.x == 0) {
        s_carry = 0;
        s_dead = 0;
        for (int i = 0; i < SK; ++i) {
            mbar_init(&kfull[i], 1);
            mbar_init(&kempty[i], 1);
        }
        for (int i = 0; i < SV; ++i) {
            mbar_init(&vfull[i], 1);
            mbar_init(&vempty[i], 1);
        }
        mbar_init(q_full, 1);
        mbar_init(q_cp, 1);
        for (int i = 0; i < 2; ++i) mbar_init(&q_free[i], 1);
        for (int i = 0; i < kTcSBuf; ++i) {
            mbar_init(&s_full[i], 1);
            mbar_init(&p_full[i], n_live);
            mbar_init(&o_ready[i], 1);
        }
        mbar_init(o_free, n_live);
        fence_barrier_init();
    }
    // a programmatic dependent of the kernel before it (inputs are read
    // below); the merge kernel may start once every CTA is past this point
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    // ---- schedule: exclusive prefix of tiles per request (x spans), clamped L
    __syncthreads();
    const int l_cap = p.max_pages * p.ps;
    for (int base = 0; base < nb; base += kTcThreads) {
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
        if (threadIdx.x == kTcThreads - 1) s_carry = before + inc;
        __syncthreads();
    }
    if (threadIdx.x == 0) {
        s_prefix[nb] = s_carry;
        // this CTA's two partial slots start unused
        p.part_span[2 * blockIdx.x] = -1;
        p.part_span[2 * blockIdx.x + 1] = -1;
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = s_tmem;

    const long long W = s_prefix[nb];
    const long long g_need = (W + kMinTilesPerCta - 1) / kMinTilesPerCta;
    const int Gc = (int)(g_need < (long long)gridDim.x ? (g_need > 0 ? g_need : 1) : gridDim.x);
    const int cta = blockIdx.x;
    const long long U = W + (long long)p.span_x * p.n_vh * nb;
    long long f0 = tiles_before(unit_start(cta, U, Gc), s_prefix, s_len, nb, p.n_vh, p.span_x);
    long long f1 = tiles_before(unit_start(cta + 1, U, Gc), s_prefix, s_len, nb, p.n_vh, p.span_x);
    if (cta >= Gc) f0 = f1 = 0;
    const int n_tiles = (int)(f1 - f0);
    // one dim half of a span's rows (trees: of its row block of q_nodes nodes)
    const uint32_t qrow_bytes = (uint32_t)(kTree ? p.n_rows : p.R * p.G) * 128u;
    const int q_nodes = p.n_rows / p.G;

    if ((warp == kTcKWarp || warp == kTcVWarp) && n_tiles > 0) {
        // --------------------------------------------------------- producers
        // warp kTcKWarp: the K tiles (and, opening a piece, the query rows) through
        // the K ring; warp kTcVWarp: the V tiles through the V ring.  Each
        // runs ahead as far as its own ring allows.
        const bool k_side = warp == kTcKWarp;
        const int S = k_side ? SK : SV;
        uint8_t* const ring = k_side ? sk : sv;
        uint64_t* const fullb = k_side ? kfull : vfull;
        uint64_t* const emptyb = k_side ? kempty : vempty;
        const CUtensorMap* const tmap = k_side ? &tmap_k : &tmap_v;
        constexpr int per_batch = 32 / kPieces;
        auto batch_pages = [&](int j0) -> int {
            const int jj = j0 + lane / kPieces;
            if (jj >= n_tiles) return -1;
            const Cursor cc = locate(f0 + jj, s_prefix, s_len, nb, p.n_vh);
            const int tok = cc.t * kTileT + (lane % kPieces) * kBoxT;
            if (tok >= s_len[cc.b]) return -1;
            return __ldg(p.page_table + (size_t)(p.b_base + cc.b) * p.max_pages + tok / p.ps);
        };
        if (lane == 0) {
            tma_prefetch_desc(tmap);
            if (k_side) tma_prefetch_desc(&tmap_q);
        }
        Cursor cur = locate(f0, s_prefix, s_len, nb, p.n_vh);
        int pg_cur = batch_pages(0);
        int pg_next = per_batch < n_tiles ? batch_pages(per_batch) : -1;
        // The next tile's page, position and flags are worked out while the
        // current one waits for its stage (the cursor walk, the page-id
        // batches and their lookups stay off the path from a free stage to
        // its copy).
        struct Next {
            int page, L, ts, h, rb, b, valid;
            bool first, last;
        } nx;
        auto prepare = [&](int jt) {
            const int jb = jt % per_batch;
            if (jt > 0 && jb == 0) {
                pg_cur = pg_next;
                pg_next = jt + per_batch < n_tiles ? batch_pages(jt + per_batch) : -1;
            }
            nx.page = __shfl_sync(0xffffffffu, pg_cur, jb * kPieces + lane % kPieces);
            nx.first = jt == 0 || cur.t == 0;
            nx.last = jt + 1 == n_tiles || cur.t + 1 == cur.T;
            nx.L = s_len[cur.b];
            nx.ts = cur.t * kTileT;
            nx.h = cur.h / p.n_rb;
            if (kTree) nx.rb = cur.h - nx.h * p.n_rb;
            nx.b = cur.b;
            advance(cur, s_len, nb, p.n_vh);
            nx.valid = 0;
            for (int pc = 0; pc < kPieces; ++pc)
                if (nx.ts + pc * kBoxT < nx.L) ++nx.valid;
        };
        prepare(0);
        int span = -1;
        // tile jt goes out once its stage is free and, K side opening a
        // piece, once the query buffer is free
        int jt = 0;
        for (; jt < n_tiles; ++jt) {
            const int st = jt % S;
            const Next c = nx;
            if (c.first) ++span;
            bool go = jt < S || tc_wait(&emptyb[st], (uint32_t)(jt / S - 1) & 1, &s_dead, p.status);
            // the query buffer is free once the previous span's rows are in tensor memory
            if (go && k_side && c.first && span >= 1)
                go = tc_wait(q_cp, (uint32_t)(span - 1) & 1, &s_dead, p.status);
            if (!__all_sync(0xffffffffu, go)) break;
            if (k_side && c.first && lane == 0) {
                // a new span piece: its query rows into the query buffer
                mbar_arrive_expect_tx(q_full, 2 * qrow_bytes);
                const uint32_t qdst = smem_u32(sq);
#pragma unroll
                for (int hh = 0; hh < 2; ++hh)
                    tma_load_4d(qdst + hh * qh, &tmap_q, q_full, hh * 64, c.h * p.G, kTree ? c.rb * q_nodes : 0,
                                p.b_base + c.b);
            }
            if (lane == 0) {
                if (k_side) s_info[st] = (c.first ? 1 : 0) | (c.last ? 2 : 0);
                else s_keys[st] = max(0, min(kTileT, c.L - c.ts));
                mbar_arrive_expect_tx(&fullb[st], (uint32_t)c.valid * kPieceBytes);
            }
            __syncwarp();
            if (lane < c.valid) {
                // one box per page piece, both dim halves: [half][kBoxT keys][128 B]
                // (page sizes are powers of two)
                const uint32_t dst = smem_u32(ring + st * kTensorTileBytes) + (uint32_t)lane * kPieceBytes;
                const int slot = (c.ts + lane * kBoxT) & (p.ps - 1);
                tma_load_5d(dst, tmap, &fullb[st], 0, slot, 0, c.h, c.page);
            }
            if (jt + 1 < n_tiles) prepare(jt + 1);
        }
        // no copy in flight at exit: every issued tile has landed
        if (lane == 0)
            for (int j = jt > S ? jt - S : 0; j < jt; ++j)
                if (!mbar_wait_bounded(&fullb[j % S], (uint32_t)(j / S) & 1)) atomicOr(p.status, CS_DEVICE_WAIT_TIMEOUT);
    } else if ((warp == kTcQkWarp || warp == kTcPvWarp) && n_tiles > 0) {
        // ---------------------------------------------------------- MMA
        // Two issuing warps, each running its loop with all lanes (the waits)
        // and one elected lane issuing (a lone lane beside 31 parked at the
        // block barrier pays hundreds of cycles per barrier probe and per
        // tcgen05 instruction).  Each commit tracks the MMAs of its own
        // thread only, and the two streams meet only through barriers:
        //   warp kTcQkWarp (QK): S_t = Q K_t^T as soon as K_t has landed and S buffer
        //     t % 4 is free (PV_{t-4} done) -- up to four tiles ahead of the
        //     softmax, whatever the PV stream is doing;
        //   warp kTcPvWarp (PV): O += P_t V_t as soon as the softmax has
        //     released P_t (and, opening a piece, the epilogue has read O).
        // Each wait names a phase its barrier can be at most one phase short
        // of (the next phase needs an MMA of this warp that is not issued
        // yet), so a parity wait is exact.  Descriptors advance by constant
        // offsets (addresses stay below 256 KB: the 14-bit start field cannot
        // carry).
        const bool qk_warp = warp == kTcQkWarp;
        // QK and PV both bf16: P enters as two bf16 terms (hi + lo) against V as stored
        constexpr uint32_t id_s = tc_idesc(kBoxT, false, false), id_o = tc_idesc(kD, true, false);
        const uint64_t dq0 = tc_sw128_desc(smem_u32(sq));
        const uint64_t qhalf16 = (uint64_t)qh >> 4;
        const uint64_t dk0 = tc_sw128_desc(smem_u32(sk)), dv0 = tc_mn_desc(smem_u32(sv), kPieceHalf);
        int span = -1, pv_piece = 0;
        Cursor cur = locate(f0, s_prefix, s_len, nb, p.n_vh);   // the PV warp's own view of the pieces
        uint64_t* last_bar = nullptr;   // the warp's latest commit: completes after all its MMAs
        uint32_t last_par = 0;
        // every lane waits; the result is made warp-uniform, so that no lane
        // leaves the loop while another still issues
        auto wait_all = [&](uint64_t* bar, uint32_t par) -> bool {
            return __all_sync(0xffffffffu, tc_wait(bar, par, &s_dead, p.status));
        };
        for (int t = 0; t < n_tiles; ++t) {
            const int sb = t % kTcSBuf;
            if (qk_warp) {
                const int st = t % SK;
                if (!wait_all(&kfull[st], (uint32_t)(t / SK) & 1)) break;
                const int info = s_info[st];
                if (info & 1) {
                    // a new piece: its query rows landed, and the QKs of the
                    // piece two back are done reading the query buffer
                    ++span;
                    if (!wait_all(q_full, (uint32_t)span & 1)) break;
                    if (span >= 2 && !wait_all(&q_free[span & 1], (uint32_t)((span - 2) >> 1) & 1)) break;
                }
                // S buffer sb held S_{t-4}: PV_{t-4} is done with it
                if (t >= kTcSBuf && !wait_all(&o_ready[sb], (uint32_t)((t - kTcSBuf) / kTcSBuf) & 1)) break;
                tc_fence_after();
                const uint32_t tq = tmem + kTcQCol + (span & 1) * 64;
                const uint64_t dk = dk0 + (uint64_t)((st * kTensorTileBytes) >> 4);
                if (elect_one()) {
                    if (info & 1) {
                        // the query rows into tensor memory once per piece, 16
                        // dims (8 columns) per copy; every QK of the piece then
                        // reads only K from shared memory
#pragma unroll
                        for (int ks = 0; ks < kD / 16; ++ks)
                            tc_cp_128x256b(tq + ks * 8, dq0 + (ks >> 2) * qhalf16 + (uint64_t)((ks & 3) * 2));
                        tc_commit(q_cp);   // the producer may refill the query buffer
                    }
                    // per page piece (N = kBoxT keys, S columns pc*kBoxT..), 8
                    // steps of 16 dims
#pragma unroll
                    for (int pc = 0; pc < kPieces; ++pc) {
#pragma unroll
                        for (int ks = 0; ks < kD / 16; ++ks) {
                            const uint64_t ko =
                                (uint64_t)(((pc * kPieceBytes + (ks >> 2) * kPieceHalf) >> 4) + (ks & 3) * 2);
                            tc_mma_ts(tmem + sb * 64 + pc * kBoxT, tq + ks * 8, dk + ko, id_s, ks > 0 ? 1u : 0u);
                        }
                    }
                    tc_commit(&s_full[sb]);
                    tc_commit(&kempty[st]);
                    if (info & 2) tc_commit(&q_free[span & 1]);
                }
                __syncwarp();
                last_bar = &s_full[sb];
                last_par = (uint32_t)(t / kTcSBuf) & 1;
            } else {
                const int st = t % SV;
                if (!wait_all(&p_full[sb], (uint32_t)(t / kTcSBuf) & 1)) break;
                // V_t has landed (the stage's next landing needs this PV first)
                if (!wait_all(&vfull[st], (uint32_t)(t / SV) & 1)) break;
                const bool first = t == 0 || cur.t == 0;
                advance(cur, s_len, nb, p.n_vh);
                if (first) {
                    // the previous piece's epilogue has read O
                    if (pv_piece > 0 && !wait_all(o_free, (uint32_t)(pv_piece - 1) & 1)) break;
                    ++pv_piece;
                }
                // a span's last tile: the slots past L_b may hold any bits (NaN
                // included) and P is 0 there, so their V rows are zeroed (128-byte
                // row r of the tile, [piece][half][kBoxT keys], holds key
                // (r / (2 kBoxT)) kBoxT + r % kBoxT)
                const int keys = s_keys[st];
                if (keys < kTileT) {
                    uint4* vt = reinterpret_cast<uint4*>(sv + st * kTensorTileBytes);
                    for (int i = lane; i < kTensorTileBytes / 16; i += 32) {
                        const int r = i >> 3;
                        if ((r / (2 * kBoxT)) * kBoxT + r % kBoxT >= keys) vt[i] = make_uint4(0, 0, 0, 0);
                    }
                    // generic writes the tensor core reads next
                    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                    __syncwarp();
                }
                tc_fence_after();
                // O += P_t V_t: 4 steps of 16 keys with P_hi (columns 0..31 of
                // the buffer), 4 with P_lo (columns 32..63), both dim halves per step
                const uint64_t dv = dv0 + (uint64_t)((st * kTensorTileBytes) >> 4);
                if (elect_one()) {
                    // keys 16kk..16kk+15: rows (16kk) % kBoxT.. of page piece 16kk / kBoxT
#pragma unroll
                    for (int kk = 0; kk < kTileT / 16; ++kk) {
                        const uint64_t vk = dv + (uint64_t)((((16 * kk) / kBoxT) * kPieceBytes + ((16 * kk) % kBoxT) * 128) >> 4);
                        tc_mma_ts(tmem + kTcOCol, tmem + sb * 64 + kk * 8, vk, id_o, (first && kk == 0) ? 0u : 1u);
                    }
#pragma unroll
                    for (int kk = 0; kk < kTileT / 16; ++kk) {
                        const uint64_t vk = dv + (uint64_t)((((16 * kk) / kBoxT) * kPieceBytes + ((16 * kk) % kBoxT) * 128) >> 4);
                        tc_mma_ts(tmem + kTcOCol, tmem + sb * 64 + 32 + kk * 8, vk, id_o, 1u);
                    }
                    tc_commit(&o_ready[sb]);
                    tc_commit(&vempty[st]);
                }
                __syncwarp();
                last_bar = &o_ready[sb];
                last_par = (uint32_t)(t / kTcSBuf) & 1;
            }
        }
        // every MMA of this warp completes before tensor memory is freed
        if (last_bar != nullptr && !mbar_wait_bounded(last_bar, last_par) && lane == 0)
            atomicOr(p.status, CS_DEVICE_WAIT_TIMEOUT);
    } else if (warp >= 4 && warp < 12 && n_tiles > 0 && ((warp & 3) * 2 + (warp >> 3)) < n_live) {
        // ---------------------------------------------------- softmax, epilogue
        // Two warps per tensor-memory lane quarter q: warp 4+q takes lanes
        // 32q..32q+15, warp 8+q lanes 32q+16..32q+31 (one query row per lane).
        // In a warp, threads t and t+16 share the row of lane t % 16: the
        // first takes keys 0..31 of every tile, the second keys 32..63 (the
        // 16x32bx2 access shape), so a row's max and sum meet in one shuffle.
        const int sub = warp & 3, hw = warp >> 3;
        const int kh = lane >> 4;                              // key half of this thread
        const int kb = kh * 32;                                // its first key of a tile
        const int lane0 = sub * 32 + hw * 16;                  // the warp's first tensor-memory lane
        const int row = lane0 + (lane & 15);                   // query row of the span = tensor-memory lane
        const uint32_t t_row = tmem + ((uint32_t)lane0 << 16);
        const float c = p.scale_log2;
        Cursor cur = locate(f0, s_prefix, s_len, nb, p.n_vh);
        int seg_t0 = cur.t;
        bool first_seg = true;
        float m_run = kNegInf, l_part = 0.f;
        int lim = 0, tree_base = 0, span_L = 0;
        // trees may come in row blocks: the query row of the request and KV
        // head is the block's first row + row, and rows past the block's
        // end are padding; a chain is one block
        int qrow = row;
        bool tree_live = false;
        uint64_t anc = ~0ull;
        auto begin_span = [&](const Cursor& cc) {
            const int L = s_len[cc.b];
            m_run = kNegInf;
            l_part = 0.f;
            if (kTree) {
                qrow = (cc.h % p.n_rb) * p.n_rows + row;
                tree_live = row < p.n_rows && qrow < p.n_rows_all;
                uint64_t ma, mb;
                tree_ancestor_masks(p.parents + (size_t)(p.b_base + cc.b) * p.R, p.R, lane, ma, mb);
                const int i = tree_live ? qrow / p.G : 0;
                const uint64_t x = __shfl_sync(0xffffffffu, ma, i & 31), y = __shfl_sync(0xffffffffu, mb, i & 31);
                anc = tree_live ? (i >= 32 ? y : x) : ~0ull;
                tree_base = L - p.R;
                span_L = L;
            } else {
                lim = row < p.n_rows_all ? L - p.R + 1 + row / p.G : L;
            }
        };
        begin_span(cur);
        for (int t = 0; t < n_tiles; ++t) {
            const int sb = t % kTcSBuf;
            const int ts = cur.t * kTileT;
            const bool piece_end = t + 1 == n_tiles || cur.t + 1 == cur.T;
            if (!tc_wait(&s_full[sb], (uint32_t)(t / kTcSBuf) & 1, &s_dead, p.status)) break;
            tc_fence_after();
            float s[32];
            tc_ld16x2_32<32>(t_row + sb * 64, s);
            // ---- mask (tree ancestors or the causal chain, and the context end);
            // padded rows see nothing
            if (kTree ? !tree_live : row >= p.n_rows_all) {
#pragma unroll
                for (int e = 0; e < 32; ++e) s[e] = kNegInf;
            } else if (kTree) {
                const int d = ts - tree_base;
                const uint64_t pre = d >= 0 ? 0ull : (d <= -64 ? ~0ull : (1ull << -d) - 1ull);
                const uint64_t live = span_L - ts >= 64 ? ~0ull : (1ull << max(span_L - ts, 0)) - 1ull;
                const uint64_t tr = d >= 64 ? 0ull : (d >= 0 ? anc >> d : (d <= -64 ? 0ull : anc << -d));
                const uint32_t vis = (uint32_t)(((pre | tr) & live) >> kb);
#pragma unroll
                for (int e = 0; e < 32; ++e)
                    if (!((vis >> e) & 1u)) s[e] = kNegInf;
            } else {
                const int lim_t = lim - ts - kb;   // keys e < lim_t of this half are visible
                if (lim_t < 32) {
#pragma unroll
                    for (int e = 0; e < 32; ++e)
                        if (e >= lim_t) s[e] = kNegInf;
                }
            }
            // three-input maxima in independent chains: exact in any order
            float m4[4];
#pragma unroll
            for (int j = 0; j < 4; ++j) m4[j] = fmax3(s[j], s[j + 4], s[j + 8]);
#pragma unroll
            for (int e = 12; e < 28; e += 8)
#pragma unroll
                for (int j = 0; j < 4; ++j) m4[j] = fmax3(m4[j], s[e + j], s[e + 4 + j]);
#pragma unroll
            for (int j = 0; j < 4; ++j) m4[j] = fmaxf(m4[j], s[28 + j]);
            const float mh = fmaxf(fmax3(m4[0], m4[1], m4[2]), m4[3]);
            const float mt = fmaxf(mh, __shfl_xor_sync(0xffffffffu, mh, 16));   // the tile's row maximum
            // ---- running max, lazily: O is rescaled only for a growth > 2^8
            float alpha = 1.f;
            if (mt != kNegInf && (m_run == kNegInf || (mt - m_run) * c > kTcRescale)) {
                alpha = m_run == kNegInf ? 0.f : ex2((m_run - mt) * c);
                m_run = mt;
            }
            // ---- P = 2^((s - m) c - 64) (the row sum carries the same 2^-64),
            // as the sum of two bf16 terms; pairs of keys in packed fp32
            const float neg = m_run == kNegInf ? 0.f : -m_run * c - kPShift;
            const uint64_t c2 = f2_pack(c, c), n2 = f2_pack(neg, neg);
            uint64_t r2[4] = {0ull, 0ull, 0ull, 0ull};   // +0.0f pairs
            uint32_t ph[16], pl[16];
#pragma unroll
            for (int e = 0; e < 16; ++e) {
                float x0, x1;
                f2_unpack(f2_fma(f2_pack(s[2 * e], s[2 * e + 1]), c2, n2), x0, x1);
                const float p0 = ex2(x0), p1 = ex2(x1);
                const uint64_t pp = f2_pack(p0, p1);
                r2[e & 3] = f2_add(r2[e & 3], pp);
                const uint32_t hi = pack_bf16x2(p0, p1);
                float d0, d1;
                f2_unpack(f2_sub(pp, f2_pack(__uint_as_float(hi << 16), __uint_as_float(hi & 0xffff0000u))), d0, d1);
                ph[e] = hi;
                pl[e] = pack_bf16x2(d0, d1);
            }
            {
                float a0, a1, b0, b1;
                f2_unpack(f2_add(r2[0], r2[1]), a0, a1);
                f2_unpack(f2_add(r2[2], r2[3]), b0, b1);
                l_part = l_part * alpha + ((a0 + a1) + (b0 + b1));
            }
            // ---- a rescale of O (this warp's 16 rows, all 128 dims) waits for
            // PV_{t-1}; the first tile of a piece needs none (its PV
            // overwrites O).  o_ready[b] completes once per tile of S buffer
            // b: PV_{t-5} is complete (QK_t waited for PV_{t-4}) and PV_{t+3}
            // is not issued, so the parity of PV_{t-1}'s phase is unambiguous.
            const unsigned need = __ballot_sync(0xffffffffu, alpha != 1.f && cur.t != seg_t0);
            if (need) {
                const int tp = t - 1;
                if (!tc_wait(&o_ready[tp % kTcSBuf], (uint32_t)(tp / kTcSBuf) & 1, &s_dead, p.status)) break;
                tc_fence_after();
#pragma unroll 1
                for (int c0 = 0; c0 < 64; c0 += 32) {
                    float o[32];
                    tc_ld16x2_32<64>(t_row + kTcOCol + c0, o);
                    uint32_t r[32];
#pragma unroll
                    for (int i = 0; i < 32; ++i) r[i] = __float_as_uint(o[i] * alpha);
                    tc_st16x2_32<64>(t_row + kTcOCol + c0, r);
                }
            }
            // P as bf16 pairs: keys kb..kb+31 are columns kb/2 .. kb/2+15 of
            // the buffer (hi) and 32 + kb/2 .. (lo); the S columns there were
            // loaded by this warp (the same lanes) before
            tc_st16x2_16<16>(t_row + sb * 64, ph);
            tc_st16x2_16<16>(t_row + sb * 64 + 32, pl);
            tc_wait_st();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&p_full[sb]);

            if (!piece_end) {
                advance(cur, s_len, nb, p.n_vh);
                continue;
            }
            // ---- end of a span piece: O after its last PV (every earlier MMA
            // completes before that commit), then written: thread t dims
            // 0..63 of its row, thread t+16 dims 64..127; the row sum is the
            // two threads' sum (the same in both: addition commutes)
            if (!tc_wait(&o_ready[sb], (uint32_t)(t / kTcSBuf) & 1, &s_dead, p.status)) break;
            tc_fence_after();
            const float l_run = l_part + __shfl_xor_sync(0xffffffffu, l_part, 16);
            const int bg = p.b_base + cur.b;
            const int head = cur.h / p.n_rb;
            const bool complete = seg_t0 == 0 && cur.t + 1 == cur.T;
            const size_t slot = 2 * (size_t)cta + (first_seg ? 0 : 1);
            const bool live_row = kTree ? tree_live : row < p.n_rows_all;
            // normalised output; a partial is the piece's own normalised output
            // (the merge takes a convex combination)
            const float inv = l_run > 0.f ? 1.f / l_run : 0.f;
#pragma unroll 1
            for (int c0 = 0; c0 < 64; c0 += 32) {
                float o[32];
                tc_ld16x2_32<64>(t_row + kTcOCol + c0, o);
                if (!live_row) continue;
                const int dim0 = kh * 64 + c0;
                if (complete) {
                    const int qr = kTree ? qrow : row;
                    const int i = qr / p.G, gi = qr % p.G;
                    __nv_bfloat16* dst =
                        p.out + (((size_t)bg * p.R + i) * p.Hq + (size_t)head * p.G + gi) * kD + dim0;
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        uint4 v;
                        v.x = pack_bf16x2(o[8 * q + 0] * inv, o[8 * q + 1] * inv);
                        v.y = pack_bf16x2(o[8 * q + 2] * inv, o[8 * q + 3] * inv);
                        v.z = pack_bf16x2(o[8 * q + 4] * inv, o[8 * q + 5] * inv);
                        v.w = pack_bf16x2(o[8 * q + 6] * inv, o[8 * q + 7] * inv);
                        *reinterpret_cast<uint4*>(dst + 8 * q) = v;
                    }
                } else {
                    float* dst = p.part_o + (slot * p.n_rows + row) * kD + dim0;
#pragma unroll
                    for (int q = 0; q < 8; ++q)
                        *reinterpret_cast<float4*>(dst + 4 * q) =
                            make_float4(o[4 * q] * inv, o[4 * q + 1] * inv, o[4 * q + 2] * inv, o[4 * q + 3] * inv);
                }
            }
            if (live_row && !complete && kh == 0)
                p.part_ml[slot * p.n_rows + row] = make_float2(m_run == kNegInf ? kNegInf : m_run * c, l_run);
            if (!complete && threadIdx.x == 128) p.part_span[slot] = cur.b * p.n_vh + cur.h;
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(o_free);
            if (t + 1 < n_tiles) {
                advance(cur, s_len, nb, p.n_vh);
                seg_t0 = cur.t;
                first_seg = false;
                begin_span(cur);
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == kTcQkWarp)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "n"(kTcTmemCols) : "memory");
}
