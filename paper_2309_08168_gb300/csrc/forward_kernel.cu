// forward_kernel.cu - one decoder forward (draft step, verification, prefill
// chunk) as a single persistent, cooperative kernel.
//
// Batch-1 decoding streams every weight byte once per forward and is bound by
// HBM (Sec. 3.1).  At LLaMA-2 7B scale a projection takes 5-30 us at full
// bandwidth, so per-kernel ramp-up and drain would cost a large fraction of
// the step.  Instead one CTA per SM walks the forward's op list
//     embed -> [QKV -> attention -> O] -> [gate/up -> down] -> ... -> lm_head
// (sublayers in the skip set z are simply absent from the draft's list,
// Sec. 3.2 / 3.3) with a grid barrier between dependent ops.  Once a CTA has
// arrived at a barrier it requests the weights of its first units of the next
// projection (they do not depend on the previous op), so the barrier's
// latency overlaps HBM streaming.  Every wait is bounded: a barrier that does
// not complete within ~2 s records an error code and the CTAs return.
//
// Projections (all of them: q/k/v + RoPE + KV write, output and down with the
// residual add, gate/up with SwiGLU, lm_head) run on the 5th-generation
// tensor cores: work unit = 128-row tile x 128-wide k chunk (32 KB of
// weights), each CTA owns an equal contiguous range of units in tile-major
// order, streamed by TMA (128-byte swizzle) through a 5-stage ring; one
// thread of the MMA warp issues tcgen05.mma kind::f16 per unit (M = 128 weight
// rows, N = the activation rows as bf16 hi + lo planes, ~16 mantissa bits of
// the fp32 activations) into a TMEM accumulator and releases the stage with
// tcgen05.commit; the consumer warps read a finished tile segment from TMEM
// (tcgen05.ld) while the next segment accumulates in the other accumulator.
// A tile split over several CTAs is summed in segment order by the CTA
// holding its first chunks; the others store their partials tagged with the
// op (value and tag in one 64-bit word), so they neither fence nor signal,
// and the finaliser polls the words themselves.
// RMSNorm is folded in: the producer of the residual stream writes the planes
// of h * g_next and per-128-column sums of h^2, the consumer scales row m by
// rsqrt(mean(h^2) + eps) in its epilogue (W (h g r) = r W (h g)).
//
// Attention: items = (KV head, group of 16 query vectors, absolute
// 128-position segment); the partial softmax of a row over a segment depends
// only on the row and the segment.  After a grid barrier every CTA combines a share
// of the (KV head, query vector) outputs over their segments in segment
// order.
//
// Coherence: L1 is not coherent across SMs within one launch, so every load of
// data another CTA wrote during this launch goes through L2 (cp.async.cg,
// ld.global.cg); stores are write-through.
//
// Batch invariance (greedy self-speculative output must equal autoregressive
// output bit for bit, Sec. 1 / App. G.2): row m's result depends only on row
// m - the MMA's output columns are independent (an input row is one column of
// D whatever N is), unit partitions and combine orders depend on the shapes
// and the grid only, epilogues are per row, attention segments are absolute
// positions.
#include "ssd_internal.cuh"

namespace ssd {
namespace {

constexpr unsigned long long kBarrierTimeoutNs = 2000000000ull;
// A wait reads the shared error flag only after this long (20 us): until
// then each poll is a single load.
constexpr unsigned long long kErrPollAfterNs = 20000ull;
// 8 consumer warps (epilogues, attention, embedding) + 1 producer warp (TMA)
// + 1 MMA warp (tcgen05.mma issue, TMEM allocation)
constexpr int kConsumers = 256;
constexpr int kFwdThreads = kConsumers + 64;

// barrier among the consumer warps only (the producer keeps streaming)
__device__ __forceinline__ void consumer_sync() { asm volatile("bar.sync 1, 256;" ::: "memory"); }


__device__ __forceinline__ unsigned long long globaltimer() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

__device__ __forceinline__ unsigned ld_acquire(const unsigned* p) {
    unsigned v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

// Grid-wide barrier for a cooperative launch (all CTAs co-resident), in two
// halves so that a CTA can do work that publishes nothing between them.  The
// counter only grows during a launch; `target` = gridDim.x * (barrier index).
// grid_arrive (one thread, after a CTA barrier that orders the CTA's stores
// before it): the release of the arrival publishes those stores and needs no
// reply.  grid_wait (the same thread): acquire - later loads, ordered after it
// by a CTA barrier, see the others' stores.  Returns false (and records
// SSD_DEV_ERR_TIMEOUT) if the others do not arrive within limit_ns, or if
// another CTA already gave up.
__device__ __forceinline__ void grid_arrive(unsigned* bar) {
    asm volatile("red.release.gpu.global.add.u32 [%0], 1;" ::"l"(bar) : "memory");
}
// Each poll is one L2 round trip: the error flag (another CTA gave up) is
// read only once the wait has lasted kErrPollAfterNs, so that a second load
// does not double the poll period of ordinary waits.
__device__ bool grid_wait(unsigned* bar, unsigned target, int* err, unsigned long long limit_ns) {
    const unsigned long long t0 = globaltimer();
    while (ld_acquire(bar) < target) {
        const unsigned long long dt = globaltimer() - t0;
        if (dt > kErrPollAfterNs) {
            if (*(volatile int*)err) return false;
            if (dt > limit_ns) {
                atomicCAS(err, 0, kDevErrTimeout);
                return false;
            }
        }
    }
    return true;
}

// Split-K partials: a float and the tag of the op that wrote it (forward
// sequence number << 10 | op index) in one 64-bit word, written and read as
// single 64-bit accesses.
__device__ __forceinline__ unsigned long long tagged(unsigned tag, float v) {
    return ((unsigned long long)tag << 32) | __float_as_uint(v);
}
__device__ __forceinline__ unsigned tag_of(unsigned long long w) { return (unsigned)(w >> 32); }
__device__ __forceinline__ float value_of(unsigned long long w) { return __uint_as_float((unsigned)w); }
__device__ __forceinline__ void st_relaxed_u64(unsigned long long* p, unsigned long long v) {
    asm volatile("st.relaxed.gpu.global.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}
__device__ __forceinline__ unsigned long long ld_relaxed_u64(const unsigned long long* p) {
    unsigned long long v;
    asm volatile("ld.relaxed.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ int unit_owner(long long u, long long U, long long G) {
    return (int)(((u + 1) * G + U - 1) / U - 1);
}

// An op's units are split over the first min(U, grid) CTAs, so every CTA that
// takes part owns at least one unit and the owners of consecutive units are
// consecutive CTAs (the segment arithmetic of the projection op relies on it).
__device__ __forceinline__ long long op_ctas(long long U) { return U < gridDim.x ? U : (long long)gridDim.x; }

__device__ __forceinline__ void my_units(long long U, int* u_begin, int* n_my) {
    const long long G = op_ctas(U), b = blockIdx.x;
    if (b >= G) { *u_begin = 0; *n_my = 0; return; }
    *u_begin = (int)(b * U / G);
    *n_my = (int)((b + 1) * U / G) - *u_begin;
}

__device__ __forceinline__ bool is_gemm(int type) { return type >= OP_QKV && type <= OP_LOGITS && type != OP_ATTN; }

__device__ __forceinline__ int epi_of(int type) {
    return type == OP_QKV ? EPI_QKV : type == OP_RESID ? EPI_RESID : type == OP_SWIGLU ? EPI_SWIGLU : EPI_LOGITS;
}

// ---------------------------------------------------------------------------
// TMA + mbarrier helpers
// ---------------------------------------------------------------------------
constexpr unsigned long long kWaitTimeoutNs = 2000000000ull;

__device__ __forceinline__ void mbar_init(uint64_t* bar, unsigned count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
// adds expected bytes without arriving (the weights of a unit, requested early)
__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, unsigned bytes) {
    asm volatile("mbarrier.expect_tx.relaxed.cta.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
                 : "memory");
}
// plain arrival (a consumer warp releasing a stage)
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
// arrives (count 1) and adds expected bytes (the activations of the unit)
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, unsigned bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, unsigned parity) {
    unsigned ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}\n"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}
// bounded wait: false after kWaitTimeoutNs (timeout recorded), or once it has
// waited kErrPollAfterNs while another thread has already recorded an error
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, unsigned parity, int* err) {
    if (mbar_try_wait(bar, parity)) return true;
    const unsigned long long t0 = globaltimer();
    while (!mbar_try_wait(bar, parity)) {
        const unsigned long long dt = globaltimer() - t0;
        if (dt > kErrPollAfterNs && *(volatile int*)err) return false;
        if (dt > kWaitTimeoutNs) {
            atomicCAS(err, 0, kDevErrTimeout);
            return false;
        }
    }
    return true;
}
// 2D tiled TMA load of one box into shared memory, completing on `bar`.  x is
// the innermost (k) coordinate; every x used here is a multiple of 64
// elements (128 bytes), so the 16-byte rule for x * element size holds.
__device__ __forceinline__ void tma_load_2d(void* dst, const void* tmap, int x, int y, uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];"
        ::"r"(smem_u32(dst)), "l"(tmap), "r"(x), "r"(y), "r"(smem_u32(bar))
        : "memory");
}

__device__ __forceinline__ void tma_load_3d(void* dst, const void* tmap, int x, int y, int z, uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], [%5];"
        ::"r"(smem_u32(dst)), "l"(tmap), "r"(x), "r"(y), "r"(z), "r"(smem_u32(bar))
        : "memory");
}

// brings a tensor map descriptor (global memory) into the descriptor cache
__device__ __forceinline__ void prefetch_tmap(const void* tmap) {
    asm volatile("prefetch.tensormap [%0];" ::"l"(tmap) : "memory");
}

// fp16 tensor-core MMA (attention: K / V are fp16) and 8x8 matrix loads
__device__ __forceinline__ void mma_f16_16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                              uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 "
        "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};\n"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}
__device__ __forceinline__ void ldsm_x4(uint32_t (&r)[4], const void* p) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(smem_u32(p)));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t (&r)[4], const void* p) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(smem_u32(p)));
}

// ---------------------------------------------------------------------------
// projection op: TMA ring -> tcgen05.mma -> TMEM -> epilogue
// ---------------------------------------------------------------------------
// Work unit = a 128-row tile x 128-wide k chunk of a weight matrix (32 KB).
// Stage layout (1 KB aligned; TMA writes the 128-byte swizzle, which is the
// canonical K-major operand layout of tcgen05.mma: row r of a 64-wide k box
// at r * 128 bytes, 8-row groups 1024 bytes apart):
//   weights : k box kb (k0 + 64 kb ..) of the tile's 128 rows at kb * 16 KB
//             (SwiGLU tiles: rows 0-63 gate, 64-127 up, of features 64 t ..)
//   inputs  : k box kb at 32 KB + kb * XKB; rows p = plane * R + row (the R
//             hi rows, then the R lo rows); rows 2R .. NP-1 are not written and
//             only feed accumulator columns that nobody reads
// One thread of the MMA warp issues, per unit, eight tcgen05.mma kind::f16
// (bf16 x bf16 -> fp32; M = 128 weight rows, N = NP input rows, K = 16) into
// one of two TMEM accumulators (one per tile segment, so the consumers read a
// finished segment while the next one accumulates) and releases the stage
// with tcgen05.commit.  The consumer warps only run the segment epilogue.
//
// attention: 64-position chunks per segment (one ring stage each).  Segments
// are absolute, so a row's softmax partials do not depend on M; two chunks
// per segment balance ~150 CTAs well at LLaMA-2 KV-head counts and contexts
// and keep the final combine short.
constexpr int kAttnSegChunks = 2;

// Attention unit in a stage: K rows of the 64-position chunk at 0 (dims 0-63,
// then 64-127 at 8 KB), V rows at 16 KB; position t, 16-byte chunk c of a
// 64-dim box at box + t * 128 + ((c ^ (t & 7)) << 4).
// After the ring: the consumers' scratch - the finished segment of a
// projection, or (same bytes: one op at a time) q / scores of attention.
// index of the input-plane tensor map of R rows
__host__ __device__ constexpr int plane_cls(int R) {
    return R == 1 ? 0 : (R == 4 ? 1 : (R == 8 ? 2 : (R == 12 ? 3 : 4)));
}

template <int R>
struct GemmSmem {
    static constexpr int NP = R <= 8 ? 16 : 32;     // MMA N: input rows (hi + lo), padded
    static constexpr int WB = kFTile * kFKC * 2;    // 32 KB of weights per unit
    static constexpr int XKB = NP * 128;            // input bytes per 64-wide k box
    static constexpr int STAGE = WB + 2 * XKB;
    static constexpr int S = 5;                     // ring depth (160 KB of weights in flight)
    static constexpr int VG = 16;  // attention: query vectors per item (one MMA M / N tile)
    static constexpr int YS = S * STAGE;            // [128][16] floats: the finished segment
    // attention scratch: q hi / lo (fp16, rows padded by 16 bytes), scores
    // (fp32), P hi / lo (fp16, padded rows)
    static constexpr int QST = 128 + 8, PST = kAttnSegChunks * kAttnChunk + 8;  // halves per row
    static constexpr int ATT = S * STAGE;
    static constexpr int ATT_SC = ATT + 2 * VG * QST * 2;
    static constexpr int ATT_P = ATT_SC + 2 * (kConsumers / 32) * VG * 4;  // per-warp maxima and sums
    static constexpr int SCRATCH_GEMM = kFTile * 16 * 4;
    static constexpr int SCRATCH_ATT = ATT_P + 2 * VG * PST * 2 - ATT;
    static constexpr size_t BYTES =
        1024 + (size_t)S * STAGE + (SCRATCH_GEMM > SCRATCH_ATT ? SCRATCH_GEMM : SCRATCH_ATT);
    static_assert(STAGE >= 2 * kAttnChunk * 128 * 2, "a stage holds the K and V rows of one 64-position chunk");
    static_assert(BYTES + 4096 <= 232448, "dynamic + static shared memory within the per-CTA limit");
};

// ---------------------------------------------------------------------------
// tcgen05 helpers
// ---------------------------------------------------------------------------
constexpr int kTmemCols = 64;  // two accumulators of up to 32 fp32 columns

// shared-memory matrix descriptor: K-major, 128-byte swizzle, 8-row groups
// 1024 bytes apart; the start address may sit 32 / 64 / 96 bytes into a
// swizzle row (k steps of 16 bf16)
__device__ __forceinline__ uint64_t umma_desc(uint32_t saddr) {
    uint64_t d = (uint64_t)((saddr & 0x3FFFFu) >> 4);  // start address
    d |= (uint64_t)1 << 16;                           // leading byte offset (unused with this swizzle)
    d |= (uint64_t)(1024 >> 4) << 32;                 // stride byte offset
    d |= (uint64_t)1 << 46;                           // descriptor version
    d |= (uint64_t)2 << 61;                           // 128-byte swizzle
    return d;
}
// instruction descriptor: kind::f16, A = B = bf16, D = fp32, both K-major,
// M = 128, N = np
__host__ __device__ constexpr uint32_t umma_idesc(int np) {
    return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(np >> 3) << 17) | ((uint32_t)(kFTile >> 4) << 24);
}
__device__ __forceinline__ void umma(uint32_t tmem_d, uint64_t ad, uint64_t bd, uint32_t idesc, uint32_t acc) {
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
        " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n"
        ::"r"(tmem_d), "l"(ad), "l"(bd), "r"(idesc), "r"(acc)
        : "memory");
}
// the mbarrier completes once every tcgen05 op this thread issued so far is done
__device__ __forceinline__ void umma_commit(uint64_t* bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(bar))
                 : "memory");
}
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// NP consecutive fp32 columns of this thread's TMEM lane
template <int NP>
__device__ __forceinline__ void tmem_ld(uint32_t taddr, float (&v)[NP]);
template <>
__device__ __forceinline__ void tmem_ld<16>(uint32_t taddr, float (&v)[16]) {
    uint32_t r[16];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}
template <>
__device__ __forceinline__ void tmem_ld<32>(uint32_t taddr, float (&v)[32]) {
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

template <>
__device__ __forceinline__ void tmem_ld<24>(uint32_t taddr, float (&v)[24]) {
    uint32_t r[24];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
                 : "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]),
                   "=r"(r[23])
                 : "r"(taddr + 16u));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 24; ++i) v[i] = __uint_as_float(r[i]);
}

// Weight rows of tile t: one 128-row box (matrix s0 from row r0), or for
// SwiGLU two 64-row boxes (the gate and the up rows of features 64 t ..).
// The q / k / v widths are whole tiles, so a q / k tile is 128 / head_dim
// whole heads in natural order and holds every RoPE pair (j, j + hd / 2).
struct TileSrc {
    int s0, r0, s1, r1;  // s1 < 0: one box
};
__device__ __forceinline__ TileSrc tile_src(const GemmArgs& a, int epi, int tile) {
    if (epi == EPI_SWIGLU) return {0, tile * 64, 1, tile * 64};
    if (epi == EPI_QKV) {
        const int qt = a.n_heads * a.head_dim / kFTile, kt = a.n_kv_heads * a.head_dim / kFTile;
        if (tile < qt) return {0, tile * kFTile, -1, 0};
        if (tile < qt + kt) return {1, (tile - qt) * kFTile, -1, 0};
        return {2, (tile - qt - kt) * kFTile, -1, 0};
    }
    return {0, tile * kFTile, -1, 0};
}

// weights of unit u into a stage (one thread): expect_tx without arriving.
// Always a full 128 x 128 tile of bytes (rows / columns out of range are
// delivered as zeros and counted).  Every x used here is a multiple of 64
// elements (128 bytes), so the 16-byte rule for x * element size holds.
template <int R>
__device__ __forceinline__ void tma_weights(const GemmArgs& a, int epi, int u, unsigned char* st, uint64_t* bar) {
    const int tile = u / a.n_chunks, k0 = (u - tile * a.n_chunks) * kFKC;
    const TileSrc ts = tile_src(a, epi, tile);
    mbar_expect_tx(bar, (unsigned)GemmSmem<R>::WB);
#pragma unroll
    for (int kb = 0; kb < 2; ++kb) {
        tma_load_2d(st + kb * 16384, a.tm_w[ts.s0], k0 + kb * 64, ts.r0, bar);
        if (ts.s1 >= 0) tma_load_2d(st + kb * 16384 + 8192, a.tm_w[ts.s1], k0 + kb * 64, ts.r1, bar);
    }
}

// input planes of unit u into a stage (one thread): arrive + expect_tx
template <int R>
__device__ __forceinline__ void tma_inputs(const GemmArgs& a, int u, unsigned char* st, uint64_t* bar) {
    using L = GemmSmem<R>;
    const int k0 = (u % a.n_chunks) * kFKC;
    const int cls = plane_cls(R);
    mbar_arrive_expect_tx(bar, 2u * 2u * (unsigned)R * 128u);
#pragma unroll
    for (int kb = 0; kb < 2; ++kb) tma_load_3d(st + L::WB + kb * L::XKB, a.tm_x[cls], k0 + kb * 64, 0, 0, bar);
}

// Pipeline state, carried across ops; every thread keeps its own copy and
// flips the bits of the waits it takes part in (or, for ring positions whose
// waits another role took, the same bits arithmetically).
//   pphase bit s : parity of the next "empty" completion of stage s (producer)
//   cphase bit s : parity of the next "full" completion of stage s (MMA thread
//                  in projections, consumers in attention)
//   afull bit b  : parity of the next completion of accumulator b (consumers)
//   aempty bit b : parity of the next release of accumulator b (MMA thread)
//   ab           : accumulator of the next tile segment
struct Pipe {
    uint64_t* full;     // [stages] TMA completion (count 1: the producer's arrive)
    uint64_t* empty;    // [stages] stage released (count 1: tcgen05.commit, or consumer thread 0)
    uint64_t* acc_full;   // [2] accumulator complete (tcgen05.commit)
    uint64_t* acc_empty;  // [2] accumulator read by the consumers (count 8: one arrival per consumer warp)
    uint32_t tmem;      // TMEM base address (two accumulators of kTmemCols / 2 columns)
    unsigned pphase;
    unsigned cphase;
    unsigned afull;
    unsigned aempty;
    int ab;
};

// flips the full-barrier parity bits of n consecutive ring positions from 0
template <int S>
__device__ __forceinline__ void advance_full(Pipe& pp, int n) {
#pragma unroll
    for (int s = 0; s < S; ++s)
        if (((n / S) + (s < n % S ? 1 : 0)) & 1) pp.cphase ^= 1u << s;
}

// Producer: requests the weights of this CTA's first S units of a projection
// before the grid barrier (they do not depend on the previous op).
// n_pre: how many (at most the ring's depth) are requested.
template <int R>
__device__ bool gemm_prefetch(const GemmArgs& a, int epi, unsigned char* smem, Pipe& pp, int* err, int n_pre) {
    constexpr int S = GemmSmem<R>::S;
    int u_begin, n_my;
    my_units(a.n_units, &u_begin, &n_my);
    bool ok = true;
    if (threadIdx.x == kConsumers) {
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        prefetch_tmap(a.tm_x[plane_cls(R)]);
        for (int s = 0; s < S && s < n_pre && s < n_my && ok; ++s) {
            ok = mbar_wait(pp.empty + s, (pp.pphase >> s) & 1u, err);
            if (!ok) break;
            pp.pphase ^= 1u << s;
            tma_weights<R>(a, epi, u_begin + s, smem + s * GemmSmem<R>::STAGE, pp.full + s);
        }
    }
    return ok;
}

// Returns false if a wait timed out (error recorded).  Three roles:
//   producer (one thread of warp 8) streams this CTA's units through the ring;
//   MMA issuer (one thread of warp 9) runs tcgen05.mma per unit into the
//     accumulator of the unit's tile segment;
//   consumers (warps 0-7), per finished segment: TMEM -> hi + lo summed ->
//     split-K exchange -> epilogue (contributors and residual finalisers
//     per warp from registers, the other finalisers through shared memory).
// ut: nullptr, or [64][4] timestamps of this CTA's first units (producer
// issue, MMAs issued, 0, segment flush done); ct: nullptr, or this CTA's op
// stamps (FwdParams::trace) - profiling aids.
template <int R>
__device__ bool gemm_op(const GemmArgs& a, int epi, int M, int pos0, int n_pre, unsigned char* smem,
                        float* r_s, Pipe& pp, unsigned tag, int* err, unsigned long long* ut,
                        unsigned long long* ct) {
    using L = GemmSmem<R>;
    constexpr int S = L::S, NP = L::NP;
    float* ys = reinterpret_cast<float*>(smem + L::YS);  // [128][16]
    bool ok = true;

    const long long U = a.n_units, G = op_ctas(U);
    const int b = blockIdx.x;
    int u_begin, n_my;
    my_units(U, &u_begin, &n_my);

    if (threadIdx.x >= kConsumers && threadIdx.x < kConsumers + 32) {  // producer warp
        if (threadIdx.x != kConsumers) return true;
        if (ut) ut[2] = globaltimer();
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        asm volatile("fence.proxy.async.global;" ::: "memory");  // inputs written by the previous op
        for (int i = 0; i < n_my; ++i) {
            const int s = i % S;
            unsigned char* st = smem + s * L::STAGE;
            if (ut && i < 64) ut[i * 4 + 0] = globaltimer();
            if (i >= n_pre) {  // (the first n_pre units' weights were requested before the op)
                if (!mbar_wait(pp.empty + s, (pp.pphase >> s) & 1u, err)) return false;
                pp.pphase ^= 1u << s;
                tma_weights<R>(a, epi, u_begin + i, st, pp.full + s);
            }
            tma_inputs<R>(a, u_begin + i, st, pp.full + s);
        }
        return true;
    }

    if (threadIdx.x >= kConsumers + 32) {  // MMA warp: one elected thread issues
        if (threadIdx.x != kConsumers + 32) return true;
        constexpr uint32_t idesc = umma_idesc(NP);
        for (int i = 0; i < n_my; ++i) {
            const int u = u_begin + i;
            const int chunk = u % a.n_chunks;
            const bool first = i == 0 || chunk == 0;
            const bool last = i == n_my - 1 || chunk == a.n_chunks - 1;
            const int ab = pp.ab;
            if (first) {  // the consumers have read this accumulator's previous segment
                if (!mbar_wait(pp.acc_empty + ab, (pp.aempty >> ab) & 1u, err)) return false;
                pp.aempty ^= 1u << ab;
            }
            const int s = i % S;
            if (!mbar_wait(pp.full + s, (pp.cphase >> s) & 1u, err)) return false;
            pp.cphase ^= 1u << s;
            tc_fence_after();
            const uint32_t st = smem_u32(smem + s * L::STAGE);
            const uint32_t d = pp.tmem + (uint32_t)(ab * (kTmemCols / 2));
#pragma unroll
            for (int kb = 0; kb < 2; ++kb)
#pragma unroll
                for (int ks = 0; ks < 4; ++ks)
                    umma(d, umma_desc(st + kb * 16384 + ks * 32), umma_desc(st + L::WB + kb * L::XKB + ks * 32),
                         idesc, (first && kb == 0 && ks == 0) ? 0u : 1u);
            umma_commit(pp.empty + s);  // the stage is free once these MMAs have read it
            if (ut && i < 64) ut[i * 4 + 1] = globaltimer();
            if (last) {
                umma_commit(pp.acc_full + ab);
                pp.ab ^= 1;
            }
        }
        return true;
    }

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // 1 / rms of each input row from the previous op's per-tile sums of
    // squares (fixed order for every M: lane-strided sums, then a shuffle tree)
    for (int m = warp; m < M; m += kConsumers / 32) {
        float r = 1.f;
        if (a.ss_in) {
            float sum = 0.f;
            for (int t = lane; t < a.ss_in_tiles; t += 32) sum += __ldcg(a.ss_in + m * a.ss_in_tiles + t);
            sum = warp_sum(sum);
            r = rsqrtf(sum * a.inv_dim + a.eps);
        }
        if (lane == 0) r_s[m] = r;
    }
    // the MMA thread took the full-barrier waits of these ring positions
    advance_full<S>(pp, n_my);

    for (int i = 0; i < n_my; ++i) {
        const int u = u_begin + i;
        const int tile = u / a.n_chunks, chunk = u - tile * a.n_chunks;
        if (threadIdx.x == 0 && ct && i == n_my - 1) ct[6] = (unsigned long long)n_my;
        if (!(i == n_my - 1 || chunk == a.n_chunks - 1)) continue;

        // this CTA's segment of the tile is complete (or completing): its
        // accumulator holds W x_hi in columns 0..R-1 and W x_lo in columns
        // R..2R-1.  Split-K: the CTA holding the tile's first chunks (its
        // segment ends last, at the end of that CTA's range) finalises; the
        // others store their partial and move on.  Each value travels with the
        // op's tag in one 64-bit word, so the finaliser needs no flag and no
        // fence: it reads each word until the tag is this op's.
        const int ab = pp.ab;
        const long long u_first = (long long)tile * a.n_chunks;
        const int seg0 = unit_owner(u_first, U, G);
        const int nseg = unit_owner(u_first + a.n_chunks - 1, U, G) - seg0 + 1;
        constexpr size_t kSlot = (size_t)kMaxRows * kFTile;
        unsigned long long* slots =
            reinterpret_cast<unsigned long long*>(a.partial) + (size_t)tile * a.n_chunks * kSlot;
        const bool contributor = nseg > 1 && b != seg0;

        if (contributor || epi == EPI_RESID) {
            // Direct path: every consumer warp reads its own TMEM rows - warp w
            // holds tile row rr = 32 (w % 4) + lane for the input rows m = w / 4,
            // w / 4 + 2, ... - so nothing goes through shared memory and no CTA
            // barrier precedes the stores.  A residual finaliser first fetches
            // the residual rows, the gains and the other segments' partials
            // while its own accumulator completes; its sum is own + (p_1 + p_2
            // + ...), the partials added in segment order.
            constexpr int HM = (R + 1) / 2;
            const int q4 = warp & 3, par = warp >> 2, rr = q4 * 32 + lane;
            const int n = tile * kFTile + rr;
            float hp[HM], ps[HM];
            const float gp = (!contributor && n < a.N && a.g_next) ? __bfloat162float(a.g_next[n]) : 0.f;
#pragma unroll
            for (int k = 0; k < HM; ++k) {
                const int m = par + 2 * k;
                hp[k] = (!contributor && m < M && n < a.N) ? __ldcg(a.out_f32 + (size_t)m * a.ldo + n) : 0.f;
                ps[k] = 0.f;
            }
            if (!contributor && nseg > 1) {
                constexpr int QB = R <= 8 ? 4 : R <= 12 ? 2 : 1;  // segments per batch (registers: QB * HM words)
                for (int sg0 = 1; sg0 < nseg; sg0 += QB) {
                    unsigned long long w[QB][HM];
#pragma unroll
                    for (int q = 0; q < QB; ++q)
#pragma unroll
                        for (int k = 0; k < HM; ++k)
                            if (sg0 + q < nseg && par + 2 * k < M)
                                w[q][k] = ld_relaxed_u64(slots + (size_t)(sg0 + q) * kSlot + (par + 2 * k) * kFTile + rr);
                    // words that do not carry this op's tag yet (their CTA has
                    // not published) are re-read together, not one at a time
                    unsigned long long t_wait = 0;
                    for (;;) {
                        bool ready = true;
#pragma unroll
                        for (int q = 0; q < QB; ++q)
#pragma unroll
                            for (int k = 0; k < HM; ++k)
                                if (sg0 + q < nseg && par + 2 * k < M && tag_of(w[q][k]) != tag) ready = false;
                        if (ready) break;
                        const unsigned long long now = globaltimer();
                        if (t_wait == 0) t_wait = now;
                        if (now - t_wait > kErrPollAfterNs) {
                            if (*(volatile int*)err) { ok = false; break; }
                            if (now - t_wait > kBarrierTimeoutNs) {
                                atomicCAS(err, 0, kDevErrTimeout);
                                ok = false;
                                break;
                            }
                        }
#pragma unroll
                        for (int q = 0; q < QB; ++q)
#pragma unroll
                            for (int k = 0; k < HM; ++k)
                                if (sg0 + q < nseg && par + 2 * k < M && tag_of(w[q][k]) != tag)
                                    w[q][k] = ld_relaxed_u64(slots + (size_t)(sg0 + q) * kSlot + (par + 2 * k) * kFTile + rr);
                    }
#pragma unroll
                    for (int q = 0; q < QB; ++q)
#pragma unroll
                        for (int k = 0; k < HM; ++k)
                            if (sg0 + q < nseg && par + 2 * k < M) ps[k] += value_of(w[q][k]);
                }
            }
            ok = mbar_wait(pp.acc_full + ab, (pp.afull >> ab) & 1u, err) && ok;
            pp.afull ^= 1u << ab;
            pp.ab ^= 1;
            tc_fence_after();
            if (threadIdx.x == 0 && ct) ct[2] = globaltimer();
            constexpr int NC = R == 12 ? 24 : NP;  // the 2R accumulator columns, rounded up
            float v[NC];
            tmem_ld<NC>(pp.tmem + (uint32_t)(ab * (kTmemCols / 2)) + ((uint32_t)(q4 * 32) << 16), v);
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(pp.acc_empty + ab);  // this warp is done with the accumulator
            float own[HM];
#pragma unroll
            for (int k = 0; k < HM; ++k) {  // input row m = par + 2k: columns m (hi) and R + m (lo)
                const float hi = par ? v[(2 * k + 1) < NC ? 2 * k + 1 : 0] : v[2 * k];
                const float lo = par ? v[(R + 2 * k + 1) < NC ? R + 2 * k + 1 : 0] : v[(R + 2 * k) < NC ? R + 2 * k : 0];
                own[k] = hi + lo;
            }
            if (contributor) {
                unsigned long long* mine = slots + (size_t)(b - seg0) * kSlot;
#pragma unroll
                for (int k = 0; k < HM; ++k)
                    if (par + 2 * k < M) st_relaxed_u64(mine + (par + 2 * k) * kFTile + rr, tagged(tag, own[k]));
                continue;
            }
            // residual finaliser: h += sum, the next norm's input planes of
            // h * g_next and the per-tile sums of h^2 (per quadrant of 32 rows,
            // then the 4 quadrants in order)
            float* ssq = ys;  // [16][4]
#pragma unroll
            for (int k = 0; k < HM; ++k) {
                const int m = par + 2 * k;
                if (m >= M) break;  // (uniform in the warp)
                float hv = 0.f;
                if (n < a.N) {
                    hv = hp[k] + (own[k] + ps[k]);
                    a.out_f32[(size_t)m * a.ldo + n] = hv;
                    if (a.g_next) {
                        const float z = hv * gp;
                        const bf16 zh = __float2bfloat16_rn(z);
                        a.xo_hi[(size_t)m * a.N + n] = zh;
                        a.xo_lo[(size_t)m * a.N + n] = __float2bfloat16_rn(z - __bfloat162float(zh));
                    }
                }
                if (a.g_next) {
                    const float sq = warp_sum(hv * hv);
                    if (lane == 0) ssq[m * 4 + q4] = sq;
                }
            }
            if (a.g_next) {
                consumer_sync();
                if (threadIdx.x < M)
                    a.ss_out[threadIdx.x * a.n_tiles + tile] = (ssq[threadIdx.x * 4 + 0] + ssq[threadIdx.x * 4 + 1]) +
                                                              (ssq[threadIdx.x * 4 + 2] + ssq[threadIdx.x * 4 + 3]);
            }
            consumer_sync();  // ys is reused by the next segment
            if (ut && i < 64 && threadIdx.x == 0) ut[i * 4 + 3] = globaltimer();
            continue;
        }

        // finalisers of the other epilogues: TMEM -> ys (warps 0-3), then the
        // other segments' partials and the epilogue over ys
        ok = mbar_wait(pp.acc_full + ab, (pp.afull >> ab) & 1u, err) && ok;
        pp.afull ^= 1u << ab;
        pp.ab ^= 1;
        tc_fence_after();
        if (threadIdx.x == 0 && ct) ct[2] = globaltimer();
        if (warp < 4) {  // warp w reads TMEM lanes (tile rows) 32w .. 32w + 31
            float v[NP];
            tmem_ld<NP>(pp.tmem + (uint32_t)(ab * (kTmemCols / 2)) + ((uint32_t)(warp * 32) << 16), v);
            const int r = warp * 32 + lane;
#pragma unroll
            for (int m = 0; m < R; ++m) ys[r * 16 + m] = v[m] + v[R + m];
        }
        tc_fence_before();
        consumer_sync();
        if (lane == 0) mbar_arrive(pp.acc_empty + ab);  // the accumulator may be refilled

        constexpr int HJ = (R * kFTile + kGemmThreads - 1) / kGemmThreads;  // elements per thread (M <= R)

        if (nseg > 1) {
            // the other segments come from later CTAs, which never wait on this
            // one.  Each thread issues the words of all its elements for a batch
            // of segments before using any (one L2 round trip per batch), then
            // adds them in segment order.
            float acc[HJ];
            int at[HJ];
#pragma unroll
            for (int j = 0; j < HJ; ++j) {
                const int idx = threadIdx.x + j * kGemmThreads;
                const int m = idx / kFTile, r = idx - m * kFTile;
                at[j] = idx < M * kFTile ? m * kFTile + r : -1;
                acc[j] = at[j] >= 0 ? ys[r * 16 + m] : 0.f;
            }
            constexpr int QB = R <= 8 ? 4 : 2;  // segments per batch (registers: QB * HJ words)
            for (int sg0 = 1; sg0 < nseg; sg0 += QB) {
                unsigned long long w[QB][HJ];
#pragma unroll
                for (int q = 0; q < QB; ++q)
#pragma unroll
                    for (int j = 0; j < HJ; ++j)
                        if (sg0 + q < nseg && at[j] >= 0) w[q][j] = ld_relaxed_u64(slots + (size_t)(sg0 + q) * kSlot + at[j]);
                // words that do not carry this op's tag yet (their segment's CTA
                // has not published) are re-read together, not one at a time
                unsigned long long t_wait = 0;
                for (;;) {
                    bool ready = true;
#pragma unroll
                    for (int q = 0; q < QB; ++q)
#pragma unroll
                        for (int j = 0; j < HJ; ++j)
                            if (sg0 + q < nseg && at[j] >= 0 && tag_of(w[q][j]) != tag) ready = false;
                    if (ready) break;
                    const unsigned long long now = globaltimer();
                    if (t_wait == 0) t_wait = now;
                    if (now - t_wait > kErrPollAfterNs) {
                        if (*(volatile int*)err) { ok = false; break; }
                        if (now - t_wait > kBarrierTimeoutNs) {
                            atomicCAS(err, 0, kDevErrTimeout);
                            ok = false;
                            break;
                        }
                    }
#pragma unroll
                    for (int q = 0; q < QB; ++q)
#pragma unroll
                        for (int j = 0; j < HJ; ++j)
                            if (sg0 + q < nseg && at[j] >= 0 && tag_of(w[q][j]) != tag)
                                w[q][j] = ld_relaxed_u64(slots + (size_t)(sg0 + q) * kSlot + at[j]);
                }
#pragma unroll
                for (int q = 0; q < QB; ++q)
#pragma unroll
                    for (int j = 0; j < HJ; ++j)
                        if (sg0 + q < nseg && at[j] >= 0) acc[j] += value_of(w[q][j]);
            }
#pragma unroll
            for (int j = 0; j < HJ; ++j)
                if (at[j] >= 0) {
                    const int m = at[j] / kFTile, r = at[j] - m * kFTile;
                    ys[r * 16 + m] = acc[j];
                }
            consumer_sync();
        }

        // epilogue of the finished tile (row m scaled by its RMSNorm factor)
        if (epi == EPI_LOGITS) {
            for (int idx = threadIdx.x; idx < M * kFTile; idx += kGemmThreads) {
                const int m = idx / kFTile, r = idx - m * kFTile;
                const int n = tile * kFTile + r;
                if (n < a.N) a.out_f32[(size_t)m * a.ldo + n] = ys[r * 16 + m] * r_s[m];
            }
        } else if (epi == EPI_SWIGLU) {
            for (int idx = threadIdx.x; idx < M * 64; idx += kGemmThreads) {
                const int m = idx >> 6, r = idx & 63;
                const int i2 = tile * 64 + r;
                if (i2 >= a.ffn) continue;
                const float gt = ys[r * 16 + m] * r_s[m], up = ys[(r + 64) * 16 + m] * r_s[m];
                const float act = gt / (1.f + expf(-gt)) * up;
                const bf16 ah = __float2bfloat16_rn(act);
                a.xo_hi[(size_t)m * a.ffn + i2] = ah;
                a.xo_lo[(size_t)m * a.ffn + i2] = __float2bfloat16_rn(act - __bfloat162float(ah));
            }
        } else {  // EPI_QKV
            const int hd = a.head_dim, half = hd >> 1;
            const int qt = a.n_heads * hd / kFTile, kt = a.n_kv_heads * hd / kFTile;
            if (tile < qt + kt) {
                const bool is_q = tile < qt;
                const int tt = is_q ? tile : tile - qt;
                for (int idx = threadIdx.x; idx < M * 64; idx += kGemmThreads) {
                    const int m = idx >> 6, pr = idx & 63;  // rotation pair pr of the tile
                    const int hl = pr / half, ii = pr - hl * half;
                    const int r1 = hl * hd + ii, r2 = r1 + half;
                    const int head = tt * (kFTile / hd) + hl, pos = pos0 + m;
                    const float x1 = ys[r1 * 16 + m] * r_s[m], x2 = ys[r2 * 16 + m] * r_s[m];
                    const float2 cs = a.rope[(size_t)pos * half + ii];
                    const float y1 = x1 * cs.x - x2 * cs.y;
                    const float y2 = x2 * cs.x + x1 * cs.y;
                    if (is_q) {
                        float* q = a.q_out + (size_t)m * a.n_heads * hd + head * hd;
                        q[ii] = y1;
                        q[ii + half] = y2;
                    } else {
                        f16* k = a.k_cache + ((size_t)head * a.max_seq + pos) * hd;
                        k[ii] = __float2half_rn(y1);
                        k[ii + half] = __float2half_rn(y2);
                    }
                }
            } else {
                const int vt = tile - qt - kt;
                for (int idx = threadIdx.x; idx < M * kFTile; idx += kGemmThreads) {
                    const int m = idx / kFTile, r = idx - m * kFTile;
                    const int f = vt * kFTile + r;
                    const int head = f / hd, e = f - head * hd;
                    a.v_cache[((size_t)head * a.max_seq + pos0 + m) * hd + e] =
                        __float2half_rn(ys[r * 16 + m] * r_s[m]);
                }
            }
        }
        consumer_sync();  // ys is reused by the next segment
        if (ut && i < 64 && threadIdx.x == 0) ut[i * 4 + 3] = globaltimer();
    }
    consumer_sync();
    return ok;
}

// ---------------------------------------------------------------------------
// attention op: items (KV head, vector group, 128-position segment), through
// the TMA ring
// ---------------------------------------------------------------------------
// A segment is kAttnSegChunks absolute 64-position chunks; the producer thread
// requests each chunk's K and V rows (TMA, 128-byte swizzle) into consecutive
// ring stages.  An item is one segment of one KV head for a group of up to 16
// of its G * M query vectors (G query heads of the KV head, M rows): scores
// and P V on tensor cores (fp16 hi + lo operands, fp32 accumulators), the
// softmax over the segment from the score accumulators; the partial (o, max,
// sum) of the segment goes to global memory.  Items run segment fastest, so a
// CTA's consecutive items share their q.  After a grid barrier every CTA
// combines a share of the (KV head, vector) partials in segment order
// (flash-decoding style split of the softmax).  Every reduction has a fixed
// order that depends only on the row's own position, not on M.
struct AttnRange {
    int n_ch, n_seg, n_vg;  // chunks, segments per KV head, groups of 16 query vectors
    int i_begin, i_end;     // this CTA's items (KV head, vector group, segment), segment fastest
};
__device__ __forceinline__ AttnRange attn_range(const AttnArgs& a, int M, int pos0) {
    constexpr int S = kAttnSegChunks;
    AttnRange r;
    r.n_ch = (pos0 + M + kAttnChunk - 1) / kAttnChunk;  // chunks holding any visible position
    r.n_seg = (r.n_ch + S - 1) / S;
    r.n_vg = (a.n_heads / a.n_kv_heads * M + 15) / 16;
    const long long I = (long long)a.n_kv_heads * r.n_seg * r.n_vg, GR = gridDim.x;
    r.i_begin = (int)((long long)blockIdx.x * I / GR);
    r.i_end = (int)((long long)(blockIdx.x + 1) * I / GR);
    return r;
}

// Producer thread: requests K / V of this CTA's chunks at ring positions
// [i_from, i_limit), in item order; with old_only it stops at the first chunk
// holding rows this forward writes (those need the q/k/v op to be finished).
// Returns the ring position reached, or -1 if a wait timed out.
template <int R, int HD>
__device__ int attn_produce(const AttnArgs& a, const AttnRange& ar, int pos0, unsigned char* smem, Pipe& pp,
                            int* err, int i_from, int i_limit, bool old_only) {
    using L = GemmSmem<R>;
    constexpr int S = L::S, SC = kAttnSegChunks;
    int i = 0;
    for (int it = ar.i_begin; it < ar.i_end; ++it) {
        const int hv = it / ar.n_seg, kvh = hv / ar.n_vg, c0 = (it - hv * ar.n_seg) * SC;
        for (int c = c0; c < min(c0 + SC, ar.n_ch); ++c, ++i) {
            if (i < i_from) continue;
            if (i >= i_limit || (old_only && (c + 1) * kAttnChunk > pos0)) return i;
            const int s = i % S;
            unsigned char* st = smem + s * L::STAGE;
            if (!mbar_wait(pp.empty + s, (pp.pphase >> s) & 1u, err)) return -1;
            pp.pphase ^= 1u << s;
            mbar_arrive_expect_tx(pp.full + s, 2u * (HD / 64) * 8192u);
#pragma unroll
            for (int bx = 0; bx < HD / 64; ++bx) {
                tma_load_3d(st + bx * 8192, a.tm_k, bx * 64, c * kAttnChunk, a.kv_z0 + kvh, pp.full + s);
                tma_load_3d(st + 16384 + bx * 8192, a.tm_v, bx * 64, c * kAttnChunk, a.kv_z0 + kvh, pp.full + s);
            }
        }
    }
    return i;
}

// Before the grid barrier ahead of an attention op: the producer requests the
// K / V chunks of its first ring stages that hold only rows of earlier
// forwards.  Returns how many (0 for other threads, -1 on a timeout).
template <int R, int HD>
__device__ int attn_prefetch(const AttnArgs& a, int M, int pos0, unsigned char* smem, Pipe& pp, int* err) {
    if (threadIdx.x != kConsumers) return 0;
    const AttnRange ar = attn_range(a, M, pos0);
    if (ar.i_begin < ar.i_end) {
        prefetch_tmap(a.tm_k);
        prefetch_tmap(a.tm_v);
    }
    return attn_produce<R, HD>(a, ar, pos0, smem, pp, err, 0, GemmSmem<R>::S, true);
}

// Returns false if a wait timed out (error recorded).  pre: ring positions the
// producer already filled before the grid barrier (attn_prefetch).
template <int R, int HD>
__device__ bool attn_op(const AttnArgs& a, int M, int pos0, unsigned char* smem, Pipe& pp, int* err,
                        unsigned long long* ct, int pre, unsigned long long* ut) {
    using L = GemmSmem<R>;
    constexpr int S = L::S, VG = L::VG, SC = kAttnSegChunks, SP = SC * kAttnChunk;  // positions per segment
    static_assert(SC <= S, "a segment's chunks are held in the ring at once");
    const int G = a.n_heads / a.n_kv_heads, NV = G * M;
    const AttnRange ar = attn_range(a, M, pos0);

    if (threadIdx.x >= kConsumers + 32) {  // MMA warp: only keeps its copy of the ring parities
        if (threadIdx.x == kConsumers + 32) {
            int n = 0;
            for (int it = ar.i_begin; it < ar.i_end; ++it) {
                const int sg = it % ar.n_seg;
                n += min(SC, ar.n_ch - sg * SC);
            }
            advance_full<S>(pp, n);
        }
        return true;
    }
    if (threadIdx.x >= kConsumers) {  // producer warp: one elected thread requests K / V
        if (threadIdx.x != kConsumers) return true;
        // K / V rows of this forward were stored by other CTAs (generic proxy)
        if (ar.i_begin < ar.i_end) asm volatile("fence.proxy.async.global;" ::: "memory");
        return attn_produce<R, HD>(a, ar, pos0, smem, pp, err, pre, 1 << 30, false) >= 0;
    }

    constexpr int QST = L::QST, PST = L::PST;
    __half* qh = reinterpret_cast<__half*>(smem + L::ATT);  // [VG][QST] q hi, then lo
    __half* ql = qh + VG * QST;
    float* sc = reinterpret_cast<float*>(smem + L::ATT_SC);  // per-warp maxima and sums
    __half* ph = reinterpret_cast<__half*>(smem + L::ATT_P);  // [VG][PST] weights hi, then lo
    __half* pl = ph + VG * PST;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int g = lane >> 2, tg = lane & 3;
    constexpr size_t part_v = attn_part_floats(HD);  // floats per partial: o[HD], max, sum, pad
    bool ok = true;
    int i = 0;       // ring position within the op
    int q_key = -1;  // (KV head, vector group) whose q is in shared memory

    // profiling aid: ut (CTA 0 of a traced forward) gets per-item phase stamps
    auto stamp = [&](int it, int k) {
        if (ut && tid == 0 && it - ar.i_begin < 31) ut[(it - ar.i_begin) * 8 + k] = globaltimer();
    };
    for (int it = ar.i_begin; it < ar.i_end; ++it) {
        stamp(it, 0);
        const int hv = it / ar.n_seg, sg = it - hv * ar.n_seg, t0 = sg * SP;
        const int kvh = hv / ar.n_vg, vg = hv - kvh * ar.n_vg;
        const int n_u = min(SC, ar.n_ch - sg * SC);  // chunks of this segment
        const int v0 = vg * VG, nv = min(VG, NV - v0);
        float* part = a.part + ((size_t)kvh * a.n_chunks + sg) * NV * part_v;
        // q of this item's vectors as fp16 hi + lo (other CTAs wrote q: L2);
        // every thread issues all its 16-byte loads before converting, and the
        // loads overlap the wait for K / V; consecutive items of one KV head
        // and vector group reuse it
        const int key = kvh * ar.n_vg + vg;
        if (key != q_key) {
            constexpr int HD4 = HD / 4, QJ = VG * HD4 / kConsumers;  // float4 per thread: 2 | 1
            static_assert(VG * HD4 % kConsumers == 0, "q tile split evenly over the consumers");
            float4 qv[QJ];
#pragma unroll
            for (int j = 0; j < QJ; ++j) {
                const int k4 = tid + j * kConsumers, vl = k4 / HD4, e = (k4 - vl * HD4) * 4;
                qv[j] = make_float4(0.f, 0.f, 0.f, 0.f);
                if (vl < nv) {
                    const int v = v0 + vl, m = v / G, gi = v - m * G;
                    qv[j] = __ldcg(reinterpret_cast<const float4*>(a.q + (size_t)m * a.n_heads * HD +
                                                                   (size_t)(kvh * G + gi) * HD + e));
                }
            }
#pragma unroll
            for (int j = 0; j < QJ; ++j) {
                const int k4 = tid + j * kConsumers, vl = k4 / HD4, e = (k4 - vl * HD4) * 4;
                const __half2 h01 = __floats2half2_rn(qv[j].x, qv[j].y), h23 = __floats2half2_rn(qv[j].z, qv[j].w);
                const float2 f01 = __half22float2(h01), f23 = __half22float2(h23);
                const __half2 l01 = __floats2half2_rn(qv[j].x - f01.x, qv[j].y - f01.y);
                const __half2 l23 = __floats2half2_rn(qv[j].z - f23.x, qv[j].w - f23.y);
                *reinterpret_cast<uint2*>(qh + vl * QST + e) =
                    make_uint2(*reinterpret_cast<const uint32_t*>(&h01), *reinterpret_cast<const uint32_t*>(&h23));
                *reinterpret_cast<uint2*>(ql + vl * QST + e) =
                    make_uint2(*reinterpret_cast<const uint32_t*>(&l01), *reinterpret_cast<const uint32_t*>(&l23));
            }
        }
        q_key = key;
        stamp(it, 1);
        for (int j = 0; j < n_u; ++j) {
            const int s = (i + j) % S;
            ok = mbar_wait(pp.full + s, (pp.cphase >> s) & 1u, err) && ok;
            pp.cphase ^= 1u << s;
        }
        if (ct && tid == 0 && it == ar.i_begin) ct[1] = globaltimer();
        stamp(it, 2);
        consumer_sync();
        stamp(it, 3);

        // scores S = K q^T on tensor cores: warp w takes positions 16w..16w+15
        // (A = K rows, 128-byte swizzled), all 16 vectors (B = q hi, then lo);
        // then the softmax of every vector over the segment straight from the
        // accumulators: per-warp maxima -> CTA barrier -> the segment maximum
        // (the 8 warps' values in order) -> weights as fp16 hi + lo, per-warp
        // sums (the partial's sum adds the 8 warps' sums in order)
        float* wmax = sc;           // [8 warps][VG vectors]
        float* wsum = sc + 8 * VG;  // [8 warps][VG vectors]
        {
            const int p0 = warp * 16, j = p0 / kAttnChunk;
            float c[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
            if (j < n_u) {
                // K q_hi and K q_lo in separate accumulators (two short
                // dependency chains instead of one long one), added at the end
                float cl[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
                const unsigned char* kst = smem + ((i + j) % S) * L::STAGE;
                const int t = (p0 % kAttnChunk) + (lane & 7) + 8 * ((lane >> 3) & 1);
                const int qv = (lane & 7) + 8 * (lane >> 4), qk = ((lane >> 3) & 1) * 8;
#pragma unroll
                for (int ks = 0; ks < HD / 16; ++ks) {
                    uint32_t af[4], bh[4], bl[4];
                    const int chunk = 2 * (ks & 3) + (lane >> 4);
                    ldsm_x4(af, kst + (ks >> 2) * 8192 + t * 128 + ((chunk ^ (t & 7)) << 4));
                    ldsm_x4(bh, qh + qv * QST + ks * 16 + qk);
                    ldsm_x4(bl, ql + qv * QST + ks * 16 + qk);
                    mma_f16_16816(c[0], af[0], af[1], af[2], af[3], bh[0], bh[1]);
                    mma_f16_16816(cl[0], af[0], af[1], af[2], af[3], bl[0], bl[1]);
                    if (nv > 8) {  // vectors 8..15
                        mma_f16_16816(c[1], af[0], af[1], af[2], af[3], bh[2], bh[3]);
                        mma_f16_16816(cl[1], af[0], af[1], af[2], af[3], bl[2], bl[3]);
                    }
                }
#pragma unroll
                for (int nt = 0; nt < 2; ++nt)
#pragma unroll
                    for (int x = 0; x < 4; ++x) c[nt][x] += cl[nt][x];
            }
            // C: rows = positions p0 + g (+8), columns = vectors 8 nt + 2 tg (+1)
#pragma unroll
            for (int nt = 0; nt < 2; ++nt)
#pragma unroll
                for (int x = 0; x < 4; ++x) {
                    const int vl = nt * 8 + 2 * tg + (x & 1), pq = p0 + g + 8 * (x >> 1);
                    const int m = (v0 + vl) / G;
                    const bool vis = j < n_u && vl < nv && t0 + pq <= pos0 + m;
                    c[nt][x] = vis ? c[nt][x] * a.scale : -INFINITY;
                }
#pragma unroll
            for (int nt = 0; nt < 2; ++nt)
#pragma unroll
                for (int cx = 0; cx < 2; ++cx) {
                    float v = fmaxf(c[nt][cx], c[nt][cx + 2]);
                    v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, 4));
                    v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, 8));
                    v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, 16));
                    if (g == 0) wmax[warp * VG + nt * 8 + 2 * tg + cx] = v;
                }
            consumer_sync();
            stamp(it, 4);
#pragma unroll
            for (int nt = 0; nt < 2; ++nt)
#pragma unroll
                for (int cx = 0; cx < 2; ++cx) {
                    const int vl = nt * 8 + 2 * tg + cx;
                    float mx = -INFINITY;
#pragma unroll
                    for (int w2 = 0; w2 < kConsumers / 32; ++w2) mx = fmaxf(mx, wmax[w2 * VG + vl]);
                    float l = 0.f;
#pragma unroll
                    for (int xh = 0; xh < 2; ++xh) {
                        const float x = c[nt][cx + 2 * xh];
                        const float pq = x == -INFINITY ? 0.f : expf(x - mx);
                        const __half hh = __float2half_rn(pq);
                        const int pos = p0 + g + 8 * xh;
                        ph[vl * PST + pos] = hh;
                        pl[vl * PST + pos] = __float2half_rn(pq - __half2float(hh));
                        l += pq;
                    }
                    l += __shfl_xor_sync(0xffffffffu, l, 4);
                    l += __shfl_xor_sync(0xffffffffu, l, 8);
                    l += __shfl_xor_sync(0xffffffffu, l, 16);
                    if (g == 0) wsum[warp * VG + vl] = l;
                }
        }
        consumer_sync();
        stamp(it, 5);
        // the segment's (max, sum) of each vector; -inf: nothing visible
        if (tid < nv) {
            const int v = v0 + tid, m = v / G;
            float mx = -INFINITY, l = 0.f;
#pragma unroll
            for (int w2 = 0; w2 < kConsumers / 32; ++w2) {
                mx = fmaxf(mx, wmax[w2 * VG + tid]);
                l += wsum[w2 * VG + tid];
            }
            float* o = part + (size_t)v * part_v;
            o[HD] = pos0 + m < t0 ? -INFINITY : mx;
            o[HD + 1] = l;
        }

        // O = P V on tensor cores: warp w takes dims 16w..16w+15 (B = V rows via
        // transposed 8x8 loads), all 16 vectors (A = P hi, then lo); rows of
        // vectors past nv hold stale weights and are not stored
        if (warp * 16 < HD) {
            // P_hi V and P_lo V in separate accumulators, added at the end
            float c[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
            float cl[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
            const int d = warp * 16 + 8 * (lane >> 4), bx = d >> 6, cc = (d & 63) >> 3;
            const int pv = (lane & 7) + 8 * ((lane >> 3) & 1), pk = (lane >> 4) * 8;
            for (int ks = 0; ks < n_u * (kAttnChunk / 16); ++ks) {
                uint32_t ah[4], al[4], bv[4];
                const int p = ks * 16 + (lane & 7) + 8 * ((lane >> 3) & 1), j = p / kAttnChunk, tt = p % kAttnChunk;
                ldsm_x4(ah, ph + pv * PST + ks * 16 + pk);
                ldsm_x4(al, pl + pv * PST + ks * 16 + pk);
                ldsm_x4_t(bv, smem + ((i + j) % S) * L::STAGE + 16384 + bx * 8192 + tt * 128 + ((cc ^ (tt & 7)) << 4));
                mma_f16_16816(c[0], ah[0], ah[1], ah[2], ah[3], bv[0], bv[1]);
                mma_f16_16816(c[1], ah[0], ah[1], ah[2], ah[3], bv[2], bv[3]);
                mma_f16_16816(cl[0], al[0], al[1], al[2], al[3], bv[0], bv[1]);
                mma_f16_16816(cl[1], al[0], al[1], al[2], al[3], bv[2], bv[3]);
            }
#pragma unroll
            for (int nt = 0; nt < 2; ++nt)
#pragma unroll
                for (int x = 0; x < 4; ++x) c[nt][x] += cl[nt][x];
            // C: rows = vectors g (+8), columns = dims 16w + 8 nt + 2 tg (+1)
#pragma unroll
            for (int nt = 0; nt < 2; ++nt)
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int vl = g + 8 * h;
                    if (vl < nv)
                        *reinterpret_cast<float2*>(part + (size_t)(v0 + vl) * part_v + warp * 16 + nt * 8 + 2 * tg) =
                            make_float2(c[nt][2 * h], c[nt][2 * h + 1]);
                }
        }
        consumer_sync();  // q / scores / weights are free for the next item
        stamp(it, 6);
        if (tid == 0)
            for (int j = 0; j < n_u; ++j) mbar_arrive(pp.empty + (i + j) % S);  // the stages are free
        i += n_u;
    }
    if (ct && tid == 0) ct[6] = (unsigned long long)(ar.i_end - ar.i_begin);
    return ok;
}

// Second phase of attention, after a grid barrier (the segment partials of
// every CTA are visible): the partials of each (KV head, query vector) are
// combined in segment order - row m uses segments 0 .. (pos0 + m) / SP - and
// written as the bf16 hi / lo planes of the attention output.  One warp per
// 64 dims of a vector (2 dims per lane), spread round-robin over the warps of
// all CTAs.  Per batch of up to kCombineBatch segments a lane loads its dims of
// every segment and lane j the (max, sum) of segment j, all at once (one L2
// round trip per batch: one for contexts up to 2048 positions); the batch
// maximum and the sum of the weighted sums are shuffle trees, the weighted
// dims are added in segment order, and batches fold into running sums scaled
// to the running maximum.  The order depends only on the row's position.
constexpr int kCombineBatch = 16;
template <int HD>
__device__ void attn_combine(const AttnArgs& a, int M, int pos0) {
    if (threadIdx.x >= kConsumers) return;
    constexpr int SP = kAttnSegChunks * kAttnChunk, HALVES = HD / 64, B = kCombineBatch;
    static_assert(B <= 32, "one lane per segment of a batch");
    const int G = a.n_heads / a.n_kv_heads, NV = G * M;
    constexpr size_t part_v = attn_part_floats(HD);  // floats per partial: o[HD], max, sum, pad
    const size_t qs_stride = (size_t)NV * part_v;    // next segment of the same vector
    const int n_work = a.n_kv_heads * NV * HALVES;   // (vector, 64 dims) per warp
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int n_warps = gridDim.x * (kConsumers / 32);
    // warp-major over the CTAs: the first work items go to warp 0 of every CTA
    for (int wk = warp * gridDim.x + blockIdx.x; wk < n_work; wk += n_warps) {
        const int gv = wk / HALVES, hf = wk - gv * HALVES;
        const int kvh = gv / NV, v = gv - kvh * NV;
        const int e = hf * 64 + 2 * lane;
        const int m = v / G, gi = v - m * G;
        const int nsg = (pos0 + m) / SP + 1;
        const float* pv = a.part + (size_t)kvh * a.n_chunks * qs_stride + (size_t)v * part_v;
        float mx = -INFINITY, l = 0.f, o0 = 0.f, o1 = 0.f;
        for (int q0 = 0; q0 < nsg; q0 += B) {
            const int nb = min(B, nsg - q0);
            float2 ml = make_float2(-INFINITY, 0.f);  // (max, sum) of segment q0 + lane
            if (lane < nb) ml = __ldcg(reinterpret_cast<const float2*>(pv + (size_t)(q0 + lane) * qs_stride + HD));
            float2 ov[B];
#pragma unroll
            for (int j = 0; j < B; ++j) {
                ov[j] = make_float2(0.f, 0.f);
                if (j < nb) ov[j] = __ldcg(reinterpret_cast<const float2*>(pv + (size_t)(q0 + j) * qs_stride + e));
            }
            float bm = ml.x;
#pragma unroll
            for (int off = 16; off; off >>= 1) bm = fmaxf(bm, __shfl_xor_sync(0xffffffffu, bm, off));
            bm = fmaxf(bm, mx);
            // empty segments (and lanes past the batch) hold max -inf, o = 0
            const float r = mx == -INFINITY ? 0.f : expf(mx - bm);
            const float f = ml.x == -INFINITY ? 0.f : expf(ml.x - bm);
            float fl = f * ml.y;
#pragma unroll
            for (int off = 16; off; off >>= 1) fl += __shfl_xor_sync(0xffffffffu, fl, off);
            l = l * r + fl;
            o0 *= r;
            o1 *= r;
#pragma unroll
            for (int j = 0; j < B; ++j) {
                const float fj = __shfl_sync(0xffffffffu, f, j);
                o0 += fj * ov[j].x;
                o1 += fj * ov[j].y;
            }
            mx = bm;
        }
        const float inv = 1.f / l;
        const size_t at = (size_t)m * a.n_heads * HD + (size_t)(kvh * G + gi) * HD + e;
        const float v0 = o0 * inv, v1 = o1 * inv;
        const bf16 h0 = __float2bfloat16_rn(v0), h1 = __float2bfloat16_rn(v1);
        __nv_bfloat162 hi, lo;
        hi.x = h0;
        hi.y = h1;
        lo.x = __float2bfloat16_rn(v0 - __bfloat162float(h0));
        lo.y = __float2bfloat16_rn(v1 - __bfloat162float(h1));
        *reinterpret_cast<__nv_bfloat162*>(a.out_hi + at) = hi;
        *reinterpret_cast<__nv_bfloat162*>(a.out_lo + at) = lo;
    }
}

// ---------------------------------------------------------------------------
// embedding op: h = E[token], planes of h * g (first RMSNorm), sums of h^2
// ---------------------------------------------------------------------------
__device__ void embed_op(const FwdParams& p, int pos0) {
    if (threadIdx.x >= kConsumers) return;
    const int d = p.d, n_tiles = d / kFTile;  // sums of squares per 128 columns
    const int lane = threadIdx.x & 31;
    const int gw = blockIdx.x * (kGemmThreads / 32) + (threadIdx.x >> 5);
    const int nw = gridDim.x * (kGemmThreads / 32);
    if (blockIdx.x == 0 && threadIdx.x == 0) p.st->pos0 = pos0;
    for (int u = gw; u < p.M * n_tiles; u += nw) {
        const int m = u / n_tiles, t = u - m * n_tiles;
        int tok;
        if (p.src == SRC_TOKENS) tok = p.toks[m];
        else if (p.src == SRC_DRAFT) tok = p.st->j == 0 ? p.st->x_last : p.st->drafts[p.st->j - 1];
        else tok = m == 0 ? p.st->x_last : p.st->drafts[m - 1];
        const bf16* row = p.embed + (size_t)tok * d;
        float sq = 0.f;
#pragma unroll
        for (int j = 0; j < kFTile / 32; ++j) {
            const int i = t * kFTile + j * 32 + lane;
            const float v = __bfloat162float(row[i]);
            p.h[(size_t)m * d + i] = v;
            const float z = v * __bfloat162float(p.g0[i]);
            const bf16 zh = __float2bfloat16_rn(z);
            p.xn_hi[(size_t)m * d + i] = zh;
            p.xn_lo[(size_t)m * d + i] = __float2bfloat16_rn(z - __bfloat162float(zh));
            sq += v * v;
        }
        sq = warp_sum(sq);
        if (lane == 0) p.ss[m * n_tiles + t] = sq;
    }
}

// Block-cooperative copy of an op descriptor into shared memory.
__device__ __forceinline__ void copy_op(const FwdOp* src, FwdOp* dst) {
    static_assert(sizeof(FwdOp) % 4 == 0, "FwdOp is copied in 4-byte words");
    const unsigned* s = reinterpret_cast<const unsigned*>(src);
    unsigned* d = reinterpret_cast<unsigned*>(dst);
    for (int i = threadIdx.x; i < (int)(sizeof(FwdOp) / 4); i += blockDim.x) d[i] = s[i];
    __syncthreads();
}

// After a timed-out wait: give copies still in flight a bounded time to land
// before the CTA exits (the error is already recorded).
__device__ void drain_before_exit() {
    if (threadIdx.x == 0) {
        const unsigned long long t0 = globaltimer();
        while (globaltimer() - t0 < 2000000ull) __nanosleep(1000);
    }
    __syncthreads();
}

// Units of the next projection whose weights the producer requests between
// its CTA's arrival at an op boundary's grid barrier and the barrier's end.
constexpr int kBoundaryPrefetch = 5;

template <int R, int HD>
__global__ void __launch_bounds__(kFwdThreads, 1) forward_kernel(const FwdParams p) {
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    __shared__ float r_s[kMaxRows];
    __shared__ int s_pos0, s_skip;
    __shared__ unsigned s_seq;
    __shared__ uint32_t s_tmem;
    constexpr int S = GemmSmem<R>::S;
    __shared__ __align__(8) uint64_t full[S];       // TMA completion per stage
    __shared__ __align__(8) uint64_t empty[S];      // stage released (tcgen05.commit, or one consumer thread)
    __shared__ __align__(8) uint64_t acc_full[2];   // TMEM accumulator complete (tcgen05.commit)
    __shared__ __align__(8) uint64_t acc_empty[2];  // TMEM accumulator read by the consumers
    __shared__ FwdOp s_op[2];                       // current and next op's arguments
    // 128-byte TMA swizzle needs 1 KB aligned boxes
    unsigned char* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
    const bool mma_warp = threadIdx.x >= kConsumers + 32;
    if (threadIdx.x == 0) {
        int pos0;
        if (p.src == SRC_TOKENS) pos0 = p.pos0_arg;
        else if (p.src == SRC_DRAFT) pos0 = p.st->len + p.st->j;
        else pos0 = p.st->len;
        s_pos0 = pos0;
        // a draft step after the round's drafting stage ended (draft exit): no work
        s_skip = p.src == SRC_DRAFT && *(volatile int*)&p.st->exited;
        s_seq = *(volatile unsigned*)p.seq;  // this forward's number (advanced by CTA 0 below)
        for (int st = 0; st < S; ++st) {
            mbar_init(full + st, 1);
            mbar_init(empty + st, 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(acc_full + b, 1);
            mbar_init(acc_empty + b, kConsumers / 32);  // one arrival per consumer warp
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        if (p.trace && blockIdx.x == 0) p.trace[0] = globaltimer();
    }
    __syncthreads();
    if (s_skip) return;
    if (mma_warp) {  // TMEM for the two projection accumulators (freed at the end)
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&s_tmem)),
                     "r"(kTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    // every stage and both accumulators start empty
    if (threadIdx.x == 0)
        for (int st = 0; st < S; ++st) mbar_arrive(empty + st);
    if (threadIdx.x < kConsumers && (threadIdx.x & 31) == 0) {
        mbar_arrive(acc_empty + 0);
        mbar_arrive(acc_empty + 1);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const int pos0 = s_pos0;
    unsigned target = 0;
    int n_barrier = 0;
    // Grid barriers of this launch, each split in two: thread 0 arrives right
    // after a CTA barrier that ends the work before it, and waits for the
    // others later, so the producer's requests for the next op (the issue of
    // which can take microseconds while HBM is busy) overlap the wait instead
    // of delaying the arrival.  The profiling hook p.stall_barrier (0: none)
    // makes barrier number n unreachable, so that its bounded wait runs out
    // and the launch ends with the timeout recorded.
    __shared__ int s_ok;
    auto barrier_arrive = [&]() {
        target += gridDim.x;
        ++n_barrier;
        if (threadIdx.x == 0) grid_arrive(p.bar);
    };
    auto barrier_wait = [&]() {  // thread 0: result in s_ok
        const unsigned extra = n_barrier == p.stall_barrier ? 1u : 0u;
        s_ok = grid_wait(p.bar, target + extra, p.err, p.wait_ns) ? 1 : 0;
        // every CTA has read the sequence number before the first barrier
        if (s_ok && n_barrier == 1 && blockIdx.x == 0) *p.seq = s_seq + 1u;
    };
    Pipe pp{full, empty, acc_full, acc_empty, s_tmem, 0u, 0u, 0u, 0u, 0};
    int n_pre = 0;  // producer: units of the op whose weights were requested before it
    bool failed = false;
    int attn_pre = 0;  // producer: K / V chunks of the next attention op requested early
    copy_op(p.ops, s_op);
    for (int o = 0; o < p.n_ops; ++o) {
        const FwdOp& op = s_op[o & 1];
        const int type = op.type;
        bool ok = true;
        unsigned long long* ct = (p.trace && o == (p.trace_op & 0xffff)) ? p.trace + kTraceCtas + blockIdx.x * 8 : nullptr;
        const bool ut_cta = ct && (int)blockIdx.x == (p.trace_op >> 16);  // the CTA whose units are stamped
        if (ct && threadIdx.x == 0) ct[0] = globaltimer();
        // the next op's arguments: the producer warp copies them (16 bytes a
        // lane, asynchronously) into their slot, which held op o-1, while op
        // o runs; the producer uses them as soon as it has issued op o
        constexpr int kOpChunks = (int)(sizeof(FwdOp) / 16);
        static_assert(sizeof(FwdOp) % 16 == 0 && kOpChunks <= 32, "an op is copied in 16-byte pieces by one warp");
        const bool has_nx = o + 1 < p.n_ops;
        const int plane = mma_warp ? -1 : (int)threadIdx.x - kConsumers;  // lane in the producer warp
        if (has_nx && plane >= 0 && plane < kOpChunks)
            asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(
                             smem_u32(reinterpret_cast<unsigned char*>(s_op + ((o + 1) & 1)) + 16 * plane)),
                         "l"(reinterpret_cast<const unsigned char*>(p.ops + o + 1) + 16 * plane)
                         : "memory");
        const FwdOp* nx = has_nx ? s_op + ((o + 1) & 1) : nullptr;
        bool early = false;  // producer: the next projection's weights already requested
        if (is_gemm(type)) {
            ok = gemm_op<R>(op.g, epi_of(type), p.M, pos0, n_pre, smem, r_s, pp, (s_seq << 10) | (unsigned)o, p.err,
                            ut_cta ? p.trace + kTraceUnits : nullptr, ct);
        } else if (type == OP_EMBED) {
            embed_op(p, pos0);
        } else {
            // attention: segment partials; a grid barrier; then every CTA
            // combines a share of the partials.  Between arriving and passing,
            // the producer requests the next projection's first weights (the
            // ring is free again); the consumers do not wait for that.
            ok = attn_op<R, HD>(op.at, p.M, pos0, smem, pp, p.err, ct, attn_pre,
                                ut_cta ? p.trace + kTraceUnits : nullptr);
            if (__syncthreads_or(!ok)) {  // (uniform)
                failed = true;
                break;
            }
            if (ct && threadIdx.x == 0) ct[2] = globaltimer();
            barrier_arrive();
            if (plane >= 0) {
                asm volatile("cp.async.wait_all;" ::: "memory");
                __syncwarp();
            }
            if (plane == 0 && nx && is_gemm(nx->type)) {
                ok = gemm_prefetch<R>(nx->g, epi_of(nx->type), smem, pp, p.err, GemmSmem<R>::S);
                early = true;
            }
            if (threadIdx.x < kConsumers) {  // (the producer and MMA warps go on to the op's end)
                if (threadIdx.x == 0) {
                    barrier_wait();
                    if (ct) ct[7] = globaltimer();
                }
                consumer_sync();
                if (s_ok) attn_combine<HD>(op.at, p.M, pos0);
                else ok = false;
            }
        }
        if (ct && threadIdx.x == 0) ct[3] = globaltimer();
        // the end of op o in this CTA (its stores ordered before thread 0's
        // arrival); the last op needs no grid barrier
        if (__syncthreads_or(!ok)) {
            failed = true;
            break;
        }
        if (ct && threadIdx.x == 0) ct[4] = globaltimer();
        if (has_nx) barrier_arrive();
        // next op: visible to the producer warp now, to every thread after
        // the CTA barrier below; the producer requests its first inputs that
        // do not depend on op o while the grid gathers
        if (plane >= 0) {
            asm volatile("cp.async.wait_all;" ::: "memory");
            __syncwarp();
        }
        n_pre = 0;
        attn_pre = 0;
        if (plane == 0 && nx) {
            if (is_gemm(nx->type)) {
                n_pre = (early || kBoundaryPrefetch > GemmSmem<R>::S) ? GemmSmem<R>::S : kBoundaryPrefetch;
                if (!early) ok = gemm_prefetch<R>(nx->g, epi_of(nx->type), smem, pp, p.err, n_pre);
            } else if (nx->type == OP_ATTN) {
                attn_pre = attn_prefetch<R, HD>(nx->at, p.M, pos0, smem, pp, p.err);
                ok = attn_pre >= 0;
            }
        }
        if (has_nx && threadIdx.x == 0) {
            barrier_wait();
            if (ct && is_gemm(type)) ct[7] = globaltimer();
        }
        if (__syncthreads_or(!ok || (has_nx && threadIdx.x == 0 && !s_ok))) {
            failed = true;
            break;
        }
        if (ct && threadIdx.x == 0) ct[5] = globaltimer();
        if (p.trace && blockIdx.x == 0 && threadIdx.x == 0) p.trace[o + 1] = globaltimer();
    }
    // After a failed wait, copies and MMAs still in flight get a bounded time
    // to land; otherwise every MMA this CTA issued has completed (the
    // consumers waited for each accumulator).  Then TMEM is freed.
    if (failed) drain_before_exit();
    tc_fence_before();
    __syncthreads();
    if (mma_warp) {
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(s_tmem), "r"(kTmemCols)
                     : "memory");
    }
}

template <int R, int HD>
int launch_fwd(const FwdParams& p, int grid, cudaStream_t s) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid, 1, 1);
    cfg.blockDim = dim3(kFwdThreads, 1, 1);
    cfg.dynamicSmemBytes = GemmSmem<R>::BYTES;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeCooperative;
    attr[0].val.cooperative = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return (int)cudaLaunchKernelEx(&cfg, forward_kernel<R, HD>, p);
}

template <int R, int HD>
int configure_fwd() {
    return (int)cudaFuncSetAttribute(forward_kernel<R, HD>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)GemmSmem<R>::BYTES);
}

}  // namespace

int forward_configure() {
    int e = 0;
    e = e ? e : configure_fwd<1, 64>();
    e = e ? e : configure_fwd<4, 64>();
    e = e ? e : configure_fwd<8, 64>();
    e = e ? e : configure_fwd<12, 64>();
    e = e ? e : configure_fwd<16, 64>();
    e = e ? e : configure_fwd<1, 128>();
    e = e ? e : configure_fwd<4, 128>();
    e = e ? e : configure_fwd<8, 128>();
    e = e ? e : configure_fwd<12, 128>();
    e = e ? e : configure_fwd<16, 128>();
    return e;
}

template <int HD>
int launch_hd(const FwdParams& p, int grid, cudaStream_t s) {
    switch (fwd_plane_rows(p.M)) {
        case 1: return launch_fwd<1, HD>(p, grid, s);
        case 4: return launch_fwd<4, HD>(p, grid, s);
        case 8: return launch_fwd<8, HD>(p, grid, s);
        case 12: return launch_fwd<12, HD>(p, grid, s);
        default: return launch_fwd<16, HD>(p, grid, s);
    }
}

int launch_forward(const FwdParams& p, int head_dim, int grid, cudaStream_t s) {
    if (head_dim == 128) return launch_hd<128>(p, grid, s);
    if (head_dim == 64) return launch_hd<64>(p, grid, s);
    return (int)cudaErrorInvalidValue;
}

}  // namespace ssd
