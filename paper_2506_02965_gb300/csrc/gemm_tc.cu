// Grouped expert GEMMs on the 5th-generation tensor cores (tcgen05, sm_103a).
//
// One persistent, warp-specialised kernel template serves all six contractions of
// the SwiGLU experts (ForwardExpert / BackwardExpert of Alg. 6):
//   fwd  [G|U] = Xp W1^T (SwiGLU epilogue)      Y  = A W2^T
//   bwd  dA = dY W2 (SwiGLU-backward epilogue)  dXp = dH W1
//        dW2 = dY^T A  and  dW1 = dH^T Xp  (contraction over the expert's rows)
// Warp 0 issues TMA loads (128B-swizzled tiles) into a 4-stage shared-memory ring,
// warp 1 issues tcgen05.mma (M=128, N=BN, K=16, bf16 in, fp32 accumulate) into a
// double-buffered TMEM accumulator, warps 2-5 drain TMEM with tcgen05.ld and run
// the fused epilogue. Every mbarrier wait is bounded in time; on a timeout the CTA
// records MOE_ERR_TIMEOUT, drains its in-flight copies and MMAs, frees TMEM and
// returns.
#include <cuda.h>

#include <algorithm>

#include "moe_common.cuh"
#include "moe_internal.h"

namespace moe {
namespace tc {

constexpr int BM = 128;
constexpr int BK = 64;  // 64 bf16 = 128 bytes = one 128B-swizzle row
// Contraction rows per k-block: BK, except for CTA-pair K-variable tiles (weight
// gradients), whose operands are both MN-major (64-element TMA boxes): 128-row boxes
// there halve the boxes and stage hand-offs per byte (3 stages of 64 KiB per CTA).
__host__ __device__ constexpr int kblock_rows(bool var_k, bool pair) { return (var_k && pair) ? 128 : BK; }
// k-blocks per operand stage: 2 for the router up to 64 experts (its stream of x is bound
// by a fixed cost per stage hand-off, so a stage carries two 64-wide boxes of each
// operand; wider B would leave too few stages) and for the M-variable CTA-pair tiles
// with a store or SwiGLU-forward epilogue (three stages of 64 KiB per CTA instead of six
// of 32: the same bytes in flight, half the hand-offs, less power per flop under the
// power cap), else 1 (the SwiGLU-backward pairs measured faster with six stages)
__host__ __device__ constexpr int kblocks_per_stage(int epi, int bn, bool pair = false, bool var_k = false) {
    return ((epi == 3 /* EPI_ROUTE */ && bn <= 64) || (pair && !var_k && epi != 2 /* EPI_SWIGLU_BWD */)) ? 2 : 1;
}
constexpr int EPI_WARPS = 4;
constexpr int THREADS = 64 + 32 * EPI_WARPS;  // TMA warp, MMA warp, epilogue warps
constexpr int EPI_BOX = 32;                     // TMA-store box: 32 columns x 32 rows (bf16)
constexpr int EPI_BUF_BYTES = EPI_BOX * EPI_BOX * 2;
// per epilogue warp: a ring of 4 output boxes (each box leaves by its own TMA store, so
// up to 3 stores are in flight while the next box is written), or for the SwiGLU
// backward 2 x (G, U) boxes
constexpr int EPI_NBUF = 4;
constexpr int EPI_STAGE_BYTES = EPI_NBUF * EPI_BUF_BYTES;
// per epilogue warp (the router-gradient partials are stored straight from registers)
__host__ __device__ constexpr int epi_stage_bytes(int epi) { return epi == EPI_DWR ? 0 : EPI_STAGE_BYTES; }
constexpr int MAX_GROUPS = 256;

struct Params {
    const int32_t* offsets;  // OFFSETS mode when non-null
    int rows;                // UNIFORM rows per group
    int64_t a_stride, b_stride, out_stride;
    int G;
    int N;       // output columns (per group)
    int K;       // contraction length (M-variable)
    int Mout;    // output rows per group (K-variable)
    int F;       // SwiGLU inner size (SWIGLU epilogues)
    int64_t b_group_rows;  // rows of B's 2D view per group (M-variable)
    const int32_t* gexp;   // group -> expert of its weights / weight gradient, or null
    void* out0;
    void* out1;
    const void* aux;
    uint64_t wait_ns;
    // EPI_ROUTE: out0 = logits, out1 = probs (fp32 [T,E]), aux = bias [P,E] or null
    int E, k, normalize, hist_n;
    int band;  // tile order: bands of `band` M-tiles, each swept along N (set at launch)
    // operand bytes for the per-group choice of the tile order: the bytes of one A row
    // (M-variable: K elements; K-variable: Mout elements per contraction row), of one B
    // contraction row (K-variable), and of all of B (M-variable: one group's weights)
    int64_t a_row_bytes, b_row_bytes, b_all_bytes;
    int32_t* topk_idx;
    float* topk_w;
    int32_t* counts;
    // EPI_ROUTE: token rows per tile (1..BM; the A box height), so that the tiles of a
    // short batch spread over every SM (each CTA streams its rows at a per-CTA rate)
    int tile_rows;
};

// ------------------------------------------------------------------------ PTX helpers
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ uint64_t gtimer() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
// One poll: the thread sleeps until the phase completes or at most ~20 us have passed.
constexpr uint32_t kSuspendHintNs = 20000;
__device__ __forceinline__ bool mbar_try(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity), "r"(kSuspendHintNs)
        : "memory");
    return ok != 0;
}
// Bounded wait. Returns false when the CTA is aborting (another role gave up) or when
// this wait ran past `limit_ns` (then it raises the abort flag and records TIMEOUT).
__device__ __noinline__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                       uint64_t limit_ns) {
    if (mbar_try(bar, parity)) return true;
    const uint64_t t0 = gtimer();
    for (;;) {
        if (mbar_try(bar, parity)) return true;
        if (*abort_flag) return false;
        if (gtimer() - t0 > limit_ns) {
            *abort_flag = 1;
            record_status(MOE_ERR_TIMEOUT);
            return false;
        }
    }
}
// --- CTA-pair (cta_group::2) helpers
__device__ __forceinline__ uint32_t cluster_rank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}
// shared::cluster address of the same shared-memory offset in CTA `rank` of the cluster
__device__ __forceinline__ uint32_t map_to_rank(uint32_t addr, uint32_t rank) {
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
    return r;
}
__device__ __forceinline__ void mbar_arrive_remote(uint32_t cluster_bar) {
    asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_bar)
                 : "memory");
}
__device__ __forceinline__ bool mbar_try_cluster(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2, %3;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity), "r"(kSuspendHintNs)
        : "memory");
    return ok != 0;
}
// TMA load into this CTA's shared memory whose completion is counted on a barrier
// that may live in the peer CTA of the pair (the leader's "full" barrier)
__device__ __forceinline__ void tma_load_2d_pair(uint32_t dst, const CUtensorMap* map,
                                                 uint32_t cluster_bar, int c0, int c1) {
    asm volatile(
        "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes "
        "[%0], [%1, {%3, %4}], [%2];" ::"r"(dst),
        "l"((uint64_t)map), "r"(cluster_bar), "r"(c0), "r"(c1)
        : "memory");
}
__device__ __forceinline__ void mma_bf16_pair(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc,
                                              uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}
// commit the pair's MMAs to the barrier at this offset in every CTA of `mask`
__device__ __forceinline__ void mma_commit_pair(uint32_t bar, uint16_t mask) {
    asm volatile(
        "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 "
        "[%0], %1;" ::"r"(bar),
        "h"(mask)
        : "memory");
}
// credit `bytes` of expected transactions to a barrier in another CTA of the cluster, as
// if that many bytes had arrived there (no arrival)
__device__ __forceinline__ void mbar_complete_tx_remote(uint32_t cluster_bar, uint32_t bytes) {
    asm volatile("mbarrier.complete_tx.relaxed.cluster.shared::cluster.b64 [%0], %1;" ::"r"(cluster_bar), "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ void cluster_sync_all() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::
                     : "memory");
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, uint32_t bar,
                                            int c0, int c1) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes "
        "[%0], [%1, {%3, %4}], [%2];" ::"r"(dst),
        "l"((uint64_t)map), "r"(bar), "r"(c0), "r"(c1)
        : "memory");
}
__device__ __forceinline__ void tma_store_2d(const CUtensorMap* map, uint32_t src, int c0, int c1) {
    asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%2, %3}], [%1];" ::"l"(
                     (uint64_t)map),
                 "r"(src), "r"(c0), "r"(c1)
                 : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read0() {
    asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
}
// wait until at most N of this thread's bulk groups are still reading shared memory
template <int N>
__device__ __forceinline__ void bulk_wait_read() {
    asm volatile("cp.async.bulk.wait_group.read %0;" ::"n"(N) : "memory");
}
__device__ __forceinline__ void bulk_wait0() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
__device__ __forceinline__ void fence_proxy_async() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
// 32 fp32 values -> 32 bf16 (64 bytes) at dst (16-byte aligned; shared or global)
__device__ __forceinline__ void store_row32(__nv_bfloat16* dst, const float* v) {
#pragma unroll
    for (int i = 0; i < 4; ++i) Vec<__nv_bfloat16>::store(dst + 8 * i, v + 8 * i);
}

// One 64-byte row (32 bf16) of a staging box in the 64B-swizzled layout the TMA store
// map uses: 16-byte chunk c of row r sits at chunk c ^ ((r >> 1) & 3).
__device__ __forceinline__ void store_row32_sw64(uint8_t* row_base, int r, const float* v) {
#pragma unroll
    for (int c = 0; c < 4; ++c)
        Vec<__nv_bfloat16>::store(reinterpret_cast<__nv_bfloat16*>(row_base + ((c ^ ((r >> 1) & 3)) << 4)),
                                  v + 8 * c);
}

__device__ __forceinline__ void fence_before() {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void fence_after() {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void mma_bf16(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc,
                                         uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}
__device__ __forceinline__ void mma_commit(uint32_t bar) {
    asm volatile(
        "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
        : "memory");
}
// 32 lanes x 32 consecutive fp32 columns of the accumulator
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float* v) {
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
        "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
          "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),
          "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),
          "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// 32 lanes x 16 consecutive fp32 columns of the accumulator
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float* v) {
    uint32_t r[16];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
        "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
          "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}
// 16-byte read-only load (the buffer is not written while the kernel runs)
__device__ __forceinline__ uint4 ldg_nc(const __nv_bfloat16* ptr) {
    uint4 r;
    asm volatile("ld.global.nc.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
                 : "l"(ptr));
    return r;
}
__device__ __forceinline__ void unpack8(uint4 u, float* v) {
    const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const float2 f = __bfloat1622float2(h[i]);
        v[2 * i] = f.x;
        v[2 * i + 1] = f.y;
    }
}

// Shared-memory matrix descriptor, 128B swizzle, sm_100 family layout:
// start>>4 [0,14), LBO>>4 [16,30), SBO>>4 [32,46), version 1 [46,48), swizzle 2 [61,64).
__device__ __forceinline__ uint64_t smem_desc(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
    uint64_t d = (uint64_t)((saddr & 0x3FFFFu) >> 4);
    d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
    d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;
    d |= (uint64_t)1 << 46;
    d |= (uint64_t)2 << 61;
    return d;
}
// Instruction descriptor of kind::f16: fp32 D [4,6), bf16 A [7,10), bf16 B [10,13),
// A major [15], B major [16] (1 = MN-major), N>>3 [17,23), M>>4 [24,29).
template <int BN, bool A_MN, bool B_MN, int M = BM>
__host__ __device__ constexpr uint32_t instr_desc() {
    return (1u << 4) | (1u << 7) | (1u << 10) | ((A_MN ? 1u : 0u) << 15) |
           ((B_MN ? 1u : 0u) << 16) | ((uint32_t)(BN >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

// Pipeline depth: as many operand stages as fit beside the epilogue's shared memory
// (staging boxes, or the router's histogram), at most 12. OCC CTAs share one SM (OCC = 2:
// about half of the SM's 228 KiB each, for launches bound by their epilogue, whose
// stores then come from twice as many warps per SM).
__host__ __device__ constexpr int epi_extra_bytes(int epi) {
    return epi == EPI_ROUTE ? 64 * 64 * 4 : EPI_WARPS * epi_stage_bytes(epi);
}
__host__ __device__ constexpr int num_stages(uint32_t stage_bytes, int epi, int occ = 1) {
    const int per_cta = occ == 1 ? 227 * 1024 : 112 * 1024;
    const int budget = per_cta - 1024 - 1024 - epi_extra_bytes(epi);  // dyn. smem, align, static
    const int n = budget / (int)stage_bytes;
    return n > 12 ? 12 : n;
}

// ------------------------------------------------------------------------ tile geometry
struct Tile {
    int g;
    int m0, n0;         // output tile origin inside the group
    int mvalid;         // rows of the group (M-variable) -> rows m0.. valid if < mvalid
    int64_t a_row;      // first A row (M-var: token row; K-var: first contraction row)
    int64_t b_row;      // K-var: first contraction row of B
    int64_t out_row;    // M-var: output row of group row 0
    int k_iters;
    int last_rows;      // K-var: valid contraction rows in the last k-block (1..64)
    bool dw;            // a tile of the second (K-variable) problem of a fused launch
    int we;             // expert whose weights (M-variable) or weight gradient (K-variable)
                        // the tile uses: group_expert[g], or g
};

// ------------------------------------------------------------------------ router epilogue
// Gating of Alg. 7 for the token of this TMEM lane: the thread holds all BN >= E
// logits of its token, adds the party's bias, writes logits and Softmax
// probabilities, picks the k largest logits (equal logits: lower expert id first),
// writes the gate weights p[I] (renormalised on request) and counts the picks.
// The loops over experts are unrolled (the logits live in registers); the loop over
// the k picks is not: each tile runs this code once per CTA, so it runs from a cold
// instruction cache, and an unrolled 8 x BN selection was fetch-bound (k = 6, E = 64).
template <int BN>
__device__ __forceinline__ void route_epilogue(const Params& p, const Tile& ti, int m, bool valid,
                                               uint32_t tbase, int* hist) {
    float z[BN];
    if constexpr (BN == 16) {
        tmem_ld16(tbase, z);
    } else {
#pragma unroll
        for (int c = 0; c < BN / 32; ++c) tmem_ld32(tbase + 32 * c, z + 32 * c);
    }
    if (!valid) return;
    const int E = p.E, k = p.k;
    const int64_t t = ti.out_row + m;
    const float* bias = (const float*)p.aux;
    float mx = -3.402823466e38f;
#pragma unroll
    for (int e = 0; e < BN; ++e) {
        if (e < E) {
            if (bias) z[e] += bias[ti.g * E + e];
            mx = fmaxf(mx, z[e]);
        }
    }
    float ez[BN];
    float sum = 0.f;
#pragma unroll
    for (int e = 0; e < BN; ++e) {
        ez[e] = e < E ? expf(z[e] - mx) : 0.f;
        if (e < E) sum += ez[e];
    }
    float* lg = (float*)p.out0 + t * E;
    float* pr = (float*)p.out1 + t * E;
#pragma unroll
    for (int e = 0; e < BN; e += 4) {
        if (e < E) {
            *reinterpret_cast<float4*>(lg + e) = make_float4(z[e], z[e + 1], z[e + 2], z[e + 3]);
            *reinterpret_cast<float4*>(pr + e) =
                make_float4(ez[e] / sum, ez[e + 1] / sum, ez[e + 2] / sum, ez[e + 3] / sum);
        }
    }
    uint64_t taken = 0;
    float wsum = 0.f;
    int32_t* ti_out = p.topk_idx + t * k;
    float* tw_out = p.topk_w + t * k;
#pragma unroll 1
    for (int j = 0; j < k; ++j) {
        int bi = -1;
        float bv = 0.f;
#pragma unroll
        for (int e = 0; e < BN; ++e) {
            if (e < E && !((taken >> e) & 1ull) && (bi < 0 || z[e] > bv)) {
                bi = e;
                bv = z[e];
            }
        }
        taken |= 1ull << bi;
        const float w = expf(bv - mx) / sum;
        wsum += w;
        ti_out[j] = bi;
        tw_out[j] = w;
        atomicAdd(&hist[ti.g * E + bi], 1);
    }
    if (p.normalize) {
#pragma unroll 1
        for (int j = 0; j < k; ++j) tw_out[j] = tw_out[j] / wsum;
    }
}

// Gating of Alg. 7 for E > 64 (BN = 128 or 256 accumulator columns): the same results
// as route_epilogue without holding all logits in registers. The accumulator stays in
// TMEM, read 32 columns at a time in three passes: (1) bias, logits out, running max and
// the k largest logits by insertion into a sorted list (ids arrive in ascending order
// and only a strictly larger logit moves ahead, so equal logits keep the lower id
// first); (2) the sum of exp(z - max); (3) the probabilities. Logits and probabilities
// are written element by element (any E). Every lane runs the TMEM loads (they are
// warp-collective); only valid rows use them.
template <int BN>
__device__ __forceinline__ void route_epilogue_wide(const Params& p, const Tile& ti, int m, bool valid,
                                                    uint32_t tbase, int* hist) {
    const int E = p.E, k = p.k;
    const int64_t t = ti.out_row + m;
    const float* bias = (const float*)p.aux;
    float* lg = (float*)p.out0 + t * E;
    float* pr = (float*)p.out1 + t * E;
    float mx = -3.402823466e38f;
    float tv[8];
    int tid[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
        tv[j] = -3.402823466e38f;
        tid[j] = -1;
    }
#pragma unroll 1
    for (int c = 0; c < BN; c += 32) {
        float z[32];
        tmem_ld32(tbase + c, z);
        if (valid) {
#pragma unroll
            for (int i = 0; i < 32; ++i) {
                const int e = c + i;
                if (e < E) {
                    float v = z[i] + (bias ? bias[ti.g * E + e] : 0.f);
                    lg[e] = v;
                    mx = fmaxf(mx, v);
                    // insert at the first slot that is empty or holds a smaller logit,
                    // then shift the rest down by one
                    float cv = v;
                    int ce = e;
                    bool shifting = false;
#pragma unroll
                    for (int j = 0; j < 8; ++j) {
                        if (j < k && (shifting || tid[j] < 0 || cv > tv[j])) {
                            const float tvj = tv[j];
                            const int tij = tid[j];
                            tv[j] = cv;
                            tid[j] = ce;
                            cv = tvj;
                            ce = tij;
                            shifting = true;
                            if (ce < 0) break;
                        }
                    }
                }
            }
        }
    }
    float sum = 0.f;
#pragma unroll 1
    for (int c = 0; c < BN; c += 32) {
        float z[32];
        tmem_ld32(tbase + c, z);
        if (valid) {
#pragma unroll
            for (int i = 0; i < 32; ++i)
                if (c + i < E) sum += expf(z[i] + (bias ? bias[ti.g * E + c + i] : 0.f) - mx);
        }
    }
#pragma unroll 1
    for (int c = 0; c < BN; c += 32) {
        float z[32];
        tmem_ld32(tbase + c, z);
        if (valid) {
#pragma unroll
            for (int i = 0; i < 32; ++i)
                if (c + i < E) pr[c + i] = expf(z[i] + (bias ? bias[ti.g * E + c + i] : 0.f) - mx) / sum;
        }
    }
    if (!valid) return;
    float wsel[8], wsum = 0.f;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
        wsel[j] = 0.f;
        if (j < k) {
            wsel[j] = expf(tv[j] - mx) / sum;
            wsum += wsel[j];
        }
    }
#pragma unroll
    for (int j = 0; j < 8; ++j) {
        if (j < k) {
            p.topk_idx[t * k + j] = tid[j];
            p.topk_w[t * k + j] = p.normalize ? wsel[j] / wsum : wsel[j];
            atomicAdd(&hist[ti.g * E + tid[j]], 1);
        }
    }
}

// ------------------------------------------------------------------------ the kernel
// PAIR: the two CTAs of a cluster compute one 256 x BN tile with tcgen05 cta_group::2
// MMAs issued by CTA 0: each CTA holds 128 rows of A and BN/2 rows of B in its own
// shared memory and 128 rows of the accumulator in its own TMEM.
// DW2: the launch also computes a second, K-variable problem with the same groups
// (p2, tmA2, tmB2, tmO2: C_g = A_g^T B_g over group g's rows, MN-major operands, bf16
// store), its tiles after all of the first problem's: one persistent launch, one tail,
// for a weight gradient and the M-variable GEMM of the same backward step. (Interleaving
// the two problems' tiles group by group measured slower: a tile with a long epilogue
// followed by one with a short mainloop leaves the MMA waiting for an accumulator.)
template <int BN, bool B_MN, bool VAR_K, int EPI, bool PAIR = false, bool DW2 = false, int OCC = 1>
__global__ void __launch_bounds__(THREADS, OCC)
    grouped_gemm_kernel(const __grid_constant__ CUtensorMap tmA,
                        const __grid_constant__ CUtensorMap tmB,
                        const __grid_constant__ CUtensorMap tmO0,
                        const __grid_constant__ CUtensorMap tmO1, const Params p,
                        const __grid_constant__ CUtensorMap tmA2,
                        const __grid_constant__ CUtensorMap tmB2,
                        const __grid_constant__ CUtensorMap tmO2, const Params p2) {
    pdl_begin();
    static_assert(!DW2 || (B_MN && !VAR_K && !PAIR && BN == 256), "fused: M-variable, MN-major B");
    static_assert(OCC == 1 || (!PAIR && !DW2 && 2 * BN * OCC <= 512), "shared SMs: single-CTA tiles, TMEM for all");
    constexpr bool A_MN = VAR_K;
    constexpr int NPAIR = PAIR ? 2 : 1;
    constexpr int BNL = BN / NPAIR;  // B rows held by this CTA
    constexpr int BMP = BM * NPAIR;  // rows of one (pair) tile
    constexpr int KB = kblock_rows(VAR_K, PAIR);  // contraction rows per k-block
    constexpr uint32_t ATOM = KB * 128;              // bytes of one 64-wide MN-major box
    constexpr int KPS = kblocks_per_stage(EPI, BN, PAIR, VAR_K);
    constexpr uint32_t A_BOX = BM * KB * 2;   // one k-block of A
    constexpr uint32_t B_BOX = BNL * KB * 2;  // one k-block of B
    constexpr uint32_t A_BYTES = A_BOX * KPS;
    constexpr uint32_t B_BYTES = B_BOX * KPS;
    constexpr uint32_t STAGE_BYTES = A_BYTES + B_BYTES;
    constexpr int NST = num_stages(STAGE_BYTES, EPI, OCC);
    constexpr uint32_t IDESC = instr_desc<BN, A_MN, B_MN, BMP>();
    constexpr uint32_t IDESC_DW = instr_desc<BN, true, true, BM>();
    constexpr int TMEM_COLS = (2 * BN <= 32) ? 32 : (2 * BN <= 64) ? 64 : (2 * BN <= 128) ? 128 : (2 * BN <= 256) ? 256 : 512;

    extern __shared__ uint8_t smem_raw[];
    // K-variable pairs: the peer's own barriers for the partial last k-block of a tile
    constexpr int NPART = (PAIR && VAR_K) ? NST : 0;
    __shared__ uint64_t bars[2 * NST + 5 + 2 * EPI_WARPS + NPART];
    __shared__ uint32_t s_tmem;
    __shared__ int s_abort;
    __shared__ int s_tile_start[MAX_GROUPS + 1];
    __shared__ int s_total1;  // fused: tiles of the first problem
    __shared__ unsigned char s_order[DW2 ? MAX_GROUPS : 1];  // fused: second problem's group order

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    volatile int* abort_flag = &s_abort;
    const uint32_t rank = PAIR ? cluster_rank() : 0u;
    const int tile0 = (int)blockIdx.x / NPAIR, tile_step = (int)gridDim.x / NPAIR;

    // group -> tile prefix
    // N-tiles per row of tiles; the last one may be ragged (N a multiple of 128 with
    // 256-wide tiles: its columns past N are computed from zero-filled or unused operand
    // columns and never stored)
    const int tiles_n = (EPI == EPI_SWIGLU_FWD) ? p.N / 256 : (EPI == EPI_ROUTE) ? 1 : (p.N + BN - 1) / BN;
    if (threadIdx.x == 0) {
        int acc = 0;
        for (int g = 0; g < p.G; ++g) {
            s_tile_start[g] = acc;
            int mt;
            if (VAR_K) {
                mt = p.Mout / BMP;
            } else {
                const int rows = p.offsets ? (p.offsets[g + 1] - p.offsets[g]) : p.rows;
                const int rpt = (EPI == EPI_ROUTE) ? p.tile_rows : BMP;  // rows per tile
                mt = rows > 0 ? (rows + rpt - 1) / rpt : 0;
            }
            acc += mt * tiles_n;
        }
        s_tile_start[p.G] = acc;
        s_total1 = acc;
        if constexpr (DW2) s_tile_start[p.G] = acc + p.G * (p2.Mout / BM) * (p2.N / BN);
        s_abort = 0;
    }
    __syncthreads();
    if constexpr (DW2) {
        // weight-gradient groups longest first (each tile of a group runs over all its
        // rows): with skewed experts the long tiles then do not form the tail. Rank of g =
        // groups with more rows, or as many and a lower index. (Row counts are read from
        // the offsets in global memory: static shared memory is at its limit here.)
        for (int g = threadIdx.x; g < p2.G; g += blockDim.x) {
            const int rg = p2.offsets[g + 1] - p2.offsets[g];
            int rank = 0;
            for (int h = 0; h < p2.G; ++h) {
                const int rh = p2.offsets[h + 1] - p2.offsets[h];
                rank += (rh > rg) || (rh == rg && h < g);
            }
            s_order[rank] = (unsigned char)g;
        }
        __syncthreads();
    }
    const int total_tiles = s_tile_start[p.G];
    if (tile0 >= total_tiles) return;  // uniform across the pair

    // Tile order inside a group: bands of `band` M-tiles, each band swept along N with
    // the M-tiles of the band innermost. The tiles that run at the same time (one round
    // of the persistent grid, C of them) then cover about band x C/band output tiles and
    // read band A blocks and C/band B blocks, instead of one A block and C B blocks when
    // whole rows of N-tiles come first (band ~ sqrt(C) minimises the blocks per round;
    // the A blocks of a band also stay in L2 while it sweeps N). When all of a group's B
    // fits in L2, whole rows of N-tiles first (band 1) read it from DRAM once and each A
    // block once; else when all of its A fits, whole columns of M-tiles first (band =
    // the group's M-tiles) do the same with A resident.
    constexpr int64_t kL2Resident = 48ll << 20;  // bytes of an operand kept in L2
    auto group_band = [&](const Params& q, int64_t rows_g, int mt_g) -> int {
        const int64_t a_all = (int64_t)rows_g * q.a_row_bytes;
        const int64_t b_all = q.b_row_bytes ? (int64_t)rows_g * q.b_row_bytes : q.b_all_bytes;
        if (b_all > 0 && b_all <= kL2Resident) return 1;
        if (a_all > 0 && a_all <= kL2Resident) return mt_g;
        return q.band;
    };
    auto band_split = [&](int local, int mt_g, int nt_g, int band, int* mt, int* nt) {
        const int gmx = band > 0 ? band : 1;
        const int b = local / (gmx * nt_g);
        const int first = b * gmx;
        const int gm = min(gmx, mt_g - first);
        const int rem = local - b * gmx * nt_g;
        *mt = first + rem % gm;
        *nt = rem / gm;
    };
    auto tile_at = [&](int t) -> Tile {
        Tile ti;
        ti.dw = false;
        if constexpr (DW2) {
            if (t >= s_total1) {  // second problem: K-variable, rows of group g
                const int per = (p2.Mout / BM) * (p2.N / BN);
                const int g = s_order[(t - s_total1) / per], l2 = (t - s_total1) % per;
                const int tn2 = p2.N / BN;
                int mt2, nt2;
                band_split(l2, p2.Mout / BM, tn2,
                           group_band(p2, p2.offsets[g + 1] - p2.offsets[g], p2.Mout / BM), &mt2, &nt2);
                ti.dw = true;
                ti.g = g;
                ti.we = p2.gexp ? p2.gexp[g] : g;
                ti.m0 = mt2 * BM;
                ti.n0 = nt2 * BN;
                const int64_t r0 = p2.offsets[g], nrows = p2.offsets[g + 1] - r0;
                ti.mvalid = p2.Mout;
                ti.a_row = ti.b_row = r0;
                ti.out_row = 0;
                ti.k_iters = (int)((nrows + BK - 1) / BK);
                ti.last_rows = (int)(nrows - (int64_t)(ti.k_iters - 1) * BK);
                return ti;
            }
        }
        // the group whose tile range holds t: last g with s_tile_start[g] <= t (binary
        // search; empty groups share their start with the next one)
        int lo = 0, hi = p.G - 1;
        while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1;
            if (s_tile_start[mid] <= t) lo = mid;
            else hi = mid - 1;
        }
        const int g = lo;
        const int local = t - s_tile_start[g];
        const int g_end = (g + 1 < p.G) ? s_tile_start[g + 1] : s_total1;
        const int mt_g = (g_end - s_tile_start[g]) / tiles_n;
        const int64_t rows_g = p.offsets ? (int64_t)(p.offsets[g + 1] - p.offsets[g]) : (int64_t)p.rows;
        int mt, nt;
        band_split(local, mt_g, tiles_n, group_band(p, rows_g, mt_g), &mt, &nt);
        ti.g = g;
        ti.we = p.gexp ? p.gexp[g] : g;
        ti.m0 = (EPI == EPI_ROUTE) ? mt * p.tile_rows : mt * BMP + (int)rank * BM;
        ti.n0 = nt * ((EPI == EPI_SWIGLU_FWD) ? 128 : BN);
        int64_t r0, nrows, a0, b0, o0;
        if (p.offsets) {
            r0 = p.offsets[g];
            nrows = p.offsets[g + 1] - r0;
            a0 = b0 = o0 = r0;
        } else {
            nrows = p.rows;
            a0 = (int64_t)g * p.a_stride;
            b0 = (int64_t)g * p.b_stride;
            o0 = (int64_t)g * p.out_stride;
        }
        if (VAR_K) {
            ti.mvalid = p.Mout;
            ti.a_row = a0;
            ti.b_row = b0;
            ti.out_row = 0;
            ti.k_iters = (int)((nrows + KB - 1) / KB);
            ti.last_rows = (int)(nrows - (int64_t)(ti.k_iters - 1) * KB);
        } else {
            // router tiles of tile_rows rows: the box's rows past them are the next tile's
            ti.mvalid = (EPI == EPI_ROUTE) ? (int)min64(nrows, (int64_t)ti.m0 + p.tile_rows) : (int)nrows;
            ti.a_row = a0;
            ti.b_row = 0;
            ti.out_row = o0;
            ti.k_iters = p.K / (BK * KPS);
            ti.last_rows = BK;
        }
        return ti;
    };

    // 1024-byte aligned stage ring
    const uint32_t raw_u32 = smem_u32(smem_raw);
    const uint32_t ring = raw_u32 + ((1024u - (raw_u32 & 1023u)) & 1023u);
    uint8_t* ring_ptr = smem_raw + (ring - raw_u32);
    uint8_t* stage_out = ring_ptr + (size_t)NST * STAGE_BYTES;  // EPI_WARPS x EPI_STAGE_BYTES
    int* route_hist = reinterpret_cast<int*>(stage_out);             // EPI_ROUTE has no staging
    if constexpr (EPI == EPI_ROUTE) {
        for (int i = threadIdx.x; i < p.hist_n; i += blockDim.x) route_hist[i] = 0;
    }
    const uint32_t bar0 = smem_u32(&bars[0]);
    auto full_bar = [&](int s) { return bar0 + 8u * s; };
    auto empty_bar = [&](int s) { return bar0 + 8u * (NST + s); };
    auto tfull_bar = [&](int a) { return bar0 + 8u * (2 * NST + a); };
    auto tempty_bar = [&](int a) { return bar0 + 8u * (2 * NST + 2 + a); };
    const uint32_t drain_bar = bar0 + 8u * (2 * NST + 4);
    auto pfull_bar = [&](int s) { return bar0 + 8u * (2 * NST + 5 + 2 * EPI_WARPS + s); };
    // waits: cluster-scope acquire when the barrier also collects the peer's arrivals
    auto wait_bar = [&](uint32_t bar, uint32_t parity) -> bool {
        if constexpr (PAIR) {
            if (mbar_try_cluster(bar, parity)) return true;
            const uint64_t t0 = gtimer();
            for (;;) {
                if (mbar_try_cluster(bar, parity)) return true;
                if (*abort_flag) return false;
                if (gtimer() - t0 > p.wait_ns) {
                    *abort_flag = 1;
                    record_status(MOE_ERR_TIMEOUT);
                    return false;
                }
            }
        } else {
            return mbar_wait(bar, parity, abort_flag, p.wait_ns);
        }
    };

    if (threadIdx.x == 0) {
        for (int s = 0; s < NST; ++s) {
            mbar_init(full_bar(s), 1);  // the (leader's) producer arms it for both CTAs' bytes
            mbar_init(empty_bar(s), 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(tfull_bar(a), 1);
            mbar_init(tempty_bar(a), EPI_WARPS * NPAIR);  // one arrival per epilogue warp
        }
        mbar_init(drain_bar, 1);
        for (int i = 0; i < 2 * EPI_WARPS; ++i) mbar_init(bar0 + 8u * (2 * NST + 5 + i), 1);
        for (int s = 0; s < NPART; ++s) mbar_init(pfull_bar(s), 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 1) {
        if constexpr (PAIR) {
            asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                             smem_u32(&s_tmem)),
                         "r"(TMEM_COLS)
                         : "memory");
            asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
        } else {
            asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                             smem_u32(&s_tmem)),
                         "r"(TMEM_COLS)
                         : "memory");
            asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
        }
    }
    fence_before();
    __syncthreads();
    if constexpr (PAIR) cluster_sync_all();  // the peer's barriers are initialised
    fence_after();
    const uint32_t tmem_base = s_tmem;
    const uint64_t limit = p.wait_ns;
    // drains after an abort wait for work that is already in flight (it completes in
    // microseconds); their bound does not shrink with a short user wait limit
    const uint64_t drain_limit = limit > 200000000ull ? limit : 200000000ull;

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            int issued_phase[NST];
            for (int s = 0; s < NST; ++s) issued_phase[s] = -1;
            // K-variable pair peer: stages whose own barrier was ever armed, and per stage
            // the parity of the next phase to arm
            uint32_t parmed = 0, pnext = 0;
            bool ok = true;
            // every TMA load is counted on the leader's full barrier (CTA 0 of a pair)
            bool local_bar = false;  // this stage's copies complete on this CTA's own barrier
            auto load = [&](uint32_t dst, const CUtensorMap* map, uint32_t fb, int c0, int c1) {
                if (PAIR && !local_bar) tma_load_2d_pair(dst, map, fb, c0, c1);
                else tma_load_2d(dst, map, fb, c0, c1);
            };
            for (int t = tile0; t < total_tiles && ok; t += tile_step) {
                const Tile ti = tile_at(t);
                for (int kb = 0; kb < ti.k_iters; ++kb) {
                    if (!wait_bar(empty_bar(stage), phase ^ 1u)) {
                        ok = false;
                        break;
                    }
                    const uint32_t sa = ring + stage * STAGE_BYTES;
                    const uint32_t sb = sa + A_BYTES;
                    // K-variable pair, peer, partial last k-block: its copies land on its own
                    // barrier; the MMA warp zeroes the rows past the group's end and then
                    // credits these bytes to the leader's full barrier
                    const bool part_peer = PAIR && VAR_K && rank == 1 && kb == ti.k_iters - 1 && ti.last_rows < KB;
                    const uint32_t fb = part_peer ? pfull_bar(stage)
                                                  : (PAIR ? map_to_rank(full_bar(stage), 0) : full_bar(stage));
                    local_bar = part_peer;
                    // In a pair only the leader arrives, expecting the bytes of both CTAs: the
                    // peer's copies complete on the leader's barrier without an arrival (a
                    // cluster-scope arrive per stage cost the producers most of their time). The
                    // peer reuses a stage only after the leader's MMAs released it, so its bytes
                    // always count towards the phase the leader arms.
                    if constexpr (PAIR) {
                        if (rank == 0) mbar_expect_tx(full_bar(stage), NPAIR * STAGE_BYTES);
                        else if (part_peer) {
                            mbar_expect_tx(fb, STAGE_BYTES);
                            parmed |= 1u << stage;
                            pnext ^= 1u << stage;
                        }
                    } else if constexpr (EPI == EPI_ROUTE) {
                        mbar_expect_tx(fb, (uint32_t)p.tile_rows * 128u * KPS + B_BYTES);  // A boxes of tile_rows rows
                    } else {
                        mbar_expect_tx(fb, STAGE_BYTES);
                    }
                    const int k0 = kb * KB * KPS;
                    const bool dw = DW2 && ti.dw;
                    if (!A_MN && !dw) {
#pragma unroll
                        for (int i = 0; i < KPS; ++i) load(sa + i * A_BOX, &tmA, fb, k0 + KB * i, (int)(ti.a_row + ti.m0));
                    } else {
                        const CUtensorMap* mA = dw ? &tmA2 : &tmA;
#pragma unroll
                        for (int i = 0; i < BM / 64; ++i)
                            load(sa + i * ATOM, mA, fb, ti.m0 + 64 * i, (int)(ti.a_row + k0));
                    }
                    if (EPI == EPI_SWIGLU_FWD) {
                        // 128 gate rows then 128 up rows of the same features; in a pair the
                        // leader holds the gate half and the peer the up half
                        const int64_t r = (int64_t)ti.we * p.b_group_rows + ti.n0;
                        if constexpr (PAIR) {
#pragma unroll
                            for (int j = 0; j < KPS; ++j)
                                load(sb + j * B_BOX, &tmB, fb, k0 + KB * j, (int)(r + (rank ? p.F : 0)));
                        } else {
                            load(sb, &tmB, fb, k0, (int)r);
                            load(sb + 128 * 128, &tmB, fb, k0, (int)(r + p.F));
                        }
                    } else if (!B_MN) {
#pragma unroll
                        for (int i = 0; i < KPS; ++i)
                            load(sb + i * B_BOX, &tmB, fb, k0 + KB * i,
                                 (int)((int64_t)ti.we * p.b_group_rows + ti.n0 + rank * BNL));
                    } else {
                        const int64_t krow = (VAR_K || dw) ? (ti.b_row + k0) : ((int64_t)ti.we * p.b_group_rows + k0);
                        const CUtensorMap* mB = dw ? &tmB2 : &tmB;
#pragma unroll
                        for (int j = 0; j < KPS; ++j)
#pragma unroll
                            for (int i = 0; i < BNL / 64; ++i)
                                load(sb + j * B_BOX + i * ATOM, mB, fb, ti.n0 + (int)rank * BNL + 64 * i,
                                     (int)(krow + KB * j));
                    }
                    issued_phase[stage] = (int)phase;
                    if (++stage == NST) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
            }
            if constexpr (PAIR && VAR_K) {
                if ((!ok || *abort_flag) && rank == 1) {
                    // partial copies on this CTA's own barriers: the last phase armed
                    for (int s2 = 0; s2 < NST; ++s2) {
                        if (!((parmed >> s2) & 1u)) continue;
                        const uint32_t par = ((pnext >> s2) & 1u) ^ 1u;
                        const uint64_t t0 = gtimer();
                        while (!mbar_try(pfull_bar(s2), par) && gtimer() - t0 < drain_limit) {
                        }
                    }
                }
            }
            if ((!ok || *abort_flag) && rank == 0) {
                // let every copy started into this pair land before the CTAs exit (the
                // leader's full barriers count the peer's bytes too)
                for (int s = 0; s < NST; ++s) {
                    if (issued_phase[s] < 0) continue;
                    const uint64_t t0 = gtimer();
                    while (!mbar_try(full_bar(s), (uint32_t)issued_phase[s]) &&
                           gtimer() - t0 < drain_limit) {
                    }
                }
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        int stage = 0;
        uint32_t phase = 0;
        int acc = 0;
        uint32_t acc_phase = 0;
        bool ok = true;
        bool issued_any = false;
        // in a pair only the leader issues MMAs (they read both CTAs' shared memory and
        // write both CTAs' TMEM)
        for (int t = tile0; t < total_tiles && ok && rank == 0; t += tile_step) {
            const Tile ti = tile_at(t);
            if (!wait_bar(tempty_bar(acc), acc_phase ^ 1u)) {
                ok = false;
                break;
            }
            fence_after();
            const uint32_t tmem_d = tmem_base + (uint32_t)(acc * BN);
            for (int kb = 0; kb < ti.k_iters; ++kb) {
                if (!wait_bar(full_bar(stage), phase)) {
                    ok = false;
                    break;
                }
                const uint32_t sa = ring + stage * STAGE_BYTES;
                const uint32_t sb = sa + A_BYTES;
                // K-variable groups: the last k-block may hold contraction rows of the next
                // group. Only K=16 steps that contain valid rows are issued, and inside the
                // last of them the A rows past the group's end are zeroed (A alone suffices:
                // their products with any finite B row vanish).
                int ksteps = KB * KPS / 16;
                const bool dwt = DW2 && ti.dw;
                if ((VAR_K || dwt) && kb == ti.k_iters - 1 && ti.last_rows < KB) {
                    ksteps = (ti.last_rows + 15) / 16;
                    const int zr0 = ti.last_rows, zr1 = ksteps * 16;
                    if (zr1 > zr0) {
                        uint8_t* base = ring_ptr + (size_t)stage * STAGE_BYTES;
                        const int per_box = (zr1 - zr0) * 8;  // 16-byte words
#pragma unroll
                        for (int b = 0; b < BM / 64; ++b) {
                            uint4* z = reinterpret_cast<uint4*>(base + b * ATOM + zr0 * 128);
                            for (int i = lane; i < per_box; i += 32) z[i] = make_uint4(0, 0, 0, 0);
                        }
                        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                    }
                    __syncwarp();
                }
                fence_after();
                if (lane == 0) {
#pragma unroll
                    for (int kk = 0; kk < KB * KPS / 16; ++kk) {
                        if (kk >= ksteps) break;
                        uint64_t ad, bd;
                        if (!A_MN && !dwt) ad = smem_desc(sa + (kk / (KB / 16)) * A_BOX + (kk % (KB / 16)) * 32, 16, 1024);
                        else ad = smem_desc(sa + (kk / (KB / 16)) * A_BOX + (kk % (KB / 16)) * 2048, ATOM, 1024);
                        if (!B_MN) bd = smem_desc(sb + (kk / (KB / 16)) * B_BOX + (kk % (KB / 16)) * 32, 16, 1024);
                        else bd = smem_desc(sb + (kk / (KB / 16)) * B_BOX + (kk % (KB / 16)) * 2048, ATOM, 1024);
                        if constexpr (PAIR) mma_bf16_pair(tmem_d, ad, bd, IDESC, (kb | kk) ? 1u : 0u);
                        else mma_bf16(tmem_d, ad, bd, dwt ? IDESC_DW : IDESC, (kb | kk) ? 1u : 0u);
                    }
                    if constexpr (PAIR) mma_commit_pair(empty_bar(stage), 3);  // both producers
                    else mma_commit(empty_bar(stage));
                    issued_any = true;
                }
                __syncwarp();
                if (++stage == NST) {
                    stage = 0;
                    phase ^= 1u;
                }
            }
            if (!ok) break;
            if (lane == 0) {
                if constexpr (PAIR) {
                    mma_commit_pair(tfull_bar(acc), 3);  // both CTAs' epilogues
                } else {
                    if (ti.k_iters > 0) mma_commit(tfull_bar(acc));
                    else mbar_arrive(tfull_bar(acc));
                }
            }
            __syncwarp();
            if (++acc == 2) {
                acc = 0;
                acc_phase ^= 1u;
            }
        }
        if ((!ok || *abort_flag) && lane == 0 && issued_any) {
            // wait for every MMA this CTA issued before TMEM is released
            if constexpr (PAIR) mma_commit_pair(drain_bar, 1);
            else mma_commit(drain_bar);
            const uint64_t t0 = gtimer();
            while (!mbar_try(drain_bar, 0) && gtimer() - t0 < drain_limit) {
            }
        }
        __syncwarp();
        if constexpr (PAIR && VAR_K) {
            // Peer of a K-variable pair: the leader's MMAs read this CTA's A rows too, so
            // the rows of a tile's last k-block past its group's end are zeroed here, as
            // the leader does for its own; then this stage's bytes are credited to the
            // leader's full barrier, which the peer's copies did not count.
            if (rank == 1) {
                int st2 = 0;
                uint32_t wpar = 0;  // per stage: parity of the next partial phase to wait for
                bool ok2 = true;
                for (int t = tile0; t < total_tiles && ok2; t += tile_step) {
                    const Tile ti = tile_at(t);
                    for (int kb = 0; kb < ti.k_iters; ++kb) {
                        if (kb == ti.k_iters - 1 && ti.last_rows < KB) {
                            if (!mbar_wait(pfull_bar(st2), (wpar >> st2) & 1u, abort_flag, p.wait_ns)) {
                                ok2 = false;
                                break;
                            }
                            wpar ^= 1u << st2;
                            const int zr0 = ti.last_rows, zr1 = ((ti.last_rows + 15) / 16) * 16;
                            if (zr1 > zr0) {
                                uint8_t* base = ring_ptr + (size_t)st2 * STAGE_BYTES;
                                const int per_box = (zr1 - zr0) * 8;  // 16-byte words
#pragma unroll
                                for (int b = 0; b < BM / 64; ++b) {
                                    uint4* z = reinterpret_cast<uint4*>(base + b * ATOM + zr0 * 128);
                                    for (int i = lane; i < per_box; i += 32) z[i] = make_uint4(0, 0, 0, 0);
                                }
                                asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                            }
                            __syncwarp();
                            if (lane == 0) {
                                asm volatile("fence.acq_rel.cluster;" ::: "memory");
                                mbar_complete_tx_remote(map_to_rank(full_bar(st2), 0), STAGE_BYTES);
                            }
                            __syncwarp();
                        }
                        if (++st2 == NST) st2 = 0;
                    }
                }
            }
        }
    } else {
        // ------------------------------------------------------------ epilogue warps 2-5
        // Warp w reads TMEM lane quarter w % 4 (32 rows). Finished 32x32 bf16 boxes are
        // staged in shared memory and written by TMA stores; a box that reaches past the
        // group's last row (the last M tile of an expert) is written row by row instead.
        const int q = warp & 3;
        const int row_local = q * 32 + lane;
        uint8_t* stg = stage_out + (size_t)(warp - 2) * epi_stage_bytes(EPI);
        const uint32_t stg_u32 = smem_u32(stg);
        int acc = 0;
        uint32_t acc_phase = 0;
        uint32_t box_seq = 0;  // output boxes this warp has staged (ring position)
        // SwiGLU backward: TMA loads of G/U chunk boxes into two staging buffers
        const uint32_t gu_bar0 = bar0 + 8u * (2 * NST + 5 + 2 * (warp - 2));
        uint32_t gu_issued = 0;  // chunks whose loads were issued (this warp)
        uint32_t gu_chunk = 0;   // chunks consumed
        auto gu_issue = [&](const Tile& tn, int cn) {
            if constexpr (EPI == EPI_SWIGLU_BWD) {
                const int b = gu_issued & 1;
                if (lane == 0) {
                    bulk_wait_read0();  // earlier stores out of this buffer have read it
                    const uint32_t dst = stg_u32 + (2 * b) * EPI_BUF_BYTES;
                    const int row0 = (int)(tn.out_row + tn.m0 + q * 32);
                    mbar_expect_tx(gu_bar0 + 8u * b, 2 * EPI_BUF_BYTES);
                    tma_load_2d(dst, &tmO1, gu_bar0 + 8u * b, tn.n0 + 32 * cn, row0);
                    tma_load_2d(dst + EPI_BUF_BYTES, &tmO1, gu_bar0 + 8u * b, p.F + tn.n0 + 32 * cn, row0);
                }
                ++gu_issued;
            }
        };
        auto gu_wait = [&](int b, uint32_t parity) -> bool {
            return mbar_wait(gu_bar0 + 8u * b, parity, abort_flag, limit);
        };
        if constexpr (EPI == EPI_SWIGLU_BWD) {
            if (tile0 < total_tiles) {
                const Tile tf = tile_at(tile0);
                if (!(DW2 && tf.dw)) gu_issue(tf, 0);
            }
        }
        for (int t = tile0; t < total_tiles; t += tile_step) {
            const Tile ti = tile_at(t);
            const int m = ti.m0 + row_local;
            const bool valid = m < ti.mvalid;
            const int wrow0 = ti.m0 + q * 32;
            const bool full_box = wrow0 + 32 <= ti.mvalid;
            const bool dwt = DW2 && ti.dw;
            const int64_t grow0 = (VAR_K || dwt) ? (int64_t)ti.we * (dwt ? p2.Mout : p.Mout) + wrow0
                                                 : ti.out_row + wrow0;
            const uint32_t tbase = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * BN);
            // write NOUT rows of 32 values each: staged + TMA when the whole box is valid
            auto emit = [&](int nout, const float* const* vals, const CUtensorMap* const* maps,
                            const int* cols, __nv_bfloat16* const* direct) {
                if (full_box) {
#pragma unroll
                    for (int o = 0; o < nout; ++o) {
                        const uint32_t b = box_seq & (EPI_NBUF - 1);
                        // the store that last used box b (EPI_NBUF boxes ago) has read it
                        if (lane == 0) bulk_wait_read<EPI_NBUF - 1>();
                        __syncwarp();
                        store_row32_sw64(stg + b * EPI_BUF_BYTES + lane * 64, lane, vals[o]);
                        fence_proxy_async();
                        __syncwarp();
                        if (lane == 0) {
                            tma_store_2d(maps[o], stg_u32 + b * EPI_BUF_BYTES, cols[o], (int)grow0);
                            bulk_commit();
                        }
                        ++box_seq;
                    }
                } else if (valid) {
                    for (int o = 0; o < nout; ++o) store_row32(direct[o], vals[o]);
                }
            };
            if (dwt) {
                // second problem: a bf16 weight-gradient tile, [Mout, N] per group
                if (!wait_bar(tfull_bar(acc), acc_phase)) break;
                fence_after();
                __nv_bfloat16* out = (__nv_bfloat16*)p2.out0 + (int64_t)ti.we * p2.Mout * p2.N + (int64_t)m * p2.N;
#pragma unroll 1
                for (int c = 0; c < BN; c += 32) {
                    float y[32];
                    if (ti.k_iters > 0) {
                        tmem_ld32(tbase + c, y);
                    } else {
#pragma unroll
                        for (int i = 0; i < 32; ++i) y[i] = 0.f;
                    }
                    const float* vals[1] = {y};
                    const CUtensorMap* maps[1] = {&tmO2};
                    const int cols[1] = {ti.n0 + c};
                    __nv_bfloat16* direct[1] = {out + ti.n0 + c};
                    emit(1, vals, maps, cols, direct);
                }
            } else if constexpr (EPI == EPI_SWIGLU_BWD) {
                // dA in TMEM. G and U of each 32-column chunk arrive by TMA in one of two
                // staging buffers (the next chunk's load is in flight while this one is
                // computed); dG and dU overwrite them in place and leave by TMA store.
                const int F = p.F;
                __nv_bfloat16* dh = (__nv_bfloat16*)p.out0 + (ti.out_row + m) * (int64_t)(2 * F) + ti.n0;
                constexpr int NCH = BN / 32;
                const int nchv = min(NCH, (F - ti.n0) / 32);  // chunks inside F (a ragged last tile)
                if (gu_issued == gu_chunk) gu_issue(ti, 0);  // not prefetched (a fused tile came before)
                if (!wait_bar(tfull_bar(acc), acc_phase)) break;
                fence_after();
                bool stop = false;
#pragma unroll 1
                for (int c = 0; c < nchv; ++c) {
                    // prefetch the next chunk (of this tile, or the first of the next tile)
                    if (c + 1 < nchv) gu_issue(ti, c + 1);
                    else if (t + tile_step < total_tiles) {
                        const Tile tn = tile_at(t + tile_step);
                        if (!(DW2 && tn.dw)) gu_issue(tn, 0);
                    }
                    const int b = gu_chunk & 1;
                    if (!gu_wait(b, (gu_chunk >> 1) & 1)) { stop = true; break; }
                    uint8_t* gbuf = stg + (2 * b) * EPI_BUF_BYTES + lane * 64;
                    uint8_t* ubuf = gbuf + EPI_BUF_BYTES;
                    float da[32], dG[32], dU[32];
                    tmem_ld32(tbase + 32 * c, da);
#pragma unroll
                    for (int v = 0; v < 4; ++v) {
                        const int sw = (v ^ ((lane >> 1) & 3)) << 4;
                        float G[8], U[8];
                        unpack8(*reinterpret_cast<const uint4*>(gbuf + sw), G);
                        unpack8(*reinterpret_cast<const uint4*>(ubuf + sw), U);
#pragma unroll
                        for (int i = 0; i < 8; ++i) {
                            const float sg = __fdividef(1.0f, 1.0f + __expf(-G[i]));
                            const float d = da[8 * v + i];
                            dU[8 * v + i] = d * G[i] * sg;
                            dG[8 * v + i] = d * U[i] * sg * (1.0f + G[i] * (1.0f - sg));
                        }
                    }
                    if (full_box) {
                        store_row32_sw64(gbuf, lane, dG);
                        store_row32_sw64(ubuf, lane, dU);
                        fence_proxy_async();
                        __syncwarp();
                        if (lane == 0) {
                            const uint32_t src = stg_u32 + (2 * b) * EPI_BUF_BYTES;
                            tma_store_2d(&tmO0, src, ti.n0 + 32 * c, (int)grow0);
                            tma_store_2d(&tmO0, src + EPI_BUF_BYTES, F + ti.n0 + 32 * c, (int)grow0);
                            bulk_commit();
                        }
                    } else if (valid) {
                        store_row32(dh + 32 * c, dG);
                        store_row32(dh + F + 32 * c, dU);
                    }
                    __syncwarp();
                    ++gu_chunk;
                }
                if (stop) break;
            } else {
                if (!wait_bar(tfull_bar(acc), acc_phase)) break;
                fence_after();
                if constexpr (EPI == EPI_SWIGLU_FWD) {
                    // accumulator columns [0,128) = G, [128,256) = U of features n0 .. n0+127
                    const int F = p.F;
                    __nv_bfloat16* hgu = (__nv_bfloat16*)p.out0 + (ti.out_row + m) * (int64_t)(2 * F);
                    __nv_bfloat16* actp = (__nv_bfloat16*)p.out1 + (ti.out_row + m) * (int64_t)F;
#pragma unroll 1
                    for (int c = 0; c < 128; c += 32) {
                        float g[32], u[32], a[32];
                        tmem_ld32(tbase + c, g);
                        tmem_ld32(tbase + 128 + c, u);
#pragma unroll
                        for (int i = 0; i < 32; ++i) a[i] = __fdividef(g[i], 1.0f + __expf(-g[i])) * u[i];
                        const int f = ti.n0 + c;
                        const float* vals[3] = {g, u, a};
                        const CUtensorMap* maps[3] = {&tmO0, &tmO0, &tmO1};
                        const int cols[3] = {f, F + f, f};
                        __nv_bfloat16* direct[3] = {hgu + f, hgu + F + f, actp + f};
                        emit(3, vals, maps, cols, direct);
                    }
                } else if constexpr (EPI == EPI_ROUTE) {
                    // the per-(party, expert) counts: a shared-memory histogram when P E fits
                    // (hist_n > 0), else straight to the global counts
                    int* hist = p.hist_n ? route_hist : p.counts;
                    if constexpr (BN <= 64) route_epilogue<BN>(p, ti, m, valid, tbase, hist);
                    else route_epilogue_wide<BN>(p, ti, m, valid, tbase, hist);
                } else if constexpr (EPI == EPI_DWR) {
                    // one token chunk's partial router gradient: accumulator row m is model
                    // column m, column e is expert e; stored transposed, fp32, part[g][e][m]
                    // (a warp's 32 rows are 32 consecutive floats of one expert row)
                    float* part = (float*)p.out0 + (int64_t)ti.g * p.E * p.Mout + m;
#pragma unroll 1
                    for (int c = 0; c < BN; c += 32) {
                        float v[32];
                        if (ti.k_iters > 0) {
                            tmem_ld32(tbase + c, v);
                        } else {
#pragma unroll
                            for (int i = 0; i < 32; ++i) v[i] = 0.f;
                        }
                        if (valid) {
#pragma unroll
                            for (int i = 0; i < 32; ++i)
                                if (c + i < p.E) part[(int64_t)(c + i) * p.Mout] = v[i];
                        }
                    }
                } else {
                    __nv_bfloat16* out;
                    if (VAR_K)
                        out = (__nv_bfloat16*)p.out0 + (int64_t)ti.we * p.Mout * p.N + (int64_t)m * p.N;
                    else
                        out = (__nv_bfloat16*)p.out0 + (ti.out_row + m) * (int64_t)p.N;
#pragma unroll 1
                    for (int c = 0; c < BN && ti.n0 + c < p.N; c += 32) {
                        float y[32];
                        if (ti.k_iters > 0) {
                            tmem_ld32(tbase + c, y);
                        } else {
#pragma unroll
                            for (int i = 0; i < 32; ++i) y[i] = 0.f;
                        }
                        const float* vals[1] = {y};
                        const CUtensorMap* maps[1] = {&tmO0};
                        const int cols[1] = {ti.n0 + c};
                        __nv_bfloat16* direct[1] = {out + ti.n0 + c};
                        emit(1, vals, maps, cols, direct);
                    }
                }
            }
            // release the accumulator: one arrival per warp on the MMA issuer's barrier
            fence_before();
            __syncwarp();
            if (lane == 0) {
                if constexpr (PAIR) mbar_arrive_remote(map_to_rank(tempty_bar(acc), 0));
                else mbar_arrive(tempty_bar(acc));
            }
            if (++acc == 2) {
                acc = 0;
                acc_phase ^= 1u;
            }
        }
        if (lane == 0) bulk_wait0();  // every TMA store of this warp has completed
        if constexpr (EPI == EPI_SWIGLU_BWD) {
            // loads issued but not consumed (only after an abort): let them land
            for (uint32_t c = gu_chunk; c < gu_issued; ++c) {
                const uint64_t t0 = gtimer();
                while (!mbar_try(gu_bar0 + 8u * (c & 1), (c >> 1) & 1) && gtimer() - t0 < drain_limit) {
                }
            }
        }
    }
    fence_before();
    __syncthreads();
    if constexpr (PAIR) cluster_sync_all();  // neither CTA leaves while the pair's MMAs run
    fence_after();
    if (warp == 1) {
        if constexpr (PAIR)
            asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem_base),
                         "r"(TMEM_COLS)
                         : "memory");
        else
            asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base),
                         "r"(TMEM_COLS)
                         : "memory");
    }
    if constexpr (EPI == EPI_ROUTE) {
        for (int i = threadIdx.x; i < p.hist_n; i += blockDim.x)
            if (route_hist[i]) atomicAdd(&p.counts[i], route_hist[i]);
    }
}

// ------------------------------------------------------------------------ host side
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = nullptr;
    if (!fn) {
        void* ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000,
                                             cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = (EncodeTiledFn)ptr;
    }
    return fn;
}

// 2D bf16 tensor [outer, inner] row-major, box {64, box_rows}, 128B swizzle, zero fill
// (operand loads); with store = true a {32, 32} box, 64B swizzle, for the epilogue's TMA stores.
static bool make_map(CUtensorMap* m, const void* base, int64_t inner, int64_t outer, int box_rows,
                     bool store = false) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[2] = {(cuuint64_t)inner, (cuuint64_t)outer};
    cuuint64_t strides[1] = {(cuuint64_t)inner * 2};
    cuuint32_t box[2] = {store ? (cuuint32_t)EPI_BOX : 64u, store ? (cuuint32_t)EPI_BOX : (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1u, 1u};
    CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides,
                    box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                    store ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

static uint64_t g_wait_ns = 2000000000ull;
static int g_pairs = MOE_PAIRS_AUTO;  // CTA-pair tiles for the 256-wide M-variable expert GEMMs

static int sm_count() {
    static int n = 0;
    if (!n) {
        int dev = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
        if (n <= 0) n = 148;
    }
    return n;
}

// M-tiles per band of the tile order for `c` tiles in flight at once (the persistent
// CTAs, or CTA pairs): about sqrt(c).
static int band_for(int c) {
    int b = 1;
    while ((b + 1) * (b + 1) <= c) ++b;
    return b;
}

template <int BN, bool B_MN, bool VAR_K, int EPI, bool PAIR = false, bool DW2 = false, int OCC = 1>
static cudaError_t launch(const CUtensorMap& ma, const CUtensorMap& mb, const CUtensorMap& mo0,
                          const CUtensorMap& mo1, const Params& p, int64_t tiles_ub,
                          cudaStream_t s, const CUtensorMap* ma2 = nullptr,
                          const CUtensorMap* mb2 = nullptr, const CUtensorMap* mo2 = nullptr,
                          const Params* p2 = nullptr) {
    auto kern = grouped_gemm_kernel<BN, B_MN, VAR_K, EPI, PAIR, DW2, OCC>;
    const CUtensorMap& A2 = ma2 ? *ma2 : ma;
    const CUtensorMap& B2 = mb2 ? *mb2 : mb;
    const CUtensorMap& O2 = mo2 ? *mo2 : mo0;
    Params P1 = p;
    Params P2 = p2 ? *p2 : p;
    constexpr int NPAIR = PAIR ? 2 : 1;
    constexpr int KB = kblock_rows(VAR_K, PAIR);
    constexpr int STB = (BM * KB * 2 + BN / NPAIR * KB * 2) * kblocks_per_stage(EPI, BN, PAIR, VAR_K);  // bytes of one operand stage
    constexpr int NST = num_stages((uint32_t)STB, EPI, OCC);
    const int extra_max = EPI == EPI_ROUTE ? 64 * 64 * 4 : EPI_WARPS * epi_stage_bytes(EPI);
    const int extra = EPI == EPI_ROUTE ? p.hist_n * 4 : EPI_WARPS * epi_stage_bytes(EPI);
    const int smem_max = NST * STB + 1024 + extra_max;
    const int smem = NST * STB + 1024 + extra;
    static bool attr_set = false;
    if (!attr_set) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_max);
        if (e != cudaSuccess) return e;
        attr_set = true;
    }
    if (tiles_ub <= 0) return cudaSuccess;
    if constexpr (PAIR) {
        // persistent 2-CTA clusters: no more than can be resident at once (a cluster needs
        // both SMs of a TPC, so fewer than SMs/2 may fit)
        static int max_clusters = 0;
        if (!max_clusters) {
            cudaLaunchConfig_t q = {};
            q.gridDim = dim3(2 * (sm_count() / 2));
            q.blockDim = dim3(THREADS);
            q.dynamicSmemBytes = smem_max;
            cudaLaunchAttribute qa[1];
            qa[0].id = cudaLaunchAttributeClusterDimension;
            qa[0].val.clusterDim.x = 2;
            qa[0].val.clusterDim.y = 1;
            qa[0].val.clusterDim.z = 1;
            q.attrs = qa;
            q.numAttrs = 1;
            int n = 0;
            if (cudaOccupancyMaxActiveClusters(&n, kern, &q) != cudaSuccess || n <= 0) {
                (void)cudaGetLastError();
                n = sm_count() / 2;
            }
            max_clusters = n;
        }
        const int clusters = (int)std::min<int64_t>(tiles_ub, max_clusters);
        P1.band = P2.band = band_for(clusters);
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(2 * clusters);
        cfg.blockDim = dim3(THREADS);
        cfg.dynamicSmemBytes = smem;
        cfg.stream = s;
        cudaLaunchAttribute attr[2];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = 2;
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = 1;
        attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[1].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 2;
        return cudaLaunchKernelEx(&cfg, kern, ma, mb, mo0, mo1, P1, A2, B2, O2, P2);
    } else {
        const int grid = (int)std::min<int64_t>(tiles_ub, (int64_t)OCC * sm_count());
        P1.band = P2.band = band_for(grid);
        (void)launch_pdl(kern, dim3(grid), dim3(THREADS), smem, s, ma, mb, mo0, mo1, P1, A2, B2, O2, P2);
        return cudaGetLastError();
    }
}

}  // namespace tc

void set_wait_limit_ns(uint64_t ns) { tc::g_wait_ns = ns ? ns : 1; }
void set_gemm_pairs(int mode) { tc::g_pairs = mode; }

// Pair tiles where they fill at least four rounds of the SMs (the last, partly empty
// round then costs little) and the operand feed, not the epilogue, bounds the tile.
// The input-gradient GEMM (plain store, MN-major weights, a long contraction) takes
// pairs with fewer tiles too: an SM ingests at most ~145 GB/s from L2 with TMA, which
// caps a single-CTA 128 x 256 tile near 80% of the MMA rate and a pair's 256 x 256 tile
// (half the B bytes per SM) does not, and its weight-gradient partner then runs beside
// it on the second stream. The SwiGLU-backward GEMM (dA) moves G, U, dG and dU in its
// epilogue: with a short contraction (d < 2048) the epilogue bounds it and single-CTA
// tiles fused with dW2 in one launch are faster; from d = 2048 the mainloop dominates
// and pairs win (d = 4096: the expert backward 17.8 -> 17.2 ms; d = 1024: +4%).
bool gemm_m_uses_pairs(const GemmMArgs& g) {
    using namespace tc;
    if (g.N % 128 != 0) return false;  // 256-wide pair tiles, the last one possibly ragged
    if (g_pairs == MOE_PAIRS_ALL) return true;
    if (g_pairs != MOE_PAIRS_AUTO) return false;
    if (g.epi == EPI_SWIGLU_BWD && g.K < 2048) return false;
    if (g.epi == EPI_STORE && !g.b_kmajor && g.K >= 512) return true;
    const int64_t pt_ub = g.rows.offsets ? ((int64_t)g.rows.rows + 2 * BM - 1) / (2 * BM) + g.G
                                         : (int64_t)g.G * ((g.rows.rows + 2 * BM - 1) / (2 * BM));
    return pt_ub * ((g.N + 255) / 256) >= 4 * (int64_t)(sm_count() / 2);
}

// K-variable weight gradients (dW = A^T B over each group's rows) as 256 x 256 CTA-pair
// tiles: both output dimensions multiples of 256, and (AUTO) at least four rounds of
// pair tiles.
bool gemm_k_uses_pairs(const GemmKArgs& g) {
    using namespace tc;
    if (g.epi != EPI_STORE || g.M % 256 != 0 || g.N % 128 != 0) return false;
    if (g_pairs == MOE_PAIRS_ALL) return true;
    if (g_pairs != MOE_PAIRS_AUTO) return false;
    return (int64_t)g.G * (g.M / 256) * ((g.N + 255) / 256) >= 4 * (int64_t)(sm_count() / 2);
}

// M-variable grouped GEMM (forward, dA, dX).
cudaError_t launch_gemm_m(const GemmMArgs& g, bool bf16, cudaStream_t s) {
    if (!bf16) return launch_gemm_m_simt(g, s);
    using namespace tc;
    if (g.G > MAX_GROUPS) return cudaErrorInvalidValue;
    Params p{};
    p.offsets = g.rows.offsets;
    p.rows = g.rows.offsets ? 0 : g.rows.rows;
    p.a_stride = g.rows.a_stride;
    p.b_stride = g.rows.b_stride;
    p.out_stride = g.rows.out_stride;
    p.G = g.G;
    p.N = g.N;
    p.K = g.K;
    p.out0 = g.out0;
    p.out1 = g.out1;
    p.aux = g.aux;
    p.wait_ns = g_wait_ns;
    p.gexp = g.group_expert;
    p.a_row_bytes = (int64_t)g.K * 2;
    p.b_all_bytes = (int64_t)g.N * (g.b_kmajor ? g.K : (g.b_rows ? g.b_rows : g.K)) * 2;
    // A rows in the 2D view: OFFSETS -> all routed rows; UNIFORM -> groups * stride (or rows)
    const int64_t a_rows = g.rows.offsets ? (int64_t)g.rows.rows
                                          : std::max<int64_t>(g.rows.rows, (int64_t)(g.G - 1) * g.rows.a_stride + g.rows.rows);
    const int64_t mt_ub = g.rows.offsets ? ((int64_t)g.rows.rows + BM - 1) / BM + g.G
                                         : (int64_t)g.G * ((g.rows.rows + BM - 1) / BM);
    // pair tiles (256 rows)
    const int64_t pt_ub = g.rows.offsets ? ((int64_t)g.rows.rows + 2 * BM - 1) / (2 * BM) + g.G
                                         : (int64_t)g.G * ((g.rows.rows + 2 * BM - 1) / (2 * BM));
    const bool pair = gemm_m_uses_pairs(g);
    // output rows in the 2D view of the outputs
    const int64_t o_rows = g.rows.offsets ? (int64_t)g.rows.rows
                                          : std::max<int64_t>(g.rows.rows, (int64_t)(g.G - 1) * g.rows.out_stride + g.rows.rows);
    CUtensorMap ma, mb, mo0, mo1;
    if (!make_map(&ma, g.a, g.K, a_rows, BM)) return cudaErrorInvalidValue;
    if (g.epi == EPI_SWIGLU_FWD) {
        const int F = g.N / 2;
        p.F = F;
        p.b_group_rows = 2 * (int64_t)F;
        if (!make_map(&mb, g.b, g.K, (int64_t)g.G * 2 * F, 128)) return cudaErrorInvalidValue;
        if (!make_map(&mo0, g.out0, 2 * (int64_t)F, o_rows, 0, true)) return cudaErrorInvalidValue;
        if (!make_map(&mo1, g.out1, F, o_rows, 0, true)) return cudaErrorInvalidValue;
        if (pair) return launch<256, false, false, EPI_SWIGLU_FWD, true>(ma, mb, mo0, mo1, p, pt_ub * (F / 128), s);
        return launch<256, false, false, EPI_SWIGLU_FWD>(ma, mb, mo0, mo1, p, mt_ub * (F / 128), s);
    }
    if (g.epi == EPI_STORE && g.b_kmajor) {  // Y = A W2^T: B = W2[e] as [N=d, K=F]
        p.b_group_rows = g.N;
        if (!make_map(&mo0, g.out0, g.N, o_rows, 0, true)) return cudaErrorInvalidValue;
        if (pair) {
            if (!make_map(&mb, g.b, g.K, (int64_t)g.G * g.N, 128)) return cudaErrorInvalidValue;
            return launch<256, false, false, EPI_STORE, true>(ma, mb, mo0, mo0, p, pt_ub * ((g.N + 255) / 256), s);
        }
        if (g.N % 256 == 0) {
            if (!make_map(&mb, g.b, g.K, (int64_t)g.G * g.N, 256)) return cudaErrorInvalidValue;
            return launch<256, false, false, EPI_STORE>(ma, mb, mo0, mo0, p, mt_ub * (g.N / 256), s);
        }
        if (!make_map(&mb, g.b, g.K, (int64_t)g.G * g.N, 128)) return cudaErrorInvalidValue;
        return launch<128, false, false, EPI_STORE>(ma, mb, mo0, mo0, p, mt_ub * (g.N / 128), s);
    }
    // MN-major B: weights stored [G*K, N] (or [G*b_rows, N])
    p.b_group_rows = g.b_rows ? g.b_rows : g.K;
    if (!make_map(&mb, g.b, g.N, (int64_t)g.G * p.b_group_rows, 64)) return cudaErrorInvalidValue;
    if (g.epi == EPI_SWIGLU_BWD) {
        p.F = g.N;
        if (!make_map(&mo0, g.out0, 2 * (int64_t)g.N, o_rows, 0, true)) return cudaErrorInvalidValue;
        if (!make_map(&mo1, g.aux, 2 * (int64_t)g.N, o_rows, 0, true)) return cudaErrorInvalidValue;
        if (pair)
            return launch<256, true, false, EPI_SWIGLU_BWD, true>(ma, mb, mo0, mo1, p, pt_ub * ((g.N + 255) / 256), s);
        if (g.N % 256 == 0) return launch<256, true, false, EPI_SWIGLU_BWD>(ma, mb, mo0, mo1, p, mt_ub * (g.N / 256), s);
        return launch<128, true, false, EPI_SWIGLU_BWD>(ma, mb, mo0, mo1, p, mt_ub * (g.N / 128), s);
    }
    if (!make_map(&mo0, g.out0, g.N, o_rows, 0, true)) return cudaErrorInvalidValue;
    if (g.slim && g.N % 128 == 0)
        return launch<128, true, false, EPI_STORE, false, false, 2>(ma, mb, mo0, mo0, p, mt_ub * (g.N / 128), s);
    if (pair) return launch<256, true, false, EPI_STORE, true>(ma, mb, mo0, mo0, p, pt_ub * ((g.N + 255) / 256), s);
    if (g.N % 256 == 0) return launch<256, true, false, EPI_STORE>(ma, mb, mo0, mo0, p, mt_ub * (g.N / 256), s);
    return launch<128, true, false, EPI_STORE>(ma, mb, mo0, mo0, p, mt_ub * (g.N / 128), s);
}

// K-variable grouped GEMM (dW1, dW2).
cudaError_t launch_gemm_k(const GemmKArgs& g, bool bf16, cudaStream_t s) {
    if (!bf16) return launch_gemm_k_simt(g, s);
    using namespace tc;
    if (g.G > MAX_GROUPS) return cudaErrorInvalidValue;
    Params p{};
    p.offsets = g.rows.offsets;
    p.rows = g.rows.offsets ? 0 : g.rows.rows;
    p.a_stride = g.rows.a_stride;
    p.b_stride = g.rows.b_stride;
    p.G = g.G;
    p.N = g.N;
    p.Mout = g.M;
    p.out0 = g.out;
    p.wait_ns = g_wait_ns;
    p.gexp = g.group_expert;
    p.a_row_bytes = (int64_t)g.M * 2;
    p.b_row_bytes = (int64_t)g.N * 2;
    const int64_t rows_a = g.rows.offsets ? (int64_t)g.rows.rows
                                          : std::max<int64_t>(g.rows.rows, (int64_t)(g.G - 1) * g.rows.a_stride + g.rows.rows);
    const int64_t rows_b = g.rows.offsets ? (int64_t)g.rows.rows
                                          : std::max<int64_t>(g.rows.rows, (int64_t)(g.G - 1) * g.rows.b_stride + g.rows.rows);
    CUtensorMap ma, mb, mo;
    const bool pair = g.epi == EPI_STORE && gemm_k_uses_pairs(g);
    const int kbr = kblock_rows(true, pair);  // box rows of the MN-major operands
    if (!make_map(&ma, g.a, g.M, rows_a, kbr)) return cudaErrorInvalidValue;
    if (!make_map(&mb, g.b, g.N, rows_b, kbr)) return cudaErrorInvalidValue;
    const int64_t tiles = (int64_t)g.G * (g.M / BM);
    if (g.epi == EPI_DWR) {  // fp32 partials, N = 64, 128 or 256 (experts, zero-padded)
        if ((g.N != 64 && g.N != 128 && g.N != 256) || g.M % BM) return cudaErrorInvalidValue;
        p.E = g.E;
        // two CTAs per SM where TMEM allows: each streams its token chunk of x from HBM at
        // a per-CTA rate, and every tile is resident in one round
        if (g.N == 64) return launch<64, true, true, EPI_DWR, false, false, 2>(ma, mb, ma, ma, p, tiles, s);
        if (g.N == 128) return launch<128, true, true, EPI_DWR, false, false, 2>(ma, mb, ma, ma, p, tiles, s);
        return launch<256, true, true, EPI_DWR>(ma, mb, ma, ma, p, tiles, s);
    }
    if (!make_map(&mo, g.out, g.N, (int64_t)g.G * g.M, 0, true)) return cudaErrorInvalidValue;
    if (pair)
        return launch<256, true, true, EPI_STORE, true>(ma, mb, mo, mo, p, (int64_t)g.G * (g.M / 256) * ((g.N + 255) / 256), s);
    if (g.N % 256 == 0) return launch<256, true, true, EPI_STORE>(ma, mb, mo, mo, p, tiles * (g.N / 256), s);
    return launch<128, true, true, EPI_STORE>(ma, mb, mo, mo, p, tiles * (g.N / 128), s);
}

// One launch of an M-variable GEMM with MN-major B (dA with the SwiGLU-backward
// epilogue, or dX) and a K-variable weight-gradient GEMM over the same groups (dW2, or
// dW1); see the DW2 kernel parameter. Falls back to two
// launches when the shapes do not fit one 256-wide template.
cudaError_t launch_gemm_mk(const GemmMArgs& g, const GemmKArgs& k, cudaStream_t s) {
    using namespace tc;
    const bool fits = g.rows.offsets && k.rows.offsets && g.G == k.G && !g.b_kmajor &&
                      (g.epi == EPI_SWIGLU_BWD || g.epi == EPI_STORE) && g.N % 256 == 0 &&
                      k.N % 256 == 0 && k.M % BM == 0 && k.epi == EPI_STORE && g.G <= MAX_GROUPS;
    if (!fits) {
        cudaError_t e = launch_gemm_m(g, true, s);
        if (e != cudaSuccess) return e;
        return launch_gemm_k(k, true, s);
    }
    // first problem (as launch_gemm_m, MN-major B)
    Params p{};
    p.offsets = g.rows.offsets;
    p.G = g.G;
    p.N = g.N;
    p.K = g.K;
    p.out0 = g.out0;
    p.out1 = g.out1;
    p.aux = g.aux;
    p.wait_ns = g_wait_ns;
    p.gexp = g.group_expert;
    p.b_group_rows = g.b_rows ? g.b_rows : g.K;
    p.a_row_bytes = (int64_t)g.K * 2;
    p.b_all_bytes = (int64_t)g.N * p.b_group_rows * 2;
    const int64_t a_rows = (int64_t)g.rows.rows, o_rows = a_rows;
    CUtensorMap ma, mb, mo0, mo1;
    if (!make_map(&ma, g.a, g.K, a_rows, BM)) return cudaErrorInvalidValue;
    if (!make_map(&mb, g.b, g.N, (int64_t)g.G * p.b_group_rows, 64)) return cudaErrorInvalidValue;
    if (g.epi == EPI_SWIGLU_BWD) {
        p.F = g.N;
        if (!make_map(&mo0, g.out0, 2 * (int64_t)g.N, o_rows, 0, true)) return cudaErrorInvalidValue;
        if (!make_map(&mo1, g.aux, 2 * (int64_t)g.N, o_rows, 0, true)) return cudaErrorInvalidValue;
    } else {
        if (!make_map(&mo0, g.out0, g.N, o_rows, 0, true)) return cudaErrorInvalidValue;
        mo1 = mo0;
    }
    // second problem (as launch_gemm_k)
    Params p2{};
    p2.offsets = k.rows.offsets;
    p2.G = k.G;
    p2.N = k.N;
    p2.Mout = k.M;
    p2.out0 = k.out;
    p2.wait_ns = g_wait_ns;
    p2.gexp = k.group_expert;
    p2.a_row_bytes = (int64_t)k.M * 2;
    p2.b_row_bytes = (int64_t)k.N * 2;
    CUtensorMap ma2, mb2, mo2;
    if (!make_map(&ma2, k.a, k.M, (int64_t)k.rows.rows, 64)) return cudaErrorInvalidValue;
    if (!make_map(&mb2, k.b, k.N, (int64_t)k.rows.rows, 64)) return cudaErrorInvalidValue;
    if (!make_map(&mo2, k.out, k.N, (int64_t)k.G * k.M, 0, true)) return cudaErrorInvalidValue;
    const int64_t tiles = (((int64_t)g.rows.rows + BM - 1) / BM + g.G) * (g.N / 256) +
                          (int64_t)k.G * (k.M / BM) * (k.N / 256);
    if (g.epi == EPI_SWIGLU_BWD)
        return launch<256, true, false, EPI_SWIGLU_BWD, false, true>(ma, mb, mo0, mo1, p, tiles, s,
                                                                     &ma2, &mb2, &mo2, &p2);
    return launch<256, true, false, EPI_STORE, false, true>(ma, mb, mo0, mo1, p, tiles, s, &ma2,
                                                            &mb2, &mo2, &p2);
}

// Router logits on the tensor cores with the gating epilogue: groups are parties
// (rows [po[p], po[p+1]) use W_r[p]); N = E rounded up to 16, 32 or 64.
cudaError_t launch_route_tc(const RouteArgs& a, cudaStream_t s) {
    using namespace tc;
    Params p{};
    if (a.po && a.P > 1) {
        p.offsets = a.po;
        p.G = a.P;
    } else {
        p.rows = (int)a.T;
        p.G = 1;
    }
    p.K = a.d;
    p.E = a.E;
    p.k = a.k;
    p.normalize = a.normalize;
    p.hist_n = a.P * a.E <= 64 * 64 ? a.P * a.E : 0;  // else counted in global memory
    p.out0 = a.logits;
    p.out1 = a.probs;
    p.aux = a.bias;
    p.topk_idx = a.topk_idx;
    p.topk_w = a.topk_w;
    p.counts = a.counts;
    p.b_group_rows = a.E;
    p.wait_ns = g_wait_ns;
    const int BNr = a.E <= 16 ? 16 : a.E <= 32 ? 32 : a.E <= 64 ? 64 : a.E <= 128 ? 128 : 256;
    if (a.E > 256) return cudaErrorInvalidValue;
    p.N = BNr;
    // rows per tile: the batch split evenly over the SMs (one tile each) when that is
    // under 128 rows, at least 16
    const int64_t share = (a.T + sm_count() - 1) / sm_count();
    p.tile_rows = (int)std::max<int64_t>(16, std::min<int64_t>(BM, share));
    CUtensorMap ma, mb;
    if (!make_map(&ma, a.x, a.d, a.T, p.tile_rows)) return cudaErrorInvalidValue;
    if (!make_map(&mb, a.w_router, a.d, (int64_t)a.P * a.E, BNr)) return cudaErrorInvalidValue;
    const int64_t tiles = (a.T + p.tile_rows - 1) / p.tile_rows + a.P;
    if (BNr == 16) return launch<16, false, false, EPI_ROUTE>(ma, mb, ma, ma, p, tiles, s);
    if (BNr == 32) return launch<32, false, false, EPI_ROUTE>(ma, mb, ma, ma, p, tiles, s);
    if (BNr == 64) return launch<64, false, false, EPI_ROUTE>(ma, mb, ma, ma, p, tiles, s);
    if (BNr == 128) return launch<128, false, false, EPI_ROUTE>(ma, mb, ma, ma, p, tiles, s);
    return launch<256, false, false, EPI_ROUTE>(ma, mb, ma, ma, p, tiles, s);
}

cudaError_t gemm_status(cudaStream_t s, int* code) { return tu_status_read_clear(s, code); }

}  // namespace moe
