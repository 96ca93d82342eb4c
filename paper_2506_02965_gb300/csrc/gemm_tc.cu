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
constexpr int STAGES = 4;
constexpr int THREADS = 192;
constexpr int MAX_GROUPS = 128;

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
    void* out0;
    void* out1;
    const void* aux;
    uint64_t wait_ns;
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
__device__ __forceinline__ bool mbar_try(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}
// Bounded wait. Returns false when the CTA is aborting (another role gave up) or when
// this wait ran past `limit_ns` (then it raises the abort flag and records TIMEOUT).
__device__ __noinline__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                       uint64_t limit_ns) {
    if (mbar_try(bar, parity)) return true;
    const uint64_t t0 = gtimer();
    for (uint32_t it = 1;; ++it) {
        if (mbar_try(bar, parity)) return true;
        if ((it & 31u) == 0) {
            if (*abort_flag) return false;
            if (gtimer() - t0 > limit_ns) {
                *abort_flag = 1;
                record_status(MOE_ERR_TIMEOUT);
                return false;
            }
        }
    }
}
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, uint32_t bar,
                                            int c0, int c1) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes "
        "[%0], [%1, {%3, %4}], [%2];" ::"r"(dst),
        "l"((uint64_t)map), "r"(bar), "r"(c0), "r"(c1)
        : "memory");
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
template <int BN, bool A_MN, bool B_MN>
__host__ __device__ constexpr uint32_t instr_desc() {
    return (1u << 4) | (1u << 7) | (1u << 10) | ((A_MN ? 1u : 0u) << 15) |
           ((B_MN ? 1u : 0u) << 16) | ((uint32_t)(BN >> 3) << 17) | ((uint32_t)(BM >> 4) << 24);
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
};

// ------------------------------------------------------------------------ the kernel
template <int BN, bool B_MN, bool VAR_K, int EPI>
__global__ void __launch_bounds__(THREADS, 1)
    grouped_gemm_kernel(const __grid_constant__ CUtensorMap tmA,
                        const __grid_constant__ CUtensorMap tmB, const Params p) {
    constexpr bool A_MN = VAR_K;
    constexpr uint32_t A_BYTES = BM * BK * 2;
    constexpr uint32_t B_BYTES = BN * BK * 2;
    constexpr uint32_t STAGE_BYTES = A_BYTES + B_BYTES;
    constexpr uint32_t IDESC = instr_desc<BN, A_MN, B_MN>();
    constexpr int TMEM_COLS = 2 * BN;

    extern __shared__ uint8_t smem_raw[];
    __shared__ uint64_t bars[2 * STAGES + 5];
    __shared__ uint32_t s_tmem;
    __shared__ int s_abort;
    __shared__ int s_tile_start[MAX_GROUPS + 1];

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    volatile int* abort_flag = &s_abort;

    // group -> tile prefix
    const int tiles_n = (EPI == EPI_SWIGLU_FWD) ? p.N / 256 : p.N / BN;
    if (threadIdx.x == 0) {
        int acc = 0;
        for (int g = 0; g < p.G; ++g) {
            s_tile_start[g] = acc;
            int mt;
            if (VAR_K) {
                mt = p.Mout / BM;
            } else {
                const int rows = p.offsets ? (p.offsets[g + 1] - p.offsets[g]) : p.rows;
                mt = rows > 0 ? (rows + BM - 1) / BM : 0;
            }
            acc += mt * tiles_n;
        }
        s_tile_start[p.G] = acc;
        s_abort = 0;
    }
    __syncthreads();
    const int total_tiles = s_tile_start[p.G];
    if ((int)blockIdx.x >= total_tiles) return;

    auto tile_at = [&](int t) -> Tile {
        Tile ti;
        int g = 0;
        while (g + 1 < p.G && s_tile_start[g + 1] <= t) ++g;
        const int local = t - s_tile_start[g];
        const int mt = local / tiles_n, nt = local % tiles_n;
        ti.g = g;
        ti.m0 = mt * BM;
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
            ti.k_iters = (int)((nrows + BK - 1) / BK);
            ti.last_rows = (int)(nrows - (int64_t)(ti.k_iters - 1) * BK);
        } else {
            ti.mvalid = (int)nrows;
            ti.a_row = a0;
            ti.b_row = 0;
            ti.out_row = o0;
            ti.k_iters = p.K / BK;
            ti.last_rows = BK;
        }
        return ti;
    };

    // 1024-byte aligned stage ring
    const uint32_t raw_u32 = smem_u32(smem_raw);
    const uint32_t ring = raw_u32 + ((1024u - (raw_u32 & 1023u)) & 1023u);
    uint8_t* ring_ptr = smem_raw + (ring - raw_u32);
    const uint32_t bar0 = smem_u32(&bars[0]);
    auto full_bar = [&](int s) { return bar0 + 8u * s; };
    auto empty_bar = [&](int s) { return bar0 + 8u * (STAGES + s); };
    auto tfull_bar = [&](int a) { return bar0 + 8u * (2 * STAGES + a); };
    auto tempty_bar = [&](int a) { return bar0 + 8u * (2 * STAGES + 2 + a); };
    const uint32_t drain_bar = bar0 + 8u * (2 * STAGES + 4);

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(full_bar(s), 1);
            mbar_init(empty_bar(s), 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(tfull_bar(a), 1);
            mbar_init(tempty_bar(a), 128);
        }
        mbar_init(drain_bar, 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         smem_u32(&s_tmem)),
                     "r"(TMEM_COLS)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    fence_before();
    __syncthreads();
    fence_after();
    const uint32_t tmem_base = s_tmem;
    const uint64_t limit = p.wait_ns;

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            int issued_phase[STAGES];
            for (int s = 0; s < STAGES; ++s) issued_phase[s] = -1;
            bool ok = true;
            for (int t = blockIdx.x; t < total_tiles && ok; t += gridDim.x) {
                const Tile ti = tile_at(t);
                for (int kb = 0; kb < ti.k_iters; ++kb) {
                    if (!mbar_wait(empty_bar(stage), phase ^ 1u, abort_flag, limit)) {
                        ok = false;
                        break;
                    }
                    const uint32_t sa = ring + stage * STAGE_BYTES;
                    const uint32_t sb = sa + A_BYTES;
                    const uint32_t fb = full_bar(stage);
                    mbar_expect_tx(fb, STAGE_BYTES);
                    const int k0 = kb * BK;
                    if (!A_MN) {
                        tma_load_2d(sa, &tmA, fb, k0, (int)(ti.a_row + ti.m0));
                    } else {
#pragma unroll
                        for (int i = 0; i < BM / 64; ++i)
                            tma_load_2d(sa + i * 8192, &tmA, fb, ti.m0 + 64 * i, (int)(ti.a_row + k0));
                    }
                    if (EPI == EPI_SWIGLU_FWD) {
                        const int64_t r = (int64_t)ti.g * p.b_group_rows + ti.n0;
                        tma_load_2d(sb, &tmB, fb, k0, (int)r);
                        tma_load_2d(sb + 128 * 128, &tmB, fb, k0, (int)(r + p.F));
                    } else if (!B_MN) {
                        tma_load_2d(sb, &tmB, fb, k0, (int)((int64_t)ti.g * p.b_group_rows + ti.n0));
                    } else {
                        const int64_t krow = VAR_K ? (ti.b_row + k0) : ((int64_t)ti.g * p.b_group_rows + k0);
#pragma unroll
                        for (int i = 0; i < BN / 64; ++i)
                            tma_load_2d(sb + i * 8192, &tmB, fb, ti.n0 + 64 * i, (int)krow);
                    }
                    issued_phase[stage] = (int)phase;
                    if (++stage == STAGES) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
            }
            if (!ok || *abort_flag) {
                // let every copy this thread started land before the CTA exits
                for (int s = 0; s < STAGES; ++s) {
                    if (issued_phase[s] < 0) continue;
                    const uint64_t t0 = gtimer();
                    while (!mbar_try(full_bar(s), (uint32_t)issued_phase[s]) &&
                           gtimer() - t0 < limit) {
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
        for (int t = blockIdx.x; t < total_tiles && ok; t += gridDim.x) {
            const Tile ti = tile_at(t);
            if (!mbar_wait(tempty_bar(acc), acc_phase ^ 1u, abort_flag, limit)) {
                ok = false;
                break;
            }
            fence_after();
            const uint32_t tmem_d = tmem_base + (uint32_t)(acc * BN);
            for (int kb = 0; kb < ti.k_iters; ++kb) {
                if (!mbar_wait(full_bar(stage), phase, abort_flag, limit)) {
                    ok = false;
                    break;
                }
                const uint32_t sa = ring + stage * STAGE_BYTES;
                const uint32_t sb = sa + A_BYTES;
                if (VAR_K && kb == ti.k_iters - 1 && ti.last_rows < BK) {
                    // contraction rows past the group's end belong to the next group:
                    // zero them in every 64-row box of A and B before the MMA reads them
                    const int nbox = BM / 64 + BN / 64;
                    const int zero_bytes = (BK - ti.last_rows) * 128;
                    uint8_t* base = ring_ptr + (size_t)stage * STAGE_BYTES;
                    for (int b = 0; b < nbox; ++b) {
                        uint4* z = reinterpret_cast<uint4*>(base + b * 8192 + ti.last_rows * 128);
                        for (int i = lane; i < zero_bytes / 16; i += 32) z[i] = make_uint4(0, 0, 0, 0);
                    }
                    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                    __syncwarp();
                }
                fence_after();
                if (lane == 0) {
#pragma unroll
                    for (int kk = 0; kk < BK / 16; ++kk) {
                        uint64_t ad, bd;
                        if (!A_MN) ad = smem_desc(sa + kk * 32, 16, 1024);
                        else ad = smem_desc(sa + kk * 2048, 8192, 1024);
                        if (!B_MN) bd = smem_desc(sb + kk * 32, 16, 1024);
                        else bd = smem_desc(sb + kk * 2048, 8192, 1024);
                        mma_bf16(tmem_d, ad, bd, IDESC, (kb | kk) ? 1u : 0u);
                    }
                    mma_commit(empty_bar(stage));
                    issued_any = true;
                }
                __syncwarp();
                if (++stage == STAGES) {
                    stage = 0;
                    phase ^= 1u;
                }
            }
            if (!ok) break;
            if (lane == 0) {
                if (ti.k_iters > 0) mma_commit(tfull_bar(acc));
                else mbar_arrive(tfull_bar(acc));
            }
            __syncwarp();
            if (++acc == 2) {
                acc = 0;
                acc_phase ^= 1u;
            }
        }
        if ((!ok || *abort_flag) && lane == 0 && issued_any) {
            // wait for every MMA this CTA issued before TMEM is released
            mma_commit(drain_bar);
            const uint64_t t0 = gtimer();
            while (!mbar_try(drain_bar, 0) && gtimer() - t0 < limit) {
            }
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------------ epilogue (warps 2-5)
        const int q = warp & 3;  // TMEM lane quarter this warp may access
        const int row_local = q * 32 + lane;
        int acc = 0;
        uint32_t acc_phase = 0;
        for (int t = blockIdx.x; t < total_tiles; t += gridDim.x) {
            const Tile ti = tile_at(t);
            if (!mbar_wait(tfull_bar(acc), acc_phase, abort_flag, limit)) break;
            fence_after();
            const uint32_t tbase = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * BN);
            const int m = ti.m0 + row_local;
            const bool valid = m < ti.mvalid;
            if (EPI == EPI_SWIGLU_FWD) {
                const int F = p.F;
                __nv_bfloat16* hgu = (__nv_bfloat16*)p.out0 + (ti.out_row + m) * (int64_t)(2 * F);
                __nv_bfloat16* act = (__nv_bfloat16*)p.out1 + (ti.out_row + m) * (int64_t)F;
#pragma unroll 1
                for (int c = 0; c < 128; c += 32) {
                    float g[32], u[32];
                    tmem_ld32(tbase + c, g);
                    tmem_ld32(tbase + 128 + c, u);
                    if (valid) {
                        const int f = ti.n0 + c;
#pragma unroll
                        for (int v = 0; v < 4; ++v) {
                            float a8[8];
#pragma unroll
                            for (int i = 0; i < 8; ++i) {
                                const float G = g[8 * v + i], U = u[8 * v + i];
                                a8[i] = G / (1.0f + expf(-G)) * U;
                            }
                            Vec<__nv_bfloat16>::store(hgu + f + 8 * v, g + 8 * v);
                            Vec<__nv_bfloat16>::store(hgu + F + f + 8 * v, u + 8 * v);
                            Vec<__nv_bfloat16>::store(act + f + 8 * v, a8);
                        }
                    }
                }
            } else if (EPI == EPI_SWIGLU_BWD) {
                const int F = p.F;
                const __nv_bfloat16* hgu =
                    (const __nv_bfloat16*)p.aux + (ti.out_row + m) * (int64_t)(2 * F);
                __nv_bfloat16* dh = (__nv_bfloat16*)p.out0 + (ti.out_row + m) * (int64_t)(2 * F);
#pragma unroll 1
                for (int c = 0; c < BN; c += 32) {
                    float da[32];
                    tmem_ld32(tbase + c, da);
                    if (valid) {
                        const int f = ti.n0 + c;
#pragma unroll
                        for (int v = 0; v < 4; ++v) {
                            float G[8], U[8], dG[8], dU[8];
                            Vec<__nv_bfloat16>::load(hgu + f + 8 * v, G);
                            Vec<__nv_bfloat16>::load(hgu + F + f + 8 * v, U);
#pragma unroll
                            for (int i = 0; i < 8; ++i) {
                                const float s = 1.0f / (1.0f + expf(-G[i]));
                                const float d = da[8 * v + i];
                                dU[i] = d * G[i] * s;
                                dG[i] = d * U[i] * s * (1.0f + G[i] * (1.0f - s));
                            }
                            Vec<__nv_bfloat16>::store(dh + f + 8 * v, dG);
                            Vec<__nv_bfloat16>::store(dh + F + f + 8 * v, dU);
                        }
                    }
                }
            } else {
                __nv_bfloat16* out;
                if (VAR_K)
                    out = (__nv_bfloat16*)p.out0 + (int64_t)ti.g * p.Mout * p.N + (int64_t)m * p.N;
                else
                    out = (__nv_bfloat16*)p.out0 + (ti.out_row + m) * (int64_t)p.N;
#pragma unroll 1
                for (int c = 0; c < BN; c += 32) {
                    float y[32];
                    if (ti.k_iters > 0) {
                        tmem_ld32(tbase + c, y);
                    } else {
#pragma unroll
                        for (int i = 0; i < 32; ++i) y[i] = 0.f;
                    }
                    if (valid) {
#pragma unroll
                        for (int v = 0; v < 4; ++v)
                            Vec<__nv_bfloat16>::store(out + ti.n0 + c + 8 * v, y + 8 * v);
                    }
                }
            }
            fence_before();
            mbar_arrive(tempty_bar(acc));
            if (++acc == 2) {
                acc = 0;
                acc_phase ^= 1u;
            }
        }
    }
    fence_before();
    __syncthreads();
    fence_after();
    if (warp == 1) {
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base),
                     "r"(TMEM_COLS)
                     : "memory");
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

// 2D bf16 tensor [outer, inner] row-major, box {64, box_rows}, 128B swizzle, zero fill.
static bool make_map(CUtensorMap* m, const void* base, int64_t inner, int64_t outer, int box_rows) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[2] = {(cuuint64_t)inner, (cuuint64_t)outer};
    cuuint64_t strides[1] = {(cuuint64_t)inner * 2};
    cuuint32_t box[2] = {64u, (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1u, 1u};
    CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides,
                    box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

static uint64_t g_wait_ns = 2000000000ull;

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

template <int BN, bool B_MN, bool VAR_K, int EPI>
static cudaError_t launch(const CUtensorMap& ma, const CUtensorMap& mb, const Params& p,
                          int64_t tiles_ub, cudaStream_t s) {
    auto kern = grouped_gemm_kernel<BN, B_MN, VAR_K, EPI>;
    const int smem = STAGES * (BM * BK * 2 + BN * BK * 2) + 1024;
    static bool attr_set = false;
    if (!attr_set) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
        if (e != cudaSuccess) return e;
        attr_set = true;
    }
    if (tiles_ub <= 0) return cudaSuccess;
    const int grid = (int)std::min<int64_t>(tiles_ub, sm_count());
    kern<<<grid, THREADS, smem, s>>>(ma, mb, p);
    return cudaGetLastError();
}

}  // namespace tc

void set_wait_limit_ns(uint64_t ns) { tc::g_wait_ns = ns ? ns : 1; }

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
    // A rows in the 2D view: OFFSETS -> all routed rows; UNIFORM -> groups * stride (or rows)
    const int64_t a_rows = g.rows.offsets ? (int64_t)g.rows.rows
                                          : std::max<int64_t>(g.rows.rows, (int64_t)(g.G - 1) * g.rows.a_stride + g.rows.rows);
    const int64_t mt_ub = g.rows.offsets ? ((int64_t)g.rows.rows + BM - 1) / BM + g.G
                                         : (int64_t)g.G * ((g.rows.rows + BM - 1) / BM);
    CUtensorMap ma, mb;
    if (!make_map(&ma, g.a, g.K, a_rows, BM)) return cudaErrorInvalidValue;
    if (g.epi == EPI_SWIGLU_FWD) {
        const int F = g.N / 2;
        p.F = F;
        p.b_group_rows = 2 * (int64_t)F;
        if (!make_map(&mb, g.b, g.K, (int64_t)g.G * 2 * F, 128)) return cudaErrorInvalidValue;
        return launch<256, false, false, EPI_SWIGLU_FWD>(ma, mb, p, mt_ub * (F / 128), s);
    }
    if (g.epi == EPI_STORE && g.b_kmajor) {  // Y = A W2^T: B = W2[e] as [N=d, K=F]
        p.b_group_rows = g.N;
        if (g.N % 256 == 0) {
            if (!make_map(&mb, g.b, g.K, (int64_t)g.G * g.N, 256)) return cudaErrorInvalidValue;
            return launch<256, false, false, EPI_STORE>(ma, mb, p, mt_ub * (g.N / 256), s);
        }
        if (!make_map(&mb, g.b, g.K, (int64_t)g.G * g.N, 128)) return cudaErrorInvalidValue;
        return launch<128, false, false, EPI_STORE>(ma, mb, p, mt_ub * (g.N / 128), s);
    }
    // MN-major B: weights stored [G*K, N]
    p.b_group_rows = g.K;
    if (!make_map(&mb, g.b, g.N, (int64_t)g.G * g.K, 64)) return cudaErrorInvalidValue;
    if (g.epi == EPI_SWIGLU_BWD) {
        p.F = g.N;
        if (g.N % 256 == 0) return launch<256, true, false, EPI_SWIGLU_BWD>(ma, mb, p, mt_ub * (g.N / 256), s);
        return launch<128, true, false, EPI_SWIGLU_BWD>(ma, mb, p, mt_ub * (g.N / 128), s);
    }
    if (g.N % 256 == 0) return launch<256, true, false, EPI_STORE>(ma, mb, p, mt_ub * (g.N / 256), s);
    return launch<128, true, false, EPI_STORE>(ma, mb, p, mt_ub * (g.N / 128), s);
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
    const int64_t rows_a = g.rows.offsets ? (int64_t)g.rows.rows
                                          : std::max<int64_t>(g.rows.rows, (int64_t)(g.G - 1) * g.rows.a_stride + g.rows.rows);
    const int64_t rows_b = g.rows.offsets ? (int64_t)g.rows.rows
                                          : std::max<int64_t>(g.rows.rows, (int64_t)(g.G - 1) * g.rows.b_stride + g.rows.rows);
    CUtensorMap ma, mb;
    if (!make_map(&ma, g.a, g.M, rows_a, 64)) return cudaErrorInvalidValue;
    if (!make_map(&mb, g.b, g.N, rows_b, 64)) return cudaErrorInvalidValue;
    const int64_t tiles = (int64_t)g.G * (g.M / BM);
    if (g.N % 256 == 0) return launch<256, true, true, EPI_STORE>(ma, mb, p, tiles * (g.N / 256), s);
    return launch<128, true, true, EPI_STORE>(ma, mb, p, tiles * (g.N / 128), s);
}

cudaError_t gemm_status(cudaStream_t s, int* code) { return tu_status_read_clear(s, code); }

}  // namespace moe
