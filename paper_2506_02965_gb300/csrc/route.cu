// Gating function of the MoE layer (Alg. 7) and its backward, plus the per-party
// load-balancing loss. Memory-bound SIMT kernels: x is read once with 16-byte
// vector loads, logits are reduced with warp shuffles, top-k is a warp argmax.
#include <cfloat>

#include <cooperative_groups.h>

#include <algorithm>

#include "moe_common.cuh"
#include "moe_internal.h"

namespace moe {

namespace cg = cooperative_groups;

// ----------------------------------------------------------------------------- top-k
// Per token, lane l owns experts l + 32 i, i < NV (E <= 32 NV). Picks the k largest
// logits, descending, equal logits by ascending expert id; writes logits (optional),
// probs, topk idx / w and bumps the block histogram (or the global counts when the
// histogram does not fit in shared memory).
__device__ __forceinline__ bool better(float va, int ia, float vb, int ib) {
    return va > vb || (va == vb && ia < ib);
}

template <int NV>
__device__ void softmax_topk_token(const float (&z)[NV], int lane, int E, int k, int normalize,
                                   int64_t t, int party, float* logits, float* probs,
                                   int32_t* topk_idx, float* topk_w, int* s_hist) {
    bool val[NV], taken[NV];
#pragma unroll
    for (int i = 0; i < NV; ++i) {
        val[i] = lane + 32 * i < E;
        taken[i] = !val[i];
    }
    if (logits) {
#pragma unroll
        for (int i = 0; i < NV; ++i)
            if (val[i]) logits[t * E + lane + 32 * i] = z[i];
    }
    float m = -FLT_MAX;
#pragma unroll
    for (int i = 0; i < NV; ++i) m = fmaxf(m, val[i] ? z[i] : -FLT_MAX);
    m = warp_max(m);
    float x[NV], loc = 0.f;
#pragma unroll
    for (int i = 0; i < NV; ++i) {
        x[i] = val[i] ? expf(z[i] - m) : 0.f;
        loc += x[i];
    }
    const float s = warp_sum(loc);
    float p[NV];
#pragma unroll
    for (int i = 0; i < NV; ++i) {
        p[i] = x[i] / s;
        if (val[i]) probs[t * E + lane + 32 * i] = p[i];
    }
    float wsel = 0.f, wsum = 0.f;
    int isel = 0;
    for (int j = 0; j < k; ++j) {
        // local candidate
        float cv = -FLT_MAX;
        int ci = 0x7fffffff;
        bool have = false;
#pragma unroll
        for (int i = 0; i < NV; ++i) {
            if (!taken[i] && (!have || better(z[i], lane + 32 * i, cv, ci))) {
                cv = z[i];
                ci = lane + 32 * i;
                have = true;
            }
        }
        int hv = have ? 1 : 0;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            float ov = __shfl_xor_sync(0xffffffffu, cv, o);
            int oi = __shfl_xor_sync(0xffffffffu, ci, o);
            int oh = __shfl_xor_sync(0xffffffffu, hv, o);
            if (oh && (!hv || better(ov, oi, cv, ci))) { cv = ov; ci = oi; hv = 1; }
        }
        // ci is the winner on every lane; its owner lane holds its probability
        const int owner = ci & 31, slot = ci >> 5;
        float mine = 0.f;
#pragma unroll
        for (int i = 0; i < NV; ++i)
            if (i == slot) mine = p[i];
        const float pw = __shfl_sync(0xffffffffu, mine, owner);
#pragma unroll
        for (int i = 0; i < NV; ++i)
            if (ci == lane + 32 * i) taken[i] = true;
        if (lane == j) { isel = ci; wsel = pw; }
        wsum += pw;
        if (lane == 0) atomicAdd(&s_hist[party * E + ci], 1);
    }
    if (lane < k) {
        topk_idx[t * k + lane] = isel;
        topk_w[t * k + lane] = normalize ? wsel / wsum : wsel;
    }
}

// ----------------------------------------------------------------------------- router fwd
// One warp handles a group of up to TPW consecutive tokens of one party. Lane l
// accumulates the dot products of its 16-byte column chunks for every expert, then
// the partial sums are combined with a butterfly (identical bits on every lane).
// FROM_LOGITS: the logits come from logits_in instead ([T,E] fp32); with a bias they
// are the router's raw products (E > 64, computed by a GEMM): the bias is added here
// and the biased logits are written back to `logits` (which may be logits_in).
// The per-(party, expert) counts go through a shared-memory histogram when P E fits
// (HIST_SMEM), else straight to the global counts.
constexpr int HIST_SMEM = 4096;
template <typename T, int EMAX, int TPW, bool FROM_LOGITS>
__global__ void __launch_bounds__(256) route_kernel(
    const T* __restrict__ x, const T* __restrict__ wr, const float* __restrict__ bias,
    const float* logits_in, const int32_t* __restrict__ po, int P, int64_t Tn,
    int d, int E, int k, int normalize, float* logits, float* probs, int32_t* topk_idx,
    float* topk_w, int32_t* counts) {
    pdl_begin();
    constexpr int NV = (EMAX + 31) / 32;
    extern __shared__ int s_hist_dyn[];  // [P*E] when it fits
    const bool hist_smem = P * E <= HIST_SMEM;
    int* s_hist = hist_smem ? s_hist_dyn : counts;
    if (hist_smem) {
        for (int i = threadIdx.x; i < P * E; i += blockDim.x) s_hist[i] = 0;
    }
    __syncthreads();
    using V = Vec<T>;
    constexpr int VN = V::N;
    const int lane = threadIdx.x & 31;
    const int warps_total = gridDim.x * (blockDim.x >> 5);
    const int64_t nvec = d / VN;
    // groups are enumerated party by party
    int64_t total_groups = 0;
    for (int p = 0; p < P; ++p) {
        int64_t a = po ? po[p] : 0, b = po ? po[p + 1] : Tn;
        total_groups += (b - a + TPW - 1) / TPW;
    }
    for (int64_t gi = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); gi < total_groups;
         gi += warps_total) {
        int party = 0;
        int64_t g = gi, t0 = 0, tend = Tn;
        for (int p = 0; p < P; ++p) {
            int64_t a = po ? po[p] : 0, b = po ? po[p + 1] : Tn;
            int64_t ng = (b - a + TPW - 1) / TPW;
            if (g < ng) { party = p; t0 = a + g * TPW; tend = b; break; }
            g -= ng;
        }
        const int n = (int)min64(TPW, tend - t0);
        float z[TPW][NV];
        if constexpr (FROM_LOGITS) {
#pragma unroll
            for (int i = 0; i < TPW; ++i)
#pragma unroll
                for (int v = 0; v < NV; ++v) {
                    const int e = lane + 32 * v;
                    z[i][v] = (i < n && e < E) ? logits_in[(t0 + i) * E + e] : 0.f;
                    if (bias && e < E) z[i][v] += bias[party * E + e];
                }
        } else {
            float acc[TPW][EMAX];
#pragma unroll
            for (int i = 0; i < TPW; ++i)
#pragma unroll
                for (int e = 0; e < EMAX; ++e) acc[i][e] = 0.f;
            const T* W = wr + (int64_t)party * E * d;
            for (int64_t v = lane; v < nvec; v += 32) {
                float xv[TPW][VN];
#pragma unroll
                for (int i = 0; i < TPW; ++i) {
                    if (i < n) V::load(x + (t0 + i) * d + v * VN, xv[i]);
                    else {
#pragma unroll
                        for (int q = 0; q < VN; ++q) xv[i][q] = 0.f;
                    }
                }
#pragma unroll
                for (int e = 0; e < EMAX; ++e) {
                    if (e < E) {
                        float wv[VN];
                        V::load(W + (int64_t)e * d + v * VN, wv);
#pragma unroll
                        for (int i = 0; i < TPW; ++i)
#pragma unroll
                            for (int q = 0; q < VN; ++q) acc[i][e] = fmaf(xv[i][q], wv[q], acc[i][e]);
                    }
                }
            }
#pragma unroll
            for (int i = 0; i < TPW; ++i) {
#pragma unroll
                for (int v = 0; v < NV; ++v) z[i][v] = 0.f;
#pragma unroll
                for (int e = 0; e < EMAX; ++e) {
                    float s = warp_sum(acc[i][e]);
#pragma unroll
                    for (int v = 0; v < NV; ++v)
                        if (e == lane + 32 * v) z[i][v] = s;
                }
                if (bias) {
#pragma unroll
                    for (int v = 0; v < NV; ++v)
                        if (lane + 32 * v < E) z[i][v] += bias[party * E + lane + 32 * v];
                }
            }
        }
#pragma unroll
        for (int i = 0; i < TPW; ++i)
            if (i < n)
                softmax_topk_token<NV>(z[i], lane, E, k, normalize, t0 + i, party,
                                       (FROM_LOGITS && !bias) ? nullptr : logits, probs, topk_idx,
                                       topk_w, s_hist);
    }
    __syncthreads();
    if (hist_smem) {
        for (int i = threadIdx.x; i < P * E; i += blockDim.x)
            if (s_hist[i]) atomicAdd(&counts[i], s_hist[i]);
    }
}

// ----------------------------------------------------------------------------- aux loss
// One 8-CTA thread-block cluster per party: each CTA sums probs[t, e] over its slice
// of the party's tokens, then CTA 0 of the cluster adds the 8 partial rows from
// distributed shared memory in rank order. Inside a CTA, thread (s, e) of S = 2^j
// stripes per expert loads AUX_U values of its stripe at once (independent loads in
// flight) and adds them in order; the stripes are then added by a fixed binary tree.
// Deterministic, no workspace, no floating-point atomics.
constexpr int AUX_CLUSTER = 8;
constexpr int AUX_THREADS = 1024;
constexpr int AUX_U = 8;

__device__ __forceinline__ int pow2_floor(int v) {
    int r = 1;
    while (2 * r <= v) r *= 2;
    return r;
}

__global__ void __cluster_dims__(AUX_CLUSTER, 1, 1) __launch_bounds__(AUX_THREADS)
    aux_loss_kernel(const float* __restrict__ probs, const int32_t* __restrict__ counts,
                    const int32_t* __restrict__ po, int64_t Tn, int E, int k, float alpha,
                    float* loss, float* coef) {
    pdl_begin();
    __shared__ float s_part[AUX_THREADS];
    __shared__ float s_col[256];
    cg::cluster_group cluster = cg::this_cluster();
    const int rank = (int)cluster.block_rank();
    const int p = blockIdx.x / AUX_CLUSTER;
    const int64_t a = po ? po[p] : 0, b = po ? po[p + 1] : Tn;
    const int64_t n = b - a;
    const int64_t per = (n + AUX_CLUSTER - 1) / AUX_CLUSTER;
    const int64_t lo = a + min64(n, per * rank), hi = a + min64(n, per * (rank + 1));
    const int tid = threadIdx.x;
    const int stripes = pow2_floor(AUX_THREADS / E);
    float acc = 0.f;
    if (tid < stripes * E) {
        const int e = tid % E, st = tid / E;
        for (int64_t t = lo + st; t < hi; t += (int64_t)AUX_U * stripes) {
            float v[AUX_U];
#pragma unroll
            for (int u = 0; u < AUX_U; ++u) {
                const int64_t tt = t + (int64_t)u * stripes;
                v[u] = tt < hi ? probs[tt * E + e] : 0.f;
            }
#pragma unroll
            for (int u = 0; u < AUX_U; ++u) acc += v[u];
        }
    }
    s_part[tid] = acc;
    __syncthreads();
    for (int h = stripes / 2; h > 0; h >>= 1) {
        if (tid < h * E) s_part[tid] += s_part[tid + h * E];
        __syncthreads();
    }
    if (tid < E) s_col[tid] = s_part[tid];
    cluster.sync();
    if (rank == 0 && tid < E) {
        float tot = 0.f;
        for (int r = 0; r < AUX_CLUSTER; ++r) tot += cluster.map_shared_rank(s_col, r)[tid];
        const float Tp = (float)n;
        const float f = (n > 0) ? (float)counts[p * E + tid] / (Tp * k) : 0.f;
        const float Pm = (n > 0) ? tot / Tp : 0.f;
        s_part[tid] = f * Pm;
        coef[p * E + tid] = (n > 0) ? alpha * E * f / Tp : 0.f;
    }
    cluster.sync();
    if (rank == 0 && tid == 0) {
        float L = 0.f;
        for (int e = 0; e < E; ++e) L += s_part[e];
        loss[p] = alpha * E * L;
    }
}

// ----------------------------------------------------------------------------- router bwd
// Token chunks never straddle a party: chunk ci of the enumeration party by party.
__device__ __forceinline__ bool chunk_of(int64_t ci, const int32_t* po, int P, int64_t Tn,
                                         int CH, int* party, int64_t* t0, int* n) {
    for (int p = 0; p < P; ++p) {
        int64_t a = po ? po[p] : 0, b = po ? po[p + 1] : Tn;
        int64_t nc = (b - a + CH - 1) / CH;
        if (ci < nc) {
            *party = p;
            *t0 = a + ci * CH;
            *n = (int)min64(CH, b - *t0);
            return true;
        }
        ci -= nc;
    }
    return false;
}

// dlogits, one warp per token (Alg. 7 backward with the picks held fixed); lane l
// holds experts l + 32 i, i < NV. For the tensor-core router gradients it also writes
// dz16 [T, EP], dlogits rounded to bf16 with zero columns past E (EP = E rounded up to
// 64, 128 or 256), and (block 0) the token chunks of the chunked dW_r contraction:
// chunk_off[c] = first token of chunk c, the chunks of CH tokens of each party in
// order, then empty chunks up to nchunk.
template <int NV>
__global__ void __launch_bounds__(256) dlogits_kernel(
    const float* __restrict__ probs, const int32_t* __restrict__ topk_idx,
    const float* __restrict__ topk_w, const float* __restrict__ dtopk_w,
    const float* __restrict__ aux_coef, const int32_t* __restrict__ po, int P, int64_t Tn, int E,
    int k, int normalize, float* dlogits, __nv_bfloat16* dz16, int EP, int32_t* chunk_off, int CH,
    int nchunk) {
    pdl_begin();
    const int lane = threadIdx.x & 31;
    const int64_t t = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    if (chunk_off && blockIdx.x == 0 && threadIdx.x == 0) {
        int c = 0;
        for (int q = 0; q < P; ++q) {
            const int64_t a = po ? po[q] : 0, b = po ? po[q + 1] : Tn;
            for (int64_t r = a; r < b && c < nchunk; r += CH) chunk_off[c++] = (int32_t)r;
        }
        for (; c <= nchunk; ++c) chunk_off[c] = (int32_t)Tn;
    }
    if (t >= Tn) return;
    const int party = party_of(po, P, t);
    float p[NV], dp[NV];
#pragma unroll
    for (int i = 0; i < NV; ++i) {
        const int e = lane + 32 * i;
        p[i] = e < E ? probs[t * E + e] : 0.f;
        dp[i] = (aux_coef && e < E) ? aux_coef[party * E + e] : 0.f;
    }
    // lane j < k holds pick j
    const int ej = lane < k ? topk_idx[t * k + lane] : -1;
    const float gj0 = lane < k ? dtopk_w[t * k + lane] : 0.f;
    const float wj = lane < k ? topk_w[t * k + lane] : 0.f;
    float gj = gj0;
    if (normalize) {
        const float inner = warp_sum(gj0 * wj);
        const float S = warp_sum((ej >= 0 && ej < E) ? probs[t * E + ej] : 0.f);
        gj = (gj0 - inner) / S;
    }
    for (int j = 0; j < k; ++j) {
        const int e = __shfl_sync(0xffffffffu, ej, j);
        const float g = __shfl_sync(0xffffffffu, gj, j);
#pragma unroll
        for (int i = 0; i < NV; ++i)
            if (e == lane + 32 * i) dp[i] += g;
    }
    float loc = 0.f;
#pragma unroll
    for (int i = 0; i < NV; ++i) loc += dp[i] * p[i];
    const float dot = warp_sum(loc);
#pragma unroll
    for (int i = 0; i < NV; ++i) {
        const int e = lane + 32 * i;
        const float zz = p[i] * (dp[i] - dot);
        if (e < E) dlogits[t * E + e] = zz;
        if (dz16 && e < EP) dz16[t * EP + e] = __float2bfloat16_rn(e < E ? zz : 0.f);
    }
}

// dbias partial of one token chunk: part_db[c][e] = sum of dlogits[t][e] over the chunk.
// Thread (g, e) of a block, g < G = 2^j <= 1024 / E token groups, loads CDB_U tokens
// g, g + G, ... at once and adds them in order; the groups are then added by a fixed
// binary tree (deterministic).
constexpr int CDB_THREADS = 1024;
constexpr int CDB_U = 8;
__global__ void __launch_bounds__(CDB_THREADS) chunk_db_kernel(const float* __restrict__ dz,
                                                              const int32_t* __restrict__ chunk_off, int E,
                                                              float* part_db) {
    pdl_begin();
    __shared__ float s_part[CDB_THREADS];
    const int c = blockIdx.x, G = pow2_floor(CDB_THREADS / E);
    const int e = threadIdx.x % E, g = threadIdx.x / E;
    const int64_t a = chunk_off[c], b = chunk_off[c + 1];
    float acc = 0.f;
    if (g < G) {
        for (int64_t t = a + g; t < b; t += (int64_t)CDB_U * G) {
            float v[CDB_U];
#pragma unroll
            for (int u = 0; u < CDB_U; ++u) {
                const int64_t tt = t + (int64_t)u * G;
                v[u] = tt < b ? dz[tt * E + e] : 0.f;
            }
#pragma unroll
            for (int u = 0; u < CDB_U; ++u) acc += v[u];
        }
    }
    s_part[threadIdx.x] = (g < G) ? acc : 0.f;
    __syncthreads();
    for (int h = G / 2; h > 0; h >>= 1) {
        if (threadIdx.x < h * E) s_part[threadIdx.x] += s_part[threadIdx.x + h * E];
        __syncthreads();
    }
    if (threadIdx.x < E) part_db[(int64_t)c * E + threadIdx.x] = s_part[threadIdx.x];
}

// Partial dW_r = dlogits^T x and db over one chunk of RB_CH tokens of one party, for
// a tile of RB_ET experts and a column slab. The two thread halves take alternate
// tokens of the chunk and are added in a fixed order at the end.
constexpr int RB_CH = 32;   // tokens per chunk
constexpr int RB_ET = 8;    // experts per tile
constexpr int RB_HALF = 128;  // threads per half

template <typename T>
__global__ void __launch_bounds__(2 * RB_HALF) route_bwd_partial_kernel(
    const T* __restrict__ x, const float* __restrict__ dz, const int32_t* __restrict__ po, int P,
    int64_t Tn, int d, int E, float* part_dw, float* part_db) {
    pdl_begin();
    constexpr int VN = Vec<T>::N;
    constexpr int SLAB = RB_HALF * VN;
    __shared__ float s_dz[RB_CH][RB_ET];
    extern __shared__ float s_acc[];  // [RB_HALF][RB_ET][VN]: the second half's sums
    int party, n;
    int64_t t0;
    if (!chunk_of(blockIdx.x, po, P, Tn, RB_CH, &party, &t0, &n)) return;
    const int e0 = blockIdx.y * RB_ET;
    const int ne = min(RB_ET, E - e0);
    for (int i = threadIdx.x; i < RB_CH * RB_ET; i += blockDim.x) {
        const int tt = i / RB_ET, e = i % RB_ET;
        s_dz[tt][e] = (tt < n && e < ne) ? dz[(t0 + tt) * E + e0 + e] : 0.f;
    }
    __syncthreads();
    const int half = threadIdx.x / RB_HALF, ht = threadIdx.x % RB_HALF;
    if (blockIdx.z == 0 && threadIdx.x < ne) {
        float sdb = 0.f;
        for (int i = 0; i < n; ++i) sdb += s_dz[i][threadIdx.x];
        part_db[(int64_t)blockIdx.x * E + e0 + threadIdx.x] = sdb;
    }
    const int64_t c = (int64_t)blockIdx.z * SLAB + ht * VN;
    const bool active = c < d;
    float acc[RB_ET][VN];
#pragma unroll
    for (int e = 0; e < RB_ET; ++e)
#pragma unroll
        for (int q = 0; q < VN; ++q) acc[e][q] = 0.f;
    if (active) {
        // four tokens' x vectors are loaded before any of them is used
        for (int i0 = half; i0 < n; i0 += 8) {
            uint4 raw[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int i = i0 + 2 * u;
                if (i < n) raw[u] = Vec<T>::raw_load(x + (t0 + i) * d + c);
            }
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int i = i0 + 2 * u;
                if (i >= n) break;
                float xv[VN];
                unpack_vec<T>(raw[u], xv);
#pragma unroll
                for (int e = 0; e < RB_ET; ++e) {
                    const float zz = s_dz[i][e];
#pragma unroll
                    for (int q = 0; q < VN; ++q) acc[e][q] = fmaf(zz, xv[q], acc[e][q]);
                }
            }
        }
    }
    if (half == 1) {
#pragma unroll
        for (int e = 0; e < RB_ET; ++e)
#pragma unroll
            for (int q = 0; q < VN; ++q) s_acc[(ht * RB_ET + e) * VN + q] = acc[e][q];
    }
    __syncthreads();
    if (half == 0 && active) {
#pragma unroll
        for (int e = 0; e < RB_ET; ++e) {
            if (e < ne) {
                float* dst = part_dw + ((int64_t)blockIdx.x * E + e0 + e) * d + c;
                float r[VN];
#pragma unroll
                for (int q = 0; q < VN; ++q) r[q] = acc[e][q] + s_acc[(ht * RB_ET + e) * VN + q];
                Vec<float>::store(dst, r);
                if (VN == 8) Vec<float>::store(dst + 4, r + 4);
            }
        }
    }
}

// Sum the partials of each party's chunks: a block takes 32 outputs; thread group g
// (of 8) adds chunks g, g+8, ... in order, then group 0 adds the 8 group sums in order.
constexpr int RR_OUT = 32, RR_GRP = 8;

template <typename T>
__global__ void __launch_bounds__(RR_OUT * RR_GRP) route_bwd_reduce_kernel(
    const float* __restrict__ part_dw, const float* __restrict__ part_db,
    const int32_t* __restrict__ po, int P, int64_t Tn, int d, int E, int CH, T* dw_router,
    float* dbias) {
    pdl_begin();
    __shared__ float s_sum[RR_GRP][RR_OUT];
    const int o = threadIdx.x % RR_OUT, g = threadIdx.x / RR_OUT;
    const int64_t i = (int64_t)blockIdx.x * RR_OUT + o;
    const int64_t per_party = (int64_t)E * d;
    auto crange = [&](int p, int64_t* first, int64_t* cnt) {
        int64_t base = 0;
        for (int q = 0; q < P; ++q) {
            int64_t a = po ? po[q] : 0, b = po ? po[q + 1] : Tn;
            int64_t nc = (b - a + CH - 1) / CH;
            if (q == p) { *first = base; *cnt = nc; return; }
            base += nc;
        }
    };
    float acc = 0.f;
    const bool ok = i < (int64_t)P * per_party;
    if (ok) {
        const int p = (int)(i / per_party);
        const int64_t rem = i % per_party;
        int64_t first, cnt;
        crange(p, &first, &cnt);
        for (int64_t c = g; c < cnt; c += RR_GRP) acc += part_dw[(first + c) * per_party + rem];
    }
    s_sum[g][o] = acc;
    __syncthreads();
    if (g == 0 && ok) {
        float tot = 0.f;
#pragma unroll
        for (int q = 0; q < RR_GRP; ++q) tot += s_sum[q][o];
        Elem<T>::store(dw_router + i, tot);
    }
    if (dbias && g == 0 && i < (int64_t)P * E) {
        const int p = (int)(i / E), e = (int)(i % E);
        int64_t first, cnt;
        crange(p, &first, &cnt);
        float sum = 0.f;
        for (int64_t c = 0; c < cnt; ++c) sum += part_db[(first + c) * E + e];
        dbias[i] = sum;
    }
}

// ----------------------------------------------------------------------------- launchers
static int num_sms() {
    static int n = 0;
    if (!n) {
        int dev = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
        if (n <= 0) n = 148;
    }
    return n;
}

template <typename T, bool FROM>
static cudaError_t launch_route_t(const RouteArgs& a, cudaStream_t s) {
    const int E = a.E;
    const size_t smem = a.P * E <= HIST_SMEM ? (size_t)a.P * E * sizeof(int) : 0;
    const int64_t groups_ub = a.T + a.P;  // upper bound with TPW = 1
    int blocks = (int)min64((groups_ub + 7) / 8, (int64_t)num_sms() * 8);
    if (blocks < 1) blocks = 1;
    const T* x = (const T*)a.x;
    const T* wr = (const T*)a.w_router;
#define MOE_ROUTE_CASE(EM, TP)                                                                   \
    (void)launch_pdl(route_kernel<T, EM, TP, FROM>, dim3(blocks), dim3(256), smem, s,                                       \
        x, wr, a.bias, a.logits_in, a.po, a.P, a.T, a.d, E, a.k, a.normalize, a.logits, a.probs, \
        a.topk_idx, a.topk_w, a.counts)
    if constexpr (FROM) {
        if (E <= 64) MOE_ROUTE_CASE(64, 4);
        else if (E <= 128) MOE_ROUTE_CASE(128, 2);
        else MOE_ROUTE_CASE(256, 1);
    } else if (E <= 8) {
        MOE_ROUTE_CASE(8, 8);
    } else if (E <= 16) {
        MOE_ROUTE_CASE(16, 4);
    } else if (E <= 32) {
        MOE_ROUTE_CASE(32, 2);
    } else {
        MOE_ROUTE_CASE(64, 1);
    }
#undef MOE_ROUTE_CASE
    return cudaGetLastError();
}

// E > 64 on the CUDA cores (fp32): the router's products x W_r[p]^T by the grouped SIMT
// GEMM into `logits` (groups = parties), then the gating pass reads them back, adds the
// bias and overwrites them with the biased logits.
static cudaError_t launch_route_wide_simt(const RouteArgs& a, cudaStream_t s) {
    GemmMArgs m{};
    m.G = (a.po && a.P > 1) ? a.P : 1;
    m.rows = (a.po && a.P > 1) ? GroupRows{a.po, (int)a.T, 0, 0, 0} : GroupRows{nullptr, (int)a.T, 0, 0, 0};
    m.a = a.x;
    m.b = a.w_router;
    m.b_group_elems = (int64_t)a.E * a.d;
    m.b_kmajor = true;
    m.N = a.E;
    m.K = a.d;
    m.epi = EPI_STORE;
    m.out0 = a.logits;
    cudaError_t e = launch_gemm_m_simt(m, s);
    if (e != cudaSuccess) return e;
    RouteArgs b = a;
    b.logits_in = a.logits;
    return launch_route_t<float, true>(b, s);
}

cudaError_t launch_route(const RouteArgs& a, bool bf16, bool from_logits, cudaStream_t s) {
    cudaError_t e = cudaMemsetAsync(a.counts, 0, sizeof(int32_t) * a.P * a.E, s);
    if (e != cudaSuccess) return e;
    if (from_logits) {
        RouteArgs b = a;
        b.bias = nullptr;  // the caller's logits are final
        return launch_route_t<float, true>(b, s);
    }
    if (bf16 && (a.E % 4 == 0 || a.E > 64) && a.T > 0) return launch_route_tc(a, s);
    if (a.E > 64) return a.T > 0 ? launch_route_wide_simt(a, s) : cudaSuccess;
    return bf16 ? launch_route_t<__nv_bfloat16, false>(a, s) : launch_route_t<float, false>(a, s);
}

cudaError_t launch_aux_loss(const float* probs, const int32_t* counts, const int32_t* po, int P,
                            int64_t T, int E, int k, float alpha, float* loss, float* coef,
                            cudaStream_t s) {
    (void)launch_pdl(aux_loss_kernel, dim3(P * AUX_CLUSTER), dim3(AUX_THREADS), 0, s, probs, counts, po, T, E, k, alpha, loss, coef);
    return cudaGetLastError();
}

// Workspace of the router backward. CUDA-core path (fp32): per-chunk partials of
// RB_CH tokens. Tensor-core path (bf16): per-chunk fp32 partials of dW_r and dbias, the
// chunk table and dz16 [T, 64] (dlogits in bf16, the A operand of dx_router = dz W_r and
// the B operand of dW_r^T = x^T dz).
static size_t align256(size_t n) { return (n + 255) / 256 * 256; }
struct RbTcLayout {
    int64_t C, nchunk;
    int EP;  // columns of dz16: E rounded up to 64, 128 or 256
    size_t dw, db, off, dz, total;
};
// Tokens per chunk of the chunked dW_r contraction: about 256 tiles of 128 model columns
// in all (one wave of 152 single-CTA tiles measured slower), at most 128 - P chunks
// (well inside the grouped GEMM's 256 groups), a multiple of 64.
static RbTcLayout rb_tc_layout(int64_t T, int P, int E, int d) {
    RbTcLayout L;
    const int64_t mt = std::max(1, d / 128);
    int64_t C = (T * mt + 255) / 256;
    C = std::max<int64_t>(C, (T + (128 - P) - 1) / (128 - P));
    C = std::max<int64_t>(C, 64);
    L.C = (C + 63) / 64 * 64;
    L.nchunk = (T + L.C - 1) / L.C + P;
    L.dw = 0;
    L.db = align256((size_t)L.nchunk * E * d * sizeof(float));
    L.off = align256(L.db + (size_t)L.nchunk * E * sizeof(float));
    L.EP = E <= 64 ? 64 : E <= 128 ? 128 : 256;
    L.dz = align256(L.off + (size_t)(L.nchunk + 1) * sizeof(int32_t));
    L.total = L.dz + (size_t)T * L.EP * 2 + 256;
    return L;
}

size_t route_bwd_workspace(int64_t T, int P, int E, int d) {
    const int64_t nch = (T + RB_CH - 1) / RB_CH + P;
    const size_t simt = (size_t)nch * E * d * sizeof(float) + (size_t)nch * E * sizeof(float) + 256;
    return std::max(simt, rb_tc_layout(T, P, E, d).total);
}

static cudaError_t launch_dlogits(const RouteBwdArgs& a, __nv_bfloat16* dz16, int EP, int32_t* chunk_off,
                                  int CH, int nchunk, cudaStream_t s) {
    const unsigned blocks = (unsigned)((a.T + 7) / 8);
#define MOE_DL(NV)                                                                                 \
    (void)launch_pdl(dlogits_kernel<NV>, dim3(blocks), dim3(256), 0, s, a.probs, a.topk_idx, a.topk_w, \
                     a.dtopk_w, a.aux_coef, a.po, a.P, a.T, a.E, a.k, a.normalize, a.dlogits, dz16, EP, \
                     chunk_off, CH, nchunk)
    if (a.E <= 64) MOE_DL(2);
    else if (a.E <= 128) MOE_DL(4);
    else MOE_DL(8);
#undef MOE_DL
    return cudaGetLastError();
}

// fp32: dlogits, CUDA-core partials and reduce, dx_router on the CUDA-core GEMM
static cudaError_t launch_route_bwd_simt(const RouteBwdArgs& a, void* ws, cudaStream_t s) {
    using T = float;
    const int64_t nch = (a.T + RB_CH - 1) / RB_CH + a.P;
    float* part_dw = (float*)ws;
    float* part_db = part_dw + nch * a.E * a.d;
    if (a.T > 0) {
        cudaError_t e = launch_dlogits(a, (__nv_bfloat16*)nullptr, 0, (int32_t*)nullptr, 0, 0, s);
        if (e != cudaSuccess) return e;
    }
    constexpr int SLAB = RB_HALF * Vec<T>::N;
    dim3 grid((unsigned)nch, (a.E + RB_ET - 1) / RB_ET, (a.d + SLAB - 1) / SLAB);
    const size_t smem = (size_t)RB_HALF * RB_ET * Vec<T>::N * sizeof(float);
    static bool attr = false;
    if (!attr) {
        cudaError_t e = cudaFuncSetAttribute(route_bwd_partial_kernel<T>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        attr = true;
    }
    (void)launch_pdl(route_bwd_partial_kernel<T>, dim3(grid), dim3(2 * RB_HALF), smem, s, (const T*)a.x,
                     a.dlogits, a.po, a.P, a.T, a.d, a.E, part_dw, part_db);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    const int64_t total = (int64_t)a.P * a.E * a.d;
    (void)launch_pdl(route_bwd_reduce_kernel<T>, dim3((unsigned)((total + RR_OUT - 1) / RR_OUT)),
                     dim3(RR_OUT * RR_GRP), 0, s, part_dw, part_db, a.po, a.P, a.T, a.d, a.E, RB_CH,
                     (T*)a.dw_router, a.dbias);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    if (a.dx_router && a.T > 0) {  // dx_router[t] = dlogits[t] W_r[p(t)], K = E
        GemmMArgs m{};
        m.G = a.po ? a.P : 1;
        m.rows = GroupRows{a.po, (int)a.T, 0, 0, 0};
        m.a = a.dlogits;
        m.b = a.w_router;
        m.b_group_elems = (int64_t)a.E * a.d;
        m.b_kmajor = false;
        m.N = a.d;
        m.K = a.E;
        m.epi = EPI_STORE;
        m.out0 = a.dx_router;
        return launch_gemm_m_simt(m, s);
    }
    return cudaSuccess;
}

// bf16: both products on the tensor cores.
//   dW_r[p]^T = sum over the chunks c of party p of x_c^T dz_c (K-variable grouped GEMM,
//               one group per chunk, fp32 partials), reduced over chunks in order;
//   dx_router = dz W_r[p(t)] (M-variable grouped GEMM over parties, K = 64 padded).
// dz is rounded to bf16 for both (the operands of every bf16 contraction are bf16).
static cudaError_t launch_route_bwd_tc(const RouteBwdArgs& a, void* ws, cudaStream_t s) {
    const RbTcLayout Lw = rb_tc_layout(a.T, a.P, a.E, a.d);
    uint8_t* base = (uint8_t*)ws;
    float* part_dw = (float*)(base + Lw.dw);
    float* part_db = (float*)(base + Lw.db);
    int32_t* chunk_off = (int32_t*)(base + Lw.off);
    __nv_bfloat16* dz16 = (__nv_bfloat16*)(base + Lw.dz);
    cudaError_t e;
    if (a.T > 0) {
        if ((e = launch_dlogits(a, dz16, Lw.EP, chunk_off, (int)Lw.C, (int)Lw.nchunk, s)) != cudaSuccess)
            return e;
        (void)launch_pdl(chunk_db_kernel, dim3((unsigned)Lw.nchunk), dim3(CDB_THREADS), 0, s,
                         (const float*)a.dlogits, (const int32_t*)chunk_off, a.E, part_db);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
        GemmKArgs g{};
        g.G = (int)Lw.nchunk;
        g.rows = GroupRows{chunk_off, (int)a.T, 0, 0, 0};
        g.a = a.x;
        g.b = dz16;
        g.M = a.d;
        g.N = Lw.EP;
        g.out = part_dw;
        g.epi = EPI_DWR;
        g.E = a.E;
        if ((e = launch_gemm_k(g, true, s)) != cudaSuccess) return e;
    }
    const int64_t total = (int64_t)a.P * a.E * a.d;
    (void)launch_pdl(route_bwd_reduce_kernel<__nv_bfloat16>, dim3((unsigned)((total + RR_OUT - 1) / RR_OUT)),
                     dim3(RR_OUT * RR_GRP), 0, s, (const float*)part_dw, (const float*)part_db, a.po, a.P,
                     a.T, a.d, a.E, (int)Lw.C, (__nv_bfloat16*)a.dw_router, a.dbias);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    if (a.dx_router && a.T > 0) {
        GemmMArgs m{};
        m.G = a.po ? a.P : 1;
        m.rows = GroupRows{a.po, (int)a.T, 0, 0, 0};
        m.a = dz16;
        m.b = a.w_router;
        m.b_group_elems = (int64_t)a.E * a.d;
        m.b_kmajor = false;
        m.N = a.d;
        m.K = Lw.EP;
        m.b_rows = a.E;
        m.epi = EPI_STORE;
        m.out0 = a.dx_router;
        m.slim = true;  // one k-block per tile: the stores bound it
        return launch_gemm_m(m, true, s);
    }
    return cudaSuccess;
}

cudaError_t launch_route_bwd(const RouteBwdArgs& a, bool bf16, void* ws, cudaStream_t s) {
    return bf16 ? launch_route_bwd_tc(a, ws, s) : launch_route_bwd_simt(a, ws, s);
}

cudaError_t route_status(cudaStream_t s, int* code) { return tu_status_read_clear(s, code); }

}  // namespace moe
