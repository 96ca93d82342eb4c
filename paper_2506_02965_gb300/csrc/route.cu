// Gating function of the MoE layer (Alg. 7) and its backward, plus the per-party
// load-balancing loss. Memory-bound SIMT kernels: x is read once with 16-byte
// vector loads, logits are reduced with warp shuffles, top-k is a warp argmax.
#include <cfloat>

#include "moe_common.cuh"
#include "moe_internal.h"

namespace moe {

// ----------------------------------------------------------------------------- top-k
// Per token, lane l owns experts l and l + 32 (E <= 64). Picks the k largest logits,
// descending, equal logits by ascending expert id; writes logits (optional), probs,
// topk idx / w and bumps the block histogram.
__device__ __forceinline__ bool better(float va, int ia, float vb, int ib) {
    return va > vb || (va == vb && ia < ib);
}

__device__ void softmax_topk_token(float z0, float z1, int lane, int E, int k, int normalize,
                                   int64_t t, int party, float* logits, float* probs,
                                   int32_t* topk_idx, float* topk_w, int* s_hist) {
    const int e0 = lane, e1 = lane + 32;
    const bool v0 = e0 < E, v1 = e1 < E;
    if (logits) {
        if (v0) logits[t * E + e0] = z0;
        if (v1) logits[t * E + e1] = z1;
    }
    float m = fmaxf(v0 ? z0 : -FLT_MAX, v1 ? z1 : -FLT_MAX);
    m = warp_max(m);
    float x0 = v0 ? expf(z0 - m) : 0.f;
    float x1 = v1 ? expf(z1 - m) : 0.f;
    float s = warp_sum(x0 + x1);
    float p0 = x0 / s, p1 = x1 / s;
    if (v0) probs[t * E + e0] = p0;
    if (v1) probs[t * E + e1] = p1;
    bool taken0 = !v0, taken1 = !v1;
    float wsel = 0.f, wsum = 0.f;
    int isel = 0;
    for (int j = 0; j < k; ++j) {
        // local candidate
        float cv = -FLT_MAX;
        int ci = 0x7fffffff;
        bool have = false;
        if (!taken0) { cv = z0; ci = e0; have = true; }
        if (!taken1 && (!have || better(z1, e1, cv, ci))) { cv = z1; ci = e1; have = true; }
        int hv = have ? 1 : 0;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            float ov = __shfl_xor_sync(0xffffffffu, cv, o);
            int oi = __shfl_xor_sync(0xffffffffu, ci, o);
            int oh = __shfl_xor_sync(0xffffffffu, hv, o);
            if (oh && (!hv || better(ov, oi, cv, ci))) { cv = ov; ci = oi; hv = 1; }
        }
        // ci is the winner on every lane
        const int owner = ci & 31;
        float pw = __shfl_sync(0xffffffffu, (ci < 32) ? p0 : p1, owner);
        if (ci == e0) taken0 = true;
        if (ci == e1) taken1 = true;
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
template <typename T, int EMAX, int TPW, bool FROM_LOGITS>
__global__ void __launch_bounds__(256) route_kernel(
    const T* __restrict__ x, const T* __restrict__ wr, const float* __restrict__ bias,
    const float* __restrict__ logits_in, const int32_t* __restrict__ po, int P, int64_t Tn,
    int d, int E, int k, int normalize, float* logits, float* probs, int32_t* topk_idx,
    float* topk_w, int32_t* counts) {
    extern __shared__ int s_hist[];  // [P*E]
    for (int i = threadIdx.x; i < P * E; i += blockDim.x) s_hist[i] = 0;
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
        float z0[TPW], z1[TPW];
        if constexpr (FROM_LOGITS) {
#pragma unroll
            for (int i = 0; i < TPW; ++i) {
                z0[i] = (i < n && lane < E) ? logits_in[(t0 + i) * E + lane] : 0.f;
                z1[i] = (i < n && lane + 32 < E) ? logits_in[(t0 + i) * E + lane + 32] : 0.f;
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
                z0[i] = 0.f;
                z1[i] = 0.f;
#pragma unroll
                for (int e = 0; e < EMAX; ++e) {
                    float s = warp_sum(acc[i][e]);
                    if (e == lane) z0[i] = s;
                    if (e == lane + 32) z1[i] = s;
                }
                if (bias) {
                    if (lane < E) z0[i] += bias[party * E + lane];
                    if (lane + 32 < E) z1[i] += bias[party * E + lane + 32];
                }
            }
        }
#pragma unroll
        for (int i = 0; i < TPW; ++i)
            if (i < n)
                softmax_topk_token(z0[i], z1[i], lane, E, k, normalize, t0 + i, party,
                                   FROM_LOGITS ? nullptr : logits, probs, topk_idx, topk_w,
                                   s_hist);
    }
    __syncthreads();
    for (int i = threadIdx.x; i < P * E; i += blockDim.x)
        if (s_hist[i]) atomicAdd(&counts[i], s_hist[i]);
}

// ----------------------------------------------------------------------------- aux loss
// One block per party; deterministic fixed-order reductions.
__global__ void __launch_bounds__(256) aux_loss_kernel(const float* __restrict__ probs,
                                                      const int32_t* __restrict__ counts,
                                                      const int32_t* __restrict__ po, int64_t Tn,
                                                      int E, int k, float alpha, float* loss,
                                                      float* coef) {
    __shared__ float s_part[256];
    __shared__ float s_term[64];
    const int p = blockIdx.x;
    const int64_t a = po ? po[p] : 0, b = po ? po[p + 1] : Tn;
    const int lpe = blockDim.x / E;  // stripes per expert
    const int tid = threadIdx.x;
    float s = 0.f;
    if (tid < lpe * E) {
        const int e = tid % E, stripe = tid / E;
        for (int64_t t = a + stripe; t < b; t += lpe) s += probs[t * E + e];
    }
    s_part[tid] = s;
    __syncthreads();
    if (tid < E) {
        float tot = 0.f;
        for (int st = 0; st < lpe; ++st) tot += s_part[st * E + tid];
        const float Tp = (float)(b - a);
        const float f = (Tp > 0) ? (float)counts[p * E + tid] / (Tp * k) : 0.f;
        const float Pm = (Tp > 0) ? tot / Tp : 0.f;
        s_term[tid] = f * Pm;
        coef[p * E + tid] = (Tp > 0) ? alpha * E * f / Tp : 0.f;
    }
    __syncthreads();
    if (tid == 0) {
        float L = 0.f;
        for (int e = 0; e < E; ++e) L += s_term[e];
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

// dlogits of one token (lane l: experts l, l+32), Alg. 7 backward with fixed picks.
__device__ __forceinline__ void dlogits_token(int64_t t, int lane, int E, int k, int normalize,
                                              int party, const float* probs,
                                              const int32_t* topk_idx, const float* topk_w,
                                              const float* dtopk_w, const float* aux_coef,
                                              float* dz0, float* dz1) {
    const int e0 = lane, e1 = lane + 32;
    float p0 = e0 < E ? probs[t * E + e0] : 0.f;
    float p1 = e1 < E ? probs[t * E + e1] : 0.f;
    float dp0 = 0.f, dp1 = 0.f;
    float inner = 0.f, S = 0.f;
    if (normalize) {
        for (int j = 0; j < k; ++j) {
            const int e = topk_idx[t * k + j];
            inner += dtopk_w[t * k + j] * topk_w[t * k + j];
            if (e >= 0 && e < E) S += probs[t * E + e];
        }
    }
    for (int j = 0; j < k; ++j) {
        const int e = topk_idx[t * k + j];
        float g = dtopk_w[t * k + j];
        if (normalize) g = (g - inner) / S;
        if (e == e0) dp0 += g;
        if (e == e1) dp1 += g;
    }
    if (aux_coef) {
        if (e0 < E) dp0 += aux_coef[party * E + e0];
        if (e1 < E) dp1 += aux_coef[party * E + e1];
    }
    const float dot = warp_sum(dp0 * p0 + dp1 * p1);
    *dz0 = p0 * (dp0 - dot);
    *dz1 = p1 * (dp1 - dot);
}

// Stage A: per (token chunk, 8-expert tile, 1024-column slab): dlogits of the chunk
// into shared memory (and to global once), then partial dW_r = dz^T x and partial db.
constexpr int RB_CH = 64;    // tokens per chunk
constexpr int RB_ET = 8;     // experts per tile
constexpr int RB_COLS = 1024;

template <typename T>
__global__ void __launch_bounds__(128) route_bwd_partial_kernel(
    const T* __restrict__ x, const float* __restrict__ probs, const int32_t* __restrict__ topk_idx,
    const float* __restrict__ topk_w, const float* __restrict__ dtopk_w,
    const float* __restrict__ aux_coef, const int32_t* __restrict__ po, int P, int64_t Tn, int d,
    int E, int k, int normalize, float* dlogits, float* part_dw, float* part_db) {
    __shared__ float s_dz[RB_CH][64];
    int party, n;
    int64_t t0;
    if (!chunk_of(blockIdx.x, po, P, Tn, RB_CH, &party, &t0, &n)) return;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const bool writer = (blockIdx.y == 0 && blockIdx.z == 0);
    for (int i = warp; i < RB_CH; i += blockDim.x >> 5) {
        float dz0 = 0.f, dz1 = 0.f;
        if (i < n) {
            dlogits_token(t0 + i, lane, E, k, normalize, party, probs, topk_idx, topk_w, dtopk_w,
                          aux_coef, &dz0, &dz1);
            if (writer) {
                if (lane < E) dlogits[(t0 + i) * E + lane] = dz0;
                if (lane + 32 < E) dlogits[(t0 + i) * E + lane + 32] = dz1;
            }
        }
        s_dz[i][lane] = dz0;
        s_dz[i][lane + 32] = dz1;
    }
    __syncthreads();
    const int e0 = blockIdx.y * RB_ET;
    if (blockIdx.z == 0 && threadIdx.x < RB_ET && e0 + threadIdx.x < E) {
        float s = 0.f;
        for (int i = 0; i < n; ++i) s += s_dz[i][e0 + threadIdx.x];
        part_db[(int64_t)blockIdx.x * E + e0 + threadIdx.x] = s;
    }
    using V = Vec<T>;
    constexpr int VN = V::N;
    const int64_t c0 = (int64_t)blockIdx.z * RB_COLS + threadIdx.x * VN;
    for (int64_t c = c0; c < min64(d, (int64_t)(blockIdx.z + 1) * RB_COLS); c += blockDim.x * VN) {
        float acc[RB_ET][VN];
#pragma unroll
        for (int e = 0; e < RB_ET; ++e)
#pragma unroll
            for (int q = 0; q < VN; ++q) acc[e][q] = 0.f;
        for (int i = 0; i < n; ++i) {
            float xv[VN];
            V::load(x + (t0 + i) * d + c, xv);
#pragma unroll
            for (int e = 0; e < RB_ET; ++e) {
                const float z = s_dz[i][(e0 + e) & 63];
#pragma unroll
                for (int q = 0; q < VN; ++q) acc[e][q] = fmaf(z, xv[q], acc[e][q]);
            }
        }
#pragma unroll
        for (int e = 0; e < RB_ET; ++e) {
            if (e0 + e < E) {
                float* dst = part_dw + ((int64_t)blockIdx.x * E + e0 + e) * d + c;
#pragma unroll
                for (int q = 0; q < VN; ++q) dst[q] = acc[e][q];
            }
        }
    }
}

// Stage B: sum the partials of each party's chunks in chunk order.
template <typename T>
__global__ void __launch_bounds__(256) route_bwd_reduce_kernel(
    const float* __restrict__ part_dw, const float* __restrict__ part_db,
    const int32_t* __restrict__ po, int P, int64_t Tn, int d, int E, T* dw_router, float* dbias) {
    const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t per_party = (int64_t)E * d;
    const int64_t total = (int64_t)P * per_party;
    // chunk range of party p
    auto crange = [&](int p, int64_t* first, int64_t* cnt) {
        int64_t base = 0;
        for (int q = 0; q < P; ++q) {
            int64_t a = po ? po[q] : 0, b = po ? po[q + 1] : Tn;
            int64_t nc = (b - a + RB_CH - 1) / RB_CH;
            if (q == p) { *first = base; *cnt = nc; return; }
            base += nc;
        }
    };
    if (i < total) {
        const int p = (int)(i / per_party);
        const int64_t rem = i % per_party;  // e*d + c
        int64_t first, cnt;
        crange(p, &first, &cnt);
        float s = 0.f;
        for (int64_t c = 0; c < cnt; ++c) s += part_dw[(first + c) * per_party + rem];
        Elem<T>::store(dw_router + i, s);
    }
    if (dbias && i < (int64_t)P * E) {
        const int p = (int)(i / E), e = (int)(i % E);
        int64_t first, cnt;
        crange(p, &first, &cnt);
        float s = 0.f;
        for (int64_t c = 0; c < cnt; ++c) s += part_db[(first + c) * E + e];
        dbias[i] = s;
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
    const size_t smem = (size_t)a.P * E * sizeof(int);
    const int64_t groups_ub = a.T + a.P;  // upper bound with TPW = 1
    int blocks = (int)min64((groups_ub + 7) / 8, (int64_t)num_sms() * 8);
    if (blocks < 1) blocks = 1;
    const T* x = (const T*)a.x;
    const T* wr = (const T*)a.w_router;
#define MOE_ROUTE_CASE(EM, TP)                                                                   \
    route_kernel<T, EM, TP, FROM><<<blocks, 256, smem, s>>>(                                      \
        x, wr, a.bias, a.logits_in, a.po, a.P, a.T, a.d, E, a.k, a.normalize, a.logits, a.probs, \
        a.topk_idx, a.topk_w, a.counts)
    if constexpr (FROM) {
        MOE_ROUTE_CASE(64, 4);
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

cudaError_t launch_route(const RouteArgs& a, bool bf16, bool from_logits, cudaStream_t s) {
    cudaError_t e = cudaMemsetAsync(a.counts, 0, sizeof(int32_t) * a.P * a.E, s);
    if (e != cudaSuccess) return e;
    if (from_logits) return launch_route_t<float, true>(a, s);
    return bf16 ? launch_route_t<__nv_bfloat16, false>(a, s) : launch_route_t<float, false>(a, s);
}

cudaError_t launch_aux_loss(const float* probs, const int32_t* counts, const int32_t* po, int P,
                            int64_t T, int E, int k, float alpha, float* loss, float* coef,
                            cudaStream_t s) {
    aux_loss_kernel<<<P, 256, 0, s>>>(probs, counts, po, T, E, k, alpha, loss, coef);
    return cudaGetLastError();
}

size_t route_bwd_workspace(int64_t T, int P, int E, int d) {
    const int64_t nch = (T + RB_CH - 1) / RB_CH + P;
    return (size_t)nch * E * d * sizeof(float) + (size_t)nch * E * sizeof(float) + 256;
}

template <typename T>
static cudaError_t launch_route_bwd_t(const RouteBwdArgs& a, void* ws, cudaStream_t s) {
    const int64_t nch = (a.T + RB_CH - 1) / RB_CH + a.P;
    float* part_dw = (float*)ws;
    float* part_db = part_dw + nch * a.E * a.d;
    dim3 grid((unsigned)nch, (a.E + RB_ET - 1) / RB_ET, (a.d + RB_COLS - 1) / RB_COLS);
    route_bwd_partial_kernel<T><<<grid, 128, 0, s>>>(
        (const T*)a.x, a.probs, a.topk_idx, a.topk_w, a.dtopk_w, a.aux_coef, a.po, a.P, a.T, a.d,
        a.E, a.k, a.normalize, a.dlogits, part_dw, part_db);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    const int64_t total = (int64_t)a.P * a.E * a.d;
    route_bwd_reduce_kernel<T><<<(unsigned)((total + 255) / 256), 256, 0, s>>>(
        part_dw, part_db, a.po, a.P, a.T, a.d, a.E, (T*)a.dw_router, a.dbias);
    return cudaGetLastError();
}

cudaError_t launch_route_bwd(const RouteBwdArgs& a, bool bf16, void* ws, cudaStream_t s) {
    return bf16 ? launch_route_bwd_t<__nv_bfloat16>(a, ws, s) : launch_route_bwd_t<float>(a, ws, s);
}

cudaError_t route_status(cudaStream_t s, int* code) { return tu_status_read_clear(s, code); }

}  // namespace moe
