// Token dispatch (the "send h to the host of idx" step of Alg. 3 as one expert-major
// buffer), the gate-weighted combine of Alg. 3 and the backward of both (Alg. 5,
// Sec. 3.2). All memory-bound: 16-byte vector loads/stores, one warp per token or
// per permuted row, no floating-point atomics (every result is deterministic).
#include "moe_common.cuh"
#include "moe_internal.h"

namespace moe {

constexpr int DCH = 128;  // tokens per dispatch chunk (one thread each)

// Per chunk: how many of its (token, pick) pairs went to each expert. Also checks
// that every index lies in [0, E) and that no token picks an expert twice.
__global__ void __launch_bounds__(DCH) chunk_count_kernel(const int32_t* __restrict__ idx,
                                                          int64_t T, int E, int k,
                                                          int32_t* chunk_counts) {
    pdl_begin();
    __shared__ int s_cnt[64];
    for (int i = threadIdx.x; i < E; i += blockDim.x) s_cnt[i] = 0;
    __syncthreads();
    const int64_t t = (int64_t)blockIdx.x * DCH + threadIdx.x;
    if (t < T) {
        for (int j = 0; j < k; ++j) {
            const int e = idx[t * k + j];
            bool ok = (e >= 0 && e < E);
            for (int jj = 0; jj < j; ++jj) ok = ok && (idx[t * k + jj] != e);
            if (ok) atomicAdd(&s_cnt[e], 1);
            else record_status(MOE_ERR_DEVICE_CHECK);
        }
    }
    __syncthreads();
    for (int i = threadIdx.x; i < E; i += blockDim.x)
        chunk_counts[(int64_t)blockIdx.x * E + i] = s_cnt[i];
}

// Per chunk: offsets (written by chunk 0), the chunk's base row inside each expert
// segment, and the stable rank of each pick among the chunk's picks of that expert
// (a bit per token and expert, counted with popc).
__global__ void __launch_bounds__(DCH) slot_kernel(const int32_t* __restrict__ idx,
                                                   const int32_t* __restrict__ chunk_counts,
                                                   int64_t T, int E, int k, int nchunks,
                                                   int32_t* offsets, int32_t* slot_of,
                                                   int32_t* token_of) {
    pdl_begin();
    __shared__ int s_pre[64];
    __shared__ int s_tot[64];
    __shared__ int s_base[64];
    __shared__ unsigned s_bits[64][DCH / 32];
    constexpr int TAB = 8192;  // chunk-count table staged in shared memory when it fits
    __shared__ int s_tab[TAB];
    const int c = blockIdx.x;
    const int64_t ntab = (int64_t)nchunks * E;
    if (ntab <= TAB) {
        for (int i = threadIdx.x; i < ntab; i += blockDim.x) s_tab[i] = chunk_counts[i];
        __syncthreads();
    }
    for (int e = threadIdx.x; e < E; e += blockDim.x) {
        int pre = 0, tot = 0;
        for (int cc = 0; cc < nchunks; ++cc) {
            const int v = ntab <= TAB ? s_tab[cc * E + e] : chunk_counts[(int64_t)cc * E + e];
            if (cc < c) pre += v;
            tot += v;
        }
        s_pre[e] = pre;
        s_tot[e] = tot;
    }
    for (int i = threadIdx.x; i < 64 * (DCH / 32); i += blockDim.x) (&s_bits[0][0])[i] = 0u;
    __syncthreads();
    if (threadIdx.x == 0) {
        int run = 0;
        for (int e = 0; e < E; ++e) {
            if (c == 0) offsets[e] = run;
            s_base[e] = run + s_pre[e];
            run += s_tot[e];
        }
        if (c == 0) offsets[E] = run;
    }
    const int i = threadIdx.x;
    const int64_t t = (int64_t)c * DCH + i;
    int es[8];
    int kk = 0;
    if (t < T) {
        for (int j = 0; j < k; ++j) {
            const int e = idx[t * k + j];
            bool ok = (e >= 0 && e < E);
            for (int jj = 0; jj < j; ++jj) ok = ok && (es[jj] != e);
            es[j] = ok ? e : -1;
            if (ok) atomicOr(&s_bits[e][i >> 5], 1u << (i & 31));
            else slot_of[t * k + j] = -1;
        }
        kk = k;
    }
    __syncthreads();
    for (int j = 0; j < kk; ++j) {
        const int e = es[j];
        if (e < 0) continue;
        int rank = 0;
        for (int w = 0; w < (i >> 5); ++w) rank += __popc(s_bits[e][w]);
        rank += __popc(s_bits[e][i >> 5] & ((1u << (i & 31)) - 1u));
        const int slot = s_base[e] + rank;
        slot_of[t * k + j] = slot;
        token_of[slot] = (int32_t)t;
    }
}

// x_perm[r] = x[token_of[r]]: one warp per permuted row, 16-byte vectors.
template <typename T>
__global__ void __launch_bounds__(256) gather_kernel(const T* __restrict__ x,
                                                     const int32_t* __restrict__ token_of,
                                                     int64_t TK, int64_t Tn, int d, T* x_perm) {
    pdl_begin();
    const int lane = threadIdx.x & 31;
    const int64_t r = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    if (r >= TK) return;
    const int64_t t = token_of[r];
    if (t < 0 || t >= Tn) {
        if (lane == 0) record_status(MOE_ERR_DEVICE_CHECK);
        return;
    }
    constexpr int VN = Vec<T>::N;
    const int nv = d / VN;
    const T* src = x + t * d;
    T* dst = x_perm + r * d;
    for (int v = lane; v < nv; v += 32) Vec<T>::raw_store(dst + v * VN, Vec<T>::raw_load(src + v * VN));
}

// out[t] = sum_j w[t,j] * y_perm[slot_of[t,j]] (+ sum_s y_sh[s,t]); fp32 accumulation.
// One warp per token; every lane issues the loads of up to UB vectors of all k rows
// before it uses any of them, so enough bytes are in flight to keep HBM busy.
template <typename T, int KMAX>
__global__ void __launch_bounds__(256, 3) combine_fwd_kernel(const T* __restrict__ y_perm,
                                                          const float* __restrict__ w,
                                                          const int32_t* __restrict__ slot_of,
                                                          const T* __restrict__ y_sh, int S,
                                                          int64_t Tn, int d, int k, T* out) {
    pdl_begin();
    const int lane = threadIdx.x & 31;
    const int64_t t = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    if (t >= Tn) return;
    constexpr int VN = Vec<T>::N;
    constexpr int UB = KMAX <= 2 ? 4 : KMAX <= 4 ? 2 : 1;  // vectors per lane in flight
    int64_t slot[KMAX];
    float wt[KMAX];
#pragma unroll
    for (int j = 0; j < KMAX; ++j) {
        slot[j] = j < k ? slot_of[t * k + j] : 0;
        wt[j] = j < k ? w[t * k + j] : 0.f;
        if (slot[j] < 0 || slot[j] >= Tn * k) {  // bad table: contribute nothing
            if (lane == 0) record_status(MOE_ERR_DEVICE_CHECK);
            slot[j] = 0;
            wt[j] = 0.f;
        }
    }
    const int nv = d / VN;
    for (int v0 = lane; v0 < nv; v0 += 32 * UB) {
        uint4 raw[UB][KMAX];
#pragma unroll
        for (int u = 0; u < UB; ++u) {
            const int v = v0 + 32 * u;
#pragma unroll
            for (int j = 0; j < KMAX; ++j)
                if (j < k && v < nv) raw[u][j] = Vec<T>::raw_load(y_perm + slot[j] * d + v * VN);
        }
#pragma unroll
        for (int u = 0; u < UB; ++u) {
            const int v = v0 + 32 * u;
            if (v >= nv) break;
            float acc[VN];
#pragma unroll
            for (int q = 0; q < VN; ++q) acc[q] = 0.f;
#pragma unroll
            for (int j = 0; j < KMAX; ++j) {
                if (j < k) {
                    float yv[VN];
                    unpack_vec<T>(raw[u][j], yv);
#pragma unroll
                    for (int q = 0; q < VN; ++q) acc[q] = fmaf(wt[j], yv[q], acc[q]);
                }
            }
            for (int s2 = 0; s2 < S; ++s2) {
                float yv[VN];
                Vec<T>::load(y_sh + ((int64_t)s2 * Tn + t) * d + v * VN, yv);
#pragma unroll
                for (int q = 0; q < VN; ++q) acc[q] += yv[q];
            }
            Vec<T>::store(out + t * d + v * VN, acc);
        }
    }
}

// dy_perm[slot(t,j)] = w[t,j] dout[t];  dw[t,j] = <dout[t], y_perm[slot(t,j)]>.
template <typename T, int KMAX>
__global__ void __launch_bounds__(256, 3) combine_bwd_kernel(const T* __restrict__ dout,
                                                          const T* __restrict__ y_perm,
                                                          const float* __restrict__ w,
                                                          const int32_t* __restrict__ slot_of,
                                                          int64_t Tn, int d, int k, T* dy_perm,
                                                          float* dw) {
    pdl_begin();
    const int lane = threadIdx.x & 31;
    const int64_t t = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    if (t >= Tn) return;
    constexpr int VN = Vec<T>::N;
    constexpr int UB = KMAX <= 2 ? 4 : KMAX <= 4 ? 2 : 1;
    int64_t slot[KMAX];
    float wt[KMAX], part[KMAX];
#pragma unroll
    for (int j = 0; j < KMAX; ++j) {
        slot[j] = j < k ? slot_of[t * k + j] : 0;
        wt[j] = j < k ? w[t * k + j] : 0.f;
        part[j] = 0.f;
        if (slot[j] < 0 || slot[j] >= Tn * k) {
            if (lane == 0) record_status(MOE_ERR_DEVICE_CHECK);
            slot[j] = -1;
        }
    }
    const int nv = d / VN;
    for (int v0 = lane; v0 < nv; v0 += 32 * UB) {
        uint4 graw[UB], yraw[UB][KMAX];
#pragma unroll
        for (int u = 0; u < UB; ++u) {
            const int v = v0 + 32 * u;
            if (v < nv) {
                graw[u] = Vec<T>::raw_load(dout + t * d + v * VN);
#pragma unroll
                for (int j = 0; j < KMAX; ++j)
                    if (j < k && slot[j] >= 0) yraw[u][j] = Vec<T>::raw_load(y_perm + slot[j] * d + v * VN);
            }
        }
#pragma unroll
        for (int u = 0; u < UB; ++u) {
            const int v = v0 + 32 * u;
            if (v >= nv) break;
            float g[VN];
            unpack_vec<T>(graw[u], g);
#pragma unroll
            for (int j = 0; j < KMAX; ++j) {
                if (j < k && slot[j] >= 0) {
                    float yv[VN], dy[VN];
                    unpack_vec<T>(yraw[u][j], yv);
#pragma unroll
                    for (int q = 0; q < VN; ++q) {
                        part[j] = fmaf(g[q], yv[q], part[j]);
                        dy[q] = wt[j] * g[q];
                    }
                    Vec<T>::store(dy_perm + slot[j] * d + v * VN, dy);
                }
            }
        }
    }
#pragma unroll
    for (int j = 0; j < KMAX; ++j) {
        if (j < k) {
            const float sum = warp_sum(part[j]);
            if (lane == 0) dw[t * k + j] = sum;
        }
    }
}

// dx[t] = sum_j dx_perm[slot(t,j)] + sum_e dlogits[t,e] W_r[p(t)][e] + sum_s dx_sh[s,t].
// A block takes UR_TOK tokens of one party and a slab of 64 * VN columns; each thread
// owns VN columns of UR_TOK / 4 tokens. The slot lookups and permuted rows of the first
// two picks are requested first; while they are in flight the party's router rows for
// the slab and the tokens' dlogits are staged in shared memory and the router term is
// accumulated.
constexpr int UR_TOK = 16;
constexpr int UR_PRE = 2;  // picks whose rows are loaded before the router term

template <typename T>
__global__ void __launch_bounds__(256) unpermute_reduce_kernel(
    const T* __restrict__ dx_perm, const int32_t* __restrict__ slot_of,
    const float* __restrict__ dz, const T* __restrict__ wr, const int32_t* __restrict__ po, int P,
    const T* __restrict__ dx_sh, int S, int64_t Tn, int d, int E, int k, T* dx) {
    pdl_begin();
    constexpr int VN = Vec<T>::N;
    constexpr int SLAB = 64 * VN;
    constexpr int TPT = UR_TOK / 4;  // tokens per thread
    extern __shared__ __align__(16) unsigned char ur_smem[];
    float* s_dz = reinterpret_cast<float*>(ur_smem);                  // [UR_TOK][E]
    T* s_w = reinterpret_cast<T*>(ur_smem + UR_TOK * 64 * sizeof(float));  // [E][SLAB]
    // tile -> (party, first token)
    int64_t ti = blockIdx.x, t0 = -1, tend = 0;
    int party = 0;
    for (int p = 0; p < P; ++p) {
        const int64_t a = po ? po[p] : 0, b = po ? po[p + 1] : Tn;
        const int64_t nt = (b - a + UR_TOK - 1) / UR_TOK;
        if (ti < nt) { party = p; t0 = a + ti * UR_TOK; tend = b; break; }
        ti -= nt;
    }
    if (t0 < 0) return;
    const int n = (int)min64(UR_TOK, tend - t0);
    const int64_t c0 = (int64_t)blockIdx.y * SLAB;
    const int ncols = (int)min64(SLAB, d - c0);
    const int cv = threadIdx.x & 63;  // column vector inside the slab
    const int tg = threadIdx.x >> 6;  // token group
    const bool active = cv * VN < ncols;
    const int64_t col = c0 + cv * VN;
    // slot of pick j of this thread's tokens (-1: no token, or a bad slot, recorded)
    auto slots_of = [&](int j, int32_t* slot) {
#pragma unroll
        for (int i = 0; i < TPT; ++i) {
            const int tt = tg * TPT + i;
            slot[i] = (active && tt < n) ? slot_of[(t0 + tt) * k + j] : -1;
            if (active && tt < n && (slot[i] < 0 || (int64_t)slot[i] >= Tn * k)) {
                if (cv == 0) record_status(MOE_ERR_DEVICE_CHECK);
                slot[i] = -1;
            }
        }
    };
    int32_t pslot[UR_PRE][TPT];
    uint4 praw[UR_PRE][TPT];
#pragma unroll
    for (int j = 0; j < UR_PRE; ++j) {
        if (j < k) {
            slots_of(j, pslot[j]);
        } else {
#pragma unroll
            for (int i = 0; i < TPT; ++i) pslot[j][i] = -1;
        }
    }
#pragma unroll
    for (int j = 0; j < UR_PRE; ++j)
#pragma unroll
        for (int i = 0; i < TPT; ++i)
            if (pslot[j][i] >= 0) praw[j][i] = Vec<T>::raw_load(dx_perm + (int64_t)pslot[j][i] * d + col);
    // router term: stage dlogits and the party's router rows for this slab
    const T* W = wr + (int64_t)party * E * d;
    for (int i = threadIdx.x; i < UR_TOK * E; i += blockDim.x) {
        const int tt = i / E, e = i % E;
        s_dz[i] = tt < n ? dz[(t0 + tt) * E + e] : 0.f;
    }
    for (int i = threadIdx.x; i < E * (SLAB / VN); i += blockDim.x) {
        const int e = i / (SLAB / VN), v = i % (SLAB / VN);
        if (v * VN < ncols) Vec<T>::raw_store(s_w + e * SLAB + v * VN, Vec<T>::raw_load(W + (int64_t)e * d + c0 + v * VN));
    }
    __syncthreads();
    if (!active) return;
    float acc[TPT][VN];
#pragma unroll
    for (int i = 0; i < TPT; ++i)
#pragma unroll
        for (int q = 0; q < VN; ++q) acc[i][q] = 0.f;
    for (int e = 0; e < E; ++e) {
        float wv[VN];
        Vec<T>::load(s_w + e * SLAB + cv * VN, wv);
#pragma unroll
        for (int i = 0; i < TPT; ++i) {
            const float zz = s_dz[(tg * TPT + i) * E + e];
#pragma unroll
            for (int q = 0; q < VN; ++q) acc[i][q] = fmaf(zz, wv[q], acc[i][q]);
        }
    }
    auto add_rows = [&](const int32_t* slot, const uint4* raw) {
#pragma unroll
        for (int i = 0; i < TPT; ++i) {
            if (slot[i] >= 0) {
                float g[VN];
                unpack_vec<T>(raw[i], g);
#pragma unroll
                for (int q = 0; q < VN; ++q) acc[i][q] += g[q];
            }
        }
    };
#pragma unroll
    for (int j = 0; j < UR_PRE; ++j) add_rows(pslot[j], praw[j]);
    // remaining picks, one at a time: the slot lookups, then the rows, in flight together
    for (int j = UR_PRE; j < k; ++j) {
        int32_t slot[TPT];
        slots_of(j, slot);
        uint4 raw[TPT];
#pragma unroll
        for (int i = 0; i < TPT; ++i)
            if (slot[i] >= 0) raw[i] = Vec<T>::raw_load(dx_perm + (int64_t)slot[i] * d + col);
        add_rows(slot, raw);
    }
#pragma unroll
    for (int i = 0; i < TPT; ++i) {
        const int tt = tg * TPT + i;
        if (tt >= n) break;
        const int64_t t = t0 + tt;
        for (int s2 = 0; s2 < S; ++s2) {
            float g[VN];
            Vec<T>::load(dx_sh + ((int64_t)s2 * Tn + t) * d + col, g);
#pragma unroll
            for (int q = 0; q < VN; ++q) acc[i][q] += g[q];
        }
        Vec<T>::store(dx + t * d + col, acc[i]);
    }
}

// ----------------------------------------------------------------------------- launchers
size_t dispatch_workspace(int64_t T, int E) {
    const int64_t nch = (T + DCH - 1) / DCH;
    return (size_t)nch * E * sizeof(int32_t) + 256;
}

cudaError_t launch_dispatch(const int32_t* topk_idx, const void* x, int64_t T, int d, int E, int k,
                            bool bf16, int32_t* offsets, int32_t* slot_of, int32_t* token_of,
                            void* x_perm, void* ws, cudaStream_t s) {
    const int nch = (int)((T + DCH - 1) / DCH);
    int32_t* cc = (int32_t*)ws;
    if (T == 0) {
        return cudaMemsetAsync(offsets, 0, sizeof(int32_t) * (E + 1), s);
    }
    (void)launch_pdl(chunk_count_kernel, dim3(nch), dim3(DCH), 0, s, topk_idx, T, E, k, cc);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    (void)launch_pdl(slot_kernel, dim3(nch), dim3(DCH), 0, s, topk_idx, cc, T, E, k, nch, offsets, slot_of, token_of);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    const int64_t TK = T * k;
    const unsigned blocks = (unsigned)((TK + 7) / 8);
    if (bf16)
        (void)launch_pdl(gather_kernel<__nv_bfloat16>, dim3(blocks), dim3(256), 0, s, (const __nv_bfloat16*)x, token_of, TK, T,
                                                            d, (__nv_bfloat16*)x_perm);
    else
        (void)launch_pdl(gather_kernel<float>, dim3(blocks), dim3(256), 0, s, (const float*)x, token_of, TK, T, d,
                                                    (float*)x_perm);
    return cudaGetLastError();
}

cudaError_t launch_combine_fwd(const void* y_perm, const float* topk_w, const int32_t* slot_of,
                               const void* y_sh, int S, int64_t T, int d, int k, bool bf16,
                               void* out, cudaStream_t s) {
    if (T == 0) return cudaSuccess;
    const unsigned blocks = (unsigned)((T + 7) / 8);
#define MOE_CF(TT, KM)                                                                           \
    (void)launch_pdl(combine_fwd_kernel<TT, KM>, dim3(blocks), dim3(256), 0, s, (const TT*)y_perm, topk_w, slot_of,         \
                                                      (const TT*)y_sh, S, T, d, k, (TT*)out)
    if (bf16) {
        if (k <= 2) MOE_CF(__nv_bfloat16, 2);
        else if (k <= 4) MOE_CF(__nv_bfloat16, 4);
        else MOE_CF(__nv_bfloat16, 8);
    } else {
        if (k <= 2) MOE_CF(float, 2);
        else if (k <= 4) MOE_CF(float, 4);
        else MOE_CF(float, 8);
    }
#undef MOE_CF
    return cudaGetLastError();
}

cudaError_t launch_combine_bwd(const void* dout, const void* y_perm, const float* topk_w,
                               const int32_t* slot_of, int64_t T, int d, int k, bool bf16,
                               void* dy_perm, float* dtopk_w, cudaStream_t s) {
    if (T == 0) return cudaSuccess;
    const unsigned blocks = (unsigned)((T + 7) / 8);
#define MOE_CB(TT, KM)                                                                           \
    (void)launch_pdl(combine_bwd_kernel<TT, KM>, dim3(blocks), dim3(256), 0, s, (const TT*)dout, (const TT*)y_perm, topk_w, \
                                                      slot_of, T, d, k, (TT*)dy_perm, dtopk_w)
    if (bf16) {
        if (k <= 2) MOE_CB(__nv_bfloat16, 2);
        else if (k <= 4) MOE_CB(__nv_bfloat16, 4);
        else MOE_CB(__nv_bfloat16, 8);
    } else {
        if (k <= 2) MOE_CB(float, 2);
        else if (k <= 4) MOE_CB(float, 4);
        else MOE_CB(float, 8);
    }
#undef MOE_CB
    return cudaGetLastError();
}

cudaError_t launch_unpermute_reduce(const void* dx_perm, const int32_t* slot_of,
                                    const float* dlogits, const void* w_router,
                                    const int32_t* po, int P, const void* dx_sh, int S, int64_t T,
                                    int d, int E, int k, bool bf16, void* dx, cudaStream_t s) {
    if (T == 0) return cudaSuccess;
    const unsigned tiles = (unsigned)((T + UR_TOK - 1) / UR_TOK + P);
    const int VN = bf16 ? 8 : 4;
    const int slab = 64 * VN;
    dim3 grid(tiles, (d + slab - 1) / slab);
    const size_t smem = UR_TOK * 64 * sizeof(float) + (size_t)E * slab * (bf16 ? 2 : 4);
    if (bf16) {
        static bool attr = false;
        if (!attr) {
            cudaError_t e = cudaFuncSetAttribute(unpermute_reduce_kernel<__nv_bfloat16>,
                                                 cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                 (int)(UR_TOK * 64 * 4 + 64 * 512 * 2));
            if (e != cudaSuccess) return e;
            attr = true;
        }
        (void)launch_pdl(unpermute_reduce_kernel<__nv_bfloat16>, dim3(grid), dim3(256), smem, s, 
            (const __nv_bfloat16*)dx_perm, slot_of, dlogits, (const __nv_bfloat16*)w_router, po, P,
            (const __nv_bfloat16*)dx_sh, S, T, d, E, k, (__nv_bfloat16*)dx);
    } else {
        static bool attr = false;
        if (!attr) {
            cudaError_t e = cudaFuncSetAttribute(unpermute_reduce_kernel<float>,
                                                 cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                 (int)(UR_TOK * 64 * 4 + 64 * 256 * 4));
            if (e != cudaSuccess) return e;
            attr = true;
        }
        (void)launch_pdl(unpermute_reduce_kernel<float>, dim3(grid), dim3(256), smem, s, 
            (const float*)dx_perm, slot_of, dlogits, (const float*)w_router, po, P,
            (const float*)dx_sh, S, T, d, E, k, (float*)dx);
    }
    return cudaGetLastError();
}

// ----------------------------------------------------------------------------- no-alloc dispatch
// Dispatch for callers that cannot allocate device memory (their interface hands them
// only input and output buffers). The per-chunk counts live in this file-scope array
// instead of a caller workspace: every GPU that loads the library holds it until the
// process exits, and every call shares it. chunk_count_kernel overwrites each entry it
// uses, so nothing has to be cleared between calls; calls whose kernels overlap on the
// GPU (different streams, or several host threads) race on it.
static __device__ __align__(256) int32_t g_dispatch_scratch[kNoAllocScratchInts];

namespace {
constexpr int kMaxDevices = 64;
int32_t* g_scratch_ptr[kMaxDevices] = {};
}  // namespace

int64_t dispatch_noalloc_max_chunk_entries() { return kNoAllocScratchInts; }

cudaError_t launch_dispatch_noalloc(const int32_t* topk_idx, const void* x, int64_t T, int d, int E,
                                    int k, bool bf16, int32_t* offsets, int32_t* slot_of,
                                    int32_t* token_of, void* x_perm, cudaStream_t s) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    if (!g_scratch_ptr[dev]) {  // first call on this device: look the array up once
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_dispatch_scratch);
        if (e != cudaSuccess) return e;
        g_scratch_ptr[dev] = static_cast<int32_t*>(p);
    }
    int32_t* cc = g_scratch_ptr[dev];
    const int nch = (int)((T + DCH - 1) / DCH);
    if ((int64_t)nch * E > kNoAllocScratchInts) return cudaErrorInvalidValue;
    if (T == 0) return cudaMemsetAsync(offsets, 0, sizeof(int32_t) * (E + 1), s);
    (void)launch_pdl(chunk_count_kernel, dim3(nch), dim3(DCH), 0, s, topk_idx, T, E, k, cc);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    (void)launch_pdl(slot_kernel, dim3(nch), dim3(DCH), 0, s, topk_idx, cc, T, E, k, nch, offsets, slot_of, token_of);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    const int64_t TK = T * k;
    const unsigned blocks = (unsigned)((TK + 7) / 8);
    if (bf16)
        (void)launch_pdl(gather_kernel<__nv_bfloat16>, dim3(blocks), dim3(256), 0, s, (const __nv_bfloat16*)x, token_of, TK, T,
                                                            d, (__nv_bfloat16*)x_perm);
    else
        (void)launch_pdl(gather_kernel<float>, dim3(blocks), dim3(256), 0, s, (const float*)x, token_of, TK, T, d,
                                                    (float*)x_perm);
    return cudaGetLastError();
}

cudaError_t dispatch_status(cudaStream_t s, int* code) { return tu_status_read_clear(s, code); }

}  // namespace moe
