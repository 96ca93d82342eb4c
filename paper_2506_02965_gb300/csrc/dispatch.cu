// Token dispatch (the "send h to the host of idx" step of Alg. 3 as one expert-major
// buffer), the gate-weighted combine of Alg. 3 and the backward of both (Alg. 5,
// Sec. 3.2). All memory-bound: 16-byte vector loads/stores, one warp per token or
// per permuted row, no floating-point atomics (every result is deterministic).
#include <algorithm>
#include <atomic>

#include "moe_common.cuh"
#include "moe_internal.h"

namespace moe {

constexpr int DCH = kDispatchChunkTokens;  // tokens per dispatch chunk (one thread each)
constexpr int EMAX = 256;                  // experts (shared-memory tables below)

// Per chunk: how many of its (token, pick) pairs went to each expert. Also checks
// that every index lies in [0, E) and that no token picks an expert twice. With `send`
// (owner-grouped dispatch) it also adds each pair to send[party(t) * P + e mod P]
// (integer additions: the totals do not depend on their order).
constexpr int SEND_SMEM = 1024;  // P*P counters staged in shared memory up to this many
__global__ void __launch_bounds__(DCH) chunk_count_kernel(const int32_t* __restrict__ idx,
                                                          int64_t T, int E, int k,
                                                          int32_t* chunk_counts,
                                                          const int32_t* __restrict__ po, int P,
                                                          int32_t* send) {
    pdl_begin();
    __shared__ int s_cnt[EMAX];
    __shared__ int s_send[SEND_SMEM];
    const bool send_smem = send && P * P <= SEND_SMEM;
    for (int i = threadIdx.x; i < E; i += blockDim.x) s_cnt[i] = 0;
    if (send_smem)
        for (int i = threadIdx.x; i < P * P; i += blockDim.x) s_send[i] = 0;
    __syncthreads();
    const int64_t t = (int64_t)blockIdx.x * DCH + threadIdx.x;
    if (t < T) {
        const int src = send ? party_of(po, P, t) : 0;
        for (int j = 0; j < k; ++j) {
            const int e = idx[t * k + j];
            bool ok = (e >= 0 && e < E);
            for (int jj = 0; jj < j; ++jj) ok = ok && (idx[t * k + jj] != e);
            if (ok) {
                atomicAdd(&s_cnt[e], 1);
                if (send_smem) atomicAdd(&s_send[src * P + e % P], 1);
                else if (send) atomicAdd(&send[src * P + e % P], 1);
            } else {
                record_status(MOE_ERR_DEVICE_CHECK);
            }
        }
    }
    __syncthreads();
    for (int i = threadIdx.x; i < E; i += blockDim.x)
        chunk_counts[(int64_t)blockIdx.x * E + i] = s_cnt[i];
    if (send_smem)
        for (int i = threadIdx.x; i < P * P; i += blockDim.x)
            if (s_send[i]) atomicAdd(&send[i], s_send[i]);
}

// Per chunk: offsets (written by chunk 0), the chunk's base row inside each expert
// segment, and the stable rank of each pick among the chunk's picks of that expert
// (a bit per token and expert, counted with popc). The expert segments follow in
// (e mod Pown, e) order: expert order for Pown = 1, owner-grouped for Pown = P (chunk 0
// then also writes group_expert[g] = the expert of segment g).
__global__ void __launch_bounds__(DCH) slot_kernel(const int32_t* __restrict__ idx,
                                                   const int32_t* __restrict__ chunk_counts,
                                                   int64_t T, int E, int k, int nchunks,
                                                   int32_t* offsets, int32_t* slot_of,
                                                   int32_t* token_of, int Pown,
                                                   int32_t* group_expert) {
    pdl_begin();
    __shared__ int s_pre[EMAX];
    __shared__ int s_tot[EMAX];
    __shared__ int s_base[EMAX];
    __shared__ unsigned s_bits[EMAX][DCH / 32];
    __shared__ int s_ppre[DCH], s_ptot[DCH];  // per (group, expert) partial sums
    constexpr int TAB = 6144;  // chunk-count table staged in shared memory when it fits
    __shared__ int s_tab[TAB];
    const int c = blockIdx.x;
    const int64_t ntab = (int64_t)nchunks * E;
    if (ntab <= TAB) {
        for (int i = threadIdx.x; i < ntab; i += blockDim.x) s_tab[i] = chunk_counts[i];
        __syncthreads();
    }
    // per expert: the picks of the chunks before this one (pre) and of all chunks (tot).
    // With E <= DCH the block's threads form G = DCH / E groups per expert, group g adding
    // the chunks g, g + G, ...; the groups are then summed (integers: exact in any order).
    auto cnt = [&](int cc, int e) {
        return ntab <= TAB ? s_tab[cc * E + e] : chunk_counts[(int64_t)cc * E + e];
    };
    if (E <= DCH) {
        const int G = DCH / E, e = threadIdx.x % E, g = threadIdx.x / E;
        int pre = 0, tot = 0;
        if (g < G) {
            for (int cc = g; cc < nchunks; cc += G) {
                const int v = cnt(cc, e);
                if (cc < c) pre += v;
                tot += v;
            }
        }
        s_ppre[threadIdx.x] = pre;
        s_ptot[threadIdx.x] = tot;
        __syncthreads();
        if (threadIdx.x < E) {
            int p2 = 0, t2 = 0;
            for (int q = 0; q < G; ++q) {
                p2 += s_ppre[q * E + threadIdx.x];
                t2 += s_ptot[q * E + threadIdx.x];
            }
            s_pre[threadIdx.x] = p2;
            s_tot[threadIdx.x] = t2;
        }
    } else {
        for (int e = threadIdx.x; e < E; e += blockDim.x) {
            int pre = 0, tot = 0;
            for (int cc = 0; cc < nchunks; ++cc) {
                const int v = cnt(cc, e);
                if (cc < c) pre += v;
                tot += v;
            }
            s_pre[e] = pre;
            s_tot[e] = tot;
        }
    }
    for (int i = threadIdx.x; i < EMAX * (DCH / 32); i += blockDim.x) (&s_bits[0][0])[i] = 0u;
    __syncthreads();
    if (threadIdx.x == 0) {
        int run = 0, g = 0;
        for (int o = 0; o < Pown; ++o) {
            for (int e = o; e < E; e += Pown, ++g) {
                if (c == 0) {
                    offsets[g] = run;
                    if (group_expert) group_expert[g] = e;
                }
                s_base[e] = run + s_pre[e];
                run += s_tot[e];
            }
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

// x_perm[slot_of[t,j]] = x[t] for every pick j: one warp per token reads its row once
// (16-byte vectors, U of them in flight per lane) and writes it to its k rows of x_perm.
// A slot outside [0, T k) is skipped and recorded as MOE_ERR_DEVICE_CHECK.
template <typename T>
__global__ void __launch_bounds__(256) gather_kernel(const T* __restrict__ x,
                                                     const int32_t* __restrict__ slot_of,
                                                     int64_t Tn, int d, int k, T* x_perm) {
    pdl_begin();
    const int lane = threadIdx.x & 31;
    const int64_t t = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    if (t >= Tn) return;
    int32_t slot[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
        slot[j] = j < k ? slot_of[t * k + j] : -1;
        if (j < k && (slot[j] < 0 || (int64_t)slot[j] >= Tn * k)) {
            if (lane == 0) record_status(MOE_ERR_DEVICE_CHECK);
            slot[j] = -1;
        }
    }
    constexpr int VN = Vec<T>::N;
    constexpr int U = 4;  // vectors per lane in flight
    const int nv = d / VN;
    const T* src = x + t * d;
    for (int v0 = lane; v0 < nv; v0 += 32 * U) {
        uint4 buf[U];
#pragma unroll
        for (int u = 0; u < U; ++u)
            if (v0 + 32 * u < nv) buf[u] = Vec<T>::raw_load(src + (v0 + 32 * u) * VN);
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            if (slot[j] < 0) continue;
            T* dst = x_perm + (int64_t)slot[j] * d;
#pragma unroll
            for (int u = 0; u < U; ++u)
                if (v0 + 32 * u < nv) Vec<T>::raw_store(dst + (v0 + 32 * u) * VN, buf[u]);
        }
    }
}

// dst[i] = src[rows[i]] for n rows of `row_vecs` 16-byte vectors: one warp per row.
// A row index outside [0, n_src) leaves dst[i] untouched and records
// MOE_ERR_DEVICE_CHECK.
__global__ void __launch_bounds__(256) gather_rows_kernel(const uint4* __restrict__ src,
                                                          const int32_t* __restrict__ rows,
                                                          int64_t n, int64_t n_src, int row_vecs,
                                                          uint4* dst) {
    pdl_begin();
    const int lane = threadIdx.x & 31;
    const int64_t i = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    if (i >= n) return;
    const int64_t r = rows[i];
    if (r < 0 || r >= n_src) {
        if (lane == 0) record_status(MOE_ERR_DEVICE_CHECK);
        return;
    }
    constexpr int U = 4;
    const uint4* s = src + r * row_vecs;
    uint4* o = dst + i * row_vecs;
    for (int v0 = lane; v0 < row_vecs; v0 += 32 * U) {
        uint4 buf[U];
#pragma unroll
        for (int u = 0; u < U; ++u)
            if (v0 + 32 * u < row_vecs) buf[u] = s[v0 + 32 * u];
#pragma unroll
        for (int u = 0; u < U; ++u)
            if (v0 + 32 * u < row_vecs) o[v0 + 32 * u] = buf[u];
    }
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

// dx[t] = sum_j dx_perm[slot(t,j)] + dx_router[t] + sum_s dx_sh[s,t]; fp32 accumulation.
// One warp per token; every lane issues the loads of up to UB vectors of all k rows (and
// of the router's row) before it uses any of them.
template <typename T, int KMAX>
__global__ void __launch_bounds__(256, 3) unpermute_reduce_kernel(
    const T* __restrict__ dx_perm, const int32_t* __restrict__ slot_of,
    const T* __restrict__ dx_router, const T* __restrict__ dx_sh, int S, int64_t Tn, int d, int k,
    T* dx) {
    pdl_begin();
    const int lane = threadIdx.x & 31;
    const int64_t t = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    if (t >= Tn) return;
    constexpr int VN = Vec<T>::N;
    constexpr int UB = KMAX <= 2 ? 4 : KMAX <= 4 ? 2 : 1;  // vectors per lane in flight
    int32_t slot[KMAX];
#pragma unroll
    for (int j = 0; j < KMAX; ++j) {
        slot[j] = j < k ? slot_of[t * k + j] : -1;
        if (j < k && (slot[j] < 0 || (int64_t)slot[j] >= Tn * k)) {  // bad table: skip the row
            if (lane == 0) record_status(MOE_ERR_DEVICE_CHECK);
            slot[j] = -1;
        }
    }
    const int nv = d / VN;
    for (int v0 = lane; v0 < nv; v0 += 32 * UB) {
        uint4 raw[UB][KMAX], rr[UB];
#pragma unroll
        for (int u = 0; u < UB; ++u) {
            const int v = v0 + 32 * u;
            if (v < nv) {
#pragma unroll
                for (int j = 0; j < KMAX; ++j)
                    if (slot[j] >= 0) raw[u][j] = Vec<T>::raw_load(dx_perm + (int64_t)slot[j] * d + v * VN);
                if (dx_router) rr[u] = Vec<T>::raw_load(dx_router + t * d + v * VN);
            }
        }
#pragma unroll
        for (int u = 0; u < UB; ++u) {
            const int v = v0 + 32 * u;
            if (v >= nv) break;
            float acc[VN];
            if (dx_router) {
                unpack_vec<T>(rr[u], acc);
            } else {
#pragma unroll
                for (int q = 0; q < VN; ++q) acc[q] = 0.f;
            }
#pragma unroll
            for (int j = 0; j < KMAX; ++j) {
                if (slot[j] >= 0) {
                    float g[VN];
                    unpack_vec<T>(raw[u][j], g);
#pragma unroll
                    for (int q = 0; q < VN; ++q) acc[q] += g[q];
                }
            }
            for (int s2 = 0; s2 < S; ++s2) {
                float g[VN];
                Vec<T>::load(dx_sh + ((int64_t)s2 * Tn + t) * d + v * VN, g);
#pragma unroll
                for (int q = 0; q < VN; ++q) acc[q] += g[q];
            }
            Vec<T>::store(dx + t * d + v * VN, acc);
        }
    }
}

// ----------------------------------------------------------------------------- launchers
static cudaError_t launch_gather(const void* x, const int32_t* slot_of, int64_t T, int d, int k, bool bf16,
                                 void* x_perm, cudaStream_t s) {
    const unsigned blocks = (unsigned)((T + 7) / 8);
    if (bf16)
        (void)launch_pdl(gather_kernel<__nv_bfloat16>, dim3(blocks), dim3(256), 0, s, (const __nv_bfloat16*)x,
                         slot_of, T, d, k, (__nv_bfloat16*)x_perm);
    else
        (void)launch_pdl(gather_kernel<float>, dim3(blocks), dim3(256), 0, s, (const float*)x, slot_of, T, d, k,
                         (float*)x_perm);
    return cudaGetLastError();
}

size_t dispatch_workspace(int64_t T, int E) {
    const int64_t nch = (T + DCH - 1) / DCH;
    return (size_t)nch * E * sizeof(int32_t) + 256;
}

cudaError_t launch_dispatch(const int32_t* topk_idx, const void* x, int64_t T, int d, int E, int k,
                            bool bf16, int32_t* offsets, int32_t* slot_of, int32_t* token_of,
                            void* x_perm, void* ws, cudaStream_t s, const int32_t* po, int P,
                            int32_t* group_expert, int32_t* send) {
    const bool owner = send != nullptr;
    const int nch = (int)std::max<int64_t>(owner ? 1 : 0, (T + DCH - 1) / DCH);
    int32_t* cc = (int32_t*)ws;
    cudaError_t e;
    if (owner) {
        if ((e = cudaMemsetAsync(send, 0, sizeof(int32_t) * P * P, s)) != cudaSuccess) return e;
    } else if (T == 0) {
        return cudaMemsetAsync(offsets, 0, sizeof(int32_t) * (E + 1), s);
    }
    (void)launch_pdl(chunk_count_kernel, dim3(nch), dim3(DCH), 0, s, topk_idx, T, E, k, cc, po,
                     owner ? P : 1, send);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    (void)launch_pdl(slot_kernel, dim3(nch), dim3(DCH), 0, s, topk_idx, cc, T, E, k, nch, offsets,
                     slot_of, token_of, owner ? P : 1, group_expert);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    if (T * k == 0) return cudaSuccess;
    return launch_gather(x, slot_of, T, d, k, bf16, x_perm, s);
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
                                    const void* dx_router, const void* dx_sh, int S, int64_t T,
                                    int d, int k, bool bf16, void* dx, cudaStream_t s) {
    if (T == 0) return cudaSuccess;
    const unsigned blocks = (unsigned)((T + 7) / 8);
#define MOE_UR(TT, KM)                                                                            \
    (void)launch_pdl(unpermute_reduce_kernel<TT, KM>, dim3(blocks), dim3(256), 0, s,              \
                     (const TT*)dx_perm, slot_of, (const TT*)dx_router, (const TT*)dx_sh, S, T, d, \
                     k, (TT*)dx)
    if (bf16) {
        if (k <= 2) MOE_UR(__nv_bfloat16, 2);
        else if (k <= 4) MOE_UR(__nv_bfloat16, 4);
        else MOE_UR(__nv_bfloat16, 8);
    } else {
        if (k <= 2) MOE_UR(float, 2);
        else if (k <= 4) MOE_UR(float, 4);
        else MOE_UR(float, 8);
    }
#undef MOE_UR
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
// Device address of g_dispatch_scratch per device, looked up on the first call there.
// Two threads that make their first call at once both look it up and store the same
// value; the atomic makes that well defined.
std::atomic<int32_t*> g_scratch_ptr[kMaxDevices] = {};
}  // namespace

int64_t dispatch_noalloc_max_chunk_entries() { return kNoAllocScratchInts; }

cudaError_t launch_dispatch_noalloc(const int32_t* topk_idx, const void* x, int64_t T, int d, int E,
                                    int k, bool bf16, int32_t* offsets, int32_t* slot_of,
                                    int32_t* token_of, void* x_perm, cudaStream_t s) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    int32_t* cc = g_scratch_ptr[dev].load(std::memory_order_acquire);
    if (!cc) {  // first call on this device: look the array up once
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_dispatch_scratch);
        if (e != cudaSuccess) return e;
        cc = static_cast<int32_t*>(p);
        g_scratch_ptr[dev].store(cc, std::memory_order_release);
    }
    const int nch = (int)((T + DCH - 1) / DCH);
    if ((int64_t)nch * E > kNoAllocScratchInts) return cudaErrorInvalidValue;
    if (T == 0) return cudaMemsetAsync(offsets, 0, sizeof(int32_t) * (E + 1), s);
    (void)launch_pdl(chunk_count_kernel, dim3(nch), dim3(DCH), 0, s, topk_idx, T, E, k, cc,
                     (const int32_t*)nullptr, 1, (int32_t*)nullptr);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    (void)launch_pdl(slot_kernel, dim3(nch), dim3(DCH), 0, s, topk_idx, cc, T, E, k, nch, offsets,
                     slot_of, token_of, 1, (int32_t*)nullptr);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    return launch_gather(x, slot_of, T, d, k, bf16, x_perm, s);
}

cudaError_t launch_gather_rows(const void* src, const int32_t* rows, int64_t n, int64_t n_src,
                               int64_t row_bytes, void* dst, cudaStream_t s) {
    if (n == 0) return cudaSuccess;
    const unsigned blocks = (unsigned)((n + 7) / 8);
    (void)launch_pdl(gather_rows_kernel, dim3(blocks), dim3(256), 0, s, (const uint4*)src, rows, n, n_src,
                     (int)(row_bytes / 16), (uint4*)dst);
    return cudaGetLastError();
}

cudaError_t dispatch_status(cudaStream_t s, int* code) { return tu_status_read_clear(s, code); }

}  // namespace moe
