// The two training-step kernels of Alg. 1 around the layer: the regression loss of the
// toy block (its value and dL/dh) and the SGD update of the parameters a batch touches
// (the active party's gating, BackwardLocal of Alg. 4, and the experts it called,
// BackwardExpert of Alg. 6). Both are HBM-bound streams: 16-byte vector loads and
// stores, grids of a few CTAs per SM, fp32 arithmetic on bf16 or fp32 storage.
#include <algorithm>

#include "moe_common.cuh"
#include "moe_internal.h"

namespace moe {

// --------------------------------------------------------------------------- SGD
// w[g] <- w[g] - lr * dw[g] for every group g with counts[g] > 0 (or every group when
// counts is null). With a master copy (fp32, MASTER): master[g] <- master[g] - lr *
// dw[g] and w[g] <- master[g] rounded to T, so that updates smaller than T's spacing
// accumulate. Grid: (blocks per group, groups); a CTA of a group that was not called
// returns before touching memory, so an uncalled expert costs no traffic.
template <typename T, bool VEC, bool MASTER>
__global__ void __launch_bounds__(256) sgd_update_kernel(T* __restrict__ w, const T* __restrict__ dw,
                                                         float* __restrict__ master, int64_t group_elems,
                                                         const int32_t* __restrict__ counts, float lr) {
    pdl_begin();
    const int64_t g = blockIdx.y;
    if (counts && counts[g] <= 0) return;
    T* wg = w + g * group_elems;
    const T* dg = dw + g * group_elems;
    float* mg = MASTER ? master + g * group_elems : nullptr;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    const int64_t i0 = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if constexpr (VEC) {
        constexpr int VN = Vec<T>::N;
        const int64_t nv = group_elems / VN;
        for (int64_t v = i0; v < nv; v += stride) {
            float a[VN], b[VN];
            if constexpr (MASTER) {
#pragma unroll
                for (int h = 0; h < VN; h += 4) Vec<float>::load(mg + v * VN + h, a + h);
            } else {
                Vec<T>::load(wg + v * VN, a);
            }
            Vec<T>::load(dg + v * VN, b);
#pragma unroll
            for (int q = 0; q < VN; ++q) a[q] = fmaf(-lr, b[q], a[q]);
            if constexpr (MASTER) {
#pragma unroll
                for (int h = 0; h < VN; h += 4) Vec<float>::store(mg + v * VN + h, a + h);
            }
            Vec<T>::store(wg + v * VN, a);
        }
    } else {
        for (int64_t i = i0; i < group_elems; i += stride) {
            const float a = MASTER ? mg[i] : Elem<T>::load(wg + i);
            const float r = fmaf(-lr, Elem<T>::load(dg + i), a);
            if constexpr (MASTER) mg[i] = r;
            Elem<T>::store(wg + i, r);
        }
    }
}

static int sm_count_train() {
    static int n = 0;
    if (!n) {
        int dev = 0;
        if (cudaGetDevice(&dev) != cudaSuccess ||
            cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
            n = 148;
    }
    return n;
}

cudaError_t launch_sgd_update(void* w, const void* dw, float* master, int64_t n_groups, int64_t group_elems,
                              const int32_t* counts, float lr, bool bf16, cudaStream_t s) {
    if (n_groups == 0 || group_elems == 0) return cudaSuccess;
    const int vn = bf16 ? 8 : 4;
    const bool vec = group_elems % vn == 0 && ((uintptr_t)w % 16 == 0) && ((uintptr_t)dw % 16 == 0) &&
                     ((uintptr_t)master % 16 == 0);
    // about 8 CTAs per SM over all groups, none with less than one vector per thread
    const int64_t work = vec ? group_elems / vn : group_elems;
    int64_t bx = std::max<int64_t>(1, (8 * (int64_t)sm_count_train() + n_groups - 1) / n_groups);
    bx = std::min<int64_t>(bx, (work + 255) / 256);
    const dim3 grid((unsigned)std::max<int64_t>(bx, 1), (unsigned)n_groups);
#define MOE_SGD(TT, V, M)                                                                      \
    (void)launch_pdl(sgd_update_kernel<TT, V, M>, grid, dim3(256), 0, s, (TT*)w, (const TT*)dw, master, \
                     group_elems, counts, lr)
    if (bf16) {
        if (master) {
            if (vec) MOE_SGD(__nv_bfloat16, true, true);
            else MOE_SGD(__nv_bfloat16, false, true);
        } else {
            if (vec) MOE_SGD(__nv_bfloat16, true, false);
            else MOE_SGD(__nv_bfloat16, false, false);
        }
    } else {
        if (master) {
            if (vec) MOE_SGD(float, true, true);
            else MOE_SGD(float, false, true);
        } else {
            if (vec) MOE_SGD(float, true, false);
            else MOE_SGD(float, false, false);
        }
    }
#undef MOE_SGD
    return cudaGetLastError();
}

// --------------------------------------------------------------------------- MSE
// Pass 1 (MSE_BLOCKS CTAs, each a fixed slice of the vectors): dout = (out - y) / T in
// the storage type, and the CTA's sum of (out - y)^2 into partial[cta]. Pass 2 (one
// CTA): the partials in a fixed order, loss = sum / (2T). The same bits on every run.
constexpr int MSE_BLOCKS = 512;
constexpr int MSE_THREADS = 256;

__device__ __forceinline__ float block_sum(float v, float* red) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) red[warp] = v;
    __syncthreads();
    float s = 0.f;
    if (warp == 0) {
        s = lane < (int)(blockDim.x >> 5) ? red[lane] : 0.f;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    }
    return s;  // valid in thread 0
}

template <typename T, bool VEC>
__global__ void __launch_bounds__(MSE_THREADS) mse_partial_kernel(const T* __restrict__ out,
                                                                   const T* __restrict__ y, int64_t n,
                                                                   float inv_T, T* __restrict__ dout,
                                                                   float* __restrict__ partial) {
    pdl_begin();
    __shared__ float red[MSE_THREADS / 32];
    float acc = 0.f;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    const int64_t i0 = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if constexpr (VEC) {
        constexpr int VN = Vec<T>::N;
        const int64_t nv = n / VN;
        for (int64_t v = i0; v < nv; v += stride) {
            float a[VN], b[VN];
            Vec<T>::load(out + v * VN, a);
            Vec<T>::load(y + v * VN, b);
#pragma unroll
            for (int q = 0; q < VN; ++q) {
                const float dlt = a[q] - b[q];
                acc = fmaf(dlt, dlt, acc);
                a[q] = dlt * inv_T;
            }
            Vec<T>::store(dout + v * VN, a);
        }
    } else {
        for (int64_t i = i0; i < n; i += stride) {
            const float dlt = Elem<T>::load(out + i) - Elem<T>::load(y + i);
            acc = fmaf(dlt, dlt, acc);
            Elem<T>::store(dout + i, dlt * inv_T);
        }
    }
    const float s = block_sum(acc, red);
    if (threadIdx.x == 0) partial[blockIdx.x] = s;
}

__global__ void __launch_bounds__(MSE_THREADS) mse_final_kernel(const float* __restrict__ partial, int nb,
                                                                 float half_inv_T, float* __restrict__ loss) {
    pdl_begin();
    __shared__ float red[MSE_THREADS / 32];
    float acc = 0.f;
    for (int i = threadIdx.x; i < nb; i += blockDim.x) acc += partial[i];
    const float s = block_sum(acc, red);
    if (threadIdx.x == 0) loss[0] = s * half_inv_T;
}

size_t mse_workspace_bytes() { return MSE_BLOCKS * sizeof(float); }

cudaError_t launch_mse_loss(const void* out, const void* y, int64_t T, int d, bool bf16, float* loss,
                            void* dout, void* workspace, cudaStream_t s) {
    const int64_t n = T * (int64_t)d;
    const int vn = bf16 ? 8 : 4;
    const bool vec = n % vn == 0 && (uintptr_t)out % 16 == 0 && (uintptr_t)y % 16 == 0 &&
                     (uintptr_t)dout % 16 == 0;
    const float inv_T = 1.0f / (float)T;
    float* partial = (float*)workspace;
#define MOE_MSE(TT, V)                                                                          \
    (void)launch_pdl(mse_partial_kernel<TT, V>, dim3(MSE_BLOCKS), dim3(MSE_THREADS), 0, s,        \
                     (const TT*)out, (const TT*)y, n, inv_T, (TT*)dout, partial)
    if (bf16) {
        if (vec) MOE_MSE(__nv_bfloat16, true);
        else MOE_MSE(__nv_bfloat16, false);
    } else {
        if (vec) MOE_MSE(float, true);
        else MOE_MSE(float, false);
    }
#undef MOE_MSE
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    (void)launch_pdl(mse_final_kernel, dim3(1), dim3(MSE_THREADS), 0, s, (const float*)partial, MSE_BLOCKS,
                     0.5f * inv_T, loss);
    return cudaGetLastError();
}

}  // namespace moe
