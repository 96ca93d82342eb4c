// fp32 grouped expert GEMMs on the CUDA cores (FFMA), for the fp32 configuration.
// TF32 tensor cores would not meet a 1e-4 relative error bound, so fp32 inputs take
// this path. Same argument meaning as the tensor-core kernels (moe_internal.h):
// M-variable groups (forward, dA, dX) and K-variable groups (dW1, dW2).
#include "moe_common.cuh"
#include "moe_internal.h"

namespace moe {

constexpr int SB_M = 64, SB_N = 64, SB_K = 16;

// Group g and first row of M-tile `mt` (64 rows) for M-variable launches.
__device__ __forceinline__ bool locate_mtile(const GroupRows& gr, int G, int mt, int* g_out,
                                             int64_t* a_row0, int64_t* out_row0, int* m0,
                                             int* mrows) {
    int acc = 0;
    for (int g = 0; g < G; ++g) {
        int64_t r0, n;
        if (gr.offsets) {
            r0 = gr.offsets[g];
            n = gr.offsets[g + 1] - r0;
        } else {
            r0 = 0;
            n = gr.rows;
        }
        const int nt = (int)((n + SB_M - 1) / SB_M);
        if (mt < acc + nt) {
            *g_out = g;
            *m0 = (mt - acc) * SB_M;
            *mrows = (int)n;
            if (gr.offsets) {
                *a_row0 = r0;
                *out_row0 = r0;
            } else {
                *a_row0 = (int64_t)g * gr.a_stride;
                *out_row0 = (int64_t)g * gr.out_stride;
            }
            return true;
        }
        acc += nt;
    }
    return false;
}

// Column c of the 64-wide tile -> weight row n. SwiGLU forward tiles hold 32 features
// f: thread column group tx owns gate f0+2tx, f0+2tx+1 and up f0+2tx, f0+2tx+1, so
// the epilogue finds G and U of the same feature in one thread.
__device__ __forceinline__ int tile_col_to_n(int epi, int c, int n0, int F) {
    if (epi != EPI_SWIGLU_FWD) return n0 + c;
    const int tx = c >> 2, q = c & 3;
    const int f = n0 + 2 * tx + (q & 1);
    return (q >> 1) ? F + f : f;
}

__global__ void __launch_bounds__(256) gemm_m_simt_kernel(GemmMArgs p) {
    pdl_begin();
    __shared__ float As[SB_K][SB_M + 4];
    __shared__ float Bs[SB_K][SB_N + 4];
    int g, m0, mrows;
    int64_t a_row0, out_row0;
    if (!locate_mtile(p.rows, p.G, blockIdx.y, &g, &a_row0, &out_row0, &m0, &mrows)) return;
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    const int K = p.K, N = p.N;
    const int F = (p.epi == EPI_SWIGLU_FWD) ? N / 2 : N;
    const int n0 = blockIdx.x * (p.epi == EPI_SWIGLU_FWD ? SB_N / 2 : SB_N);
    const float* A = (const float*)p.a;
    const float* B = (const float*)p.b + (int64_t)(p.group_expert ? p.group_expert[g] : g) * p.b_group_elems;
    const int Nb = (p.epi == EPI_SWIGLU_FWD) ? N : N;  // rows of B viewed as [Nb, K]
    float acc[4][4] = {};
    for (int k0 = 0; k0 < K; k0 += SB_K) {
        // A tile: 64 rows x 16 k
        for (int i = tid; i < SB_M * SB_K; i += 256) {
            const int r = i / SB_K, kk = i % SB_K;
            const int m = m0 + r;
            float v = 0.f;
            if (m < mrows && k0 + kk < K) v = A[(a_row0 + m) * K + k0 + kk];
            As[kk][r] = v;
        }
        for (int i = tid; i < SB_N * SB_K; i += 256) {
            int c, kk;
            if (p.b_kmajor) { c = i / SB_K; kk = i % SB_K; }
            else { kk = i / SB_N; c = i % SB_N; }
            const int n = tile_col_to_n(p.epi, c, n0, F);
            float v = 0.f;
            if (n < Nb && k0 + kk < K)
                v = p.b_kmajor ? B[(int64_t)n * K + k0 + kk] : B[(int64_t)(k0 + kk) * Nb + n];
            Bs[kk][c] = v;
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < SB_K; ++kk) {
            float a[4], b[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) a[i] = As[kk][ty * 4 + i];
#pragma unroll
            for (int j = 0; j < 4; ++j) b[j] = Bs[kk][tx * 4 + j];
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
        }
        __syncthreads();
    }
    // epilogue
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int m = m0 + ty * 4 + i;
        if (m >= mrows) continue;
        const int64_t row = out_row0 + m;
        if (p.epi == EPI_SWIGLU_FWD) {
            float* hgu = (float*)p.out0;
            float* act = (float*)p.out1;
#pragma unroll
            for (int q = 0; q < 2; ++q) {
                const int f = n0 + 2 * tx + q;
                if (f >= F) continue;
                const float G = acc[i][q], U = acc[i][2 + q];
                hgu[row * 2 * F + f] = G;
                hgu[row * 2 * F + F + f] = U;
                act[row * F + f] = G * sigmoidf_(G) * U;
            }
        } else if (p.epi == EPI_STORE) {
            float* out = (float*)p.out0;
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int n = n0 + tx * 4 + j;
                if (n < N) out[row * N + n] = acc[i][j];
            }
        } else {  // SWIGLU_BWD: acc = dA[row, f], N = F
            const float* hgu = (const float*)p.aux;
            float* dh = (float*)p.out0;
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int f = n0 + tx * 4 + j;
                if (f >= N) continue;
                const float G = hgu[row * 2 * N + f], U = hgu[row * 2 * N + N + f];
                const float s = sigmoidf_(G);
                const float dA = acc[i][j];
                dh[row * 2 * N + N + f] = dA * G * s;
                dh[row * 2 * N + f] = dA * U * s * (1.f + G * (1.f - s));
            }
        }
    }
}

__global__ void __launch_bounds__(256) gemm_k_simt_kernel(GemmKArgs p) {
    pdl_begin();
    __shared__ float As[SB_K][SB_M + 4];
    __shared__ float Bs[SB_K][SB_N + 4];
    const int g = blockIdx.z;
    const int m0 = blockIdx.y * SB_M, n0 = blockIdx.x * SB_N;
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    int64_t ra, rb, nrows;
    if (p.rows.offsets) {
        ra = rb = p.rows.offsets[g];
        nrows = p.rows.offsets[g + 1] - ra;
    } else {
        ra = (int64_t)g * p.rows.a_stride;
        rb = (int64_t)g * p.rows.b_stride;
        nrows = p.rows.rows;
    }
    const float* A = (const float*)p.a;
    const float* B = (const float*)p.b;
    const int M = p.M, N = p.N;
    float acc[4][4] = {};
    for (int64_t k0 = 0; k0 < nrows; k0 += SB_K) {
        for (int i = tid; i < SB_M * SB_K; i += 256) {
            const int kk = i / SB_M, c = i % SB_M;
            float v = 0.f;
            if (k0 + kk < nrows && m0 + c < M) v = A[(ra + k0 + kk) * M + m0 + c];
            As[kk][c] = v;
        }
        for (int i = tid; i < SB_N * SB_K; i += 256) {
            const int kk = i / SB_N, c = i % SB_N;
            float v = 0.f;
            if (k0 + kk < nrows && n0 + c < N) v = B[(rb + k0 + kk) * N + n0 + c];
            Bs[kk][c] = v;
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < SB_K; ++kk) {
            float a[4], b[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) a[i] = As[kk][ty * 4 + i];
#pragma unroll
            for (int j = 0; j < 4; ++j) b[j] = Bs[kk][tx * 4 + j];
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
        }
        __syncthreads();
    }
    float* out = (float*)p.out + (int64_t)(p.group_expert ? p.group_expert[g] : g) * M * N;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int m = m0 + ty * 4 + i;
        if (m >= M) continue;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int n = n0 + tx * 4 + j;
            if (n < N) out[(int64_t)m * N + n] = acc[i][j];
        }
    }
}

cudaError_t launch_gemm_m_simt(const GemmMArgs& g, cudaStream_t s) {
    const int ncols = (g.epi == EPI_SWIGLU_FWD) ? g.N / 2 : g.N;
    const int per = (g.epi == EPI_SWIGLU_FWD) ? SB_N / 2 : SB_N;
    int64_t mt_ub;
    if (g.rows.offsets) {
        // sum over groups of ceil(M_g/64) <= ceil(total/64) + G; total rows <= caller's bound
        mt_ub = g.rows.rows / SB_M + g.G + 1;  // rows holds the total row count here
    } else {
        mt_ub = (int64_t)g.G * ((g.rows.rows + SB_M - 1) / SB_M);
    }
    if (mt_ub <= 0) return cudaSuccess;
    dim3 grid((ncols + per - 1) / per, (unsigned)mt_ub);
    (void)launch_pdl(gemm_m_simt_kernel, dim3(grid), dim3(256), 0, s, g);
    return cudaGetLastError();
}

cudaError_t launch_gemm_k_simt(const GemmKArgs& g, cudaStream_t s) {
    dim3 grid((g.N + SB_N - 1) / SB_N, (g.M + SB_M - 1) / SB_M, g.G);
    (void)launch_pdl(gemm_k_simt_kernel, dim3(grid), dim3(256), 0, s, g);
    return cudaGetLastError();
}

cudaError_t simt_status(cudaStream_t s, int* code) { return tu_status_read_clear(s, code); }

}  // namespace moe
