// Launchers shared between the kernel translation units and the C ABI (host side).
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

namespace moe {

struct RouteArgs {
    const void* x;          // [T,d] dtype
    const void* w_router;   // [P,E,d] dtype
    const float* bias;      // [P,E] or null
    const float* logits_in; // [T,E] (from-logits path)
    const int32_t* po;      // [P+1] or null
    int P;
    int64_t T;
    int d, E, k, normalize;
    float* logits;
    float* probs;
    int32_t* topk_idx;
    float* topk_w;
    int32_t* counts;        // [P,E]
};

struct RouteBwdArgs {
    const void* x;
    const float* probs;
    const int32_t* topk_idx;
    const float* topk_w;
    const float* dtopk_w;
    const float* aux_coef;  // [P,E] or null
    const int32_t* po;
    int P;
    int64_t T;
    int d, E, k, normalize;
    float* dlogits;
    void* dw_router;
    float* dbias;
    const void* w_router;  // [P,E,d]
    void* dx_router;       // [T,d] or null
};

cudaError_t launch_route(const RouteArgs& a, bool bf16, bool from_logits, cudaStream_t s);
// bf16 router logits on the tensor cores with the gating epilogue (E <= 64, E % 4 == 0)
cudaError_t launch_route_tc(const RouteArgs& a, cudaStream_t s);
cudaError_t launch_aux_loss(const float* probs, const int32_t* counts, const int32_t* po, int P,
                            int64_t T, int E, int k, float alpha, float* loss, float* coef,
                            cudaStream_t s);
size_t route_bwd_workspace(int64_t T, int P, int E, int d);
cudaError_t launch_route_bwd(const RouteBwdArgs& a, bool bf16, void* ws, cudaStream_t s);
cudaError_t route_status(cudaStream_t s, int* code);

// dispatch / combine
constexpr int kDispatchChunkTokens = 128;  // tokens per dispatch chunk (per-chunk expert counts)
size_t dispatch_workspace(int64_t T, int E);
cudaError_t launch_dispatch(const int32_t* topk_idx, const void* x, int64_t T, int d, int E, int k,
                            bool bf16, int32_t* offsets, int32_t* slot_of, int32_t* token_of,
                            void* x_perm, void* ws, cudaStream_t s,
                            const int32_t* po = nullptr, int P = 1,
                            int32_t* group_expert = nullptr, int32_t* send = nullptr);
cudaError_t launch_combine_fwd(const void* y_perm, const float* topk_w, const int32_t* slot_of,
                               const void* y_sh, int S, int64_t T, int d, int k, bool bf16,
                               void* out, cudaStream_t s);
cudaError_t launch_combine_bwd(const void* dout, const void* y_perm, const float* topk_w,
                               const int32_t* slot_of, int64_t T, int d, int k, bool bf16,
                               void* dy_perm, float* dtopk_w, cudaStream_t s);
cudaError_t launch_unpermute_reduce(const void* dx_perm, const int32_t* slot_of,
                                    const void* dx_router, const void* dx_sh, int S, int64_t T,
                                    int d, int k, bool bf16, void* dx, cudaStream_t s);
cudaError_t dispatch_status(cudaStream_t s, int* code);
// dst[i] = src[rows[i]] (row_bytes a multiple of 16)
cudaError_t launch_gather_rows(const void* src, const int32_t* rows, int64_t n, int64_t n_src,
                               int64_t row_bytes, void* dst, cudaStream_t s);
// dispatch with its per-chunk counts in a fixed device array (no workspace argument)
constexpr int64_t kNoAllocScratchInts = 1 << 16;  // 256 KiB of int32 chunk counts
int64_t dispatch_noalloc_max_chunk_entries();
cudaError_t launch_dispatch_noalloc(const int32_t* topk_idx, const void* x, int64_t T, int d, int E,
                                    int k, bool bf16, int32_t* offsets, int32_t* slot_of,
                                    int32_t* token_of, void* x_perm, cudaStream_t s);

// grouped GEMMs -------------------------------------------------------------------------
enum EpiKind { EPI_SWIGLU_FWD = 0, EPI_STORE = 1, EPI_SWIGLU_BWD = 2, EPI_ROUTE = 3, EPI_DWR = 4 };

// How the groups (experts) of a grouped GEMM are laid out along the rows that vary:
//  OFFSETS: group g owns rows [offsets[g], offsets[g+1]) of A / out (M-variable) or of
//           both operands (K-variable);
//  UNIFORM: every group has `rows` rows; group g starts at g*a_stride in A (or in the
//           first operand), g*b_stride in the second operand (K-variable) and at
//           g*out_stride in the output.
struct GroupRows {
    const int32_t* offsets;  // OFFSETS mode when non-null
    int rows;                // UNIFORM: rows per group; OFFSETS: total rows of all groups
    int64_t a_stride, b_stride, out_stride;
};

// C[M_g, N] = A_g[M_g, K] * B_g[N, K]^T per group g, M varying per group.
//  A: [rows, K] dtype row-major (rows of all groups)
//  B: group g's weight at b + g * b_group_elems, viewed as [N, K] (b_kmajor) or as
//     [K, N] (MN-major, i.e. the transpose is stored)
struct GemmMArgs {
    int G;                 // groups
    GroupRows rows;
    const void* a;
    const void* b;
    int64_t b_group_elems;
    bool b_kmajor;
    int N, K;
    int b_rows;  // MN-major B: rows of one group's [K, N] view when they are fewer than K
                 // (the rows past them multiply zero columns of A); 0 means K
    const int32_t* group_expert;  // device [G]: the weights of group g are group_expert[g]'s
                                  // (owner-grouped layout); null: group g's
    int epi;
    // EPI_SWIGLU_FWD: out0 = h_gu [rows, 2F] (G at cols [0,F), U at [F,2F)),
    //                 out1 = act [rows, F]; N = 2F (B holds gate rows then up rows).
    // EPI_STORE:      out0 = [rows, N].
    // EPI_SWIGLU_BWD: aux = h_gu [rows, 2F] (input), out0 = dh [rows, 2F]; N = F.
    void* out0;
    void* out1;
    const void* aux;
    // EPI_STORE with MN-major B and N % 128 == 0: two CTAs per SM with 128-wide tiles, for
    // a short contraction whose time is the epilogue's stores (the router's dx_router)
    bool slim;
};

// C_g[M, N] = sum over the rows r of group g of A[r, m] * B[r, n]  (K varies per group)
//  A: [rows, M] row-major; B: [rows, N] row-major; C: out + g*M*N, [M, N] row-major.
struct GemmKArgs {
    int G;
    GroupRows rows;
    const void* a;
    const void* b;
    int M, N;
    void* out;
    // EPI_STORE: out = dtype C as above. EPI_DWR (bf16 only, N = 64): out = fp32 partials
    // stored transposed, out + (g*E + e)*M + m = C_g[m, e] for e < E.
    int epi = EPI_STORE;
    int E = 0;
    const int32_t* group_expert = nullptr;  // device [G]: group g's output is group_expert[g]'s
};

cudaError_t launch_gemm_m(const GemmMArgs& g, bool bf16, cudaStream_t s);
cudaError_t launch_gemm_k(const GemmKArgs& g, bool bf16, cudaStream_t s);
// bf16: an M-variable GEMM (MN-major B) and a K-variable GEMM over the same groups in
// one persistent launch (the second problem's tiles after the first's)
cudaError_t launch_gemm_mk(const GemmMArgs& m, const GemmKArgs& k, cudaStream_t s);
// whether launch_gemm_m runs this GEMM as CTA-pair tiles (bf16)
bool gemm_m_uses_pairs(const GemmMArgs& g);
bool gemm_k_uses_pairs(const GemmKArgs& g);
void set_wait_limit_ns(uint64_t ns);
void set_gemm_pairs(int mode);  // MOE_PAIRS_*
cudaError_t gemm_status(cudaStream_t s, int* code);
cudaError_t simt_status(cudaStream_t s, int* code);

// fp32 SIMT versions (the fp32 configuration); same argument meaning.
cudaError_t launch_gemm_m_simt(const GemmMArgs& g, cudaStream_t s);
cudaError_t launch_gemm_k_simt(const GemmKArgs& g, cudaStream_t s);

// training step around the layer (train.cu)
cudaError_t launch_sgd_update(void* w, const void* dw, float* master, int64_t n_groups, int64_t group_elems,
                              const int32_t* counts, float lr, bool bf16, cudaStream_t s);
size_t mse_workspace_bytes();
cudaError_t launch_mse_loss(const void* out, const void* y, int64_t T, int d, bool bf16, float* loss,
                            void* dout, void* workspace, cudaStream_t s);

}  // namespace moe
