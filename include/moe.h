/*
 * moe.h — C ABI of the GB300 (sm_103a) sparse MoE expert layer, forward and backward.
 *
 * The layer is the one every party's hidden states pass through in PC-MoE
 * (arXiv 2506.02965): the gating function of Alg. 7 (softmax over the router
 * logits, top-k picks, gate weights w = p[I]), the ProcessExperts step of Alg. 3
 * (each token's hidden state goes to every expert it picked; the expert outputs
 * are summed with the gate weights), the expert passes of Alg. 6, and
 * BackwardExperts of Alg. 5 together with the gradient contract of Sec. 3.2: an
 * expert host receives the gradient w.r.t. its output and returns one
 * activation-sized gradient w.r.t. its input.
 *
 * Conventions shared by every entry point
 *  - Pointers named x, w_*, logits, ... are DEVICE pointers unless the comment says
 *    HOST. The caller allocates and owns every buffer; the library never frees or
 *    keeps a pointer after the call returns. Tensors are dense and row-major.
 *  - "dtype" buffers hold cfg->dtype elements (float32 for MOE_F32, bfloat16 for
 *    MOE_BF16). Router logits, probabilities, gate weights and their gradients are
 *    always float32; counts and index tables are int32.
 *  - Shapes use T tokens, d = d_model, E experts, F = d_ff, k = top_k, P parties,
 *    S shared experts with Fs = d_ff_shared, TK = T*k.
 *  - Every call is asynchronous on `stream` (NULL = legacy default stream). Bad
 *    arguments are reported synchronously as MOE_ERR_INVALID_ARG (no work queued;
 *    moe_last_error() gives the reason). Errors found by a kernel (an index out of
 *    range, a bounded wait that ran out) are recorded in a device status word and
 *    returned by moe_device_status().
 *  - bf16 paths need d % 128 == 0, F % 128 == 0, Fs % 128 == 0 and 16-byte aligned
 *    dtype buffers; fp32 paths need d % 4 == 0.
 *  - Party layout (Sec. 3.1): tokens are party-contiguous; party p owns tokens
 *    [party_offsets[p], party_offsets[p+1]) and routes them with its own router
 *    W_r[p] over the GLOBAL pool of E experts. party_offsets is a device int32
 *    array of P+1 entries, party_offsets[0] = 0, party_offsets[P] = T; it may be
 *    NULL when P == 1.
 *  - Nothing here allocates device memory. Scratch comes from the caller's
 *    workspace, sized by moe_workspace_size().
 */
#ifndef MOE_H
#define MOE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* moe_stream_t; /* same handle as cudaStream_t */

typedef enum {
    MOE_OK = 0,
    MOE_ERR_INVALID_ARG = 1,  /* bad argument, found on the host before any launch */
    MOE_ERR_CUDA = 2,         /* a CUDA runtime/driver call failed */
    MOE_ERR_DEVICE_CHECK = 3, /* a kernel found an index or size out of range */
    MOE_ERR_TIMEOUT = 4,      /* a bounded wait inside a kernel ran out */
    MOE_ERR_UNSUPPORTED = 5   /* valid request this build does not implement */
} moe_status;

typedef enum { MOE_F32 = 0, MOE_BF16 = 1 } moe_dtype;

/* Layer configuration (HOST struct, 48 bytes). */
typedef struct {
    int64_t T;              /* tokens in the batch (all parties) */
    int32_t d_model;        /* hidden size d */
    int32_t n_experts;      /* E, global expert pool, 1..256 (MOE_ERR_UNSUPPORTED above) */
    int32_t d_ff;           /* F, SwiGLU inner size of each routed expert */
    int32_t top_k;          /* k, 1..8, k <= E */
    int32_t n_parties;      /* P >= 1 */
    int32_t n_shared;       /* S >= 0 always-on shared experts */
    int32_t d_ff_shared;    /* Fs, inner size of each shared expert (0 if S == 0) */
    int32_t normalize_topk; /* 0: w = p[I] exactly as Alg. 7; 1: w renormalised over the k picks */
    float aux_alpha;        /* alpha of the load-balancing loss */
    int32_t dtype;          /* moe_dtype */
} moe_config;

/* Bytes of device workspace the calls that take `workspace` need for this config. */
moe_status moe_workspace_size(const moe_config* cfg, size_t* bytes /* HOST out */);

/*
 * Gating, Alg. 7: z_t = W_r[p(t)] x_t (+ b[p(t)]), p_t = Softmax(z_t),
 * I_t = the k largest logits in descending order (equal logits: lower expert id
 * first), w_tj = p_t[I_tj] (renormalised over the picks if cfg->normalize_topk).
 *   x        [T,d] dtype            w_router [P,E,d] dtype
 *   router_bias [P,E] f32 or NULL   party_offsets [P+1] i32 or NULL (P == 1)
 *   logits, probs [T,E] f32 out     topk_idx [T,k] i32 out    topk_w [T,k] f32 out
 *   counts [P,E] i32 out: how many (token, pick) pairs of party p went to expert e.
 * Logits are accumulated in fp32; the picks are decided on those fp32 logits.
 */
moe_status moe_route(const moe_config* cfg, const void* x, const void* w_router,
                     const float* router_bias, const int32_t* party_offsets,
                     float* logits, float* probs, int32_t* topk_idx, float* topk_w,
                     int32_t* counts, moe_stream_t stream);

/* The softmax / top-k / count part of moe_route on caller-supplied fp32 logits [T,E]
 * (Alg. 7). With identical logits the picks and counts are exact integers. */
moe_status moe_route_from_logits(const moe_config* cfg, const float* logits,
                                 const int32_t* party_offsets, float* probs,
                                 int32_t* topk_idx, float* topk_w, int32_t* counts,
                                 moe_stream_t stream);

/*
 * Load-balancing loss per party (the paper has none; this is the Switch-Transformer
 * form it cites in Sec. 1): L_p = alpha * E * sum_e f_pe * P_pe with
 * f_pe = counts[p,e] / (T_p k) (no gradient) and P_pe = mean over the party's tokens
 * of probs[t,e].
 *   probs [T,E] f32, counts [P,E] i32 (from moe_route)
 *   loss [P] f32 out; aux_coef [P,E] f32 out = dL_p/dprobs[t,e] for t in party p.
 */
moe_status moe_aux_loss(const moe_config* cfg, const float* probs, const int32_t* counts,
                        const int32_t* party_offsets, float* loss, float* aux_coef,
                        moe_stream_t stream);

/*
 * Token dispatch, the "send h to the host of idx" step of Alg. 3 laid out as one
 * expert-major buffer:
 *   offsets [E+1] i32 out: offsets[e] = number of picks of experts < e, offsets[E] = TK
 *   slot_of [T*k] i32 out: row of x_perm holding pick j of token t (index t*k + j):
 *                          offsets[e] + #{t' < t : token t' picked e}  (stable)
 *   token_of [T*k] i32 out: token_of[slot_of[t*k+j]] = t
 *   x_perm [T*k,d] dtype out: x_perm[r] = x[token_of[r]]
 *   workspace: device scratch of at least moe_workspace_size() bytes.
 * Returns MOE_ERR_DEVICE_CHECK (via moe_device_status) if an index is outside [0,E).
 */
moe_status moe_dispatch(const moe_config* cfg, const int32_t* topk_idx, const void* x,
                        int32_t* offsets, int32_t* slot_of, int32_t* token_of, void* x_perm,
                        void* workspace, size_t workspace_bytes, moe_stream_t stream);

/*
 * Owner-grouped dispatch: the layout of the cross-party sends of Alg. 3 ("send h to the
 * host of idx") when expert e is hosted by party owner(e) = e mod P (round-robin,
 * Sec. 3.1). As moe_dispatch, but the expert segments of x_perm are ordered by
 * (owner, expert): every party's received rows are contiguous, and inside a segment the
 * rows follow the token order (tokens are party-contiguous, so each source party's rows
 * are contiguous and in party order).
 *   group_expert [E] i32 out: the expert of segment g ((e mod P, e) order)
 *   offsets [E+1] i32 out:    segment g holds rows [offsets[g], offsets[g+1])
 *   slot_of, token_of, x_perm: as moe_dispatch, in this layout
 *   send_counts [P,P] i32 out: (token, pick) pairs of source party s received by owner o
 * The expert FFN calls take group_expert to find each segment's weights. P = 1 gives
 * the expert-major layout of moe_dispatch. workspace: at least moe_workspace_size()
 * bytes (also when T == 0). Returns MOE_ERR_DEVICE_CHECK (via moe_device_status) if an
 * index is outside [0,E).
 */
moe_status moe_dispatch_owner(const moe_config* cfg, const int32_t* topk_idx, const void* x,
                              const int32_t* party_offsets, int32_t* group_expert,
                              int32_t* offsets, int32_t* slot_of, int32_t* token_of, void* x_perm,
                              int32_t* send_counts, void* workspace, size_t workspace_bytes,
                              moe_stream_t stream);

/*
 * moe_dispatch without a workspace argument, for callers that cannot allocate device
 * memory: code whose host framework hands it only input and output buffers (an op or
 * plugin interface with no scratch), or that must not allocate while it runs (a
 * fixed device-memory budget). The paper has no counterpart; this is a library
 * convenience. Same arguments and results as moe_dispatch.
 *  - Scratch: a fixed device array inside the library of 65536 int32 entries
 *    (256 KiB), held by every GPU that loads the library until the process exits.
 *    It bounds the size: ceil(T/128) * E <= 65536 (e.g. T <= 131072 with E = 64);
 *    larger requests return MOE_ERR_INVALID_ARG and queue no work.
 *  - Calls no cudaMalloc or cudaFree. The first call on a device looks up the
 *    array's device address once (cudaGetSymbolAddress) and keeps it for the process;
 *    make that first call before any stream capture. The kept address belongs to the
 *    device's context at that time: after cudaDeviceReset on that device, do not call
 *    moe_dispatch_noalloc there again in this process.
 *  - Every call shares the one array. Each call overwrites the entries it uses, so
 *    back-to-back calls on one stream are fine; calls whose kernels overlap on the GPU
 *    (several streams or host threads at once) race and give wrong tables.
 */
moe_status moe_dispatch_noalloc(const moe_config* cfg, const int32_t* topk_idx, const void* x,
                                int32_t* offsets, int32_t* slot_of, int32_t* token_of,
                                void* x_perm, moe_stream_t stream);

/*
 * Row gather: dst[i] = src[rows[i]] for i < n_rows, rows of row_elems elements of dtype.
 * The reordering between the blocks an expert host receives from the parties
 * (source-major, Alg. 3 "send h to the host of idx") and the expert-major order its
 * grouped GEMMs take, and back (Sec. 3.2: the gradient returned to each data owner).
 *   src [n_src_rows, row_elems], dst [n_rows, row_elems]: device, 16-byte aligned,
 *   row_elems * element size a multiple of 16 bytes; rows [n_rows] i32 device.
 * A row index outside [0, n_src_rows) leaves that dst row untouched and is recorded as
 * MOE_ERR_DEVICE_CHECK (moe_device_status). Bad sizes: MOE_ERR_INVALID_ARG.
 */
moe_status moe_gather_rows(const void* src, const int32_t* rows, int64_t n_rows, int64_t n_src_rows,
                           int64_t row_elems, moe_dtype dtype, void* dst, moe_stream_t stream);

/*
 * ForwardExpert of Alg. 6 for every routed expert, on its rows of x_perm, plus the
 * always-on shared experts on every token. Expert e is SwiGLU:
 *   [G|U] = x_perm_e W1[e]^T, A = silu(G) * U, Y = A W2[e]^T
 *   x_perm [TK,d]; offsets [E+1] (from moe_dispatch); w1 [E,2F,d] (gate rows, then
 *   up rows); w2 [E,d,F]; h_gu [TK,2F] out (G then U, kept for the backward);
 *   act [TK,F] out; y_perm [TK,d] out.
 * Shared experts (all NULL when S == 0): x [T,d]; ws1 [S,2Fs,d]; ws2 [S,d,Fs];
 *   h_gu_sh [S,T,2Fs] out; act_sh [S,T,Fs] out; y_sh [S,T,d] out.
 * bf16: tcgen05 tensor-core GEMMs, fp32 accumulation in TMEM, bf16 outputs.
 * group_expert [E] i32 (from moe_dispatch_owner) or NULL: segment g of x_perm (rows
 *   [offsets[g], offsets[g+1])) belongs to expert group_expert[g] (NULL: to expert g).
 */
moe_status moe_expert_ffn_fwd(const moe_config* cfg, const void* x_perm, const int32_t* offsets,
                              const void* w1, const void* w2, void* h_gu, void* act,
                              void* y_perm, const void* x, const void* ws1, const void* ws2,
                              void* h_gu_sh, void* act_sh, void* y_sh,
                              const int32_t* group_expert, moe_stream_t stream);

/* Number of CUDA kernels one moe_expert_ffn_bwd call with this configuration launches
 * (host only, no device work): per weight, the input-gradient GEMM and the weight
 * gradient in one persistent launch, or in two (CTA-pair tiles, moe_set_gemm_pairs,
 * and the fp32 path), plus four for the shared experts; 0 GEMMs when T*k == 0. */
moe_status moe_expert_ffn_bwd_kernels(const moe_config* cfg, int32_t* count /* HOST out */);

/*
 * The weighted sum of Alg. 3: out_t = sum_j topk_w[t,j] * y_perm[slot_of[t*k+j]]
 * (+ sum_s y_sh[s,t] when S > 0, shared experts enter with weight 1).
 *   out [T,d] dtype out (fp32 accumulation).
 */
moe_status moe_combine_fwd(const moe_config* cfg, const void* y_perm, const float* topk_w,
                           const int32_t* slot_of, const void* y_sh, void* out,
                           moe_stream_t stream);

/*
 * Backward of the weighted sum (Alg. 5 with the chain rule completed):
 *   dy_perm[slot_of[t*k+j]] = topk_w[t,j] * dout[t]   (the gradient sent to the host)
 *   dtopk_w[t,j] = <dout[t], y_perm[slot_of[t*k+j]]>   (fp32)
 *   dout [T,d]; dy_perm [TK,d] out; dtopk_w [T,k] f32 out.
 */
moe_status moe_combine_bwd(const moe_config* cfg, const void* dout, const void* y_perm,
                           const float* topk_w, const int32_t* slot_of, void* dy_perm,
                           float* dtopk_w, moe_stream_t stream);

/*
 * BackwardExpert of Alg. 6 for every routed expert (and the shared experts):
 *   dA = dY W2;  dU = dA*silu(G);  dG = dA*U*s*(1+G*(1-s)), s = sigmoid(G)
 *   dh [TK,2F] out = [dG|dU];  dx_perm [TK,d] out = dh W1 (the gradient w.r.t. the
 *   expert input returned to the data owner, Sec. 3.2);
 *   dw1 [E,2F,d] out = dh^T x_perm;  dw2 [E,d,F] out = dY^T act  (dtype).
 * Inputs: x_perm, offsets, w1, w2, h_gu, act (from the forward), dy_perm (from
 * moe_combine_bwd). Experts with no rows get zero weight gradients.
 * Shared experts (NULL when S == 0): x [T,d], dout [T,d] (their dY), ws1, ws2,
 *   h_gu_sh, act_sh (forward), dh_sh [S,T,2Fs] out, dx_sh [S,T,d] out,
 *   dws1 [S,2Fs,d] out, dws2 [S,d,Fs] out.
 * group_expert: as in moe_expert_ffn_fwd (dw1[e], dw2[e] are always expert e's).
 * Several host threads may call this at once: a weight gradient that runs on the
 * library's second stream of the device (CTA-pair tiles, or fp32) is forked from and
 * joined back to the caller's stream under a lock, so each call waits on its own
 * stream's work only (calls on different streams then share that second stream).
 */
moe_status moe_expert_ffn_bwd(const moe_config* cfg, const void* x_perm, const int32_t* offsets,
                              const void* w1, const void* w2, const void* h_gu, const void* act,
                              const void* dy_perm, void* dh, void* dx_perm, void* dw1, void* dw2,
                              const void* x, const void* dout, const void* ws1, const void* ws2,
                              const void* h_gu_sh, const void* act_sh, void* dh_sh, void* dx_sh,
                              void* dws1, void* dws2, const int32_t* group_expert,
                              moe_stream_t stream);

/*
 * Backward of the gating function (the router is part of the party's local
 * layers L_i, Sec. 3.1; the picks are constants):
 *   dp[t,e] = sum_j [topk_idx[t,j] == e] * g_tj + aux_coef[p(t),e]
 *     with g_tj = dtopk_w[t,j] (paper), or (dtopk_w[t,j] - <dtopk_w[t], topk_w[t]>) /
 *     sum_j probs[t, topk_idx[t,j]] when normalize_topk;
 *   dlogits[t,e] = probs[t,e] * (dp[t,e] - <dp[t], probs[t]>)   [T,E] f32 out
 *   dw_router[p] = sum_{t in p} dlogits[t]^T x[t]                [P,E,d] dtype out
 *   dbias[p]     = sum_{t in p} dlogits[t]                       [P,E] f32 out or NULL
 *   dx_router[t] = dlogits[t] W_r[p(t)]  (the router's share of the input gradient)
 *                                                               [T,d] dtype out or NULL
 * aux_coef may be NULL (no aux term). bf16: the two products run on the tensor cores
 * with dlogits rounded to bf16 as their operand (fp32 accumulation); fp32: CUDA cores.
 * Deterministic: partial sums go to the workspace and are reduced in a fixed order.
 */
moe_status moe_route_bwd(const moe_config* cfg, const void* x, const void* w_router,
                         const float* probs, const int32_t* topk_idx, const float* topk_w,
                         const float* dtopk_w, const float* aux_coef,
                         const int32_t* party_offsets, float* dlogits, void* dw_router,
                         float* dbias, void* dx_router, void* workspace,
                         size_t workspace_bytes, moe_stream_t stream);

/*
 * Input gradient of the layer: the returned expert-input gradients summed per token
 * (Sec. 3.2), plus the router's share (dx_router from moe_route_bwd) and the shared
 * experts' share:
 *   dx[t] = sum_j dx_perm[slot_of[t*k+j]] + dx_router[t] + sum_s dx_sh[s,t]
 *   dx [T,d] dtype out (overwritten; fp32 accumulation). dx_router NULL: no router
 *   term. dx_sh NULL when S == 0. A slot outside [0, T*k) is skipped and recorded as
 *   MOE_ERR_DEVICE_CHECK (moe_device_status).
 */
moe_status moe_dispatch_bwd(const moe_config* cfg, const void* dx_perm, const int32_t* slot_of,
                            const void* dx_router, const void* dx_sh, void* dx,
                            moe_stream_t stream);

/*
 * Training step of Alg. 1 around the layer (toy block: the layer output is the block
 * output). The loss of the batch, Loss(h, y) of Alg. 1, read as mean-squared error:
 *   loss[0] = sum_t ||out_t - target_t||^2 / (2T)          (fp32, device out)
 *   dout    = (out - target) / T                            [T,d] dtype out
 * out, target [T,d] dtype (cfg->dtype). fp32 arithmetic; the reduction runs in a fixed
 * order (the same bits on every call). workspace: device scratch of at least
 * moe_workspace_size(cfg) bytes (only its first 2 KB are used here).
 * Errors: MOE_ERR_INVALID_ARG for NULL pointers or a short workspace. T == 0 writes 0.
 */
moe_status moe_mse_loss(const moe_config* cfg, const void* out, const void* target, float* loss,
                        void* dout, void* workspace, size_t workspace_bytes, moe_stream_t stream);

/*
 * One SGD step on a parameter stored as n_groups groups of group_elems elements (an
 * expert stack [E, ...] or one party's router slice): the updates of Alg. 1, where
 * only the active party's gating (BackwardLocal, Alg. 4) and the experts its batch
 * called (BackwardExpert, Alg. 6) change and nothing is broadcast. For every group g
 * with group_counts[g] > 0 (every group when group_counts is NULL):
 *   w_master == NULL:  w[g] <- w[g] - lr * dw[g]
 *   w_master != NULL:  w_master[g] <- w_master[g] - lr * dw[g];  w[g] <- w_master[g]
 * w, dw [n_groups * group_elems] of dtype, device memory, updated in place; w_master
 * (optional) fp32 [n_groups * group_elems] device memory, the master copy of w for
 * bf16 training (updates below the bf16 spacing accumulate there); group_counts
 * [n_groups] int32 device memory or NULL (e.g. the per-expert counts moe_route wrote
 * for a one-party batch). fp32 arithmetic (one fused multiply-add), rounded to dtype.
 * A group that is not called is neither read nor written.
 * Errors: MOE_ERR_INVALID_ARG for negative sizes, more than 65535 groups, an unknown
 * dtype, a non-finite lr or NULL w / dw with work to do.
 */
moe_status moe_sgd_update(void* w, const void* dw, float* w_master, int64_t n_groups, int64_t group_elems,
                          const int32_t* group_counts, float lr, moe_dtype dtype, moe_stream_t stream);

/* Synchronises `stream`, returns the first error code any kernel recorded since the
 * last call (MOE_OK if none) in *code and clears it. */
moe_status moe_device_status(moe_stream_t stream, int32_t* code /* HOST out */);

/* Upper bound, in nanoseconds, of every bounded wait inside the tensor-core kernels
 * (default 2e9). A wait that runs out records MOE_ERR_TIMEOUT and the kernel returns. */
moe_status moe_set_wait_limit_ns(uint64_t ns);

/* Tile shape of the 256-wide expert GEMMs (forward, dA, dX and the weight gradients),
 * for all later calls of this process. A CTA-pair tile is 256 x 256, computed by
 * two CTAs on two SMs with tcgen05 cta_group::2 MMAs, each SM holding half of the B
 * operand (half the operand traffic per SM of a single-CTA 128 x 256 tile), but twice
 * as few tiles share the SMs, so a launch with few tiles loses to its last round.
 *   MOE_PAIRS_OFF  (0): single-CTA tiles everywhere;
 *   MOE_PAIRS_ALL  (1): pair tiles for every such GEMM;
 *   MOE_PAIRS_AUTO (2, default): pair tiles for the input-gradient GEMM dX = dH W1
 *                   (contraction 2F) and wherever a launch has at least four rounds
 *                   of them, except under the SwiGLU backward epilogue when d < 2048
 *                   (there the epilogue, not the operand feed, bounds the dA GEMM).
 * The weight-gradient GEMMs launched on their own (dW1; dW2 when dA runs as pairs; the
 * shared experts') follow the same mode with 256 x 256 output tiles where both output
 * dimensions are multiples of 256.
 * Results agree up to fp32 summation order. Any other mode: MOE_ERR_INVALID_ARG. */
enum { MOE_PAIRS_OFF = 0, MOE_PAIRS_ALL = 1, MOE_PAIRS_AUTO = 2 };
moe_status moe_set_gemm_pairs(int mode);

const char* moe_status_string(moe_status s);
/* Reason for the last MOE_ERR_INVALID_ARG / MOE_ERR_CUDA returned on this thread. */
const char* moe_last_error(void);
/* Library version string. */
const char* moe_version(void);

#ifdef __cplusplus
}
#endif
#endif /* MOE_H */
