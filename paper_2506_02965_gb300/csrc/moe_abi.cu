// C ABI of the MoE expert layer (declared in include/moe.h): argument checks,
// launches, status handling. No device allocation happens here.
#include <algorithm>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <string>

#include "../../include/moe.h"
#include "moe_internal.h"

using namespace moe;

namespace {

thread_local std::string g_last_error;

moe_status fail(moe_status s, const char* fmt, ...) __attribute__((format(printf, 2, 3)));
moe_status fail(moe_status s, const char* fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof(buf), fmt, ap);
    va_end(ap);
    g_last_error = buf;
    return s;
}

moe_status cuda_status(cudaError_t e, const char* where) {
    if (e == cudaSuccess) return MOE_OK;
    return fail(MOE_ERR_CUDA, "%s: %s", where, cudaGetErrorString(e));
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Validate the configuration; fills the commonly used derived values.
moe_status check_cfg(const moe_config* c) {
    if (!c) return fail(MOE_ERR_INVALID_ARG, "cfg is NULL");
    if (c->dtype != MOE_F32 && c->dtype != MOE_BF16)
        return fail(MOE_ERR_INVALID_ARG, "dtype %d is not MOE_F32 or MOE_BF16", c->dtype);
    if (c->T < 0) return fail(MOE_ERR_INVALID_ARG, "T=%lld < 0", (long long)c->T);
    if (c->d_model <= 0 || c->d_ff <= 0)
        return fail(MOE_ERR_INVALID_ARG, "d_model=%d and d_ff=%d must be > 0", c->d_model, c->d_ff);
    if (c->n_experts < 1)
        return fail(MOE_ERR_INVALID_ARG, "n_experts=%d < 1", c->n_experts);
    if (c->n_experts > 256)
        return fail(MOE_ERR_UNSUPPORTED, "n_experts=%d > 256, the largest expert pool this build handles",
                    c->n_experts);
    if (c->top_k < 1 || c->top_k > 8 || c->top_k > c->n_experts)
        return fail(MOE_ERR_INVALID_ARG, "top_k=%d outside [1, min(8, E)]", c->top_k);
    if (c->n_parties < 1 || c->n_parties > 64)
        return fail(MOE_ERR_INVALID_ARG, "n_parties=%d outside [1,64]", c->n_parties);
    if (c->n_shared < 0 || c->n_shared > 8)
        return fail(MOE_ERR_INVALID_ARG, "n_shared=%d outside [0,8]", c->n_shared);
    if (c->n_shared > 0 && c->d_ff_shared <= 0)
        return fail(MOE_ERR_INVALID_ARG, "d_ff_shared must be > 0 with shared experts");
    if (c->normalize_topk != 0 && c->normalize_topk != 1)
        return fail(MOE_ERR_INVALID_ARG, "normalize_topk must be 0 or 1");
    const int64_t TK = c->T * c->top_k;
    if (TK >= (int64_t)1 << 31) return fail(MOE_ERR_INVALID_ARG, "T*k must be < 2^31");
    if (c->dtype == MOE_BF16) {
        if (c->d_model % 128 || c->d_ff % 128 || (c->n_shared && c->d_ff_shared % 128))
            return fail(MOE_ERR_INVALID_ARG,
                        "bf16 needs d_model, d_ff, d_ff_shared multiples of 128 (got %d, %d, %d)",
                        c->d_model, c->d_ff, c->d_ff_shared);
    } else {
        if (c->d_model % 4) return fail(MOE_ERR_INVALID_ARG, "fp32 needs d_model %% 4 == 0");
    }
    return MOE_OK;
}

#define REQUIRE(ptr)                                                                  \
    do {                                                                              \
        if (!(ptr)) return fail(MOE_ERR_INVALID_ARG, "%s is NULL", #ptr);             \
    } while (0)
#define REQUIRE_VEC(ptr)                                                              \
    do {                                                                              \
        if (!(ptr)) return fail(MOE_ERR_INVALID_ARG, "%s is NULL", #ptr);             \
        if (!aligned16(ptr))                                                          \
            return fail(MOE_ERR_INVALID_ARG, "%s is not 16-byte aligned", #ptr);      \
    } while (0)

moe_status check_parties(const moe_config* c, const int32_t* po) {
    if (c->n_parties > 1 && !po)
        return fail(MOE_ERR_INVALID_ARG, "party_offsets is NULL with n_parties=%d", c->n_parties);
    return MOE_OK;
}

size_t elem_size(const moe_config* c) { return c->dtype == MOE_BF16 ? 2 : 4; }

// A second stream per device on which the backward runs the weight-gradient GEMMs
// while the input-gradient GEMMs run on the caller's stream, so that the tail wave of
// one persistent kernel is filled by the other. Fork and join are event waits, so all
// work stays ordered with respect to the caller's stream. Created on the first call
// on a device (that call must not be inside a stream capture). The events are shared
// by every call on the device, so a call holds g_side_mu (side_stream's caller passes
// its lock) from the fork record until its join wait is queued: two host threads
// cannot re-record each other's events in between.
struct SideStream {
    cudaStream_t s = nullptr;
    cudaEvent_t fork = nullptr, mid = nullptr, join = nullptr;
};
constexpr int kMaxDev = 64;
SideStream g_side[kMaxDev];
std::mutex g_side_mu;

// Requires g_side_mu held by the caller.
cudaError_t side_stream(SideStream** out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDev) return cudaErrorInvalidDevice;
    SideStream& ss = g_side[dev];
    if (!ss.s) {
        if ((e = cudaStreamCreateWithFlags(&ss.s, cudaStreamNonBlocking)) != cudaSuccess) return e;
        if ((e = cudaEventCreateWithFlags(&ss.fork, cudaEventDisableTiming)) != cudaSuccess) return e;
        if ((e = cudaEventCreateWithFlags(&ss.mid, cudaEventDisableTiming)) != cudaSuccess) return e;
        if ((e = cudaEventCreateWithFlags(&ss.join, cudaEventDisableTiming)) != cudaSuccess) return e;
    }
    *out = &ss;
    return cudaSuccess;
}

}  // namespace

extern "C" {

const char* moe_version(void) { return "pcmoe-gb300 0.1 (sm_103a)"; }

const char* moe_last_error(void) { return g_last_error.c_str(); }

const char* moe_status_string(moe_status s) {
    switch (s) {
        case MOE_OK: return "MOE_OK";
        case MOE_ERR_INVALID_ARG: return "MOE_ERR_INVALID_ARG";
        case MOE_ERR_CUDA: return "MOE_ERR_CUDA";
        case MOE_ERR_DEVICE_CHECK: return "MOE_ERR_DEVICE_CHECK";
        case MOE_ERR_TIMEOUT: return "MOE_ERR_TIMEOUT";
        case MOE_ERR_UNSUPPORTED: return "MOE_ERR_UNSUPPORTED";
    }
    return "MOE_ERR_UNKNOWN";
}

moe_status moe_set_wait_limit_ns(uint64_t ns) {
    if (ns == 0) return fail(MOE_ERR_INVALID_ARG, "wait limit must be > 0");
    set_wait_limit_ns(ns);
    return MOE_OK;
}

moe_status moe_set_gemm_pairs(int mode) {
    if (mode != MOE_PAIRS_OFF && mode != MOE_PAIRS_ALL && mode != MOE_PAIRS_AUTO)
        return fail(MOE_ERR_INVALID_ARG, "pair mode must be MOE_PAIRS_OFF, _ALL or _AUTO");
    set_gemm_pairs(mode);
    return MOE_OK;
}

moe_status moe_workspace_size(const moe_config* cfg, size_t* bytes) {
    moe_status st = check_cfg(cfg);
    if (st) return st;
    REQUIRE(bytes);
    *bytes = std::max(std::max(dispatch_workspace(cfg->T, cfg->n_experts),
                               route_bwd_workspace(cfg->T, cfg->n_parties, cfg->n_experts, cfg->d_model)),
                      mse_workspace_bytes());
    return MOE_OK;
}

static moe_status route_common(const moe_config* cfg, const void* x, const void* w_router,
                               const float* bias, const float* logits_in, const int32_t* po,
                               float* logits, float* probs, int32_t* topk_idx, float* topk_w,
                               int32_t* counts, moe_stream_t stream) {
    RouteArgs a{};
    a.x = x;
    a.w_router = w_router;
    a.bias = bias;
    a.logits_in = logits_in;
    a.po = po;
    a.P = cfg->n_parties;
    a.T = cfg->T;
    a.d = cfg->d_model;
    a.E = cfg->n_experts;
    a.k = cfg->top_k;
    a.normalize = cfg->normalize_topk;
    a.logits = logits;
    a.probs = probs;
    a.topk_idx = topk_idx;
    a.topk_w = topk_w;
    a.counts = counts;
    return cuda_status(launch_route(a, cfg->dtype == MOE_BF16, logits_in != nullptr,
                                    (cudaStream_t)stream),
                       "moe_route");
}

moe_status moe_route(const moe_config* cfg, const void* x, const void* w_router,
                     const float* router_bias, const int32_t* party_offsets, float* logits,
                     float* probs, int32_t* topk_idx, float* topk_w, int32_t* counts,
                     moe_stream_t stream) {
    moe_status st = check_cfg(cfg);
    if (st) return st;
    if ((st = check_parties(cfg, party_offsets))) return st;
    REQUIRE(counts);
    if (cfg->T == 0)
        return cuda_status(cudaMemsetAsync(counts, 0, sizeof(int32_t) * cfg->n_parties * cfg->n_experts,
                                           (cudaStream_t)stream), "moe_route");
    REQUIRE_VEC(x);
    REQUIRE_VEC(w_router);
    REQUIRE(logits);
    REQUIRE(probs);
    REQUIRE(topk_idx);
    REQUIRE(topk_w);
    REQUIRE(counts);
    return route_common(cfg, x, w_router, router_bias, nullptr, party_offsets, logits, probs,
                        topk_idx, topk_w, counts, stream);
}

moe_status moe_route_from_logits(const moe_config* cfg, const float* logits,
                                 const int32_t* party_offsets, float* probs, int32_t* topk_idx,
                                 float* topk_w, int32_t* counts, moe_stream_t stream) {
    moe_status st = check_cfg(cfg);
    if (st) return st;
    if ((st = check_parties(cfg, party_offsets))) return st;
    REQUIRE(counts);
    if (cfg->T == 0)
        return cuda_status(cudaMemsetAsync(counts, 0, sizeof(int32_t) * cfg->n_parties * cfg->n_experts,
                                           (cudaStream_t)stream), "moe_route_from_logits");
    REQUIRE(logits);
    REQUIRE(probs);
    REQUIRE(topk_idx);
    REQUIRE(topk_w);
    return route_common(cfg, nullptr, nullptr, nullptr, logits, party_offsets, nullptr, probs,
                        topk_idx, topk_w, counts, stream);
}

moe_status moe_aux_loss(const moe_config* cfg, const float* probs, const int32_t* counts,
                        const int32_t* party_offsets, float* loss, float* aux_coef,
                        moe_stream_t stream) {
    moe_status st = check_cfg(cfg);
    if (st) return st;
    if ((st = check_parties(cfg, party_offsets))) return st;
    if (cfg->T > 0) REQUIRE(probs);
    REQUIRE(counts);
    REQUIRE(loss);
    REQUIRE(aux_coef);
    return cuda_status(launch_aux_loss(probs, counts, party_offsets, cfg->n_parties, cfg->T,
                                       cfg->n_experts, cfg->top_k, cfg->aux_alpha, loss, aux_coef,
                                       (cudaStream_t)stream),
                       "moe_aux_loss");
}

moe_status moe_dispatch(const moe_config* cfg, const int32_t* topk_idx, const void* x,
                        int32_t* offsets, int32_t* slot_of, int32_t* token_of, void* x_perm,
                        void* workspace, size_t workspace_bytes, moe_stream_t stream) {
    moe_status st = check_cfg(cfg);
    if (st) return st;
    REQUIRE(offsets);
    if (cfg->T > 0) {
        REQUIRE(topk_idx);
        REQUIRE_VEC(x);
        REQUIRE(slot_of);
        REQUIRE(token_of);
        REQUIRE_VEC(x_perm);
        REQUIRE(workspace);
        const size_t need = dispatch_workspace(cfg->T, cfg->n_experts);
        if (workspace_bytes < need)
            return fail(MOE_ERR_INVALID_ARG, "workspace of %zu bytes < %zu needed", workspace_bytes,
                        need);
    }
    return cuda_status(launch_dispatch(topk_idx, x, cfg->T, cfg->d_model, cfg->n_experts,
                                       cfg->top_k, cfg->dtype == MOE_BF16, offsets, slot_of,
                                       token_of, x_perm, workspace, (cudaStream_t)stream),
                       "moe_dispatch");
}

moe_status moe_dispatch_owner(const moe_config* cfg, const int32_t* topk_idx, const void* x,
                              const int32_t* party_offsets, int32_t* group_expert,
                              int32_t* offsets, int32_t* slot_of, int32_t* token_of, void* x_perm,
                              int32_t* send_counts, void* workspace, size_t workspace_bytes,
                              moe_stream_t stream) {
    moe_status st = check_cfg(cfg);
    if (st) return st;
    if ((st = check_parties(cfg, party_offsets))) return st;
    REQUIRE(group_expert);
    REQUIRE(offsets);
    REQUIRE(send_counts);
    REQUIRE(workspace);
    const size_t need = dispatch_workspace(std::max<int64_t>(cfg->T, 1), cfg->n_experts);
    if (workspace_bytes < need)
        return fail(MOE_ERR_INVALID_ARG, "workspace of %zu bytes < %zu needed", workspace_bytes, need);
    if (cfg->T > 0) {
        REQUIRE(topk_idx);
        REQUIRE_VEC(x);
        REQUIRE(slot_of);
        REQUIRE(token_of);
        REQUIRE_VEC(x_perm);
    }
    return cuda_status(launch_dispatch(topk_idx, x, cfg->T, cfg->d_model, cfg->n_experts,
                                       cfg->top_k, cfg->dtype == MOE_BF16, offsets, slot_of,
                                       token_of, x_perm, workspace, (cudaStream_t)stream,
                                       cfg->n_parties > 1 ? party_offsets : nullptr,
                                       cfg->n_parties, group_expert, send_counts),
                       "moe_dispatch_owner");
}

moe_status moe_dispatch_noalloc(const moe_config* cfg, const int32_t* topk_idx, const void* x,
                                int32_t* offsets, int32_t* slot_of, int32_t* token_of,
                                void* x_perm, moe_stream_t stream) {
    moe_status st = check_cfg(cfg);
    if (st) return st;
    REQUIRE(offsets);
    const int64_t nch = (cfg->T + kDispatchChunkTokens - 1) / kDispatchChunkTokens;
    if (nch * cfg->n_experts > dispatch_noalloc_max_chunk_entries())
        return fail(MOE_ERR_INVALID_ARG,
                    "moe_dispatch_noalloc: ceil(T/128)*E = %lld exceeds its fixed scratch of %lld "
                    "entries; use moe_dispatch with a workspace",
                    (long long)(nch * cfg->n_experts), (long long)dispatch_noalloc_max_chunk_entries());
    if (cfg->T > 0) {
        REQUIRE(topk_idx);
        REQUIRE_VEC(x);
        REQUIRE(slot_of);
        REQUIRE(token_of);
        REQUIRE_VEC(x_perm);
    }
    return cuda_status(launch_dispatch_noalloc(topk_idx, x, cfg->T, cfg->d_model, cfg->n_experts,
                                               cfg->top_k, cfg->dtype == MOE_BF16, offsets, slot_of,
                                               token_of, x_perm, (cudaStream_t)stream),
                       "moe_dispatch_noalloc");
}

moe_status moe_expert_ffn_fwd(const moe_config* cfg, const void* x_perm, const int32_t* offsets,
                              const void* w1, const void* w2, void* h_gu, void* act, void* y_perm,
                              const void* x, const void* ws1, const void* ws2, void* h_gu_sh,
                              void* act_sh, void* y_sh, const int32_t* group_expert,
                              moe_stream_t stream) {
    moe_status st = check_cfg(cfg);
    if (st) return st;
    const bool bf16 = cfg->dtype == MOE_BF16;
    const int64_t T = cfg->T, TK = T * cfg->top_k;
    const int d = cfg->d_model, F = cfg->d_ff, E = cfg->n_experts, S = cfg->n_shared;
    if (T == 0) return MOE_OK;
    REQUIRE_VEC(x_perm);
    REQUIRE(offsets);
    REQUIRE_VEC(w1);
    REQUIRE_VEC(w2);
    REQUIRE_VEC(h_gu);
    REQUIRE_VEC(act);
    REQUIRE_VEC(y_perm);
    if (S) {
        REQUIRE_VEC(x);
        REQUIRE_VEC(ws1);
        REQUIRE_VEC(ws2);
        REQUIRE_VEC(h_gu_sh);
        REQUIRE_VEC(act_sh);
        REQUIRE_VEC(y_sh);
    }
    cudaStream_t s = (cudaStream_t)stream;
    // routed experts: [G|U] = Xp W1^T with SwiGLU epilogue, then Y = A W2^T
    GemmMArgs g1{};
    g1.group_expert = group_expert;
    g1.G = E;
    g1.rows = GroupRows{offsets, (int)TK, 0, 0, 0};
    g1.a = x_perm;
    g1.b = w1;
    g1.b_group_elems = (int64_t)2 * F * d;
    g1.b_kmajor = true;
    g1.N = 2 * F;
    g1.K = d;
    g1.epi = EPI_SWIGLU_FWD;
    g1.out0 = h_gu;
    g1.out1 = act;
    if ((st = cuda_status(launch_gemm_m(g1, bf16, s), "expert gemm1"))) return st;
    GemmMArgs g2{};
    g2.group_expert = group_expert;
    g2.G = E;
    g2.rows = GroupRows{offsets, (int)TK, 0, 0, 0};
    g2.a = act;
    g2.b = w2;
    g2.b_group_elems = (int64_t)d * F;
    g2.b_kmajor = true;
    g2.N = d;
    g2.K = F;
    g2.epi = EPI_STORE;
    g2.out0 = y_perm;
    if ((st = cuda_status(launch_gemm_m(g2, bf16, s), "expert gemm2"))) return st;
    if (S) {
        const int Fs = cfg->d_ff_shared;
        GemmMArgs h1 = g1;
        h1.group_expert = nullptr;  // shared experts: one group per expert
        h1.G = S;
        h1.rows = GroupRows{nullptr, (int)T, 0, 0, T};
        h1.a = x;
        h1.b = ws1;
        h1.b_group_elems = (int64_t)2 * Fs * d;
        h1.N = 2 * Fs;
        h1.out0 = h_gu_sh;
        h1.out1 = act_sh;
        if ((st = cuda_status(launch_gemm_m(h1, bf16, s), "shared gemm1"))) return st;
        GemmMArgs h2 = g2;
        h2.group_expert = nullptr;  // shared experts: one group per expert
        h2.G = S;
        h2.rows = GroupRows{nullptr, (int)T, T, 0, T};
        h2.a = act_sh;
        h2.b = ws2;
        h2.b_group_elems = (int64_t)d * Fs;
        h2.K = Fs;
        h2.out0 = y_sh;
        if ((st = cuda_status(launch_gemm_m(h2, bf16, s), "shared gemm2"))) return st;
    }
    return MOE_OK;
}

moe_status moe_combine_fwd(const moe_config* cfg, const void* y_perm, const float* topk_w,
                           const int32_t* slot_of, const void* y_sh, void* out,
                           moe_stream_t stream) {
    moe_status st = check_cfg(cfg);
    if (st) return st;
    if (cfg->T == 0) return MOE_OK;
    REQUIRE_VEC(y_perm);
    REQUIRE(topk_w);
    REQUIRE(slot_of);
    REQUIRE_VEC(out);
    if (cfg->n_shared) REQUIRE_VEC(y_sh);
    return cuda_status(launch_combine_fwd(y_perm, topk_w, slot_of, y_sh, cfg->n_shared, cfg->T,
                                          cfg->d_model, cfg->top_k, cfg->dtype == MOE_BF16, out,
                                          (cudaStream_t)stream),
                       "moe_combine_fwd");
}

moe_status moe_combine_bwd(const moe_config* cfg, const void* dout, const void* y_perm,
                           const float* topk_w, const int32_t* slot_of, void* dy_perm,
                           float* dtopk_w, moe_stream_t stream) {
    moe_status st = check_cfg(cfg);
    if (st) return st;
    if (cfg->T == 0) return MOE_OK;
    REQUIRE_VEC(dout);
    REQUIRE_VEC(y_perm);
    REQUIRE(topk_w);
    REQUIRE(slot_of);
    REQUIRE_VEC(dy_perm);
    REQUIRE(dtopk_w);
    return cuda_status(launch_combine_bwd(dout, y_perm, topk_w, slot_of, cfg->T, cfg->d_model,
                                          cfg->top_k, cfg->dtype == MOE_BF16, dy_perm, dtopk_w,
                                          (cudaStream_t)stream),
                       "moe_combine_bwd");
}

moe_status moe_expert_ffn_bwd(const moe_config* cfg, const void* x_perm, const int32_t* offsets,
                              const void* w1, const void* w2, const void* h_gu, const void* act,
                              const void* dy_perm, void* dh, void* dx_perm, void* dw1, void* dw2,
                              const void* x, const void* dout, const void* ws1, const void* ws2,
                              const void* h_gu_sh, const void* act_sh, void* dh_sh, void* dx_sh,
                              void* dws1, void* dws2, const int32_t* group_expert,
                              moe_stream_t stream) {
    moe_status st = check_cfg(cfg);
    if (st) return st;
    const bool bf16 = cfg->dtype == MOE_BF16;
    const int64_t T = cfg->T, TK = T * cfg->top_k;
    const int d = cfg->d_model, F = cfg->d_ff, E = cfg->n_experts, S = cfg->n_shared;
    const int Fs = cfg->d_ff_shared;
    const size_t es = elem_size(cfg);
    REQUIRE_VEC(dw1);
    REQUIRE_VEC(dw2);
    if (S) {
        REQUIRE_VEC(dws1);
        REQUIRE_VEC(dws2);
    }
    cudaStream_t s = (cudaStream_t)stream;
    if (T == 0) {  // no rows: all weight gradients are zero
        if ((st = cuda_status(cudaMemsetAsync(dw1, 0, es * E * 2 * F * d, s), "memset"))) return st;
        if ((st = cuda_status(cudaMemsetAsync(dw2, 0, es * E * d * F, s), "memset"))) return st;
        if (S) {
            if ((st = cuda_status(cudaMemsetAsync(dws1, 0, es * S * 2 * Fs * d, s), "memset"))) return st;
            if ((st = cuda_status(cudaMemsetAsync(dws2, 0, es * S * d * Fs, s), "memset"))) return st;
        }
        return MOE_OK;
    }
    REQUIRE_VEC(x_perm);
    REQUIRE(offsets);
    REQUIRE_VEC(w1);
    REQUIRE_VEC(w2);
    REQUIRE_VEC(h_gu);
    REQUIRE_VEC(act);
    REQUIRE_VEC(dy_perm);
    REQUIRE_VEC(dh);
    REQUIRE_VEC(dx_perm);
    if (S) {
        REQUIRE_VEC(x);
        REQUIRE_VEC(dout);
        REQUIRE_VEC(ws1);
        REQUIRE_VEC(ws2);
        REQUIRE_VEC(h_gu_sh);
        REQUIRE_VEC(act_sh);
        REQUIRE_VEC(dh_sh);
        REQUIRE_VEC(dx_sh);
    }
    // dA = dY W2 with the SwiGLU-backward epilogue -> dH
    GemmMArgs a{};
    a.group_expert = group_expert;
    a.G = E;
    a.rows = GroupRows{offsets, (int)TK, 0, 0, 0};
    a.a = dy_perm;
    a.b = w2;
    a.b_group_elems = (int64_t)d * F;
    a.b_kmajor = false;  // W2[e] is [d, F] = [K, N]
    a.N = F;
    a.K = d;
    a.epi = EPI_SWIGLU_BWD;
    a.aux = h_gu;
    a.out0 = dh;
    // dXp = dH W1
    GemmMArgs b{};
    b.group_expert = group_expert;
    b.G = E;
    b.rows = GroupRows{offsets, (int)TK, 0, 0, 0};
    b.a = dh;
    b.b = w1;
    b.b_group_elems = (int64_t)2 * F * d;
    b.b_kmajor = false;  // W1[e] is [2F, d] = [K, N]
    b.N = d;
    b.K = 2 * F;
    b.epi = EPI_STORE;
    b.out0 = dx_perm;
    // dW2[e] = dY_e^T A_e ; dW1[e] = dH_e^T Xp_e
    GemmKArgs w2g{};
    w2g.group_expert = group_expert;
    w2g.G = E;
    w2g.rows = GroupRows{offsets, (int)TK, 0, 0, 0};
    w2g.a = dy_perm;
    w2g.b = act;
    w2g.M = d;
    w2g.N = F;
    w2g.out = dw2;
    GemmKArgs w1g{};
    w1g.group_expert = group_expert;
    w1g.G = E;
    w1g.rows = GroupRows{offsets, (int)TK, 0, 0, 0};
    w1g.a = dh;
    w1g.b = x_perm;
    w1g.M = 2 * F;
    w1g.N = d;
    w1g.out = dw1;
    // Each M-variable GEMM runs with its weight gradient in one persistent launch (one
    // tail instead of two, and no two persistent grids contending for SMs): dA then dW2
    // (which needs only dY and A), dX then dW1 (which needs dH). A GEMM that runs as
    // CTA-pair tiles, and the CUDA-core path, instead put the weight gradient on a side
    // stream: dW2 alongside dA, dW1 alongside dX once dH exists.
    const bool fuse_a = bf16 && !gemm_m_uses_pairs(a);
    const bool fuse_b = bf16 && !gemm_m_uses_pairs(b);  // the same rule as moe_expert_ffn_bwd_kernels
    SideStream* ss = nullptr;
    std::unique_lock<std::mutex> side_lock(g_side_mu, std::defer_lock);
    if (!fuse_a || !fuse_b) {
        side_lock.lock();  // held until the join wait is queued (the events are shared)
        if ((st = cuda_status(side_stream(&ss), "side stream"))) return st;
        if ((st = cuda_status(cudaEventRecord(ss->fork, s), "fork"))) return st;
        if ((st = cuda_status(cudaStreamWaitEvent(ss->s, ss->fork, 0), "fork"))) return st;
    }
    if (fuse_a) {
        if ((st = cuda_status(launch_gemm_mk(a, w2g, s), "expert dA+dW2 gemm"))) return st;
    } else {
        if ((st = cuda_status(launch_gemm_k(w2g, bf16, ss->s), "expert dW2 gemm"))) return st;
        if ((st = cuda_status(launch_gemm_m(a, bf16, s), "expert dA gemm"))) return st;
    }
    if (fuse_b) {
        if ((st = cuda_status(launch_gemm_mk(b, w1g, s), "expert dX+dW1 gemm"))) return st;
    } else {
        if ((st = cuda_status(cudaEventRecord(ss->mid, s), "mid"))) return st;
        if ((st = cuda_status(launch_gemm_m(b, bf16, s), "expert dX gemm"))) return st;
        if ((st = cuda_status(cudaStreamWaitEvent(ss->s, ss->mid, 0), "mid"))) return st;
        if ((st = cuda_status(launch_gemm_k(w1g, bf16, ss->s), "expert dW1 gemm"))) return st;
    }
    if (ss) {
        if ((st = cuda_status(cudaEventRecord(ss->join, ss->s), "join"))) return st;
        if ((st = cuda_status(cudaStreamWaitEvent(s, ss->join, 0), "join"))) return st;
        side_lock.unlock();
    }
    if (S) {
        GemmMArgs sa = a;
        sa.group_expert = nullptr;  // shared experts: one group per expert
        sa.G = S;
        sa.rows = GroupRows{nullptr, (int)T, 0, 0, T};
        sa.a = dout;
        sa.b = ws2;
        sa.b_group_elems = (int64_t)d * Fs;
        sa.N = Fs;
        sa.aux = h_gu_sh;
        sa.out0 = dh_sh;
        if ((st = cuda_status(launch_gemm_m(sa, bf16, s), "shared dA gemm"))) return st;
        GemmMArgs sb = b;
        sb.group_expert = nullptr;  // shared experts: one group per expert
        sb.G = S;
        sb.rows = GroupRows{nullptr, (int)T, T, 0, T};
        sb.a = dh_sh;
        sb.b = ws1;
        sb.b_group_elems = (int64_t)2 * Fs * d;
        sb.K = 2 * Fs;
        sb.out0 = dx_sh;
        if ((st = cuda_status(launch_gemm_m(sb, bf16, s), "shared dX gemm"))) return st;
        GemmKArgs sw2 = w2g;
        sw2.group_expert = nullptr;  // shared experts: one group per expert
        sw2.G = S;
        sw2.rows = GroupRows{nullptr, (int)T, 0, T, 0};
        sw2.a = dout;
        sw2.b = act_sh;
        sw2.N = Fs;
        sw2.out = dws2;
        if ((st = cuda_status(launch_gemm_k(sw2, bf16, s), "shared dW2 gemm"))) return st;
        GemmKArgs sw1 = w1g;
        sw1.group_expert = nullptr;  // shared experts: one group per expert
        sw1.G = S;
        sw1.rows = GroupRows{nullptr, (int)T, T, 0, 0};
        sw1.a = dh_sh;
        sw1.b = x;
        sw1.M = 2 * Fs;
        sw1.out = dws1;
        if ((st = cuda_status(launch_gemm_k(sw1, bf16, s), "shared dW1 gemm"))) return st;
    }
    return MOE_OK;
}

moe_status moe_route_bwd(const moe_config* cfg, const void* x, const void* w_router,
                         const float* probs, const int32_t* topk_idx, const float* topk_w,
                         const float* dtopk_w, const float* aux_coef,
                         const int32_t* party_offsets, float* dlogits, void* dw_router,
                         float* dbias, void* dx_router, void* workspace,
                         size_t workspace_bytes, moe_stream_t stream) {
    moe_status st = check_cfg(cfg);
    if (st) return st;
    if ((st = check_parties(cfg, party_offsets))) return st;
    REQUIRE_VEC(dw_router);
    if (dx_router && cfg->T > 0) {
        REQUIRE_VEC(dx_router);
        REQUIRE_VEC(w_router);
    }
    if (cfg->T > 0) {
        REQUIRE_VEC(x);
        REQUIRE(probs);
        REQUIRE(topk_idx);
        REQUIRE(topk_w);
        REQUIRE(dtopk_w);
        REQUIRE(dlogits);
    }
    REQUIRE(workspace);
    const size_t need = route_bwd_workspace(cfg->T, cfg->n_parties, cfg->n_experts, cfg->d_model);
    if (workspace_bytes < need)
        return fail(MOE_ERR_INVALID_ARG, "workspace of %zu bytes < %zu needed", workspace_bytes, need);
    RouteBwdArgs a{};
    a.x = x;
    a.probs = probs;
    a.topk_idx = topk_idx;
    a.topk_w = topk_w;
    a.dtopk_w = dtopk_w;
    a.aux_coef = aux_coef;
    a.po = party_offsets;
    a.P = cfg->n_parties;
    a.T = cfg->T;
    a.d = cfg->d_model;
    a.E = cfg->n_experts;
    a.k = cfg->top_k;
    a.normalize = cfg->normalize_topk;
    a.dlogits = dlogits;
    a.dw_router = dw_router;
    a.dbias = dbias;
    a.w_router = w_router;
    a.dx_router = dx_router;
    return cuda_status(launch_route_bwd(a, cfg->dtype == MOE_BF16, workspace, (cudaStream_t)stream),
                       "moe_route_bwd");
}

moe_status moe_dispatch_bwd(const moe_config* cfg, const void* dx_perm, const int32_t* slot_of,
                            const void* dx_router, const void* dx_sh, void* dx,
                            moe_stream_t stream) {
    moe_status st = check_cfg(cfg);
    if (st) return st;
    if (cfg->T == 0) return MOE_OK;
    REQUIRE_VEC(dx_perm);
    REQUIRE(slot_of);
    if (dx_router) REQUIRE_VEC(dx_router);
    REQUIRE_VEC(dx);
    if (cfg->n_shared) REQUIRE_VEC(dx_sh);
    return cuda_status(launch_unpermute_reduce(dx_perm, slot_of, dx_router, dx_sh, cfg->n_shared,
                                               cfg->T, cfg->d_model, cfg->top_k,
                                               cfg->dtype == MOE_BF16, dx, (cudaStream_t)stream),
                       "moe_dispatch_bwd");
}

moe_status moe_gather_rows(const void* src, const int32_t* rows, int64_t n_rows, int64_t n_src_rows,
                           int64_t row_elems, moe_dtype dtype, void* dst, moe_stream_t stream) {
    if (dtype != MOE_F32 && dtype != MOE_BF16) return fail(MOE_ERR_INVALID_ARG, "unknown dtype %d", (int)dtype);
    if (n_rows < 0 || n_src_rows < 0 || row_elems < 0)
        return fail(MOE_ERR_INVALID_ARG, "negative size (n_rows=%lld, n_src_rows=%lld, row_elems=%lld)",
                    (long long)n_rows, (long long)n_src_rows, (long long)row_elems);
    const int64_t row_bytes = row_elems * (dtype == MOE_BF16 ? 2 : 4);
    if (row_bytes % 16) return fail(MOE_ERR_INVALID_ARG, "row of %lld bytes is not a multiple of 16", (long long)row_bytes);
    if (n_rows == 0 || row_elems == 0) return MOE_OK;
    REQUIRE_VEC(src);
    REQUIRE(rows);
    REQUIRE_VEC(dst);
    if (row_bytes / 16 > INT32_MAX) return fail(MOE_ERR_INVALID_ARG, "row too long");
    return cuda_status(launch_gather_rows(src, rows, n_rows, n_src_rows, row_bytes, dst, (cudaStream_t)stream),
                       "moe_gather_rows");
}

moe_status moe_expert_ffn_bwd_kernels(const moe_config* cfg, int32_t* count) {
    moe_status st = check_cfg(cfg);
    if (st) return st;
    REQUIRE(count);
    const bool bf16 = cfg->dtype == MOE_BF16;
    const int64_t TK = cfg->T * cfg->top_k;
    static const int32_t marker = 0;  // offsets mode: only its non-null-ness is looked at
    GemmMArgs a{}, b{};
    a.G = b.G = cfg->n_experts;
    a.rows = b.rows = GroupRows{&marker, (int)TK, 0, 0, 0};
    a.b_kmajor = b.b_kmajor = false;
    a.N = cfg->d_ff;
    a.K = cfg->d_model;
    a.epi = EPI_SWIGLU_BWD;
    b.N = cfg->d_model;
    b.K = 2 * cfg->d_ff;
    b.epi = EPI_STORE;
    int n = 0;
    if (TK > 0) {
        n += (bf16 && !gemm_m_uses_pairs(a)) ? 1 : 2;
        n += (bf16 && !gemm_m_uses_pairs(b)) ? 1 : 2;
    }
    if (cfg->n_shared && cfg->T > 0) n += 4;
    *count = n;
    return MOE_OK;
}

moe_status moe_mse_loss(const moe_config* cfg, const void* out, const void* target, float* loss,
                        void* dout, void* workspace, size_t workspace_bytes, moe_stream_t stream) {
    moe_status st = check_cfg(cfg);
    if (st) return st;
    REQUIRE(loss);
    if (cfg->T == 0)
        return cuda_status(cudaMemsetAsync(loss, 0, sizeof(float), (cudaStream_t)stream), "moe_mse_loss");
    REQUIRE(out);
    REQUIRE(target);
    REQUIRE(dout);
    REQUIRE(workspace);
    if (workspace_bytes < mse_workspace_bytes())
        return fail(MOE_ERR_INVALID_ARG, "workspace_bytes %zu < %zu", workspace_bytes, mse_workspace_bytes());
    return cuda_status(launch_mse_loss(out, target, cfg->T, cfg->d_model, cfg->dtype == MOE_BF16, loss, dout,
                                       workspace, (cudaStream_t)stream),
                       "moe_mse_loss");
}

moe_status moe_sgd_update(void* w, const void* dw, float* w_master, int64_t n_groups, int64_t group_elems,
                          const int32_t* group_counts, float lr, moe_dtype dtype, moe_stream_t stream) {
    if (n_groups < 0 || group_elems < 0)
        return fail(MOE_ERR_INVALID_ARG, "negative size (n_groups=%lld, group_elems=%lld)",
                    (long long)n_groups, (long long)group_elems);
    if (n_groups > 65535) return fail(MOE_ERR_INVALID_ARG, "n_groups=%lld > 65535", (long long)n_groups);
    if (dtype != MOE_F32 && dtype != MOE_BF16) return fail(MOE_ERR_INVALID_ARG, "unknown dtype %d", (int)dtype);
    if (!(lr == lr) || lr - lr != 0.0f) return fail(MOE_ERR_INVALID_ARG, "lr is not finite");
    if (n_groups == 0 || group_elems == 0) return MOE_OK;
    REQUIRE(w);
    REQUIRE(dw);
    return cuda_status(launch_sgd_update(w, dw, w_master, n_groups, group_elems, group_counts, lr, dtype == MOE_BF16,
                                         (cudaStream_t)stream),
                       "moe_sgd_update");
}

moe_status moe_device_status(moe_stream_t stream, int32_t* code) {
    REQUIRE(code);
    cudaStream_t s = (cudaStream_t)stream;
    int c[4] = {0, 0, 0, 0};
    cudaError_t e;
    if ((e = route_status(s, &c[0])) != cudaSuccess) return cuda_status(e, "status");
    if ((e = dispatch_status(s, &c[1])) != cudaSuccess) return cuda_status(e, "status");
    if ((e = gemm_status(s, &c[2])) != cudaSuccess) return cuda_status(e, "status");
    if ((e = simt_status(s, &c[3])) != cudaSuccess) return cuda_status(e, "status");
    *code = 0;
    for (int i = 0; i < 4; ++i)
        if (c[i] && !*code) *code = c[i];
    return MOE_OK;
}

}  // extern "C"
