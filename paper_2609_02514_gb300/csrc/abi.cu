// C ABI of the AceSpec path: argument validation, launch configuration and
// workspace carving.  Nothing here allocates memory.
#include <climits>
#include <cmath>
#include <mutex>

#define ACES_FILE 1  // site numbers of the checked build
#include "common.cuh"

using namespace aces;

namespace {

bool aligned16(const void *p) { return ((uintptr_t)p & 15u) == 0; }

int sm_count() {
    int dev = 0, n = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 132;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) return 132;
    return n;
}

size_t elem_size(aces_dtype dt) { return dt == ACES_BF16 ? 2 : 4; }

// Common checks of the target-row arguments.  Returns ACES_OK or the error.
aces_status check_rows(const void *logits, aces_dtype dt, long long rows, int V, float T, float top_p,
                       int k, bool need_payload, const void *ids, const void *probs, const void *tail,
                       const void *status) {
    if (dt != ACES_F32 && dt != ACES_BF16) return ACES_ERR_UNSUPPORTED;
    if (!logits || !status) return ACES_ERR_INVALID_ARG;
    if (rows < 1 || rows > INT_MAX / 2) return ACES_ERR_INVALID_ARG;
    if (V < 2 || V > ACES_MAX_V) return ACES_ERR_INVALID_ARG;
    if (T == 0.0f) return ACES_ERR_UNSUPPORTED;  // greedy decoding is not a distribution
    if (!(T > 0.0f) || !std::isfinite(T)) return ACES_ERR_INVALID_ARG;
    if (!(top_p > 0.0f && top_p <= 1.0f)) return ACES_ERR_INVALID_ARG;
    if (k < 0 || k > ACES_MAX_TOPK || k > V) return ACES_ERR_INVALID_ARG;
    if (need_payload && k < 1) return ACES_ERR_INVALID_ARG;
    if (k > 0 && (!ids || !probs || !tail)) return ACES_ERR_INVALID_ARG;
    (void)elem_size;
    return ACES_OK;
}

// Row kernels: the single-pass capture kernel when rows are 16-byte
// aligned, then the exact general kernel for every row it handed over (or
// for every row otherwise).
aces_status run_rows(RowArgs &a, aces_dtype dt, bool exact, cudaStream_t s) {
    const size_t es = elem_size(dt);
    const bool vec = aligned16(a.logits) && ((size_t)a.V * es) % 16 == 0;
    const int nsm = sm_count();
    const int nseq = a.K > 0 ? a.rows / (a.K + 1) : a.rows;
    if (cudaMemsetAsync(a.ws.fb_count, 0, ws_clear_bytes(nseq, a.K), s) != cudaSuccess) return ACES_ERR_CUDA;
    const int grid = a.rows < 2 * nsm ? a.rows : 2 * nsm;
    a.nsm = nsm;
    // With many waves of rows the four CTAs an SM starts with would reach
    // their epilogues (when few loads are in flight) together, wave after
    // wave: their starts are spread over about a quarter of a row's time.
    a.stagger_ns = a.rows >= 16 * nsm ? STAGGER_NS : 0;
    if (vec) {
        rows_cap_layout(a, dt);
        a.force_fb = exact ? 1 : 0;
        if (launch_rows_cap(a, dt, s) != cudaSuccess) return ACES_ERR_CUDA;
        if (launch_rows_general(a, dt, true, 0, grid, s) != cudaSuccess) return ACES_ERR_CUDA;
    } else {
        a.force_fb = 0;
        if (launch_rows_general(a, dt, false, 1, grid, s) != cudaSuccess) return ACES_ERR_CUDA;
    }
    return ACES_OK;
}

}  // namespace

extern "C" {

size_t aces_workspace_bytes(int B, int K, int V, int k) {
    if (B < 1 || K < 0 || K > ACES_MAX_K || V < 2 || V > ACES_MAX_V || k < 0 || k > ACES_MAX_TOPK)
        return 0;
    long long rows = (long long)B * (K + 1);
    if (rows > INT_MAX / 2) return 0;
    return ws_bytes((int)rows, B, K, true);
}

}  // extern "C"

// The argument checks of aces_verify (nothing is launched).
static aces_status verify_check(const void *target_logits, aces_dtype dt, const float *draft_probs,
                                const int32_t *draft_tokens, const float *uniforms, int B, int K, int V,
                                float T, float top_p, int32_t *accept_len, int32_t *out_token, int k,
                                int32_t *topk_ids, float *topk_probs, float *tail_mass, int32_t *row_status,
                                void *workspace, size_t workspace_bytes, bool lists) {
    if (B < 1 || K < 1 || K > ACES_MAX_K) return ACES_ERR_INVALID_ARG;
    aces_status st = check_rows(target_logits, dt, (long long)B * (K + 1), V, T, top_p, k, false,
                                topk_ids, topk_probs, tail_mass, row_status);
    if (st != ACES_OK) return st;
    if (!draft_probs || !draft_tokens || !uniforms || !accept_len || !out_token || !workspace)
        return ACES_ERR_INVALID_ARG;
    if (!aligned16(workspace) || workspace_bytes < ws_bytes(B * (K + 1), B, K, lists))
        return ACES_ERR_INVALID_ARG;
    return ACES_OK;
}

// Results depend on neither `lists` (without them the residual draw scans its
// whole row instead of the stored nucleus) nor `exact` (every row on the
// general kernel).
aces_status aces::verify_impl(const void *target_logits, aces_dtype dt, const float *draft_probs,
                        const int32_t *draft_tokens, const float *uniforms, int B, int K, int V,
                        float T, float top_p, int32_t *accept_len, int32_t *out_token, int k,
                        int32_t *topk_ids, float *topk_probs, float *tail_mass,
                        int32_t *row_status, void *workspace, size_t workspace_bytes, bool lists,
                        bool exact, aces_stream_t stream) {
    aces_status st = verify_check(target_logits, dt, draft_probs, draft_tokens, uniforms, B, K, V, T, top_p,
                                  accept_len, out_token, k, topk_ids, topk_probs, tail_mass, row_status,
                                  workspace, workspace_bytes, lists);
    if (st != ACES_OK) return st;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    const int rows = B * (K + 1);
    RowArgs a;
    a.logits = target_logits;
    a.rows = rows;
    a.V = V;
    a.K = K;
    a.T = T;
    a.c = (float)(1.4426950408889634 / (double)T);
    a.inv_w = (float)(BIN_PER_T / (double)T);
    a.top_p = top_p;
    a.k = k;
    a.q = draft_probs;
    a.xt = draft_tokens;
    a.u = uniforms;
    a.topk_ids = topk_ids;
    a.topk_probs = topk_probs;
    a.tail = tail_mass;
    a.row_status = row_status;
    a.ws = ws_carve(workspace, rows, B, K, lists && top_p < 1.0f);
    a.accept_len = accept_len;
    a.out_token = out_token;
    st = run_rows(a, dt, exact, s);
    if (st != ACES_OK) return st;
    ResolveArgs r;
    r.logits = target_logits;
    r.q = draft_probs;
    r.u = uniforms;
    r.B = B;
    r.K = K;
    r.V = V;
    r.T = T;
    r.top_p = top_p;
    r.k = k;
    r.ws = a.ws;
    r.accept_len = accept_len;
    r.out_token = out_token;
    r.row_status = row_status;
    const bool vec = aligned16(target_logits) && ((size_t)V * elem_size(dt)) % 16 == 0 &&
                     aligned16(draft_probs) && V % 4 == 0;
    if (launch_resolve(r, dt, vec, s) != cudaSuccess) return ACES_ERR_CUDA;
    return ACES_OK;
}

extern "C" {

aces_status aces_verify(const void *target_logits, aces_dtype dt, const float *draft_probs,
                        const int32_t *draft_tokens, const float *uniforms, int B, int K, int V,
                        float T, float top_p, int32_t *accept_len, int32_t *out_token, int k,
                        int32_t *topk_ids, float *topk_probs, float *tail_mass,
                        int32_t *row_status, void *workspace, size_t workspace_bytes,
                        aces_stream_t stream) {
    if (B < 1 || K < 1 || K > ACES_MAX_K) return ACES_ERR_INVALID_ARG;
    if (workspace_bytes < aces_workspace_bytes(B, K, V, k)) return ACES_ERR_INVALID_ARG;
    return verify_impl(target_logits, dt, draft_probs, draft_tokens, uniforms, B, K, V, T, top_p,
                       accept_len, out_token, k, topk_ids, topk_probs, tail_mass, row_status,
                       workspace, workspace_bytes, true, false, stream);
}

aces_status aces_verify_exact(const void *target_logits, aces_dtype dt, const float *draft_probs,
                              const int32_t *draft_tokens, const float *uniforms, int B, int K, int V,
                              float T, float top_p, int32_t *accept_len, int32_t *out_token, int k,
                              int32_t *topk_ids, float *topk_probs, float *tail_mass,
                              int32_t *row_status, void *workspace, size_t workspace_bytes,
                              aces_stream_t stream) {
    if (B < 1 || K < 1 || K > ACES_MAX_K) return ACES_ERR_INVALID_ARG;
    if (workspace_bytes < aces_workspace_bytes(B, K, V, k)) return ACES_ERR_INVALID_ARG;
    return verify_impl(target_logits, dt, draft_probs, draft_tokens, uniforms, B, K, V, T, top_p,
                       accept_len, out_token, k, topk_ids, topk_probs, tail_mass, row_status,
                       workspace, workspace_bytes, true, true, stream);
}

aces_status aces_sparsify(const void *target_logits, aces_dtype dt, int rows, int V, float T,
                          float top_p, int k, int32_t *topk_ids, float *topk_probs,
                          float *tail_mass, int32_t *row_status, void *workspace,
                          size_t workspace_bytes, aces_stream_t stream) {
    aces_status st = check_rows(target_logits, dt, rows, V, T, top_p, k, true, topk_ids, topk_probs,
                                tail_mass, row_status);
    if (st != ACES_OK) return st;
    if (!workspace || !aligned16(workspace) || workspace_bytes < aces_workspace_bytes(rows, 0, V, k))
        return ACES_ERR_INVALID_ARG;
    RowArgs a;
    a.logits = target_logits;
    a.rows = rows;
    a.V = V;
    a.K = 0;
    a.T = T;
    a.c = (float)(1.4426950408889634 / (double)T);
    a.inv_w = (float)(BIN_PER_T / (double)T);
    a.top_p = top_p;
    a.k = k;
    a.q = nullptr;
    a.xt = nullptr;
    a.u = nullptr;
    a.topk_ids = topk_ids;
    a.topk_probs = topk_probs;
    a.tail = tail_mass;
    a.row_status = row_status;
    a.ws = ws_carve(workspace, rows, rows, 0, false);
    a.accept_len = nullptr;
    a.out_token = nullptr;
    return run_rows(a, dt, false, reinterpret_cast<cudaStream_t>(stream));
}

static aces_status fill_cache_args(CacheArgs &c, const int32_t *F_host, int B, int K, int V) {
    if (!F_host || B < 1 || K < 1 || K > ACES_MAX_K || V < 2 || V > ACES_MAX_V) return ACES_ERR_INVALID_ARG;
    if ((long long)B * K > INT_MAX / 2) return ACES_ERR_INVALID_ARG;
    int tot = 0;
    c.off[0] = 0;
    for (int d = 0; d < K; ++d) {
        int f = F_host[d];
        if (f < 0 || f > V - 1) return ACES_ERR_INVALID_ARG;
        if (f > ACES_MAX_BRANCH) return ACES_ERR_UNSUPPORTED;
        c.F[d] = f;
        tot += f;
        c.off[d + 1] = tot;
    }
    for (int d = K; d < ACES_MAX_K; ++d) c.F[d] = 0;
    c.total = tot;
    c.B = B;
    c.K = K;
    c.V = V;
    return ACES_OK;
}

// The argument checks of aces_cache_build and its kernel arguments.
static aces_status cache_prepare(CacheArgs &c, const float *draft_probs, const int32_t *draft_tokens,
                                 const int32_t *F_host, int B, int K, int V, int32_t *branch_tok,
                                 float *branch_prob) {
    aces_status st = fill_cache_args(c, F_host, B, K, V);
    if (st != ACES_OK) return st;
    if (!draft_probs || !draft_tokens) return ACES_ERR_INVALID_ARG;
    if (c.total > 0 && (!branch_tok || !branch_prob)) return ACES_ERR_INVALID_ARG;
    c.q = draft_probs;
    c.xt = draft_tokens;
    c.bt = branch_tok;
    c.bp = branch_prob;
    return ACES_OK;
}

static aces_status cache_launch(const CacheArgs &c, cudaStream_t s) {
    if (c.total == 0) return ACES_OK;
    const bool vec = aligned16(c.q) && c.V % 4 == 0;
    return launch_cache_build(c, vec, s) == cudaSuccess ? ACES_OK : ACES_ERR_CUDA;
}

// The library's side stream of the current device, with a fork and a join
// event: created on the first aces_cloud_step on that device and kept until
// the process exits.  Held under g_side_mu while a call records and waits.
struct SideStream {
    cudaStream_t s;
    cudaEvent_t fork, join;
};
constexpr int SIDE_MAX_DEVICES = 64;
static std::mutex g_side_mu;
static SideStream g_side[SIDE_MAX_DEVICES];
static bool g_side_ok[SIDE_MAX_DEVICES];

static aces_status side_stream(SideStream **out) {  // called with g_side_mu held
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= SIDE_MAX_DEVICES) return ACES_ERR_CUDA;
    if (!g_side_ok[dev]) {
        SideStream ss;
        if (cudaStreamCreateWithFlags(&ss.s, cudaStreamNonBlocking) != cudaSuccess) return ACES_ERR_CUDA;
        if (cudaEventCreateWithFlags(&ss.fork, cudaEventDisableTiming) != cudaSuccess) return ACES_ERR_CUDA;
        if (cudaEventCreateWithFlags(&ss.join, cudaEventDisableTiming) != cudaSuccess) return ACES_ERR_CUDA;
        g_side[dev] = ss;
        g_side_ok[dev] = true;
    }
    *out = &g_side[dev];
    return ACES_OK;
}

aces_status aces_cache_build(const float *draft_probs, const int32_t *draft_tokens,
                             const int32_t *F_host, int B, int K, int V, int32_t *branch_tok,
                             float *branch_prob, aces_stream_t stream) {
    CacheArgs c;
    const aces_status st = cache_prepare(c, draft_probs, draft_tokens, F_host, B, K, V, branch_tok, branch_prob);
    if (st != ACES_OK) return st;
    return cache_launch(c, reinterpret_cast<cudaStream_t>(stream));
}

aces_status aces_cloud_step(const void *target_logits, aces_dtype dt, const float *draft_probs,
                            const int32_t *draft_tokens, const float *uniforms, int B, int K, int V,
                            float T, float top_p, int32_t *accept_len, int32_t *out_token, int k,
                            int32_t *topk_ids, float *topk_probs, float *tail_mass, int32_t *row_status,
                            const int32_t *F_host, int32_t *branch_tok, float *branch_prob, void *workspace,
                            size_t workspace_bytes, aces_stream_t stream) {
    aces_status st = verify_check(target_logits, dt, draft_probs, draft_tokens, uniforms, B, K, V, T, top_p,
                                  accept_len, out_token, k, topk_ids, topk_probs, tail_mass, row_status,
                                  workspace, workspace_bytes, true);
    if (st != ACES_OK) return st;
    if (workspace_bytes < aces_workspace_bytes(B, K, V, k)) return ACES_ERR_INVALID_ARG;
    CacheArgs c;
    st = cache_prepare(c, draft_probs, draft_tokens, F_host, B, K, V, branch_tok, branch_prob);
    if (st != ACES_OK) return st;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    std::lock_guard<std::mutex> lock(g_side_mu);
    SideStream *ss = nullptr;
    st = side_stream(&ss);
    if (st != ACES_OK) return st;
    // fork: the cache build on the side stream after everything before it on `stream`
    if (cudaEventRecord(ss->fork, s) != cudaSuccess || cudaStreamWaitEvent(ss->s, ss->fork, 0) != cudaSuccess)
        return ACES_ERR_CUDA;
    const aces_status sc = cache_launch(c, ss->s);
    const aces_status sv = verify_impl(target_logits, dt, draft_probs, draft_tokens, uniforms, B, K, V, T, top_p,
                                       accept_len, out_token, k, topk_ids, topk_probs, tail_mass, row_status,
                                       workspace, workspace_bytes, true, false, stream);
    // join: later work on `stream` waits for the cache build (also after a failure)
    if (cudaEventRecord(ss->join, ss->s) != cudaSuccess || cudaStreamWaitEvent(s, ss->join, 0) != cudaSuccess)
        return ACES_ERR_CUDA;
    return sc != ACES_OK ? sc : sv;
}

aces_status aces_cache_lookup(const int32_t *branch_tok, const int32_t *F_host, int B, int K,
                              const int32_t *accept_len, const int32_t *token, int32_t *slot,
                              aces_stream_t stream) {
    CacheArgs c;
    if (!F_host || B < 1 || K < 1 || K > ACES_MAX_K) return ACES_ERR_INVALID_ARG;
    int tot = 0;
    c.off[0] = 0;
    for (int d = 0; d < K; ++d) {
        if (F_host[d] < 0 || F_host[d] > ACES_MAX_BRANCH) return ACES_ERR_INVALID_ARG;
        c.F[d] = F_host[d];
        tot += F_host[d];
        c.off[d + 1] = tot;
    }
    for (int d = K; d < ACES_MAX_K; ++d) c.F[d] = 0;
    c.total = tot;
    c.B = B;
    c.K = K;
    c.V = 0;
    c.q = nullptr;
    c.xt = nullptr;
    c.bt = nullptr;
    c.bp = nullptr;
    if (!accept_len || !token || !slot || (tot > 0 && !branch_tok)) return ACES_ERR_INVALID_ARG;
    if (launch_cache_lookup(branch_tok, c, accept_len, token, slot,
                            reinterpret_cast<cudaStream_t>(stream)) != cudaSuccess)
        return ACES_ERR_CUDA;
    return ACES_OK;
}

aces_status aces_resample_sparse(const int32_t *accept_len, const int32_t *topk_ids, const float *topk_probs,
                                 const float *tail_mass, const int32_t *row_status, const float *draft_probs,
                                 const float *uniforms, int B, int K, int V, int k, int32_t *token,
                                 int32_t *status, aces_stream_t stream) {
    if (B < 1 || K < 1 || K > ACES_MAX_K || V < 2 || V > ACES_MAX_V) return ACES_ERR_INVALID_ARG;
    if (k < 1 || k > ACES_MAX_TOPK || k > V) return ACES_ERR_INVALID_ARG;
    if ((long long)B * (K + 1) > INT_MAX / 2) return ACES_ERR_INVALID_ARG;
    if (!accept_len || !topk_ids || !topk_probs || !tail_mass || !row_status || !draft_probs || !uniforms ||
        !token || !status)
        return ACES_ERR_INVALID_ARG;
    const bool vec = aligned16(draft_probs) && V % 4 == 0;
    if (launch_resample_sparse(accept_len, topk_ids, topk_probs, tail_mass, row_status, draft_probs, uniforms, B,
                               K, V, k, token, status, vec, reinterpret_cast<cudaStream_t>(stream)) !=
        cudaSuccess)
        return ACES_ERR_CUDA;
    return ACES_OK;
}

aces_status aces_compact_kv(void *kv, int elem_bytes, int planes, int B, int H, int S, int D,
                            const int32_t *prefix_len, const int32_t *accept_len, const int32_t *slot, int K,
                            int branch_len, int32_t *new_len, aces_stream_t stream) {
    if (!kv || !prefix_len || !accept_len || !slot || !new_len) return ACES_ERR_INVALID_ARG;
    if (elem_bytes != 1 && elem_bytes != 2 && elem_bytes != 4 && elem_bytes != 8) return ACES_ERR_INVALID_ARG;
    if (planes < 1 || B < 1 || H < 1 || S < 1 || D < 1 || K < 1 || K > ACES_MAX_K || branch_len < 1)
        return ACES_ERR_INVALID_ARG;
    const size_t row_bytes = (size_t)D * (size_t)elem_bytes;
    if (row_bytes % 16 != 0 || !aligned16(kv)) return ACES_ERR_INVALID_ARG;
    if ((long long)B * planes * H > (long long)INT_MAX * 8) return ACES_ERR_INVALID_ARG;
    if (launch_compact_kv(kv, planes, B, H, S, row_bytes, prefix_len, accept_len, slot, K, branch_len, new_len,
                          reinterpret_cast<cudaStream_t>(stream)) != cudaSuccess)
        return ACES_ERR_CUDA;
    return ACES_OK;
}

int aces_tree_tokens(const int32_t *F_host, int K, int branch_len) {
    if (!F_host || K < 1 || K > ACES_MAX_K || branch_len < 1) return -1;
    long long n = K;
    for (int d = 0; d < K; ++d) {
        if (F_host[d] < 0 || F_host[d] > ACES_MAX_BRANCH) return -1;
        n += (long long)F_host[d] * branch_len;
    }
    return n > (1 << 20) ? -1 : (int)n;
}

aces_status aces_tree_mask(const int32_t *F_host, int K, int branch_len, uint32_t *mask, int32_t *depth,
                           aces_stream_t stream) {
    const int n = aces_tree_tokens(F_host, K, branch_len);
    if (n < 0 || !mask || !depth) return ACES_ERR_INVALID_ARG;
    int off[ACES_MAX_K + 1];
    off[0] = 0;
    for (int d = 0; d < K; ++d) off[d + 1] = off[d] + F_host[d];
    const int words = (n + 31) / 32;
    if (launch_tree_mask(off, K, branch_len, n, words, mask, depth, reinterpret_cast<cudaStream_t>(stream)) !=
        cudaSuccess)
        return ACES_ERR_CUDA;
    return ACES_OK;
}

const char *aces_status_string(aces_status s) {
    switch (s) {
        case ACES_OK: return "ok";
        case ACES_ERR_INVALID_ARG: return "invalid argument";
        case ACES_ERR_UNSUPPORTED: return "unsupported argument";
        case ACES_ERR_CUDA: return "CUDA launch error";
    }
    return "unknown status";
}

}  // extern "C"

#ifdef ACES_CHECKED
// The first out-of-range index met by any kernel since the last call (see
// ACES_IN in common.cuh): out = {site, index, bound}, site 0 when none.
// Waits for the device.  Clears every word.
extern "C" aces_status aces_checked_violation(unsigned long long out[3]) {
    if (!out) return ACES_ERR_INVALID_ARG;
    if (cudaDeviceSynchronize() != cudaSuccess) return ACES_ERR_CUDA;
    cudaError_t (*take[])(unsigned long long *) = {check_take_rows_cap, check_take_rows_general, check_take_resolve,
                                                   check_take_cache, check_take_resample, check_take_kv,
                                                   check_take_mask};
    out[0] = out[1] = out[2] = 0ull;
    for (auto f : take) {
        unsigned long long w[3];
        if (f(w) != cudaSuccess) return ACES_ERR_CUDA;
        if (out[0] == 0ull && w[0] != 0ull) {
            out[0] = w[0];
            out[1] = w[1];
            out[2] = w[2];
        }
    }
    return ACES_OK;
}
#endif
