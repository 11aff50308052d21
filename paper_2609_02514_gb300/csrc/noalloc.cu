// aces_verify_noalloc: aces_verify for callers that cannot allocate device
// memory themselves.
//
// aces_verify needs a caller-provided device workspace.  Some callers have no
// way to provide one on their serving path: cudaMalloc synchronizes the whole
// device (a latency-bound verification loop cannot afford that stall), and
// some host runtimes that embed this library own all device memory and give
// libraries none.  This entry point uses a fixed scratch area that lives in
// the library itself (a file-scope __device__ array, ACES_NOALLOC_SCRATCH_BYTES
// bytes, present on every GPU that loads the library until the process
// exits) and calls no allocator at all.
//
// The scratch is shared by every call on a device and keeps what the last
// call left there.  aces_verify clears the counters it needs at the start of
// every call and writes every other scratch word before reading it, so no
// extra clearing is needed here.  Calls whose work overlaps on the GPU (two
// streams, or calls on one stream that a caller reorders) race on the scratch
// and must not be issued.
#include <mutex>

#define ACES_FILE 6  // site numbers of the checked build
#include "common.cuh"

namespace {

static __device__ __align__(256) unsigned char g_noalloc_scratch[ACES_NOALLOC_SCRATCH_BYTES];

constexpr int MAX_DEVICES = 64;
void *g_scratch_addr[MAX_DEVICES];  // device address of g_noalloc_scratch, per device
std::mutex g_scratch_mu;

// Device address of the scratch array on the current device.  The array's
// name is only a host-side stand-in, so the address is looked up once per
// device with that device current.
aces_status scratch_address(void **out) {
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= MAX_DEVICES) return ACES_ERR_CUDA;
    std::lock_guard<std::mutex> lock(g_scratch_mu);
    if (g_scratch_addr[dev] == nullptr) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr) return ACES_ERR_CUDA;
        g_scratch_addr[dev] = p;
    }
    *out = g_scratch_addr[dev];
    return ACES_OK;
}

}  // namespace

extern "C" aces_status aces_verify_noalloc(const void *target_logits, aces_dtype dt, const float *draft_probs,
                                           const int32_t *draft_tokens, const float *uniforms, int B, int K,
                                           int V, float T, float top_p, int32_t *accept_len,
                                           int32_t *out_token, int k, int32_t *topk_ids, float *topk_probs,
                                           float *tail_mass, int32_t *row_status, aces_stream_t stream) {
    if (B < 1 || K < 1 || K > ACES_MAX_K) return ACES_ERR_INVALID_ARG;
    const size_t full = aces_workspace_bytes(B, K, V, k);
    if (full == 0) return ACES_ERR_INVALID_ARG;
    // The nucleus lists (4 KiB per row) fit for small batches only; without
    // them the call needs ws_bytes(rows, B, K, false) bytes.
    const int rows = B * (K + 1);
    const size_t cap = (size_t)ACES_NOALLOC_SCRATCH_BYTES;
    const bool lists = full <= cap;
    if (aces::ws_bytes(rows, B, K, false) > cap) return ACES_ERR_UNSUPPORTED;  // batch too large
    void *scratch = nullptr;
    const aces_status st = scratch_address(&scratch);
    if (st != ACES_OK) return st;
    return aces::verify_impl(target_logits, dt, draft_probs, draft_tokens, uniforms, B, K, V, T, top_p,
                             accept_len, out_token, k, topk_ids, topk_probs, tail_mass, row_status, scratch,
                             cap, lists, false, stream);
}
