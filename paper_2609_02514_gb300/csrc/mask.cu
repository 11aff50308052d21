// Tree attention mask of the packed branch forward (Sec. III-C): all
// branches are drafted in one forward pass, each tree token attending to
// the shared prefix (not stored here: every row sees all of it), to the
// main-chain tokens before its branch point (the main-path block) and to
// its own branch up to itself (the suffix-diagonal block).
//
// Packed order: the main chain (K tokens), then the branches in slot order
// (the slots of the cache lookup), branch_len tokens each.  One thread
// writes one 32-bit word of one row: a token's allowed keys are at most two
// intervals, [0, a) of the main chain and [b, c] of its own branch, so each
// word is two interval masks.
#define ACES_FILE 5  // site numbers of the checked build
#include "common.cuh"

namespace aces {

struct MaskArgs {
    int K, branch_len, n, words;
    int off[ACES_MAX_K + 1];  // first slot of every depth, off[K] = number of branches
    uint32_t *mask;
    int32_t *depth;
};

// bits [lo, hi) of the word covering keys [w0, w0 + 32)
__device__ __forceinline__ uint32_t interval_bits(int lo, int hi, int w0) {
    const int a = max(lo - w0, 0), b = min(hi - w0, 32);
    if (a >= b) return 0u;
    const uint32_t upto_b = b >= 32 ? 0xFFFFFFFFu : ((1u << b) - 1u);
    const uint32_t upto_a = (1u << a) - 1u;  // a < 32 here
    return upto_b & ~upto_a;
}

__global__ void k_tree_mask(MaskArgs a) {
    const long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= (long long)a.n * a.words) return;
    const int q = (int)(i / a.words), w = (int)(i % a.words);
    int main_hi, br_lo, br_hi, dep;  // keys [0, main_hi) and [br_lo, br_hi)
    if (q < a.K) {
        main_hi = q + 1;
        br_lo = br_hi = 0;
        dep = q;
    } else {
        const int s = (q - a.K) / a.branch_len, o = (q - a.K) % a.branch_len;
        int d = 0;
        while (d + 1 <= a.K && a.off[d + 1] <= s) ++d;  // depth of slot s
        main_hi = d;
        br_lo = a.K + s * a.branch_len;
        br_hi = q + 1;
        dep = d + o;
    }
    const int w0 = w * 32;
    a.mask[i] = interval_bits(0, main_hi, w0) | interval_bits(br_lo, br_hi, w0);
    if (w == 0) a.depth[q] = dep;
}

cudaError_t launch_tree_mask(const int *off, int K, int branch_len, int n, int words, uint32_t *mask,
                             int32_t *depth, cudaStream_t s) {
    MaskArgs a;
    a.K = K;
    a.branch_len = branch_len;
    a.n = n;
    a.words = words;
    for (int d = 0; d <= K; ++d) a.off[d] = off[d];
    a.mask = mask;
    a.depth = depth;
    const long long tot = (long long)n * words;
    k_tree_mask<<<(unsigned)((tot + 255) / 256), 256, 0, s>>>(a);
    return cudaGetLastError();
}

#ifdef ACES_CHECKED
cudaError_t check_take_mask(unsigned long long out[3]) { return check_take(out); }
#endif

}  // namespace aces
