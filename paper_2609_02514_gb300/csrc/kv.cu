// COMPACT_KV / ROLLBACK_KV of the edge pipeline (Alg. 1; Sec. III-C): after
// the lookup, the KV rows of the hit branch move right behind the accepted
// tokens, so the next cycle continues from a contiguous cache.
//
// KV layout: [planes, B, H, S, D] with planes = layers x {K, V}; the tree
// of sequence b sits after its prefix of prefix_len[b] positions: the main
// chain (K positions), then the branches in slot order, branch_len
// positions each.  One warp per (sequence, plane, head) block copies the
// branch's branch_len rows in 16-byte vectors.  Source and destination can
// overlap (the source always lies above the destination), so each warp
// moves them in increasing order, in rounds no longer than the distance
// between the two, loading a whole round before storing it.
#define ACES_FILE 4  // site numbers of the checked build
#include "common.cuh"

namespace aces {

constexpr int NTK = 256;
constexpr int KU = 4;  // 16-byte vectors per lane and round

struct KvArgs {
    char *kv;
    int planes, B, H, S;
    size_t row_bytes;  // D * element size, a multiple of 16
    const int32_t *prefix_len, *accept_len, *slot;
    int K, branch_len;
    int32_t *new_len;
};

__global__ void __launch_bounds__(NTK) k_compact_kv(KvArgs a) {
    const long long w = (long long)blockIdx.x * (NTK / 32) + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    const long long nblk = (long long)a.B * a.planes * a.H;
    if (w >= nblk) return;
    const int h = (int)(w % a.H);
    const int plane = (int)((w / a.H) % a.planes);
    const int b = (int)(w / ((long long)a.H * a.planes));
    const int t = a.prefix_len[b], pi = a.accept_len[b], s = a.slot[b];
    const int L = a.branch_len;
    const bool valid = t >= 0 && pi >= 0 && pi <= a.K;
    long long src = -1, len;
    if (s >= 0) {
        src = (long long)t + a.K + (long long)s * L;
        len = (valid && src + L <= a.S) ? (long long)t + pi + L : -1;
    } else if (s == -2) {
        len = (valid && (long long)t + a.K <= a.S) ? (long long)t + a.K : -1;
    } else {
        len = (valid && (long long)t + pi <= a.S) ? (long long)t + pi : -1;
    }
    if (plane == 0 && h == 0 && lane == 0) a.new_len[b] = (int32_t)len;
    if (s < 0 || len < 0) return;
    const long long dst = (long long)t + pi;
    if (src == dst) return;
    char *base = a.kv + (((size_t)plane * a.B + b) * a.H + h) * (size_t)a.S * a.row_bytes;
    if (!ACES_IN(src + L - 1, a.S) || !ACES_IN(dst, a.S)) return;
    const char *from = base + (size_t)src * a.row_bytes;
    char *to = base + (size_t)dst * a.row_bytes;
    const size_t total = (size_t)L * a.row_bytes;
    const size_t dist = (size_t)(src - dst) * a.row_bytes;
    const size_t cap = (size_t)32 * 16 * KU;
    const size_t round = dist < cap ? dist : cap;  // multiple of 16: row_bytes is
    for (size_t off = 0; off < total; off += round) {
        const size_t end = off + round < total ? off + round : total;
        uint4 v[KU];
#pragma unroll
        for (int u = 0; u < KU; ++u) {
            const size_t i = off + ((size_t)u * 32 + lane) * 16;
            if (i < end) v[u] = *reinterpret_cast<const uint4 *>(from + i);
        }
        __syncwarp();
#pragma unroll
        for (int u = 0; u < KU; ++u) {
            const size_t i = off + ((size_t)u * 32 + lane) * 16;
            if (i < end) *reinterpret_cast<uint4 *>(to + i) = v[u];
        }
        __syncwarp();
    }
}

cudaError_t launch_compact_kv(void *kv, int planes, int B, int H, int S, size_t row_bytes,
                              const int32_t *prefix_len, const int32_t *accept_len, const int32_t *slot, int K,
                              int branch_len, int32_t *new_len, cudaStream_t s) {
    KvArgs a;
    a.kv = reinterpret_cast<char *>(kv);
    a.planes = planes;
    a.B = B;
    a.H = H;
    a.S = S;
    a.row_bytes = row_bytes;
    a.prefix_len = prefix_len;
    a.accept_len = accept_len;
    a.slot = slot;
    a.K = K;
    a.branch_len = branch_len;
    a.new_len = new_len;
    const long long nblk = (long long)B * planes * H;
    const long long grid = (nblk + NTK / 32 - 1) / (NTK / 32);
    k_compact_kv<<<(unsigned)grid, NTK, 0, s>>>(a);
    return cudaGetLastError();
}

#ifdef ACES_CHECKED
cudaError_t check_take_kv(unsigned long long out[3]) { return check_take(out); }
#endif

}  // namespace aces
