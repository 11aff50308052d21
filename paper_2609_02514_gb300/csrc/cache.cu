// Probabilistic state cache of the AceSpec edge step (Sec. III-C,
// Algorithm 1 TREE_DRAFT and the O(1) lookup of w = (pi, x_resampled)).
//
//   k_cache_build   one CTA per (sequence, depth) row of the draft
//                   distribution: the F_d largest q over ids != x~_d, in
//                   (q desc, id asc) order, with probability q / (1 - q(x~_d)).
//                   One HBM pass keeps a sorted top-TOPL list per thread
//                   (TOPL = 4 when every F_d <= 4, else 8), filtered by one
//                   integer max and compare per four values against the raw
//                   bits of the list's last entry.  F_d <= TOPL: the block
//                   extracts maxima one at a time.  F_d > TOPL: the 2048
//                   entries of all lists are sorted in shared memory; every
//                   id a thread dropped lies below its full list's last
//                   entry, so when the largest such entry is below the
//                   F_d-th sorted entry, the first F_d are the answer (one
//                   pass).  Otherwise the pass is repeated below the last
//                   extracted order value, TOPL maxima at a time.
//   k_cache_lookup  one thread per sequence scanning the F_pi branches.
#define ACES_FILE 3  // site numbers of the checked build
#include "common.cuh"

namespace aces {


constexpr int NTC = 256;  // threads per row
constexpr int CLD = 8;    // 16-byte loads in flight per thread

template <int TOPL>
__device__ __forceinline__ void list_insert(unsigned long long (&Lst)[TOPL], unsigned long long o) {
    Lst[TOPL - 1] = o;
#pragma unroll
    for (int i = TOPL - 1; i > 0; --i) {
        if (Lst[i] > Lst[i - 1]) {
            const unsigned long long t = Lst[i];
            Lst[i] = Lst[i - 1];
            Lst[i - 1] = t;
        }
    }
}

// TOPL: per-thread list length (4 when every fan-out is at most 4, else 8)
template <bool VEC, int TOPL>
__global__ void __launch_bounds__(NTC, 4) k_cache_build(CacheArgs a) {
    __shared__ unsigned long long redu[NTC / 32];
    // the union of the per-thread lists (fan-outs above TOPL)
    __shared__ unsigned long long uni[TOPL == 8 ? NTC * TOPL : 1];
    __shared__ int s_done;
    const int row = blockIdx.x, tid = threadIdx.x;
    const int b = row / a.K, d = row % a.K;
    const int Fd = a.F[d];
    if (Fd == 0) return;
    const float *qr = a.q + (size_t)row * a.V;
    int32_t *bt = a.bt + (size_t)b * a.total + a.off[d];
    float *bp = a.bp + (size_t)b * a.total + a.off[d];
    const int xd = a.xt[row];
    float den = 0.0f;
    if (xd >= 0 && xd < a.V) den = 1.0f - __ldg(qr + xd);
    int got = 0;
    if (den > 0.0f) {
        unsigned long long ub = ~0ull;  // exclusive upper bound of this pass
        while (got < Fd) {
            unsigned long long Lst[TOPL];
#pragma unroll
            for (int i = 0; i < TOPL; ++i) Lst[i] = 0ull;
            // An element can only enter the list when its raw bits reach thr,
            // those of the list's last entry (at least 1: q > 0).  Positive
            // floats order like their bits; negative or NaN q pass this test
            // and are rejected below.
            uint32_t thr = 1u;
            auto consider = [&](float qv, int x) {
                if (!(qv > 0.0f) || x == xd) return;
                const unsigned long long o = order_val(__float_as_uint(qv) | 0x80000000u, (uint32_t)x);
                if (o < ub && o > Lst[TOPL - 1]) {
                    list_insert<TOPL>(Lst, o);
                    const uint32_t t = (uint32_t)(Lst[TOPL - 1] >> 32) & 0x7FFFFFFFu;
                    thr = t > 1u ? t : 1u;
                }
            };
            // Fd <= TOPL: a lane's Fd-th entry bounds the Fd largest of the
            // row from below (that lane alone holds Fd values at or above
            // it), so the warp's largest such entry raises every lane's
            // threshold; refreshed once per round of loads (the filter then
            // drops what no list could keep, and insertions stay rare)
            if (VEC) {
                const int nch = a.V >> 2;
                for (int c0 = tid; c0 < nch; c0 += NTC * CLD) {
                    if (TOPL == 8 && c0 != tid && Fd <= TOPL) {  // (warp-uniform; the short lists filter enough)
                        unsigned long long e = 0ull;
#pragma unroll
                        for (int i = 0; i < TOPL; ++i) e = i == Fd - 1 ? Lst[i] : e;
                        const uint32_t wb = __reduce_max_sync(0xffffffffu, (uint32_t)(e >> 32) & 0x7FFFFFFFu);
                        thr = wb > thr ? wb : thr;
                    }
                    uint4 w[CLD];
#pragma unroll
                    for (int u = 0; u < CLD; ++u) {
                        const int cc = c0 + u * NTC;
                        w[u] = cc < nch ? ldg16(qr + (size_t)cc * 4) : make_uint4(0u, 0u, 0u, 0u);
                    }
                    if (TOPL == 8) {
                        // the values reaching thr as bits of one mask, then
                        // one insertion site in a loop over them (unrolled
                        // sites of the eight-entry insertion overflow the
                        // instruction cache)
                        uint32_t mk = 0u;
#pragma unroll
                        for (int u = 0; u < CLD; ++u)
                            mk |= ((uint32_t)(w[u].x >= thr) | (uint32_t)(w[u].y >= thr) << 1 |
                                   (uint32_t)(w[u].z >= thr) << 2 | (uint32_t)(w[u].w >= thr) << 3) << (4 * u);
                        while (mk) {
                            const int bit = __ffs(mk) - 1;
                            mk &= mk - 1u;
                            const int u = bit >> 2, j = bit & 3;
                            uint4 x = w[0];
#pragma unroll
                            for (int k = 1; k < CLD; ++k) x = u == k ? w[k] : x;
                            const uint32_t v = j == 0 ? x.x : j == 1 ? x.y : j == 2 ? x.z : x.w;
                            consider(__uint_as_float(v), (c0 + u * NTC) * 4 + j);
                        }
                    } else {
#pragma unroll
                        for (int u = 0; u < CLD; ++u) {
                            // one test per four values: the largest raw bits
                            if (max(max(w[u].x, w[u].y), max(w[u].z, w[u].w)) >= thr) {
                                const int x0 = (c0 + u * NTC) * 4;
                                if (w[u].x >= thr) consider(__uint_as_float(w[u].x), x0);
                                if (w[u].y >= thr) consider(__uint_as_float(w[u].y), x0 + 1);
                                if (w[u].z >= thr) consider(__uint_as_float(w[u].z), x0 + 2);
                                if (w[u].w >= thr) consider(__uint_as_float(w[u].w), x0 + 3);
                            }
                        }
                    }
                }
            } else {
                for (int x = tid; x < a.V; x += NTC) {
                    const float qv = __ldg(qr + x);
                    if (__float_as_uint(qv) >= thr) consider(qv, x);
                }
            }
            if (TOPL == 8 && Fd > TOPL && got == 0 && ub == ~0ull) {
                // one pass for the whole fan-out when the union of the lists
                // provably holds the Fd largest
                const unsigned long long bound = Lst[TOPL - 1];  // 0: nothing dropped
                const unsigned long long D = block_reduce_n<NTC>(bound, redu, MaxU64());
#pragma unroll
                for (int i = 0; i < TOPL; ++i) uni[tid * TOPL + i] = Lst[i];
                __syncthreads();
                bitonic_sort_desc(uni, NTC * TOPL);
                const unsigned long long vF = ACES_IN(Fd - 1, NTC * TOPL) ? uni[Fd - 1] : ~0ull;
                if (tid == 0) s_done = D == 0ull || D < vF;
                __syncthreads();
                if (s_done) {
                    int n = 0;  // positive entries among the first Fd
                    for (int j = tid; j < Fd; j += NTC) {
                        const unsigned long long o = uni[j];
                        if (o != 0ull) {
                            bt[j] = (int32_t)order_id(o);
                            bp[j] = order_value(o) / den;
                            ++n;
                        }
                    }
                    got = (int)block_reduce_n<NTC>((unsigned long long)n, redu, SumU64());
                    break;
                }
            }
            const int take = min(TOPL, Fd - got);
            bool exhausted = false;
            for (int t = 0; t < take; ++t) {
                const unsigned long long best = block_reduce_n<NTC>(Lst[0], redu, MaxU64());
                if (best == 0ull) {
                    exhausted = true;
                    break;
                }
                if (Lst[0] == best) {  // order values are unique: one owner
#pragma unroll
                    for (int i = 0; i < TOPL - 1; ++i) Lst[i] = Lst[i + 1];
                    Lst[TOPL - 1] = 0ull;
                }
                if (tid == 0) {
                    bt[got] = (int32_t)order_id(best);
                    bp[got] = order_value(best) / den;
                }
                ++got;
                ub = best;
            }
            if (exhausted) break;
        }
    }
    for (int j = got + tid; j < Fd; j += NTC) {
        bt[j] = -1;
        bp[j] = 0.0f;
    }
}

__global__ void k_cache_lookup(const int32_t *bt, CacheArgs a, const int32_t *accept_len,
                               const int32_t *token, int32_t *slot) {
    const int b = blockIdx.x * blockDim.x + threadIdx.x;
    if (b >= a.B) return;
    const int pi = accept_len[b];
    if (pi == a.K) {
        slot[b] = -2;
        return;
    }
    int s = -1;
    const int tok = token[b];
    if (pi >= 0 && pi < a.K && tok >= 0) {
        const int32_t *row = bt + (size_t)b * a.total + a.off[pi];
        for (int j = 0; j < a.F[pi]; ++j)
            if (row[j] == tok) {
                s = a.off[pi] + j;
                break;
            }
    }
    slot[b] = s;
}

cudaError_t launch_cache_build(const CacheArgs &a, bool vec, cudaStream_t s) {
    int fmax = 0;
    for (int d = 0; d < a.K; ++d) fmax = a.F[d] > fmax ? a.F[d] : fmax;
    const int g = a.B * a.K;
    if (fmax <= 4) {
        if (vec) k_cache_build<true, 4><<<g, NTC, 0, s>>>(a);
        else k_cache_build<false, 4><<<g, NTC, 0, s>>>(a);
    } else {
        if (vec) k_cache_build<true, 8><<<g, NTC, 0, s>>>(a);
        else k_cache_build<false, 8><<<g, NTC, 0, s>>>(a);
    }
    return cudaGetLastError();
}

cudaError_t launch_cache_lookup(const int32_t *bt, const CacheArgs &a, const int32_t *accept_len,
                                const int32_t *token, int32_t *slot, cudaStream_t s) {
    k_cache_lookup<<<(a.B + 255) / 256, 256, 0, s>>>(bt, a, accept_len, token, slot);
    return cudaGetLastError();
}

#ifdef ACES_CHECKED
cudaError_t check_take_cache(unsigned long long out[3]) { return check_take(out); }
#endif

}  // namespace aces
