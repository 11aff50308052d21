// Edge-side resample from the sparse downlink payload (Alg. 1
// RESAMPLE(P^_target, Q); Sec. III-B): the cloud returns the rejection index
// pi and the partial target distribution of row pi, and the edge draws the
// corrected token itself from that payload and its own draft row q_pi.
//
// The edge knows the target p only on the payload ids I (probs p^_I) and the
// mass tau = tail outside them.  For pi < K the tail is spread like the
// draft: p^(x) = tau * q(x) / q_rest outside I, with q_rest the draft mass
// outside I, so the residual r^ = max(0, p^ - q) is max(0, p^_x - q(x)) on I
// and q(x) * max(0, tau / q_rest - 1) outside.  For pi = K (bonus) the draw
// uses p^_I alone.  When the nucleus of row pi fits in the payload, tau = 0
// and the draw is the exact residual draw of aces_verify.
//
// One thread-block cluster of 8 CTAs (256 threads each) per sequence:
//   1. the payload of row pi is ordered by id in shared memory (direct rank
//      counting), and its weights (p^ - q on I) are gathered;
//   2. only when tau > 0, the 8 CTAs split q_pi's 2048-id tiles: one pass
//      gives each CTA's share of q_rest (compensated fp32), combined through
//      distributed shared memory; once the spread factor is known a second
//      pass gives the weight of every tile (four tiles' loads in flight per
//      thread), and the CTA holding the draw rescans its tile.  Otherwise
//      the first CTA draws alone and the others exit at once;
//   3. the draw: smallest id j whose prefix sum exceeds floor(u * R), with
//      every weight an integer in units of 2^-52 (exact, order independent).
#include <cooperative_groups.h>

#define ACES_FILE 7  // site numbers of the checked build
#include "common.cuh"

namespace aces {

constexpr int NTS = 256;
constexpr int SEPT = 8;                // consecutive ids per thread
constexpr int STILE = NTS * SEPT;      // ids per tile
constexpr int SPAY = ACES_MAX_TOPK;    // payload entries
constexpr int STILES = (ACES_MAX_V + STILE - 1) / STILE;
constexpr int TPI = 4;                 // tiles per round of the q passes
constexpr int SCL = 8;                 // CTAs per sequence: one thread-block cluster

// floor(x * 2^52) of a float x in [0, 2^11) from its bits (0 for x <= 0 or NaN)
__device__ __forceinline__ unsigned long long to_fx52(float x) {
    if (!(x > 0.0f)) return 0ull;
    const uint32_t u = __float_as_uint(x);
    const uint32_t be = u >> 23;
    const unsigned long long mant = (unsigned long long)((u & 0x7FFFFFu) | 0x800000u);
    const int sh = (int)be - 98;  // x * 2^52 = mant * 2^(be - 127 - 23 + 52)
    if (sh >= 40) return ~0ull >> 1;
    return sh >= 0 ? (mant << sh) : (sh > -64 ? (mant >> (-sh)) : 0ull);
}

struct SparseArgs {
    const int32_t *accept_len, *ids, *row_status;
    const float *probs, *tail, *q, *u;
    int B, K, V, k;
    int32_t *token, *status;
};

// first index i in sid[0, n) with sid[i] >= x
__device__ __forceinline__ int lower_bound_id(const int *sid, int n, int x) {
    int lo = 0, hi = n;
    while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (sid[mid] < x) lo = mid + 1;
        else hi = mid;
    }
    return lo;
}

// q at ids [x0, x0 + SEPT) (0 past V)
template <bool VEC>
__device__ __forceinline__ void load_q(const float *qr, int V, int x0, float (&qv)[SEPT]) {
    if (VEC && x0 + SEPT <= V) {
        const uint4 w0 = ldg16(qr + x0), w1 = ldg16(qr + x0 + 4);
        qv[0] = __uint_as_float(w0.x); qv[1] = __uint_as_float(w0.y);
        qv[2] = __uint_as_float(w0.z); qv[3] = __uint_as_float(w0.w);
        qv[4] = __uint_as_float(w1.x); qv[5] = __uint_as_float(w1.y);
        qv[6] = __uint_as_float(w1.z); qv[7] = __uint_as_float(w1.w);
    } else {
#pragma unroll
        for (int e = 0; e < SEPT; ++e) qv[e] = x0 + e < V ? __ldg(qr + x0 + e) : 0.0f;
    }
}

template <bool VEC>
__global__ void __cluster_dims__(SCL, 1, 1) __launch_bounds__(NTS) k_resample_sparse(SparseArgs a) {
    namespace cg = cooperative_groups;
    __shared__ unsigned long long skey[SPAY];  // id << 32 | entry (all ones: invalid id)
    __shared__ int sid[SPAY];                  // valid payload ids, ascending
    __shared__ int sidx[SPAY];                 // their payload entries
    __shared__ unsigned long long sw[SPAY];    // their weights (2^-52 units)
    __shared__ unsigned long long tsum[(STILES + SCL - 1) / SCL];  // this CTA's tiles
    __shared__ unsigned long long red[NTS / 32];
    __shared__ unsigned long long red4[TPI][NTS / 32];
    __shared__ float redh[NTS / 32], redl[NTS / 32];
    __shared__ float s_ph, s_pl;               // this CTA's share of q_rest (read by the cluster)
    __shared__ int s_pbad;
    __shared__ int s_n, s_bad, s_tok, s_tile;
    __shared__ float s_gam;
    __shared__ unsigned long long s_thr, s_base, s_R;
    cg::cluster_group cl = cg::this_cluster();
    const int rank = (int)cl.block_rank();
    const int b = blockIdx.x / SCL, tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    const int R1 = a.K + 1;
    const int pi = a.accept_len[b];
    const bool bad_row = pi < 0 || pi > a.K || (a.row_status[(size_t)b * R1 + pi] & ACES_ROW_NONFINITE);
    const size_t row = (size_t)b * R1 + (bad_row ? 0 : pi);
    const float tau = a.tail[row];
    const float *qr = (!bad_row && pi < a.K) ? a.q + ((size_t)b * a.K + pi) * a.V : nullptr;
    // The whole cluster takes part only when the tail may be spread (pi < K,
    // tau > 0): every CTA then decides the same way from the same inputs, so
    // all of them reach every cluster barrier.  Otherwise rank 0 works alone.
    const bool cluster_work = qr != nullptr && tau > 0.0f;
    if (!cluster_work && rank != 0) return;
    if (bad_row) {
        if (tid == 0) {
            a.token[b] = -1;
            a.status[b] = ACES_ROW_NONFINITE;
        }
        return;
    }
    const int32_t *I = a.ids + row * a.k;
    const float *P = a.probs + row * a.k;
    const int V = a.V;

    // ---- 1. payload sorted by id, weights on it ----
    // The valid entries (0 <= id < V) are ordered by (id, entry) by direct
    // rank counting: one pass, no barrier stages.
    if (tid == 0) {
        s_n = 0;
        s_bad = 0;
        s_tok = -1;
        s_tile = -1;
        s_gam = 0.0f;
    }
    for (int j = tid; j < a.k; j += NTS) {
        unsigned long long key = ~0ull;  // invalid: after every valid key
        const int x = I[j];
        if (x >= 0 && x < V) key = ((unsigned long long)x << 32) | (unsigned long long)j;
        skey[j] = key;
    }
    __syncthreads();
    for (int j = tid; j < a.k; j += NTS) {
        const unsigned long long key = skey[j];
        if (key == ~0ull) continue;
        int rank = 0;
        for (int i = 0; i < a.k; ++i) rank += skey[i] < key;
        if (ACES_IN(rank, SPAY)) {
            sid[rank] = (int)(key >> 32);
            sidx[rank] = (int)(key & 0xFFFFFFFFull);
        }
        atomicAdd(&s_n, 1);
    }
    __syncthreads();
    const int n = s_n;
    for (int i = tid; i < n; i += NTS) {
        const int x = sid[i], j = sidx[i];
        float w = fmaxf(P[j], 0.0f);
        if (qr && ACES_IN(x, V)) {
            const float qx = __ldg(qr + x);
            if (!(qx >= 0.0f)) s_bad = 1;
            w = fmaxf(P[j] - qx, 0.0f);
        }
        sw[i] = to_fx52(w);
    }
    __syncthreads();
    if (s_bad || n == 0) {  // the same in every CTA of the cluster
        if (rank == 0 && tid == 0) {
            a.token[b] = -1;
            a.status[b] = s_bad ? ACES_ROW_BAD_Q : 0;
        }
        return;
    }

    // ---- 2. the tail, spread like the draft (pi < K, tau > 0): the cluster ----
    const int ntile = (V + STILE - 1) / STILE;  // 2048-id tiles
    const int per = (ntile + SCL - 1) / SCL;     // tiles of each CTA
    const int t_lo = rank * per < ntile ? rank * per : ntile;
    const int t_hi = t_lo + per < ntile ? t_lo + per : ntile;
    bool spread = false;
    if (cluster_work) {
        float hi = 0.0f, lo = 0.0f;  // compensated sum of q outside the payload
        int bad = 0;
        for (int t0 = t_lo; t0 < t_hi; t0 += TPI) {  // TPI tiles' loads in flight
            float qv[TPI][SEPT];
#pragma unroll
            for (int h = 0; h < TPI; ++h) {
                const int x0 = (t0 + h) * STILE + tid * SEPT;
                if (t0 + h < t_hi && x0 < V) load_q<VEC>(qr, V, x0, qv[h]);
            }
#pragma unroll
            for (int h = 0; h < TPI; ++h) {
                const int x0 = (t0 + h) * STILE + tid * SEPT;
                if (t0 + h >= t_hi || x0 >= V) break;
                int j = lower_bound_id(sid, n, x0);
#pragma unroll
                for (int e = 0; e < SEPT; ++e) {
                    const int x = x0 + e;
                    if (x >= V) break;
                    const float qx = qv[h][e];
                    if (!(qx >= 0.0f)) bad = 1;
                    while (j < n && sid[j] < x) ++j;
                    if (j < n && sid[j] == x) continue;
                    const float t = hi + qx;
                    if (fabsf(hi) >= fabsf(qx)) lo += (hi - t) + qx;
                    else lo += (qx - t) + hi;
                    hi = t;
                }
            }
        }
        if (bad) s_bad = 1;
        for (int o = 16; o > 0; o >>= 1) {
            const float h2 = __shfl_xor_sync(0xffffffffu, hi, o);
            const float l2 = __shfl_xor_sync(0xffffffffu, lo, o);
            const float sm = hi + h2;
            const float bb = sm - hi;
            lo = lo + l2 + ((hi - (sm - bb)) + (h2 - bb));
            hi = sm;
        }
        if (lane == 0) {
            redh[wid] = hi;
            redl[wid] = lo;
        }
        __syncthreads();
        if (tid == 0) {
            float h = 0.0f, l = 0.0f;
            for (int i = 0; i < NTS / 32; ++i) {
                const float sm = h + redh[i];
                const float bb = sm - h;
                l = l + redl[i] + ((h - (sm - bb)) + (redh[i] - bb));
                h = sm;
            }
            s_ph = h;
            s_pl = l;
            s_pbad = s_bad;
        }
        cl.sync();  // every CTA's share is written
        if (tid == 0) {  // every CTA sums the shares in rank order: the same value everywhere
            double qrest = 0.0;
            int anybad = 0;
            for (int j = 0; j < SCL; ++j) {
                qrest += (double)*cl.map_shared_rank(&s_ph, j) + (double)*cl.map_shared_rank(&s_pl, j);
                anybad |= *cl.map_shared_rank(&s_pbad, j);
            }
            const double g = qrest > 0.0 ? (double)tau / qrest - 1.0 : 0.0;
            s_gam = g > 0.0 ? (float)g : 0.0f;
            s_bad = anybad;
        }
        cl.sync();  // the shares are read before any CTA moves on or exits
        if (s_bad) {
            if (rank == 0 && tid == 0) {
                a.token[b] = -1;
                a.status[b] = ACES_ROW_BAD_Q;
            }
            return;
        }
        spread = s_gam > 0.0f;
        if (!spread && rank != 0) return;
    }

    // ---- 3. the draw ----
    if (spread) {
        const float gam = s_gam;
        // weight of each of this CTA's tiles: q * gam outside the payload, sw on it
        for (int t0 = t_lo; t0 < t_hi; t0 += TPI) {
            float qv[TPI][SEPT];
#pragma unroll
            for (int h = 0; h < TPI; ++h) {
                const int x0 = (t0 + h) * STILE + tid * SEPT;
                if (t0 + h < t_hi && x0 < V) load_q<VEC>(qr, V, x0, qv[h]);
            }
            unsigned long long loc[TPI];
#pragma unroll
            for (int h = 0; h < TPI; ++h) {
                const int x0 = (t0 + h) * STILE + tid * SEPT;
                loc[h] = 0ull;
                if (t0 + h >= t_hi || x0 >= V) continue;
                int j = lower_bound_id(sid, n, x0);
#pragma unroll
                for (int e = 0; e < SEPT; ++e) {
                    const int x = x0 + e;
                    if (x >= V) break;
                    while (j < n && sid[j] < x) ++j;
                    loc[h] += (j < n && sid[j] == x) ? sw[j] : to_fx52(qv[h][e] * gam);
                }
            }
#pragma unroll
            for (int h = 0; h < TPI; ++h) loc[h] = warp_sum(loc[h]);
            if (lane == 0)
#pragma unroll
                for (int h = 0; h < TPI; ++h) red4[h][wid] = loc[h];
            __syncthreads();
            if (tid < TPI && t0 + tid < t_hi) {
                unsigned long long ts = 0ull;
                for (int i = 0; i < NTS / 32; ++i) ts += red4[tid][i];
                tsum[t0 + tid - t_lo] = ts;
            }
            __syncthreads();
        }
        cl.sync();  // every CTA's tile weights are written
        if (tid == 0) {  // the same walk over all tiles in every CTA
            unsigned long long tot = 0ull;
            for (int j = 0; j < SCL; ++j) {
                const int lo_j = j * per < ntile ? j * per : ntile;
                const int hi_j = lo_j + per < ntile ? lo_j + per : ntile;
                const unsigned long long *rt = cl.map_shared_rank(tsum, j);
                for (int t = lo_j; t < hi_j; ++t) tot += rt[t - lo_j];
            }
            s_R = tot;
            s_tile = -1;
            if (tot > 0ull) {
                const unsigned long long thr = floor_u_times(a.u[(size_t)b * R1 + a.K], tot);
                unsigned long long base = 0ull;
                int tt = ntile - 1;
                bool found = false;
                for (int j = 0; j < SCL && !found; ++j) {
                    const int lo_j = j * per < ntile ? j * per : ntile;
                    const int hi_j = lo_j + per < ntile ? lo_j + per : ntile;
                    const unsigned long long *rt = cl.map_shared_rank(tsum, j);
                    for (int t = lo_j; t < hi_j; ++t) {
                        if (base + rt[t - lo_j] > thr) {
                            tt = t;
                            found = true;
                            break;
                        }
                        base += rt[t - lo_j];
                    }
                }
                if (tt >= t_lo && tt < t_hi) s_tile = tt;
                s_base = base;
                s_thr = thr;
            }
        }
        cl.sync();  // the tile weights are read before any CTA exits
        if (s_R == 0ull) {  // nothing above 2^-52: rank 0 draws on the payload
            spread = false;
            if (rank != 0) return;
        } else if (s_tile < 0) {
            return;  // another CTA holds the draw
        }
    }
    if (spread) {
        const float gam = s_gam;
        // rescan the tile holding the draw
        const int x0 = s_tile * STILE + tid * SEPT;
        unsigned long long wv[SEPT];
        unsigned long long loc = 0ull;
        float qv[SEPT];
        if (x0 < V) load_q<VEC>(qr, V, x0, qv);
        int j = x0 < V ? lower_bound_id(sid, n, x0) : n;
#pragma unroll
        for (int e = 0; e < SEPT; ++e) {
            const int x = x0 + e;
            wv[e] = 0ull;
            if (x < V) {
                while (j < n && sid[j] < x) ++j;
                wv[e] = (j < n && sid[j] == x) ? sw[j] : to_fx52(qv[e] * gam);
            }
            loc += wv[e];
        }
        unsigned long long tot;
        const unsigned long long ex = block_exscan_n<NTS>(loc, red, &tot);
        const unsigned long long thr = s_thr;
        unsigned long long c = s_base + ex;
        if (c <= thr && thr < c + loc) {
#pragma unroll
            for (int e = 0; e < SEPT; ++e) {
                c += wv[e];
                if (c > thr) {
                    s_tok = x0 + e;
                    break;
                }
            }
        }
        __syncthreads();
    } else {
        // weights on the payload only (ascending id): one entry per thread
        unsigned long long w = tid < n ? sw[tid] : 0ull;
        unsigned long long tot;
        unsigned long long ex = block_exscan_n<NTS>(w, red, &tot);
        if (tot == 0ull) {  // p^ <= q wherever it is known: draw from p^ on the payload
            __syncthreads();
            if (tid < n) sw[tid] = to_fx52(fmaxf(P[sidx[tid]], 0.0f));
            __syncthreads();
            w = tid < n ? sw[tid] : 0ull;
            ex = block_exscan_n<NTS>(w, red, &tot);
        }
        if (tot > 0ull) {
            const unsigned long long thr = floor_u_times(a.u[(size_t)b * R1 + a.K], tot);
            if (ex <= thr && thr < ex + w) s_tok = sid[tid];
        }
        __syncthreads();
    }
    if (tid == 0) {
        a.token[b] = s_tok;
        a.status[b] = 0;
    }
}

cudaError_t launch_resample_sparse(const int32_t *accept_len, const int32_t *ids, const float *probs,
                                   const float *tail, const int32_t *row_status, const float *q,
                                   const float *u, int B, int K, int V, int k, int32_t *token,
                                   int32_t *status, bool vec, cudaStream_t s) {
    SparseArgs a;
    a.accept_len = accept_len;
    a.ids = ids;
    a.row_status = row_status;
    a.probs = probs;
    a.tail = tail;
    a.q = q;
    a.u = u;
    a.B = B;
    a.K = K;
    a.V = V;
    a.k = k;
    a.token = token;
    a.status = status;
    if (vec) k_resample_sparse<true><<<B * SCL, NTS, 0, s>>>(a);
    else k_resample_sparse<false><<<B * SCL, NTS, 0, s>>>(a);
    return cudaGetLastError();
}

#ifdef ACES_CHECKED
cudaError_t check_take_resample(unsigned long long out[3]) { return check_take(out); }
#endif

}  // namespace aces
