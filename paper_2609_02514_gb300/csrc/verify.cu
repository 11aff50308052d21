// Verification and sparse-payload kernels of the AceSpec cloud step
// (Sec. III-B: accept test, first rejection pi, packaging of the target
// distribution; Sec. II-A: modified rejection sampling; Sec. V-C: compact
// downlink payload).
//
// Row kernels (one CTA per target row r = b*(K+1)+i):
//   k_rows_fast     one HBM pass (online max / exp-sum and a per-group max
//                   sketch kept in shared memory), then an exact selection
//                   over the few ids the sketch proves can matter.
//   k_rows_general  exact radix selection over the 64-bit (logit, id) order
//                   with fixed-point masses; takes every row the fast path
//                   cannot certify.
// Sequence kernel (one CTA per sequence):
//   k_resolve       first rejection pi by a scan of the accept bits, then the
//                   residual (or bonus) inverse-CDF draw over row pi in
//                   vocabulary order with exact integer prefix sums.
#include <climits>

#include "common.cuh"

namespace aces {

// ---------------------------------------------------------------------------
// Row epilogue shared by both row kernels: payload, tail, accept test, stats.
// `sorted` holds the first L ids of the nucleus in order (descending order
// values).  Called by all threads of the CTA.
template <int DT>
__device__ void finish_row(const RowArgs &a, int r, const char *row, float m, double S_nuc,
                           unsigned long long cut, int flags, const unsigned long long *sorted,
                           int L, double *redd) {
    const int tid = threadIdx.x;
    double loc = 0.0;
    if (a.k > 0) {
        for (int j = tid; j < a.k; j += NT) {
            size_t o = (size_t)r * a.k + j;
            if (j < L) {
                unsigned long long ov = sorted[j];
                float e = ex2((order_value(ov) - m) * a.c);
                loc += (double)e;
                a.topk_ids[o] = (int32_t)order_id(ov);
                a.topk_probs[o] = (float)((double)e / S_nuc);
            } else {
                a.topk_ids[o] = -1;
                a.topk_probs[o] = 0.0f;
            }
        }
    }
    double tot = block_reduce(loc, redd, SumD());
    if (tid != 0) return;
    if (a.k > 0) a.tail[r] = (float)((S_nuc - tot) / S_nuc);
    int st = 0;
    if (a.K > 0) {
        int b = r / (a.K + 1), i = r % (a.K + 1);
        if (i < a.K) {
            int x = a.xt[(size_t)b * a.K + i];
            int accept = 0;
            if (x < 0 || x >= a.V) {
                st |= ACES_ROW_BAD_Q;
            } else {
                float v = Elem<DT>::load1(row, x);
                bool in = (flags & RS_ALL_IN) ? (v > -INFINITY) : (order_val(fkey(v), (uint32_t)x) >= cut);
                double p = in ? (double)ex2((v - m) * a.c) / S_nuc : 0.0;
                float qx = a.q[((size_t)b * a.K + i) * a.V + x];
                if (!(qx > 0.0f)) {
                    st |= ACES_ROW_BAD_Q;
                } else {
                    double ratio = p / (double)qx;
                    accept = (double)a.u[(size_t)b * (a.K + 1) + i] < fmin(1.0, ratio);
                }
            }
            a.ws.acc[(size_t)b * a.K + i] = accept;
        }
    }
    a.row_status[r] = st;
    RowStat s;
    s.m = m;
    s.c = a.c;
    s.S_nuc = S_nuc;
    s.cut = cut;
    s.flags = flags;
    s.pad = 0;
    a.ws.stats[r] = s;
}

// Outputs of a row whose logits are not a distribution.
__device__ void nonfinite_row(const RowArgs &a, int r) {
    const int tid = threadIdx.x;
    for (int j = tid; j < a.k; j += NT) {
        a.topk_ids[(size_t)r * a.k + j] = -1;
        a.topk_probs[(size_t)r * a.k + j] = 0.0f;
    }
    if (tid == 0) {
        if (a.k > 0) a.tail[r] = 1.0f;
        a.row_status[r] = ACES_ROW_NONFINITE;
        if (a.K > 0) {
            int b = r / (a.K + 1), i = r % (a.K + 1);
            if (i < a.K) a.ws.acc[(size_t)b * a.K + i] = 0;
        }
        RowStat s;
        s.m = 0.f;
        s.c = a.c;
        s.S_nuc = 1.0;
        s.cut = 0;
        s.flags = RS_NONFINITE;
        s.pad = 0;
        a.ws.stats[r] = s;
    }
}

// ---------------------------------------------------------------------------
// Fast path.  GC = 16-byte chunks per sketch group.
template <int DT, int GC>
__global__ void __launch_bounds__(NT, 2) k_rows_fast(RowArgs a) {
    using E = Elem<DT>;
    constexpr int EPC = E::EPC;
    extern __shared__ __align__(16) unsigned char smem[];
    uint32_t *sketch = reinterpret_cast<uint32_t *>(smem);
    unsigned long long *cand = reinterpret_cast<unsigned long long *>(smem + align16((size_t)a.ng * 4));
    __shared__ uint32_t bins[NBIN];
    __shared__ double redd[NWARP];
    __shared__ float redf[NWARP];
    __shared__ int s_ncand, s_nstar, s_bc;
    __shared__ double s_Snuc;

    const int r = blockIdx.x;
    const int tid = threadIdx.x;
    const char *row = reinterpret_cast<const char *>(a.logits) + (size_t)r * a.V * E::SIZE;
    const int nch = a.V / EPC;
    const uint32_t NI = E::NEG_INF_WORD;

    // ---- pass 1: online max and exp-sum, per-group max sketch ----
    float m_t = -FLT_MAX, s_t = 0.f, e_t = 0.f;
    constexpr int GPI = GC >= 4 ? 1 : 2;  // groups per iteration (4 loads in flight)
    for (int g0 = tid; g0 < a.ng; g0 += NT * GPI) {
        uint4 w[GPI][GC];
#pragma unroll
        for (int h = 0; h < GPI; ++h) {
            int g = g0 + h * NT;
#pragma unroll
            for (int j = 0; j < GC; ++j) {
                int cc = g * GC + j;
                w[h][j] = (g < a.ng && cc < nch) ? ldg16(row + (size_t)cc * 16) : make_uint4(NI, NI, NI, NI);
            }
        }
#pragma unroll
        for (int h = 0; h < GPI; ++h) {
            int g = g0 + h * NT;
            float gm = -INFINITY;
#pragma unroll
            for (int j = 0; j < GC; ++j)
#pragma unroll
                for (int e = 0; e < EPC; ++e) gm = fmaxf(gm, E::get(w[h][j], e));
            if (gm > m_t) {
                float sc = ex2((m_t - gm) * a.c);
                s_t *= sc;
                e_t *= sc;
                m_t = gm;
            }
            float gs = 0.f;
#pragma unroll
            for (int j = 0; j < GC; ++j) {
                float cs[EPC];
#pragma unroll
                for (int e = 0; e < EPC; ++e) cs[e] = ex2((E::get(w[h][j], e) - m_t) * a.c);
#pragma unroll
                for (int wdt = 1; wdt < EPC; wdt <<= 1)
#pragma unroll
                    for (int e = 0; e < EPC; e += 2 * wdt) cs[e] += cs[e + wdt];
                gs += cs[0];
            }
            float t = s_t + gs;
            if (fabsf(s_t) >= fabsf(gs)) e_t += (s_t - t) + gs;
            else e_t += (gs - t) + s_t;
            s_t = t;
            if (g < a.ng) sketch[g] = fkey(gm);
        }
    }
    const float m = block_reduce(m_t, redf, MaxF());
    const double S = block_reduce((double)(s_t + e_t) * (double)ex2((m_t - m) * a.c), redd, SumD());
    if (!(S > 0.0 && S < 1e300) || !(m < INFINITY)) {
        nonfinite_row(a, r);
        return;
    }
    const bool all_in = a.top_p >= 1.0f;

    // ---- sketch bins: groups by floor((m - gmax) / (T/8)) ----
    for (int i = tid; i < NBIN; i += NT) bins[i] = 0u;
    __syncthreads();
    for (int g = tid; g < a.ng; g += NT) {
        float d = (m - fkey_inv(sketch[g])) * a.inv_w;
        if (d < (float)NBIN) atomicAdd(&bins[(int)d], 1u);
    }
    __syncthreads();
    if (tid < 32) {
        // each lane owns 8 consecutive bins; the lower bound of a bin's mass
        // per group is exp(-(b+1)/8), shaded by 1e-5 for rounding
        constexpr int PER = NBIN / 32;
        double lb[PER];
        unsigned cn[PER];
        double lsum = 0.0;
        unsigned csum = 0;
#pragma unroll
        for (int j = 0; j < PER; ++j) {
            int b = tid * PER + j;
            cn[j] = bins[b];
            lb[j] = (double)cn[j] * (double)ex2(-(float)(b + 1) * (1.4426950408889634f / BIN_PER_T)) * (1.0 - 1e-5);
            lsum += lb[j];
            csum += cn[j];
        }
        double lpre = lsum;
        unsigned cpre = csum;
        for (int o = 1; o < 32; o <<= 1) {
            double t = __shfl_up_sync(0xffffffffu, lpre, o);
            unsigned c = __shfl_up_sync(0xffffffffu, cpre, o);
            if (tid >= o) {
                lpre += t;
                cpre += c;
            }
        }
        lpre -= lsum;
        cpre -= csum;
        const double target = (double)a.top_p * S * (1.0 + 1e-5);
        int hit = -1;
#pragma unroll
        for (int j = 0; j < PER; ++j) {
            lpre += lb[j];
            cpre += cn[j];
            bool ok = all_in ? (cpre >= (unsigned)a.k) : (lpre >= target);
            if (ok && hit < 0) hit = tid * PER + j;
        }
        unsigned bal = __ballot_sync(0xffffffffu, hit >= 0);
        int first = bal ? __ffs(bal) - 1 : -1;
        int bc = first >= 0 ? __shfl_sync(0xffffffffu, hit, first) : -1;
        if (tid == 0) {
            s_bc = bc;
            s_ncand = 0;
            s_nstar = INT_MAX;
        }
    }
    __syncthreads();
    const int bc = s_bc;
    bool fallback = bc < 0;

    // ---- candidates: every id whose bin is <= bc (re-read only flagged groups) ----
    int n = 0;
    if (!fallback) {
        const float lim = (float)(bc + 1);
        for (int g = tid; g < a.ng; g += NT) {
            if ((m - fkey_inv(sketch[g])) * a.inv_w < lim) {
#pragma unroll
                for (int j = 0; j < GC; ++j) {
                    int cc = g * GC + j;
                    if (cc < nch) {
                        uint4 w = ldg16(row + (size_t)cc * 16);
#pragma unroll
                        for (int e = 0; e < EPC; ++e) {
                            float v = E::get(w, e);
                            if ((m - v) * a.inv_w < lim) {
                                int pos = atomicAdd(&s_ncand, 1);
                                if (pos < CAND_CAP) cand[pos] = order_val(fkey(v), (uint32_t)(cc * EPC + e));
                            }
                        }
                    }
                }
            }
        }
        __syncthreads();
        n = s_ncand;
        fallback = n > CAND_CAP;
    }
    if (fallback) {
        if (tid == 0) {
            int pos = atomicAdd(a.ws.fb_count, 1);
            a.ws.fb_list[pos] = r;
        }
        return;
    }
    const int np = next_pow2(n < 2 ? 2 : n);
    for (int i = n + tid; i < np; i += NT) cand[i] = 0ull;
    __syncthreads();
    bitonic_sort_desc(cand, np);

    // ---- exact nucleus over the sorted candidates ----
    double S_nuc = S;
    unsigned long long cut = 0ull;
    int L;
    if (all_in) {
        L = n < a.k ? n : a.k;
    } else {
        const int per = (n + NT - 1) / NT;
        const int lo = tid * per, hi = min(n, lo + per);
        double loc = 0.0;
        for (int i = lo; i < hi; ++i) loc += (double)ex2((order_value(cand[i]) - m) * a.c);
        double tot;
        const double ex0 = block_exscan(loc, redd, &tot);
        const double target = (double)a.top_p * S;
        double cum = ex0;
        for (int i = lo; i < hi; ++i) {
            cum += (double)ex2((order_value(cand[i]) - m) * a.c);
            if (cum >= target) {
                atomicMin(&s_nstar, i);
                break;
            }
        }
        __syncthreads();
        const int nstar = s_nstar;
        if (nstar == INT_MAX) {  // candidates hold too little mass: exact general path
            if (tid == 0) {
                int pos = atomicAdd(a.ws.fb_count, 1);
                a.ws.fb_list[pos] = r;
            }
            return;
        }
        if (nstar >= lo && nstar < hi) {  // the owner of the crossing id sums up to it
            double c3 = ex0;
            for (int i = lo; i <= nstar; ++i) c3 += (double)ex2((order_value(cand[i]) - m) * a.c);
            s_Snuc = c3;
        }
        __syncthreads();
        S_nuc = s_Snuc;
        cut = cand[nstar];
        L = (nstar + 1) < a.k ? (nstar + 1) : a.k;
    }
    finish_row<DT>(a, r, row, m, S_nuc, cut, all_in ? RS_ALL_IN : 0, cand, L, redd);
}

// ---------------------------------------------------------------------------
// General path: exact radix selection over the 64-bit order value
// O = key(z) << 32 | (2^32 - 1 - id), 8 bits per pass, masses in 2^-40
// fixed point so that every partial sum is exact and order-independent.
template <int DT, bool VEC, class F>
__device__ __forceinline__ void for_each_elem(const char *row, int V, F f) {
    using E = Elem<DT>;
    if (VEC) {
        const int nch = V / E::EPC;
#pragma unroll 2
        for (int cc = threadIdx.x; cc < nch; cc += NT) {
            uint4 w = ldg16(row + (size_t)cc * 16);
#pragma unroll
            for (int e = 0; e < E::EPC; ++e) f(cc * E::EPC + e, E::get(w, e));
        }
    } else {
        for (int x = threadIdx.x; x < V; x += NT) f(x, E::load1(row, x));
    }
}

struct SelState {
    uint32_t cnt[256];
    unsigned long long mass[256];
    unsigned long long prefix;
    unsigned long long above;
    unsigned long long S_fx;
    unsigned long long found;
    unsigned above_cnt;
    int sel;
    unsigned sel_cnt;
    int done;
};

// One radix selection.  mode 0: first id where the cumulative mass reaches
// target_fx (as a double); mode 1: the kk-th id (1-based) by count.
// Returns the order value of the selected id; st->above / above_cnt hold the
// mass / count strictly before it; when want_S, st->S_fx gets the total mass.
template <int DT, bool VEC>
__device__ unsigned long long radix_select(const char *row, int V, float m, float c, int mode,
                                           double target, unsigned kk, bool want_S, SelState *st) {
    const int tid = threadIdx.x;
    if (tid == 0) {
        st->prefix = 0ull;
        st->above = 0ull;
        st->above_cnt = 0u;
        st->done = 0;
        st->S_fx = 0ull;
    }
    int nbits = 0;
    for (int s = 56; s >= 0; s -= 8) {
        // digits known in advance: the low 16 key bits of a bf16 value are 0,
        // and ids below 2^24 give 0xFF in bits 31..24 of (2^32 - 1 - id)
        int known = -1;
        if (DT == ACES_BF16 && (s == 40 || s == 32)) known = 0;
        if (s == 24) known = 0xFF;
        if (known >= 0) {
            if (tid == 0) st->prefix = (st->prefix << 8) | (unsigned long long)known;
            nbits += 8;
            __syncthreads();
            continue;
        }
        for (int i = tid; i < 256; i += NT) {
            st->cnt[i] = 0u;
            st->mass[i] = 0ull;
        }
        __syncthreads();
        const unsigned long long prefix = st->prefix;
        const int sh = 64 - nbits;
        for_each_elem<DT, VEC>(row, V, [&](int x, float v) {
            if (!(v > -INFINITY)) return;
            unsigned long long o = order_val(fkey(v), (uint32_t)x);
            if (nbits != 0 && (o >> sh) != prefix) return;
            int d = (int)((o >> s) & 255ull);
            atomicAdd(&st->cnt[d], 1u);
            if (mode == 0 || want_S) atomicAdd(&st->mass[d], to_fx(ex2((v - m) * c)));
        });
        __syncthreads();
        if (tid == 0) {
            if (nbits == 0) {
                unsigned long long S = 0ull;
                for (int d = 0; d < 256; ++d) S += st->mass[d];
                st->S_fx = S;
                if (mode == 0) target *= (double)S;  // target arrives as top_p
            }
            int sel = -1;
            int lowest = -1;
            for (int d = 255; d >= 0; --d) {
                if (st->cnt[d] == 0u) continue;
                lowest = d;
                bool hit = mode == 0 ? ((double)(st->above + st->mass[d]) >= target)
                                     : (st->above_cnt + st->cnt[d] >= kk);
                if (hit) {
                    sel = d;
                    break;
                }
                st->above += st->mass[d];
                st->above_cnt += st->cnt[d];
            }
            if (sel < 0) {  // target not reached (rounding at top_p ~ 1): take the last id
                sel = lowest;
                st->above -= st->mass[sel];
                st->above_cnt -= st->cnt[sel];
            }
            st->sel = sel;
            st->sel_cnt = st->cnt[sel];
            st->prefix = (st->prefix << 8) | (unsigned long long)sel;
            if (mode == 0) st->found = st->mass[sel];  // mass of the bin (of the id when unique)
        }
        __syncthreads();
        nbits += 8;
        if (st->sel_cnt == 1u && s > 0) {
            // a single id carries this prefix: fetch its full order value
            const unsigned long long pf = st->prefix;
            const int sh2 = 64 - nbits;
            for_each_elem<DT, VEC>(row, V, [&](int x, float v) {
                if (!(v > -INFINITY)) return;
                unsigned long long o = order_val(fkey(v), (uint32_t)x);
                if ((o >> sh2) == pf) st->prefix = o;
            });
            __syncthreads();
            break;
        }
    }
    return st->prefix;
}

template <int DT, bool VEC>
__global__ void __launch_bounds__(NT) k_rows_general(RowArgs a, int direct) {
    using E = Elem<DT>;
    __shared__ SelState st;
    __shared__ unsigned long long buf[ACES_MAX_TOPK];
    __shared__ double redd[NWARP];
    __shared__ float redf[NWARP];
    __shared__ unsigned long long redu[NWARP];
    __shared__ int s_bad;
    __shared__ int s_nbuf;
    const int tid = threadIdx.x;
    const int nrows = direct ? a.rows : *a.ws.fb_count;
    for (int idx = blockIdx.x; idx < nrows; idx += gridDim.x) {
        const int r = direct ? idx : a.ws.fb_list[idx];
        const char *row = reinterpret_cast<const char *>(a.logits) + (size_t)r * a.V * E::SIZE;
        // pass 0: max, finite count, invalid values
        if (tid == 0) s_bad = 0;
        __syncthreads();
        float mx = -INFINITY;
        unsigned long long nfin = 0;
        int bad = 0;
        for_each_elem<DT, VEC>(row, a.V, [&](int, float v) {
            if (v != v || v == INFINITY) bad = 1;
            if (v > -INFINITY) ++nfin;
            mx = fmaxf(mx, v);
        });
        if (bad) s_bad = 1;
        const float m = block_reduce(mx, redf, MaxF());
        const unsigned long long n_fin = block_reduce(nfin, redu, SumU64());
        if (s_bad || n_fin == 0ull) {
            nonfinite_row(a, r);
            __syncthreads();
            continue;
        }
        const bool all_in = a.top_p >= 1.0f;
        unsigned long long cut = 0ull;
        double S_nuc;
        unsigned long long n_nuc;
        if (!all_in) {
            cut = radix_select<DT, VEC>(row, a.V, m, a.c, 0, (double)a.top_p, 0u, true, &st);
            S_nuc = (double)(st.above + st.found) / (double)FX_SCALE;
            n_nuc = (unsigned long long)st.above_cnt + 1ull;
        } else {
            unsigned long long sfx = 0ull;
            for_each_elem<DT, VEC>(row, a.V, [&](int, float v) {
                if (v > -INFINITY) sfx += to_fx(ex2((v - m) * a.c));
            });
            S_nuc = (double)block_reduce(sfx, redu, SumU64()) / (double)FX_SCALE;
            n_nuc = n_fin;
        }
        __syncthreads();
        // the payload boundary: the last nucleus id, or the k-th id when the
        // nucleus is longer than the payload
        unsigned long long lim = all_in ? 0ull : cut;
        int L = (int)(n_nuc < (unsigned long long)a.k ? n_nuc : (unsigned long long)a.k);
        if (a.k > 0 && n_nuc > (unsigned long long)a.k)
            lim = radix_select<DT, VEC>(row, a.V, m, a.c, 1, 0.0, (unsigned)a.k, false, &st);
        __syncthreads();
        // collect the payload ids (order value >= lim)
        if (tid == 0) s_nbuf = 0;
        __syncthreads();
        if (a.k > 0) {
            for_each_elem<DT, VEC>(row, a.V, [&](int x, float v) {
                if (!(v > -INFINITY)) return;
                unsigned long long o = order_val(fkey(v), (uint32_t)x);
                if (o >= lim) {
                    int pos = atomicAdd(&s_nbuf, 1);
                    if (pos < ACES_MAX_TOPK) buf[pos] = o;
                }
            });
        }
        __syncthreads();
        const int nb = min(s_nbuf, ACES_MAX_TOPK);
        const int np = next_pow2(nb < 2 ? 2 : nb);
        for (int i = nb + tid; i < np; i += NT) buf[i] = 0ull;
        __syncthreads();
        bitonic_sort_desc(buf, np);
        if (L > nb) L = nb;
        finish_row<DT>(a, r, row, m, S_nuc, cut, all_in ? RS_ALL_IN : 0, buf, L, redd);
        __syncthreads();
    }
}

// ---------------------------------------------------------------------------
// Sequence kernel: pi, accept_len, and the residual / bonus token.
constexpr int EPT = 8;                 // consecutive ids per thread in a tile
constexpr int TILE = NT * EPT;
constexpr int MAX_TILES = (ACES_MAX_V + TILE - 1) / TILE;


// r_fx of ids [x0, x0 + EPT) into out[]; sets *bad on a NaN / negative q.
template <int DT, bool VEC>
__device__ __forceinline__ void resid_fx(const char *zrow, const float *qrow, int V, int x0,
                                         const RowStat &rs, float inv_S, int mode,
                                         unsigned long long out[EPT], int *bad) {
    using E = Elem<DT>;
    float zv[EPT], qv[EPT];
    if (VEC && x0 + EPT <= V) {
        if (DT == ACES_BF16) {
            uint4 w = ldg16(zrow + (size_t)x0 * 2);
#pragma unroll
            for (int e = 0; e < EPT; ++e) zv[e] = E::get(w, e);
        } else {
            uint4 w0 = ldg16(zrow + (size_t)x0 * 4), w1 = ldg16(zrow + (size_t)x0 * 4 + 16);
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                zv[e] = Elem<ACES_F32>::get(w0, e);
                zv[e + 4] = Elem<ACES_F32>::get(w1, e);
            }
        }
        if (qrow) {
            uint4 w0 = ldg16(qrow + x0), w1 = ldg16(qrow + x0 + 4);
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                qv[e] = Elem<ACES_F32>::get(w0, e);
                qv[e + 4] = Elem<ACES_F32>::get(w1, e);
            }
        }
    } else {
#pragma unroll
        for (int e = 0; e < EPT; ++e) {
            int x = x0 + e;
            zv[e] = x < V ? E::load1(zrow, x) : -INFINITY;
            qv[e] = (qrow && x < V) ? __ldg(qrow + x) : 0.0f;
        }
    }
#pragma unroll
    for (int e = 0; e < EPT; ++e) {
        const int x = x0 + e;
        const float v = zv[e];
        bool in = x < V && ((rs.flags & RS_ALL_IN) ? (v > -INFINITY)
                                                   : (order_val(fkey(v), (uint32_t)x) >= rs.cut));
        float p = in ? ex2((v - rs.m) * rs.c) * inv_S : 0.0f;
        float rr = p;
        if (qrow && mode == 0 && x < V) {
            float qx = qv[e];
            if (!(qx >= 0.0f)) *bad = 1;
            rr = fmaxf(p - qx, 0.0f);
        }
        out[e] = x < V ? to_fx(rr) : 0ull;
    }
}

template <int DT, bool VEC>
__global__ void __launch_bounds__(NT) k_resolve(ResolveArgs a) {
    using E = Elem<DT>;
    __shared__ unsigned long long tile_sum[MAX_TILES];
    __shared__ unsigned long long redu[NWARP];
    __shared__ int s_pi, s_bad, s_tile, s_tok;
    __shared__ unsigned long long s_base, s_thr;
    const int b = blockIdx.x, tid = threadIdx.x;
    if (tid == 0) {
        int pi = a.K;
        for (int i = 0; i < a.K; ++i)
            if (!a.ws.acc[(size_t)b * a.K + i]) {
                pi = i;
                break;
            }
        s_pi = pi;
        s_bad = 0;
        s_tok = -1;
        a.accept_len[b] = pi;
    }
    __syncthreads();
    const int pi = s_pi;
    const int r = b * (a.K + 1) + pi;
    const RowStat rs = a.ws.stats[r];
    if (rs.flags & RS_NONFINITE) {
        if (tid == 0) a.out_token[b] = -1;
        return;
    }
    const char *zrow = reinterpret_cast<const char *>(a.logits) + (size_t)r * a.V * E::SIZE;
    const float *qrow = pi < a.K ? a.q + ((size_t)b * a.K + pi) * a.V : nullptr;
    const float inv_S = (float)(1.0 / rs.S_nuc);
    const int ntiles = (a.V + TILE - 1) / TILE;
    int mode = 0;
    unsigned long long R = 0ull;
    for (int pass = 0; pass < 2; ++pass) {
        int bad = 0;
        for (int t = 0; t < ntiles; ++t) {
            unsigned long long v[EPT];
            resid_fx<DT, VEC>(zrow, qrow, a.V, t * TILE + tid * EPT, rs, inv_S, mode, v, &bad);
            unsigned long long loc = 0ull;
#pragma unroll
            for (int e = 0; e < EPT; ++e) loc += v[e];
            unsigned long long ts = block_reduce(loc, redu, SumU64());
            if (tid == 0) tile_sum[t] = ts;
        }
        if (bad) s_bad = 1;
        __syncthreads();
        if (s_bad) {
            if (tid == 0) {
                a.out_token[b] = -1;
                a.row_status[r] |= ACES_ROW_BAD_Q;
            }
            return;
        }
        R = 0ull;
        for (int t = 0; t < ntiles; ++t) R += tile_sum[t];
        if (R > 0ull) break;
        if (mode == 1) {  // no mass anywhere (cannot happen for a finite row)
            if (tid == 0) a.out_token[b] = -1;
            return;
        }
        mode = 1;  // p <= q everywhere: draw from p itself
        __syncthreads();
    }
    if (tid == 0) {
        // thr = floor(u * R) exactly: u = M * 2^E with a 24-bit integer M
        float uu = a.u[(size_t)b * (a.K + 1) + a.K];
        int ex;
        float fr = frexpf(uu, &ex);                  // uu = fr * 2^ex, fr in [0.5, 1)
        unsigned long long M = (unsigned long long)ldexpf(fr, 24);
        int sh = 24 - ex;                            // uu = M / 2^sh
        unsigned long long lo = M * R;
        unsigned long long hi = __umul64hi(M, R);
        unsigned long long thr;
        if (sh >= 128) thr = 0ull;
        else if (sh >= 64) thr = hi >> (sh - 64);
        else if (sh == 0) thr = lo;
        else thr = (lo >> sh) | (hi << (64 - sh));
        if (!(uu > 0.0f)) thr = 0ull;
        if (thr >= R) thr = R - 1ull;
        unsigned long long base = 0ull;
        int tt = ntiles - 1;
        for (int t = 0; t < ntiles; ++t) {
            if (base + tile_sum[t] > thr) {
                tt = t;
                break;
            }
            base += tile_sum[t];
        }
        s_tile = tt;
        s_base = base;
        s_thr = thr;
    }
    __syncthreads();
    const int tt = s_tile;
    unsigned long long v[EPT];
    int bad = 0;
    resid_fx<DT, VEC>(zrow, qrow, a.V, tt * TILE + tid * EPT, rs, inv_S, mode, v, &bad);
    unsigned long long loc = 0ull;
#pragma unroll
    for (int e = 0; e < EPT; ++e) loc += v[e];
    unsigned long long tot;
    unsigned long long ex = block_exscan(loc, redu, &tot);
    const unsigned long long thr = s_thr;
    unsigned long long cum = s_base + ex;
    if (cum <= thr && thr < cum + loc) {
#pragma unroll
        for (int e = 0; e < EPT; ++e) {
            cum += v[e];
            if (cum > thr) {
                s_tok = tt * TILE + tid * EPT + e;
                break;
            }
        }
    }
    __syncthreads();
    if (tid == 0) a.out_token[b] = s_tok;
}

// ---------------------------------------------------------------------------
// host launchers
template <int DT>
static cudaError_t launch_fast_dt(const RowArgs &a, int gc, size_t smem, cudaStream_t s) {
    void (*fn)(RowArgs) = nullptr;
    switch (gc) {
        case 2: fn = k_rows_fast<DT, 2>; break;
        case 4: fn = k_rows_fast<DT, 4>; break;
        case 8: fn = k_rows_fast<DT, 8>; break;
        default:
            if (DT == ACES_F32) fn = k_rows_fast<ACES_F32, 16>;
            break;
    }
    if (!fn) return cudaErrorInvalidValue;
    cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    fn<<<a.rows, NT, smem, s>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_rows_fast(const RowArgs &a, int dt, int gc, size_t smem, cudaStream_t s) {
    return dt == ACES_BF16 ? launch_fast_dt<ACES_BF16>(a, gc, smem, s) : launch_fast_dt<ACES_F32>(a, gc, smem, s);
}

cudaError_t launch_rows_general(const RowArgs &a, int dt, bool vec, int direct, int grid, cudaStream_t s) {
    if (dt == ACES_BF16) {
        if (vec) k_rows_general<ACES_BF16, true><<<grid, NT, 0, s>>>(a, direct);
        else k_rows_general<ACES_BF16, false><<<grid, NT, 0, s>>>(a, direct);
    } else {
        if (vec) k_rows_general<ACES_F32, true><<<grid, NT, 0, s>>>(a, direct);
        else k_rows_general<ACES_F32, false><<<grid, NT, 0, s>>>(a, direct);
    }
    return cudaGetLastError();
}

cudaError_t launch_resolve(const ResolveArgs &a, int dt, bool vec, cudaStream_t s) {
    if (dt == ACES_BF16) {
        if (vec) k_resolve<ACES_BF16, true><<<a.B, NT, 0, s>>>(a);
        else k_resolve<ACES_BF16, false><<<a.B, NT, 0, s>>>(a);
    } else {
        if (vec) k_resolve<ACES_F32, true><<<a.B, NT, 0, s>>>(a);
        else k_resolve<ACES_F32, false><<<a.B, NT, 0, s>>>(a);
    }
    return cudaGetLastError();
}

}  // namespace aces
