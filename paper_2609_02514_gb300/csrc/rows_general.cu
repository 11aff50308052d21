// Exact general row kernel of the AceSpec cloud step (Sec. III-B; Sec. II-A
// modified rejection sampling; Sec. V-C payload).  It takes every row that
// the fast kernel cannot certify (and every row when the logits are not
// 16-byte aligned): exact radix selection over the 64-bit order value
// O = key(z) << 32 | (2^32 - 1 - id), 8 bits per pass, with masses in 2^-40
// fixed point so that every partial sum is exact and order-independent.
// One CTA of 512 threads per row; a persistent grid walks the list of rows
// handed over by the fast kernel.
#include <climits>

#include "common.cuh"

namespace aces {

// ---------------------------------------------------------------------------
// Row epilogue shared by both row kernels: payload, tail, accept test, stats.
// `sorted` holds the first L ids of the nucleus in order (descending order
// values).  Called by all threads of the CTA.
template <int DT>
__device__ void finish_row(const RowArgs &a, int r, const char *row, float kref, double S_nuc,
                           unsigned long long cut, int flags, const unsigned long long *sorted,
                           int L, double *redd) {
    const int tid = threadIdx.x;
    // same formulas as the fast row kernel, so a row gets bit-identical
    // outputs whichever kernel finishes it: p = e * (float)(1/S_nuc), and the
    // tail from the exact fixed-point sum of the payload masses
    const float inv_S = (float)(1.0 / S_nuc);
    unsigned long long loc = 0ull;
    if (a.k > 0) {
        for (int j = tid; j < a.k; j += NT) {
            size_t o = (size_t)r * a.k + j;
            if (j < L) {
                unsigned long long ov = sorted[j];
                float e = ex2(fmaf(order_value(ov), a.c, -kref));
                loc += to_fx(e);
                a.topk_ids[o] = (int32_t)order_id(ov);
                a.topk_probs[o] = e * inv_S;
            } else {
                a.topk_ids[o] = -1;
                a.topk_probs[o] = 0.0f;
            }
        }
    }
    __shared__ unsigned long long s_redl[NWARP];
    const unsigned long long tot = block_reduce(loc, s_redl, SumU64());
    if (tid != 0) return;
    if (a.k > 0) a.tail[r] = (float)((S_nuc - (double)tot / (double)FX_SCALE) / S_nuc);
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
                double p = in ? (double)ex2(fmaf(v, a.c, -kref)) / S_nuc : 0.0;
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
    s.kref = kref;
    s.c = a.c;
    s.S_nuc = S_nuc;
    s.cut = cut;
    s.flags = flags;
    s.nnuc = -1;  // the residual step scans the row
    a.ws.stats[r] = s;
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
__device__ unsigned long long radix_select(const char *row, int V, float kref, float c, int mode,
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
            if (mode == 0 || want_S) atomicAdd(&st->mass[d], to_fx(ex2(fmaf(v, c, -kref))));
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
        const float kref = ceilf(m * a.c);  // masses are 2^(z*c - kref) <= 1
        const unsigned long long n_fin = block_reduce(nfin, redu, SumU64());
        if (s_bad || n_fin == 0ull || !(kref < 1e30f)) {
            nonfinite_row<NT>(a, r);
            __syncthreads();
            continue;
        }
        const bool all_in = a.top_p >= 1.0f;
        unsigned long long cut = 0ull;
        double S_nuc;
        unsigned long long n_nuc;
        if (!all_in) {
            cut = radix_select<DT, VEC>(row, a.V, kref, a.c, 0, (double)a.top_p, 0u, true, &st);
            S_nuc = (double)(st.above + st.found) / (double)FX_SCALE;
            n_nuc = (unsigned long long)st.above_cnt + 1ull;
        } else {
            unsigned long long sfx = 0ull;
            for_each_elem<DT, VEC>(row, a.V, [&](int, float v) {
                if (v > -INFINITY) sfx += to_fx(ex2(fmaf(v, a.c, -kref)));
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
            lim = radix_select<DT, VEC>(row, a.V, kref, a.c, 1, 0.0, (unsigned)a.k, false, &st);
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
        finish_row<DT>(a, r, row, kref, S_nuc, cut, all_in ? RS_ALL_IN : 0, buf, L, redd);
        __syncthreads();
    }
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

}  // namespace aces
