// Exact general row kernel of the AceSpec cloud step (Sec. III-B; Sec. II-A
// modified rejection sampling; Sec. V-C payload).  It takes every row that
// the fast kernel cannot certify (and every row when the logits are not
// 16-byte aligned).  Masses are in 2^-40 fixed point, so every partial sum
// is exact and order-independent.  One CTA of 512 threads per row; a
// persistent grid walks the list of rows handed over by the fast kernel.
//   value histogram  (aligned bfloat16 rows) ids counted per bfloat16 value
//                below the max, the crossing and payload values found by a
//                prefix scan, their ids collected and ranked: two row reads;
//   binned path  exact per-bin masses over bins of distance below the max
//                (warp-aggregated shared-memory atomics, farther elements
//                summed in registers), then the crossing bin and the payload
//                bins are collected and ordered: three to four row reads;
//   radix path   when a needed bin is too full or too far: exact radix
//                selection over the 64-bit order value
//                O = key(z) << 32 | (2^32 - 1 - id), 8 bits per pass.
#include <climits>
#include <type_traits>

#include <cuda_bf16.h>

#define ACES_FILE 10  // site numbers of the checked build
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
    // outputs whichever kernel finishes it: p = e * inv_mass(S_nuc), and the
    // tail from the exact fixed-point sum of the payload masses
    const float inv_S = inv_mass(S_nuc);
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
    if (a.k > 0) a.tail[r] = (float)(S_nuc - (double)tot * FX_INV) * inv_S;
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
                const float e = in ? ex2(fmaf(v, a.c, -kref)) : 0.0f;
                float qx = a.q[((size_t)b * a.K + i) * a.V + x];
                if (!(qx > 0.0f)) st |= ACES_ROW_BAD_Q;
                else accept = accept_test(a.u[(size_t)b * (a.K + 1) + i], qx, e, S_nuc);
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

// Warp-uniform walk over the row: every lane of a warp takes part in every
// round (f gets valid = false past the end), so f may use warp collectives.
template <int DT, bool VEC, class F>
__device__ __forceinline__ void for_each_elem_warp(const char *row, int V, F f) {
    using E = Elem<DT>;
    if (VEC) {
        const int nch = V / E::EPC;
        for (int c0 = threadIdx.x & ~31; c0 < nch; c0 += NT) {
            const int cc = c0 + (threadIdx.x & 31);
            const bool in = cc < nch;
            const uint4 w = in ? ldg16(row + (size_t)cc * 16) : make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
            for (int e = 0; e < E::EPC; ++e) f(in, cc * E::EPC + e, E::get(w, e));
        }
    } else {
        for (int x0 = threadIdx.x & ~31; x0 < V; x0 += NT) {
            const int x = x0 + (threadIdx.x & 31);
            const bool in = x < V;
            f(in, x, in ? E::load1(row, x) : 0.0f);
        }
    }
}

// cnt[d] += 1 and mass[d] += m for every lane with ok; a warp whose lanes
// all hit one bin (the common case in the first digits, where the logits
// share their leading key bits) adds its totals with one atomic each
__device__ __forceinline__ void hist_add(uint32_t *cnt, unsigned long long *mass, bool ok, int d,
                                         unsigned long long m, bool with_mass) {
    const unsigned act = __ballot_sync(0xffffffffu, ok);
    if (act == 0u) return;
    const int d0 = __shfl_sync(0xffffffffu, d, __ffs(act) - 1);
    if (__all_sync(0xffffffffu, !ok || d == d0)) {
        const unsigned long long ms = with_mass ? warp_sum(ok ? m : 0ull) : 0ull;
        if ((threadIdx.x & 31) == 0 && ACES_IN(d0, 256)) {
            atomicAdd(&cnt[d0], (uint32_t)__popc(act));
            if (with_mass) atomicAdd(&mass[d0], ms);
        }
    } else if (ok && ACES_IN(d, 256)) {
        atomicAdd(&cnt[d], 1u);
        if (with_mass) atomicAdd(&mass[d], m);
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
        const bool with_mass = mode == 0 || want_S;
        for_each_elem_warp<DT, VEC>(row, V, [&](bool in, int x, float v) {
            const unsigned long long o = order_val(fkey(v), (uint32_t)x);
            const bool ok = in && v > -INFINITY && (nbits == 0 || (o >> sh) == prefix);
            const int d = (int)((o >> s) & 255ull);
            const unsigned long long m = (ok && with_mass) ? to_fx(ex2(fmaf(v, c, -kref))) : 0ull;
            hist_add(st->cnt, st->mass, ok, d, m, with_mass);
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

// ---------------------------------------------------------------------------
// Binned exact selection.  Elements are binned by their distance below the
// row max, d = (m - z) * inv_w (width T/8, bin 255 = everything farther),
// with exact fixed-point masses per bin.  Bins are ordered by value, so the
// nucleus crossing lies in the first bin whose cumulative mass reaches the
// target, and the first k nucleus ids in the bins up to the one where the
// cumulative count reaches k.  Those bins' elements are collected (at most
// GB_CAP each) and ordered in shared memory.  Returns false, having
// written nothing, when a needed bin is the far bin or too full; the radix
// selection then finishes the row.
constexpr int GB_CAP = 2048;

constexpr int GB_WIN = 96;  // bins of the first pass (12 temperatures below the max)

struct BinState {
    uint32_t cnt[NBIN];              // counts of every bin seen so far
    unsigned long long mass[NBIN];   // masses of the current window's bins
    unsigned long long S_fx;         // total mass of the row
    unsigned long long xs[GB_CAP];  // order values of the crossing bin
    unsigned long long ps[GB_CAP];  // order values of the payload bins
    int nx, np_, bx, bk, ok, nbelow;
    unsigned long long above;       // mass of the bins before the crossing bin
    double target;
};

// appends o to arr[*n] for every lane with take (one atomic per warp)
__device__ __forceinline__ void warp_append(unsigned long long *arr, int *n, bool take, unsigned long long o) {
    const unsigned bal = __ballot_sync(0xffffffffu, take);
    if (bal == 0u) return;
    const int lane = threadIdx.x & 31;
    int base = 0;
    if (lane == __ffs(bal) - 1) base = atomicAdd(n, __popc(bal));
    base = __shfl_sync(0xffffffffu, base, __ffs(bal) - 1);
    const int pos = base + __popc(bal & ((1u << lane) - 1u));
    if (take && pos < GB_CAP) arr[pos] = o;
}

template <int DT, bool VEC>
__device__ bool binned_row(const RowArgs &a, int r, const char *row, float m, float kref,
                           unsigned long long n_fin, BinState *bs, unsigned long long *buf, double *redd,
                           unsigned long long *redu) {
    const int tid = threadIdx.x;
    const bool all_in = a.top_p >= 1.0f;
    // Two windows: the first pass histograms the GB_WIN bins nearest the max
    // with shared-memory atomics and only sums the farther elements in
    // registers, so most elements of a peaked row cost no atomic; a second
    // pass over the remaining bins runs only when the crossing (or the k-th
    // id) lies farther out.
    if (tid == 0) {
        bs->nx = 0;
        bs->np_ = 0;
        bs->above = 0ull;
        bs->nbelow = 0;
        bs->bx = -2;  // crossing bin, -2 while unknown
        bs->bk = -2;  // last payload bin, -2 while unknown
        bs->ok = 1;
    }
    for (int i = tid; i < NBIN; i += NT) bs->cnt[i] = 0u;
    for (int W = 0; W < NBIN - 1; W = W == 0 ? GB_WIN : NBIN - 1) {
        const int WN = W == 0 ? GB_WIN : NBIN - 1 - W;  // bins of this window
        for (int i = tid; i < WN; i += NT) bs->mass[i] = 0ull;
        __syncthreads();
        unsigned long long far_cnt = 0ull, far_mass = 0ull;
        for_each_elem_warp<DT, VEC>(row, a.V, [&](bool in, int, float v) {
            const bool fin = in && v > -INFINITY;
            const float dd = (m - v) * a.inv_w;
            const int d = dd < (float)(NBIN - 1) ? (int)dd : NBIN - 1;
            const bool near = fin && d >= W && d < W + WN && d < NBIN - 1;
            unsigned long long mf = 0ull;
            if (fin && d >= W) mf = to_fx(ex2(fmaf(v, a.c, -kref)));
            if (fin && d >= W && !near) {
                far_cnt += 1ull;
                far_mass += mf;
            }
            hist_add(bs->cnt + W, bs->mass, near, d - W, mf, true);
        });
        far_cnt = block_reduce(far_cnt, redu, SumU64());
        far_mass = block_reduce(far_mass, redu, SumU64());
        if (tid == 0) {
            if (W == 0) {  // the first window sees every element: the total
                unsigned long long S = far_mass;
                for (int j = 0; j < WN; ++j) S += bs->mass[j];
                bs->target = (double)a.top_p * (double)S;
                bs->S_fx = S;
            }
            unsigned long long above = bs->above;
            int nbelow = bs->nbelow;
            const int wend = W + WN;
            if (!all_in && bs->bx == -2) {
                for (int d = W; d < wend; ++d) {
                    if ((double)(above + bs->mass[d - W]) >= bs->target) {
                        bs->bx = d;
                        break;
                    }
                    above += bs->mass[d - W];
                    nbelow += (int)bs->cnt[d];
                }
                bs->above = above;
                bs->nbelow = nbelow;
            }
            // once the nucleus size is bounded, the payload needs min(k, it) ids
            const bool bx_known = all_in || bs->bx >= 0;
            if (bx_known && bs->bk == -2) {
                const long long nnuc_max = all_in ? (long long)n_fin : (long long)bs->nbelow + bs->cnt[bs->bx];
                const long long want = a.k < nnuc_max ? a.k : nnuc_max;
                long long c = 0;
                bs->bk = -1;  // k = 0: no payload
                for (int d = 0; d < wend && want > 0; ++d) {
                    c += bs->cnt[d];
                    if (c >= want) {
                        bs->bk = d;
                        break;
                    }
                }
                if (want > 0 && bs->bk < 0) bs->bk = -2;  // farther than this window
                if (bs->bk >= 0 && c > GB_CAP) bs->ok = 0;
            }
            if (bs->bx >= 0 && bs->cnt[bs->bx] > (uint32_t)GB_CAP) bs->ok = 0;
        }
        __syncthreads();
        if (!bs->ok) return false;
        if ((all_in || bs->bx >= 0) && bs->bk != -2) break;
    }
    if ((!all_in && bs->bx < 0) || bs->bk == -2) return false;  // beyond the binned range
    if (tid == 0 && all_in) bs->bx = -1;
    __syncthreads();
    const int bx = bs->bx, bk = bs->bk;
    // collect the crossing bin and the payload bins
    for_each_elem_warp<DT, VEC>(row, a.V, [&](bool in, int x, float v) {
        const bool fin = in && v > -INFINITY;
        const float dd = (m - v) * a.inv_w;
        const int d = dd < (float)(NBIN - 1) ? (int)dd : NBIN - 1;
        const unsigned long long o = order_val(fkey(v), (uint32_t)x);
        warp_append(bs->xs, &bs->nx, fin && d == bx, o);
        warp_append(bs->ps, &bs->np_, fin && d <= bk, o);
    });
    __syncthreads();
    const int nx = bs->nx, npl = bs->np_;
    // the payload bins' ids ranked by direct counting (order values are
    // distinct): the first min(npl, k) ranks go straight to buf
    const int lp = npl < a.k ? npl : a.k;
    for (int i = tid; i < npl; i += NT) {
        const unsigned long long key = bs->ps[i];
        int rank = 0;
#pragma unroll 4
        for (int t = 0; t < npl; ++t) rank += bs->ps[t] > key;
        if (rank < lp && ACES_IN(rank, ACES_MAX_TOPK)) buf[rank] = key;
    }
    // the crossing bin in order (descending order value)
    {
        const int p2 = next_pow2(nx < 2 ? 2 : nx);
        for (int i = nx + tid; i < p2; i += NT) bs->xs[i] = 0ull;
        __syncthreads();
        if (bx >= 0) bitonic_sort_desc(bs->xs, p2);
    }
    // the crossing id: the first id of the crossing bin where the cumulative
    // mass reaches the target (the bin's last id if rounding keeps it short);
    // its masses go to ps (free now) and a block scan finds it
    double S_nuc;
    unsigned long long cut = 0ull;
    long long n_nuc;
    if (bx >= 0) {
        for (int i = tid; i < nx; i += NT) bs->ps[i] = to_fx(ex2(fmaf(order_value(bs->xs[i]), a.c, -kref)));
        if (tid == 0) bs->bk = -1;  // reuse: the crossing position, -1 until found
        __syncthreads();
        const int per = (nx + NT - 1) / NT;
        const int lo = tid * per < nx ? tid * per : nx, hi = lo + per < nx ? lo + per : nx;
        unsigned long long loc = 0ull;
        for (int i = lo; i < hi; ++i) loc += bs->ps[i];
        unsigned long long tot;
        unsigned long long cum = bs->above + block_exscan_n<NT>(loc, redu, &tot);
        for (int i = lo; i < hi; ++i) {
            const unsigned long long prev = cum;
            cum += bs->ps[i];
            if ((double)prev < bs->target && (double)cum >= bs->target) {  // one id crosses
                bs->bk = i;
                redd[0] = (double)cum * FX_INV;
            }
        }
        __syncthreads();
        int ix = bs->bk;
        if (ix < 0) {  // rounding: the bin's last id
            ix = nx - 1;
            if (tid == 0) redd[1] = (double)(bs->above + tot) * FX_INV;
            __syncthreads();
            S_nuc = redd[1];
        } else {
            S_nuc = redd[0];
        }
        cut = ACES_IN(ix, GB_CAP) ? bs->xs[ix] : 0ull;
        n_nuc = (long long)bs->nbelow + ix + 1;
    } else {
        S_nuc = (double)bs->S_fx * FX_INV;
        n_nuc = (long long)n_fin;
    }
    int L = (int)(n_nuc < (long long)a.k ? n_nuc : (long long)a.k);
    if (L > lp) L = lp;
    __syncthreads();
    finish_row<DT>(a, r, row, kref, S_nuc, cut, all_in ? RS_ALL_IN : 0, buf, L, redd);
    return true;
}

// ---------------------------------------------------------------------------
// Value-histogram path for bfloat16 rows.  A bfloat16 logit takes one of
// 65536 values, and equal values have equal masses, so counting the elements
// of each value is enough: the values of a window below the row max (at most
// VH_W of them) get a count, one shared-memory atomic per element and no
// per-element mass.  The exp-sum S of the whole row comes with a row handed
// over by the fast kernel; otherwise the counting pass sums it in compensated
// fp32, as the fast kernel does.  A prefix scan over the values then gives,
// exactly in 2^-40 fixed point (count x the value's mass), the value holding
// the nucleus crossing (first prefix reaching ceil(top_p * S * 2^40)) and the
// value holding the k-th payload id; the elements of those values (ties are
// taken in id order, which is the order-value order) are collected and ranked
// in shared memory.  Returns false, having written nothing, when a needed
// value lies below the window or a collected set exceeds VH_CAP; the binned
// path then takes the row.
constexpr int VH_W = 4096;    // values below the max with a count
constexpr int VH_CAP = 1024;  // collected ids per set (payload values, crossing value)
constexpr int VH_U = 4;       // 16-byte loads per thread in flight in the counting pass

struct ValHist {
    uint32_t cnt[VH_W];                // elements of value key16(max) - d
    unsigned long long pay[VH_CAP];    // order values of the payload values
    unsigned long long tie[VH_CAP];    // order values of the crossing value
    int npay, ntie;
    int dstar, dk, j;                  // crossing value, last payload value, ids of dstar in the nucleus
    unsigned long long above, cnt_above, npay_need;
    unsigned long long above_cut;      // the cut: order value of the crossing value's j-th id
};

// 16-bit order key of a bfloat16 value: 0x8000 plus the value's signed
// magnitude, so keys sort like values and -0 and +0 share one key (-inf has
// 0x80, the finite values 0x81..0xFF7F); and the value of a key
__device__ __forceinline__ uint32_t bkey16(uint32_t b) {
    const uint32_t mag = b & 0x7FFFu;
    return (b & 0x8000u) ? 0x8000u - mag : 0x8000u + mag;
}
__device__ __forceinline__ float bval16(uint32_t k) {
    const uint32_t b = k >= 0x8000u ? k - 0x8000u : (0x8000u | (0x8000u - k));
    return __uint_as_float(b << 16);
}

// appends o to arr[*n] for every lane with take (one atomic per warp); *n
// may pass cap, entries beyond it are dropped
__device__ __forceinline__ void warp_append_cap(unsigned long long *arr, int *n, bool take, unsigned long long o,
                                                int cap) {
    const unsigned bal = __ballot_sync(0xffffffffu, take);
    if (bal == 0u) return;
    const int lane = threadIdx.x & 31;
    int base = 0;
    if (lane == __ffs(bal) - 1) base = atomicAdd(n, __popc(bal));
    base = __shfl_sync(0xffffffffu, base, __ffs(bal) - 1);
    const int pos = base + __popc(bal & ((1u << lane) - 1u));
    if (take && pos < cap) arr[pos] = o;
}

// (aligned bfloat16 rows; all threads of the CTA)
// S_in: the row's exp-sum in units of 2^kref for a row handed over by the
// fast kernel, 0 otherwise.  *n_fin_out gets the row's count of finite ids
// when top_p = 1 or S_in = 0 (its only uses), even when the row is declined.
__device__ bool valhist_row(const RowArgs &a, int r, const char *row, float m, float kref, double S_in,
                            unsigned long long *n_fin_out, ValHist *vh, unsigned long long *buf, double *redd,
                            unsigned long long *redu) {
    using E = Elem<ACES_BF16>;
    const int tid = threadIdx.x, lane = tid & 31;
    const bool all_in = a.top_p >= 1.0f;
    const bool have_S = S_in > 0.0;
    const uint32_t km = bkey16(__float_as_uint(m) >> 16);  // m is a bfloat16 value
    for (int i = tid; i < VH_W; i += NT) vh->cnt[i] = 0u;
    if (tid == 0) {
        vh->npay = 0;
        vh->ntie = 0;
        vh->dstar = all_in ? -1 : -2;  // -2: not (yet) found in the window
        vh->dk = -2;
    }
    // the window: values km - d for d <= D (never -inf, whose key is 0x80)
    uint32_t D = km - 0x81u < (uint32_t)(VH_W - 1) ? km - 0x81u : (uint32_t)(VH_W - 1);
    if (have_S && !all_in) {
        // Every id below a value of mass e_lo = (1 - top_p) S / (16 V) has
        // less mass than that, so all of them together hold less than a
        // sixteenth of the mass outside the nucleus and the crossing lies at
        // or above that value; an id whose fixed-point mass is 0 (below
        // 2^-40) is never needed either.  D is the last value reaching it.
        const float g = fmaxf(log2f((1.0f - a.top_p) * (float)S_in / (16.0f * (float)a.V)), -41.0f);
        const float vt = (kref + g) / a.c;
        uint32_t lo = 0u, hi = D;  // bval16(km) = m >= vt
        while (lo < hi) {
            const uint32_t mid = (lo + hi + 1u) >> 1;
            if (bval16(km - mid) >= vt) lo = mid;
            else hi = mid - 1u;
        }
        D = lo;
    }
    __syncthreads();
    // ---- pass 1: counts per value (with the finite count and the
    // compensated exp-sum where they are needed) ----
    float hi = 0.f, lo = 0.f;
    unsigned long long nfin = 0ull;
    const int nch = a.V / E::EPC;
    // (-inf words past the end count nowhere)
    auto count_pass = [&](auto with_sum, auto with_nfin) {
        constexpr bool WS = decltype(with_sum)::value, WN = decltype(with_nfin)::value;
        for (int c0 = tid; c0 < nch; c0 += VH_U * NT) {
            uint4 wu[VH_U];
#pragma unroll
            for (int u = 0; u < VH_U; ++u) {
                const int cc = c0 + u * NT;
                wu[u] = cc < nch ? ldg16(row + (size_t)cc * 16) : make_uint4(0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u);
            }
            float cs = 0.f;
            uint32_t nf = 0u;
#pragma unroll
            for (int u = 0; u < VH_U; ++u) {
                const uint32_t wd[4] = {wu[u].x, wu[u].y, wu[u].z, wu[u].w};
#pragma unroll
                for (int q = 0; q < 4; ++q) {
#pragma unroll
                    for (int h = 0; h < 2; ++h) {
                        const uint32_t b = h ? (wd[q] >> 16) : (wd[q] & 0xFFFFu);
                        if (WS) cs += ex2(fmaf(__uint_as_float(b << 16), a.c, -kref));  // 0 for -inf
                        if (WN) nf += b != 0xFF80u;
                        const uint32_t d = km - bkey16(b);
                        if (d <= D && ACES_IN(d, VH_W)) atomicAdd(&vh->cnt[d], 1u);
                    }
                }
            }
            if (WN) nfin += nf;
            if (WS) {
                const float t = hi + cs;  // Neumaier
                if (fabsf(hi) >= fabsf(cs)) lo += (hi - t) + cs;
                else lo += (cs - t) + hi;
                hi = t;
            }
        }
    };
    if (!have_S) count_pass(std::true_type(), std::true_type());
    else if (all_in) count_pass(std::false_type(), std::true_type());
    else count_pass(std::false_type(), std::false_type());
    const unsigned long long n_fin = block_reduce(nfin, redu, SumU64());  // (its barriers order the counts)
    *n_fin_out = n_fin;
    const double S = have_S ? S_in : block_reduce((double)hi + (double)lo, redd, SumD());
    if (!(S > 0.0 && S < 1e300)) return false;
    const unsigned long long tg = all_in ? 0ull : (unsigned long long)ceil((double)a.top_p * S * (double)FX_SCALE);
    // ---- prefix scan over the values, PER consecutive values per thread ----
    constexpr int PER = VH_W / NT;
    static_assert(VH_W % NT == 0, "whole values per thread");
    const int d0 = tid * PER;
    // the mass of the c ids of value km - d (exact: c equal fixed-point masses)
    auto bin_mass = [&](int d, uint32_t c) -> unsigned long long {
        return c ? (unsigned long long)c * to_fx(ex2(fmaf(bval16(km - (uint32_t)d), a.c, -kref))) : 0ull;
    };
    unsigned long long bm_loc = 0ull, bc_loc = 0ull;
#pragma unroll
    for (int i = 0; i < PER; ++i) {
        const uint32_t c = vh->cnt[d0 + i];
        bm_loc += bin_mass(d0 + i, c);
        bc_loc += c;
    }
    unsigned long long m_tot, c_tot;
    const unsigned long long m_ex = block_exscan_n<NT>(bm_loc, redu, &m_tot);
    const unsigned long long c_ex = block_exscan_n<NT>(bc_loc, redu, &c_tot);
    if (!all_in) {  // the value whose masses cross tg (at most one thread finds it)
        unsigned long long cm = m_ex, cc = c_ex;
#pragma unroll
        for (int i = 0; i < PER; ++i) {
            const uint32_t c = vh->cnt[d0 + i];
            const unsigned long long bm = bin_mass(d0 + i, c);
            if (bm > 0ull && cm < tg && cm + bm >= tg) {
                const unsigned long long e = bm / c;  // one id's mass
                vh->dstar = d0 + i;
                vh->above = cm;
                vh->cnt_above = cc;
                vh->j = (int)((tg - cm + e - 1) / e);  // ids of this value in the nucleus
            }
            cm += bm;
            cc += c;
        }
    }
    __syncthreads();
    if (vh->dstar == -2) return false;  // the crossing lies below the window
    const unsigned long long n_nuc = all_in ? n_fin : vh->cnt_above + (unsigned long long)vh->j;
    const int L = (int)(n_nuc < (unsigned long long)a.k ? n_nuc : (unsigned long long)a.k);
    if (L > 0) {  // the value holding the L-th id (at most one thread finds it)
        unsigned long long cc = c_ex;
#pragma unroll
        for (int i = 0; i < PER; ++i) {
            const unsigned long long c = vh->cnt[d0 + i];
            if (cc < (unsigned long long)L && cc + c >= (unsigned long long)L) {
                vh->dk = d0 + i;
                vh->npay_need = cc + c;  // ids of the values up to it
            }
            cc += c;
        }
    } else if (tid == 0) {
        vh->dk = -1;  // no payload
    }
    __syncthreads();
    const int dstar = vh->dstar, dk = vh->dk;
    if (dk == -2) return false;  // the L-th id lies below the window
    if (dk >= 0 && vh->npay_need > (unsigned long long)VH_CAP) return false;
    if (dstar >= 0 && vh->cnt[dstar] > (uint32_t)VH_CAP) return false;
    // ---- collect every id of the values up to dk, and those of dstar ----
    // A packed bfloat16 compare per pair of ids (value >= that of dk, or
    // == that of dstar: IEEE order, where -0 == +0 as in the keys) lets a
    // warp skip a round in which no id of its 32 chunks is wanted.
    const float vk = dk >= 0 ? bval16(km - (uint32_t)dk) : INFINITY;
    const float vs = dstar >= 0 ? bval16(km - (uint32_t)dstar) : NAN;
    const __nv_bfloat162 vk2 = __floats2bfloat162_rn(vk, vk), vs2 = __floats2bfloat162_rn(vs, vs);
    // (the next round's chunk is loaded before this round's ids are examined)
    uint4 pw = tid < nch ? ldg16(row + (size_t)tid * 16) : make_uint4(0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u);
    for (int c0 = tid & ~31; c0 < nch; c0 += NT) {  // warp-uniform rounds
        const int c = c0 + lane;
        const bool in = c < nch;
        const uint4 w = pw;
        pw = c + NT < nch ? ldg16(row + (size_t)(c + NT) * 16) : make_uint4(0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u);
        const uint32_t wd[4] = {w.x, w.y, w.z, w.w};
        uint32_t hm = 0u;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const __nv_bfloat162 x = *reinterpret_cast<const __nv_bfloat162 *>(&wd[q]);
            hm |= __hge2_mask(x, vk2) | __heq2_mask(x, vs2);
        }
        if (!__any_sync(0xffffffffu, hm != 0u)) continue;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const uint32_t b = h ? (wd[q] >> 16) : (wd[q] & 0xFFFFu);
                const uint32_t d = km - bkey16(b);
                const bool fin = in && b != 0xFF80u;
                const bool tp = fin && dk >= 0 && d <= (uint32_t)dk;
                const bool tt = fin && dstar >= 0 && d == (uint32_t)dstar;
                if (!__any_sync(0xffffffffu, tp || tt)) continue;
                const unsigned long long o =
                    order_val(fkey(__uint_as_float(b << 16)), (uint32_t)(c * E::EPC + 2 * q + h));
                warp_append_cap(vh->pay, &vh->npay, tp, o, VH_CAP);
                warp_append_cap(vh->tie, &vh->ntie, tt, o, VH_CAP);
            }
        }
    }
    __syncthreads();
    const int npay = vh->npay, ntie = vh->ntie;
    // ---- rank by direct counting (order values are distinct; descending
    // order, ties by ascending id): the first L payload ids go straight to
    // buf, and the cut is the crossing value's id of rank j - 1 ----
    const int LL = L < npay ? L : npay;
    for (int i = tid; i < npay; i += NT) {
        const unsigned long long key = vh->pay[i];
        int rank = 0;
#pragma unroll 4
        for (int t = 0; t < npay; ++t) rank += vh->pay[t] > key;
        if (rank < LL && ACES_IN(rank, ACES_MAX_TOPK)) buf[rank] = key;
    }
    const int jt = dstar >= 0 ? vh->j - 1 : -1;
    for (int i = tid; i < ntie; i += NT) {
        const unsigned long long key = vh->tie[i];
        int rank = 0;
#pragma unroll 4
        for (int t = 0; t < ntie; ++t) rank += vh->tie[t] > key;
        if (rank == jt) vh->above_cut = key;
    }
    __syncthreads();
    double S_nuc = S;
    unsigned long long cut = 0ull;
    if (dstar >= 0) {
        cut = vh->above_cut;
        const unsigned long long ed = to_fx(ex2(fmaf(bval16(km - (uint32_t)dstar), a.c, -kref)));
        S_nuc = (double)(vh->above + (unsigned long long)vh->j * ed) * FX_INV;
    }
    if (tid == 0) atomicAdd(&a.ws.fb_count[6], 1);
    finish_row<ACES_BF16>(a, r, row, kref, S_nuc, cut, all_in ? RS_ALL_IN : 0, buf, LL, redd);
    return true;
}

template <int DT, bool VEC>
__global__ void __launch_bounds__(NT) k_rows_general(RowArgs a, int direct) {
    using E = Elem<DT>;
    __shared__ SelState st;
    __shared__ union {
        BinState bs;   // binned path
        ValHist vh;    // value-histogram path (bfloat16)
    } paths;
    BinState &bst = paths.bs;
    __shared__ unsigned long long buf[ACES_MAX_TOPK];
    __shared__ double redd[NWARP];
    __shared__ float redf[NWARP];
    __shared__ unsigned long long redu[NWARP];
    __shared__ int s_bad;
    __shared__ int s_nbuf;
    const int tid = threadIdx.x;
    pdl_wait();  // after the fast row kernel: its fallback list is complete
    const int nrows = direct ? a.rows : *a.ws.fb_count;
    for (int idx = blockIdx.x; idx < nrows; idx += gridDim.x) {
        const int r = direct ? idx : a.ws.fb_list[idx];
        if (!ACES_IN(r, a.rows)) continue;  // (the same r in every thread)
        const char *row = reinterpret_cast<const char *>(a.logits) + (size_t)r * a.V * E::SIZE;
        // a row the fast kernel handed over comes with its max and its
        // exp-sum (and is finite); the max pass runs only where the paths
        // need the finite count it takes (top_p = 1 on float32 rows)
        RowStat hs;
        hs.flags = 0;
        if (VEC && !direct) hs = a.ws.stats[r];
        const bool handed = hs.flags == RS_HANDOFF;
        float m;
        unsigned long long n_fin = 0ull;
        if (handed && (DT == ACES_BF16 || a.top_p < 1.0f)) {
            m = hs.kref;
        } else {
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
            m = block_reduce(mx, redf, MaxF());
            n_fin = block_reduce(nfin, redu, SumU64());
            if (s_bad || n_fin == 0ull || !(ceilf(m * a.c) < 1e30f)) {
                nonfinite_row<NT>(a, r);
                __syncthreads();
                continue;
            }
        }
        const float kref = ceilf(m * a.c);  // masses are 2^(z*c - kref) <= 1
        if (DT == ACES_BF16 && VEC) {
            // the handed exp-sum in units of 2^kref (its reference is the same
            // ceil(m c); the power-of-two rescale is exact)
            const double S_in = handed ? ldexp(hs.S_nuc, (int)(hs.c - kref)) : 0.0;
            unsigned long long nf = 0ull;
            const bool done = valhist_row(a, r, row, m, kref, S_in, &nf, &paths.vh, buf, redd, redu);
            __syncthreads();
            if (done) continue;
            n_fin = nf;
        }
        if (binned_row<DT, VEC>(a, r, row, m, kref, n_fin, &bst, buf, redd, redu)) {
            __syncthreads();
            continue;
        }
        if (tid == 0) atomicAdd(&a.ws.fb_count[4], 1);
        const bool all_in = a.top_p >= 1.0f;
        unsigned long long cut = 0ull;
        double S_nuc;
        unsigned long long n_nuc;
        if (!all_in) {
            cut = radix_select<DT, VEC>(row, a.V, kref, a.c, 0, (double)a.top_p, 0u, true, &st);
            S_nuc = (double)(st.above + st.found) * FX_INV;
            n_nuc = (unsigned long long)st.above_cnt + 1ull;
        } else {
            unsigned long long sfx = 0ull;
            for_each_elem<DT, VEC>(row, a.V, [&](int, float v) {
                if (v > -INFINITY) sfx += to_fx(ex2(fmaf(v, a.c, -kref)));
            });
            S_nuc = (double)block_reduce(sfx, redu, SumU64()) * FX_INV;
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
    // only now: resolve CTAs waiting beside busy rows would slow them down
    pdl_trigger();
}

// direct = 0 follows the fast row kernel and overlaps its drain
cudaError_t launch_rows_general(const RowArgs &a, int dt, bool vec, int direct, int grid, cudaStream_t s) {
    void (*fn)(RowArgs, int) = dt == ACES_BF16 ? (vec ? k_rows_general<ACES_BF16, true> : k_rows_general<ACES_BF16, false>)
                                               : (vec ? k_rows_general<ACES_F32, true> : k_rows_general<ACES_F32, false>);
    if (direct) {
        fn<<<grid, NT, 0, s>>>(a, direct);
        return cudaGetLastError();
    }
    return launch_after(fn, (unsigned)grid, NT, s, a, direct);
}

#ifdef ACES_CHECKED
cudaError_t check_take_rows_general(unsigned long long out[3]) { return check_take(out); }
#endif

}  // namespace aces
