// Fast row kernel of the AceSpec cloud step (Sec. III-B: accept test and
// packaging of the target distribution; Sec. V-C: compact payload; the
// acceptance rule is the modified rejection sampling of Sec. II-A).
//
// One CTA of 256 threads per target row r = b*(K+1)+i, four CTAs per SM
// (64 registers per thread with eight 16-byte loads in flight, and a sketch
// of at most 16 KB), so that the per-row epilogue of one row overlaps the
// HBM stream of the others.
//
//   pass 1   every logit is read once from HBM with 16-byte loads (eight in
//            flight per thread): an online exp-sum in log2 units against an
//            integer reference k_t = ceil(max z * log2(e)/T) (one paired
//            FFMA per two logits, one ex2 per logit, rescales are exact
//            powers of two), the two largest group maxima per thread, and the
//            max of every group of GC consecutive 16-byte chunks into a sketch.
//   certify  group maxima are binned by (m - gmax) / (T/8); one max per
//            group is a lower bound of the mass above a bin edge, so the
//            first bin whose bound reaches top_p * S proves that the nucleus
//            lies above that edge (for top_p = 1: the first bin holding k
//            groups proves the top k lie above it).  First tier: the two
//            largest group maxima of every thread, kept in registers during
//            pass 1; second tier (only when the first cannot certify): every
//            group of the sketch.  Rows neither can certify go to the exact
//            general kernel.
//   select   a binary search turns the edge into a key threshold; groups
//            whose sketch key reaches it are listed, re-read (one 16-byte
//            chunk per thread), and their ids above the threshold ordered by
//            the 64-bit (logit, id) order (direct ranking up to 512 ids,
//            bitonic sort above); the nucleus crossing is found with exact
//            fixed-point prefix sums in one warp.
//   finish   payload (first k of the nucleus), tail mass, accept test of the
//            draft token at this position, per-row state for the resolve
//            kernels.
#include <climits>
#include <type_traits>
#include <cuda_bf16.h>

#include "common.cuh"

namespace aces {

constexpr int NTF = 256;
constexpr int NWF = NTF / 32;
constexpr int CAND_CAP_F = 2048;
constexpr int RANK_MAX = 512;       // candidates ordered by direct ranking (more: bitonic sort)

template <int DT> struct Sketch;
template <> struct Sketch<ACES_F32> {
    using T = uint32_t;
    __device__ __forceinline__ static T enc(uint32_t key) { return key; }
    __device__ __forceinline__ static float dec(T s) { return fkey_inv(s); }
};
template <> struct Sketch<ACES_BF16> {
    using T = uint16_t;  // a bf16 key has 16 zero low bits
    __device__ __forceinline__ static T enc(uint32_t key) { return (T)(key >> 16); }
    __device__ __forceinline__ static float dec(T s) { return fkey_inv((uint32_t)s << 16); }
};

__device__ __forceinline__ void two_sum(float a, float b, float &s, float &e) {
    s = a + b;
    const float bb = s - a;
    e = (a - (s - bb)) + (b - bb);
}

// 2^d for an integer-valued d <= 0, exactly
__device__ __forceinline__ float pow2_int(float d) {
    return d >= -126.0f ? __int_as_float((127 + __float2int_rn(d)) << 23) : 0.0f;
}

template <int DT, int GC>
__device__ __forceinline__ float group_max(const uint4 (&w)[GC]) {
    if (DT == ACES_BF16) {
        __nv_bfloat162 mx = *reinterpret_cast<const __nv_bfloat162 *>(&w[0].x);
#pragma unroll
        for (int j = 0; j < GC; ++j) {
            const uint32_t wd[4] = {w[j].x, w[j].y, w[j].z, w[j].w};
#pragma unroll
            for (int q = 0; q < 4; ++q) mx = __hmax2(mx, *reinterpret_cast<const __nv_bfloat162 *>(&wd[q]));
        }
        const uint32_t u = *reinterpret_cast<const uint32_t *>(&mx);
        return fmaxf(__uint_as_float(u << 16), __uint_as_float(u & 0xFFFF0000u));
    } else {
        float gm = -INFINITY;
#pragma unroll
        for (int j = 0; j < GC; ++j)
            gm = fmaxf(gm, fmaxf(fmaxf(__uint_as_float(w[j].x), __uint_as_float(w[j].y)),
                                 fmaxf(__uint_as_float(w[j].z), __uint_as_float(w[j].w))));
        return gm;
    }
}

// Paired fp32 arithmetic (one instruction for two lanes of a 64-bit register
// pair; each lane rounds exactly like the scalar operation).
__device__ __forceinline__ unsigned long long pack2(float lo, float hi) {
    unsigned long long r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
    return r;
}
__device__ __forceinline__ void unpack2(unsigned long long v, float &lo, float &hi) {
    asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ unsigned long long ffma2(unsigned long long a, unsigned long long b,
                                                    unsigned long long c) {
    unsigned long long d;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
    return d;
}
__device__ __forceinline__ unsigned long long fadd2(unsigned long long a, unsigned long long b) {
    unsigned long long d;
    asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
    return d;
}
// (2^(lo*c + nk), 2^(hi*c + nk)) for a pair of logits
__device__ __forceinline__ unsigned long long ex2_pair(unsigned long long z2, unsigned long long c2,
                                                       unsigned long long nk2) {
    float lo, hi;
    unpack2(ffma2(z2, c2, nk2), lo, hi);
    return pack2(ex2(lo), ex2(hi));
}

// sum over the group of 2^(z*c - k), two logits per instruction
template <int DT, int GC>
__device__ __forceinline__ float group_expsum(const uint4 (&w)[GC], float c, float nk) {
    const unsigned long long c2 = pack2(c, c), nk2 = pack2(nk, nk);
    unsigned long long acc = 0ull;
#pragma unroll
    for (int j = 0; j < GC; ++j) {
        unsigned long long s;
        if (DT == ACES_BF16) {
            const uint32_t wd[4] = {w[j].x, w[j].y, w[j].z, w[j].w};
            unsigned long long p[4];
#pragma unroll
            for (int q = 0; q < 4; ++q)
                p[q] = ex2_pair(pack2(__uint_as_float(wd[q] << 16), __uint_as_float(wd[q] & 0xFFFF0000u)),
                                c2, nk2);
            s = fadd2(fadd2(p[0], p[1]), fadd2(p[2], p[3]));
        } else {
            const unsigned long long p0 = ex2_pair(pack2(__uint_as_float(w[j].x), __uint_as_float(w[j].y)), c2, nk2);
            const unsigned long long p1 = ex2_pair(pack2(__uint_as_float(w[j].z), __uint_as_float(w[j].w)), c2, nk2);
            s = fadd2(p0, p1);
        }
        acc = j == 0 ? s : fadd2(acc, s);
    }
    float a, b;
    unpack2(acc, a, b);
    return a + b;
}

// Called by all threads when this CTA has written row r's outputs and state.
// The CTA that finishes the last row of a sequence (rows handed to the
// general kernel are never counted) draws the sequence's token from the
// stored nucleus, so most sequences need no separate resolve launch.
template <int NTH>
__device__ void row_finished(const RowArgs &a, int r, unsigned char *scratch) {
    if (a.ws.seqcnt == nullptr) return;  // sparsify
    __shared__ int s_last;
    __shared__ unsigned long long s_red[NTH / 32];
    __shared__ DrawShared s_draw;
    const int b = r / (a.K + 1);
    __syncthreads();  // every thread's writes of this row are issued
    // releases this row's writes; the last row acquires the others'
    if (threadIdx.x == 0) s_last = atomic_add_acq_rel(&a.ws.seqcnt[b], 1) == a.K;
    __syncthreads();
    if (!s_last) return;
    unsigned long long *skey = reinterpret_cast<unsigned long long *>(scratch);  // 4 * NUC_CAP entries
    draw_from_list<NTH>(a.ws, a.q, a.u, a.K, a.V, b, a.accept_len, a.out_token, a.row_status, skey,
                        skey + NUC_CAP, skey + 2 * NUC_CAP, skey + 3 * NUC_CAP, s_red, &s_draw);
}

// Hands row r to the general kernel with its max m and its exp-sum S (in
// units of 2^kref), which spare that kernel a pass and the exponentials of
// another (the row is finite: rows with NaN or +inf were marked NONFINITE
// before any handoff).
__device__ __forceinline__ void fallback_row(const RowArgs &a, int r, float m, float kref, double S) {
    RowStat s;
    s.kref = m;
    s.c = kref;
    s.S_nuc = S;
    s.cut = 0ull;
    s.flags = RS_HANDOFF;
    s.nnuc = -1;
    a.ws.stats[r] = s;
    const int pos = atomicAdd(a.ws.fb_count, 1);
    a.ws.fb_list[pos] = r;
}

// the CTA's exp-sum from the per-warp (hi, lo) pairs, in fp64, by warp 0 (a
// shuffle tree: three dependent fp64 adds instead of sixteen in one thread)
__device__ __forceinline__ double warp0_mass(const float *hi, const float *lo, int lane) {
    double v = lane < NWF ? (double)hi[lane] + (double)lo[lane] : 0.0;
#pragma unroll
    for (int o = NWF / 2; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

template <int DT, int GC>
__global__ void __launch_bounds__(NTF, 4) k_rows_fast(RowArgs a) {
    using E = Elem<DT>;
    using SK = typename Sketch<DT>::T;
    constexpr int EPC = E::EPC;
    extern __shared__ __align__(16) unsigned char smem[];
    const int ng = a.ng;
    SK *sketch = reinterpret_cast<SK *>(smem);
    const size_t sk_bytes = align16((size_t)ng * sizeof(SK)) > (size_t)CAND_CAP_F * 8
                                ? align16((size_t)ng * sizeof(SK)) : (size_t)CAND_CAP_F * 8;
    unsigned long long *sorted = reinterpret_cast<unsigned long long *>(smem);  // after collection
    unsigned long long *cand = reinterpret_cast<unsigned long long *>(smem + sk_bytes);

    __shared__ uint32_t bins[NBIN];
    __shared__ float redf[NWF], redk[NWF], redh[NWF], redl[NWF];
    __shared__ int s_ncand, s_ngl, s_bc, s_nstar, s_L;
    __shared__ uint32_t s_thr;
    __shared__ double s_S, s_Snuc;
    __shared__ float s_inv_S;
    __shared__ unsigned long long s_cut, s_Snuc_fx, s_cumL_fx;

    static_assert(NTF == SPLIT_NT, "split rows keep two group maxima per thread of SPLIT_NT");
    // rows r < r_full take one CTA each; each later row takes P CTAs, one per
    // range of gper sketch groups
    const bool split = (int)blockIdx.x >= a.r_full;
    const int sj = split ? (int)blockIdx.x - a.r_full : 0;
    const int r = split ? a.r_full + sj / a.P : (int)blockIdx.x;
    const int part = split ? sj % a.P : 0;
    const int g_lo = split ? part * a.gper : 0;
    const int g_hi = split ? min(ng, g_lo + a.gper) : ng;
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    const char *row = reinterpret_cast<const char *>(a.logits) + (size_t)r * a.V * E::SIZE;
    const int nch = a.V / EPC;
    const uint32_t NI = E::NEG_INF_WORD;

    // the draft token of this position, fetched early by thread 0
    int xb = -1, bq = 0, iq = 0;
    if (a.K > 0) {
        bq = r / (a.K + 1);
        iq = r % (a.K + 1);
        if (tid == 0 && iq < a.K) xb = a.xt[(size_t)bq * a.K + iq];
    }

    // ---- pass 1 ----
    float k_t = -1e30f, m_t = -INFINITY, s_t = 0.f, e_t = 0.f;
    float t1 = -INFINITY, t2 = -INFINITY;  // this thread's two largest group maxima
    // groups per iteration: eight 16-byte loads in flight per thread
    constexpr int GPI = GC >= 8 ? 1 : 8 / GC;
    const int ngf = nch / GC;  // groups without a ragged end
    // one iteration: GPI groups, one reference check and one compensated add
    auto step = [&](int g0, auto checked) {
        constexpr bool CHK = decltype(checked)::value;
        uint4 w[GPI][GC];
#pragma unroll
        for (int h = 0; h < GPI; ++h) {
            const int g = g0 + h * NTF;
#pragma unroll
            for (int j = 0; j < GC; ++j) {
                const int cc = g * GC + j;
                w[h][j] = (!CHK || (g < g_hi && cc < nch)) ? ldg16(row + (size_t)cc * 16) : make_uint4(NI, NI, NI, NI);
            }
        }
        float im = -INFINITY;
#pragma unroll
        for (int h = 0; h < GPI; ++h) {
            const int g = g0 + h * NTF;
            const float gm = group_max<DT, GC>(w[h]);
            im = fmaxf(im, gm);
            if (gm > t2) {
                t2 = fminf(gm, t1);
                t1 = fmaxf(gm, t1);
            }
            if (!CHK || g < g_hi) sketch[g] = Sketch<DT>::enc(fkey(gm));
        }
        m_t = fmaxf(m_t, im);
        const float gk = im * a.c;
        if (gk > k_t) {
            const float nk = ceilf(gk);
            const float sc = pow2_int(k_t - nk);
            s_t *= sc;
            e_t *= sc;
            k_t = nk;
        }
        float gs[GPI];
#pragma unroll
        for (int h = 0; h < GPI; ++h) gs[h] = group_expsum<DT, GC>(w[h], a.c, -k_t);
#pragma unroll
        for (int wdt = 1; wdt < GPI; wdt <<= 1)
#pragma unroll
            for (int h = 0; h < GPI; h += 2 * wdt) gs[h] += gs[h + wdt];
        const float t = s_t + gs[0];
        if (fabsf(s_t) >= fabsf(gs[0])) e_t += (s_t - t) + gs[0];
        else e_t += (gs[0] - t) + s_t;
        s_t = t;
    };
    int g0 = g_lo + tid;
    const int gf_hi = ngf < g_hi ? ngf : g_hi;  // groups of this CTA without a ragged end
    for (; g0 + (GPI - 1) * NTF < gf_hi; g0 += NTF * GPI) step(g0, std::false_type());
    for (; g0 < g_hi; g0 += NTF * GPI) step(g0, std::true_type());
    // dependent loads of the accept test, consumed at the end
    float zx = 0.f, qx = 0.f, ux = 0.f;
    if (xb >= 0 && xb < a.V) {
        zx = E::load1(row, xb);
        qx = __ldg(a.q + ((size_t)bq * a.K + iq) * a.V + xb);
        ux = __ldg(a.u + (size_t)bq * (a.K + 1) + iq);
    }

    // ---- row max, reference and exp-sum (fp32 two-sum tree, fp64 in thread 0) ----
    {
        const float mw = warp_max(m_t), kw = warp_max(k_t);
        if (lane == 0) {
            redf[wid] = mw;
            redk[wid] = kw;
        }
    }
    for (int i = tid; i < NBIN; i += NTF) bins[i] = 0u;
    __syncthreads();
    float m = redf[0], kref = redk[0];  // this CTA's (the row's unless split)
#pragma unroll
    for (int i = 1; i < NWF; ++i) {
        m = fmaxf(m, redf[i]);
        kref = fmaxf(kref, redk[i]);
    }
    {
        const float f = pow2_int(fmaxf(k_t - kref, -1000.0f));
        float hi = s_t * f, lo = e_t * f;
        for (int o = 16; o > 0; o >>= 1) {
            const float h2 = __shfl_xor_sync(0xffffffffu, hi, o);
            const float l2 = __shfl_xor_sync(0xffffffffu, lo, o);
            float sm, er;
            two_sum(hi, h2, sm, er);
            lo = lo + l2 + er;
            hi = sm;
        }
        if (lane == 0) {
            redh[wid] = hi;
            redl[wid] = lo;
        }
    }
    if (split) {
        // Publish this part (max, reference, exp-sum, top group maxima and
        // its sketch groups); the CTA that finishes the row's last part
        // gathers the others and runs the rest of the row.  No CTA waits.
        const int si = r - a.r_full;
        unsigned char *pr = a.ws.parts + (size_t)si * a.ws.part_stride;
        PartStat *ps = reinterpret_cast<PartStat *>(pr);
        float *tops = reinterpret_cast<float *>(pr + SPLIT_P_MAX * sizeof(PartStat));
        SK *gsk = reinterpret_cast<SK *>(pr + SPLIT_P_MAX * sizeof(PartStat) + (size_t)SPLIT_P_MAX * 2 * NTF * 4);
        tops[(part * 2 + 0) * NTF + tid] = t1;
        tops[(part * 2 + 1) * NTF + tid] = t2;
        for (int g = g_lo + tid; g < g_hi; g += NTF) gsk[g] = sketch[g];
        __syncthreads();
        if (wid == 0) {
            const double S = warp0_mass(redh, redl, lane);
            if (lane == 0) {
                PartStat st;
                st.m = m;
                st.kref = kref;
                st.S = S;
                ps[part] = st;
            }
        }
        __syncthreads();
        // releases this part; the last part acquires the others
        if (tid == 0) s_ncand = atomic_add_acq_rel(&a.ws.rowcnt[si], 1) == a.P - 1;  // s_ncand reused as a flag
        __syncthreads();
        if (!s_ncand) return;  // another part finishes the row
        if (tid == 0) {
            atomicAdd(&a.ws.fb_count[5], 1);
            float mm = -INFINITY, kk = -1e30f;
            for (int p2 = 0; p2 < a.P; ++p2) {
                mm = fmaxf(mm, ps[p2].m);
                kk = fmaxf(kk, ps[p2].kref);
            }
            double S = 0.0;  // each part's sum rescaled by an exact power of two
            for (int p2 = 0; p2 < a.P; ++p2) S += ps[p2].S * (double)pow2_int(fmaxf(ps[p2].kref - kk, -1000.0f));
            s_S = S;
            redf[0] = mm;
            redk[0] = kk;
        }
        for (int p2 = 0; p2 < a.P; ++p2) {
            if (p2 == part) continue;
            const int lo = p2 * a.gper, hi = min(ng, lo + a.gper);
            for (int g = lo + tid; g < hi; g += NTF) sketch[g] = gsk[g];
        }
        __syncthreads();
        m = redf[0];
        kref = redk[0];
        // first tier over every part's top group maxima
        for (int i = tid; i < a.P * 2 * NTF; i += NTF) {
            const float t = tops[i];
            const float d = (m - t) * a.inv_w;
            if (d < (float)NBIN) atomicAdd(&bins[(int)d], 1u);
        }
        __syncthreads();
    } else {
        // first tier: bins of the 2 * NTF largest group maxima (two per
        // thread); they carry a lower bound of the mass above every bin edge
        const float d1 = (m - t1) * a.inv_w, d2 = (m - t2) * a.inv_w;
        if (d1 < (float)NBIN) atomicAdd(&bins[(int)d1], 1u);
        if (d2 < (float)NBIN) atomicAdd(&bins[(int)d2], 1u);
        __syncthreads();
        if (wid == 0) {
            const double S = warp0_mass(redh, redl, lane);
            if (lane == 0) s_S = S;
        }
    }
    const bool all_in = a.top_p >= 1.0f;
    for (int pass = 0; pass < 2; ++pass) {
        if (pass == 1) {  // second tier: every group of the sketch
            __syncthreads();
            if (s_bc >= 0) break;
            if (tid == 0) atomicAdd(&a.ws.fb_count[2], 1);
            for (int i = tid; i < NBIN; i += NTF) bins[i] = 0u;
            __syncthreads();
            for (int g = tid; g < ng; g += NTF) {
                const float d = (m - Sketch<DT>::dec(sketch[g])) * a.inv_w;
                if (d < (float)NBIN) atomicAdd(&bins[(int)d], 1u);
            }
            __syncthreads();
        }
        if (wid == 0) {
            constexpr int PER = NBIN / 32;
            float lb[PER];
            unsigned cn[PER];
            float lsum = 0.f;
            unsigned csum = 0;
            // a group in bin b carries at least 2^((m - (b+1)T/8) c - kref)
            const float base2 = ex2(fmaf(m, a.c, -kref));
#pragma unroll
            for (int j = 0; j < PER; ++j) {
                const int b = lane * PER + j;
                cn[j] = bins[b];
                lb[j] = (float)cn[j] * ex2(-(float)(b + 1) * (1.4426950408889634f / BIN_PER_T)) * base2;
                lsum += lb[j];
                csum += cn[j];
            }
            float lpre = lsum;
            unsigned cpre = csum;
            for (int o = 1; o < 32; o <<= 1) {
                const float tt = __shfl_up_sync(0xffffffffu, lpre, o);
                const unsigned cc = __shfl_up_sync(0xffffffffu, cpre, o);
                if (lane >= o) {
                    lpre += tt;
                    cpre += cc;
                }
            }
            lpre -= lsum;
            cpre -= csum;
            double S = 0.0;  // lane 0 of warp 0 is thread 0, which wrote s_S above
            if (lane == 0) S = s_S;
            S = __shfl_sync(0xffffffffu, S, 0);
            // 1e-4 covers the fp32 sums of the bound and of S
            const float target = (float)((double)a.top_p * S) * (1.0f + 1e-4f);
            int hit = -1;
#pragma unroll
            for (int j = 0; j < PER; ++j) {
                lpre += lb[j];
                cpre += cn[j];
                const bool okb = all_in ? (cpre >= (unsigned)a.k) : (lpre * (1.0f - 1e-4f) >= target);
                if (okb && hit < 0) hit = lane * PER + j;
            }
            const unsigned bal = __ballot_sync(0xffffffffu, hit >= 0);
            const int first = bal ? __ffs(bal) - 1 : -1;
            const int bc = first >= 0 ? __shfl_sync(0xffffffffu, hit, first) : -1;
            // Bins are monotone in the order key, so a binary search finds
            // the smallest sketch key in a bin <= bc; the scans below then
            // select exactly those ids by integer compares.
            uint32_t thr = 0;
            if (bc >= 0) {
                const float lim = (float)(bc + 1);
                uint32_t lo = 0, hi = Sketch<DT>::enc(fkey(m));  // the max itself is in bin 0
                while (lo < hi) {
                    const uint32_t mid = lo + ((hi - lo) >> 1);
                    if ((m - Sketch<DT>::dec((SK)mid)) * a.inv_w < lim) hi = mid;
                    else lo = mid + 1;
                }
                thr = hi;
            }
            if (lane == 0) {
                s_bc = bc;
                s_thr = thr;
                s_ncand = 0;
                s_ngl = 0;
            }
        }
    }
    __syncthreads();
    const double S = s_S;
    const int bc = s_bc;
    if (!(S > 0.0 && S < 1e300) || !(m < INFINITY) || !(kref < 1e30f)) {
        nonfinite_row<NTF>(a, r);
        row_finished<NTF>(a, r, smem);
        return;
    }
    if (bc < 0) {
        if (tid == 0) fallback_row(a, r, m, kref, S);
        return;
    }
    // ---- candidates: every id whose key reaches thr (bin <= bc) ----
    const uint32_t thr = s_thr;
    const uint32_t thr_key = DT == ACES_BF16 ? thr << 16 : thr;  // for 32-bit element keys
    // groups holding candidates: the sketch is scanned 16 bytes at a time
    // with packed compares; each warp lists its hits in cand[] (free until
    // ranking) with one atomic per warp and round
    int *glist = reinterpret_cast<int *>(cand);
    {
        constexpr int SPW = 16 / sizeof(SK);  // sketch entries per 16-byte word
        const int nw = (ng + SPW - 1) / SPW;
        const uint4 *sk4 = reinterpret_cast<const uint4 *>(sketch);
        for (int i0 = 0; i0 < nw; i0 += NTF) {  // warp-uniform rounds
            const int i = i0 + tid;
            unsigned hm = 0;  // hit mask over the word's SPW entries
            if (i < nw) {
                const uint4 wd = sk4[i];
                const uint32_t x[4] = {wd.x, wd.y, wd.z, wd.w};
                if (DT == ACES_BF16) {
                    const uint32_t t2x = thr * 0x00010001u;
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        const uint32_t c = __vcmpgeu2(x[q], t2x);
                        hm |= ((c >> 15) & 1u) << (2 * q) | ((c >> 31) & 1u) << (2 * q + 1);
                    }
                } else {
#pragma unroll
                    for (int q = 0; q < 4; ++q) hm |= (unsigned)(x[q] >= thr) << q;
                }
                if (i == nw - 1 && ng % SPW) hm &= (1u << (ng % SPW)) - 1u;  // past the last group
            }
            if (!__any_sync(0xffffffffu, hm != 0u)) continue;
            const int cnt = __popc(hm);
            int inc = cnt;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int t = __shfl_up_sync(0xffffffffu, inc, o);
                if (lane >= o) inc += t;
            }
            int base = 0;
            if (lane == 31) base = atomicAdd(&s_ngl, inc);
            base = __shfl_sync(0xffffffffu, base, 31) + inc - cnt;
            while (hm) {
                const int e = __ffs(hm) - 1;
                hm &= hm - 1u;
                if (base < CAND_CAP_F) glist[base] = i * SPW + e;
                ++base;
            }
        }
    }
    __syncthreads();
    const int ngl = s_ngl;
    if (ngl > CAND_CAP_F) {  // every listed group holds a candidate: too many
        if (tid == 0) fallback_row(a, r, m, kref, S);
        return;
    }
    // re-read the listed groups, one 16-byte chunk per thread and round;
    // candidates go to sorted[] (the sketch is no longer needed)
    unsigned long long *cv = sorted;
    {
        const int nck = ngl * GC;
        for (int c0 = 0; c0 < nck; c0 += 2 * NTF) {
            uint4 wv[2];
            int cc[2];
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const int c = c0 + h * NTF + tid;
                cc[h] = c < nck ? glist[c / GC] * GC + c % GC : nch;
                wv[h] = cc[h] < nch ? ldg16(row + (size_t)cc[h] * 16) : make_uint4(NI, NI, NI, NI);
            }
#pragma unroll
            for (int h = 0; h < 2; ++h)
#pragma unroll
                for (int e = 0; e < EPC; ++e) {
                    const uint32_t key = fkey(E::get(wv[h], e));
                    if (cc[h] < nch && key >= thr_key) {
                        const int pos = atomicAdd(&s_ncand, 1);
                        if (pos < CAND_CAP_F) cv[pos] = order_val(key, (uint32_t)(cc[h] * EPC + e));
                    }
                }
        }
    }
    __syncthreads();
    const int n = s_ncand;
    if (n > CAND_CAP_F) {
        if (tid == 0) fallback_row(a, r, m, kref, S);
        return;
    }
    // ---- order the candidates (descending order value) into ord[] (the
    // cand[] bytes), their masses in 2^-40 units into efx[] ----
    unsigned long long *ord = cand;
    unsigned long long *efx;
    if (n <= RANK_MAX) {  // rank of each candidate by direct count
        efx = sorted + RANK_MAX;
        for (int i = tid; i < n; i += NTF) {
            const unsigned long long v = cv[i];
            int rank = 0;
#pragma unroll 4
            for (int j = 0; j < n; ++j) rank += cv[j] > v;
            ord[rank] = v;
            efx[rank] = to_fx(ex2(fmaf(order_value(v), a.c, -kref)));
        }
    } else {
        if (tid == 0) atomicAdd(&a.ws.fb_count[3], 1);
        const int np = next_pow2(n);
        for (int i = tid; i < np; i += NTF) ord[i] = i < n ? cv[i] : 0ull;
        __syncthreads();
        bitonic_sort_desc(ord, np);
        efx = sorted;
        for (int i = tid; i < n; i += NTF) efx[i] = to_fx(ex2(fmaf(order_value(ord[i]), a.c, -kref)));
    }
    __syncthreads();

    // ---- nucleus crossing with exact fixed-point prefix sums (warp 0) ----
    if (wid == 0) {
        const int per = (n + 31) / 32;
        const int lo = lane * per, hi = min(n, lo + per);
        unsigned long long loc = 0ull;
        for (int i = lo; i < hi; ++i) loc += efx[i];
        unsigned long long inc = loc;
        for (int o = 1; o < 32; o <<= 1) {
            const unsigned long long tt = __shfl_up_sync(0xffffffffu, inc, o);
            if (lane >= o) inc += tt;
        }
        const unsigned long long ex = inc - loc;
        int nstar = n - 1;
        if (!all_in) {
            const unsigned long long tg = (unsigned long long)ceil((double)a.top_p * S * (double)FX_SCALE);
            int found = INT_MAX;
            unsigned long long c = ex;
            for (int i = lo; i < hi; ++i) {
                c += efx[i];
                if (c >= tg) {
                    found = i;
                    break;
                }
            }
            const unsigned bal = __ballot_sync(0xffffffffu, found != INT_MAX);
            nstar = bal ? __shfl_sync(0xffffffffu, found, __ffs(bal) - 1) : INT_MAX;
        }
        int L = 0;
        if (nstar != INT_MAX) L = all_in ? min(n, a.k) : min(nstar + 1, a.k);
        unsigned long long cN = 0ull, cL = 0ull, c = ex;
        for (int i = lo; i < hi; ++i) {
            c += efx[i];
            if (i == nstar) cN = c;
            if (i == L - 1) cL = c;
        }
        cN = warp_sum(cN);
        cL = warp_sum(cL);
        if (lane == 0) {
            s_nstar = nstar;
            s_L = L;
            s_Snuc_fx = cN;
            s_cumL_fx = cL;
            const double sn = all_in ? S : (double)cN * FX_INV;
            s_Snuc = sn;
            s_inv_S = inv_mass(sn);
            s_cut = (nstar != INT_MAX && !all_in) ? ord[nstar] : 0ull;
        }
    }
    __syncthreads();
    if (s_nstar == INT_MAX) {  // the candidates carry too little mass: exact path
        if (tid == 0) fallback_row(a, r, m, kref, S);
        return;
    }
    // keep the nucleus (in order) for the residual step when it fits
    const int nnuc = (a.ws.nuc != nullptr && !all_in && s_nstar + 1 <= NUC_CAP) ? s_nstar + 1 : -1;
    if (nnuc > 0)
        for (int i = tid; i < nnuc; i += NTF) a.ws.nuc[(size_t)r * NUC_CAP + i] = ord[i];
    const int L = s_L;
    const float inv_S = s_inv_S;
    for (int j = tid; j < a.k; j += NTF) {
        const size_t o = (size_t)r * a.k + j;
        if (j < L) {
            const unsigned long long ov = ord[j];
            a.topk_ids[o] = (int32_t)order_id(ov);
            a.topk_probs[o] = ex2(fmaf(order_value(ov), a.c, -kref)) * inv_S;
        } else {
            a.topk_ids[o] = -1;
            a.topk_probs[o] = 0.0f;
        }
    }
    if (tid == 0) {
        const double S_nuc = s_Snuc;
        const double cumL = (double)s_cumL_fx * FX_INV;
        if (a.k > 0) a.tail[r] = (float)(S_nuc - cumL) * inv_S;
        const unsigned long long cut = s_cut;
        int stt = 0;
        if (a.K > 0 && iq < a.K) {
            int accept = 0;
            if (xb < 0 || xb >= a.V) {
                stt |= ACES_ROW_BAD_Q;
            } else {
                const bool in = all_in ? (zx > -INFINITY) : (order_val(fkey(zx), (uint32_t)xb) >= cut);
                const float e = in ? ex2(fmaf(zx, a.c, -kref)) : 0.0f;
                if (!(qx > 0.0f)) stt |= ACES_ROW_BAD_Q;
                else accept = accept_test(ux, qx, e, S_nuc);
            }
            a.ws.acc[(size_t)bq * a.K + iq] = accept;
        }
        a.row_status[r] = stt;
        RowStat rs;
        rs.kref = kref;
        rs.c = a.c;
        rs.S_nuc = S_nuc;
        rs.cut = cut;
        rs.flags = all_in ? RS_ALL_IN : 0;
        rs.nnuc = nnuc;
        a.ws.stats[r] = rs;
    }
    row_finished<NTF>(a, r, smem);
}

// Chunks per sketch group: the smallest power of two >= 4 that keeps the
// sketch within SKETCH_CAP groups; 0 when the fast kernel cannot take the row.
// Four chunks (32 bf16 / 16 fp32 logits) per group keep the sketch at 16 KB
// for a 256000-id bf16 row, which leaves room for four CTAs per SM.
int rows_fast_gc(int dt, int V) {
    const int nch = (int)((size_t)V * (dt == ACES_BF16 ? 2 : 4) / 16);
    const int gmax = 8;  // 16 chunks per group would not fit the register budget
    for (int gc = 4; gc <= gmax; gc *= 2)
        if ((nch + gc - 1) / gc <= SKETCH_CAP) return gc;
    return 0;
}

size_t rows_fast_smem(int dt, int gc, int nch) {
    const size_t skw = dt == ACES_BF16 ? 2 : 4;
    const int ng = (nch + gc - 1) / gc;
    size_t sk = align16((size_t)ng * skw);
    if (sk < (size_t)CAND_CAP_F * 8) sk = (size_t)CAND_CAP_F * 8;
    return sk + (size_t)CAND_CAP_F * 8;
}

template <int DT>
static cudaError_t launch_fast_dt(const RowArgs &a, int gc, size_t smem, cudaStream_t s) {
    void (*fn)(RowArgs) = nullptr;
    switch (gc) {
        case 4: fn = k_rows_fast<DT, 4>; break;
        case 8: fn = k_rows_fast<DT, 8>; break;
        default: break;
    }
    if (!fn) return cudaErrorInvalidValue;
    const cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const long long grid = (long long)a.r_full + (long long)(a.rows - a.r_full) * a.P;
    fn<<<(unsigned)grid, NTF, smem, s>>>(a);
    return cudaGetLastError();
}

template <int DT>
static int per_sm_dt(int gc, size_t smem) {
    void (*fn)(RowArgs) = nullptr;
    switch (gc) {
        case 4: fn = k_rows_fast<DT, 4>; break;
        case 8: fn = k_rows_fast<DT, 8>; break;
        default: return 0;
    }
    if (cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess) return 0;
    int n = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, fn, NTF, smem) != cudaSuccess) return 0;
    return n;
}

// resident CTAs per SM of the fast row kernel (0 when unknown)
int rows_fast_per_sm(int dt, int gc, size_t smem) {
    return dt == ACES_BF16 ? per_sm_dt<ACES_BF16>(gc, smem) : per_sm_dt<ACES_F32>(gc, smem);
}

// one CTA per row r < r_full, P CTAs per later row
cudaError_t launch_rows_fast(const RowArgs &a, int dt, int gc, size_t smem, cudaStream_t s) {
    return dt == ACES_BF16 ? launch_fast_dt<ACES_BF16>(a, gc, smem, s) : launch_fast_dt<ACES_F32>(a, gc, smem, s);
}

}  // namespace aces
