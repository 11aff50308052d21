// Sequence step of AceSpec verification (Sec. III-B, Algorithm 1): the first
// rejection index pi of each drafted chain and the token emitted at pi,
// drawn from norm(max(0, p_pi - q_pi)) when pi < K (from p_pi itself when
// that is all zero) or from p_K when the whole chain was accepted.
//
// The draw is the smallest id j whose prefix sum over ids 0..j exceeds
// u[b, K] times the total.  Every probability enters as an integer in units
// of 2^-40, so all partial sums are exact and independent of the order in
// which threads add them; the segment sums of pass one and the prefix scan
// of pass two therefore agree bit for bit.
//
//   draw_from_list  (common.cuh; run by the row kernel's CTA that finishes a
//                   sequence's last row) when row pi's nucleus was kept
//                   (top_p < 1 and at most NUC_CAP ids): the residual
//                   max(0, p - q) is zero outside the nucleus, so q is read at
//                   those ids only, they are ordered by id, and the draw is
//                   taken from their prefix sums.  Identical to the scan
//                   below, whose other terms are all zero.
//   k_resolve_seg   every other sequence: sums over segments of row pi of
//                   the residual and of p, added atomically (exact integers)
//                   by warps that each take a few 2048-id tasks (1024 for float32); when row pi
//                   kept its cut as (value v, count j) (RS_LAZY: the nucleus
//                   ends among the ids of one bfloat16 value, which the row
//                   kernel did not list), the ids of value v are summed and
//                   counted apart
//   k_resolve_pick  (B CTAs of 1024 threads) with a lazy cut, scans the
//                   segment holding the j-th id of value v for the residual
//                   of its first ones (the nucleus holds the first j in id
//                   order); then locates the segment holding the draw and
//                   scans it in 8192-id rounds until the crossing id is found
#define ACES_FILE 8  // site numbers of the checked build
#include <cuda_bf16.h>

#include "common.cuh"

namespace aces {

constexpr int EPT = 8;                  // consecutive ids per thread and chunk
constexpr int NTS = 256;                // threads of a segment-sum CTA
constexpr int NTP = 1024;               // threads of a pick CTA
constexpr int PTILE = NTP * EPT;        // ids of a pick round
// chunks per lane in a warp task (its logits are loaded at once: 4 KB of a
// row per warp in flight), and the ids of a task
template <int DT>
struct SegTask {
    static constexpr int WCH = DT == ACES_BF16 ? 8 : 4;
    static constexpr int IDS = 32 * EPT * WCH;
};
static_assert(PTILE % SegTask<ACES_BF16>::IDS == 0 && PTILE % SegTask<ACES_F32>::IDS == 0, "segments of whole tasks");

// the raw 16-byte words of ids [x0, x0 + EPT) (vector path, whole chunk):
// logits in zr (one word for bfloat16, two for float32)
template <int DT>
__device__ __forceinline__ void z_load(const char *zrow, int x0, uint4 (&zr)[2]) {
    if (DT == ACES_BF16) {
        zr[0] = ldg16(zrow + (size_t)x0 * 2);
        zr[1] = make_uint4(0u, 0u, 0u, 0u);
    } else {
        zr[0] = ldg16(zrow + (size_t)x0 * 4);
        zr[1] = ldg16(zrow + (size_t)x0 * 4 + 16);
    }
}

// the logits of ids [x0, x0 + EPT) (-inf at ids >= V): from the words of the
// vector path when the whole chunk lies below V, else one by one
template <int DT, bool VEC>
__device__ __forceinline__ void z_values(const char *zrow, const uint4 (&zr)[2], int V, int x0, float (&zv)[EPT]) {
    using E = Elem<DT>;
    if (VEC && x0 + EPT <= V) {
        if (DT == ACES_BF16) {
#pragma unroll
            for (int e = 0; e < EPT; ++e) zv[e] = E::get(zr[0], e);
        } else {
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                zv[e] = Elem<ACES_F32>::get(zr[0], e);
                zv[e + 4] = Elem<ACES_F32>::get(zr[1], e);
            }
        }
    } else {
#pragma unroll
        for (int e = 0; e < EPT; ++e) zv[e] = x0 + e < V ? E::load1(zrow, x0 + e) : -INFINITY;
    }
}

// q of ids [x0, x0 + EPT) (0 at ids >= V)
template <bool VEC>
__device__ __forceinline__ void q_values(const float *qrow, int V, int x0, float (&qv)[EPT]) {
    if (VEC && x0 + EPT <= V) {
        const uint4 w0 = ldg16(qrow + x0), w1 = ldg16(qrow + x0 + 4);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            qv[e] = Elem<ACES_F32>::get(w0, e);
            qv[e + 4] = Elem<ACES_F32>::get(w1, e);
        }
    } else {
#pragma unroll
        for (int e = 0; e < EPT; ++e) qv[e] = x0 + e < V ? __ldg(qrow + x0 + e) : 0.0f;
    }
}

// membership of ids [x0, x0 + EPT) from their logits zv: bit e of the result
// when id x0 + e is in the nucleus (or holds a lazy cut's value: also in *tie)
__device__ __forceinline__ uint32_t member_bits(const float (&zv)[EPT], int V, int x0, const RowStat &rs,
                                                uint32_t *tie) {
    const bool lazy = (rs.flags & RS_LAZY) != 0;
    const uint32_t vkey = (uint32_t)(rs.cut >> 32);
    uint32_t in = 0u, tm = 0u;
#pragma unroll
    for (int e = 0; e < EPT; ++e) {
        const int x = x0 + e;
        const float v = zv[e];
        bool i, t = false;
        if (!(x < V)) {
            i = false;
        } else if (rs.flags & RS_ALL_IN) {
            i = v > -INFINITY;
        } else if (lazy) {
            const uint32_t k = fkey(v);
            t = k == vkey;
            i = k >= vkey;
        } else {
            i = order_val(fkey(v), (uint32_t)x) >= rs.cut;
        }
        in |= (uint32_t)i << e;
        tm |= (uint32_t)t << e;
    }
    *tie = tm;
    return in;
}

// member_bits of a whole bfloat16 chunk of a lazy cut (value vv) from its
// word, two ids per compare: members are the ids >= vv, ties the ids == vv
// (as order keys: +0 and -0 are one value)
__device__ __forceinline__ uint32_t member_bits_lazy_bf16(const uint4 &w, float vv, uint32_t *tie) {
    const __nv_bfloat162 t2 = __floats2bfloat162_rn(vv, vv);
    const uint32_t wd[4] = {w.x, w.y, w.z, w.w};
    uint32_t in = 0u, tm = 0u;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const __nv_bfloat162 h = *reinterpret_cast<const __nv_bfloat162 *>(&wd[q]);
        const uint32_t ge = __hge2_mask(h, t2), eq = __heq2_mask(h, t2);
        in |= ((ge & 1u) | ((ge >> 15) & 2u)) << (2 * q);
        tm |= ((eq & 1u) | ((eq >> 15) & 2u)) << (2 * q);
    }
    *tie = tm;
    return in;
}

// element e (a run-time index) of eight values
__device__ __forceinline__ float sel8(const float (&v)[EPT], int e) {
    const float a = (e & 1) ? v[1] : v[0], b = (e & 1) ? v[3] : v[2];
    const float c = (e & 1) ? v[5] : v[4], d = (e & 1) ? v[7] : v[6];
    const float lo = (e & 2) ? b : a, hi = (e & 2) ? d : c;
    return (e & 4) ? hi : lo;
}

// the logit of id x0 + e (e a run-time index) of a chunk below V: from its
// words on the vector path, else loaded
template <int DT, bool VEC>
__device__ __forceinline__ float z_at(const char *zrow, const uint4 (&zr)[2], int V, int x0, int e) {
    if (VEC && x0 + EPT <= V) {
        if (DT == ACES_BF16) return Elem<ACES_BF16>::get(zr[0], e);
        return Elem<ACES_F32>::get((e & 4) ? zr[1] : zr[0], e & 3);
    }
    return Elem<DT>::load1(zrow, x0 + e);
}

// the mass of one member id with logit v: p in units of 2^-40 (*pf) and the
// residual max(0, p - q) likewise (return value); *bad on a NaN / negative q
// (q is read where p > 0 only: r = 0 elsewhere)
__device__ __forceinline__ unsigned long long member_mass(float v, float qx, bool has_q, const RowStat &rs,
                                                          float inv_S, unsigned long long *pf, int *bad) {
    const float p = ex2(fmaf(v, rs.c, -rs.kref)) * inv_S;
    float rr = p;
    if (has_q) {
        if (!(qx >= 0.0f)) *bad = 1;
        rr = fmaxf(p - qx, 0.0f);
    }
    *pf = to_fx(p);
    return to_fx(rr);
}

// Segment sums.  The tasks are the 2048-id (float32: 1024) pieces of every sequence's row
// pi, in (sequence, id) order; a warp takes tpw consecutive ones, so that
// it reads a sequence's statistics once and adds its sums once per segment
// (u64 atomics on the cleared sums: exact, and in any order the same).
template <int DT, bool VEC>
__global__ void __launch_bounds__(NTS, 2) k_resolve_seg(ResolveArgs a, int nseg, int seglen, int tps, int tpw) {
    pdl_wait();  // the row kernels are complete
    const int lane = threadIdx.x & 31;
    if (blockIdx.x == 0 && threadIdx.x < WS_COUNTERS / 4) {
        // the hints of this call's rows, for the first rows of the next call
        // with the same shape (the row kernels read them only when fewer
        // than their minimum of this call's rows have finished)
        const int i = threadIdx.x;
        int v = i >= WS_DEPTH ? __ldcg(&a.ws.fb_count[i]) : 0;
        if (i == 0) v = CARRY_MAGIC;
        if (i == 1) v = __float_as_int(a.T);
        if (i == 2) v = __float_as_int(a.top_p);
        if (i == 3) v = a.k;
        if (i == 4) v = a.V;
        if (i == 5) v = DT;
        if (i == 6) v = __ldcg(&a.ws.fb_count[8]);
        if (i == 7) v = __ldcg(&a.ws.fb_count[11]);
        a.ws.carry[i] = v;
    }
    const long long gw = (long long)blockIdx.x * (NTS / 32) + (threadIdx.x >> 5);
    const long long ntask = (long long)a.B * tps;
    const long long t_lo = gw * tpw;
    const long long t_hi = t_lo + tpw < ntask ? t_lo + tpw : ntask;
    int cb = -1, csg = -1;  // sequence and segment of the sums being gathered
    bool skip = true;
    RowStat rs = {};
    const char *zrow = nullptr;
    const float *qrow = nullptr;
    float inv_S = 0.0f, vv = 0.0f;  // vv: the value of a lazy cut
    bool lazy_bf = false;
    unsigned long long sr = 0ull, sp = 0ull, st = 0ull;
    uint32_t nt = 0u;
    int bad = 0;
    auto flush = [&]() {  // (warp-uniform)
        if (csg < 0) return;
        const unsigned long long r_ = warp_sum(sr), p_ = warp_sum(sp), t_ = warp_sum(st);
        const uint32_t n_ = __reduce_add_sync(0xffffffffu, nt);
        const uint32_t bd = __reduce_or_sync(0xffffffffu, (uint32_t)bad);
        const size_t si = (size_t)cb * nseg + csg;
        if (lane == 0 && ACES_IN(si, (size_t)a.B * NSEG_MAX)) {
            SegSum *o = a.ws.seg + si;
            if (r_) atomicAdd(&o->r, r_);
            if (p_) atomicAdd(&o->p, p_);
            if (t_) atomicAdd(&o->tr, t_);
            if (n_) atomicAdd(&o->nt, (int)n_);
            if (bd) atomicOr(&o->bad, 1);
        }
        sr = sp = st = 0ull;
        nt = 0u;
        bad = 0;
        csg = -1;
    };
    for (long long t = t_lo; t < t_hi; ++t) {
        const int b = (int)(t / tps), x_task = (int)(t % tps) * SegTask<DT>::IDS;
        if (b != cb) {
            flush();
            cb = b;
            const int done = a.ws.seqdone[b];
            const int pi = first_reject_warp(a.ws, b, a.K);
            skip = done != 0;  // (drawn from row pi's nucleus list)
            if (!skip) {
                const int r = b * (a.K + 1) + pi;
                rs = a.ws.stats[r];
                skip = (rs.flags & RS_NONFINITE) != 0;
                zrow = reinterpret_cast<const char *>(a.logits) + (size_t)r * a.V * Elem<DT>::SIZE;
                qrow = pi < a.K ? a.q + ((size_t)b * a.K + pi) * a.V : nullptr;
                inv_S = inv_mass(rs.S_nuc);
                lazy_bf = (rs.flags & RS_LAZY) != 0 && !(rs.flags & RS_ALL_IN);
                vv = fkey_inv((uint32_t)(rs.cut >> 32));
            }
        }
        if (skip) continue;
        const int sg = x_task / seglen;
        if (sg != csg) {
            flush();
            csg = sg;
        }
        // the logits of the task's chunks, then q (four chunks at a time)
        // where a chunk has members
        constexpr int WCH = SegTask<DT>::WCH;
        uint4 zr[WCH][2];
#pragma unroll
        for (int i = 0; i < WCH; ++i) {
            const int x0 = x_task + (i * 32 + lane) * EPT;
            if (VEC && x0 + EPT <= a.V) z_load<DT>(zrow, x0, zr[i]);
        }
        unsigned long long inm = 0ull, tmm = 0ull;  // 8 bits per chunk
#pragma unroll
        for (int i = 0; i < WCH; ++i) {
            const int x0 = x_task + (i * 32 + lane) * EPT;
            uint32_t in, tb;
            if (DT == ACES_BF16 && VEC && lazy_bf && x0 + EPT <= a.V) {
                in = member_bits_lazy_bf16(zr[i][0], vv, &tb);
            } else {
                float zv[EPT];
                z_values<DT, VEC>(zrow, zr[i], a.V, x0, zv);
                in = member_bits(zv, a.V, x0, rs, &tb);
            }
            inm |= (unsigned long long)in << (8 * i);
            tmm |= (unsigned long long)tb << (8 * i);
        }
#pragma unroll
        for (int g = 0; g < WCH; g += 4) {
            float qv[4][EPT];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int x0 = x_task + ((g + i) * 32 + lane) * EPT;
                if (qrow && ((inm >> (8 * (g + i))) & 0xFFull)) {
                    q_values<VEC>(qrow, a.V, x0, qv[i]);
                } else {
#pragma unroll
                    for (int e = 0; e < EPT; ++e) qv[i][e] = 0.0f;
                }
            }
            // the members, one per lane and step (the steps of a chunk are
            // the most members any lane holds in it: members are sparse)
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                uint32_t m = (uint32_t)(inm >> (8 * (g + i))) & 0xFFu;
                const uint32_t tb = (uint32_t)(tmm >> (8 * (g + i))) & 0xFFu;
                const int x0 = x_task + ((g + i) * 32 + lane) * EPT;
                while (__any_sync(0xffffffffu, m != 0u)) {
                    if (m) {
                        const int e = __ffs(m) - 1;
                        m &= m - 1u;
                        unsigned long long pfe;
                        const unsigned long long rfe = member_mass(z_at<DT, VEC>(zrow, zr[g + i], a.V, x0, e),
                                                                   sel8(qv[i], e), qrow != nullptr, rs, inv_S,
                                                                   &pfe, &bad);
                        if ((tb >> e) & 1u) {
                            st += rfe;
                            ++nt;
                        } else {
                            sr += rfe;
                            sp += pfe;
                        }
                    }
                }
            }
        }
    }
    flush();
}

// One CTA per sequence: the draw from the segment sums.  With a lazy cut
// (value v, count j) the nucleus holds the first j ids of value v in id
// order: the segment holding the j-th is scanned for the residual of its
// first ones, then the segment holding floor(u * total) is scanned with the
// same rule.
template <int DT, bool VEC>
__global__ void __launch_bounds__(NTP, 1) k_resolve_pick(ResolveArgs a, int nseg, int seglen) {
    __shared__ unsigned long long red[NTP / 32];
    __shared__ int s_tok, s_done, s_pi, s_mode, s_sp, s_sd;
    __shared__ unsigned long long s_need, s_tbd, s_base, s_thr, s_partR;
    const int b = blockIdx.x, tid = threadIdx.x, lane = tid & 31;
    pdl_wait();  // the segment sums are complete
    if (a.ws.seqdone[b]) return;  // drawn from row pi's nucleus list
    if (tid < 32) {
        const int pi0 = first_reject_warp(a.ws, b, a.K);
        if (tid == 0) {
            s_pi = pi0;
            s_tok = -1;
            s_done = 0;
            a.accept_len[b] = pi0;
        }
    }
    __syncthreads();
    const int pi = s_pi;
    const int r = b * (a.K + 1) + pi;
    const RowStat rs = a.ws.stats[r];
    if (rs.flags & RS_NONFINITE) {
        if (tid == 0) a.out_token[b] = -1;
        return;
    }
    const SegSum *seg = a.ws.seg + (size_t)b * nseg;
    const char *zrow = reinterpret_cast<const char *>(a.logits) + (size_t)r * a.V * Elem<DT>::SIZE;
    const float *qrow = pi < a.K ? a.q + ((size_t)b * a.K + pi) * a.V : nullptr;
    const float inv_S = inv_mass(rs.S_nuc);
    const bool lazy = (rs.flags & RS_LAZY) != 0;
    const unsigned long long j = lazy ? (unsigned long long)(uint32_t)rs.cut : 0ull;
    // the mass of one id of the cut's value (the same formula as member_mass)
    const unsigned long long pstar =
        lazy ? to_fx(ex2(fmaf(fkey_inv((uint32_t)(rs.cut >> 32)), rs.c, -rs.kref)) * inv_S) : 0ull;
    // warp 0: the segment holding the j-th id of the cut's value (lane t
    // holds segment t)
    if (tid < 32) {
        const bool ok = lazy && lane < nseg;
        const unsigned long long c = ok ? (unsigned long long)seg[lane].nt : 0ull;
        unsigned long long inc = c;
        for (int o = 1; o < 32; o <<= 1) {
            const unsigned long long v = __shfl_up_sync(0xffffffffu, inc, o);
            if (lane >= o) inc += v;
        }
        const unsigned bal = __ballot_sync(0xffffffffu, ok && inc >= j);
        const int sp = bal ? __ffs(bal) - 1 : -1;
        if (lane == 0) {
            if (lazy && sp < 0) s_done = 1;  // (fewer ids of the cut's value than j: cannot happen)
            s_sp = sp;
            if (!lazy || sp < 0) s_need = 0ull;
        }
        if (sp >= 0 && lane == sp) s_need = j - (inc - c);  // the cut's ids in segment sp inside the nucleus
    }
    __syncthreads();
    if (s_done) {
        if (tid == 0) a.out_token[b] = -1;
        return;
    }
    const int sp = s_sp;
    const unsigned long long need = s_need;
    // the residual of the first `need` ids of the cut's value in segment sp
    if (lazy) {
        const int x_lo = sp * seglen, x_hi = min(a.V, x_lo + seglen);
        unsigned long long seen = 0ull, acc = 0ull;
        for (int t0 = x_lo; t0 < x_hi && seen < need; t0 += PTILE) {
            const int x0 = t0 + tid * EPT;
            float zv[EPT];
            uint4 zr[2];
            if (VEC && x0 + EPT <= x_hi) z_load<DT>(zrow, x0, zr);
            z_values<DT, VEC>(zrow, zr, x_hi, x0, zv);
            uint32_t tm = 0u;
            member_bits(zv, x_hi, x0, rs, &tm);
            unsigned long long ttot;
            unsigned long long rk = seen + block_exscan_n<NTP>((unsigned long long)__popc(tm), red, &ttot);
            unsigned long long loc = 0ull;
            if (tm && rk < need) {
                float qv[EPT];
                if (qrow) {
                    q_values<VEC>(qrow, x_hi, x0, qv);
                } else {
#pragma unroll
                    for (int e = 0; e < EPT; ++e) qv[e] = 0.0f;
                }
                int bad = 0;
#pragma unroll
                for (int e = 0; e < EPT; ++e)
                    if ((tm >> e) & 1u) {
                        unsigned long long pfe;
                        const unsigned long long rfe =
                            member_mass(zv[e], qv[e], qrow != nullptr, rs, inv_S, &pfe, &bad);
                        if (rk < need) loc += rfe;
                        ++rk;
                    }
            }
            acc += block_reduce_n<NTP>(loc, red, SumU64());
            seen += ttot;
        }
        if (tid == 0) s_partR = acc;
    }
    // warp 0: the totals and the segment holding the draw; per segment its
    // weight (residual, or p) with the cut's ids that are in
    if (tid < 32) {
        const unsigned long long partR = lazy ? s_partR : 0ull;
        const bool ok = lane < nseg;
        SegSum sgl = {0ull, 0ull, 0ull, 0, 0};
        if (ok) sgl = seg[lane];
        const unsigned long long ntl = (unsigned long long)sgl.nt;
        const unsigned long long tn = !lazy ? 0ull : (lane < sp ? ntl : (lane == sp ? need : 0ull));
        const unsigned long long trr = !lazy ? 0ull : (lane < sp ? sgl.tr : (lane == sp ? partR : 0ull));
        const unsigned long long wr = ok ? sgl.r + trr : 0ull, wp = ok ? sgl.p + tn * pstar : 0ull;
        unsigned long long R = warp_sum(wr);
        const unsigned long long P = warp_sum(wp);
        const bool bad = __any_sync(0xffffffffu, ok && sgl.bad != 0);
        int mode = 0;
        if (bad) {
            if (lane == 0) {
                a.row_status[r] |= ACES_ROW_BAD_Q;
                s_done = 1;
            }
        } else {
            if (R == 0ull) {
                mode = 1;  // p <= q everywhere: draw from p itself
                R = P;
            }
            if (R == 0ull) {
                if (lane == 0) s_done = 1;
            } else {
                const unsigned long long thr = floor_u_times(a.u[(size_t)b * (a.K + 1) + a.K], R);
                const unsigned long long w = mode ? wp : wr;
                unsigned long long inc = w, tinc = ntl;
                for (int o = 1; o < 32; o <<= 1) {
                    const unsigned long long v = __shfl_up_sync(0xffffffffu, inc, o);
                    const unsigned long long tv = __shfl_up_sync(0xffffffffu, tinc, o);
                    if (lane >= o) {
                        inc += v;
                        tinc += tv;
                    }
                }
                const unsigned bal = __ballot_sync(0xffffffffu, ok && inc > thr);
                const int sd = bal ? __ffs(bal) - 1 : nseg - 1;
                const unsigned long long base = __shfl_sync(0xffffffffu, inc - w, sd);
                const unsigned long long tbd = __shfl_sync(0xffffffffu, tinc - ntl, sd);
                if (lane == 0) {
                    s_sd = sd;
                    s_base = base;
                    s_thr = thr;
                    s_tbd = tbd;  // ids of the cut's value before segment sd
                }
            }
        }
        if (lane == 0) s_mode = mode;
    }
    __syncthreads();
    if (s_done) {
        if (tid == 0) a.out_token[b] = -1;
        return;
    }
    const int mode = s_mode;
    const unsigned long long thr = s_thr;
    unsigned long long base = s_base, rb = s_tbd;
    // the draw: the smallest id whose prefix sum passes thr
    {
        const int x_lo = s_sd * seglen, x_hi = min(a.V, x_lo + seglen);
        for (int t0 = x_lo; t0 < x_hi; t0 += PTILE) {
            const int x0 = t0 + tid * EPT;
            float zv[EPT];
            uint4 zr[2];
            if (VEC && x0 + EPT <= x_hi) z_load<DT>(zrow, x0, zr);
            z_values<DT, VEC>(zrow, zr, x_hi, x0, zv);
            uint32_t tm = 0u;
            uint32_t in = member_bits(zv, x_hi, x0, rs, &tm);
            unsigned long long ttot = 0ull;
            unsigned long long rk = lazy ? rb + block_exscan_n<NTP>((unsigned long long)__popc(tm), red, &ttot) : 0ull;
            // the cut's ids of rank < j are in the nucleus
#pragma unroll
            for (int e = 0; e < EPT; ++e)
                if ((tm >> e) & 1u) {
                    if (!(rk < j)) in &= ~(1u << e);
                    ++rk;
                }
            float qv[EPT];
            if (qrow && !mode && in) {
                q_values<VEC>(qrow, x_hi, x0, qv);
            } else {
#pragma unroll
                for (int e = 0; e < EPT; ++e) qv[e] = 0.0f;
            }
            unsigned long long wv[EPT], loc = 0ull;
            int bad = 0;
#pragma unroll
            for (int e = 0; e < EPT; ++e) {
                wv[e] = 0ull;
                if ((in >> e) & 1u) {
                    unsigned long long pfe;
                    const unsigned long long rfe =
                        member_mass(zv[e], qv[e], qrow != nullptr && !mode, rs, inv_S, &pfe, &bad);
                    wv[e] = mode ? pfe : rfe;
                }
                loc += wv[e];
            }
            unsigned long long tot;
            const unsigned long long exs = block_exscan_n<NTP>(loc, red, &tot);
            unsigned long long cum = base + exs;
            if (cum <= thr && thr < cum + loc) {
#pragma unroll
                for (int e = 0; e < EPT; ++e) {
                    cum += wv[e];
                    if (cum > thr) {
                        s_tok = x0 + e;
                        break;
                    }
                }
                s_done = 1;
            }
            __syncthreads();
            if (s_done) break;
            base += tot;
            rb += ttot;
        }
    }
    if (tid == 0) a.out_token[b] = s_tok;
}

// The kernels follow the row kernels of the same call and overlap their drain.
// Segments: at most NSEG_MAX per sequence, each a whole number of warp tasks.
// The segment-sum warps: about 16 per SM in all (one wave), each with a few tasks.
cudaError_t launch_resolve(const ResolveArgs &a, int dt, bool vec, cudaStream_t s) {
    static int nsm_of[64];
    int dev = 0, nsm = 132;
    if (cudaGetDevice(&dev) == cudaSuccess && dev >= 0 && dev < 64) {
        if (nsm_of[dev] <= 0) {
            int n = 0;
            if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess && n > 0)
                nsm_of[dev] = n;
        }
        if (nsm_of[dev] > 0) nsm = nsm_of[dev];
    }
    const int wtask = dt == ACES_BF16 ? SegTask<ACES_BF16>::IDS : SegTask<ACES_F32>::IDS;
    const int tps = (a.V + wtask - 1) / wtask;  // tasks per sequence
    int nseg = tps < NSEG_MAX ? tps : NSEG_MAX;
    const int seglen = ((a.V + nseg - 1) / nseg + wtask - 1) / wtask * wtask;
    nseg = (a.V + seglen - 1) / seglen;
    const long long ntask = (long long)a.B * tps;
    const long long target = (long long)nsm * 16;
    const int tpw = (int)((ntask + target - 1) / target);
    const long long nwarp = (ntask + tpw - 1) / tpw;
    const unsigned g1 = (unsigned)((nwarp + NTS / 32 - 1) / (NTS / 32));
    void (*seg)(ResolveArgs, int, int, int, int);
    void (*pick)(ResolveArgs, int, int);
    if (dt == ACES_BF16) {
        seg = vec ? k_resolve_seg<ACES_BF16, true> : k_resolve_seg<ACES_BF16, false>;
        pick = vec ? k_resolve_pick<ACES_BF16, true> : k_resolve_pick<ACES_BF16, false>;
    } else {
        seg = vec ? k_resolve_seg<ACES_F32, true> : k_resolve_seg<ACES_F32, false>;
        pick = vec ? k_resolve_pick<ACES_F32, true> : k_resolve_pick<ACES_F32, false>;
    }
    const cudaError_t e = launch_after(seg, g1, NTS, s, a, nseg, seglen, tps, tpw);
    if (e != cudaSuccess) return e;
    return launch_after(pick, (unsigned)a.B, NTP, s, a, nseg, seglen);
}

#ifdef ACES_CHECKED
cudaError_t check_take_resolve(unsigned long long out[3]) { return check_take(out); }
#endif

}  // namespace aces
