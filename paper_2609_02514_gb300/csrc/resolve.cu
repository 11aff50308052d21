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
//   draw_from_list  (common.cuh; run by the fast row kernel's CTA that
//                   finishes a sequence's last row) when row pi's nucleus was
//                   kept (top_p < 1 and at most NUC_CAP ids): the residual
//                   max(0, p - q) is zero outside the nucleus, so q is read at
//                   those ids only, they are ordered by id, and the draw is
//                   taken from their prefix sums.  Identical to the scan
//                   below, whose other terms are all zero.
//   k_resolve_cut   (B x nseg CTAs) when row pi kept its cut as (value v,
//                   count j) (RS_LAZY: the nucleus ends among the ids of one
//                   bfloat16 value, which the row kernel did not list): each
//                   CTA counts the ids of value v in its segment, the last
//                   CTA of the sequence finds the segment holding the j-th
//                   and scans it for that id, the exact cut
//   k_resolve_seg   (B x nseg CTAs) every other sequence: segment sums of
//                   the residual and of p over the whole row
//   k_resolve_pick  (B CTAs) locates the segment holding the draw and scans
//                   it in 2048-id tiles until the crossing id is found
#define ACES_FILE 8  // site numbers of the checked build
#include "common.cuh"

namespace aces {

constexpr int NTR = 256;
constexpr int EPT = 8;               // consecutive ids per thread
constexpr int TILE = NTR * EPT;

// r_fx (residual) and p_fx of ids [x0, x0 + EPT); *bad on a NaN / negative q.
template <int DT, bool VEC>
__device__ __forceinline__ void mass_fx(const char *zrow, const float *qrow, int V, int x0, const RowStat &rs,
                                        float inv_S, unsigned long long rf[EPT], unsigned long long pf[EPT],
                                        int *bad) {
    using E = Elem<DT>;
    float zv[EPT], qv[EPT];
    if (VEC && x0 + EPT <= V) {
        if (DT == ACES_BF16) {
            const uint4 w = ldg16(zrow + (size_t)x0 * 2);
#pragma unroll
            for (int e = 0; e < EPT; ++e) zv[e] = E::get(w, e);
        } else {
            const uint4 w0 = ldg16(zrow + (size_t)x0 * 4), w1 = ldg16(zrow + (size_t)x0 * 4 + 16);
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                zv[e] = Elem<ACES_F32>::get(w0, e);
                zv[e + 4] = Elem<ACES_F32>::get(w1, e);
            }
        }
        if (qrow) {
            const uint4 w0 = ldg16(qrow + x0), w1 = ldg16(qrow + x0 + 4);
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                qv[e] = Elem<ACES_F32>::get(w0, e);
                qv[e + 4] = Elem<ACES_F32>::get(w1, e);
            }
        }
    } else {
#pragma unroll
        for (int e = 0; e < EPT; ++e) {
            const int x = x0 + e;
            zv[e] = x < V ? E::load1(zrow, x) : -INFINITY;
            qv[e] = (qrow && x < V) ? __ldg(qrow + x) : 0.0f;
        }
    }
#pragma unroll
    for (int e = 0; e < EPT; ++e) {
        const int x = x0 + e;
        const float v = zv[e];
        const bool in = x < V && ((rs.flags & RS_ALL_IN) ? (v > -INFINITY)
                                                         : (order_val(fkey(v), (uint32_t)x) >= rs.cut));
        const float p = in ? ex2(fmaf(v, rs.c, -rs.kref)) * inv_S : 0.0f;
        float rr = p;
        if (qrow && x < V) {  // r = max(0, p - q) is 0 where p = 0: q is read where p > 0
            const float qx = qv[e];
            if (in && !(qx >= 0.0f)) *bad = 1;
            rr = in ? fmaxf(p - qx, 0.0f) : 0.0f;
        }
        pf[e] = x < V ? to_fx(p) : 0ull;
        rf[e] = x < V ? to_fx(rr) : 0ull;
    }
}


// ids of [x0, x0 + EPT) whose logit has order key vkey (bit e of the result)
template <int DT, bool VEC>
__device__ __forceinline__ uint32_t ties_of(const char *zrow, int V, int x0, uint32_t vkey) {
    using E = Elem<DT>;
    uint32_t m = 0u;
    if (VEC && x0 + EPT <= V) {
        if (DT == ACES_BF16) {
            const uint4 w = ldg16(zrow + (size_t)x0 * 2);
#pragma unroll
            for (int e = 0; e < EPT; ++e) m |= (uint32_t)(fkey(E::get(w, e)) == vkey) << e;
        } else {
            const uint4 w0 = ldg16(zrow + (size_t)x0 * 4), w1 = ldg16(zrow + (size_t)x0 * 4 + 16);
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                m |= (uint32_t)(fkey(Elem<ACES_F32>::get(w0, e)) == vkey) << e;
                m |= (uint32_t)(fkey(Elem<ACES_F32>::get(w1, e)) == vkey) << (e + 4);
            }
        }
    } else {
#pragma unroll
        for (int e = 0; e < EPT; ++e) {
            const int x = x0 + e;
            if (x < V) m |= (uint32_t)(fkey(E::load1(zrow, x)) == vkey) << e;
        }
    }
    return m;
}

template <int DT, bool VEC>
__global__ void __launch_bounds__(NTR) k_resolve_cut(ResolveArgs a, int nseg, int seglen) {
    using E = Elem<DT>;
    __shared__ int s_pi, s_last, s_seg, s_need, s_id;
    __shared__ unsigned long long red[NTR / 32];
    const int b = blockIdx.x / nseg, sg = blockIdx.x % nseg, tid = threadIdx.x;
    pdl_wait();  // the row kernels are complete
    if (a.ws.fb_count[5] == 0 || a.ws.seqdone[b]) return;  // no cut left open / token already drawn
    if (tid < 32) {
        const int pi0 = first_reject_warp(a.ws, b, a.K);
        if (tid == 0) s_pi = pi0;
    }
    __syncthreads();
    const int r = b * (a.K + 1) + s_pi;
    const RowStat rs = a.ws.stats[r];
    if (!(rs.flags & RS_LAZY)) return;
    const uint32_t vkey = (uint32_t)(rs.cut >> 32);
    const int j = (int)(uint32_t)rs.cut;  // >= 1
    const char *zrow = reinterpret_cast<const char *>(a.logits) + (size_t)r * a.V * E::SIZE;
    const int x_lo = sg * seglen, x_hi = min(a.V, x_lo + seglen);
    unsigned long long cnt = 0ull;
#pragma unroll 4
    for (int x0 = x_lo + tid * EPT; x0 < x_hi; x0 += TILE) cnt += __popc(ties_of<DT, VEC>(zrow, x_hi, x0, vkey));
    const unsigned long long tot = block_reduce_n<NTR>(cnt, red, SumU64());
    if (tid == 0) {
        a.ws.tiecnt[(size_t)b * NSEG_MAX + sg] = (int)tot;
        // releases the count; the last segment acquires the others'
        s_last = atomic_add_acq_rel(&a.ws.cutcnt[b], 1) == nseg - 1;
    }
    __syncthreads();
    if (!s_last) return;
    if (tid == 0) {
        int before = 0, seg = nseg - 1;
        for (int t = 0; t < nseg; ++t) {
            const int c = a.ws.tiecnt[(size_t)b * NSEG_MAX + t];
            if (before + c >= j) {
                seg = t;
                break;
            }
            before += c;
        }
        s_seg = seg;
        s_need = j - before;  // rank (1-based) of the cut among the segment's ties
        s_id = -1;
    }
    __syncthreads();
    const int y_lo = s_seg * seglen, y_hi = min(a.V, y_lo + seglen);
    unsigned long long base = 0ull;
    for (int t0 = y_lo; t0 < y_hi; t0 += TILE) {
        const int x0 = t0 + tid * EPT;
        const uint32_t m = x0 < y_hi ? ties_of<DT, VEC>(zrow, y_hi, x0, vkey) : 0u;
        unsigned long long total;
        const unsigned long long ex = base + block_exscan_n<NTR>((unsigned long long)__popc(m), red, &total);
        const unsigned long long need = (unsigned long long)s_need;
        if (ex < need && need <= ex + (unsigned long long)__popc(m) && ACES_IN(x0, y_hi)) {
            uint32_t mm = m;
            for (unsigned long long q = ex + 1ull; q < need; ++q) mm &= mm - 1u;
            s_id = x0 + __ffs(mm) - 1;
        }
        __syncthreads();
        if (s_id >= 0) break;
        base += total;
    }
    if (tid == 0 && s_id >= 0 && ACES_IN(s_id, a.V)) {
        a.ws.stats[r].cut = order_val(vkey, (uint32_t)s_id);
        a.ws.stats[r].flags = rs.flags & ~RS_LAZY;
    }
}

template <int DT, bool VEC>
__global__ void __launch_bounds__(NTR) k_resolve_seg(ResolveArgs a, int nseg, int seglen) {
    using E = Elem<DT>;
    __shared__ int s_pi;
    __shared__ unsigned long long red[NTR / 32];
    __shared__ int s_bad;
    const int b = blockIdx.x / nseg, sg = blockIdx.x % nseg, tid = threadIdx.x;
    pdl_wait();  // the row kernels are complete
    if (a.ws.seqdone[b]) return;  // drawn from row pi's nucleus list
    const int pi0 = tid < 32 ? first_reject_warp(a.ws, b, a.K) : 0;
    if (tid == 0) {
        const int pi = pi0;
        s_pi = pi;
        s_bad = 0;
        if (sg == 0) a.accept_len[b] = pi;
    }
    __syncthreads();
    const int pi = s_pi;
    const int r = b * (a.K + 1) + pi;
    const RowStat rs = a.ws.stats[r];
    SegSum *out = a.ws.seg + (size_t)b * nseg + sg;
    if (rs.flags & RS_NONFINITE) {
        if (tid == 0) *out = SegSum{0ull, 0ull, 0, 0};
        return;
    }
    const char *zrow = reinterpret_cast<const char *>(a.logits) + (size_t)r * a.V * E::SIZE;
    const float *qrow = pi < a.K ? a.q + ((size_t)b * a.K + pi) * a.V : nullptr;
    const float inv_S = inv_mass(rs.S_nuc);
    const int x_lo = sg * seglen, x_hi = min(a.V, x_lo + seglen);
    unsigned long long sr = 0ull, sp = 0ull;
    int bad = 0;
#pragma unroll 4
    for (int x0 = x_lo + tid * EPT; x0 < x_hi; x0 += TILE) {
        unsigned long long rf[EPT], pf[EPT];
        mass_fx<DT, VEC>(zrow, qrow, x_hi, x0, rs, inv_S, rf, pf, &bad);
#pragma unroll
        for (int e = 0; e < EPT; ++e) {
            sr += rf[e];
            sp += pf[e];
        }
    }
    if (bad) s_bad = 1;
    const unsigned long long tr = block_reduce_n<NTR>(sr, red, SumU64());
    const unsigned long long tp = block_reduce_n<NTR>(sp, red, SumU64());
    if (tid == 0) *out = SegSum{tr, tp, s_bad, 0};
}

template <int DT, bool VEC>
__global__ void __launch_bounds__(NTR) k_resolve_pick(ResolveArgs a, int nseg, int seglen) {
    using E = Elem<DT>;
    __shared__ unsigned long long red[NTR / 32];
    __shared__ int s_seg, s_tok, s_done;
    __shared__ unsigned long long s_base, s_thr;
    __shared__ int s_mode, s_pi;
    const int b = blockIdx.x, tid = threadIdx.x;
    pdl_wait();  // the segment sums are complete
    if (a.ws.seqdone[b]) return;  // drawn from row pi's nucleus list
    const int pi0 = tid < 32 ? first_reject_warp(a.ws, b, a.K) : 0;
    if (tid == 0) {
        s_pi = pi0;
        s_tok = -1;
        s_done = 0;
        s_seg = -1;
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
    if (tid == 0) {
        unsigned long long R = 0ull, P = 0ull;
        int bad = 0;
        for (int s = 0; s < nseg; ++s) {
            R += seg[s].r;
            P += seg[s].p;
            bad |= seg[s].bad;
        }
        int mode = 0;
        if (bad) {
            a.row_status[r] |= ACES_ROW_BAD_Q;
            s_done = 1;
        } else {
            if (R == 0ull) {
                mode = 1;  // p <= q everywhere: draw from p itself
                R = P;
            }
            if (R == 0ull) {
                s_done = 1;
            } else {
                const unsigned long long thr = floor_u_times(a.u[(size_t)b * (a.K + 1) + a.K], R);
                unsigned long long base = 0ull;
                int sg = nseg - 1;
                for (int s = 0; s < nseg; ++s) {
                    const unsigned long long v = mode ? seg[s].p : seg[s].r;
                    if (base + v > thr) {
                        sg = s;
                        break;
                    }
                    base += v;
                }
                s_seg = sg;
                s_base = base;
                s_thr = thr;
            }
        }
        s_mode = mode;
    }
    __syncthreads();
    if (s_done) {
        if (tid == 0) a.out_token[b] = -1;
        return;
    }
    const char *zrow = reinterpret_cast<const char *>(a.logits) + (size_t)r * a.V * E::SIZE;
    const float *qrow = pi < a.K ? a.q + ((size_t)b * a.K + pi) * a.V : nullptr;
    const float inv_S = inv_mass(rs.S_nuc);
    const int mode = s_mode;
    const unsigned long long thr = s_thr;
    const int x_lo = s_seg * seglen, x_hi = min(a.V, x_lo + seglen);
    unsigned long long base = s_base;
    for (int t0 = x_lo; t0 < x_hi; t0 += TILE) {
        const int x0 = t0 + tid * EPT;
        unsigned long long rf[EPT], pf[EPT];
        int bad = 0;
        if (x0 < x_hi) {
            mass_fx<DT, VEC>(zrow, qrow, x_hi, x0, rs, inv_S, rf, pf, &bad);
        } else {
#pragma unroll
            for (int e = 0; e < EPT; ++e) rf[e] = pf[e] = 0ull;
        }
        unsigned long long loc = 0ull;
#pragma unroll
        for (int e = 0; e < EPT; ++e) loc += mode ? pf[e] : rf[e];
        unsigned long long tot;
        const unsigned long long exs = block_exscan_n<NTR>(loc, red, &tot);
        unsigned long long cum = base + exs;
        if (cum <= thr && thr < cum + loc) {
#pragma unroll
            for (int e = 0; e < EPT; ++e) {
                cum += mode ? pf[e] : rf[e];
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
    }
    if (tid == 0) a.out_token[b] = s_tok;
}


// segments of about 8192 ids (four tiles), at most NSEG_MAX per sequence
int resolve_segments(int V) {
    int nseg = (V + 8191) / 8192;
    return nseg < 1 ? 1 : (nseg > NSEG_MAX ? NSEG_MAX : nseg);
}

// The kernels follow the row kernels of the same call and overlap their drain.
cudaError_t launch_resolve(const ResolveArgs &a, int dt, bool vec, cudaStream_t s) {
    const int nseg = resolve_segments(a.V);
    int seglen = (a.V + nseg - 1) / nseg;
    seglen = (seglen + EPT - 1) / EPT * EPT;
    const int g1 = a.B * nseg;
    void (*seg)(ResolveArgs, int, int), (*pick)(ResolveArgs, int, int), (*cut)(ResolveArgs, int, int);
    if (dt == ACES_BF16) {
        cut = vec ? k_resolve_cut<ACES_BF16, true> : k_resolve_cut<ACES_BF16, false>;
        seg = vec ? k_resolve_seg<ACES_BF16, true> : k_resolve_seg<ACES_BF16, false>;
        pick = vec ? k_resolve_pick<ACES_BF16, true> : k_resolve_pick<ACES_BF16, false>;
    } else {
        cut = nullptr;  // only bfloat16 rows leave a cut open
        seg = vec ? k_resolve_seg<ACES_F32, true> : k_resolve_seg<ACES_F32, false>;
        pick = vec ? k_resolve_pick<ACES_F32, true> : k_resolve_pick<ACES_F32, false>;
    }
    cudaError_t e = cudaSuccess;
    if (cut) e = launch_after(cut, (unsigned)g1, NTR, s, a, nseg, seglen);
    if (e != cudaSuccess) return e;
    e = launch_after(seg, (unsigned)g1, NTR, s, a, nseg, seglen);
    if (e != cudaSuccess) return e;
    return launch_after(pick, (unsigned)a.B, NTR, s, a, nseg, seglen);
}

#ifdef ACES_CHECKED
cudaError_t check_take_resolve(unsigned long long out[3]) { return check_take(out); }
#endif

}  // namespace aces
