// Single-pass row kernel of the AceSpec cloud step (Sec. III-B: accept test
// and packaging of the target distribution; Sec. V-C: compact payload; the
// acceptance rule is the modified rejection sampling of Sec. II-A).
//
// One CTA of 256 threads per target row r = b*(K+1)+i, four CTAs per SM.
// Every logit is read from HBM exactly once, with 16-byte loads, eight in
// flight per thread.  The row is read in tiles of 32 chunks (one coalesced
// 512-byte warp load) in the order t -> (t * pstride) mod ntile, so that the
// first iteration (64 tiles) is a strided sample of the whole row.
//
//   stream    an online exp-sum in log2 units against an integer reference
//             k_t = ceil(max z * log2(e)/T) (one paired FFMA per two logits,
//             one ex2 per logit, exact power-of-two rescales) and the max.
//   estimate  after the first iteration the sample's mass profile (bins of
//             T/4 below its max) gives an estimate of the nucleus crossing
//             and of the logit above which the payload lies; theta is put
//             1.5 T below the estimated crossing (and low enough that about
//             max(4k, 256) ids lie above it).  The estimate only decides what
//             is kept: every result below is proved from exact sums.
//   capture   every id >= theta is kept on chip while the row streams:
//             list mode    (few ids expected; both dtypes): the id's 64-bit
//                          order value goes to a shared-memory list;
//             value mode   (bfloat16, many ids expected, theta > 0): one
//                          shared-memory counter per bfloat16 value in a
//                          window of 1024 values above theta is incremented,
//                          and only ids above a second, higher threshold
//                          (about max(4k, 64) ids) are listed.
//   finish    from the exact row max and exp-sum, exact 2^-40 fixed-point
//             masses prove that the nucleus crossing and the payload lie in
//             the capture (else the row goes to the exact general kernel):
//             list mode    the listed ids are binned by (m - z)/(T/8) with
//                          exact masses; the bins up to the crossing bin are
//                          ordered (direct ranking up to 512 ids, bitonic sort
//                          above) and one warp finds the crossing;
//             value mode   a prefix scan over the value counts gives the
//                          crossing value, the number j of its ids inside the
//                          nucleus and the payload's last value; the listed
//                          payload ids are ranked.  When the crossing value's
//                          ids are listed too, the j-th of them (in id order)
//                          is the cut; otherwise the row keeps (value, j) and
//                          the resolve step finds that id only for the rows it
//                          draws from.
//             Then the payload, the tail mass, the accept test of the draft
//             token at this position and the per-row state; the CTA that
//             finishes a sequence's last row draws its token when row pi's
//             nucleus was listed.
#include <climits>
#include <mutex>
#include <type_traits>

#include <cuda_bf16.h>

#define ACES_FILE 9  // site numbers of the checked build
#include "common.cuh"

namespace aces {

constexpr int NTC = 256;            // threads per CTA
constexpr int NWC = NTC / 32;
constexpr int UC = 8;               // 16-byte chunks per thread and iteration
constexpr int TCH = 32;             // chunks per tile
constexpr int TPI = NWC * UC;       // tiles per iteration
constexpr int NSB = 40;             // sample bins (at most 64: two per lane of a warp)
constexpr int SPB = 4;              // sample bins per temperature
constexpr int MARGIN_BINS = 2;      // theta below the sample's crossing (0.5 T; the sample errs deep)
constexpr int HW = 1024;            // value-mode window (bfloat16 values above theta)
constexpr int CREC = 1536;          // recorded chunks (16-byte chunk + its index) per row
constexpr int LCAP = 2048;          // listed ids, expanded from the records after the stream
constexpr int PCAP = 1024;          // value mode: payload candidates, crossing-value ids
constexpr int VALUE_MIN = 6000;     // expected capture above which value mode is used
constexpr int RANK_MAX = 512;       // ids ordered by direct ranking (more: bitonic sort)
constexpr int WCAP = 2048;          // work area: ordered candidates, or payload + crossing-value ids
// dynamic shared memory: [records: CREC x (16 + 4) bytes | list: LCAP u64 | window: HW u32];
// the work area reuses the records once they are expanded
constexpr int CAP_SMEM = CREC * 20 + LCAP * 8 + HW * 4;
static_assert(WCAP * 8 <= CREC * 20, "the work area fits in the records' place");
constexpr int HINT_MIN = 16;        // finished rows before their depths set theta
constexpr int HINT_MARGIN = 1;      // sample bins of margin below that depth
constexpr float HINT_Q = 0.99f;     // the quantile of the finished rows' depths theta covers
static_assert(WS_DEPTH0 + NSB <= WS_COUNTERS / 4, "the depth histogram fits the counters area");

__device__ __forceinline__ void two_sum(float a, float b, float &s, float &e) {
    s = a + b;
    const float bb = s - a;
    e = (a - (s - bb)) + (b - bb);
}

// 2^d for an integer-valued d <= 0, exactly
__device__ __forceinline__ float pow2_int(float d) {
    return d >= -126.0f ? __int_as_float((127 + __float2int_rn(d)) << 23) : 0.0f;
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

// Max of one chunk, as a packed pair (bfloat16: the max of its even and of
// its odd elements; float32: the max of elements 0,2 and of 1,3).
template <int DT>
__device__ __forceinline__ uint32_t chunk_max2(const uint4 &w) {
    if (DT == ACES_BF16) {
        const __nv_bfloat162 a = __hmax2(*reinterpret_cast<const __nv_bfloat162 *>(&w.x),
                                         *reinterpret_cast<const __nv_bfloat162 *>(&w.y));
        const __nv_bfloat162 b = __hmax2(*reinterpret_cast<const __nv_bfloat162 *>(&w.z),
                                         *reinterpret_cast<const __nv_bfloat162 *>(&w.w));
        const __nv_bfloat162 m = __hmax2(a, b);
        return *reinterpret_cast<const uint32_t *>(&m);
    } else {
        return __float_as_uint(fmaxf(fmaxf(__uint_as_float(w.x), __uint_as_float(w.y)),
                                     fmaxf(__uint_as_float(w.z), __uint_as_float(w.w))));
    }
}
template <int DT>
__device__ __forceinline__ float max2_value(uint32_t m2) {
    if (DT == ACES_BF16) return fmaxf(__uint_as_float(m2 << 16), __uint_as_float(m2 & 0xFFFF0000u));
    return __uint_as_float(m2);
}

// sum over the chunks of 2^(z*c - k), two logits per instruction
template <int DT>
__device__ __forceinline__ float chunks_expsum(const uint4 (&w)[UC], float c, float nk) {
    const unsigned long long c2 = pack2(c, c), nk2 = pack2(nk, nk);
    unsigned long long acc0 = 0ull, acc1 = 0ull;
#pragma unroll
    for (int j = 0; j < UC; ++j) {
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
        if (j & 1) acc1 = j == 1 ? s : fadd2(acc1, s);
        else acc0 = j == 0 ? s : fadd2(acc0, s);
    }
    float a, b;
    unpack2(fadd2(acc0, acc1), a, b);
    return a + b;
}

// element e of a chunk (e may be a run-time index)
template <int DT>
__device__ __forceinline__ float chunk_elem(const uint4 &w, int e) {
    if (DT == ACES_BF16) {
        const uint32_t lo = (e & 4) ? w.z : w.x, hi = (e & 4) ? w.w : w.y;
        const uint32_t wd = (e & 2) ? hi : lo;
        return __uint_as_float((e & 1) ? (wd & 0xFFFF0000u) : (wd << 16));
    } else {
        const uint32_t lo = (e & 2) ? w.z : w.x, hi = (e & 2) ? w.w : w.y;
        return __uint_as_float((e & 1) ? hi : lo);
    }
}

// bits of the chunk's elements >= th (bfloat16: th is a bfloat16 value)
template <int DT>
__device__ __forceinline__ uint32_t chunk_hits(const uint4 &w, float th) {
    if (DT == ACES_BF16) {
        const __nv_bfloat162 t2 = __floats2bfloat162_rn(th, th);
        const uint32_t wd[4] = {w.x, w.y, w.z, w.w};
        uint32_t hm = 0u;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const uint32_t m = __hge2_mask(*reinterpret_cast<const __nv_bfloat162 *>(&wd[q]), t2);
            hm |= ((m & 1u) | ((m >> 15) & 2u)) << (2 * q);
        }
        return hm;
    } else {
        return (uint32_t)(__uint_as_float(w.x) >= th) | (uint32_t)(__uint_as_float(w.y) >= th) << 1 |
               (uint32_t)(__uint_as_float(w.z) >= th) << 2 | (uint32_t)(__uint_as_float(w.w) >= th) << 3;
    }
}

// bfloat16 order key of a bfloat16 bit pattern (keys sort like values, -0
// and +0 share one key), and the value of a key
__device__ __forceinline__ uint32_t key16(uint32_t b) {
    const uint32_t mag = b & 0x7FFFu;
    return (b & 0x8000u) ? 0x8000u - mag : 0x8000u + mag;
}
__device__ __forceinline__ float val16(uint32_t k) {
    const uint32_t b = k >= 0x8000u ? k - 0x8000u : (0x8000u | (0x8000u - k));
    return __uint_as_float(b << 16);
}

// Called by all threads when this CTA has written row r's outputs and state.
// The CTA that finishes the last row of a sequence (rows handed to the
// general kernel are never counted) draws the sequence's token from the
// stored nucleus, so most sequences need no separate resolve launch.
__device__ void row_finished(const RowArgs &a, int r, unsigned char *scratch) {
    if (a.ws.seqcnt == nullptr) return;  // sparsify
    __shared__ int s_last;
    __shared__ unsigned long long s_red[NWC];
    __shared__ DrawShared s_draw;
    const int b = r / (a.K + 1);
    __syncthreads();  // every thread's writes of this row are issued
    // releases this row's writes; the last row acquires the others'
    if (threadIdx.x == 0) s_last = atomic_add_acq_rel(&a.ws.seqcnt[b], 1) == a.K;
    __syncthreads();
    if (!s_last) return;
    unsigned long long *skey = reinterpret_cast<unsigned long long *>(scratch);  // 4 * NUC_CAP entries
    draw_from_list<NTC>(a.ws, a.q, a.u, a.K, a.V, b, a.accept_len, a.out_token, a.row_status, skey,
                        skey + NUC_CAP, skey + 2 * NUC_CAP, skey + 3 * NUC_CAP, s_red, &s_draw);
}

// Hands row r to the general kernel with its max m and its exp-sum S (in
// units of 2^kref), which spare that kernel a pass and the exponentials of
// another (the row is finite: rows with NaN or +inf are marked NONFINITE
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
// shuffle tree: three dependent fp64 adds instead of eight in one thread)
__device__ __forceinline__ double warp0_mass(const float *hi, const float *lo, int lane) {
    double v = lane < NWC ? (double)hi[lane] + (double)lo[lane] : 0.0;
#pragma unroll
    for (int o = NWC / 2; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// appends o to arr[*n] for every lane with take (one atomic per warp); *n
// may pass cap, entries beyond it are dropped (all lanes of the warp call it)
__device__ __forceinline__ void append_cap(unsigned long long *arr, int *n, bool take, unsigned long long o, int cap) {
    const unsigned bal = __ballot_sync(0xffffffffu, take);
    if (bal == 0u) return;
    const int lane = threadIdx.x & 31;
    int base = 0;
    if (lane == __ffs(bal) - 1) base = atomicAdd(n, __popc(bal));
    base = __shfl_sync(0xffffffffu, base, __ffs(bal) - 1);
    const int pos = base + __popc(bal & ((1u << lane) - 1u));
    if (take && pos < cap) arr[pos] = o;
}

// mass of one id of logit v in 2^-40 units (the same formula in every kernel)
__device__ __forceinline__ unsigned long long id_fx(float v, float c, float kref) {
    return to_fx(ex2(fmaf(v, c, -kref)));
}

template <int DT>
__global__ void __launch_bounds__(NTC, 4) k_rows_cap(RowArgs a) {
    using E = Elem<DT>;
    constexpr int EPC = E::EPC;
    constexpr bool BF = DT == ACES_BF16;
    extern __shared__ __align__(16) unsigned char smem[];
    uint4 *rec_dat = reinterpret_cast<uint4 *>(smem);                                  // CREC
    uint32_t *rec_idx = reinterpret_cast<uint32_t *>(smem + CREC * 16);                 // CREC
    unsigned long long *list = reinterpret_cast<unsigned long long *>(smem + CREC * 20);  // LCAP
    uint32_t *hist = reinterpret_cast<uint32_t *>(smem + CREC * 20 + LCAP * 8);         // HW (value mode)
    unsigned long long *work = reinterpret_cast<unsigned long long *>(smem);            // WCAP, after expansion
    // list-mode bin counts alias the value window (never both in one row)
    uint32_t *bcnt = hist;

    __shared__ uint32_t sbin[NWC][NSB];  // per warp, relative to the warp's own max
    __shared__ float redf[NWC], redk[NWC], redh[NWC], redl[NWC];
    __shared__ int s_nrec, s_nl, s_mode, s_fb, s_n, s_bsel, s_nstar, s_L, s_npay, s_ntie, s_vs, s_vk, s_j, s_nn;
    __shared__ float s_thlo, s_thpay, s_zx, s_m1;
    __shared__ int s_xb;
    __shared__ double s_S, s_Snuc;
    __shared__ float s_inv_S;
    __shared__ unsigned long long s_cut, s_cumL_fx, s_above, s_cab;
    __shared__ unsigned long long s_redu[NWC];

    const int r = blockIdx.x;
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    const char *row = reinterpret_cast<const char *>(a.logits) + (size_t)r * a.V * E::SIZE;
    const int nch = a.V / EPC, ntile = a.ntile;
    const uint32_t NI = E::NEG_INF_WORD;
    const bool all_in = a.top_p >= 1.0f;

    // the draft token of this position, fetched early by thread 0
    int xb = -1, bq = 0, iq = 0;
    if (a.K > 0) {
        bq = r / (a.K + 1);
        iq = r % (a.K + 1);
        if (tid == 0 && iq < a.K) xb = a.xt[(size_t)bq * a.K + iq];
    }
    for (int i = tid; i < NWC * NSB; i += NTC) (&sbin[0][0])[i] = 0u;
    if (BF)
        for (int i = tid; i < HW; i += NTC) hist[i] = 0u;
    if (tid == 0) s_nrec = 0;

    // ---- stream ----
    float k_t = -1e30f, m_t = -INFINITY, s_t = 0.f, e_t = 0.f;
    uint4 w[UC];
    int tile0 = (int)(((long long)wid * a.pstride) % ntile);  // tile of (iteration 0, u = 0)
    // (iterations whose tiles all exist and are whole load without checks:
    // only the last iteration can hold fewer tiles, and only the row's last
    // tile can be partial)
    auto load = [&](int it) {
        int tile = tile0;
        const bool checked = (it + 1) * TPI > ntile || it == a.it_partial;
#pragma unroll
        for (int u = 0; u < UC; ++u) {
            const int t = it * TPI + u * NWC + wid;
            const int c = tile * TCH + lane;
            w[u] = (!checked || (t < ntile && c < nch)) ? ldg16(row + (size_t)c * 16) : make_uint4(NI, NI, NI, NI);
            tile += a.pstride_w;
            if (tile >= ntile) tile -= ntile;
        }
    };
    // bit u: chunk u holds an id >= th
    auto mask_of = [&](float th) -> uint32_t {
        uint32_t hb = 0u;
#pragma unroll
        for (int u = 0; u < UC; ++u) hb |= (uint32_t)(max2_value<DT>(chunk_max2<DT>(w[u])) >= th) << u;
        return hb;
    };
    // max and exp-sum of this iteration; returns mask_of(th)
    auto math = [&](float th) -> uint32_t {
        float im = -INFINITY;
        uint32_t hb = 0u;
#pragma unroll
        for (int u = 0; u < UC; ++u) {
            const float cmx = max2_value<DT>(chunk_max2<DT>(w[u]));
            im = fmaxf(im, cmx);
            hb |= (uint32_t)(cmx >= th) << u;
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
        const float gs = chunks_expsum<DT>(w, a.c, -k_t);
        const float t = s_t + gs;  // Neumaier
        if (fabsf(s_t) >= fabsf(gs)) e_t += (s_t - t) + gs;
        else e_t += (gs - t) + s_t;
        s_t = t;
        return hb;
    };
    // records the chunks in hb (those holding an id >= the capture
    // threshold): one vote per iteration, one warp-aggregated atomic per chunk
    // position that has any; the ids are extracted after the stream
    auto record_hits = [&](uint32_t hb) {
        if (!__any_sync(0xffffffffu, hb != 0u)) return;
        int tile = tile0;
#pragma unroll
        for (int u = 0; u < UC; ++u) {
            const bool hit = (hb >> u) & 1u;
            const unsigned bal = __ballot_sync(0xffffffffu, hit);
            if (bal != 0u) {
                const int lead = __ffs(bal) - 1;
                int base = 0;
                if (lane == lead) base = atomicAdd(&s_nrec, __popc(bal));
                base = __shfl_sync(0xffffffffu, base, lead);
                if (hit) {
                    const int at = base + __popc(bal & ((1u << lane) - 1u));
                    if (at < CREC && ACES_IN(at, CREC)) {
                        rec_dat[at] = w[u];
                        rec_idx[at] = (uint32_t)(tile * TCH + lane);
                    }
                }
            }
            tile += a.pstride_w;
            if (tile >= ntile) tile -= ntile;
        }
    };
    // value mode: one count per id of each bfloat16 value in [theta, theta + HW
    // values), branch-free (theta > 0: the bit patterns of positive values are
    // their order, and every other id falls outside the window); ids above the
    // window are caught by the max check at the end
    auto count_all = [&](uint32_t thb) {
#pragma unroll
        for (int u = 0; u < UC; ++u) {
            const uint32_t wd[4] = {w[u].x, w[u].y, w[u].z, w[u].w};
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const uint32_t rl = (wd[q] & 0xFFFFu) - thb, rh = (wd[q] >> 16) - thb;
                if (rl < (uint32_t)HW && ACES_IN(rl, HW)) atomicAdd(&hist[rl], 1u);
                if (rh < (uint32_t)HW && ACES_IN(rh, HW)) atomicAdd(&hist[rh], 1u);
            }
        }
    };

    // iteration 0: the sample.  Each warp bins its ids near its own max
    // (bins of T/SPB, NSB of them); warp 0 aligns the warps' bins and takes
    // the sample's mass from the exact exp-sums.
    load(0);
    math(INFINITY);
    {
        const float mw = warp_max(m_t);
        // every id of the sample within NSB bins of the warp's max is binned
        // (few are); chunks holding none are skipped by a vote
        if (mw > -INFINITY && mw < INFINITY) {
#pragma unroll
            for (int u = 0; u < UC; ++u) {
                const float cmx = max2_value<DT>(chunk_max2<DT>(w[u]));
                if (!__any_sync(0xffffffffu, (mw - cmx) * a.inv_ws < (float)NSB)) continue;
#pragma unroll 1  // (unrolled, the independent atomics spill registers)
                for (int e = 0; e < EPC; ++e) {
                    const float d = (mw - chunk_elem<DT>(w[u], e)) * a.inv_ws;
                    if (d < (float)NSB && ACES_IN((int)d, NSB)) atomicAdd(&sbin[wid][(int)d], 1u);
                }
            }
        }
        // the sample's mass: this warp's exp-sum against its largest reference
        const float kw = warp_max(k_t);
        float sw = (s_t + e_t) * pow2_int(fmaxf(k_t - kw, -1000.0f));
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) sw += __shfl_xor_sync(0xffffffffu, sw, o);
        if (lane == 0) {
            redf[wid] = mw;
            redk[wid] = kw;
            redh[wid] = sw;
        }
    }
    __syncthreads();
    float m1 = redf[0];
#pragma unroll
    for (int i = 1; i < NWC; ++i) m1 = fmaxf(m1, redf[i]);
    const bool have = m1 > -INFINITY && m1 < INFINITY;
    if (wid == 0 && have) {
        // bins 2 * lane and 2 * lane + 1 below m1, from the warps' bins shifted
        // by the (rounded) distance of their maxima; the sample's mass in units
        // of 2^((z - m1) c) from the warps' sums
        uint32_t c0 = 0u, c1 = 0u;
        float M = 0.0f;
#pragma unroll
        for (int i = 0; i < NWC; ++i) {
            const float mwi = redf[i];
            if (!(mwi > -INFINITY)) continue;
            const int off = __float2int_rn((m1 - mwi) * a.inv_ws);
            const int s0 = 2 * lane - off, s1 = 2 * lane + 1 - off;
            if (s0 >= 0 && s0 < NSB) c0 += sbin[i][s0];
            if (s1 >= 0 && s1 < NSB) c1 += sbin[i][s1];
            M += redh[i] * ex2(redk[i] - m1 * a.c);
        }
        constexpr float L2B = 1.4426950408889634f / SPB;
        const float ms0 = (float)c0 * ex2(-(2 * lane + 0.5f) * L2B), ms1 = (float)c1 * ex2(-(2 * lane + 1.5f) * L2B);
        float pm = ms0 + ms1;
        uint32_t pc = c0 + c1;
        for (int o = 1; o < 32; o <<= 1) {
            const float tm = __shfl_up_sync(0xffffffffu, pm, o);
            const uint32_t tc = __shfl_up_sync(0xffffffffu, pc, o);
            if (lane >= o) {
                pm += tm;
                pc += tc;
            }
        }
        const float pm0 = pm - ms1, pc0f = (float)(pc - c1);  // cumulative through bin 2*lane
        // first bin whose cumulative reaches a target (NSB when none)
        auto first_bin = [&](bool h0, bool h1) -> int {
            const int hb = h0 ? 2 * lane : (h1 ? 2 * lane + 1 : NSB);
            const unsigned bal = __ballot_sync(0xffffffffu, hb < NSB);
            return bal ? __shfl_sync(0xffffffffu, hb, __ffs(bal) - 1) : NSB;
        };
        const float f = a.samp_frac;
        auto bin_of_count = [&](float n) { return first_bin(pc0f >= n * f, (float)pc >= n * f); };
        int blo;
        if (all_in) {
            blo = bin_of_count((float)a.nmin);
        } else {
            const float tm = a.top_p * M;
            const int bx = first_bin(pm0 >= tm, pm >= tm);
            blo = max(bx + MARGIN_BINS, bin_of_count((float)a.nmin));
        }
        // rows of this call already finished: the depth (crossing or payload
        // end, whichever is deeper) that HINT_Q of them needed sets theta
        // instead; a row that needs more falls back to the exact kernel
        const int hrows = __ldcg(&a.ws.fb_count[8]);
        if (hrows >= HINT_MIN) {
            const int h0 = 2 * lane < NSB ? __ldcg(&a.ws.fb_count[WS_DEPTH0 + 2 * lane]) : 0;
            const int h1 = 2 * lane + 1 < NSB ? __ldcg(&a.ws.fb_count[WS_DEPTH0 + 2 * lane + 1]) : 0;
            int hc = h0 + h1, hi = hc;
            for (int o = 1; o < 32; o <<= 1) {
                const int t = __shfl_up_sync(0xffffffffu, hi, o);
                if (lane >= o) hi += t;
            }
            const int htot = __shfl_sync(0xffffffffu, hi, 31);
            const float need = HINT_Q * (float)htot;
            const int hb0 = (float)(hi - h1) >= need ? 2 * lane : ((float)hi >= need ? 2 * lane + 1 : NSB);
            const unsigned hbal = __ballot_sync(0xffffffffu, hb0 < NSB);
            const int hd = hbal ? __shfl_sync(0xffffffffu, hb0, __ffs(hbal) - 1) : NSB - 1;
            blo = hd + HINT_MARGIN;
            (void)hc;
        }
        blo = min(blo, NSB - 1);
        // expected ids >= theta
        const float cum_lo = __shfl_sync(0xffffffffu, (blo & 1) ? (float)pc : pc0f, blo >> 1);
        const float n_est = cum_lo / f;
        const float thlo = m1 - (float)(blo + 1) * (a.T / SPB);
        int mode = 0;  // list mode
        float thpay = thlo;
        if (BF && !all_in && n_est > (float)VALUE_MIN && thlo > 0.0f) {
            mode = 1;  // value mode
            const int bp = min(bin_of_count((float)a.npay), blo);
            thpay = m1 - (float)(bp + 1) * (a.T / SPB);
        }
        if (lane == 0) {
            float tl = thlo, tp = thpay;
            if (BF) {  // thresholds are bfloat16 values (rounded down)
                tl = __bfloat162float(__float2bfloat16_rd(tl));
                tp = __bfloat162float(__float2bfloat16_rd(tp));
                if (mode == 1 && !(tl > 0.0f)) tl = __uint_as_float(0x00010000u);  // smallest positive
                if (tp < tl) tp = tl;
            }
            s_thlo = tl;
            s_thpay = tp;
            s_mode = mode;
            s_m1 = m1;
        }
    }
    __syncthreads();
    const int mode = have ? s_mode : 0;
    const float thlo = have ? s_thlo : INFINITY;  // no estimate: keep nothing
    const float thpay = have ? s_thpay : INFINITY;
    const int nit = (ntile + TPI - 1) / TPI;
    if (mode == 0) {
        uint32_t hb = mask_of(thlo);  // (iteration 0 is loaded and summed)
        for (int it = 0; it < nit; ++it) {
            if (it > 0) {
                tile0 += a.pstride_it;
                if (tile0 >= ntile) tile0 -= ntile;
                load(it);
                hb = math(thlo);
            }
            record_hits(hb);
        }
    } else {
        const uint32_t thb = __float_as_uint(thlo) >> 16;  // bit pattern of theta (> 0)
        uint32_t hb = mask_of(thpay);
        for (int it = 0; it < nit; ++it) {
            if (it > 0) {
                tile0 += a.pstride_it;
                if (tile0 >= ntile) tile0 -= ntile;
                load(it);
                hb = math(thpay);
            }
            count_all(thb);
            record_hits(hb);
        }
    }
    // dependent loads of the accept test, consumed at the end
    float zx = 0.f, qx = 0.f, ux = 0.f;
    if (xb >= 0 && xb < a.V) {
        zx = E::load1(row, xb);
        qx = __ldg(a.q + ((size_t)bq * a.K + iq) * a.V + xb);
        ux = __ldg(a.u + (size_t)bq * (a.K + 1) + iq);
    }

    // ---- row max, reference and exp-sum (fp32 two-sum tree, fp64 in warp 0) ----
    {
        const float mw = warp_max(m_t), kw = warp_max(k_t);
        if (lane == 0) {
            redf[wid] = mw;
            redk[wid] = kw;
        }
    }
    __syncthreads();
    float m = redf[0], kref = redk[0];
#pragma unroll
    for (int i = 1; i < NWC; ++i) {
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
    __syncthreads();
    if (wid == 0) {
        const double S = warp0_mass(redh, redl, lane);
        if (lane == 0) {
            s_S = S;
            s_fb = 0;
            s_nstar = INT_MAX;
        }
    }
    __syncthreads();
    const double S = s_S;
    if (!(S > 0.0 && S < 1e300) || !(m < INFINITY) || !(kref < 1e30f)) {
        nonfinite_row<NTC>(a, r);
        row_finished(a, r, smem);
        return;
    }
    const int nrec = s_nrec;
    if (a.force_fb || nrec > CREC) {
        if (tid == 0) fallback_row(a, r, m, kref, S);
        return;
    }
    // expand the records: the ids >= the capture threshold of every recorded
    // chunk (all such ids lie in recorded chunks), as 64-bit order values
    {
        const float th = mode == 0 ? thlo : thpay;
        if (tid == 0) s_nl = 0;
        __syncthreads();
        for (int i0 = 0; i0 < nrec; i0 += NTC) {  // warp-uniform rounds
            const int i = i0 + tid;
            const bool in = i < nrec;
            const uint4 dat = in ? rec_dat[i] : make_uint4(NI, NI, NI, NI);
            const uint32_t base = in ? rec_idx[i] * (uint32_t)EPC : 0u;
#pragma unroll
            for (int e = 0; e < EPC; ++e) {
                const float v = Elem<DT>::get(dat, e);
                append_cap(list, &s_nl, in && v >= th, order_val(fkey(v), base + (uint32_t)e), LCAP);
            }
        }
        __syncthreads();
    }
    const int nl = s_nl;
    if (nl > LCAP) {
        if (tid == 0) fallback_row(a, r, m, kref, S);
        return;
    }
    const unsigned long long tg = all_in ? 0ull : (unsigned long long)ceil((double)a.top_p * S * (double)FX_SCALE);
    unsigned long long *ord;  // the first ids of the nucleus in order (at least the payload)
    int lazy = 0;
    int nnuc = -1;            // nucleus ids written to the row's list (-1: none)

    if (mode == 0) {
        // ================= list mode =================
        // counts of the listed ids in bins of T/8 below m; a bin's ids each
        // carry at least its lower edge's mass, so the first bin where that
        // lower bound of the cumulative mass reaches the target holds or
        // follows the crossing (top_p = 1: the first bin where the count
        // reaches k).  The exact crossing is found below among the ids of
        // the bins up to it.
        for (int i = tid; i < NBIN; i += NTC) bcnt[i] = 0u;
        __syncthreads();
        for (int i = tid; i < nl; i += NTC) {
            const float d = (m - order_value(list[i])) * a.inv_w;
            const int bn = d < (float)(NBIN - 1) ? (int)d : NBIN - 1;
            if (ACES_IN(bn, NBIN)) atomicAdd(&bcnt[bn], 1u);
        }
        __syncthreads();
        if (wid == 0) {
            constexpr int PER = NBIN / 32;
            // lower edge of bin b in units of 2^kref: 2^(m c - kref) 2^(-(b+1) log2(e)/8)
            const float base2 = ex2(fmaf(m, a.c, -kref));
            constexpr float L2E8 = 1.4426950408889634f / BIN_PER_T;
            float lm = 0.0f;
            unsigned lc = 0u;
#pragma unroll
            for (int j = 0; j < PER; ++j) {
                const int bn = lane * PER + j;
                lm += (float)bcnt[bn] * base2 * ex2(-(float)(bn + 1) * L2E8);
                lc += bcnt[bn];
            }
            float pm = lm;
            unsigned pc = lc;
            for (int o = 1; o < 32; o <<= 1) {
                const float tm = __shfl_up_sync(0xffffffffu, pm, o);
                const unsigned tc = __shfl_up_sync(0xffffffffu, pc, o);
                if (lane >= o) {
                    pm += tm;
                    pc += tc;
                }
            }
            pm -= lm;
            pc -= lc;
            // 1e-4 covers the fp32 rounding of the bound and of S
            const float tgf = (float)((double)a.top_p * S) * (1.0f + 1e-4f);
            int hit = -1;
            unsigned ncand = 0u;
#pragma unroll
            for (int j = 0; j < PER; ++j) {
                const int bn = lane * PER + j;
                pm += (float)bcnt[bn] * base2 * ex2(-(float)(bn + 1) * L2E8) * (1.0f - 1e-4f);
                pc += bcnt[bn];
                const bool okb = all_in ? (pc >= (unsigned)a.k) : (pm >= tgf);
                if (okb && hit < 0) {
                    hit = bn;
                    ncand = pc;
                }
            }
            const unsigned bal = __ballot_sync(0xffffffffu, hit >= 0);
            const int src = bal ? __ffs(bal) - 1 : 0;
            const int bsel = __shfl_sync(0xffffffffu, hit, src);
            const unsigned nc = __shfl_sync(0xffffffffu, ncand, src);
            // no bin reaches the bound: take every listed id (the exact sums
            // below still decide whether they hold the crossing); top_p = 1
            // with fewer than k listed ids goes to the exact kernel (the row
            // may hold finite ids below theta)
            if (lane == 0) {
                s_fb = all_in && bal == 0u;
                s_bsel = bal ? bsel : NBIN - 1;
                s_n = bal ? (int)nc : nl;
                s_npay = 0;
            }
        }
        __syncthreads();
        if (s_fb || s_n > WCAP) {
            if (tid == 0) fallback_row(a, r, m, kref, S);
            return;
        }
        // candidates: the listed ids in bins up to bsel
        const int bsel = s_bsel, n = s_n;
        unsigned long long *cv = work;
        for (int i0 = 0; i0 < nl; i0 += NTC) {  // warp-uniform rounds
            const int i = i0 + tid;
            unsigned long long o = 0ull;
            bool take = false;
            if (i < nl) {
                o = list[i];
                const float d = (m - order_value(o)) * a.inv_w;
                const int bn = d < (float)(NBIN - 1) ? (int)d : NBIN - 1;
                take = bn <= bsel;
            }
            const unsigned bal = __ballot_sync(0xffffffffu, take);
            if (bal == 0u) continue;
            int base = 0;
            if (lane == __ffs(bal) - 1) base = atomicAdd(&s_npay, __popc(bal));
            base = __shfl_sync(0xffffffffu, base, __ffs(bal) - 1);
            const int at = base + __popc(bal & ((1u << lane) - 1u));
            if (take && ACES_IN(at, WCAP)) cv[at] = o;
        }
        __syncthreads();
        // order them (descending order value) into ord[], masses into efx[]
        unsigned long long *efx;
        if (n <= RANK_MAX) {
            ord = list;
            efx = list + RANK_MAX;
            for (int i = tid; i < n; i += NTC) {
                const unsigned long long v = cv[i];
                int rank = 0;
#pragma unroll 4
                for (int j = 0; j < n; ++j) rank += cv[j] > v;
                if (ACES_IN(rank, RANK_MAX)) {
                    ord[rank] = v;
                    efx[rank] = id_fx(order_value(v), a.c, kref);
                }
            }
        } else {
            if (tid == 0) atomicAdd(&a.ws.fb_count[3], 1);
            ord = list;
            efx = work;
            const int np = next_pow2(n);
            for (int i = tid; i < np; i += NTC)
                if (ACES_IN(i, LCAP)) ord[i] = i < n ? cv[i] : 0ull;
            __syncthreads();
            bitonic_sort_desc(ord, np);
            for (int i = tid; i < n; i += NTC)
                if (ACES_IN(i, WCAP)) efx[i] = id_fx(order_value(ord[i]), a.c, kref);
        }
        __syncthreads();
        // nucleus crossing with exact fixed-point prefix sums (warp 0)
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
                s_cumL_fx = cL;
                const double sn = all_in ? S : (double)cN * FX_INV;
                s_Snuc = sn;
                s_inv_S = inv_mass(sn);
                s_cut = (nstar != INT_MAX && !all_in) ? ord[nstar] : 0ull;
            }
        }
        __syncthreads();
        if (s_nstar == INT_MAX) {
            if (tid == 0) fallback_row(a, r, m, kref, S);
            return;
        }
        // keep the nucleus for the residual step when it fits
        nnuc = (a.ws.nuc != nullptr && !all_in && s_nstar + 1 <= NUC_CAP) ? s_nstar + 1 : -1;
        if (nnuc > 0)
            for (int i = tid; i < nnuc; i += NTC)
                if (ACES_IN(i, NUC_CAP)) a.ws.nuc[(size_t)r * NUC_CAP + i] = ord[i];
    } else {
        // ================= value mode (bfloat16) =================
        const uint32_t thk = key16(__float_as_uint(thlo) >> 16);
        const uint32_t km = key16(__float_as_uint(m) >> 16);
        if (km - thk >= (uint32_t)HW) {  // ids above the window were not counted
            if (tid == 0) fallback_row(a, r, m, kref, S);
            return;
        }
        if (tid == 0) atomicAdd(&a.ws.fb_count[2], 1);
        // prefix scan over the values, highest first, four per thread
        constexpr int PERV = HW / NTC;
        const int d0 = tid * PERV;  // values thk + HW - 1 - d0 - i
        auto vmass = [&](int i, uint32_t cn) -> unsigned long long {
            return cn ? (unsigned long long)cn * id_fx(val16(thk + (uint32_t)(HW - 1 - d0 - i)), a.c, kref) : 0ull;
        };
        uint32_t cnv[PERV];
        unsigned long long bm = 0ull, bc = 0ull;
#pragma unroll
        for (int i = 0; i < PERV; ++i) {
            cnv[i] = hist[HW - 1 - d0 - i];
            bm += vmass(i, cnv[i]);
            bc += cnv[i];
        }
        if (tid == 0) {
            s_vs = -1;
            s_vk = -1;
        }
        unsigned long long mtot, ctot;
        const unsigned long long mex = block_exscan_n<NTC>(bm, s_redu, &mtot);
        const unsigned long long cex = block_exscan_n<NTC>(bc, s_redu, &ctot);
        {
            unsigned long long cmv = mex, ccv = cex;
#pragma unroll
            for (int i = 0; i < PERV; ++i) {
                const unsigned long long mm = vmass(i, cnv[i]);
                if (cnv[i] && cmv < tg && cmv + mm >= tg) {
                    const unsigned long long e1 = mm / cnv[i];
                    s_vs = HW - 1 - d0 - i;
                    s_above = cmv;
                    s_cab = ccv;
                    s_j = (int)((tg - cmv + e1 - 1) / e1);
                }
                cmv += mm;
                ccv += cnv[i];
            }
        }
        __syncthreads();
        if (s_vs < 0) {  // the counted ids hold too little mass
            if (tid == 0) fallback_row(a, r, m, kref, S);
            return;
        }
        const unsigned long long n_nuc = s_cab + (unsigned long long)s_j;
        const int L = (int)(n_nuc < (unsigned long long)a.k ? n_nuc : (unsigned long long)a.k);
        if (L > 0) {
            unsigned long long ccv = cex;
#pragma unroll
            for (int i = 0; i < PERV; ++i) {
                if (ccv < (unsigned long long)L && ccv + cnv[i] >= (unsigned long long)L) s_vk = HW - 1 - d0 - i;
                ccv += cnv[i];
            }
        }
        if (tid == 0) {
            s_npay = 0;
            s_ntie = 0;
            s_nn = 0;
        }
        __syncthreads();
        const uint32_t vsk = thk + (uint32_t)s_vs;                       // crossing value's key
        const uint32_t vkk = L > 0 ? thk + (uint32_t)s_vk : 0xFFFFFFFFu;  // last payload value's key
        const uint32_t tpk = key16(__float_as_uint(thpay) >> 16);
        if (L > 0 && vkk < tpk) {  // payload ids below the listed range
            if (tid == 0) fallback_row(a, r, m, kref, S);
            return;
        }
        const bool exact = vsk >= tpk;  // the crossing value's ids are listed
        const bool keep = exact && a.ws.nuc != nullptr && n_nuc <= (unsigned long long)NUC_CAP;
        unsigned long long *pay = work, *tie = work + PCAP;
        for (int i0 = 0; i0 < nl; i0 += NTC) {  // warp-uniform rounds
            const int i = i0 + tid;
            unsigned long long o = 0ull;
            uint32_t kk = 0u;
            if (i < nl) {
                o = list[i];
                kk = key16(__float_as_uint(order_value(o)) >> 16);
            }
            const bool in = i < nl;
            append_cap(pay, &s_npay, in && kk >= vkk, o, PCAP);
            append_cap(tie, &s_ntie, in && exact && kk == vsk, o, PCAP);
            if (keep) {  // nucleus ids above the crossing value
                const bool tk = in && kk > vsk;
                const unsigned bal = __ballot_sync(0xffffffffu, tk);
                if (bal) {
                    int base = 0;
                    if (lane == __ffs(bal) - 1) base = atomicAdd(&s_nn, __popc(bal));
                    base = __shfl_sync(0xffffffffu, base, __ffs(bal) - 1);
                    const int at = base + __popc(bal & ((1u << lane) - 1u));
                    if (tk && ACES_IN(at, NUC_CAP)) a.ws.nuc[(size_t)r * NUC_CAP + at] = o;
                }
            }
        }
        __syncthreads();
        const int npay = s_npay, ntie = s_ntie;
        if (npay > PCAP || ntie > PCAP) {
            if (tid == 0) fallback_row(a, r, m, kref, S);
            return;
        }
        // rank: the first L payload ids go to ord (the list is no longer
        // needed), the crossing value's id of rank j - 1 is the cut
        ord = list;
        const int LL = L < npay ? L : npay;
        for (int i = tid; i < npay; i += NTC) {
            const unsigned long long key = pay[i];
            int rank = 0;
#pragma unroll 4
            for (int t = 0; t < npay; ++t) rank += pay[t] > key;
            if (rank < LL && ACES_IN(rank, LCAP)) ord[rank] = key;
        }
        const int j = s_j;
        if (exact) {
            const int nb = s_nn;
            for (int i = tid; i < ntie; i += NTC) {
                const unsigned long long key = tie[i];
                int rank = 0;
#pragma unroll 4
                for (int t = 0; t < ntie; ++t) rank += tie[t] > key;
                if (rank == j - 1) s_cut = key;
                if (keep && rank < j && ACES_IN(nb + rank, NUC_CAP)) a.ws.nuc[(size_t)r * NUC_CAP + nb + rank] = key;
            }
        }
        if (keep) nnuc = (int)n_nuc;
        // exact sum of the payload masses, for the tail
        unsigned long long loc = 0ull;
        __syncthreads();
        for (int i = tid; i < LL; i += NTC) loc += id_fx(order_value(ord[i]), a.c, kref);
        const unsigned long long cumL = block_reduce_n<NTC>(loc, s_redu, SumU64());
        if (tid == 0) {
            const float vsv = val16(vsk);
            const unsigned long long es = id_fx(vsv, a.c, kref);
            const unsigned long long snfx = s_above + (unsigned long long)j * es;
            s_Snuc = (double)snfx * FX_INV;
            s_inv_S = inv_mass(s_Snuc);
            s_cumL_fx = cumL;
            s_L = LL;
            if (!exact) {
                s_cut = ((unsigned long long)fkey(vsv) << 32) | (unsigned long long)(uint32_t)j;
                atomicAdd(&a.ws.fb_count[5], 1);
            }
            s_zx = zx;
            s_xb = xb;
        }
        lazy = !exact;
        __syncthreads();
        // the draft token's value equals the crossing value and that value's
        // ids were not listed: its rank among them (ids below it) decides
        if (lazy && s_xb >= 0 && s_xb < a.V && key16(__float_as_uint(s_zx) >> 16) == vsk) {
            const int xr = s_xb;
            const __nv_bfloat162 v2 = __floats2bfloat162_rn(val16(vsk), val16(vsk));
            uint32_t cnt = 0u;
            for (int cc = tid; cc * EPC < xr; cc += NTC) {
                const uint4 wv = ldg16(row + (size_t)cc * 16);
                const uint32_t wd[4] = {wv.x, wv.y, wv.z, wv.w};
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const uint32_t mk = __heq2_mask(*reinterpret_cast<const __nv_bfloat162 *>(&wd[q]), v2);
                    const int x0 = cc * EPC + 2 * q;
                    cnt += ((mk & 1u) && x0 < xr) + ((mk >> 16 & 1u) && x0 + 1 < xr);
                }
            }
            const unsigned long long below = block_reduce_n<NTC>((unsigned long long)cnt, s_redu, SumU64());
            if (tid == 0) {
                atomicAdd(&a.ws.fb_count[7], 1);
                // x~ is in the nucleus iff fewer than j ids of its value precede it
                s_zx = below < (unsigned long long)j ? 1.0f : 0.0f;
            }
            __syncthreads();
            if (tid == 0) zx = s_zx > 0.0f ? val16(vsk) : -INFINITY;  // in: keep its value; out: mass 0
        }
    }
    // ---- outputs ----
    const int L = s_L;
    if (tid == 0) {  // publish the depths this row needed, for later rows
        const float vx = all_in ? m : (lazy ? fkey_inv((uint32_t)(s_cut >> 32)) : order_value(s_cut));
        const float vl = L > 0 ? order_value(ord[L - 1]) : m;
        const float m1s = s_m1;  // the sample max (written by the estimate, which ran: no fallback here)
        const float dxf = (m1s - vx) * a.inv_ws, dkf = (m1s - vl) * a.inv_ws;
        const int dx = all_in ? 0 : (dxf > 0.0f ? (int)fminf(dxf, (float)(NSB - 1)) : 0);
        const int dk = dkf > 0.0f ? (int)fminf(dkf, (float)(NSB - 1)) : 0;
        const int dd = max(dx, dk);
        if (ACES_IN(dd, NSB)) atomicAdd(&a.ws.fb_count[WS_DEPTH0 + dd], 1);
        atomicAdd(&a.ws.fb_count[8], 1);
    }
    const float inv_S = s_inv_S;
    for (int j = tid; j < a.k; j += NTC) {
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
                bool in;
                if (all_in) in = zx > -INFINITY;
                else if (lazy) in = fkey(zx) >= (uint32_t)(cut >> 32);  // ties were decided above
                else in = order_val(fkey(zx), (uint32_t)xb) >= cut;
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
        rs.flags = (all_in ? RS_ALL_IN : 0) | (lazy ? RS_LAZY : 0);
        rs.nnuc = nnuc;
        a.ws.stats[r] = rs;
    }
    row_finished(a, r, smem);
}

static int gcd_int(int x, int y) {
    while (y) {
        const int t = x % y;
        x = y;
        y = t;
    }
    return x;
}

// Tile order and sample size of a row of a.V elements of type dt: the
// stride is the smallest integer >= ntile / TPI coprime with ntile, so the
// first TPI tiles are spread over the whole row.
void rows_cap_layout(RowArgs &a, int dt) {
    const int epc = dt == ACES_BF16 ? 8 : 4;
    const int nch = a.V / epc;
    const int ntile = (nch + TCH - 1) / TCH;
    int p = ntile / TPI;
    if (p < 1) p = 1;
    while (gcd_int(p, ntile) != 1) ++p;
    a.ntile = ntile;
    a.pstride = p;
    a.pstride_w = (int)((long long)NWC * p % ntile);
    a.pstride_it = (int)((long long)TPI * p % ntile);
    long long samp = 0;
    const int first = ntile < TPI ? ntile : TPI;
    for (int t = 0; t < first; ++t) {
        const long long tile = (long long)t * p % ntile;
        const long long c0 = tile * TCH, c1 = c0 + TCH < nch ? c0 + TCH : nch;
        samp += (c1 - c0) * epc;
    }
    a.samp_frac = (float)((double)samp / (double)a.V);
    a.it_partial = -1;  // the iteration that reads the partial last tile
    if (nch % TCH != 0)
        for (int t = 0; t < ntile; ++t)
            if ((long long)t * p % ntile == ntile - 1) {
                a.it_partial = t / TPI;
                break;
            }
    a.inv_ws = (float)(SPB / (double)a.T);
    a.nmin = 4 * a.k > 256 ? 4 * a.k : 256;
    a.npay = 4 * a.k > 64 ? 4 * a.k : 64;
}

// The dynamic shared memory above 48 KB needs an opt-in per device, set
// once per device on the first launch there (outside any stream capture).
template <int DT>
static cudaError_t launch_cap_dt(const RowArgs &a, cudaStream_t s) {
    static std::mutex mu;
    static bool ready[64];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    {
        std::lock_guard<std::mutex> lock(mu);
        if (!ready[dev]) {
            const cudaError_t e = cudaFuncSetAttribute(k_rows_cap<DT>, cudaFuncAttributeMaxDynamicSharedMemorySize, CAP_SMEM);
            if (e != cudaSuccess) return e;
            ready[dev] = true;
        }
    }
    k_rows_cap<DT><<<(unsigned)a.rows, NTC, CAP_SMEM, s>>>(a);
    return cudaGetLastError();
}

// one CTA per row (16-byte aligned rows)
cudaError_t launch_rows_cap(const RowArgs &a, int dt, cudaStream_t s) {
    return dt == ACES_BF16 ? launch_cap_dt<ACES_BF16>(a, s) : launch_cap_dt<ACES_F32>(a, s);
}

#ifdef ACES_CHECKED
cudaError_t check_take_rows_cap(unsigned long long out[3]) { return check_take(out); }
#endif

}  // namespace aces
