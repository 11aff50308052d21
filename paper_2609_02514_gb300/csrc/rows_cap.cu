// Single-pass row kernel of the AceSpec cloud step (Sec. III-B: accept test
// and packaging of the target distribution; Sec. V-C: compact payload; the
// acceptance rule is the modified rejection sampling of Sec. II-A).
//
// One CTA of 256 threads per target row r = b*(K+1)+i, four CTAs per SM.
// Every logit is read from HBM once, with 16-byte loads, eight in flight per
// thread.  The row is read in tiles of 32 chunks (one coalesced 512-byte warp
// load) in the order t -> (t * pstride) mod ntile, so that the first
// iteration (64 tiles) is a strided sample of the whole row.
//
//   stream    an online exp-sum in log2 units against an integer reference
//             k_t = ceil(max z * log2(e)/T) (one paired FFMA per two logits,
//             one ex2 per logit, exact power-of-two rescales), the max, and a
//             running max shared by the CTA's warps.
//   depth     D bounds how far below the row max the nucleus crossing (top_p
//             = 1: the payload's end) lies: a quantile of the depths that the
//             call's finished rows published, plus a margin (before 32 have
//             finished: those the previous call on the same workspace left,
//             for bfloat16 rows of the same shape; else NSB bins of T/4).  D
//             only decides what is kept; every result below is proved from
//             exact sums.
//   keep      bfloat16, counting pass: every id >= (running max - D)
//             increments a shared-memory counter of its bfloat16 value (a
//             window of HW values); sketch-led pass (when nearly all finished
//             rows had short nuclei): nothing is counted while streaming.
//             Both keep the max of every group of 4 to 8 chunks in a sketch.
//             float32: every 16-byte chunk holding an id >= the threshold is
//             recorded (chunk and index).  The running max only rises, so at
//             the end every id >= (row max - D) was kept (or, sketch-led,
//             lies in a group whose max reaches it).
//   finish    from the exact row max and exp-sum, exact 2^-40 fixed-point
//             masses give the nucleus crossing (a crossing below the kept
//             values: a second counting pass over the row; a capacity
//             exceeded: the exact general kernel):
//             bfloat16  (sketch-led: the groups reaching row max - D are read
//                       back and their ids counted first) one warp scans the
//                       value counts for the crossing value, the number j of
//                       its ids inside the nucleus and the payload's last
//                       value; the sketch's groups whose max reaches that
//                       value are re-read and their ids at or above it
//                       ordered.  When the crossing value's ids are among them
//                       the j-th (in id order) is the cut; otherwise the row
//                       keeps (value, j) and the resolve step finds that id
//                       only for the rows it draws from.
//             float32   the recorded ids are binned by (m - z)/(T/8); the bins
//                       up to the one where a lower bound of the mass reaches
//                       the target are ordered (direct ranking up to 512 ids,
//                       else bin by bin with a rank inside each bin) and one
//                       warp finds the crossing with exact prefix sums.
//             Then the payload, the tail mass, the accept test of the draft
//             token at this position and the per-row state; the CTA that
//             finishes a sequence's last row draws its token when row pi's
//             nucleus was kept.
// On launches of four waves or more, the j-th CTA each SM starts with waits
// j x 10 us first, so that the first wave's epilogues do not coincide.
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
constexpr int NSB = 40;             // depth bins (of T/SPB) of the hints; D before any hint
constexpr int SPB = 4;              // depth bins per temperature
constexpr int MARGIN_BINS = 2;      // float32 first rows: theta below the sample's crossing
constexpr int HINT_MIN = 32;        // finished rows before their depths set D
constexpr int HINT_MARGIN = 2;      // depth bins of margin above that quantile
constexpr float HINT_Q = 0.99f;     // the quantile of the finished rows' depths D covers
// bfloat16
constexpr int HW = 1024;            // counted values (bfloat16 bit patterns) per row
constexpr int HEADROOM = 256;       // of them above the sample's max at least
constexpr int SKG = 16384;          // sketch entries (group maxima, as 16-bit order keys)
constexpr int PCAP = 1024;          // ids at or above the payload's last value
constexpr int GCAP = 1024;          // sketch groups re-read
constexpr int SMEM_BF = HW * 4 + SKG * 2 + PCAP * 8;
// sketch-led pass: a row is short when at most SHORT_IDS ids reach its
// crossing (top_p = 1: when k <= SHORT_IDS); later rows take the pass when
// at least SHORT_NUM / SHORT_DEN of the finished rows were short.  Its areas
// inside the sketch's (in 8-byte units): the ordered ids [0, 1024), the
// groups read back, then the kept ids [2048, 3072), the per-value masses
// [3072, 4096)
constexpr int SHORT_IDS = 256;
constexpr int SHORT_NUM = 49, SHORT_DEN = 50;
constexpr int SK_TMP = 2048, SK_EMASS = 3072;
// float32
constexpr int CREC = 1536;          // recorded chunks (16-byte chunk + its index) per row
constexpr int LCAP = 2048;          // listed ids, expanded from the records after the stream
constexpr int WCAP = 2048;          // work area: ordered candidates
constexpr int SMEM_F32 = CREC * 20 + LCAP * 8 + NBIN * 4;
// float32 rows of a launch that fits one wave at two CTAs per SM take wider
// areas (and a deeper first capture): more records and list entries per row
template <int W>
struct F32Caps {
    static constexpr int CR = W == 2 ? 3584 : CREC;  // recorded chunks
    static constexpr int LC = W == 2 ? 4096 : LCAP;  // listed ids
    static constexpr int WC = W == 2 ? 4096 : WCAP;  // ordered candidates
    static constexpr int MARGIN = W == 2 ? MARGIN_BINS + 2 : MARGIN_BINS;
    static constexpr int SMEM = CR * 20 + LC * 8 + NBIN * 4;
};

constexpr int RANK_MAX = 512;       // ids ordered by direct ranking (more: bitonic sort)
static_assert(WS_DEPTH + NSB <= WS_COUNTERS / 4, "the depth histogram fits the counters area");
static_assert(4 * NUC_CAP * 8 <= SMEM_BF && 4 * NUC_CAP * 8 <= SMEM_F32, "the draw's scratch fits");
static_assert(GCAP * 4 <= HW * 4 && PCAP * 8 <= SKG * 2 && HW <= PCAP, "the aliased areas fit");
static_assert(PCAP <= SK_TMP && GCAP * 4 <= (SK_EMASS - SK_TMP) * 8 && PCAP <= SK_EMASS - SK_TMP &&
                  SK_EMASS + HW <= SKG / 4, "the sketch-led areas fit");
static_assert(WCAP * 8 <= CREC * 20 && RANK_MAX * 2 <= LCAP, "the float32 work areas fit");
static_assert(F32Caps<2>::WC * 8 <= F32Caps<2>::CR * 20 && RANK_MAX * 2 <= F32Caps<2>::LC &&
                  2 * (F32Caps<2>::SMEM + 1024) <= 228 * 1024,
              "the wide float32 areas fit, two CTAs per SM");

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

// 2^(z*c - k) summed over one chunk, as a packed pair of partial sums
template <int DT>
__device__ __forceinline__ unsigned long long chunk_expsum2(const uint4 &x, unsigned long long c2,
                                                            unsigned long long nk2) {
    if (DT == ACES_BF16) {
        const uint32_t wd[4] = {x.x, x.y, x.z, x.w};
        unsigned long long p[4];
#pragma unroll
        for (int q = 0; q < 4; ++q)
            p[q] = ex2_pair(pack2(__uint_as_float(wd[q] << 16), __uint_as_float(wd[q] & 0xFFFF0000u)), c2, nk2);
        return fadd2(fadd2(p[0], p[1]), fadd2(p[2], p[3]));
    } else {
        const unsigned long long p0 = ex2_pair(pack2(__uint_as_float(x.x), __uint_as_float(x.y)), c2, nk2);
        const unsigned long long p1 = ex2_pair(pack2(__uint_as_float(x.z), __uint_as_float(x.w)), c2, nk2);
        return fadd2(p0, p1);
    }
}

// adds a chunk's pair s into the two accumulators (even and odd chunks)
__device__ __forceinline__ void acc_pair(int j, unsigned long long s, unsigned long long &acc0,
                                         unsigned long long &acc1) {
    if (j & 1) acc1 = j == 1 ? s : fadd2(acc1, s);
    else acc0 = j == 0 ? s : fadd2(acc0, s);
}

__device__ __forceinline__ float acc_total(unsigned long long acc0, unsigned long long acc1) {
    float a, b;
    unpack2(fadd2(acc0, acc1), a, b);
    return a + b;
}

// sum over the chunks of 2^(z*c - k), two logits per instruction
template <int DT>
__device__ __forceinline__ float chunks_expsum(const uint4 (&w)[UC], float c, float nk) {
    const unsigned long long c2 = pack2(c, c), nk2 = pack2(nk, nk);
    unsigned long long acc0 = 0ull, acc1 = 0ull;
#pragma unroll
    for (int j = 0; j < UC; ++j) acc_pair(j, chunk_expsum2<DT>(w[j], c2, nk2), acc0, acc1);
    return acc_total(acc0, acc1);
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

// adds 1 to the shared-memory counter at address addr when x < lim (one
// predicated reduction: no branch)
__device__ __forceinline__ void red_inc_lt(uint32_t addr, uint32_t x, uint32_t lim) {
    asm volatile(
        "{\n\t.reg .pred q;\n\tsetp.lt.u32 q, %1, %2;\n\t@q red.shared.add.u32 [%0], 1;\n\t}"
        :: "r"(addr), "r"(x), "r"(lim) : "memory");
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

template <int DT, int W>
__global__ void __launch_bounds__(NTC, 4) k_rows_cap(RowArgs a) {
    constexpr int CREC = F32Caps<W>::CR, LCAP = F32Caps<W>::LC, WCAP = F32Caps<W>::WC;
    constexpr int MARGIN_BINS = F32Caps<W>::MARGIN;
    using E = Elem<DT>;
    constexpr int EPC = E::EPC;
    constexpr bool BF = DT == ACES_BF16;
    extern __shared__ __align__(16) unsigned char smem[];
    // bfloat16: [value counts: HW u32 | sketch: SKG u16 | ids >= the payload's
    //           last value: PCAP u64]; the list of re-read groups reuses the
    //           counts, the ordered ids the sketch, once each is read
    uint32_t *hist = reinterpret_cast<uint32_t *>(smem);
    uint16_t *sk = reinterpret_cast<uint16_t *>(smem + HW * 4);
    unsigned long long *pay = reinterpret_cast<unsigned long long *>(smem + HW * 4 + SKG * 2);
    uint32_t *glist = hist;
    unsigned long long *sorted = reinterpret_cast<unsigned long long *>(sk);
    // float32:  [records: CREC x (16 + 4) bytes | list: LCAP u64 | bin counts:
    //           NBIN u32]; the work area reuses the records once they are expanded
    uint4 *rec_dat = reinterpret_cast<uint4 *>(smem);
    uint32_t *rec_idx = reinterpret_cast<uint32_t *>(smem + CREC * 16);
    unsigned long long *list = reinterpret_cast<unsigned long long *>(smem + CREC * 20);
    uint32_t *bcnt = reinterpret_cast<uint32_t *>(smem + CREC * 20 + LCAP * 8);
    unsigned long long *work = reinterpret_cast<unsigned long long *>(smem);

    __shared__ uint32_t sbin[NWC][NSB];  // float32 estimate: per warp, below the sample max
    __shared__ float redf[NWC], redk[NWC], redh[NWC], redl[NWC];
    __shared__ int s_nrec, s_nl, s_fb, s_n, s_bsel, s_nstar, s_L, s_npay, s_ng, s_nge, s_j, s_vs, s_vk, s_nnuc;
    __shared__ float s_thlo, s_zx;
    __shared__ int s_dbins, s_xb;  // s_dbins: D in depth bins (-1: no hints yet)
    __shared__ int s_skm;          // bfloat16: the sketch-led pass (no counting while streaming)
    __shared__ uint32_t s_mr;  // order key of the running max
    __shared__ double s_Snuc;
    __shared__ float s_inv_S;
    __shared__ unsigned long long s_cut, s_cumL_fx;
    __shared__ unsigned long long s_redu[NWC];

    const int r = blockIdx.x;
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    if (a.stagger_ns > 0 && r < 4 * a.nsm) {
        // the j-th CTA an SM starts with (blocks are placed on the SMs in
        // turn) waits j times stagger_ns on the global timer (bounded: at
        // most 3 x stagger_ns)
        const unsigned long long wait = (unsigned long long)(r / a.nsm) * (unsigned long long)a.stagger_ns;
        const unsigned long long t0 = globaltimer_ns();
        for (int i = 0; i < 1000 && globaltimer_ns() - t0 < wait; ++i) __nanosleep(1000);
    }
    const char *row = reinterpret_cast<const char *>(a.logits) + (size_t)r * a.V * E::SIZE;
    const int nch = a.V / EPC, ntile = a.ntile;
    const int nit = (ntile + TPI - 1) / TPI;
    const uint32_t NI = E::NEG_INF_WORD;
    const bool all_in = a.top_p >= 1.0f;

    // the draft token of this position, fetched early by thread 0 and kept
    // in shared memory across the stream (xb, bq, iq are set after it)
    int xb = -1, bq = 0, iq = 0;
    int xb0 = -1;
    if (a.K > 0 && tid == 0 && r % (a.K + 1) < a.K) xb0 = a.xt[(size_t)(r / (a.K + 1)) * a.K + r % (a.K + 1)];
    if (BF) {
        for (int i = tid; i < HW; i += NTC) hist[i] = 0u;
    } else {
        for (int i = tid; i < NWC * NSB; i += NTC) (&sbin[0][0])[i] = 0u;
    }
    if (tid == 0) {
        s_nrec = 0;
        s_nl = 0;
        s_fb = 0;
        s_nstar = INT_MAX;
        s_mr = fkey(-INFINITY);
    }
    // the depths published by the call's finished rows (read by warp 0 only,
    // once: they change while this row streams)
    int hr = 0, hc0 = 0, hc1 = 0, hs = 0;
    if (wid == 0) {
        hr = __ldcg(&a.ws.fb_count[8]);
        hs = __ldcg(&a.ws.fb_count[11]);
        hc0 = 2 * lane < NSB ? __ldcg(&a.ws.fb_count[WS_DEPTH + 2 * lane]) : 0;
        hc1 = 2 * lane + 1 < NSB ? __ldcg(&a.ws.fb_count[WS_DEPTH + 2 * lane + 1]) : 0;
        if (BF && hr < HINT_MIN) {
            // too few yet: those the previous call on this workspace carried,
            // when it had the same T, top_p, k, V and logit type (bfloat16
            // rows: a float32 row's capture from its own sample overflows
            // less often than from the carried depth)
            const int *cy = a.ws.carry;
            const bool same = __ldcg(cy) == CARRY_MAGIC && __ldcg(cy + 1) == __float_as_int(a.T) &&
                              __ldcg(cy + 2) == __float_as_int(a.top_p) && __ldcg(cy + 3) == a.k &&
                              __ldcg(cy + 4) == a.V && __ldcg(cy + 5) == DT && __ldcg(cy + 6) >= HINT_MIN;
            if (same) {
                hr = __ldcg(cy + 6);
                hs = __ldcg(cy + 7);
                hc0 = 2 * lane < NSB ? __ldcg(cy + WS_DEPTH + 2 * lane) : 0;
                hc1 = 2 * lane + 1 < NSB ? __ldcg(cy + WS_DEPTH + 2 * lane + 1) : 0;
            }
        }
    }

    // ---- stream ----
    float k_t = -1e30f, m_t = -INFINITY, s_t = 0.f, e_t = 0.f;
    uint4 w[UC];
    int tile0 = (int)(((long long)wid * a.pstride) % ntile);  // tile of (iteration 0, u = 0)
    // (iterations whose tiles all exist and are whole load without checks:
    // only the last iteration can hold fewer tiles, and only the row's last
    // tile can be partial)
    // chunk u of iteration it, starting at tile `tile` (checked: bounds tested)
    auto load_chunk = [&](int it, int u, int tile, bool checked) {
        const int t = it * TPI + u * NWC + wid;
        const int c = tile * TCH + lane;
        w[u] = (!checked || (t < ntile && c < nch)) ? ldg16(row + (size_t)c * 16) : make_uint4(NI, NI, NI, NI);
    };
    auto load = [&](int it) {
        int tile = tile0;
        const bool checked = (it + 1) * TPI > ntile || it == a.it_partial;
#pragma unroll
        for (int u = 0; u < UC; ++u) {
            load_chunk(it, u, tile, checked);
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
    // max and exp-sum of this iteration; returns mask_of(th), the iteration's
    // max in im and the maxima of chunks 0..3 and 4..7 in g0, g1
    // the iteration's maxima and the reference k_t raised to them; returns
    // mask_of(th), the iteration's max in im and the maxima of chunks 0..3
    // and 4..7 in g0, g1
    auto head = [&](float th, float &im, float &g0, float &g1) -> uint32_t {
        uint32_t hb = 0u;
        g0 = -INFINITY;
        g1 = -INFINITY;
#pragma unroll
        for (int u = 0; u < UC; ++u) {
            const float cmx = max2_value<DT>(chunk_max2<DT>(w[u]));
            if (u < UC / 2) g0 = fmaxf(g0, cmx);
            else g1 = fmaxf(g1, cmx);
            hb |= (uint32_t)(cmx >= th) << u;
        }
        im = fmaxf(g0, g1);
        m_t = fmaxf(m_t, im);
        const float gk = im * a.c;
        if (gk > k_t) {
            const float nk = ceilf(gk);
            const float sc = pow2_int(k_t - nk);
            s_t *= sc;
            e_t *= sc;
            k_t = nk;
        }
        return hb;
    };
    auto add_sum = [&](float gs) {
        const float t = s_t + gs;  // Neumaier
        if (fabsf(s_t) >= fabsf(gs)) e_t += (s_t - t) + gs;
        else e_t += (gs - t) + s_t;
        s_t = t;
    };
    // max and exp-sum of this iteration (head, then the sum)
    auto math = [&](float th, float &im, float &g0, float &g1) -> uint32_t {
        const uint32_t hb = head(th, im, g0, g1);
        add_sum(chunks_expsum<DT>(w, a.c, -k_t));
        return hb;
    };
    // the running max of the CTA (a lower bound of the row max at any time)
    auto publish_max = [&](float im) {
        const float wm = warp_max(im);
        if (lane == 0 && wm > -INFINITY) atomicMax(&s_mr, fkey(wm));
    };
    auto running_max = [&]() -> float { return fkey_inv(*reinterpret_cast<volatile uint32_t *>(&s_mr)); };

    // iteration 0: a strided sample (1/8 to 1/16 of a large row, spread over it)
    float im, g0, g1;
    load(0);
    math(INFINITY, im, g0, g1);
    // D: how far below the row max the nucleus crossing (top_p = 1: the
    // payload's end) can lie.  Rows of this call that have finished published
    // their depths (in bins of T/4 below their max); the HINT_Q quantile of
    // those depths, plus a margin, sets D (in bins; -1: before HINT_MIN rows
    // have finished, a fixed NSB bins).  One value for the whole CTA.
    if (wid == 0) {
        int inc = hc0 + hc1;
        for (int o = 1; o < 32; o <<= 1) {
            const int t = __shfl_up_sync(0xffffffffu, inc, o);
            if (lane >= o) inc += t;
        }
        const float need = HINT_Q * (float)__shfl_sync(0xffffffffu, inc, 31);
        const int hb = (float)(inc - hc1) >= need ? 2 * lane : ((float)inc >= need ? 2 * lane + 1 : NSB);
        const unsigned bal = __ballot_sync(0xffffffffu, hb < NSB);
        const int hq = bal ? __shfl_sync(0xffffffffu, hb, __ffs(bal) - 1) : NSB - 1;
        if (lane == 0) {
            s_dbins = hr >= HINT_MIN ? min(hq + HINT_MARGIN, NSB - 1) + 1 : -1;
            // the sketch-led pass when nearly every finished row was short
            s_skm = BF && hr >= HINT_MIN && (long long)hs * SHORT_DEN >= (long long)hr * SHORT_NUM;
        }
    }
    publish_max(im);
    if (tid == 0) s_xb = xb0;
    __syncthreads();
    const float m1 = running_max();  // the sample's max
    const bool have = m1 > -INFINITY && m1 < INFINITY;
    const int hbins = s_dbins;
    const bool hinted = have && hbins > 0;
    const float D = (float)(hinted ? hbins : NSB) * (a.T / SPB);

    // dependent loads of the accept test, consumed at the end
    float zx = 0.f, qx = 0.f, ux = 0.f;
    int L = 0;
    unsigned long long *ord = nullptr;  // the payload in order (and, when kept, the nucleus)
    int lazy = 0;
    int nnuc = -1;  // nucleus ids written to the row's list (-1: none)
    float m = -INFINITY, kref = -1e30f;
    double S = 0.0;
    float v_need = 0.0f;  // the crossing (top_p = 1: the payload's end), for the hints
    bool short_row = false;  // (bfloat16) few ids reach the crossing: published for later rows' pass

    // reduces the row max, the reference and the exp-sum (fp32 two-sum tree,
    // fp64 in warp 0); true when the row is not a distribution (handled)
    auto finish_sums = [&]() -> bool {
        if (a.K > 0) {
            bq = r / (a.K + 1);
            iq = r % (a.K + 1);
        }
        xb = tid == 0 ? s_xb : -1;
        if (xb >= 0 && xb < a.V) {
            zx = E::load1(row, xb);
            qx = __ldg(a.q + ((size_t)bq * a.K + iq) * a.V + xb);
            ux = __ldg(a.u + (size_t)bq * (a.K + 1) + iq);
        }
        // each warp: its max, reference kw and exp-sum in units of 2^kw (a
        // compensated fp32 tree over rescales by exact powers of two)
        {
            const float mw = warp_max(m_t), kw = warp_max(k_t);
            const float f = pow2_int(fmaxf(k_t - kw, -1000.0f));
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
                redf[wid] = mw;
                redk[wid] = kw;
                redh[wid] = hi;
                redl[wid] = lo;
            }
        }
        __syncthreads();
        // every thread combines the warps' parts (fp64, exact rescales)
        m = redf[0];
        kref = redk[0];
#pragma unroll
        for (int i = 1; i < NWC; ++i) {
            m = fmaxf(m, redf[i]);
            kref = fmaxf(kref, redk[i]);
        }
        // (fp32 two-sums over exact power-of-two rescales: fp64 is slow here)
        float sh = 0.0f, sl = 0.0f;
#pragma unroll
        for (int i = 0; i < NWC; ++i) {
            const float f = pow2_int(fmaxf(redk[i] - kref, -1000.0f));  // (an integer <= 0)
            float sm, er;
            two_sum(sh, redh[i] * f, sm, er);
            sl += er + redl[i] * f;
            sh = sm;
        }
        const double Sa = (double)sh + (double)sl;
        S = Sa;
        if (!(S > 0.0 && S < 1e300) || !(m < INFINITY) || !(kref < 1e30f)) {
            nonfinite_row<NTC>(a, r);
            row_finished(a, r, smem);
            return true;
        }
        return false;
    };

    if constexpr (BF) {
        // ================= bfloat16: value counts and sketch =================
        // Every id >= lim(running max) is counted in the window of HW values
        // [thb0, thb0 + HW) (positive bit patterns, which sort like the
        // values); the running max only rises, so at the end every id >=
        // lim(row max) has been counted.  The sketch keeps the max of every
        // group of chunks (4 or 8 chunks of one thread and iteration, or 8
        // chunks of 2^ish iterations).
        uint32_t thb0 = 1u;
        bool count_on = false;
        // (the sketch-led pass keeps its work areas past a sketch of at most
        // SK_TMP * 4 slots)
        const int sk_slots = a.sk_gpi == 2 ? nit * NTC * 2 : ((nit + (1 << a.sk_ish) - 1) >> a.sk_ish) * NTC;
        const bool skm = s_skm != 0 && sk_slots <= SK_TMP * 4;
        if (have && m1 > 0.0f && !skm) {
            const float t = m1 - D;
            int lo = t > 0.0f ? (int)__bfloat16_as_ushort(__float2bfloat16_rd(t)) : 1;
            lo = max(lo, (int)(__float_as_uint(m1) >> 16) + HEADROOM - (HW - 1));
            lo = max(lo, 1);
            if (lo + HW - 1 <= 0x7F7F) {  // (then negative values, inf and NaN fall outside)
                count_on = true;
                thb0 = (uint32_t)lo;
            }
        }
        auto lim_of = [&](float mr) -> uint32_t {
            const float t = mr - D;
            uint32_t b = t > 0.0f ? (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rd(t)) : 0u;
            b = b > thb0 ? b : thb0;
            return b < thb0 + HW ? b : thb0 + HW;
        };
        // (the counts' shared-memory address, offset so that a value's bit
        // pattern times 4 indexes its counter)
        const uint32_t hbase = (uint32_t)__cvta_generic_to_shared(hist) - thb0 * 4u;
        // counts the ids of chunk u that reach thb (every lane checks every
        // element: the callers' branches are warp-uniform)
        auto count_chunk = [&](int u, uint32_t thb) {
            const uint32_t span = thb0 + HW - thb;
            const uint32_t wd[4] = {w[u].x, w[u].y, w[u].z, w[u].w};
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const uint32_t lo = wd[q] & 0xFFFFu, hi = wd[q] >> 16;
#ifdef ACES_CHECKED
                if (lo - thb < span && ACES_IN(lo - thb0, HW)) atomicAdd(&hist[lo - thb0], 1u);
                if (hi - thb < span && ACES_IN(hi - thb0, HW)) atomicAdd(&hist[hi - thb0], 1u);
#else
                red_inc_lt(hbase + lo * 4u, lo - thb, span);
                red_inc_lt(hbase + hi * 4u, hi - thb, span);
#endif
            }
        };
        const int gpi = a.sk_gpi, ish = a.sk_ish;
        uint32_t gacc = 0u;
        auto sketch_put = [&](int it) {
            const uint32_t k0 = key16(__float_as_uint(g0) >> 16), k1 = key16(__float_as_uint(g1) >> 16);
            if (gpi == 2) {
                const int s2 = it * NTC + tid;
                if (ACES_IN(2 * s2 + 1, SKG)) reinterpret_cast<uint32_t *>(sk)[s2] = k0 | (k1 << 16);
            } else {
                gacc = max(gacc, max(k0, k1));
                if (((it + 1) & ((1 << ish) - 1)) == 0 || it == nit - 1) {
                    const int s1 = (it >> ish) * NTC + tid;
                    if (ACES_IN(s1, SKG)) sk[s1] = (uint16_t)gacc;
                    gacc = 0u;
                }
            }
        };
        {
            uint32_t thb = count_on ? lim_of(m1) : 0u;
            float thf = count_on ? __uint_as_float(thb << 16) : INFINITY;
            uint32_t hb = mask_of(thf);  // (iteration 0 is loaded and summed)
            for (int it = 0; it < nit; ++it) {
                if (it > 0) {
                    tile0 += a.pstride_it;
                    if (tile0 >= ntile) tile0 -= ntile;
                    load(it);
                    if (count_on) {
                        thb = lim_of(running_max());
                        thf = __uint_as_float(thb << 16);
                    }
                    hb = math(thf, im, g0, g1);
                    publish_max(im);
                }
                if (count_on) {
                    // chunk positions where some lane of the warp reaches thb
                    const uint32_t any = __reduce_or_sync(0xffffffffu, hb);
#pragma unroll
                    for (int u = 0; u < UC; ++u)
                        if ((any >> u) & 1u) count_chunk(u, thb);
                }
                sketch_put(it);
            }
        }
        if (finish_sums()) return;
        const uint32_t km = __float_as_uint(m) >> 16;
        if (a.force_fb || !(m > 0.0f)) {
            if (tid == 0) fallback_row(a, r, m, kref, S);
            return;
        }
        auto vmass = [&](int idx) { return id_fx(val16(0x8000u + thb0 + (uint32_t)idx), a.c, kref); };
        unsigned long long *emass = pay;  // (until the re-read) the mass of one id of each counted value
        // ---- the crossing, the payload's end and the values to re-read,
        // from the counts of values thc..m (warp 0).  Returns 0, or 1 when
        // they lie below the counted values, 2 when more ids than the
        // re-read keeps share the payload's last value ----
        auto scan = [&](uint32_t thc) -> int {
            if (wid == 0) {
                const unsigned long long tg =
                    all_in ? 0ull : (unsigned long long)ceil((double)a.top_p * S * (double)FX_SCALE);
                const int top = (int)(km - thb0), lo = (int)(thc - thb0);
                const int per = (top - lo + 32) >> 5;
                const int b0 = top - lane * per;  // this lane's values: b0, b0 - 1, ... (>= lo)
                unsigned long long lm = 0ull, lc = 0ull;
                for (int i = 0; i < per; ++i) {
                    const int idx = b0 - i;
                    if (idx < lo) break;
                    const uint32_t cn = hist[idx];
                    if (cn) {
                        const unsigned long long e1 = vmass(idx);
                        if (ACES_IN(idx, PCAP)) emass[idx] = e1;
                        lm += (unsigned long long)cn * e1;
                        lc += cn;
                    }
                }
                unsigned long long incm = lm, incc = lc;
                for (int o = 1; o < 32; o <<= 1) {
                    const unsigned long long tm = __shfl_up_sync(0xffffffffu, incm, o);
                    const unsigned long long tc = __shfl_up_sync(0xffffffffu, incc, o);
                    if (lane >= o) {
                        incm += tm;
                        incc += tc;
                    }
                }
                const unsigned long long exm = incm - lm, exc = incc - lc;
                const unsigned long long totc = __shfl_sync(0xffffffffu, incc, 31);
                int fail = 0, vs = -1, jj = 0;
                unsigned long long above = 0ull, cab = 0ull, cnvs = 0ull;
                if (!all_in) {
                    if (exm < tg && incm >= tg) {
                        unsigned long long cm = exm, cc = exc;
                        for (int i = 0; i < per; ++i) {
                            const int idx = b0 - i;
                            if (idx < lo) break;
                            const uint32_t cn = hist[idx];
                            if (!cn) continue;
                            const unsigned long long e1 = emass[idx];
                            const unsigned long long mm = (unsigned long long)cn * e1;
                            if (cm + mm >= tg) {
                                vs = idx;
                                above = cm;
                                cab = cc;
                                cnvs = cn;
                                // the fewest ids of this value reaching the target
                                const unsigned long long rem = tg - cm;
                                unsigned long long q = (unsigned long long)((float)rem / (float)e1);
                                while (q * e1 < rem) ++q;
                                while (q > 1ull && (q - 1ull) * e1 >= rem) --q;
                                jj = (int)q;
                                break;
                            }
                            cm += mm;
                            cc += cn;
                        }
                    }
                    const unsigned bal = __ballot_sync(0xffffffffu, vs >= 0);
                    if (bal) {
                        const int src = __ffs(bal) - 1;
                        vs = __shfl_sync(0xffffffffu, vs, src);
                        jj = __shfl_sync(0xffffffffu, jj, src);
                        above = __shfl_sync(0xffffffffu, above, src);
                        cab = __shfl_sync(0xffffffffu, cab, src);
                        cnvs = __shfl_sync(0xffffffffu, cnvs, src);
                    } else {
                        fail = 1;
                    }
                }
                const unsigned long long nn = all_in ? (unsigned long long)a.V : cab + (unsigned long long)jj;
                const int Lw = fail ? 0 : (int)(nn < (unsigned long long)a.k ? nn : (unsigned long long)a.k);
                if (!fail && (unsigned long long)Lw > totc) fail = 1;  // (top_p = 1) the payload reaches below them
                int vk = -1;
                unsigned long long cabk = 0ull, mabk = 0ull, cnk = 0ull;
                if (!fail && Lw > 0) {
                    const unsigned long long Lu = (unsigned long long)Lw;
                    if (exc < Lu && incc >= Lu) {
                        unsigned long long cm = exm, cc = exc;
                        for (int i = 0; i < per; ++i) {
                            const int idx = b0 - i;
                            if (idx < lo) break;
                            const uint32_t cn = hist[idx];
                            if (!cn) continue;
                            if (cc + cn >= Lu) {
                                vk = idx;
                                cabk = cc;
                                mabk = cm;
                                cnk = cn;
                                break;
                            }
                            cc += cn;
                            cm += (unsigned long long)cn * emass[idx];
                        }
                    }
                    const unsigned bal = __ballot_sync(0xffffffffu, vk >= 0);
                    const int src = bal ? __ffs(bal) - 1 : 0;
                    vk = __shfl_sync(0xffffffffu, vk, src);
                    cabk = __shfl_sync(0xffffffffu, cabk, src);
                    mabk = __shfl_sync(0xffffffffu, mabk, src);
                    cnk = __shfl_sync(0xffffffffu, cnk, src);
                    if (vk < 0) fail = 1;
                }
                // the values to re-read: down to the crossing value when the
                // nucleus is short (then it is kept and the cut is exact),
                // else down to the payload's last value
                int vr = -1;
                unsigned long long nge = 0ull;
                if (!fail) {
                    if (!all_in && cab + cnvs <= (unsigned long long)PCAP && nn <= (unsigned long long)NUC_CAP) {
                        vr = vs;
                        nge = cab + cnvs;
                    } else if (Lw > 0) {
                        vr = vk;
                        nge = cabk + cnk;
                        if (nge > (unsigned long long)PCAP) fail = 2;
                    }
                }
                if (lane == 0) {
                    s_fb = fail;
                    s_vs = vs;
                    s_vk = vr;
                    s_j = jj;
                    s_L = Lw;
                    s_nnuc = all_in ? -1 : (int)(nn < (unsigned long long)INT_MAX ? nn : (unsigned long long)INT_MAX);
                    s_nge = (int)nge;
                    s_ng = 0;
                    s_npay = 0;
                    if (!fail) {
                        const unsigned long long ek = vk >= 0 ? emass[vk] : 0ull;
                        s_cumL_fx = mabk + ((unsigned long long)Lw - cabk) * ek;
                        s_Snuc = all_in ? S : (double)(above + (unsigned long long)jj * emass[vs]) * FX_INV;
                        s_inv_S = inv_mass(s_Snuc);
                    }
                }
            }
            __syncthreads();
            return s_fb;
        };
        // ---- reading groups of the sketch back ----
        const int ng_all = gpi == 2 ? nit * NTC * 2 : ((nit + (1 << ish) - 1) >> ish) * NTC;
        // cnt items of each lane get consecutive places from *ctr (one atomic
        // per warp); returns the lane's first place (all lanes of the warp)
        auto warp_place = [&](int cnt, int *ctr) -> int {
            int inc = cnt;
            for (int o = 1; o < 32; o <<= 1) {
                const int t = __shfl_up_sync(0xffffffffu, inc, o);
                if (lane >= o) inc += t;
            }
            int base = 0;
            if (lane == 31 && inc > 0) base = atomicAdd(ctr, inc);
            return __shfl_sync(0xffffffffu, base, 31) + inc - cnt;
        };
        // lists in gl the slots whose group max (16-bit order key) reaches
        // key; returns their count (all threads)
        auto compact = [&](uint32_t key, uint32_t *gl) -> int {
            if (tid == 0) s_ng = 0;
            __syncthreads();
            const int per_t = ng_all / NTC;  // (at most 64: slot i * NTC + tid)
            unsigned long long hm = 0ull;
            for (int i = 0; i < per_t; ++i) {
                const int slot = i * NTC + tid;
                if (ACES_IN(slot, SKG) && sk[slot] >= key) hm |= 1ull << i;
            }
            int at = warp_place(__popcll(hm), &s_ng);
            __syncthreads();  // (gl may overlap slots of the sketch read above)
            while (hm) {
                const int i = __ffsll((long long)hm) - 1;
                hm &= hm - 1ull;
                if (at < GCAP && ACES_IN(at, GCAP)) gl[at] = (uint32_t)(i * NTC + tid);
                ++at;
            }
            __syncthreads();
            return s_ng;
        };
        // reads the ng groups of gl (one per thread, four chunks at a time) and
        // hands every id whose bit pattern is >= vb (> 0) to put(place, bits,
        // id), places counted by *ctr
        auto reread = [&](const uint32_t *gl, int ng, uint32_t vb, int *ctr, auto put) {
            const int cpt = gpi == 2 ? UC / 2 : UC << ish;  // chunks per group
            for (int g0i = 0; g0i < ng; g0i += NTC) {      // warp-uniform rounds
                const int gi = g0i + tid;
                const bool has = gi < ng;
                const uint32_t slot = has ? gl[gi] : 0u;
                const int tl = gpi == 2 ? (int)((slot >> 1) % NTC) : (int)(slot % NTC);
                const int itg = gpi == 2 ? (int)((slot >> 1) / NTC) : (int)((slot / NTC) << ish);
                const int ub = gpi == 2 ? (int)(slot & 1u) * (UC / 2) : 0;
                for (int q0 = 0; q0 < cpt; q0 += 4) {
                    uint4 dat[4];
                    int cc[4];
#pragma unroll
                    for (int h = 0; h < 4; ++h) {
                        const int q = q0 + h;
                        const int it = itg + q / UC, u = ub + q % UC;
                        const int t = it * TPI + u * NWC + (tl >> 5);
                        cc[h] = -1;
                        if (has && it < nit && t < ntile) {
                            const int c = (int)((long long)t * a.pstride % ntile) * TCH + (tl & 31);
                            if (c < nch) cc[h] = c;
                        }
                        dat[h] = cc[h] >= 0 ? ldg16(row + (size_t)cc[h] * 16) : make_uint4(NI, NI, NI, NI);
                    }
                    uint32_t hm = 0u;
#pragma unroll
                    for (int h = 0; h < 4; ++h) {
                        const uint32_t wd[4] = {dat[h].x, dat[h].y, dat[h].z, dat[h].w};
#pragma unroll
                        for (int e = 0; e < EPC; ++e) {
                            const uint32_t bits = (e & 1) ? wd[e >> 1] >> 16 : wd[e >> 1] & 0xFFFFu;
                            hm |= (uint32_t)(bits - vb < 0x8000u - vb) << (h * EPC + e);
                        }
                    }
                    int at = warp_place(__popc(hm), ctr);
#pragma unroll
                    for (int h = 0; h < 4; ++h) {
                        uint32_t m8 = (hm >> (h * EPC)) & 0xFFu;
                        while (m8) {
                            const int e = __ffs(m8) - 1;
                            m8 &= m8 - 1u;
                            put(at, __float_as_uint(chunk_elem<DT>(dat[h], e)) >> 16, (uint32_t)(cc[h] * EPC + e));
                            ++at;
                        }
                    }
                }
            }
            __syncthreads();
        };
        auto put_pay = [&](int at, uint32_t bits, uint32_t id) {
            if (at < PCAP && ACES_IN(at, PCAP)) pay[at] = order_val(fkey(__uint_as_float(bits << 16)), id);
        };
        // ---- sketch-led pass (rows of a call whose finished rows were
        // short; nothing was counted while streaming).  Every id >= the
        // hinted window's lower end thb0 (row max - D) lies in a group whose
        // max reaches thb0: those groups are read back, their ids >= thb0
        // counted and kept, and the scan of those exact counts follows.
        // Returns 0 (pay holds the ids >= the scan's vr), 1 when the second
        // counting pass is needed, 2 when the row goes to the general kernel ----
        auto sketch_led = [&]() -> int {
            {
                const float t = m - D;
                const uint32_t lb = t > 0.0f ? (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rd(t)) : 1u;
                const uint32_t kfull = km > (uint32_t)(HW - 1) ? km - (uint32_t)(HW - 1) : 1u;
                thb0 = lb > kfull ? lb : kfull;
            }
            uint32_t *gls = reinterpret_cast<uint32_t *>(reinterpret_cast<unsigned long long *>(sk) + SK_TMP);
            const int nc = compact(0x8000u + thb0, gls);  // (ends with a barrier)
            if (nc > GCAP) return 1;
            if (tid == 0) s_npay = 0;
            __syncthreads();
            reread(gls, nc, thb0, &s_npay, [&](int at, uint32_t bits, uint32_t id) {  // (hist is clear)
                const uint32_t idx = bits - thb0;
                if (idx < (uint32_t)HW) atomicAdd(&hist[idx], 1u);
                if (at < PCAP && ACES_IN(at, PCAP)) pay[at] = order_val(fkey(__uint_as_float(bits << 16)), id);
            });
            const int nall = s_npay;
            if (nall > PCAP) return 1;
            emass = reinterpret_cast<unsigned long long *>(sk) + SK_EMASS;
            const int f = scan(thb0);
            if (f != 0) return f;
            // keep in pay the ids >= the scan's vr
            if (s_vk >= 0) {
                const uint32_t kr = fkey(val16(0x8000u + thb0 + (uint32_t)s_vk));
                unsigned long long *tmp = reinterpret_cast<unsigned long long *>(sk) + SK_TMP;
                for (int i0 = 0; i0 < nall; i0 += NTC) {  // warp-uniform rounds
                    const int i = i0 + tid;
                    const unsigned long long o = i < nall ? pay[i] : 0ull;
                    const bool keep = i < nall && (uint32_t)(o >> 32) >= kr;
                    const int at = warp_place(keep ? 1 : 0, &s_npay);
                    if (keep && ACES_IN(at, PCAP)) tmp[at] = o;
                }
                __syncthreads();
                const int nk = s_npay;
                for (int i = tid; i < nk; i += NTC)
                    if (ACES_IN(i, PCAP)) pay[i] = tmp[i];
                __syncthreads();
            }
            return 0;
        };
        int fb = 1;
        bool pay_ready = false;  // (sketch-led) pay holds the ids >= vr
        if (skm) {
            fb = sketch_led();
            pay_ready = fb == 0;
            if (tid == 0 && fb == 0) atomicAdd(&a.ws.fb_count[12], 1);
        } else if (count_on && km < thb0 + HW) {
            fb = scan(lim_of(m));
        }
        if (fb == 1) {
            emass = pay;
            // the crossing (or the row max) lies outside the counted values:
            // a second pass counts the row again, from the row max down as far
            // as the window reaches
            thb0 = km > (uint32_t)(HW - 1) ? km - (uint32_t)(HW - 1) : 1u;
            for (int i = tid; i < HW; i += NTC) hist[i] = 0u;
            __syncthreads();
            const uint32_t span = km + 1u - thb0;
            for (int c0 = 0; c0 < nch; c0 += NTC * UC) {
#pragma unroll
                for (int u = 0; u < UC; ++u) {
                    const int c = c0 + u * NTC + tid;
                    w[u] = c < nch ? ldg16(row + (size_t)c * 16) : make_uint4(NI, NI, NI, NI);
                }
#pragma unroll
                for (int u = 0; u < UC; ++u) {
                    const uint32_t wd[4] = {w[u].x, w[u].y, w[u].z, w[u].w};
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        const uint32_t lo = (wd[q] & 0xFFFFu) - thb0, hi = (wd[q] >> 16) - thb0;
                        if (lo < span && ACES_IN(lo, HW)) atomicAdd(&hist[lo], 1u);
                        if (hi < span && ACES_IN(hi, HW)) atomicAdd(&hist[hi], 1u);
                    }
                }
            }
            __syncthreads();
            if (tid == 0) atomicAdd(&a.ws.fb_count[10], 1);
            fb = scan(thb0);
        }
        if (fb != 0) {
            if (tid == 0) fallback_row(a, r, m, kref, S);
            return;
        }
        L = s_L;
        const int vs = s_vs, j = s_j, vr = s_vk;
        const uint32_t vsb = thb0 + (uint32_t)vs;  // crossing value (bit pattern)
        const bool exact = !all_in && vr == vs;    // every id of the crossing value is read below
        if (vr >= 0) {
            // ---- the ids at or above value vr, then ordered ----
            const uint32_t vrb = thb0 + (uint32_t)vr;  // its bit pattern
            if (!pay_ready) {
                const int ng = compact(0x8000u + vrb, glist);
                if (ng > GCAP) {
                    if (tid == 0) fallback_row(a, r, m, kref, S);
                    return;
                }
                reread(glist, ng, vrb, &s_npay, put_pay);
            }
            const int npay = s_npay;
            if (npay != s_nge) {  // (cannot happen: the counts and the ids agree)
                if (tid == 0) fallback_row(a, r, m, kref, S);
                return;
            }
            // order them (descending order value)
            if (npay <= RANK_MAX) {
                ord = sorted;
                for (int i = tid; i < npay; i += NTC) {
                    const unsigned long long key = pay[i];
                    int rank = 0;
#pragma unroll 4
                    for (int t = 0; t < npay; ++t) rank += pay[t] > key;
                    if (ACES_IN(rank, PCAP)) ord[rank] = key;
                }
            } else {
                if (tid == 0) atomicAdd(&a.ws.fb_count[3], 1);
                ord = pay;
                const int np = next_pow2(npay);
                for (int i = npay + tid; i < np; i += NTC)
                    if (ACES_IN(i, PCAP)) pay[i] = 0ull;
                __syncthreads();
                bitonic_sort_desc(pay, np);
            }
            __syncthreads();
        }
        const int n_nuc = s_nnuc;
        if (tid == 0) {
            if (all_in) {
                s_cut = 0ull;
            } else if (exact) {
                s_cut = ord[n_nuc - 1];
            } else {
                s_cut = ((unsigned long long)fkey(val16(0x8000u + vsb)) << 32) | (unsigned long long)(uint32_t)j;
                atomicAdd(&a.ws.fb_count[5], 1);
            }
            s_zx = zx;
            s_xb = xb;
        }
        // keep the nucleus for the residual step when it fits
        if (exact && a.ws.nuc != nullptr && n_nuc <= NUC_CAP) {
            for (int i = tid; i < n_nuc; i += NTC)
                if (ACES_IN(i, NUC_CAP)) a.ws.nuc[(size_t)r * NUC_CAP + i] = ord[i];
            nnuc = n_nuc;
        }
        lazy = !all_in && !exact;
        __syncthreads();
        // the draft token's value equals the crossing value and that value's
        // ids were not read: its rank among them (ids below it) decides
        if (lazy && s_xb >= 0 && s_xb < a.V && key16(__float_as_uint(s_zx) >> 16) == 0x8000u + vsb) {
            const int xr = s_xb;
            const float vsv = val16(0x8000u + vsb);
            const __nv_bfloat162 v2 = __floats2bfloat162_rn(vsv, vsv);
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
                zx = below < (unsigned long long)j ? vsv : -INFINITY;
            }
        }
        v_need = all_in ? (L > 0 ? order_value(ord[L - 1]) : m) : val16(0x8000u + vsb);
        short_row = all_in ? a.k <= SHORT_IDS : (n_nuc >= 0 && n_nuc <= SHORT_IDS);
        if (tid == 0) atomicAdd(&a.ws.fb_count[2], 1);
    } else {
        // ================= float32: list mode =================
        // Chunks holding an id >= the capture threshold are recorded (16-byte
        // chunk and index).  Hinted rows: the threshold is the running max
        // minus D, so at the end every id >= (row max - D) was recorded.
        // The first rows: the sample's ids within NSB bins of its max are
        // binned; the bins where the sample's mass (from the exact exp-sums)
        // reaches top_p and where its count reaches nmin set a fixed
        // threshold.
        float thlo = INFINITY;
        if (!hinted) {
            if (have) {
#pragma unroll
                for (int u = 0; u < UC; ++u) {
                    const float cmx = max2_value<DT>(chunk_max2<DT>(w[u]));
                    if (!__any_sync(0xffffffffu, (m1 - cmx) * a.inv_ws < (float)NSB)) continue;
#pragma unroll 1  // (unrolled, the independent atomics spill registers)
                    for (int e = 0; e < EPC; ++e) {
                        const float d = (m1 - chunk_elem<DT>(w[u], e)) * a.inv_ws;
                        if (d < (float)NSB && ACES_IN((int)d, NSB)) atomicAdd(&sbin[wid][(int)d], 1u);
                    }
                }
            }
            // the sample's mass in units of 2^((z - m1) c)
            {
                const float kw = warp_max(k_t);
                float sw = (s_t + e_t) * pow2_int(fmaxf(k_t - kw, -1000.0f));
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) sw += __shfl_xor_sync(0xffffffffu, sw, o);
                if (lane == 0) redh[wid] = have ? sw * ex2(kw - m1 * a.c) : 0.0f;
            }
            __syncthreads();
            if (wid == 0 && have) {
                uint32_t c0 = 0u, c1 = 0u;
                float M = 0.0f;
#pragma unroll
                for (int i = 0; i < NWC; ++i) {
                    if (2 * lane < NSB) c0 += sbin[i][2 * lane];
                    if (2 * lane + 1 < NSB) c1 += sbin[i][2 * lane + 1];
                    M += redh[i];
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
                const float f = a.samp_frac;
                // first bin whose cumulative reaches a target (NSB when none)
                auto first_bin = [&](bool h0, bool h1) -> int {
                    const int hb = h0 ? 2 * lane : (h1 ? 2 * lane + 1 : NSB);
                    const unsigned bal = __ballot_sync(0xffffffffu, hb < NSB);
                    return bal ? __shfl_sync(0xffffffffu, hb, __ffs(bal) - 1) : NSB;
                };
                auto bin_of_count = [&](float n) { return first_bin(pc0f >= n * f, (float)pc >= n * f); };
                int blo;
                if (all_in) {
                    blo = bin_of_count((float)a.nmin);
                } else {
                    const float tm = a.top_p * M;
                    const int bx = first_bin(pm0 >= tm, pm >= tm);
                    blo = max(bx + MARGIN_BINS, bin_of_count((float)a.nmin));
                }
                blo = min(blo, NSB - 1);
                if (lane == 0) s_thlo = m1 - (float)(blo + 1) * (a.T / SPB);
            }
            __syncthreads();
            if (have) thlo = s_thlo;
        }
        // records the chunks in hb (those holding an id >= the capture
        // threshold): one vote per iteration, one warp-aggregated atomic per
        // chunk position that has any; the ids are extracted after the stream
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
        {
            float th = hinted ? m1 - D : thlo;
            uint32_t hb = mask_of(th);  // (iteration 0 is loaded and summed)
            for (int it = 0; it < nit; ++it) {
                if (it > 0) {
                    tile0 += a.pstride_it;
                    if (tile0 >= ntile) tile0 -= ntile;
                    load(it);
                    if (hinted) th = running_max() - D;
                    hb = math(th, im, g0, g1);
                    if (hinted) publish_max(im);
                }
                record_hits(hb);
            }
        }
        if (finish_sums()) return;
        const int nrec = s_nrec;
        if (a.force_fb || nrec > CREC) {
            if (tid == 0) fallback_row(a, r, m, kref, S);
            return;
        }
        const float thc = hinted ? m - D : thlo;  // every id >= thc was recorded
        // expand the records: the ids >= thc of every recorded chunk (all such
        // ids lie in recorded chunks), as 64-bit order values
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
                append_cap(list, &s_nl, in && v >= thc, order_val(fkey(v), base + (uint32_t)e), LCAP);
            }
        }
        __syncthreads();
        const int nl = s_nl;
        if (nl > LCAP) {
            if (tid == 0) fallback_row(a, r, m, kref, S);
            return;
        }
        const unsigned long long tg = all_in ? 0ull : (unsigned long long)ceil((double)a.top_p * S * (double)FX_SCALE);
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
            // more: bin by bin (the bins of T/8 below m order the values), and
            // inside a bin by direct ranking among its own ids
            if (tid == 0) atomicAdd(&a.ws.fb_count[3], 1);
            auto bin_of = [&](unsigned long long o) -> int {
                const float d = (m - order_value(o)) * a.inv_w;
                return d < (float)(NBIN - 1) ? (int)d : NBIN - 1;
            };
            if (wid == 0) {  // bcnt[b] <- the first place of bin b (bins 0..bsel hold the candidates)
                constexpr int PER = NBIN / 32;
                uint32_t c[PER], loc = 0u;
#pragma unroll
                for (int j = 0; j < PER; ++j) {
                    const int bn = lane * PER + j;
                    c[j] = bn <= bsel ? bcnt[bn] : 0u;
                    loc += c[j];
                }
                uint32_t inc = loc;
                for (int o = 1; o < 32; o <<= 1) {
                    const uint32_t t = __shfl_up_sync(0xffffffffu, inc, o);
                    if (lane >= o) inc += t;
                }
                uint32_t run = inc - loc;
#pragma unroll
                for (int j = 0; j < PER; ++j) {
                    bcnt[lane * PER + j] = run;
                    run += c[j];
                }
            }
            __syncthreads();
            unsigned long long *binned = list;
            for (int i = tid; i < n; i += NTC) {
                const unsigned long long o = ACES_IN(i, WCAP) ? cv[i] : 0ull;
                const int bn = bin_of(o);
                const uint32_t at = ACES_IN(bn, NBIN) ? atomicAdd(&bcnt[bn], 1u) : 0u;
                if (ACES_IN(at, LCAP)) binned[at] = o;
            }
            __syncthreads();  // (bcnt[b] is now the end of bin b)
            ord = work;
            for (int i = tid; i < n; i += NTC) {
                const unsigned long long o = ACES_IN(i, LCAP) ? binned[i] : 0ull;
                const int bn = bin_of(o);
                const int st = bn > 0 && ACES_IN(bn - 1, NBIN) ? (int)bcnt[bn - 1] : 0;
                const int en = ACES_IN(bn, NBIN) ? (int)bcnt[bn] : 0;
                int rank = 0;
                for (int j = st; j < en; ++j) rank += (ACES_IN(j, LCAP) ? binned[j] : 0ull) > o;
                if (ACES_IN(st + rank, WCAP)) ord[st + rank] = o;
            }
            __syncthreads();
            efx = list;
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

        L = s_L;
        v_need = all_in ? (L > 0 ? order_value(ord[L - 1]) : m) : order_value(s_cut);
    }
    // ---- outputs ----
    if (tid == 0) {  // publish the depth this row needed, for later rows
        const float dxf = (m - v_need) * a.inv_ws;
        const int dx = dxf > 0.0f ? (int)fminf(dxf, (float)(NSB - 1)) : 0;
        if (ACES_IN(dx, NSB)) atomicAdd(&a.ws.fb_count[WS_DEPTH + dx], 1);
        atomicAdd(&a.ws.fb_count[8], 1);
        if (hinted) atomicAdd(&a.ws.fb_count[9], 1);
        if (short_row) atomicAdd(&a.ws.fb_count[11], 1);
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
    a.nmin = 2 * a.k + 64 > 256 ? 2 * a.k + 64 : 256;
    // sketch groups: 4 chunks (two per thread and iteration) when they fit,
    // else 8 chunks of 2^sk_ish iterations
    const int nit = (ntile + TPI - 1) / TPI;
    a.sk_gpi = 2;
    a.sk_ish = 0;
    if ((long long)nit * NTC * 2 > SKG) {
        a.sk_gpi = 1;
        while ((long long)((nit + (1 << a.sk_ish) - 1) >> a.sk_ish) * NTC > SKG) ++a.sk_ish;
    }
}

// The dynamic shared memory above 48 KB needs an opt-in per device, set
// once per device on the first launch there (outside any stream capture).
template <int DT, int W>
static cudaError_t launch_cap_dt(const RowArgs &a, cudaStream_t s) {
    constexpr int smem = DT == ACES_BF16 ? SMEM_BF : F32Caps<W>::SMEM;
    static std::mutex mu;
    static bool ready[64];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    {
        std::lock_guard<std::mutex> lock(mu);
        if (!ready[dev]) {
            const cudaError_t e = cudaFuncSetAttribute(k_rows_cap<DT, W>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
            if (e != cudaSuccess) return e;
            ready[dev] = true;
        }
    }
    k_rows_cap<DT, W><<<(unsigned)a.rows, NTC, smem, s>>>(a);
    return cudaGetLastError();
}

// one CTA per row (16-byte aligned rows)
cudaError_t launch_rows_cap(const RowArgs &a, int dt, cudaStream_t s) {
    if (dt == ACES_BF16) return launch_cap_dt<ACES_BF16, 1>(a, s);
    // (float32: the wide areas when the launch is one wave at two CTAs per SM)
    return a.rows <= 2 * a.nsm ? launch_cap_dt<ACES_F32, 2>(a, s) : launch_cap_dt<ACES_F32, 1>(a, s);
}

#ifdef ACES_CHECKED
cudaError_t check_take_rows_cap(unsigned long long out[3]) { return check_take(out); }
#endif

}  // namespace aces
