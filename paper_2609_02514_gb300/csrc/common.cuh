// Device helpers shared by the AceSpec kernels (sm_103a).
#pragma once
#include <cuda_runtime.h>
#include <float.h>
#include <stdint.h>

#include "../../include/acespec.h"

namespace aces {

// ---------------------------------------------------------------------------
// Checked build (compiled with -DACES_CHECKED, for tests).  ACES_IN(i, n) is
// true when 0 <= i < n; otherwise it records the first violation met in this
// translation unit -- the site (file number * 10000 + line), the index and
// the bound -- in a device word, and the caller skips the access (a store)
// or reads nothing (a load).  Nothing traps.  In the normal build it is the
// constant true and costs nothing.  Each .cu file defines ACES_FILE (its
// number) before including this header.
#ifndef ACES_FILE
#define ACES_FILE 0
#endif
#ifdef ACES_CHECKED
static __device__ unsigned long long g_check[3];  // site (0: none), index, bound
static __device__ __noinline__ bool check_fail(long long i, long long n, int site) {
    if (atomicCAS(&g_check[0], 0ull, (unsigned long long)site) == 0ull) {
        g_check[1] = (unsigned long long)i;
        g_check[2] = (unsigned long long)n;
        __threadfence();
    }
    return false;
}
#define ACES_IN(i, n)                                                              \
    ((unsigned long long)(long long)(i) < (unsigned long long)(long long)(n)       \
         ? true                                                                    \
         : ::aces::check_fail((long long)(i), (long long)(n), ACES_FILE * 10000 + __LINE__))
// reads this translation unit's word into out[3] and clears it
static inline cudaError_t check_take(unsigned long long out[3]) {
    cudaError_t e = cudaMemcpyFromSymbol(out, g_check, sizeof(g_check));
    if (e != cudaSuccess) return e;
    const unsigned long long z[3] = {0ull, 0ull, 0ull};
    return cudaMemcpyToSymbol(g_check, z, sizeof(z));
}
cudaError_t check_take_rows_cap(unsigned long long out[3]);
cudaError_t check_take_rows_general(unsigned long long out[3]);
cudaError_t check_take_resolve(unsigned long long out[3]);
cudaError_t check_take_cache(unsigned long long out[3]);
cudaError_t check_take_resample(unsigned long long out[3]);
cudaError_t check_take_kv(unsigned long long out[3]);
cudaError_t check_take_mask(unsigned long long out[3]);
#else
#define ACES_IN(i, n) true
#endif

constexpr int NT = 512;             // threads per CTA for the general row kernel
constexpr int NWARP = NT / 32;
constexpr int NBIN = 256;           // bins of width T/8 below the row max
constexpr int BIN_PER_T = 8;

// Row-level flags kept in the workspace.
constexpr int RS_ALL_IN = 1;        // top_p >= 1: every finite id is in the nucleus
constexpr int RS_NONFINITE = 2;
// handed to the general kernel: kref holds the row max, c the log2 reference
// of the row's exp-sum and S_nuc that exp-sum
constexpr int RS_HANDOFF = 4;
// the nucleus ends among the ids of one bfloat16 value whose ids were not
// kept: cut holds that value's 32-bit order key in its high word and j, the
// number of its ids (in id order) inside the nucleus, in its low word; the
// resolve step turns it into the order value of the last nucleus id before
// it reads the row
constexpr int RS_LAZY = 8;

// Per-row state written by the row kernels and read by the resolve kernel.
struct RowStat {
    float kref;              // log2 reference: masses are 2^(z*c - kref)
    float c;                 // log2(e) / T
    double S_nuc;            // nucleus mass in the same units
    unsigned long long cut;  // order value of the last nucleus id
    int flags;
    int nnuc;                // nucleus ids stored in the row's list (-1: none stored)
};
static_assert(sizeof(RowStat) == 32, "RowStat layout");

// ---------------------------------------------------------------------------
// order keys: unsigned integers that sort like the float values, with -0 == +0
__device__ __forceinline__ uint32_t fkey(float f) {
    uint32_t u = __float_as_uint(f);
    if (u == 0x80000000u) u = 0u;
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float fkey_inv(uint32_t k) {
    uint32_t u = (k & 0x80000000u) ? (k & 0x7FFFFFFFu) : ~k;
    return __uint_as_float(u);
}
// (value desc, id asc) order as one descending 64-bit integer
__device__ __forceinline__ unsigned long long order_val(uint32_t key, uint32_t id) {
    return ((unsigned long long)key << 32) | (unsigned long long)(0xFFFFFFFFu - id);
}
__device__ __forceinline__ uint32_t order_id(unsigned long long o) {
    return 0xFFFFFFFFu - (uint32_t)(o & 0xFFFFFFFFull);
}
__device__ __forceinline__ float order_value(unsigned long long o) {
    return fkey_inv((uint32_t)(o >> 32));
}

// ---------------------------------------------------------------------------
// Programmatic dependent launch inside one call: a kernel launched with
// launch_after() is scheduled once every CTA of the previous kernel of the
// stream has exited or executed pdl_trigger(), without waiting for that
// kernel's completion and memory flush.  Every CTA of such a kernel executes
// pdl_wait() before it reads anything the previous kernel wrote (and before
// it exits, so that its completion implies the previous kernel's).  The fast
// row kernel never triggers early: general-kernel CTAs placed on the first
// SMs its last wave frees would crowd there and unbalance that persistent
// grid.  Without the launch attribute both calls are no-ops.
__device__ __forceinline__ unsigned long long globaltimer_ns() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

template <typename... P, typename... A>
inline cudaError_t launch_after(void (*fn)(P...), unsigned grid, unsigned block, cudaStream_t s, A... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(block);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = s;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, fn, args...);
}

// 2^x on the special-function unit
__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// ---------------------------------------------------------------------------
// logit access: a 16-byte chunk holds 8 bf16 or 4 fp32 values
template <int DT> struct Elem;
template <> struct Elem<ACES_F32> {
    static constexpr int EPC = 4;
    static constexpr int SIZE = 4;
    static constexpr uint32_t NEG_INF_WORD = 0xFF800000u;
    __device__ __forceinline__ static float get(const uint4 &w, int j) {
        uint32_t v = j == 0 ? w.x : j == 1 ? w.y : j == 2 ? w.z : w.w;
        return __uint_as_float(v);
    }
    __device__ __forceinline__ static float load1(const void *row, int x) {
        return __ldg(reinterpret_cast<const float *>(row) + x);
    }
};
template <> struct Elem<ACES_BF16> {
    static constexpr int EPC = 8;
    static constexpr int SIZE = 2;
    static constexpr uint32_t NEG_INF_WORD = 0xFF80FF80u;
    __device__ __forceinline__ static float get(const uint4 &w, int j) {
        uint32_t v = (j >> 1) == 0 ? w.x : (j >> 1) == 1 ? w.y : (j >> 1) == 2 ? w.z : w.w;
        return __uint_as_float((j & 1) ? (v & 0xFFFF0000u) : (v << 16));
    }
    __device__ __forceinline__ static float load1(const void *row, int x) {
        unsigned short h = __ldg(reinterpret_cast<const unsigned short *>(row) + x);
        return __uint_as_float((uint32_t)h << 16);
    }
};

// 16 bytes of read-only data, not kept in L1 (streamed once)
__device__ __forceinline__ uint4 ldg16(const void *p) {
    uint4 v;
    asm("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}

// ---------------------------------------------------------------------------
// block reductions (NT threads)
__device__ __forceinline__ float warp_max(float v) {
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}
__device__ __forceinline__ double warp_sum(double v) {
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}
__device__ __forceinline__ unsigned long long warp_sum(unsigned long long v) {
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}
__device__ __forceinline__ unsigned long long warp_max(unsigned long long v) {
    for (int o = 16; o > 0; o >>= 1) {
        unsigned long long w = __shfl_xor_sync(0xffffffffu, v, o);
        v = w > v ? w : v;
    }
    return v;
}

// `red` must hold NTH/32 entries; every thread gets the result.
template <int NTH, class T, class Op>
__device__ __forceinline__ T block_reduce_n(T v, T *red, Op op) {
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    v = op(v);
    __syncthreads();
    if (lane == 0) red[wid] = v;
    __syncthreads();
    T r = red[0];
    for (int i = 1; i < NTH / 32; ++i) r = op.combine(r, red[i]);
    return r;
}
template <class T, class Op>
__device__ __forceinline__ T block_reduce(T v, T *red, Op op) {
    return block_reduce_n<NT>(v, red, op);
}
struct SumD {
    __device__ double operator()(double v) const { return warp_sum(v); }
    __device__ double combine(double a, double b) const { return a + b; }
};
struct MaxF {
    __device__ float operator()(float v) const { return warp_max(v); }
    __device__ float combine(float a, float b) const { return fmaxf(a, b); }
};
struct SumU64 {
    __device__ unsigned long long operator()(unsigned long long v) const { return warp_sum(v); }
    __device__ unsigned long long combine(unsigned long long a, unsigned long long b) const { return a + b; }
};
struct MaxU64 {
    __device__ unsigned long long operator()(unsigned long long v) const { return warp_max(v); }
    __device__ unsigned long long combine(unsigned long long a, unsigned long long b) const {
        return a > b ? a : b;
    }
};

// Exclusive scan over the block of one u64 per thread; `red` holds NTH/32
// entries.  Returns the exclusive prefix; *total gets the block sum.
template <int NTH>
__device__ __forceinline__ unsigned long long block_exscan_n(unsigned long long v,
                                                             unsigned long long *red,
                                                             unsigned long long *total) {
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    unsigned long long inc = v;
    for (int o = 1; o < 32; o <<= 1) {
        unsigned long long t = __shfl_up_sync(0xffffffffu, inc, o);
        if (lane >= o) inc += t;
    }
    __syncthreads();
    if (lane == 31) red[wid] = inc;
    __syncthreads();
    unsigned long long base = 0, all = 0;
    for (int i = 0; i < NTH / 32; ++i) {
        if (i < wid) base += red[i];
        all += red[i];
    }
    *total = all;
    return base + inc - v;
}
__device__ __forceinline__ double block_exscan(double v, double *red, double *total) {
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    double inc = v;
    for (int o = 1; o < 32; o <<= 1) {
        double t = __shfl_up_sync(0xffffffffu, inc, o);
        if (lane >= o) inc += t;
    }
    __syncthreads();
    if (lane == 31) red[wid] = inc;
    __syncthreads();
    double base = 0, all = 0;
    for (int i = 0; i < NWARP; ++i) {
        if (i < wid) base += red[i];
        all += red[i];
    }
    *total = all;
    return base + inc - v;
}

// Descending bitonic sort of n_pow2 u64 values in shared memory (all threads).
__device__ __forceinline__ void bitonic_sort_desc(unsigned long long *a, int n_pow2) {
    for (int k = 2; k <= n_pow2; k <<= 1) {
        for (int j = k >> 1; j > 0; j >>= 1) {
            for (int i = threadIdx.x; i < n_pow2; i += blockDim.x) {
                int ixj = i ^ j;
                if (ixj > i) {
                    unsigned long long x = a[i], y = a[ixj];
                    bool up = (i & k) == 0;
                    if (up ? (x < y) : (x > y)) {
                        a[i] = y;
                        a[ixj] = x;
                    }
                }
            }
            __syncthreads();
        }
    }
}

__host__ __device__ __forceinline__ int next_pow2(int n) {
    int p = 1;
    while (p < n) p <<= 1;
    return p;
}

// 1/S as a float, the same in every kernel: a probability is always
// e * inv_mass(S) for a mass e, so a row's outputs do not depend on which
// kernel finished it (and no fp64 divide sits on the row's critical path)
__device__ __forceinline__ float inv_mass(double S) { return __frcp_rn((float)S); }

// atomicAdd that releases this CTA's earlier writes (ordered before it by a
// __syncthreads) and acquires those released by earlier adds to *p
__device__ __forceinline__ int atomic_add_acq_rel(int *p, int v) {
    int old;
    asm volatile("atom.acq_rel.gpu.global.add.s32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
    return old;
}

// fixed point for exact, order-independent sums of probabilities: floor(x * 2^40)
// for 0 <= x < 2^23, from the float's bits with integer operations only
constexpr float FX_SCALE = 1099511627776.0f;  // 2^40
constexpr double FX_INV = 1.0 / 1099511627776.0;  // 2^-40

// Accept test of Sec. II-A, u < min(1, p/q) with p = e / S, written without
// a divide: for u < 1 it is u * q * S < e (q > 0).
__device__ __forceinline__ int accept_test(float u, float q, float e, double S) {
    return u < 1.0f && (double)u * (double)q * S < (double)e;
}
__device__ __forceinline__ unsigned long long to_fx(float x) {
    const uint32_t u = __float_as_uint(x);
    const uint32_t be = u >> 23;                      // biased exponent (sign is 0)
    if (be == 0u) return 0ull;
    const unsigned long long mant = (unsigned long long)((u & 0x7FFFFFu) | 0x800000u);
    const int sh = (int)be - 110;                     // x * 2^40 = mant * 2^(be - 127 - 23 + 40)
    return sh >= 0 ? (mant << sh) : (sh > -64 ? (mant >> (-sh)) : 0ull);
}

// floor(u * R) exactly for a uniform u = M / 2^sh with a 24-bit integer M
// (0 < u < 1), via a 128-bit product; clamped to R - 1
__device__ __forceinline__ unsigned long long floor_u_times(float uu, unsigned long long R) {
    int ex;
    const float fr = frexpf(uu, &ex);
    const unsigned long long M = (unsigned long long)ldexpf(fr, 24);
    const int sh = 24 - ex;
    const unsigned long long lo = M * R, hi = __umul64hi(M, R);
    unsigned long long thr;
    if (!(uu > 0.0f) || sh >= 128) thr = 0ull;
    else if (sh >= 64) thr = hi >> (sh - 64);
    else if (sh == 0) thr = lo;
    else thr = (lo >> sh) | (hi << (64 - sh));
    if (thr >= R) thr = R - 1ull;
    return thr;
}

// Exact sums of one vocabulary segment of a sequence's row pi (2^-40 units).
struct SegSum {
    unsigned long long r;   // residual max(0, p - q) of the nucleus ids, those of a lazy cut's value aside
    unsigned long long p;   // p itself, likewise
    unsigned long long tr;  // residual of the ids of a lazy cut's value
    int bad;                // a NaN / negative draft probability was seen
    int nt;                 // ids of a lazy cut's value
};
constexpr int NSEG_MAX = 16;
constexpr int STAGGER_NS = 10000;  // row kernel: first-wave start spread per CTA of an SM
constexpr int NUC_CAP = 512;  // nucleus entries kept per row for the residual step

constexpr int WS_CARRY = 256;         // bytes of the hints carried from the previous call, at the start
constexpr int WS_COUNTERS = 256;      // bytes of path counters and depth hints, after them
constexpr int WS_DEPTH = 16;          // first of the 40 depth counters of the row kernel's hints (int index)
constexpr int CARRY_MAGIC = 0x41434531;  // marks a written carry area
// Workspace layout (all offsets 16-byte aligned)
struct Workspace {
    int *carry;                // [64] never cleared: the previous call's hints (written by the resolve
                               //       step): [0] CARRY_MAGIC, [1] T bits, [2] top_p bits, [3] k, [4] V,
                               //       [5] dtype, [6] rows that published a depth, [7] short rows,
                               //       [16..55] how many rows needed each depth
    int *fb_count;             // [64] path counters and depth hints, cleared by every call: [0] rows handed to the
                               //       general kernel, [1] reserved (no kernel waits on another),
                               //       [2] bfloat16 rows finished from their value counts, [3] rows
                               //       ordered by bitonic sort, [4] rows the general kernel finished
                               //       by radix selection, [5] rows whose cut was left to the resolve
                               //       step, [6] rows the general kernel finished by value histogram,
                               //       [7] accept tests that ranked the draft token among ties,
                               //       [8] rows that published the depth they needed, [9] rows that
                               //       took their depth from finished rows, [10] rows counted again
                               //       in a second pass, [11] bfloat16 rows that published a short
                               //       nucleus, [12] rows finished by the sketch-led pass,
                               //       [16..55] how many rows needed each depth (in bins of T/4
                               //       below the row max)
    RowStat *stats;            // [rows]
    int *acc;                  // [B*K] accept bits
    int *fb_list;              // [rows]
    SegSum *seg;               // [B*NSEG_MAX]     (verify only) cleared by every call
    int *seqcnt;               // [B]              (verify only) rows of the sequence finished by the row kernel
    int *seqdone;              // [B]              (verify only) token already drawn
    unsigned long long *nuc;   // [rows*NUC_CAP]   (verify with lists) nucleus order values
};
__host__ __device__ inline size_t align16(size_t x) { return (x + 15) & ~(size_t)15; }
// rows = B*(K+1) target rows; nseq = B sequences with K draft positions (K = 0: sparsify);
// lists: keep every row's nucleus (up to NUC_CAP ids) for the residual step
__host__ __device__ inline size_t ws_bytes(int rows, int nseq, int K, bool lists) {
    size_t b = WS_CARRY + WS_COUNTERS + align16((size_t)rows * sizeof(RowStat)) + align16((size_t)nseq * K * 4) +
               align16((size_t)rows * 4);
    if (K > 0) {
        b += 2 * align16((size_t)nseq * 4) + align16((size_t)nseq * NSEG_MAX * sizeof(SegSum));
        if (lists) b += (size_t)rows * NUC_CAP * 8;
    }
    return b;
}
// bytes at the start of the workspace that every call clears: the counters
// and, for verification, the per-sequence row counts and done flags and the
// segment sums (added to atomically)
__host__ __device__ inline size_t ws_clear_bytes(int nseq, int K) {
    return WS_COUNTERS +
           (K > 0 ? 2 * align16((size_t)nseq * 4) + align16((size_t)nseq * NSEG_MAX * sizeof(SegSum)) : 0);
}
__host__ __device__ inline Workspace ws_carve(void *base, int rows, int nseq, int K, bool lists) {
    char *p = (char *)base;
    Workspace w;
    w.carry = (int *)p;
    p += WS_CARRY;
    w.fb_count = (int *)p;
    p += WS_COUNTERS;
    w.seqcnt = nullptr;
    w.seqdone = nullptr;
    w.seg = nullptr;
    if (K > 0) {
        w.seqcnt = (int *)p;
        p += align16((size_t)nseq * 4);
        w.seqdone = (int *)p;
        p += align16((size_t)nseq * 4);
        w.seg = (SegSum *)p;
        p += align16((size_t)nseq * NSEG_MAX * sizeof(SegSum));
    }
    w.stats = (RowStat *)p;
    p += align16((size_t)rows * sizeof(RowStat));
    w.acc = (int *)p;
    p += align16((size_t)nseq * K * 4);
    w.fb_list = (int *)p;
    p += align16((size_t)rows * 4);
    w.nuc = nullptr;
    if (K > 0) {
        if (lists) {
            w.nuc = (unsigned long long *)p;
            p += (size_t)rows * NUC_CAP * 8;
        }
    }
    return w;
}

// Arguments of the row kernels.
struct RowArgs {
    const void *logits;
    int rows, V, K;        // K = 0: sparsify only (no accept tests)
    float T, c, inv_w, top_p;
    int k;
    const float *q;
    const int32_t *xt;
    const float *u;
    int32_t *topk_ids;
    float *topk_probs;
    float *tail;
    int32_t *row_status;
    int32_t *accept_len;   // verification outputs (null for sparsify)
    int32_t *out_token;
    Workspace ws;
    // capture row kernel (16-byte aligned rows): the row's 16-byte chunks are
    // read in tiles of 32 (one coalesced warp load), tile t of the row order
    // at position (t * pstride) mod ntile, so that the first iteration reads
    // a strided sample of samp_frac of the row
    int ntile, pstride, pstride_w, pstride_it;
    int it_partial;        // iteration that reads the row's partial last tile (-1: none)
    float samp_frac;
    float inv_ws;          // sample bins per unit of logit: SPB / T
    int nmin;              // float32 first rows: ids the capture must reach
    int sk_gpi, sk_ish;    // bfloat16 sketch: groups per thread and iteration (2: 4 chunks each; 1: 8
                           // chunks of 2^sk_ish iterations)
    int force_fb;          // hand every row to the general kernel (the library's exact reference path)
    int nsm;               // SMs of the device
    int stagger_ns;        // start of the first-wave CTAs of an SM spread by this (0: none)
};

// Arguments of the sequence kernel.
struct ResolveArgs {
    const void *logits;
    const float *q;
    const float *u;
    int B, K, V;
    float T, top_p;  // (with k: the key of the hints carried to the next call)
    int k;
    Workspace ws;
    int32_t *accept_len;
    int32_t *out_token;
    int32_t *row_status;
};

// Arguments of the cache kernels.
struct CacheArgs {
    const float *q;
    const int32_t *xt;
    int B, K, V;
    int F[ACES_MAX_K];
    int off[ACES_MAX_K + 1];
    int total;
    int32_t *bt;
    float *bp;
};

// first rejection index pi_b (K when every draft token was accepted), by a
// whole warp: one load per lane and a vote
static_assert(ACES_MAX_K <= 32, "one accept bit per lane");
__device__ __forceinline__ int first_reject_warp(const Workspace &ws, int b, int K) {
    const int lane = threadIdx.x & 31;
    const bool rej = lane < K && !ws.acc[(size_t)b * K + lane];
    const unsigned bal = __ballot_sync(0xffffffffu, rej);
    return bal ? __ffs(bal) - 1 : K;
}

struct DrawShared {
    int pi, bad, tok;
    unsigned long long thr;
};

// Residual (pi < K) or bonus (pi = K) draw of sequence b from row pi's stored
// nucleus (the residual max(0, p - q) is zero outside it): q is read at the
// nucleus ids only, which are ordered by id, and the token is the smallest id
// whose prefix sum of 2^-40 fixed-point masses exceeds floor(u * total).
// Writes accept_len, out_token and seqdone; returns without writing when row
// pi has no stored nucleus (the scan kernels then draw the sequence).  The
// ids are ordered by direct rank counting (one pass, no barrier stages).
// All NTH threads call it, NTH * 2 >= NUC_CAP; skey, srt, rfx, pfx hold
// NUC_CAP entries, red NTH / 32.
template <int NTH>
__device__ void draw_from_list(const Workspace &ws, const float *q, const float *u, int K, int V, int b,
                               int32_t *accept_len, int32_t *out_token, int32_t *row_status,
                               unsigned long long *skey, unsigned long long *srt, unsigned long long *rfx,
                               unsigned long long *pfx, unsigned long long *red, DrawShared *sh) {
    static_assert(2 * NTH >= NUC_CAP, "two nucleus entries per thread");
    const int tid = threadIdx.x;
    if (tid < 32) {
        const int pi0 = first_reject_warp(ws, b, K);
        if (tid == 0) sh->pi = pi0;
    }
    if (tid == 0) {
        sh->bad = 0;
        sh->tok = -1;
    }
    __syncthreads();
    const int pi = sh->pi;
    const int r = b * (K + 1) + pi;
    const RowStat rs = ws.stats[r];
    if (rs.flags & RS_NONFINITE) {
        if (tid == 0) {
            accept_len[b] = pi;
            out_token[b] = -1;
            ws.seqdone[b] = 1;
        }
        return;
    }
    if (rs.nnuc < 0) return;  // no list: the scan kernels draw this sequence
    const int n = ACES_IN(rs.nnuc - 1, NUC_CAP) ? rs.nnuc : 0;
    const unsigned long long *lst = ws.nuc + (size_t)r * NUC_CAP;
    const float *qrow = pi < K ? q + ((size_t)b * K + pi) * V : nullptr;
    const float inv_S = inv_mass(rs.S_nuc);
    for (int i = tid; i < n; i += NTH) {
        const unsigned long long o = lst[i];
        const uint32_t id = order_id(o);
        const float p = ex2(fmaf(order_value(o), rs.c, -rs.kref)) * inv_S;
        float rr = p;
        if (qrow && ACES_IN(id, V)) {
            const float qx = __ldg(qrow + id);
            if (!(qx >= 0.0f)) sh->bad = 1;
            rr = fmaxf(p - qx, 0.0f);
        }
        rfx[i] = to_fx(rr);
        pfx[i] = to_fx(p);
        skey[i] = ((unsigned long long)id << 32) | (unsigned long long)i;  // distinct keys
    }
    __syncthreads();
    if (sh->bad) {
        if (tid == 0) {
            row_status[r] |= ACES_ROW_BAD_Q;
            accept_len[b] = pi;
            out_token[b] = -1;
            ws.seqdone[b] = 1;
        }
        return;
    }
    for (int i = tid; i < n; i += NTH) {  // ascending id: each key's rank among the others
        const unsigned long long key = skey[i];
        int rank = 0;
#pragma unroll 4
        for (int j = 0; j < n; ++j) rank += skey[j] < key;
        if (ACES_IN(rank, NUC_CAP)) srt[rank] = key;
    }
    __syncthreads();
    // two consecutive entries (in id order) per thread
    const int e0 = 2 * tid, e1 = 2 * tid + 1;
    int i0 = e0 < n ? (int)(srt[e0] & 0xFFFFFFFFull) : -1;
    int i1 = e1 < n ? (int)(srt[e1] & 0xFFFFFFFFull) : -1;
    if (i0 >= 0 && !ACES_IN(i0, NUC_CAP)) i0 = -1;
    if (i1 >= 0 && !ACES_IN(i1, NUC_CAP)) i1 = -1;
    const unsigned long long r0 = i0 >= 0 ? rfx[i0] : 0ull, r1 = i1 >= 0 ? rfx[i1] : 0ull;
    const unsigned long long R = block_reduce_n<NTH>(r0 + r1, red, SumU64());
    const int mode = R == 0ull;  // p <= q everywhere: draw from p itself
    const unsigned long long w0 = mode ? (i0 >= 0 ? pfx[i0] : 0ull) : r0;
    const unsigned long long w1 = mode ? (i1 >= 0 ? pfx[i1] : 0ull) : r1;
    unsigned long long tot;
    const unsigned long long ex = block_exscan_n<NTH>(w0 + w1, red, &tot);
    if (tid == 0) sh->thr = tot > 0ull ? floor_u_times(u[(size_t)b * (K + 1) + K], tot) : 0ull;
    __syncthreads();
    const unsigned long long thr = sh->thr;
    if (tot > 0ull) {
        if (ex <= thr && thr < ex + w0) sh->tok = (int)(srt[e0] >> 32);
        else if (ex + w0 <= thr && thr < ex + w0 + w1) sh->tok = (int)(srt[e1] >> 32);
    }
    __syncthreads();
    if (tid == 0) {
        accept_len[b] = pi;
        out_token[b] = sh->tok;
        ws.seqdone[b] = 1;
    }
}

// Outputs of a row whose logits are not a distribution.
template <int NTH>
__device__ void nonfinite_row(const RowArgs &a, int r) {
    const int tid = threadIdx.x;
    for (int j = tid; j < a.k; j += NTH) {
        a.topk_ids[(size_t)r * a.k + j] = -1;
        a.topk_probs[(size_t)r * a.k + j] = 0.0f;
    }
    if (tid == 0) {
        if (a.k > 0) a.tail[r] = 1.0f;
        a.row_status[r] = ACES_ROW_NONFINITE;
        if (a.K > 0) {
            const int b = r / (a.K + 1), i = r % (a.K + 1);
            if (i < a.K) a.ws.acc[(size_t)b * a.K + i] = 0;
        }
        RowStat s;
        s.kref = 0.f;
        s.c = a.c;
        s.S_nuc = 1.0;
        s.cut = 0;
        s.flags = RS_NONFINITE;
        s.nnuc = -1;
        a.ws.stats[r] = s;
    }
}

// host launchers (defined next to their kernels)
void rows_cap_layout(RowArgs &a, int dt);
cudaError_t launch_rows_cap(const RowArgs &a, int dt, cudaStream_t s);
cudaError_t launch_rows_general(const RowArgs &a, int dt, bool vec, int direct, int grid, cudaStream_t s);
cudaError_t launch_resolve(const ResolveArgs &a, int dt, bool vec, cudaStream_t s);
// aces_verify with two choices, neither of which changes the results: lists =
// false keeps no nucleus lists (the residual draw scans its row; the call then
// needs ws_bytes(rows, B, K, lists) bytes of workspace), exact = true hands
// every row to the general kernel.
aces_status verify_impl(const void *target_logits, aces_dtype dt, const float *draft_probs,
                        const int32_t *draft_tokens, const float *uniforms, int B, int K, int V,
                        float T, float top_p, int32_t *accept_len, int32_t *out_token, int k,
                        int32_t *topk_ids, float *topk_probs, float *tail_mass,
                        int32_t *row_status, void *workspace, size_t workspace_bytes, bool lists,
                        bool exact, aces_stream_t stream);
cudaError_t launch_cache_build(const CacheArgs &a, bool vec, cudaStream_t s);
cudaError_t launch_tree_mask(const int *off, int K, int branch_len, int n, int words, uint32_t *mask,
                             int32_t *depth, cudaStream_t s);
cudaError_t launch_compact_kv(void *kv, int planes, int B, int H, int S, size_t row_bytes,
                              const int32_t *prefix_len, const int32_t *accept_len, const int32_t *slot, int K,
                              int branch_len, int32_t *new_len, cudaStream_t s);
cudaError_t launch_resample_sparse(const int32_t *accept_len, const int32_t *ids, const float *probs,
                                   const float *tail, const int32_t *row_status, const float *q,
                                   const float *u, int B, int K, int V, int k, int32_t *token,
                                   int32_t *status, bool vec, cudaStream_t s);
cudaError_t launch_cache_lookup(const int32_t *bt, const CacheArgs &a, const int32_t *accept_len,
                                const int32_t *token, int32_t *slot, cudaStream_t s);

}  // namespace aces
