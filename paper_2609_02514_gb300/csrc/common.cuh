// Device helpers shared by the AceSpec kernels (sm_103a).
#pragma once
#include <cuda_runtime.h>
#include <float.h>
#include <stdint.h>

#include "../../include/acespec.h"

namespace aces {

constexpr int NT = 512;             // threads per CTA for every row kernel
constexpr int NWARP = NT / 32;
constexpr int SKETCH_CAP = 16384;   // max sketch groups per row (fast path)
constexpr int CAND_CAP = 4096;      // max candidates per row (fast path)
constexpr int NBIN = 256;           // sketch bins of width T/8 below the max
constexpr int BIN_PER_T = 8;

// Row-level flags kept in the workspace.
constexpr int RS_ALL_IN = 1;        // top_p >= 1: every finite id is in the nucleus
constexpr int RS_NONFINITE = 2;

// Per-row state written by the row kernels and read by the resolve kernel.
struct RowStat {
    float m;                 // row max logit
    float c;                 // log2(e) / T
    double S_nuc;            // nucleus mass, in units of exp((z - m)/T)
    unsigned long long cut;  // order value of the last nucleus id
    int flags;
    int pad;
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

__device__ __forceinline__ uint4 ldg16(const void *p) {
    return __ldg(reinterpret_cast<const uint4 *>(p));
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

// `red` must hold NWARP entries; every thread gets the result.
template <class T, class Op>
__device__ __forceinline__ T block_reduce(T v, T *red, Op op) {
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    v = op(v);
    __syncthreads();
    if (lane == 0) red[wid] = v;
    __syncthreads();
    T r = red[0];
    for (int i = 1; i < NWARP; ++i) r = op.combine(r, red[i]);
    return r;
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

// Exclusive scan over the block of one u64 per thread; `red` holds NWARP
// entries.  Returns the exclusive prefix; *total gets the block sum.
__device__ __forceinline__ unsigned long long block_exscan(unsigned long long v,
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
    for (int i = 0; i < NWARP; ++i) {
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

// fixed point for exact, order-independent sums of probabilities in [0, 1]
constexpr float FX_SCALE = 1099511627776.0f;  // 2^40
__device__ __forceinline__ unsigned long long to_fx(float x) {
    return __float2ull_rn(x * FX_SCALE);
}

// Workspace layout (all offsets 16-byte aligned)
struct Workspace {
    int *fb_count;    // [4]   number of rows handed to the general path
    RowStat *stats;   // [rows]
    int *acc;         // [B*K] accept bits
    int *fb_list;     // [rows]
};
__host__ __device__ inline size_t align16(size_t x) { return (x + 15) & ~(size_t)15; }
__host__ __device__ inline size_t ws_bytes(int rows, int nacc) {
    return 16 + align16((size_t)rows * sizeof(RowStat)) + align16((size_t)nacc * 4) +
           align16((size_t)rows * 4);
}
__host__ __device__ inline Workspace ws_carve(void *base, int rows, int nacc) {
    char *p = (char *)base;
    Workspace w;
    w.fb_count = (int *)p;
    p += 16;
    w.stats = (RowStat *)p;
    p += align16((size_t)rows * sizeof(RowStat));
    w.acc = (int *)p;
    p += align16((size_t)nacc * 4);
    w.fb_list = (int *)p;
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
    Workspace ws;
    int ng;                // sketch groups per row
};

// Arguments of the sequence kernel.
struct ResolveArgs {
    const void *logits;
    const float *q;
    const float *u;
    int B, K, V;
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

// host launchers (defined next to their kernels)
cudaError_t launch_rows_fast(const RowArgs &a, int dt, int gc, size_t smem, cudaStream_t s);
cudaError_t launch_rows_general(const RowArgs &a, int dt, bool vec, int direct, int grid, cudaStream_t s);
cudaError_t launch_resolve(const ResolveArgs &a, int dt, bool vec, cudaStream_t s);
cudaError_t launch_cache_build(const CacheArgs &a, bool vec, cudaStream_t s);
cudaError_t launch_cache_lookup(const int32_t *bt, const CacheArgs &a, const int32_t *accept_len,
                                const int32_t *token, int32_t *slot, cudaStream_t s);

}  // namespace aces
