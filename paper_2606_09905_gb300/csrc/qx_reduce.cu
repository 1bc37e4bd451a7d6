// qx_reduce.cu -- the memory-bound operators of Table 2: min/max reduction
// (INT32, INT16; FP32 too) and 2-D max / average pooling (the paper's rows
// are AvgPool 2x2/2 INT32 and MaxPool 2x2/2 FP32).  Both stream their input
// once from HBM, so they are written for bandwidth: 16-byte vector loads in a
// grid-stride loop with several loads in flight per thread.
//
// Min/max: every block reduces its share to one (min, max) pair in the plan's
// workspace; the last block to finish (arrival counter) reduces the pairs in
// block order and writes the result, then rearms the counter.
//
// Pooling: NCHW, no padding.  Max takes the window maximum; the integer
// average is floor(window sum / window size) (an arithmetic shift for 2x2),
// the float average the FP32 mean.  The 2x2 / stride 2 case reads two input
// rows of 8 values and writes 4 outputs per thread when rows are 16-byte
// aligned; any other window runs one output per thread.
#include <cuda_runtime.h>

#include <cfloat>
#include <climits>
#include <type_traits>

#include "qx_device.cuh"
#include "qx_internal.h"

namespace qx {

// ------------------------------------------------------------- min / max
template <typename T>
struct MinMaxTraits;
template <>
struct MinMaxTraits<int32_t> {
    using Acc = int32_t;
    static constexpr int VEC = 4;
    __device__ static Acc lo_init() { return INT_MAX; }
    __device__ static Acc hi_init() { return INT_MIN; }
};
template <>
struct MinMaxTraits<int16_t> {
    using Acc = int32_t;
    static constexpr int VEC = 8;
    __device__ static Acc lo_init() { return INT_MAX; }
    __device__ static Acc hi_init() { return INT_MIN; }
};
template <>
struct MinMaxTraits<float> {
    using Acc = float;
    static constexpr int VEC = 4;
    __device__ static Acc lo_init() { return FLT_MAX; }
    __device__ static Acc hi_init() { return -FLT_MAX; }
};

template <typename A>
__device__ __forceinline__ void mm_update(A &lo, A &hi, A v) {
    lo = v < lo ? v : lo;
    hi = v > hi ? v : hi;
}

// merge two partial results (either may still hold the empty-set sentinels)
template <typename A>
__device__ __forceinline__ void mm_merge(A &lo, A &hi, A olo, A ohi) {
    lo = olo < lo ? olo : lo;
    hi = ohi > hi ? ohi : hi;
}

template <typename A>
__device__ __forceinline__ A shfl_xor(A v, int m) {
    return __shfl_xor_sync(0xffffffffu, v, m);
}

struct MinMaxArgs {
    const void *x;
    int64_t n;
    void *result;          // 2 elements of the input type: min, max
    void *partial;         // [gridDim.x][2] accumulators
    unsigned *counter;     // zero between calls
    int vec;               // x is 16-byte aligned
};

template <typename T>
__global__ void __launch_bounds__(512) minmax_kernel(const MinMaxArgs p) {
    using Tr = MinMaxTraits<T>;
    using A = typename Tr::Acc;
    constexpr int V = Tr::VEC;
    const T *x = static_cast<const T *>(p.x);
    A lo = Tr::lo_init(), hi = Tr::hi_init();
    const int64_t tid = int64_t(blockIdx.x) * blockDim.x + threadIdx.x;
    const int64_t nthreads = int64_t(gridDim.x) * blockDim.x;
    int64_t done = 0;
    if (p.vec) {
        const int64_t nvec = p.n / V;
        const uint4 *xv = reinterpret_cast<const uint4 *>(x);
        int64_t i = tid;
        // four independent 16-byte loads per iteration keep enough bytes in flight
        for (; i + 3 * nthreads < nvec; i += 4 * nthreads) {
            uint4 u[4];
#pragma unroll
            for (int j = 0; j < 4; ++j) u[j] = __ldcs(xv + i + j * nthreads);
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const T *e = reinterpret_cast<const T *>(&u[j]);
#pragma unroll
                for (int k = 0; k < V; ++k) mm_update<A>(lo, hi, A(e[k]));
            }
        }
        for (; i < nvec; i += nthreads) {
            const uint4 u = __ldcs(xv + i);
            const T *e = reinterpret_cast<const T *>(&u);
#pragma unroll
            for (int k = 0; k < V; ++k) mm_update<A>(lo, hi, A(e[k]));
        }
        done = nvec * V;
    }
    for (int64_t i = done + tid; i < p.n; i += nthreads) mm_update<A>(lo, hi, A(x[i]));

    // block reduction
    __shared__ A s_lo[16], s_hi[16];
    __shared__ bool s_last;
#pragma unroll
    for (int m = 16; m > 0; m >>= 1) mm_merge<A>(lo, hi, shfl_xor(lo, m), shfl_xor(hi, m));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) {
        s_lo[warp] = lo;
        s_hi[warp] = hi;
    }
    __syncthreads();
    A *part = static_cast<A *>(p.partial);
    if (threadIdx.x == 0) {
        for (int w = 1; w < int(blockDim.x >> 5); ++w) mm_merge<A>(lo, hi, s_lo[w], s_hi[w]);
        part[2 * blockIdx.x] = lo;
        part[2 * blockIdx.x + 1] = hi;
        __threadfence();
        s_last = atomicAdd(p.counter, 1u) == gridDim.x - 1;
    }
    __syncthreads();
    if (!s_last) return;
    // last block: reduce the block results in block order
    __threadfence();
    lo = Tr::lo_init();
    hi = Tr::hi_init();
    for (int b = threadIdx.x; b < int(gridDim.x); b += blockDim.x)
        mm_merge<A>(lo, hi, __ldcg(part + 2 * b), __ldcg(part + 2 * b + 1));
#pragma unroll
    for (int m = 16; m > 0; m >>= 1) mm_merge<A>(lo, hi, shfl_xor(lo, m), shfl_xor(hi, m));
    __syncthreads();
    if (lane == 0) {
        s_lo[warp] = lo;
        s_hi[warp] = hi;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        for (int w = 1; w < int(blockDim.x >> 5); ++w) mm_merge<A>(lo, hi, s_lo[w], s_hi[w]);
        T *out = static_cast<T *>(p.result);
        out[0] = T(lo);
        out[1] = T(hi);
        *p.counter = 0u;   // rearm for the next call
    }
}

int minmax_blocks(int num_sms) { return num_sms * 4; }

cudaError_t launch_minmax(int dtype, const void *x, int64_t n, void *result, void *partial,
                          unsigned *counter, int num_sms, cudaStream_t st) {
    MinMaxArgs p;
    p.x = x;
    p.n = n;
    p.result = result;
    p.partial = partial;
    p.counter = counter;
    p.vec = (reinterpret_cast<uintptr_t>(x) % 16) == 0;
    const int grid = minmax_blocks(num_sms);
    switch (dtype) {
        case QX_I16: minmax_kernel<int16_t><<<grid, 512, 0, st>>>(p); break;
        case QX_I32: minmax_kernel<int32_t><<<grid, 512, 0, st>>>(p); break;
        case QX_F32: minmax_kernel<float><<<grid, 512, 0, st>>>(p); break;
        default: return cudaErrorInvalidValue;
    }
    return cudaGetLastError();
}

// --------------------------------------------------------------- pooling
struct PoolArgs {
    const void *x;
    void *y;
    int n, c, h, w, kh, kw, stride, P, Q;
    int is_max;
    int fast;              // 2x2 / stride 2, rows of 8-aligned 16-byte vectors
};

template <typename T>
__device__ __forceinline__ T pool_reduce_window(const T *img, int w, int r0, int c0, int kh, int kw,
                                                bool is_max) {
    if (is_max) {
        T m = img[int64_t(r0) * w + c0];
        for (int r = 0; r < kh; ++r)
            for (int s = 0; s < kw; ++s) {
                const T v = img[int64_t(r0 + r) * w + c0 + s];
                m = v > m ? v : m;
            }
        return m;
    }
    if constexpr (std::is_floating_point<T>::value) {     // float mean
        float acc = 0.f;
        for (int r = 0; r < kh; ++r)
            for (int s = 0; s < kw; ++s) acc += float(img[int64_t(r0 + r) * w + c0 + s]);
        return T(acc / float(kh * kw));
    } else {                                              // integer floor mean
        int64_t acc = 0;
        for (int r = 0; r < kh; ++r)
            for (int s = 0; s < kw; ++s) acc += int64_t(img[int64_t(r0 + r) * w + c0 + s]);
        const int64_t k = kh * kw;
        int64_t q = acc / k;
        if ((acc % k) != 0 && acc < 0) --q;
        return T(q);
    }
}

// 2x2 / stride 2 on 8 input columns -> 4 outputs
template <typename T>
__device__ __forceinline__ T pool4(T a, T b, T c, T d, bool is_max) {
    if (is_max) {
        const T m1 = a > b ? a : b, m2 = c > d ? c : d;
        return m1 > m2 ? m1 : m2;
    }
    if constexpr (std::is_floating_point<T>::value) {
        return T((float(a) + float(b) + float(c) + float(d)) * 0.25f);
    } else {
        const int64_t s = int64_t(a) + int64_t(b) + int64_t(c) + int64_t(d);
        return T(s >> 2);   // arithmetic shift = floor division by 4
    }
}

template <typename T>
__global__ void __launch_bounds__(256) pool_kernel(const PoolArgs p) {
    const T *x = static_cast<const T *>(p.x);
    T *y = static_cast<T *>(p.y);
    const bool is_max = p.is_max != 0;
    const int64_t planes = int64_t(p.n) * p.c;
    if (p.fast) {
        // each item: 4 consecutive outputs of one row (8 input columns x 2 rows)
        constexpr int IN_V = 16 / sizeof(T);              // elements per 16-byte vector
        const int groups = p.Q / 4;
        const int64_t items = planes * p.P * groups;
        for (int64_t it = int64_t(blockIdx.x) * blockDim.x + threadIdx.x; it < items;
             it += int64_t(gridDim.x) * blockDim.x) {
            const int g = int(it % groups);
            const int64_t rest = it / groups;
            const int pr = int(rest % p.P);
            const int64_t plane = rest / p.P;
            const T *r0 = x + (plane * p.h + 2 * pr) * p.w + g * 8;
            const T *r1 = r0 + p.w;
            T a[8], b[8];
#pragma unroll
            for (int v = 0; v < 8 / IN_V; ++v) {
                *reinterpret_cast<uint4 *>(a + v * IN_V) = __ldcs(reinterpret_cast<const uint4 *>(r0) + v);
                *reinterpret_cast<uint4 *>(b + v * IN_V) = __ldcs(reinterpret_cast<const uint4 *>(r1) + v);
            }
            T o[4];
#pragma unroll
            for (int j = 0; j < 4; ++j) o[j] = pool4<T>(a[2 * j], a[2 * j + 1], b[2 * j], b[2 * j + 1], is_max);
            T *dst = y + (plane * p.P + pr) * p.Q + g * 4;
            if constexpr (sizeof(T) == 4) {
                __stcs(reinterpret_cast<uint4 *>(dst), *reinterpret_cast<uint4 *>(o));
            } else {
#pragma unroll
                for (int j = 0; j < 4; ++j) dst[j] = o[j];
            }
        }
        return;
    }
    const int64_t items = planes * p.P * p.Q;
    for (int64_t it = int64_t(blockIdx.x) * blockDim.x + threadIdx.x; it < items;
         it += int64_t(gridDim.x) * blockDim.x) {
        const int q = int(it % p.Q);
        const int64_t rest = it / p.Q;
        const int pr = int(rest % p.P);
        const int64_t plane = rest / p.P;
        y[it] = pool_reduce_window<T>(x + plane * p.h * p.w, p.w, pr * p.stride, q * p.stride, p.kh,
                                      p.kw, is_max);
    }
}

cudaError_t launch_pool2d(int dtype, bool is_max, const void *x, void *y, int n, int c, int h, int w,
                          int kh, int kw, int stride, int num_sms, cudaStream_t st) {
    PoolArgs p;
    p.x = x;
    p.y = y;
    p.n = n;
    p.c = c;
    p.h = h;
    p.w = w;
    p.kh = kh;
    p.kw = kw;
    p.stride = stride;
    p.P = (h - kh) / stride + 1;
    p.Q = (w - kw) / stride + 1;
    p.is_max = is_max ? 1 : 0;
    const int esz = dtype == QX_I16 ? 2 : 4;
    p.fast = kh == 2 && kw == 2 && stride == 2 && (w % 8) == 0 && (h % 2) == 0 &&
             (reinterpret_cast<uintptr_t>(x) % 16) == 0 && (int64_t(w) * esz) % 16 == 0 &&
             (esz == 2 || ((reinterpret_cast<uintptr_t>(y) % 16) == 0 && (p.Q % 4) == 0));
    const int grid = num_sms * 8;
    switch (dtype) {
        case QX_I16: pool_kernel<int16_t><<<grid, 256, 0, st>>>(p); break;
        case QX_I32: pool_kernel<int32_t><<<grid, 256, 0, st>>>(p); break;
        case QX_F32: pool_kernel<float><<<grid, 256, 0, st>>>(p); break;
        default: return cudaErrorInvalidValue;
    }
    return cudaGetLastError();
}

}  // namespace qx
