// Depthwise convolution (groups == C == K) with the checksum group.
//
// Output channel c of pixel (n, p, q) = sum over taps (r, s), in that order,
// of w[r][s][c] * x[n, p*stride + r - pad, q*stride + s - pad, c] (FFMA
// chain from 0), + bias, ReLU.  The paper builds its carry-through filter
// for dense convolutions; in a depthwise layer the checksum is one more
// group, whose filter sees only the incoming checksum channel: its output is
// the incoming checksum at the centre tap (weight 1), + residual checksum,
// ReLU.  A fault on that group's filter (not stored) adds dv * the checksum
// input at the flipped tap.  Data filters have no structural zeros, so their
// faults are stored-word flips.
//
// Memory-bound (9 MACs per input element): one thread per output pixel and
// 16 bytes of channels (8 FP16 or 4 FP32), 16-byte loads along C, weights
// laid out [R*S][C] so a tap's weights for those channels are one load.
#include "ct_internal.h"

namespace ct {

namespace {

template <typename T> struct Vec;
template <> struct Vec<float> {
    static constexpr int N = 4;
    __device__ static void load(const float *p, float *v) {
        const float4 a = *reinterpret_cast<const float4 *>(p);
        v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
    }
    __device__ static void store(float *p, const float *v) {
        *reinterpret_cast<float4 *>(p) = make_float4(v[0], v[1], v[2], v[3]);
    }
    __device__ static float one(const float *p, size_t i) { return p[i]; }
    __device__ static void put(float *p, size_t i, float v) { p[i] = v; }
};
template <> struct Vec<__half> {
    static constexpr int N = 8;
    __device__ static void load(const __half *p, float *v) {
        const uint4 a = *reinterpret_cast<const uint4 *>(p);
        const __half2 *h = reinterpret_cast<const __half2 *>(&a);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float2 f = __half22float2(h[i]);
            v[2 * i] = f.x; v[2 * i + 1] = f.y;
        }
    }
    __device__ static void store(__half *p, const float *v) {
        uint32_t pk[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            __half2 h = __floats2half2_rn(v[2 * i], v[2 * i + 1]);
            pk[i] = *reinterpret_cast<uint32_t *>(&h);
        }
        *reinterpret_cast<uint4 *>(p) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
    }
    __device__ static float one(const __half *p, size_t i) { return __half2float(p[i]); }
    __device__ static void put(__half *p, size_t i, float v) { p[i] = __float2half_rn(v); }
};

__device__ __forceinline__ float relu_nan(float v) { return v < 0.f ? 0.f : v; }

template <typename T>
__global__ void __launch_bounds__(256) conv_dw_kernel(const ConvArgs a) {
    pdl_wait();
    pdl_trigger();
    using V = Vec<T>;
    constexpr int VE = V::N;
    const int groups = a.C / VE;
    const long long M = (long long)a.N * a.P * a.Q;
    const long long total = M * groups;
    const T *x = static_cast<const T *>(a.x);
    const T *w = static_cast<const T *>(a.w);
    T *y = static_cast<T *>(a.y);
    const FaultDelta fd = a.fd;
    const int ctr_r = (a.R - 1) / 2, ctr_s = (a.S - 1) / 2;
    for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < total;
         e += (long long)gridDim.x * blockDim.x) {
        const int g = (int)(e % groups);
        const long long m = e / groups;
        const int q = (int)(m % a.Q);
        const long long t = m / a.Q;
        const int p = (int)(t % a.P), n = (int)(t / a.P);
        const int c0 = g * VE;
        float acc[VE];
#pragma unroll
        for (int i = 0; i < VE; ++i) acc[i] = 0.f;
        for (int r = 0; r < a.R; ++r) {
            const int h = p * a.stride + r - a.pad;
            if (h < 0 || h >= a.H) continue;
            for (int s = 0; s < a.S; ++s) {
                const int ww = q * a.stride + s - a.pad;
                if (ww < 0 || ww >= a.W) continue;
                float xv[VE], wv[VE];
                V::load(x + (((size_t)n * a.H + h) * a.W + ww) * a.C + c0, xv);
                V::load(w + (size_t)(r * a.S + s) * a.C + c0, wv);
#pragma unroll
                for (int i = 0; i < VE; ++i) acc[i] = fmaf(xv[i], wv[i], acc[i]);
            }
        }
        float out[VE];
#pragma unroll
        for (int i = 0; i < VE; ++i) {
            float o = acc[i] + __ldg(a.bias + c0 + i);
            if (a.res) o += V::one(static_cast<const T *>(a.res), (size_t)m * a.K + c0 + i);
            if (a.relu) o = relu_nan(o);
            out[i] = o;
        }
        V::store(y + (size_t)m * a.K + c0, out);
        if (g == 0 && a.cs_out) {
            const T *csi = static_cast<const T *>(a.cs_in);
            const int hc = p * a.stride + ctr_r - a.pad, wc = q * a.stride + ctr_s - a.pad;
            float o = 0.f;
            if (a.role == CT_ROLE_PASS && csi && hc >= 0 && hc < a.H && wc >= 0 && wc < a.W)
                o = V::one(csi, ((size_t)n * a.H + hc) * a.W + wc);
            if (fd.active && fd.kout == a.K && csi) {
                const int h = p * a.stride + fd.r - a.pad, ws = q * a.stride + fd.s - a.pad;
                if (h >= 0 && h < a.H && ws >= 0 && ws < a.W) o += fd.dv * V::one(csi, ((size_t)n * a.H + h) * a.W + ws);
            }
            if (a.res_cs) o += V::one(static_cast<const T *>(a.res_cs), (size_t)m);
            if (a.relu) o = relu_nan(o);
            V::put(static_cast<T *>(a.cs_out), (size_t)m, o);
        }
    }
}

}  // namespace

bool dw_supported(int C, int K, bool half) { return C == K && C % (half ? 8 : 4) == 0; }

cudaError_t launch_conv_dw(const ConvArgs &a, bool half, cudaStream_t st) {
    const long long total = (long long)a.N * a.P * a.Q * (a.C / (half ? 8 : 4));
    const int threads = 256;
    const long long want = (total + threads - 1) / threads;
    const int grid = (int)std::min<long long>(std::max<long long>(want, 1), 152LL * 16);
    if (half) pdl_launch(conv_dw_kernel<__half>, grid, threads, 0, st, a);
    else pdl_launch(conv_dw_kernel<float>, grid, threads, 0, st, a);
    return cudaGetLastError();
}

}  // namespace ct
