// Split-K for convolutions whose output tiles cannot fill the GPU (small
// batches: re-execution of flagged images, deep layers with few pixels, FC
// layers run as 1x1 convolutions).  The conv kernels then write FP32 partial
// sums of their K range to a workspace [splits][M][ws_ld] (data channels in
// columns 0..K-1, the carry-through partial, already scaled by coef, in
// column K), and this kernel adds the partials in split order and applies
// the epilogue of Sec. II-A to data and checksum alike: bias (0 on the
// checksum), fault delta, residual, ReLU, store in the storage type.
#include "ct_internal.h"

namespace ct {

namespace {

__device__ __forceinline__ float relu_keep_nan(float v) { return v < 0.f ? 0.f : v; }

template <typename T> __device__ __forceinline__ float ld(const void *p, size_t i);
template <> __device__ __forceinline__ float ld<float>(const void *p, size_t i) {
    return static_cast<const float *>(p)[i];
}
template <> __device__ __forceinline__ float ld<__half>(const void *p, size_t i) {
    return __half2float(static_cast<const __half *>(p)[i]);
}

// input value behind a fault delta: data channel fd.cin of x, or the
// incoming checksum plane when fd.cin == C
template <typename T>
__device__ __forceinline__ float fault_source(const ConvArgs &a, int n, int p, int q) {
    const FaultDelta &fd = a.fd;
    const int h = p * a.stride + fd.r - a.pad, w = q * a.stride + fd.s - a.pad;
    if (h < 0 || h >= a.H || w < 0 || w >= a.W) return 0.f;
    const size_t pix = ((size_t)n * a.H + h) * a.W + w;
    if (fd.cin < a.C) return ld<T>(a.x, pix * a.C + fd.cin);
    return a.cs_in ? ld<T>(a.cs_in, pix) : 0.f;
}

// one thread: 8 channels of one output pixel, or (chunk == K / 8) its checksum
template <typename T>
__global__ void splitk_reduce_kernel(const ConvArgs a, int splits, int ws_ld) {
    pdl_wait();
    pdl_trigger();
    const int M = a.N * a.P * a.Q;
    const int chunks = a.K / 8 + (a.cs_out ? 1 : 0);
    const long long total = (long long)M * chunks;
    const size_t plane = (size_t)M * ws_ld;
    for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < total;
         e += (long long)gridDim.x * blockDim.x) {
        const int m = (int)(e / chunks), ck = (int)(e % chunks);
        const int q = m % a.Q, t = m / a.Q, p = t % a.P, n = t / a.P;
        const float *wsm = a.ws + (size_t)m * ws_ld;
        const bool fault = a.fd.active != 0;
        if (ck < a.K / 8) {
            const int k0 = ck * 8;
            float v[8];
            {
                const float4 *s0 = reinterpret_cast<const float4 *>(wsm + k0);
                float4 x0 = s0[0], x1 = s0[1];
                v[0] = x0.x; v[1] = x0.y; v[2] = x0.z; v[3] = x0.w;
                v[4] = x1.x; v[5] = x1.y; v[6] = x1.z; v[7] = x1.w;
            }
            // loads of four splits in flight, added in split order
            for (int z0 = 1; z0 < splits; z0 += 4) {
                float4 x[4][2];
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    if (z0 + u < splits) {
                        const float4 *s = reinterpret_cast<const float4 *>(wsm + (z0 + u) * plane + k0);
                        x[u][0] = s[0];
                        x[u][1] = s[1];
                    }
                }
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    if (z0 + u < splits) {
                        v[0] += x[u][0].x; v[1] += x[u][0].y; v[2] += x[u][0].z; v[3] += x[u][0].w;
                        v[4] += x[u][1].x; v[5] += x[u][1].y; v[6] += x[u][1].z; v[7] += x[u][1].w;
                    }
                }
            }
            const float fsrc = (fault && a.fd.kout >= k0 && a.fd.kout < k0 + 8) ? fault_source<T>(a, n, p, q) : 0.f;
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const int k = k0 + i;
                float o = v[i] + __ldg(a.bias + k);
                if (fault && a.fd.kout == k) o += a.fd.dv * fsrc;
                if (a.res) o += ld<T>(a.res, (size_t)m * a.K + k);
                if (a.relu) o = relu_keep_nan(o);
                v[i] = o;
            }
            if constexpr (sizeof(T) == 4) {
                float4 *y = reinterpret_cast<float4 *>(static_cast<float *>(a.y) + (size_t)m * a.K + k0);
                y[0] = make_float4(v[0], v[1], v[2], v[3]);
                y[1] = make_float4(v[4], v[5], v[6], v[7]);
            } else {
                uint32_t pk[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    __half2 h = __floats2half2_rn(v[2 * i], v[2 * i + 1]);
                    pk[i] = *reinterpret_cast<uint32_t *>(&h);
                }
                *reinterpret_cast<uint4 *>(static_cast<__half *>(a.y) + (size_t)m * a.K + k0) =
                    make_uint4(pk[0], pk[1], pk[2], pk[3]);
            }
        } else {
            float ctv = 0.f;
            for (int z0 = 0; z0 < splits; z0 += 4) {
                float c[4];
#pragma unroll
                for (int u = 0; u < 4; ++u) c[u] = z0 + u < splits ? wsm[(z0 + u) * plane + a.K] : 0.f;
#pragma unroll
                for (int u = 0; u < 4; ++u) ctv += c[u];
            }
            float cin = 0.f;
            if (a.cs_in && a.cs_rowsum > 0) {            // FC layer: every incoming checksum feature
                for (int i = 0; i < a.cs_rowsum; ++i) cin += ld<T>(a.cs_in, (size_t)m * a.cs_rowsum + i);
            } else if (a.cs_in) {
                const int hc = p * a.stride + (a.R - 1) / 2 - a.pad, wc = q * a.stride + (a.S - 1) / 2 - a.pad;
                if (hc >= 0 && hc < a.H && wc >= 0 && wc < a.W) cin = ld<T>(a.cs_in, ((size_t)n * a.H + hc) * a.W + wc);
            }
            float o = 0.f;
            if (a.role == CT_ROLE_CT) o = ctv + a.coef * cin;
            else if (a.role == CT_ROLE_PASS) o = cin;
            if (fault && a.fd.kout == a.K) o += a.fd.dv * fault_source<T>(a, n, p, q);
            if (a.res_cs) o += ld<T>(a.res_cs, (size_t)m);
            if (a.relu) o = relu_keep_nan(o);
            if constexpr (sizeof(T) == 4) static_cast<float *>(a.cs_out)[m] = o;
            else static_cast<__half *>(a.cs_out)[m] = __float2half_rn(o);
        }
    }
}

}  // namespace

int splitk_choose(int tiles, int n_kblocks, int min_kb_per_split, int target_ctas, int M, int ws_ld,
                  size_t ws_bytes) {
    if (ws_bytes == 0 || tiles * 2 > target_ctas || n_kblocks < 2 * min_kb_per_split) return 1;
    int s = (target_ctas + tiles - 1) / tiles;
    s = std::min(s, n_kblocks / min_kb_per_split);
    const size_t per = (size_t)M * ws_ld * sizeof(float);
    if (per == 0) return 1;
    s = (int)std::min<size_t>((size_t)s, ws_bytes / per);
    s = std::min(s, 64);
    if (s < 2) return 1;
    // equal K ranges: recompute the count from the per-split length
    const int kps = (n_kblocks + s - 1) / s;
    return (n_kblocks + kps - 1) / kps;
}

cudaError_t launch_splitk_reduce(const ConvArgs &a, int splits, int ws_ld, bool half, cudaStream_t st) {
    const long long total = (long long)a.N * a.P * a.Q * (a.K / 8 + (a.cs_out ? 1 : 0));
    const int threads = 256;
    const long long want = (total + threads - 1) / threads;
    const int grid = (int)std::min<long long>(std::max<long long>(want, 1), 4096);
    if (half) pdl_launch(splitk_reduce_kernel<__half>, grid, threads, 0, st, a, splits, ws_ld);
    else pdl_launch(splitk_reduce_kernel<float>, grid, threads, 0, st, a, splits, ws_ld);
    return cudaGetLastError();
}

}  // namespace ct
