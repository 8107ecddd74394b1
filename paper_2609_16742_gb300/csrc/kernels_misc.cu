// FC layers with the carry-through neuron and the output verification,
// pooling, layout conversion, fault injection and re-execution gathers.
#include "ct_internal.h"

namespace ct {
namespace {

__device__ __forceinline__ float to_f(float v) { return v; }
__device__ __forceinline__ float to_f(__half v) { return __half2float(v); }
template <typename T> __device__ __forceinline__ T from_f(float v);
template <> __device__ __forceinline__ float from_f<float>(float v) { return v; }
template <> __device__ __forceinline__ __half from_f<__half>(float v) { return __float2half_rn(v); }
__device__ __forceinline__ float relu_keep_nan(float v) { return v < 0.f ? 0.f : v; }

// ---------------------------------------------------------------------------
// FC: y[b, j] = act(sum_i W[j, i] x[b, i] + bias[j]) over the data features
// only (the checksum features are structural zeros of every data neuron,
// Sec. II-A); the carry-through neuron (hidden layers) or the
// accumulated-checksum neuron S (final layer, Sec. II-B) is coef times the
// sum of every input, checksum features included.  The final layer also
// writes the verdict flag = NOT(|S - ref| <= tau), compared in double.
//
// Block: 256 threads = 8 warps, 16 neurons x 64 images.  Lanes own images
// (l and l + 32), warps split the K chunk, so one staged x value feeds 16
// FMAs and one staged weight value is a broadcast.
// ---------------------------------------------------------------------------
constexpr int FC_J = 16, FC_IMG = 64, FC_KC = 64, FC_WARPS = 8;
// input rows in shared memory: FC_KC values + 4 of padding (16-byte rows; a
// warp's 16-byte reads of 32 rows at one k then hit every bank once per phase)
constexpr int FC_XP = FC_KC + 4;
static_assert((FC_KC / 4) % FC_WARPS == 0, "each warp takes whole groups of four inputs");

// four consecutive inputs k .. k + 3 of one row as FP32 (16 or 8 bytes, aligned)
__device__ __forceinline__ float4 load4_f(const float *p) { return *reinterpret_cast<const float4 *>(p); }
__device__ __forceinline__ float4 load4_f(const __half *p) {
    const uint2 u = *reinterpret_cast<const uint2 *>(p);
    const float2 a = __half22float2(*reinterpret_cast<const __half2 *>(&u.x));
    const float2 b = __half22float2(*reinterpret_cast<const __half2 *>(&u.y));
    return make_float4(a.x, a.y, b.x, b.y);
}

// Row b of a layer's output: a row of this batch, or (final layer with
// re-run rows) the re-executed image's row of the earlier batch's logits
template <typename TY>
__device__ __forceinline__ TY *fc_out_row(const FcArgs &a, int b) {
    if (a.rr_idx && b >= a.rr_split) return reinterpret_cast<TY *>(a.rr_y) + (size_t)a.rr_idx[b - a.rr_split] * a.n_out;
    return static_cast<TY *>(a.y) + (size_t)b * a.n_out;
}
// S and verdict of image row b of the final layer; a re-run row writes its
// S to the earlier batch and no flag (Sec. II-B: the re-run's flag is ignored)
__device__ __forceinline__ void fc_final_out(const FcArgs &a, int b, float s, uint8_t fv) {
    if (a.rr_idx && b >= a.rr_split) {
        if (a.rr_S) a.rr_S[a.rr_idx[b - a.rr_split]] = s;
        return;
    }
    if (a.S) a.S[b] = s;
    if (a.flag) a.flag[b] = fv;
    if (a.flag2) a.flag2[b] = fv;
}
static_assert((FC_IMG * FC_XP) % 4 == 0, "weight tile must start 16-byte aligned (float4 reads)");

template <typename TX, typename TW, typename TY>
__global__ void __launch_bounds__(256, 2) fc_kernel(FcArgs a) {
    pdl_wait();
    pdl_trigger();
    extern __shared__ __align__(16) float smem[];
    // two stages of [FC_IMG][FC_XP] inputs and [FC_KC][FC_J] weights (each
    // offset a multiple of 4 floats: 16-byte aligned float4 reads), then the
    // cross-warp reduction [FC_WARPS][FC_J + 1][FC_IMG]
    constexpr int XS = FC_IMG * FC_XP, WS = FC_KC * FC_J;
    float *red = smem + 2 * (XS + WS);
    const TX *x = static_cast<const TX *>(a.x);
    const TW *w = static_cast<const TW *>(a.w);
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int j0 = blockIdx.x * FC_J, b0 = blockIdx.y * FC_IMG;
    const bool ct_block = a.protect && blockIdx.x == 0;

    float acc[FC_J][2];
    float act[2] = {0.f, 0.f};
#pragma unroll
    for (int j = 0; j < FC_J; ++j) acc[j][0] = acc[j][1] = 0.f;

    // K range of this block: all inputs, or one split's range (gridDim.z > 1)
    const int nkc = (a.n_in + FC_KC - 1) / FC_KC;
    const int kc_per = (nkc + gridDim.z - 1) / gridDim.z;
    const int k_lo = blockIdx.z * kc_per * FC_KC, k_hi = min(a.n_in, k_lo + kc_per * FC_KC);
    // x[b0 .. b0+63][k0 .. k0+63] and W[j0..j0+15][k0..k0+63] (transposed):
    // the next chunk's values are loaded into registers while this chunk is
    // multiplied, then stored to the other stage.  The inputs move as four
    // consecutive values per load when every row starts 16-byte aligned
    // (n_in a multiple of 4; the K ranges end on multiples of 4 then too).
    constexpr int XR = FC_KC * FC_IMG / 256, WR = FC_KC * FC_J / 256;
    const bool xvec = (a.n_in & 3) == 0;
    float4 xr[XR / 4];
    float xs[XR];
    float wr[WR];
    auto load_chunk = [&](int k0) {
        if (xvec) {
#pragma unroll
            for (int i = 0; i < XR / 4; ++i) {
                const int e = tid + 256 * i, k4 = (e % (FC_KC / 4)) * 4, bb = e / (FC_KC / 4);
                const int b = b0 + bb, k = k0 + k4;
                xr[i] = (b < a.B && k < k_hi) ? load4_f(x + (size_t)b * a.n_in + k) : make_float4(0.f, 0.f, 0.f, 0.f);
            }
        } else {
#pragma unroll
            for (int i = 0; i < XR; ++i) {
                const int e = tid + 256 * i, kk = e % FC_KC, bb = e / FC_KC;
                const int b = b0 + bb, k = k0 + kk;
                xs[i] = (b < a.B && k < k_hi) ? to_f(x[(size_t)b * a.n_in + k]) : 0.f;
            }
        }
#pragma unroll
        for (int i = 0; i < WR; ++i) {
            const int e = tid + 256 * i, kk = e % FC_KC, jj = e / FC_KC;
            const int j = j0 + jj, k = k0 + kk;
            wr[i] = (j < a.n_out && k < k_hi) ? to_f(w[(size_t)j * a.n_in + k]) : 0.f;
        }
    };
    auto store_chunk = [&](int stage) {
        float *Xd = smem + stage * (XS + WS), *Wd = Xd + XS;
        if (xvec) {
#pragma unroll
            for (int i = 0; i < XR / 4; ++i) {
                const int e = tid + 256 * i;
                *reinterpret_cast<float4 *>(&Xd[(e / (FC_KC / 4)) * FC_XP + (e % (FC_KC / 4)) * 4]) = xr[i];
            }
        } else {
#pragma unroll
            for (int i = 0; i < XR; ++i) {
                const int e = tid + 256 * i;
                Xd[(e / FC_KC) * FC_XP + e % FC_KC] = xs[i];
            }
        }
#pragma unroll
        for (int i = 0; i < WR; ++i) {
            const int e = tid + 256 * i;
            Wd[(e % FC_KC) * FC_J + e / FC_KC] = wr[i];
        }
    };
    if (k_lo < k_hi) {
        load_chunk(k_lo);
        store_chunk(0);
    }
    __syncthreads();
    int stage = 0;
    for (int k0 = k_lo; k0 < k_hi; k0 += FC_KC, stage ^= 1) {
        const bool more = k0 + FC_KC < k_hi;
        if (more) load_chunk(k0 + FC_KC);
        const float *Xs = smem + stage * (XS + WS), *Ws = Xs + XS;
        // warp w takes the groups of four inputs g = w, w + FC_WARPS, ...;
        // lanes are images (lane, lane + 32)
#pragma unroll
        for (int g = warp; g < FC_KC / 4; g += FC_WARPS) {
            const float4 x04 = *reinterpret_cast<const float4 *>(&Xs[lane * FC_XP + 4 * g]);
            const float4 x14 = *reinterpret_cast<const float4 *>(&Xs[(lane + 32) * FC_XP + 4 * g]);
            const float x0v[4] = {x04.x, x04.y, x04.z, x04.w}, x1v[4] = {x14.x, x14.y, x14.z, x14.w};
#pragma unroll
            for (int t = 0; t < 4; ++t) {
                const float x0 = x0v[t], x1 = x1v[t];
                const float4 *wrow = reinterpret_cast<const float4 *>(&Ws[(4 * g + t) * FC_J]);
#pragma unroll
                for (int q = 0; q < FC_J / 4; ++q) {
                    float4 wv = wrow[q];
                    acc[4 * q + 0][0] = fmaf(wv.x, x0, acc[4 * q + 0][0]);
                    acc[4 * q + 0][1] = fmaf(wv.x, x1, acc[4 * q + 0][1]);
                    acc[4 * q + 1][0] = fmaf(wv.y, x0, acc[4 * q + 1][0]);
                    acc[4 * q + 1][1] = fmaf(wv.y, x1, acc[4 * q + 1][1]);
                    acc[4 * q + 2][0] = fmaf(wv.z, x0, acc[4 * q + 2][0]);
                    acc[4 * q + 2][1] = fmaf(wv.z, x1, acc[4 * q + 2][1]);
                    acc[4 * q + 3][0] = fmaf(wv.w, x0, acc[4 * q + 3][0]);
                    acc[4 * q + 3][1] = fmaf(wv.w, x1, acc[4 * q + 3][1]);
                }
                if (ct_block) { act[0] += x0; act[1] += x1; }
            }
        }
        if (more) store_chunk(stage ^ 1);
        __syncthreads();
    }
    // cross-warp reduction
#pragma unroll
    for (int j = 0; j < FC_J; ++j) {
        red[(warp * (FC_J + 1) + j) * FC_IMG + lane] = acc[j][0];
        red[(warp * (FC_J + 1) + j) * FC_IMG + lane + 32] = acc[j][1];
    }
    red[(warp * (FC_J + 1) + FC_J) * FC_IMG + lane] = act[0];
    red[(warp * (FC_J + 1) + FC_J) * FC_IMG + lane + 32] = act[1];
    __syncthreads();
    if (gridDim.z > 1) {
        // split K: FP32 partial sums [z][B][n_out + 1] (column n_out: the
        // carry-through neuron's sum of data inputs); fc_reduce_kernel finishes
        const int ldw = a.n_out + 1;
        float *wz = a.ws + (size_t)blockIdx.z * a.B * ldw;
        for (int e = tid; e < (FC_J + 1) * FC_IMG; e += 256) {
            const int jj = e / FC_IMG, bb = e % FC_IMG;
            const int b = b0 + bb;
            if (b >= a.B) continue;
            if (jj == FC_J && !ct_block) continue;
            const int j = jj == FC_J ? a.n_out : j0 + jj;
            if (jj < FC_J && j >= a.n_out) continue;
            float sum = 0.f;
            for (int wv = 0; wv < FC_WARPS; ++wv) sum += red[(wv * (FC_J + 1) + jj) * FC_IMG + bb];
            wz[(size_t)b * ldw + j] = sum;
        }
        return;
    }
    for (int e = tid; e < FC_J * FC_IMG; e += 256) {
        int jj = e / FC_IMG, bb = e % FC_IMG;
        int j = j0 + jj, b = b0 + bb;
        if (j >= a.n_out || b >= a.B) continue;
        float s = 0.f;
        for (int wv = 0; wv < FC_WARPS; ++wv) s += red[(wv * (FC_J + 1) + jj) * FC_IMG + bb];
        s += a.bias[j];
        if (a.relu) s = relu_keep_nan(s);
        fc_out_row<TY>(a, b)[j] = from_f<TY>(s);
    }
    if (!ct_block) {
        if (a.final_layer && blockIdx.x == 0 && !a.protect) {
            for (int bb = tid; bb < FC_IMG; bb += 256) {
                int b = b0 + bb;
                if (b >= a.B) continue;
                fc_final_out(a, b, __int_as_float(0x7fc00000), 0);
            }
        }
        return;
    }
    const TX *xcs = static_cast<const TX *>(a.xcs);
    for (int bb = tid; bb < FC_IMG; bb += 256) {
        int b = b0 + bb;
        if (b >= a.B) continue;
        float s = 0.f;
        for (int wv = 0; wv < FC_WARPS; ++wv) s += red[(wv * (FC_J + 1) + FC_J) * FC_IMG + bb];
        if (xcs)
            for (int i = 0; i < a.n_cs; ++i) s += to_f(xcs[(size_t)b * a.n_cs + i]);
        s *= a.coef;
        if (a.final_layer) {
            fc_final_out(a, b, s, !(fabs((double)s - a.ref) <= a.tau));
        } else {
            if (a.relu) s = relu_keep_nan(s);
            static_cast<TY *>(a.ycs)[b] = from_f<TY>(s);
        }
    }
}

// Split-K FC: adds the partials in split order, then bias and ReLU (data
// neurons), and the carry-through / accumulated-checksum neuron:
// coef * (sum of data inputs + sum of checksum inputs), with the verdict
// for the final layer.  One thread per (image, neuron), neuron n_out = the
// checksum neuron.
template <typename TX, typename TY>
__global__ void fc_reduce_kernel(FcArgs a, int splits) {
    pdl_wait();
    pdl_trigger();
    const int ldw = a.n_out + 1;
    const long long total = (long long)a.B * ldw;
    const size_t plane = (size_t)a.B * ldw;
    for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < total;
         e += (long long)gridDim.x * blockDim.x) {
        const int b = (int)(e / ldw), j = (int)(e % ldw);
        if (j < a.n_out) {
            float s = 0.f;
            for (int z = 0; z < splits; ++z) s += a.ws[z * plane + (size_t)b * ldw + j];
            s += a.bias[j];
            if (a.relu) s = relu_keep_nan(s);
            fc_out_row<TY>(a, b)[j] = from_f<TY>(s);
            continue;
        }
        if (!a.protect) {
            if (a.final_layer) fc_final_out(a, b, __int_as_float(0x7fc00000), 0);
            continue;
        }
        float s = 0.f;
        for (int z = 0; z < splits; ++z) s += a.ws[z * plane + (size_t)b * ldw + j];
        const TX *xcs = static_cast<const TX *>(a.xcs);
        if (xcs)
            for (int i = 0; i < a.n_cs; ++i) s += to_f(xcs[(size_t)b * a.n_cs + i]);
        s *= a.coef;
        if (a.final_layer) {
            fc_final_out(a, b, s, !(fabs((double)s - a.ref) <= a.tau));
        } else {
            if (a.relu) s = relu_keep_nan(s);
            static_cast<TY *>(a.ycs)[b] = from_f<TY>(s);
        }
    }
}

// ---------------------------------------------------------------------------
// Max-pool over NHWC data and the [N, H, W] checksum plane together.  The
// window maximum is taken on stored values (exact); padding never wins; a
// NaN anywhere in the window gives NaN.  Data: one thread per output pixel
// and 8 (fp16) or 4 (fp32) consecutive channels, 16-byte loads and stores;
// the checksum plane: one thread per output pixel.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void vmax(float &m, float v) { m = (v > m || v != v) ? v : m; }

template <typename T>
__global__ void maxpool_kernel(PoolArgs a) {
    pdl_wait();
    pdl_trigger();
    constexpr int VE = 16 / sizeof(T);
    using V = uint4;
    const int CV = a.C / VE;                       // vectors per pixel (C % VE == 0)
    const int n_pix = a.N * a.P * a.Q;
    const int n_data = n_pix * CV;
    const int n_all = n_data + (a.cs_in ? n_pix : 0);
    for (int e = blockIdx.x * blockDim.x + threadIdx.x; e < n_all; e += gridDim.x * blockDim.x) {
        const bool is_cs = e >= n_data;
        const int i = is_cs ? e - n_data : e;
        const int cv = is_cs ? 0 : i % CV;
        const int pix = is_cs ? i : i / CV;
        const int q = pix % a.Q, t = pix / a.Q, p = t % a.P, n = t / a.P;
        if (is_cs) {
            const T *src = static_cast<const T *>(a.cs_in);
            float m = -INFINITY;
            for (int r = 0; r < a.k; ++r) {
                const int h = p * a.stride + r - a.pad;
                if (h < 0 || h >= a.H) continue;
                for (int s = 0; s < a.k; ++s) {
                    const int w = q * a.stride + s - a.pad;
                    if (w < 0 || w >= a.W) continue;
                    vmax(m, to_f(src[((size_t)n * a.H + h) * a.W + w]));
                }
            }
            static_cast<T *>(a.cs_out)[pix] = from_f<T>(m);
            continue;
        }
        float m[VE];
#pragma unroll
        for (int j = 0; j < VE; ++j) m[j] = -INFINITY;
        const T *src = static_cast<const T *>(a.x);
        for (int r = 0; r < a.k; ++r) {
            const int h = p * a.stride + r - a.pad;
            if (h < 0 || h >= a.H) continue;
            for (int s = 0; s < a.k; ++s) {
                const int w = q * a.stride + s - a.pad;
                if (w < 0 || w >= a.W) continue;
                const V v = *reinterpret_cast<const V *>(src + (((size_t)n * a.H + h) * a.W + w) * a.C + cv * VE);
                const T *tv = reinterpret_cast<const T *>(&v);
#pragma unroll
                for (int j = 0; j < VE; ++j) vmax(m[j], to_f(tv[j]));
            }
        }
        V o;
        T *to = reinterpret_cast<T *>(&o);
#pragma unroll
        for (int j = 0; j < VE; ++j) to[j] = from_f<T>(m[j]);
        *reinterpret_cast<V *>(static_cast<T *>(a.y) + (size_t)pix * a.C + cv * VE) = o;
    }
}

// Scalar fallback for channel counts that are not a multiple of the vector.
template <typename T>
__global__ void maxpool_scalar_kernel(PoolArgs a) {
    pdl_wait();
    pdl_trigger();
    const int64_t n_data = (int64_t)a.N * a.P * a.Q * a.C;
    const int64_t n_cs = a.cs_in ? (int64_t)a.N * a.P * a.Q : 0;
    for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < n_data + n_cs;
         e += (int64_t)gridDim.x * blockDim.x) {
        const bool is_cs = e >= n_data;
        const int64_t i = is_cs ? e - n_data : e;
        const int C = is_cs ? 1 : a.C;
        const int c = (int)(i % C);
        int64_t t = i / C;
        const int q = (int)(t % a.Q); t /= a.Q;
        const int p = (int)(t % a.P);
        const int n = (int)(t / a.P);
        const T *src = static_cast<const T *>(is_cs ? a.cs_in : a.x);
        float m = -INFINITY;
        for (int r = 0; r < a.k; ++r) {
            int h = p * a.stride + r - a.pad;
            if (h < 0 || h >= a.H) continue;
            for (int s = 0; s < a.k; ++s) {
                int w = q * a.stride + s - a.pad;
                if (w < 0 || w >= a.W) continue;
                vmax(m, to_f(src[(((size_t)n * a.H + h) * a.W + w) * C + c]));
            }
        }
        T *dst = static_cast<T *>(is_cs ? a.cs_out : a.y);
        dst[i] = from_f<T>(m);
    }
}

// Global average pool: float [N, C] features (+ float [N] checksum feature).
template <typename T>
__global__ void gap_kernel(PoolArgs a) {
    pdl_wait();
    pdl_trigger();
    const int HW = a.H * a.W;
    const int n = blockIdx.y;
    const int c = blockIdx.x * blockDim.x + threadIdx.x;
    const T *x = static_cast<const T *>(a.x);
    if (c < a.C) {
        float s = 0.f;
        for (int i = 0; i < HW; ++i) s += to_f(x[((size_t)n * HW + i) * a.C + c]);
        static_cast<float *>(a.y)[(size_t)n * a.C + c] = s / (float)HW;
    } else if (c == a.C && a.cs_in) {
        const T *cs = static_cast<const T *>(a.cs_in);
        float s = 0.f;
        for (int i = 0; i < HW; ++i) s += to_f(cs[(size_t)n * HW + i]);
        static_cast<float *>(a.cs_out)[n] = s / (float)HW;
    }
}

// NCHW fp32 -> NHWC storage type, one thread per pixel; channels C..Cp-1
// of the output (padding to Cp channels) are written as zeros.
template <typename T>
__global__ void convert_input_kernel(const float *in, T *out, int N, int C, int Cp, int H, int W, const int32_t *idx) {
    pdl_wait();
    pdl_trigger();
    const int HW = H * W;
    const int total = N * HW;
    for (int e = blockIdx.x * blockDim.x + threadIdx.x; e < total; e += gridDim.x * blockDim.x) {
        const int n = e / HW, hw = e % HW;
        const float *src = in + (size_t)(idx ? idx[n] : n) * C * HW + hw;
        T *dst = out + (size_t)e * Cp;
        for (int c = 0; c < Cp; ++c) dst[c] = from_f<T>(c < C ? src[(size_t)c * HW] : 0.f);
    }
}

__global__ void xor_bit_kernel(void *base, int64_t word, int bit, int word_bytes) {
    pdl_wait();
    pdl_trigger();
    if (word_bytes == 2) static_cast<uint16_t *>(base)[word] ^= (uint16_t)(1u << bit);
    else static_cast<uint32_t *>(base)[word] ^= (1u << bit);
}

// Copies image idx[i] of `in` to row i of `out` (NCHW float rows of `per`
// elements).  16-byte vectors when every row starts 16-byte aligned.
__global__ void gather_images_kernel(const float *in, float *out, const int32_t *idx, int64_t per) {
    pdl_wait();
    pdl_trigger();
    const int i = blockIdx.y;
    const float *s = in + (size_t)idx[i] * per;
    float *d = out + (size_t)i * per;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    const int64_t t0 = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
    if (per % 4 == 0) {
        const float4 *src = reinterpret_cast<const float4 *>(s);
        float4 *dst = reinterpret_cast<float4 *>(d);
        for (int64_t e = t0; e < per / 4; e += stride) dst[e] = src[e];
    } else {
        for (int64_t e = t0; e < per; e += stride) d[e] = s[e];
    }
}

__global__ void scatter_rows_kernel(const float *src, float *dst, const int32_t *idx, int n, int row) {
    pdl_wait();
    pdl_trigger();
    for (int e = blockIdx.x * blockDim.x + threadIdx.x; e < n * row; e += gridDim.x * blockDim.x) {
        int i = e / row, c = e % row;
        dst[(size_t)idx[i] * row + c] = src[e];
    }
}

int grid_for(int64_t n, int threads) {
    int64_t g = (n + threads - 1) / threads;
    if (g > 152 * 32) g = 152 * 32;
    return (int)(g < 1 ? 1 : g);
}

template <typename TX, typename TW, typename TY>
cudaError_t fc_go(const FcArgs &a, cudaStream_t st, int *n_kernels) {
    const size_t smem =
        sizeof(float) * (2 * (FC_IMG * FC_XP + FC_KC * FC_J) + FC_WARPS * (FC_J + 1) * FC_IMG);
    static bool attr = false;
    if (!attr) {
        cudaError_t e = cudaFuncSetAttribute(fc_kernel<TX, TW, TY>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        attr = true;
    }
    const int gx = (a.n_out + FC_J - 1) / FC_J, gy = (a.B + FC_IMG - 1) / FC_IMG;
    // split K when the output blocks leave most SMs idle (at least 4 chunks of 64 inputs each)
    static int sms = 0;
    if (sms == 0) sms = device_sm_count();
    const int nkc = (a.n_in + FC_KC - 1) / FC_KC;
    const int splits = splitk_choose(gx * gy, nkc, 4, 2 * sms, a.B, a.n_out + 1, a.ws ? a.ws_bytes : 0);
    dim3 grid(gx, gy, splits);
    pdl_launch(fc_kernel<TX, TW, TY>, grid, 256, smem, st, a);
    cudaError_t e = cudaGetLastError();
    if (n_kernels) *n_kernels = 1;
    if (e != cudaSuccess || splits == 1) return e;
    if (n_kernels) *n_kernels = 2;
    const long long total = (long long)a.B * (a.n_out + 1);
    pdl_launch(fc_reduce_kernel<TX, TY>, (int)std::min<long long>((total + 255) / 256, 4096), 256, 0, st, a, splits);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_fc(const FcArgs &a, bool half, bool x_float, cudaStream_t st, int *n_kernels) {
    if (!half) return fc_go<float, float, float>(a, st, n_kernels);
    if (a.final_layer)
        return x_float ? fc_go<float, __half, float>(a, st, n_kernels) : fc_go<__half, __half, float>(a, st, n_kernels);
    return x_float ? fc_go<float, __half, __half>(a, st, n_kernels) : fc_go<__half, __half, __half>(a, st, n_kernels);
}

cudaError_t launch_maxpool(const PoolArgs &a, bool half, cudaStream_t st) {
    const int ve = half ? 8 : 4;
    const int64_t pix = (int64_t)a.N * a.P * a.Q;
    if (a.C % ve == 0 && pix * (a.C / ve + 1) < (1ll << 31)) {
        const int64_t n = pix * (a.C / ve + (a.cs_in ? 1 : 0));
        if (half) pdl_launch(maxpool_kernel<__half>, grid_for(n, 256), 256, 0, st, a);
        else pdl_launch(maxpool_kernel<float>, grid_for(n, 256), 256, 0, st, a);
    } else {
        const int64_t n = pix * (a.C + (a.cs_in ? 1 : 0));
        if (half) pdl_launch(maxpool_scalar_kernel<__half>, grid_for(n, 256), 256, 0, st, a);
        else pdl_launch(maxpool_scalar_kernel<float>, grid_for(n, 256), 256, 0, st, a);
    }
    return cudaGetLastError();
}

cudaError_t launch_gap(const PoolArgs &a, bool half, cudaStream_t st) {
    dim3 grid((a.C + 1 + 127) / 128, a.N);
    if (half) pdl_launch(gap_kernel<__half>, grid, 128, 0, st, a);
    else pdl_launch(gap_kernel<float>, grid, 128, 0, st, a);
    return cudaGetLastError();
}

cudaError_t launch_convert_input(const float *in, void *out, int N, int C, int Cp, int H, int W, bool half,
                                 cudaStream_t st, const int32_t *idx) {
    const int64_t n = (int64_t)N * H * W;
    if (half) pdl_launch(convert_input_kernel<__half>, grid_for(n, 256), 256, 0, st, in, (__half *)out, N, C, Cp, H, W, idx);
    else pdl_launch(convert_input_kernel<float>, grid_for(n, 256), 256, 0, st, in, (float *)out, N, C, Cp, H, W, idx);
    return cudaGetLastError();
}

cudaError_t launch_xor_bit(void *base, int64_t word, int bit, int word_bytes, cudaStream_t st) {
    pdl_launch(xor_bit_kernel, 1, 1, 0, st, base, word, bit, word_bytes);
    return cudaGetLastError();
}

cudaError_t launch_gather_images(const float *in, float *out, const int32_t *idx, int n,
                                 int64_t per_image, cudaStream_t st) {
    if (n <= 0) return cudaSuccess;
    const int64_t blocks = (per_image / 4 + 255) / 256 + 1;
    dim3 grid((unsigned)(blocks > 64 ? 64 : blocks), n);
    pdl_launch(gather_images_kernel, grid, 256, 0, st, in, out, idx, per_image);
    return cudaGetLastError();
}

cudaError_t launch_scatter_rows(const float *src, float *dst, const int32_t *idx, int n, int row,
                                cudaStream_t st) {
    if (n <= 0) return cudaSuccess;
    pdl_launch(scatter_rows_kernel, grid_for((int64_t)n * row, 256), 256, 0, st, src, dst, idx, n, row);
    return cudaGetLastError();
}

}  // namespace ct
