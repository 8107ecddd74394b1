// CUDA-core implicit-GEMM convolution with the carry-through filter.
//
// GEMM view: M = N*P*Q output pixels, N_gemm = K output channels,
// K_gemm = R*S*C taps-by-channels (C innermost, matching NHWC activations
// and KRSC weights).  FP32 FFMA accumulation (no TF32) for both FP32 and
// FP16 storage.
//
// The carry-through filter of Sec. II-A (a 1 at the kernel centre over every
// input channel) is not materialised as a GEMM column: its output is the
// channel sum of the centre-tap slice of the im2col tile, which this kernel
// already stages in shared memory.  Blocks of the first channel tile add the
// staged centre-tap values row by row while they run the main loop, so the
// checksum costs R*S times fewer adds than one more GEMM column would.  The
// incoming checksum plane enters only the checksum output (coefficient 1 at
// the centre), never the data outputs, whose zero slice is thus structural.
//
// Epilogue on data and checksum alike: + bias (0 for the checksum),
// + residual, ReLU (x < 0 -> +0, NaN kept), store in the storage type.
#include "ct_internal.h"

namespace ct {
namespace {

template <typename T> struct Vec;
template <> struct Vec<float> { using type = float4; static constexpr int n = 4; };
template <> struct Vec<__half> { using type = uint4; static constexpr int n = 8; };

__device__ __forceinline__ float to_f(float v) { return v; }
__device__ __forceinline__ float to_f(__half v) { return __half2float(v); }
template <typename T> __device__ __forceinline__ T from_f(float v);
template <> __device__ __forceinline__ float from_f<float>(float v) { return v; }
template <> __device__ __forceinline__ __half from_f<__half>(float v) { return __float2half_rn(v); }

__device__ __forceinline__ float relu_keep_nan(float v) { return v < 0.f ? 0.f : v; }

template <typename T>
__device__ __forceinline__ void unpack(const typename Vec<T>::type &v, float *o);
template <> __device__ __forceinline__ void unpack<float>(const float4 &v, float *o) {
    o[0] = v.x; o[1] = v.y; o[2] = v.z; o[3] = v.w;
}
template <> __device__ __forceinline__ void unpack<__half>(const uint4 &v, float *o) {
    const __half2 *h = reinterpret_cast<const __half2 *>(&v);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        float2 f = __half22float2(h[i]);
        o[2 * i] = f.x; o[2 * i + 1] = f.y;
    }
}

// Value of input element (n, h, w, c) of an NHWC tensor, 0 outside.
template <typename T>
__device__ __forceinline__ float load_x(const T *x, int n, int h, int w, int c, int H, int W, int C) {
    if (h < 0 || h >= H || w < 0 || w >= W) return 0.f;
    return to_f(x[(((size_t)n * H + h) * W + w) * C + c]);
}

// Output column j (0 .. TN) of thread column tx within the block's BN columns:
// groups of 4 consecutive columns, the groups of one thread BN / (TN / 4)
// apart, so that the 16-byte shared-memory reads of a warp's threads cover
// consecutive 16-byte pieces (no bank conflicts) for every TN.
template <int BN, int TN>
__device__ __forceinline__ int col_of(int tx, int j) {
    return (j / 4) * (BN / (TN / 4)) + tx * 4 + (j % 4);
}

// two blocks per SM: 256-thread blocks stay at or below 128 registers
template <typename T, int BM, int BN, int BK, int TM, int TN, bool VEC>
__global__ void __launch_bounds__((BM / TM) * (BN / TN), 2)
conv_simt_kernel(ConvArgs a) {
    pdl_wait();
    pdl_trigger();
    constexpr int NT = (BM / TM) * (BN / TN);
    constexpr int VE = Vec<T>::n;                 // elements per 16-byte vector
    constexpr int UPR = VEC ? BK / VE : 1;        // load units per tile row
    constexpr int A_UNITS = VEC ? BM * UPR : BM * BK;
    constexpr int B_UNITS = VEC ? BN * UPR : BN * BK;
    constexpr int A_PER = (A_UNITS + NT - 1) / NT;
    constexpr int B_PER = (B_UNITS + NT - 1) / NT;
    constexpr int AE = VEC ? VE : 1;              // elements per unit
    static_assert(!VEC || BK % VE == 0, "BK must hold whole vectors");

    // row pitches BM + 4 and BN + 4 keep every row 16-byte aligned (float4 reads)
    __shared__ __align__(16) float As[2][BK][BM + 4];
    __shared__ __align__(16) float Bs[2][BK][BN + 4];

    const T *x = static_cast<const T *>(a.x);
    const T *w = static_cast<const T *>(a.w);
    const int tid = threadIdx.x;
    const int tx = tid % (BN / TN), ty = tid / (BN / TN);
    const int M = a.N * a.P * a.Q;
    const int m0 = blockIdx.x * BM, n0 = blockIdx.y * BN;
    const int Ktot = a.R * a.S * a.C;
    const int ctr_tap = ((a.R - 1) / 2) * a.S + (a.S - 1) / 2;
    const bool do_cs = (a.role == CT_ROLE_CT) && a.cs_out != nullptr && blockIdx.y == 0;
    // K indices of the centre tap: [ctr_tap * C, (ctr_tap + 1) * C)
    const int ctr_lo = ctr_tap * a.C, ctr_hi = ctr_lo + a.C;

    // per-unit pixel decode for the A loads (fixed rows across the K loop)
    int a_row[A_PER], a_n[A_PER], a_h0[A_PER], a_w0[A_PER], a_sub[A_PER];
#pragma unroll
    for (int i = 0; i < A_PER; ++i) {
        int u = tid + i * NT;
        int row = VEC ? u / UPR : u / BK;
        a_sub[i] = VEC ? (u % UPR) * VE : u % BK;
        a_row[i] = (u < A_UNITS) ? row : -1;
        int m = m0 + row;
        if (u >= A_UNITS || m >= M) { a_n[i] = -1; a_h0[i] = 0; a_w0[i] = 0; continue; }
        int q = m % a.Q, t = m / a.Q, p = t % a.P;
        a_n[i] = t / a.P;
        a_h0[i] = p * a.stride - a.pad;
        a_w0[i] = q * a.stride - a.pad;
    }

    float areg[A_PER][AE];
    float breg[B_PER][AE];

    auto load_tiles = [&](int kt) {
        const int k0 = kt * BK;
        // the tap and channel of this K tile (C is a multiple of BK on the
        // vector path: one tap per K tile), computed once per tile
        const int tap_k = VEC ? k0 / a.C : 0;
        const int c_k = VEC ? k0 - tap_k * a.C : 0;
        const int r_k = VEC ? tap_k / a.S : 0, s_k = VEC ? tap_k - r_k * a.S : 0;
#pragma unroll
        for (int i = 0; i < A_PER; ++i) {
#pragma unroll
            for (int e = 0; e < AE; ++e) areg[i][e] = 0.f;
            if (a_n[i] < 0) continue;
            if (VEC) {
                const int c0 = c_k + a_sub[i];
                const int h = a_h0[i] + r_k, ww = a_w0[i] + s_k;
                if (h >= 0 && h < a.H && ww >= 0 && ww < a.W) {
                    const typename Vec<T>::type *p = reinterpret_cast<const typename Vec<T>::type *>(
                        x + (((size_t)a_n[i] * a.H + h) * a.W + ww) * a.C + c0);
                    unpack<T>(__ldg(p), areg[i]);
                }
            } else {
                int k = k0 + a_sub[i];
                if (k < Ktot) {
                    int tap = k / a.C, c = k % a.C;
                    int r = tap / a.S, s = tap % a.S;
                    areg[i][0] = load_x(x, a_n[i], a_h0[i] + r, a_w0[i] + s, c, a.H, a.W, a.C);
                }
            }
        }
#pragma unroll
        for (int i = 0; i < B_PER; ++i) {
            int u = tid + i * NT;
#pragma unroll
            for (int e = 0; e < AE; ++e) breg[i][e] = 0.f;
            if (u >= B_UNITS) continue;
            int row = VEC ? u / UPR : u / BK;
            int sub = VEC ? (u % UPR) * VE : u % BK;
            int n = n0 + row;
            if (n >= a.K) continue;
            if (VEC) {
                const typename Vec<T>::type *p = reinterpret_cast<const typename Vec<T>::type *>(
                    w + (size_t)n * Ktot + k0 + sub);
                unpack<T>(__ldg(p), breg[i]);
            } else {
                int k = k0 + sub;
                if (k < Ktot) breg[i][0] = to_f(w[(size_t)n * Ktot + k]);
            }
        }
    };
    auto store_tiles = [&](int buf) {
#pragma unroll
        for (int i = 0; i < A_PER; ++i) {
            if (a_row[i] < 0) continue;
#pragma unroll
            for (int e = 0; e < AE; ++e) As[buf][a_sub[i] + e][a_row[i]] = areg[i][e];
        }
#pragma unroll
        for (int i = 0; i < B_PER; ++i) {
            int u = tid + i * NT;
            if (u >= B_UNITS) continue;
            int row = VEC ? u / UPR : u / BK;
            int sub = VEC ? (u % UPR) * VE : u % BK;
#pragma unroll
            for (int e = 0; e < AE; ++e) Bs[buf][sub + e][row] = breg[i][e];
        }
    };

    float acc[TM][TN];
    float csum[TM];
#pragma unroll
    for (int i = 0; i < TM; ++i) {
        csum[i] = 0.f;
#pragma unroll
        for (int j = 0; j < TN; ++j) acc[i][j] = 0.f;
    }

    // K tiles of this block: all of them, or one split's range (gridDim.z > 1)
    const int nk_all = (Ktot + BK - 1) / BK;
    const int kps = (nk_all + gridDim.z - 1) / gridDim.z;
    const int kt_lo = blockIdx.z * kps, kt_hi = min(nk_all, kt_lo + kps);
    if (kt_lo < kt_hi) {
        load_tiles(kt_lo);
        store_tiles(0);
    }
    __syncthreads();
    // one K step: TM x TN FFMAs from two rows of the staged tiles; on the
    // centre tap's K tiles of the first channel tile the A values are also
    // summed for the carry-through output (same order as before: k ascending)
    auto kstep = [&](int buf, int kk, bool ctr) {
        float av[TM], bv[TN];
#pragma unroll
        for (int i = 0; i < TM; i += 4) {
            float4 v = *reinterpret_cast<const float4 *>(&As[buf][kk][ty * TM + i]);
            av[i] = v.x; av[i + 1] = v.y; av[i + 2] = v.z; av[i + 3] = v.w;
        }
#pragma unroll
        for (int j = 0; j < TN; j += 4) {
            float4 v = *reinterpret_cast<const float4 *>(&Bs[buf][kk][col_of<BN, TN>(tx, j)]);
            bv[j] = v.x; bv[j + 1] = v.y; bv[j + 2] = v.z; bv[j + 3] = v.w;
        }
#pragma unroll
        for (int i = 0; i < TM; ++i)
#pragma unroll
            for (int j = 0; j < TN; ++j) acc[i][j] = fmaf(av[i], bv[j], acc[i][j]);
        if (ctr) {
#pragma unroll
            for (int i = 0; i < TM; ++i) csum[i] += av[i];
        }
    };
    for (int kt = kt_lo; kt < kt_hi; ++kt) {
        const int buf = (kt - kt_lo) & 1;
        if (kt + 1 < kt_hi) load_tiles(kt + 1);
        const int k0 = kt * BK;
        // a K tile lies wholly inside or outside the centre tap's K range
        // when C is a multiple of BK (vector path); otherwise test each k
        if (!do_cs) {
#pragma unroll
            for (int kk = 0; kk < BK; ++kk) kstep(buf, kk, false);
        } else if (VEC) {
            const bool ctr = k0 >= ctr_lo && k0 < ctr_hi;
            if (ctr) {
#pragma unroll
                for (int kk = 0; kk < BK; ++kk) kstep(buf, kk, true);
            } else {
#pragma unroll
                for (int kk = 0; kk < BK; ++kk) kstep(buf, kk, false);
            }
        } else {
#pragma unroll
            for (int kk = 0; kk < BK; ++kk) kstep(buf, kk, k0 + kk >= ctr_lo && k0 + kk < ctr_hi);
        }
        if (kt + 1 < kt_hi) store_tiles(buf ^ 1);
        __syncthreads();
    }

    if (gridDim.z > 1) {
        // split-K: FP32 partial sums; the reduction kernel applies the epilogue
        const int ws_ld = (a.K + 1 + 3) & ~3;
        float *wz = a.ws + (size_t)blockIdx.z * M * ws_ld;
#pragma unroll
        for (int i = 0; i < TM; ++i) {
            const int m = m0 + ty * TM + i;
            if (m >= M) break;
#pragma unroll
            for (int j = 0; j < TN; ++j) {
                const int k = n0 + col_of<BN, TN>(tx, j);
                if (k < a.K) wz[(size_t)m * ws_ld + k] = acc[i][j];
            }
            if (a.cs_out != nullptr && blockIdx.y == 0 && tx == 0)
                wz[(size_t)m * ws_ld + a.K] = do_cs ? a.coef * csum[i] : 0.f;
        }
        return;
    }

    // ---- epilogue ----
    const T *res = static_cast<const T *>(a.res);
    T *y = static_cast<T *>(a.y);
    const FaultDelta fd = a.fd;
    const int ctr_r = (a.R - 1) / 2, ctr_s = (a.S - 1) / 2;
#pragma unroll
    for (int i = 0; i < TM; ++i) {
        const int m = m0 + ty * TM + i;
        if (m >= M) break;
        const int q = m % a.Q, t = m / a.Q, p = t % a.P, n = t / a.P;
        float v[TN];
#pragma unroll
        for (int j = 0; j < TN; ++j) {
            const int k = n0 + col_of<BN, TN>(tx, j);
            v[j] = 0.f;
            if (k >= a.K) continue;
            float o = acc[i][j] + a.bias[k];
            if (fd.active && fd.kout == k) {
                int h = p * a.stride + fd.r - a.pad, ww = q * a.stride + fd.s - a.pad;
                float src = 0.f;
                if (fd.cin < a.C) src = load_x(x, n, h, ww, fd.cin, a.H, a.W, a.C);
                else if (a.cs_in && h >= 0 && h < a.H && ww >= 0 && ww < a.W)
                    src = to_f(static_cast<const T *>(a.cs_in)[((size_t)n * a.H + h) * a.W + ww]);
                o += fd.dv * src;
            }
            if (res) o += to_f(res[(size_t)m * a.K + k]);
            if (a.relu) o = relu_keep_nan(o);
            v[j] = o;
        }
        // groups of 4 consecutive columns: vector stores when the group is whole
#pragma unroll
        for (int j = 0; j < TN; j += 4) {
            const int kb = n0 + col_of<BN, TN>(tx, j);
            if (kb + 4 <= a.K && (a.K % 4) == 0) {
                if constexpr (sizeof(T) == 4) {
                    *reinterpret_cast<float4 *>(&y[(size_t)m * a.K + kb]) = make_float4(v[j], v[j + 1], v[j + 2], v[j + 3]);
                } else {
                    __half2 h0 = __floats2half2_rn(v[j], v[j + 1]);
                    __half2 h1 = __floats2half2_rn(v[j + 2], v[j + 3]);
                    uint2 pk;
                    pk.x = *reinterpret_cast<uint32_t *>(&h0);
                    pk.y = *reinterpret_cast<uint32_t *>(&h1);
                    *reinterpret_cast<uint2 *>(&y[(size_t)m * a.K + kb]) = pk;
                }
            } else {
#pragma unroll
                for (int e = 0; e < 4; ++e)
                    if (kb + e < a.K) y[(size_t)m * a.K + kb + e] = from_f<T>(v[j + e]);
            }
        }
        // checksum output: one thread column of the first channel tile
        if (a.cs_out != nullptr && blockIdx.y == 0 && tx == 0) {
            const T *csi = static_cast<const T *>(a.cs_in);
            const int hc = p * a.stride + ctr_r - a.pad, wc = q * a.stride + ctr_s - a.pad;
            const bool inb = hc >= 0 && hc < a.H && wc >= 0 && wc < a.W;
            float cin = (csi && inb) ? to_f(csi[((size_t)n * a.H + hc) * a.W + wc]) : 0.f;
            float o = 0.f;
            if (a.role == CT_ROLE_CT) o = a.coef * (csum[i] + cin);
            else if (a.role == CT_ROLE_PASS) o = cin;
            if (fd.active && fd.kout == a.K) {
                int h = p * a.stride + fd.r - a.pad, ww = q * a.stride + fd.s - a.pad;
                float src = 0.f;
                if (fd.cin < a.C) src = load_x(x, n, h, ww, fd.cin, a.H, a.W, a.C);
                else if (csi && h >= 0 && h < a.H && ww >= 0 && ww < a.W)
                    src = to_f(csi[((size_t)n * a.H + h) * a.W + ww]);
                o += fd.dv * src;
            }
            if (a.res_cs) o += to_f(static_cast<const T *>(a.res_cs)[m]);
            if (a.relu) o = relu_keep_nan(o);
            static_cast<T *>(a.cs_out)[m] = from_f<T>(o);
        }
    }
}

int sm_count_cached() {
    static int n = 0;
    if (n == 0) n = device_sm_count();
    return n;
}

template <typename T, int BM, int BN, int BK, int TM, int TN, bool VEC>
cudaError_t go(const ConvArgs &a, cudaStream_t st, int *n_kernels) {
    const int M = a.N * a.P * a.Q;
    const int gx = (M + BM - 1) / BM, gy = (a.K + BN - 1) / BN;
    // split K when the output tiles leave most SMs idle (at least 8 K tiles per split)
    const int ws_ld = (a.K + 1 + 3) & ~3;
    const int nk = (a.R * a.S * a.C + BK - 1) / BK;
    const int splits = (a.K % 8 == 0) ? splitk_choose(gx * gy, nk, 8, 2 * sm_count_cached(), M, ws_ld,
                                                      a.ws ? a.ws_bytes : 0) : 1;
    dim3 grid(gx, gy, splits);
    pdl_launch(conv_simt_kernel<T, BM, BN, BK, TM, TN, VEC>, grid, (BM / TM) * (BN / TN), 0, st, a);
    cudaError_t e = cudaGetLastError();
    if (n_kernels) *n_kernels = 1;
    if (e != cudaSuccess || splits == 1) return e;
    if (n_kernels) *n_kernels = 2;
    return launch_splitk_reduce(a, splits, ws_ld, sizeof(T) == 2, st);
}

template <typename T>
cudaError_t dispatch(const ConvArgs &a, cudaStream_t st, int *nk) {
    constexpr int VE = Vec<T>::n;
    const bool vec = (a.C % 16 == 0) && (a.C % VE == 0);
    if (vec) {
        if (a.K >= 128) return go<T, 128, 128, 16, 8, 8, true>(a, st, nk);
        return go<T, 128, 64, 16, 8, 4, true>(a, st, nk);
    }
    if (a.K <= 16) return go<T, 64, 16, 16, 4, 4, false>(a, st, nk);
    return go<T, 128, 64, 16, 8, 4, false>(a, st, nk);
}

}  // namespace

cudaError_t launch_conv_simt(const ConvArgs &a, bool half, cudaStream_t st, int *n_kernels) {
    return half ? dispatch<__half>(a, st, n_kernels) : dispatch<float>(a, st, n_kernels);
}

}  // namespace ct
