// Tensor-core (tcgen05) implicit-GEMM convolutions with the carry-through
// filter, FP16 storage, FP32 accumulation in TMEM.
//
// GEMM view: D[m, n] = sum_k A[m, k] B[n, k] with m = output pixel (n, p, q),
// n = output channel, k = (tap, channel), channels innermost.
//   A (128 pixels x 64 channels of one tap) is fetched by TMA in im2col mode
//     from the NHWC input (conv_tc_kernel), or as one 18 x 10 pixel patch
//     whose nine shifted views are the nine taps (conv_tc_halo_kernel); the
//     tiles are 128-byte swizzled and K-major.
//   B (BN channels x 64) is fetched by tiled TMA from the KRSC weights.
//   The carry-through filter of Sec. II-A is one more GEMM row: coef at the
//     centre tap of every input channel, 0 elsewhere.  For BN <= 128 its
//     non-zero part is a constant 16-row tile (row 0 = coef) kept after the
//     weight rows in shared memory, and the centre-tap K blocks, which the
//     K loop visits first, are issued with N = BN + 16: the tensor core
//     computes the checksum column.  For BN = 256 two spare warps compute it
//     from the same A tiles with warp-level MMAs against a ones vector
//     (conv_tc_kernel), or the epilogue adds up the centre-tap pixel's
//     channels (conv_tc_pair_kernel).
//   The incoming checksum plane (weight coef at the centre), the residual
//   checksum and the epilogue (bias, residual, ReLU) are applied by the
//   epilogue warps.
//
// The kernels are persistent: one CTA per SM walks a static list of output
// tiles.  The TMA producers run ahead across tile boundaries through a ring
// of shared-memory stages.  N = 64 tiles spread consecutive K blocks over
// four independent TMEM accumulators (chains), because back-to-back short
// MMAs into one accumulator wait on each other; the epilogue sums the
// chains.  N = 128 and N = 256 tiles use one accumulator, and two of them
// alternate in TMEM, so that a tile's MMAs overlap the previous tile's
// epilogue.  A 1x1 shortcut that reads the same input at the same stride
// (a ResNet downsample) can run in the launch of its block's first
// convolution, whose centre-tap K blocks are its A operand (UnitSeq).
//
// With N = 256 and no split K, conv_tc_pair_kernel runs the tiles on pairs of
// CTAs (a cluster of two, tcgen05 cta_group::2): one M = 256 MMA reads the
// 128 A rows and 128 weight rows each CTA holds, which halves the weight
// bytes every SM copies and reads per step.  Its epilogue sums the
// carry-through column from the centre-tap input pixel.
//
// Warp roles.  conv_tc_kernel: a producer group (producer warps, each owning
// whole ring slots, plus for N = 256 the two carry-through warps), one MMA
// warp (one elected lane issues tcgen05.mma), eight epilogue warps;
// conv_tc_pair_kernel: three producer warps, each owning two ring slots (with
// two, the copy issue held the 7 x 7 layers back by 8%, measured), the MMA
// warp (issuing in the even CTA only), eight epilogue warps.
// conv_tc_halo_kernel (320 threads): warp 0 issues TMA, warp 1 the MMAs,
// warps 2-9 the epilogue.  Each TMEM lane quadrant (32 output pixels) is
// read by two epilogue warps, each taking half of the tile's channels.
// Every mbarrier wait is bounded; on expiry the kernel records an error code
// in a device word, stops issuing work and exits after releasing TMEM.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <string.h>

#include <algorithm>
#include <mutex>
#include <vector>

#include "ct_internal.h"
#include "tc_common.cuh"

namespace ct {

namespace {

using namespace tc;

constexpr int BM = 128;            // output pixels per tile (TMEM lanes)
constexpr int BK = 64;             // channels per K block (128 bytes of fp16)
constexpr int A_BYTES = BM * BK * 2;
constexpr int NTHREADS = 320;      // 1 TMA warp, 1 MMA warp, 8 epilogue warps
constexpr int N_EPI_WARPS = 8;
// conv_tc_kernel: a producer group (TMA producer warps, each owning whole ring
// slots, plus for N = 256 two carry-through warps), one MMA warp, 8 epilogue
// warps.  The group is as large as the variant needs: a warp fewer raises the
// register budget of a 1-CTA-per-SM kernel (384 threads: 168 registers, 416:
// 128).
constexpr int tc_nprod(int BN, int STAGES) {
    return BN > 128 ? 2 : STAGES % 4 == 0 ? 4 : STAGES % 3 == 0 ? 3 : STAGES % 2 == 0 ? 2 : 1;
}
constexpr int tc_npg(int BN, int STAGES) { return BN > 128 ? 4 : tc_nprod(BN, STAGES); }
constexpr int tc_threads(int BN, int STAGES) { return 32 * (tc_npg(BN, STAGES) + 1 + N_EPI_WARPS); }

enum CtMode { CT_NONE_ = 0, CT_MERGED = 1, CT_SEPARATE = 2 };

struct TcGeom {
    int M, PQ, Q, stride, pad, C, K, RSC;
    int n_kb, cpb, ctr_tap, S;
    int ct_mode;
    int tmem_cols;
    int m_tiles, n_tiles;
    int splits, kps, ws_ld;      // split-K: K blocks per split, workspace row length
    // conv_tc_pair_kernel<true>: tiles t_first .. end are each run as two
    // 128-channel halves, units 0 .. units - t_first - 1 (unit 2 * (tile -
    // t_first) + half); whole tiles 0 .. t_first - 1 follow them
    int t_first, units;
    // a 1x1 shortcut convolution run by the same launch (its items follow
    // this layer's; see UnitSeq): its item count (0: none), and its split:
    // CTAs (or pairs) 0 .. sc_s0 - 1 share items 0 .. sc_x - 1 evenly, the
    // others the rest
    int sc_items, sc_s0, sc_x;
    uint16_t coef_h;
};

// K-block range [lo, hi) and output tile of persistent work item `item`.
struct TileRef {
    int m0, n_tile, sp, kb_lo, kb_hi;
};
__device__ __forceinline__ TileRef tile_ref(int item, const TcGeom &g) {
    TileRef t;
    const int per = g.m_tiles * g.n_tiles;
    t.sp = item / per;
    const int rt = item - t.sp * per;
    t.m0 = (rt / g.n_tiles) * BM;
    t.n_tile = rt % g.n_tiles;
    t.kb_lo = t.sp * g.kps;
    t.kb_hi = min(g.n_kb, t.kb_lo + g.kps);
    return t;
}


// Work units of one CTA (or CTA pair) cid of ncl: first this layer's n1
// units, round-robin (cid, cid + ncl, ...), then a contiguous share of the
// shortcut's items: CTAs 0 .. sc_s0 - 1 split items 0 .. sc_x - 1 evenly and
// the others split the rest, so that the host can give more of them to the
// CTAs with fewer units of this layer.
// The shortcut is a 1x1 convolution of the same input at the same stride,
// whose pixel is this layer's centre tap: its A operand is this layer's
// centre-tap K blocks (same tensor map and coordinates); its weights,
// epilogue arguments and geometry are its own.  Its units are numbered
// n1 + item.
struct UnitSeq {
    int n1, k1, lo, cnt;
};
template <bool SC>
__device__ __forceinline__ UnitSeq unit_seq(int cid, int ncl, int n1, const TcGeom &g) {
    UnitSeq s;
    s.n1 = n1;
    s.k1 = cid < n1 ? (n1 - 1 - cid) / ncl + 1 : 0;
    s.lo = 0;
    s.cnt = 0;
    if (SC && g.sc_items > 0) {
        if (cid < g.sc_s0) {
            s.lo = (int)(((long long)cid * g.sc_x) / g.sc_s0);
            s.cnt = (int)(((long long)(cid + 1) * g.sc_x) / g.sc_s0) - s.lo;
        } else {
            const int nc = ncl - g.sc_s0, c = cid - g.sc_s0, rest = g.sc_items - g.sc_x;
            s.lo = g.sc_x + (int)(((long long)c * rest) / nc);
            s.cnt = g.sc_x + (int)(((long long)(c + 1) * rest) / nc) - s.lo;
        }
    }
    return s;
}
__device__ __forceinline__ int unit_at(const UnitSeq &s, int k, int cid, int ncl) {
    return k < s.k1 ? cid + k * ncl : s.n1 + s.lo + (k - s.k1);
}

// tap visited at K-block kb: the centre tap first, the others in order
__device__ __forceinline__ int tap_of(int t, int ctr) { return t == 0 ? ctr : (t <= ctr ? t - 1 : t); }

// Epilogue of one 16-channel chunk for one output pixel m: bias, fault delta,
// residual, ReLU, fp16 store (32 bytes).
__device__ __forceinline__ void store_chunk(const float *v, const ConvArgs &a, int K, size_t m, int k0,
                                            float fsrc) {
    const __half *res = static_cast<const __half *>(a.res);
    const size_t base = m * K + k0;
    float rv[16];
    if (res) {
        const uint4 *rp = reinterpret_cast<const uint4 *>(res + base);
        uint4 r0 = rp[0], r1 = rp[1];
        const __half2 *h0 = reinterpret_cast<const __half2 *>(&r0);
        const __half2 *h1 = reinterpret_cast<const __half2 *>(&r1);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            float2 f0 = __half22float2(h0[i]), f1 = __half22float2(h1[i]);
            rv[2 * i] = f0.x; rv[2 * i + 1] = f0.y; rv[8 + 2 * i] = f1.x; rv[8 + 2 * i + 1] = f1.y;
        }
    }
    const FaultDelta &fd = a.fd;
    uint32_t packed[8];
#pragma unroll
    for (int i = 0; i < 16; i += 2) {
        float o[2];
#pragma unroll
        for (int j = 0; j < 2; ++j) {
            const int k = k0 + i + j;
            float t = v[i + j] + __ldg(a.bias + k);
            if (fd.active && fd.kout == k) t += fd.dv * fsrc;
            if (res) t += rv[i + j];
            if (a.relu) t = relu_keep_nan(t);
            o[j] = t;
        }
        __half2 hh = __floats2half2_rn(o[0], o[1]);
        packed[i / 2] = *reinterpret_cast<uint32_t *>(&hh);
    }
    uint4 *yp = reinterpret_cast<uint4 *>(static_cast<__half *>(a.y) + base);
    yp[0] = make_uint4(packed[0], packed[1], packed[2], packed[3]);
    yp[1] = make_uint4(packed[4], packed[5], packed[6], packed[7]);
}

// Residual of 16 channels of one pixel, loaded before the accumulator is
// ready so that its memory latency overlaps the MMAs.
struct Res16 {
    uint4 r0, r1;
};
__device__ __forceinline__ Res16 load_res16(const ConvArgs &a, int K, size_t m, int k0) {
    Res16 r;
    if (a.res) {
        // K and k0 are multiples of 16 channels: 32-byte aligned
        uint32_t w[8];
        ld_global_nc_v8(static_cast<const __half *>(a.res) + m * K + k0, w);
        r.r0 = make_uint4(w[0], w[1], w[2], w[3]);
        r.r1 = make_uint4(w[4], w[5], w[6], w[7]);
    } else {
        r.r0 = r.r1 = make_uint4(0u, 0u, 0u, 0u);
    }
    return r;
}

// store_chunk with the residual already loaded
__device__ __forceinline__ void store_chunk_pre(const float *v, const Res16 &r, const ConvArgs &a, int K, size_t m,
                                                int k0, float fsrc) {
    float rv[16];
    {
        const __half2 *h0 = reinterpret_cast<const __half2 *>(&r.r0);
        const __half2 *h1 = reinterpret_cast<const __half2 *>(&r.r1);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            float2 f0 = __half22float2(h0[i]), f1 = __half22float2(h1[i]);
            rv[2 * i] = f0.x; rv[2 * i + 1] = f0.y; rv[8 + 2 * i] = f1.x; rv[8 + 2 * i + 1] = f1.y;
        }
    }
    const bool res = a.res != nullptr;
    const FaultDelta &fd = a.fd;
    uint32_t packed[8];
#pragma unroll
    for (int i = 0; i < 16; i += 2) {
        float o[2];
#pragma unroll
        for (int j = 0; j < 2; ++j) {
            const int k = k0 + i + j;
            float t = v[i + j] + __ldg(a.bias + k);
            if (fd.active && fd.kout == k) t += fd.dv * fsrc;
            if (res) t += rv[i + j];
            if (a.relu) t = relu_keep_nan(t);
            o[j] = t;
        }
        __half2 hh = __floats2half2_rn(o[0], o[1]);
        packed[i / 2] = *reinterpret_cast<uint32_t *>(&hh);
    }
    uint4 *yp = reinterpret_cast<uint4 *>(static_cast<__half *>(a.y) + m * K + k0);
    yp[0] = make_uint4(packed[0], packed[1], packed[2], packed[3]);
    yp[1] = make_uint4(packed[4], packed[5], packed[6], packed[7]);
}

// Fault-free epilogue of 16 channels k0 .. k0 + 15 of one pixel: the same
// FP32 operations in the same order as store_chunk_pre without a fault
// ((accumulator + bias) + residual, then ReLU), with the bias read as four
// 16-byte vectors and ReLU and the FP16 rounding (nearest even) fused into
// one conversion per channel pair (negative values become +0, NaN stays NaN).
struct Bias16 {
    float4 q[4];
};
__device__ __forceinline__ Bias16 load_bias16(const float *bias, int k0) {
    const float4 *p = reinterpret_cast<const float4 *>(bias + k0);
    Bias16 b;
#pragma unroll
    for (int i = 0; i < 4; ++i) b.q[i] = __ldg(p + i);
    return b;
}
// Bias of the conv kernels' epilogue: a copy in shared memory (up to
// BIAS_SMEM output channels), filled once per CTA, so that the per-chunk
// bias read costs no global-memory round trip; else the global array.
constexpr int BIAS_SMEM = 1024;
__device__ __forceinline__ Bias16 bias16_at(const float *bias_s, const float *bias_g, bool in_smem, int k0) {
    if (in_smem) {
        const float4 *p = reinterpret_cast<const float4 *>(bias_s + k0);
        Bias16 b;
#pragma unroll
        for (int i = 0; i < 4; ++i) b.q[i] = p[i];
        return b;
    }
    return load_bias16(bias_g, k0);
}
// Copy of the bias into shared memory by the epilogue warps (named barrier 1
// over those warps only).  Returns whether the copy was made.
__device__ __forceinline__ bool stage_bias(float *bias_s, const float *bias_g, int K, int t, int nthreads) {
    const bool in_smem = bias_g != nullptr && K <= BIAS_SMEM;
    if (in_smem) {
        for (int i = t; i < K; i += nthreads) bias_s[i] = __ldg(bias_g + i);
        asm volatile("bar.sync 1, %0;" ::"r"(nthreads) : "memory");
    }
    return in_smem;
}
// stage_bias for a launch that also runs a shortcut convolution: the
// shortcut's bias follows this layer's (bias_s[K .. 2K)).
__device__ __forceinline__ bool stage_bias2(float *bias_s, const float *b1, const float *b2, int K, int t,
                                            int nthreads) {
    const bool in_smem = b1 != nullptr && b2 != nullptr && 2 * K <= BIAS_SMEM;
    if (in_smem) {
        for (int i = t; i < K; i += nthreads) {
            bias_s[i] = __ldg(b1 + i);
            bias_s[K + i] = __ldg(b2 + i);
        }
        asm volatile("bar.sync 1, %0;" ::"r"(nthreads) : "memory");
    }
    return in_smem;
}
__device__ __forceinline__ uint32_t cvt_h2(float lo, float hi, bool relu) {
    uint32_t r;
    if (relu) asm("cvt.rn.relu.f16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
    else asm("cvt.rn.f16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
    return r;
}
__device__ __forceinline__ void store16_fast(const float *v, const Bias16 &b, const Res16 &r, bool res, bool relu,
                                             __half *dst) {
    const float *bb = reinterpret_cast<const float *>(b.q);
    float t[16];
#pragma unroll
    for (int i = 0; i < 16; ++i) t[i] = v[i] + bb[i];
    if (res) {
        const __half2 *h0 = reinterpret_cast<const __half2 *>(&r.r0);
        const __half2 *h1 = reinterpret_cast<const __half2 *>(&r.r1);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float2 f0 = __half22float2(h0[i]), f1 = __half22float2(h1[i]);
            t[2 * i] += f0.x; t[2 * i + 1] += f0.y; t[8 + 2 * i] += f1.x; t[8 + 2 * i + 1] += f1.y;
        }
    }
    uint32_t pk[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) pk[i] = cvt_h2(t[2 * i], t[2 * i + 1], relu);
    st_global_v8(dst, pk);          // 16 channels of one pixel: 32-byte aligned
}

// store16_fast without a residual, into registers: FP16 pairs of
// (accumulator + bias), ReLU fused into the rounding (the same bits).
__device__ __forceinline__ void pack16(const float *v, const Bias16 &b, bool relu, uint32_t (&pk)[8]) {
    const float *bb = reinterpret_cast<const float *>(b.q);
#pragma unroll
    for (int i = 0; i < 8; ++i) pk[i] = cvt_h2(v[2 * i] + bb[2 * i], v[2 * i + 1] + bb[2 * i + 1], relu);
}
// 4 x 4 transpose of 32-byte pieces among the lanes 4a .. 4a + 3 of a warp
// (i = lane & 3): on entry pk[p] is piece p (channels 16p .. 16p + 15) of
// this lane's pixel, on exit pk[k] is piece i of the pixel of lane 4a + k.
// Two butterfly rounds of shuffles; then a warp's store of pk[k] writes
// eight pixels' 64 channels, eight whole 128-byte lines, where a store of
// each lane's own piece touches 32 lines.
__device__ __forceinline__ void transpose4_pieces(uint32_t (&pk)[4][8], int i) {
#pragma unroll
    for (int mk = 1; mk <= 2; mk <<= 1) {
        const bool up = (i & mk) != 0;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            if (q & mk) continue;
#pragma unroll
            for (int r = 0; r < 8; ++r) {
                const uint32_t send = up ? pk[q][r] : pk[q + mk][r];
                const uint32_t recv = __shfl_xor_sync(0xffffffffu, send, mk);
                if (up) pk[q][r] = recv;
                else pk[q + mk][r] = recv;
            }
        }
    }
}

// Epilogue values of 16 channels k0 .. k0 + 15 of one pixel in FP32, in the
// order of store_chunk_pre: accumulator + bias, fault delta, residual, ReLU.
__device__ __forceinline__ void epi16_vals(const float *v, const Bias16 &b, const Res16 &r, bool res, bool relu,
                                           const FaultDelta &fd, int k0, float fsrc, float *t) {
    const float *bb = reinterpret_cast<const float *>(b.q);
    float rv[16];
    {
        const __half2 *h0 = reinterpret_cast<const __half2 *>(&r.r0);
        const __half2 *h1 = reinterpret_cast<const __half2 *>(&r.r1);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float2 f0 = __half22float2(h0[i]), f1 = __half22float2(h1[i]);
            rv[2 * i] = f0.x; rv[2 * i + 1] = f0.y; rv[8 + 2 * i] = f1.x; rv[8 + 2 * i + 1] = f1.y;
        }
    }
#pragma unroll
    for (int i = 0; i < 16; ++i) {
        float x = v[i] + bb[i];
        if (fd.active && fd.kout == k0 + i) x += fd.dv * fsrc;
        if (res) x += rv[i];
        if (relu) x = relu_keep_nan(x);
        t[i] = x;
    }
}

// Maximum over the 2 x 2 window of a halo tile's epilogue lanes: a warp holds
// four tile rows of 8 pixels, lane = 8 * row + column, so the window's other
// pixels are lanes l ^ 1 and l ^ 8.  NaN wins (a window with a NaN is NaN).
__device__ __forceinline__ float fmax_nan(float a, float b) {
    float r;
    asm("max.NaN.f32 %0, %1, %2;" : "=f"(r) : "f"(a), "f"(b));
    return r;
}
__device__ __forceinline__ float pool2x2_lanes(float v) {
    v = fmax_nan(v, __shfl_xor_sync(0xffffffffu, v, 1));
    return fmax_nan(v, __shfl_xor_sync(0xffffffffu, v, 8));
}

// The checksum output of one pixel: carry-through column + coef * incoming
// checksum (centre pixel, or the sum of an FC layer's checksum features),
// fault delta, residual checksum, ReLU.
// Inputs of a checksum output other than the carry-through column: the
// incoming checksum at the centre pixel (or the sum of an FC layer's
// checksum features) and the residual checksum.  Loaded before the
// accumulator is ready so that their latency overlaps the MMAs.
// The centre-pixel and residual checksums are kept as FP16 bits and
// converted where they are used, so that their loads stay in flight while
// the epilogue waits for the accumulator (a conversion right after the load
// would stall the warp on it).
struct CsIn {
    float cin_sum;                 // FC layer: the sum of its incoming checksum features
    unsigned short cin_h, rcs_h;   // FP16 bits of the incoming and residual checksums (0: +0)
};
__device__ __forceinline__ float h2f_bits(unsigned short b) { return __half2float(__ushort_as_half(b)); }
__device__ __forceinline__ CsIn load_cs_inputs(const ConvArgs &a, const TcGeom &g, int m, int nimg, int p, int q) {
    CsIn c{0.f, 0, 0};
    const __half *csi = static_cast<const __half *>(a.cs_in);
    const int ctr_r = g.ctr_tap / g.S, ctr_s = g.ctr_tap % g.S;
    const int hc = p * g.stride + ctr_r - g.pad, wc = q * g.stride + ctr_s - g.pad;
    const bool inb = hc >= 0 && hc < a.H && wc >= 0 && wc < a.W;
    if (csi && a.cs_rowsum > 0) {                  // FC layer: every incoming checksum feature
        for (int i = 0; i < a.cs_rowsum; ++i) c.cin_sum += ldh(csi, (size_t)m * a.cs_rowsum + i);
    } else if (csi && inb) {
        c.cin_h = __ldg(reinterpret_cast<const unsigned short *>(csi) + ((size_t)nimg * a.H + hc) * a.W + wc);
    }
    if (a.res_cs) c.rcs_h = __ldg(static_cast<const unsigned short *>(a.res_cs) + m);
    return c;
}

__device__ __forceinline__ float checksum_value(float ctv, const CsIn &c, const ConvArgs &a, const TcGeom &g,
                                                float fsrc) {
    const float cin = a.cs_rowsum > 0 ? c.cin_sum : h2f_bits(c.cin_h);
    float o = 0.f;
    if (a.role == CT_ROLE_CT) o = ctv + a.coef * cin;
    else if (a.role == CT_ROLE_PASS) o = cin;
    if (a.fd.active && a.fd.kout == g.K) o += a.fd.dv * fsrc;
    if (a.res_cs) o += h2f_bits(c.rcs_h);
    if (a.relu) o = relu_keep_nan(o);
    return o;
}

__device__ __forceinline__ void store_checksum_pre(float ctv, const CsIn &c, const ConvArgs &a, const TcGeom &g,
                                                   int m, float fsrc) {
    static_cast<__half *>(a.cs_out)[m] = __float2half_rn(checksum_value(ctv, c, a, g, fsrc));
}


// K-block kb accumulates into chain kb % NCH: back-to-back MMAs into one
// TMEM accumulator serialise on it, so NCH independent chains keep the
// tensor pipe busy when one 128 x BN x 16 MMA is short (BN = 64).  The
// epilogue adds the chains.  SUB K-blocks share one pipeline stage (one
// barrier round trip).  When two buffers of the chains fit in TMEM (NACC),
// tiles alternate between them; for BN <= 128 the epilogue also copies its
// buffer to registers and releases it before its global stores.
// SC: the launch also runs a 1x1 shortcut convolution (bmap2, a2, g2; see
// UnitSeq); otherwise those arguments are unused.
template <int BN, int STAGES, int SUB, int NCH, bool SC>
__global__ void __launch_bounds__(tc_threads(BN, STAGES), 1)
conv_tc_kernel(const __grid_constant__ CUtensorMap amap, const __grid_constant__ CUtensorMap bmap,
               const __grid_constant__ ConvArgs a, const __grid_constant__ TcGeom g,
               const __grid_constant__ CUtensorMap bmap2, const __grid_constant__ ConvArgs a2,
               const __grid_constant__ TcGeom g2) {
    constexpr int B_ROWS = BN + 16;                       // 16 constant carry-through rows
    constexpr int B_SUB_BYTES = B_ROWS * BK * 2;
    constexpr int B_TMA_BYTES = BN * BK * 2;
    constexpr int CH = BN + 16;                           // TMEM columns per chain
    constexpr bool EARLY = BN <= 128;                     // release TMEM before the stores
    // N = 256: two 256-column accumulators fill TMEM, so the carry-through
    // column is summed (warp-level MMAs against a ones vector) from the
    // centre-tap A tiles in shared memory by the warps of the producer group
    // that do not issue copies (they consume every stage, like the MMA warp),
    // and the epilogue of one tile overlaps the MMAs of the next
    constexpr bool DBUF = !EARLY;
    // accumulator buffers, 256 TMEM columns apart: two when both fit (N =
    // 256; N <= 128 with one chain), so that a tile's MMAs never wait for
    // the previous tile's epilogue to read TMEM
    constexpr int NACC = (DBUF || 2 * NCH * CH <= 512) ? 2 : 1;
    static_assert(NACC == 1 || DBUF || NCH * CH <= 256, "an accumulator buffer spans at most 256 columns");
    // producer warps (each owns whole ring slots) and carry-through warps
    constexpr int NPROD = tc_nprod(BN, STAGES);
    constexpr int NPG = tc_npg(BN, STAGES);               // producer group: producers + carry-through warps
    constexpr int NCT = DBUF ? NPG - NPROD : 0;
    constexpr int TC_MMA_WARP = NPG;
    constexpr int TC_EPI_WARP0 = NPG + 1;
    static_assert(STAGES % NPROD == 0, "producer warps must own whole ring slots");
    static_assert(DBUF ? NCT > 0 : NCT == 0, "carry-through warps only beside double-buffered accumulators");
    static_assert(!DBUF || (NCT > 0 && BM % (16 * (NCT > 0 ? NCT : 1)) == 0), "carry-through warps split the tile rows");
    static_assert(!SC || !DBUF, "a shortcut only beside single-buffered accumulators");
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint8_t *As = smem;                                   // [STAGES][SUB][A_BYTES]
    uint8_t *Bs = As + STAGES * SUB * A_BYTES;            // [STAGES][SUB][B_SUB_BYTES]
    uint8_t *CTt = Bs + STAGES * SUB * B_SUB_BYTES;       // separate 16-row carry-through tile
    float *ct_sum = (float *)(CTt + 16 * BK * 2);          // [2][BM] carry-through sums (DBUF)
    uint64_t *full = (uint64_t *)(ct_sum + 2 * BM);
    uint64_t *empty = full + STAGES;
    uint64_t *acc_full = empty + STAGES;                  // [2]
    uint64_t *acc_empty = acc_full + 2;                   // [2]
    uint64_t *ct_ready = acc_empty + 2;                   // [2]
    uint32_t *tmem_holder = (uint32_t *)(ct_ready + 2);
    volatile uint32_t *abort_flag = tmem_holder + 1;
    float *bias_s = (float *)(((uintptr_t)(tmem_holder + 2) + 15) & ~(uintptr_t)15);   // [BIAS_SMEM]

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int cid = blockIdx.x, ncl = gridDim.x;
    const int n1 = g.m_tiles * g.n_tiles * g.splits;     // this layer's items
    const UnitSeq us = unit_seq<SC>(cid, ncl, n1, g);
    const int n_units = us.k1 + us.cnt;                 // this CTA's units

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(smem_u32(&full[s]), 1);
            mbar_init(smem_u32(&empty[s]), 1 + NCT);   // MMA commit + carry-through warps
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(smem_u32(&acc_full[b]), 1);
            mbar_init(smem_u32(&acc_empty[b]), N_EPI_WARPS);
            mbar_init(smem_u32(&ct_ready[b]), NCT > 0 ? NCT : 1);
        }
        *abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == TC_MMA_WARP) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_holder)),
                     "r"((uint32_t)g.tmem_cols));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    if (warp >= TC_EPI_WARP0) {
        // constant carry-through rows: row 0 = coef, rows 1..15 = 0 (swizzle-invariant)
        const uint32_t coef2 = (uint32_t)g.coef_h | ((uint32_t)g.coef_h << 16);
        const int t = threadIdx.x - 32 * TC_EPI_WARP0;
        for (int sb = 0; sb < STAGES * SUB; ++sb) {
            uint32_t *rows = (uint32_t *)(Bs + sb * B_SUB_BYTES + BN * BK * 2);
            for (int i = t; i < 16 * BK / 2; i += 32 * N_EPI_WARPS) rows[i] = (i < BK / 2) ? coef2 : 0u;
        }
        uint32_t *ctt = (uint32_t *)CTt;
        for (int i = t; i < 16 * BK / 2; i += 32 * N_EPI_WARPS) ctt[i] = (i < BK / 2) ? coef2 : 0u;
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tmem = *tmem_holder;
    // the previous kernel's outputs (and any fault flip) are visible from here
    pdl_wait();
    pdl_trigger();

    if (warp < NPROD) {
        // ---------------- TMA producers ----------------
        // One lane of one thread issues TMA copies one after another, so the
        // ring slots are dealt to NPROD producer warps whose copies proceed
        // in parallel.  Slot s always belongs to warp s % NPROD (NPROD
        // divides STAGES): every slot is refilled by one warp in order, so a
        // parity wait on its empty barrier can never see a phase two ahead.
        if (elect_one()) {
            asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&amap) : "memory");
            asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&bmap) : "memory");
            if (SC) asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&bmap2) : "memory");
        }
        __syncwarp();
        int it = 0;
        for (int k = 0; k < n_units; ++k) {
            if (__any_sync(0xffffffffu, *abort_flag)) break;
            const int unit = unit_at(us, k, cid, ncl);
            const bool sc = SC && unit >= n1;
            // A coordinates: this layer's geometry (a shortcut reads its centre tap)
            const TileRef tr = sc ? tile_ref(unit - n1, g2) : tile_ref(unit, g);
            const CUtensorMap *bm = sc ? &bmap2 : &bmap;
            const int m0 = tr.m0, n_tile = tr.n_tile;
            const int nimg = m0 / g.PQ, rem = m0 % g.PQ;
            const int p = rem / g.Q, q = rem % g.Q;
            const int w0 = q * g.stride - g.pad, h0 = p * g.stride - g.pad;
            bool ok = true;
            for (int kb0 = tr.kb_lo; kb0 < tr.kb_hi; kb0 += SUB, ++it) {
                const int s = it % STAGES;
                if (s % NPROD != warp) continue;
                const uint32_t ph = (uint32_t)(it / STAGES) & 1u;
                if (!warp_wait(smem_u32(&empty[s]), ph ^ 1u, a.err, 1u)) { ok = false; break; }
                const int nsub = min(SUB, tr.kb_hi - kb0);
                const uint32_t fb = smem_u32(&full[s]);
                if (elect_one()) {
                    mbar_arrive_expect_tx(fb, nsub * (A_BYTES + B_TMA_BYTES));
                    for (int j = 0; j < nsub; ++j) {
                        const int kb = kb0 + j;
                        const int tap = tap_of(kb / g.cpb, g.ctr_tap);
                        const int c0 = (kb % g.cpb) * BK;
                        const int r = tap / g.S, sx = tap % g.S;
                        tma_load_im2col(smem_u32(As + (s * SUB + j) * A_BYTES), &amap, fb, c0, w0, h0, nimg,
                                        (uint16_t)sx, (uint16_t)r);
                        tma_load_2d(smem_u32(Bs + (s * SUB + j) * B_SUB_BYTES), bm, fb, (sc ? 0 : tap) * g.C + c0,
                                    n_tile * BN);
                    }
                }
                __syncwarp();
            }
            if (!ok) { if (lane == 0) *abort_flag = 1; break; }
        }
    } else if (warp == TC_MMA_WARP) {
        // ---------------- MMA issuer (whole warp, one lane issues) ----------------
        const uint32_t id_main = idesc_f16(BM, BN);
        const uint32_t id_merged = idesc_f16(BM, BN + 16);
        const uint32_t id_ct = idesc_f16(BM, 16);
        const uint32_t ct_base = smem_u32(CTt);
        int it = 0;
        for (int lt = 0; lt < n_units; ++lt) {
            if (__any_sync(0xffffffffu, *abort_flag)) break;
            const int unit = unit_at(us, lt, cid, ncl);
            const bool sc = SC && unit >= n1;
            const TcGeom &G = sc ? g2 : g;
            const TileRef tr = tile_ref(sc ? unit - n1 : unit, G);
            const int n_tile = tr.n_tile;
            const bool ct_here = G.ct_mode != CT_NONE_ && n_tile == 0;
            const int ab = NACC == 2 ? (lt & 1) : 0;
            const uint32_t aph = NACC == 2 ? ((uint32_t)(lt >> 1) & 1u) : ((uint32_t)lt & 1u);
            if (!warp_wait(smem_u32(&acc_empty[ab]), aph ^ 1u, a.err, 8u)) {
                if (lane == 0) *abort_flag = 1;
                break;
            }
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            bool ok = true;
            for (int kb0 = tr.kb_lo; kb0 < tr.kb_hi; kb0 += SUB, ++it) {
                const int s = it % STAGES;
                const uint32_t ph = (uint32_t)(it / STAGES) & 1u;
                if (!warp_wait(smem_u32(&full[s]), ph, a.err, 2u)) { ok = false; break; }
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                const int nsub = min(SUB, tr.kb_hi - kb0);
                if (elect_one()) {
                    // descriptors advance 32 bytes (2 in the 16-byte address field)
                    // per 16-element K step; the instruction choice is per K block
                    for (int j = 0; j < nsub; ++j) {
                        const int kb = kb0 + j;
                        const int kr = kb - tr.kb_lo;               // position within this split
                        const uint32_t d = tmem + (uint32_t)(ab * 256 + (kr % NCH) * CH);
                        const bool centre = kb < G.cpb;
                        const uint64_t ad0 = smem_desc_sw128(smem_u32(As + (s * SUB + j) * A_BYTES));
                        const uint64_t bd0 = smem_desc_sw128(smem_u32(Bs + (s * SUB + j) * B_SUB_BYTES));
                        const uint32_t acc0 = kr >= NCH ? 1u : 0u;  // first use of the chain
                        if (!DBUF && ct_here && centre && G.ct_mode == CT_SEPARATE) {
                            const uint64_t cd0 = smem_desc_sw128(ct_base);
#pragma unroll
                            for (int k16 = 0; k16 < BK / 16; ++k16) {
                                umma_f16(d, ad0 + 2 * k16, bd0 + 2 * k16, id_main, k16 ? 1u : acc0);
                                umma_f16(d + BN, ad0 + 2 * k16, cd0 + 2 * k16, id_ct, k16 ? 1u : acc0);
                            }
                        } else {
                            const uint32_t idm = (!DBUF && ct_here && centre && G.ct_mode == CT_MERGED) ? id_merged : id_main;
#pragma unroll
                            for (int k16 = 0; k16 < BK / 16; ++k16)
                                umma_f16(d, ad0 + 2 * k16, bd0 + 2 * k16, idm, k16 ? 1u : acc0);
                        }
                    }
                }
                __syncwarp();
                if (elect_one()) umma_commit(smem_u32(&empty[s]));
                __syncwarp();
            }
            if (!ok) { if (lane == 0) *abort_flag = 1; break; }
            if (elect_one()) umma_commit(smem_u32(&acc_full[ab]));   // fires when the tile's MMAs have completed
            __syncwarp();
        }
    } else if (warp < NPG) {
        if (NCT > 0) {
            // ---------------- carry-through sums (N = 256) ----------------
            // Consumes every stage in order (arrives on its empty barrier);
            // on the centre-tap K blocks of the first N tile it adds each A
            // row's 64 channels.  The row sums run on the warp-level MMA
            // against a B of ones (FP32 accumulation, like the tcgen05
            // column of the other kernels): per K block and 64-row share,
            // 16 ldmatrix + 16 MMAs.  Rows are read through the 128-byte
            // swizzle (chunk c of row r sits at chunk c ^ (r & 7)), so the
            // eight rows of one 8x8 matrix hit eight different bank groups.
            constexpr int ROWS_W = BM / (NCT > 0 ? NCT : 1);       // rows per carry-through warp
            constexpr int MT = ROWS_W / 16;                          // 16-row MMA tiles per warp
            const float coef = __half2float(__ushort_as_half(g.coef_h));
            const int w = warp - NPROD;
            // ldmatrix row address of this lane: matrix lane / 8 = (rows +8, chunk +1) bits
            const int lm_row = (lane & 7) + ((lane >> 3) & 1) * 8, lm_chk = lane >> 4;
            int it = 0;
            bool ok = true;
            for (int lt = 0; lt < n_units && ok; ++lt) {
                if (__any_sync(0xffffffffu, *abort_flag)) break;
                const TileRef tr = tile_ref(unit_at(us, lt, cid, ncl), g);
                const bool ct_here = g.ct_mode != CT_NONE_ && tr.n_tile == 0;
                const int ab = lt & 1;
                float acc[MT][4];
#pragma unroll
                for (int m = 0; m < MT; ++m)
#pragma unroll
                    for (int e = 0; e < 4; ++e) acc[m][e] = 0.f;
                for (int kb0 = tr.kb_lo; kb0 < tr.kb_hi; kb0 += SUB, ++it) {
                    const int s = it % STAGES;
                    if (!warp_wait(smem_u32(&full[s]), (uint32_t)(it / STAGES) & 1u, a.err, 2u)) { ok = false; break; }
                    const int nsub = min(SUB, tr.kb_hi - kb0);
                    for (int j = 0; j < nsub; ++j) {
                        if (!(ct_here && kb0 + j < g.cpb)) continue;
                        const uint32_t tbase = smem_u32(As + (s * SUB + j) * A_BYTES);
#pragma unroll
                        for (int m = 0; m < MT; ++m) {
                            const int row = w * ROWS_W + m * 16 + lm_row;
                            const uint32_t rbase = tbase + (uint32_t)row * 128u;
#pragma unroll
                            for (int t = 0; t < 4; ++t) {
                                const uint32_t chk = (uint32_t)((2 * t + lm_chk) ^ (row & 7));
                                uint32_t a0, a1, a2, a3;
                                ldsm_x4(rbase + chk * 16u, a0, a1, a2, a3);
                                mma_rowsum_16x16(acc[m], a0, a1, a2, a3);
                            }
                        }
                    }
                    __syncwarp();
                    if (lane == 0) mbar_arrive(smem_u32(&empty[s]));
                }
                if (!ok) break;
                // ct_sum[ab] is free once the epilogue released accumulator ab
                if (!warp_wait(smem_u32(&acc_empty[ab]), ((uint32_t)(lt >> 1) & 1u) ^ 1u, a.err, 8u)) { ok = false; break; }
                // D fragment: lane l holds rows l / 4 (acc[m][0]) and l / 4 + 8 (acc[m][2]) of tile m
                if ((lane & 3) == 0) {
#pragma unroll
                    for (int m = 0; m < MT; ++m) {
                        const int r0 = w * ROWS_W + m * 16 + (lane >> 2);
                        ct_sum[ab * BM + r0] = coef * acc[m][0];
                        ct_sum[ab * BM + r0 + 8] = coef * acc[m][2];
                    }
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(&ct_ready[ab]));
            }
            if (!ok && lane == 0) *abort_flag = 1;
        }
    } else if (warp >= TC_EPI_WARP0) {
        // ---------------- epilogue: 8 warps ----------------
        // (producer warps beyond NPROD have no role)
        const int ep = warp - TC_EPI_WARP0;
        const int quad = warp & 3;                 // TMEM lanes this warp may read
        const int half = ep >> 2;                  // which half of the tile's channels
        const int row = quad * 32 + lane;
        const int et = threadIdx.x - 32 * TC_EPI_WARP0;
        const bool bias_sm = SC ? stage_bias2(bias_s, a.bias, a2.bias, g.K, et, 32 * N_EPI_WARPS)
                                : stage_bias(bias_s, a.bias, g.K, et, 32 * N_EPI_WARPS);
        for (int lt = 0; lt < n_units; ++lt) {
            const int unit = unit_at(us, lt, cid, ncl);
            const bool sc = SC && unit >= n1;
            const ConvArgs &A = sc ? a2 : a;       // this unit's layer
            const TcGeom &G = sc ? g2 : g;
            const float *bias_l = bias_s + (sc ? G.K : 0);
            const __half *x = static_cast<const __half *>(A.x);
            const FaultDelta fd = A.fd;
            const bool split = G.splits > 1;
            const bool has_res = A.res != nullptr, relu = A.relu != 0;
            const TileRef tr = tile_ref(sc ? unit - n1 : unit, G);
            const int m0 = tr.m0, n_tile = tr.n_tile;
            // residual loads in flight while the MMAs run
            Res16 rs[BN / 32];
            {
                const int mp = m0 + row;
#pragma unroll
                for (int c = 0; c < BN / 32; ++c)
                    rs[c] = (mp < G.M && G.splits == 1)
                                ? load_res16(A, G.K, (size_t)mp, n_tile * BN + half * (BN / 2) + 16 * c)
                                : Res16{make_uint4(0u, 0u, 0u, 0u), make_uint4(0u, 0u, 0u, 0u)};
            }
            CsIn csv{0.f, 0, 0};
            {
                const int mp = m0 + row;
                if (half == 0 && A.cs_out != nullptr && n_tile == 0 && mp < G.M && G.splits == 1) {
                    const int ni = mp / G.PQ, rm = mp % G.PQ;
                    csv = load_cs_inputs(A, G, mp, ni, rm / G.Q, rm % G.Q);
                }
            }
            const int chains = min(NCH, tr.kb_hi - tr.kb_lo);                    // chains that received MMAs
            // chains whose first K block is a centre block hold a carry-through column
            const int ct_chains = max(0, min(NCH, min(G.cpb, tr.kb_hi) - tr.kb_lo));
            const int ab = NACC == 2 ? (lt & 1) : 0;
            const uint32_t aph = NACC == 2 ? ((uint32_t)(lt >> 1) & 1u) : ((uint32_t)lt & 1u);
            bool ok = mbar_wait(smem_u32(&acc_full[ab]), aph, A.err, 4u) && !*abort_flag;
            if (DBUF) ok = ok && mbar_wait(smem_u32(&ct_ready[ab]), aph, A.err, 4u);
            ok = __all_sync(0xffffffffu, ok);      // tcgen05.ld below is warp-collective
            if (!ok) break;
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            const uint32_t trow = tmem + (uint32_t)(ab * 256) + ((uint32_t)(quad * 32) << 16);
            const int m = m0 + row;
            const bool valid = m < G.M;
            const int mm = valid ? m : 0;
            const int nimg = mm / G.PQ, rem = mm % G.PQ, p = rem / G.Q, q = rem % G.Q;
            float fsrc = 0.f;
            if (fd.active && !split) {
                const int h = p * G.stride + fd.r - G.pad, w = q * G.stride + fd.s - G.pad;
                if (h >= 0 && h < A.H && w >= 0 && w < A.W) {
                    if (fd.cin < G.C) fsrc = ldh(x, (((size_t)nimg * A.H + h) * A.W + w) * G.C + fd.cin);
                    else if (A.cs_in) fsrc = ldh(static_cast<const __half *>(A.cs_in), ((size_t)nimg * A.H + h) * A.W + w);
                }
            }
            const int n0 = n_tile * BN;
            const bool do_cs = half == 0 && A.cs_out != nullptr && n_tile == 0;
            float ctv = 0.f;
            if (EARLY) {
                // TMEM reads in few round trips: chain 0 (all of this warp's
                // columns) with the carry-through columns, then the other
                // chains two chunks at a time; the sums keep the order
                // ((chain 0 + chain 1) + chain 2) + ...
                float vals[BN / 2];
                const bool ld_ct = do_cs && G.ct_mode != CT_NONE_;
                uint32_t ctr[NCH];
                {
                    uint32_t tv[BN / 32][16];
#pragma unroll
                    for (int c = 0; c < BN / 2; c += 16) tmem_ld16_nw(trow + half * (BN / 2) + c, tv[c / 16]);
#pragma unroll
                    for (int ch = 0; ch < NCH; ++ch)
                        if (ld_ct && ch < ct_chains) tmem_ld1_nw(trow + ch * CH + BN, ctr[ch]);
                    tmem_wait_ld();
#pragma unroll
                    for (int c = 0; c < BN / 2; c += 16) tmem_done16(tv[c / 16], vals + c);
                }
                for (int ch = 1; ch < chains; ++ch) {
#pragma unroll
                    for (int c = 0; c < BN / 2; c += 32) {
                        uint32_t t2[2][16];
                        tmem_ld16_nw(trow + ch * CH + half * (BN / 2) + c, t2[0]);
                        tmem_ld16_nw(trow + ch * CH + half * (BN / 2) + c + 16, t2[1]);
                        tmem_wait_ld();
                        float t[16];
                        tmem_done16(t2[0], t);
#pragma unroll
                        for (int i = 0; i < 16; ++i) vals[c + i] += t[i];
                        tmem_done16(t2[1], t);
#pragma unroll
                        for (int i = 0; i < 16; ++i) vals[c + 16 + i] += t[i];
                    }
                }
#pragma unroll
                for (int ch = 0; ch < NCH; ++ch)
                    if (ld_ct && ch < ct_chains) ctv += tmem_done(ctr[ch]);
                asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(&acc_empty[ab]));   // accumulators free for a later tile
                if (valid && split) {
                    float *wrow = A.ws + ((size_t)tr.sp * G.M + m) * G.ws_ld;
#pragma unroll
                    for (int c = 0; c < BN / 2; c += 4)
                        *reinterpret_cast<float4 *>(wrow + n0 + half * (BN / 2) + c) =
                            make_float4(vals[c], vals[c + 1], vals[c + 2], vals[c + 3]);
                    if (do_cs) wrow[G.K] = ctv;
                } else if (valid && fd.active) {
#pragma unroll
                    for (int c = 0; c < BN / 2; c += 16)
                        store_chunk_pre(vals + c, rs[c / 16], A, G.K, (size_t)m, n0 + half * (BN / 2) + c, fsrc);
                    if (do_cs) store_checksum_pre(ctv, csv, A, G, m, fsrc);
                } else if (BN == 128 && !split && !fd.active && !has_res) {
                    // whole lines: the lanes of each group of four swap their
                    // 16-channel pieces (all lanes take part; stores of pixels
                    // past M are skipped)
                    uint32_t pk[4][8];
#pragma unroll
                    for (int c = 0; c < 4; ++c)
                        pack16(vals + 16 * c, bias16_at(bias_l, A.bias, bias_sm, n0 + half * (BN / 2) + 16 * c), relu,
                               pk[c]);
                    transpose4_pieces(pk, lane & 3);
#pragma unroll
                    for (int k = 0; k < 4; ++k) {
                        const int mk = m0 + quad * 32 + (lane & ~3) + k;
                        if (mk < G.M)
                            st_global_v8(static_cast<__half *>(A.y) + (size_t)mk * G.K + n0 + half * (BN / 2) +
                                             16 * (lane & 3), pk[k]);
                    }
                    if (do_cs && valid) store_checksum_pre(ctv, csv, A, G, m, 0.f);
                } else if (valid) {
                    __half *yrow = static_cast<__half *>(A.y) + (size_t)m * G.K + n0 + half * (BN / 2);
#pragma unroll
                    for (int c = 0; c < BN / 2; c += 16)
                        store16_fast(vals + c, bias16_at(bias_l, A.bias, bias_sm, n0 + half * (BN / 2) + c), rs[c / 16], has_res,
                                     relu, yrow + c);
                    if (do_cs) store_checksum_pre(ctv, csv, A, G, m, 0.f);
                }
            } else {
#pragma unroll
                for (int c = half * (BN / 2); c < (half + 1) * (BN / 2); c += 16) {
                    float v[16];
                    tmem_ld16(trow + c, v);
                    for (int ch = 1; ch < chains; ++ch) {
                        float t[16];
                        tmem_ld16(trow + ch * CH + c, t);
#pragma unroll
                        for (int i = 0; i < 16; ++i) v[i] += t[i];
                    }
                    if (valid && split) {
                        float4 *wp = reinterpret_cast<float4 *>(A.ws + ((size_t)tr.sp * G.M + m) * G.ws_ld + n0 + c);
#pragma unroll
                        for (int i = 0; i < 4; ++i) wp[i] = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
                    } else if (valid && fd.active) {
                        store_chunk_pre(v, rs[(c - half * (BN / 2)) / 16], A, G.K, (size_t)m, n0 + c, fsrc);
                    } else if (valid) {
                        store16_fast(v, bias16_at(bias_l, A.bias, bias_sm, n0 + c), rs[(c - half * (BN / 2)) / 16], has_res,
                                     relu, static_cast<__half *>(A.y) + (size_t)m * G.K + n0 + c);
                    }
                }
                if (do_cs && G.ct_mode != CT_NONE_) ctv = ct_sum[ab * BM + row];
                if (do_cs && valid && split) A.ws[((size_t)tr.sp * G.M + m) * G.ws_ld + G.K] = ctv;
                else if (do_cs && valid) store_checksum_pre(ctv, csv, A, G, m, fsrc);
                asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(&acc_empty[ab]));
            }
        }
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (warp == TC_MMA_WARP) {
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"((uint32_t)g.tmem_cols));
    }
}

// ---------------------------------------------------------------------------
// N = 256 over CTA pairs (tcgen05 cta_group::2).  A cluster of two CTAs
// computes a 256-pixel x 256-channel tile: each CTA copies its own 128 A rows
// and its half (128 rows) of the tile's weights; the even CTA issues M = 256
// MMAs that read both CTAs' shared memory and leave each CTA's 128 rows of D
// in its own TMEM.  Per SM and 128 x 256 x 16 step the shared memory then
// takes 8 KB of copies and 8 KB of MMA reads instead of 12 + 12, the bound
// of the single-CTA N = 256 tiles.
//
// The carry-through column at the centre tap is coef * the channel sum of
// one input pixel, so each epilogue thread adds it up from the input tensor
// (rows of C FP16 values, just copied through L2) with FP32 accumulation;
// the stage pipeline carries only the GEMM.  Hand-over (all waits bounded):
//   full[s]        even CTA: stage s landed in both CTAs (one expect_tx
//                  arrival + the bytes of both CTAs' copies)
//   empty[s]       each CTA: the pair's MMAs on stage s completed (commit
//                  multicast): the stage may be refilled
//   acc_full[b]    each CTA: accumulator b complete (commit multicast)
//   pair_empty[b]  even CTA: both epilogues have read accumulator b
//   mma_done       each CTA: every MMA of the pair completed (before dealloc)
//
// Last-round balance (conv_tc_pair_kernel<true>).  When the last round of
// tiles would leave more than half the pairs idle, each tile of that round
// runs as two units of 128 channels (M = 256, N = 128 MMAs: each CTA copies
// 64 weight rows), on different pairs and before the whole tiles.  Every
// output is still one full-K accumulation, so the result does not depend on
// the split.
constexpr int PR_STAGES = 6;
constexpr int PR_NPROD = 3;
constexpr int PR_MMA_WARP = PR_NPROD;
constexpr int PR_EPI_WARP0 = PR_MMA_WARP + 1;
constexpr int PR_THREADS = 32 * (PR_EPI_WARP0 + N_EPI_WARPS);
constexpr int PR_BH_BYTES = BM * BK * 2;                  // this CTA's 128 weight rows of a stage
constexpr int PR_NBAR = 2 * PR_STAGES + 5;                // full, empty per stage; acc_full, pair_empty, mma_done

// Work unit u of a pair kernel: its tile (256 pixels x 256 channels), first
// output channel, and whether it is a 128-channel half (else all 256).
struct PairUnit {
    int item, nb;
    bool narrow;
};
template <bool VARN>
__device__ __forceinline__ PairUnit pair_unit(int u, const TcGeom &g) {
    if (!VARN) return PairUnit{u, (u % g.n_tiles) * 256, false};
    const int n_h = g.units - g.t_first;
    if (u >= n_h) {
        const int it = u - n_h;
        return PairUnit{it, (it % g.n_tiles) * 256, false};
    }
    const int it = g.t_first + (u >> 1);
    return PairUnit{it, (it % g.n_tiles) * 256 + (u & 1) * 128, true};
}

// unit u of a pair kernel that may also run a shortcut (units n1 ..: its
// whole tiles)
template <bool VARN, bool SC>
__device__ __forceinline__ PairUnit pair_unit_sc(int u, int n1, const TcGeom &g, const TcGeom &g2) {
    if (SC && u >= n1) return PairUnit{u - n1, ((u - n1) % g2.n_tiles) * 256, false};
    return pair_unit<VARN>(u, g);
}

size_t pair_smem_bytes() {
    return 1024 + (size_t)PR_STAGES * (A_BYTES + PR_BH_BYTES) + 8 * PR_NBAR + 16 + 16 + 4 * BIAS_SMEM;
}

// SC: the launch also runs a 1x1 shortcut convolution as whole tiles after
// this layer's units (bmap2: its 128-row weight halves; a2, g2; see UnitSeq).
template <bool VARN, bool SC>
__global__ void __launch_bounds__(PR_THREADS, 1)
conv_tc_pair_kernel(const __grid_constant__ CUtensorMap amap, const __grid_constant__ CUtensorMap bmap,
                    const __grid_constant__ CUtensorMap bmap64, const __grid_constant__ ConvArgs a,
                    const __grid_constant__ TcGeom g, const __grid_constant__ CUtensorMap bmap2,
                    const __grid_constant__ ConvArgs a2, const __grid_constant__ TcGeom g2) {
    constexpr int BN = 256;
    static_assert(PR_STAGES % PR_NPROD == 0, "producer warps must own whole ring slots");
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint8_t *As = smem;                                    // [STAGES][A_BYTES]
    uint8_t *Bs = As + PR_STAGES * A_BYTES;                // [STAGES][PR_BH_BYTES]
    uint64_t *full = (uint64_t *)(Bs + PR_STAGES * PR_BH_BYTES);
    uint64_t *empty = full + PR_STAGES;
    uint64_t *acc_full = empty + PR_STAGES;                // [2]
    uint64_t *pair_empty = acc_full + 2;                   // [2]
    uint64_t *mma_done = pair_empty + 2;
    uint32_t *tmem_holder = (uint32_t *)(mma_done + 1);
    volatile uint32_t *abort_flag = tmem_holder + 1;
    float *bias_s = (float *)(((uintptr_t)(tmem_holder + 2) + 15) & ~(uintptr_t)15);   // [BIAS_SMEM]

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t crank = cluster_ctarank();
    const bool leader = crank == 0;
    const int cid = blockIdx.x >> 1, ncl = gridDim.x >> 1;
    const int n1 = VARN ? g.units : ((g.m_tiles + 1) >> 1) * g.n_tiles;    // this layer's units
    const UnitSeq us = unit_seq<SC>(cid, ncl, n1, g);
    const int n_units = us.k1 + us.cnt;                                     // this pair's units

    if (threadIdx.x == 0) {
        for (int s = 0; s < PR_STAGES; ++s) {
            mbar_init(smem_u32(&full[s]), 1);
            mbar_init(smem_u32(&empty[s]), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(smem_u32(&acc_full[b]), 1);
            mbar_init(smem_u32(&pair_empty[b]), 2 * N_EPI_WARPS);
        }
        mbar_init(smem_u32(mma_done), 1);
        *abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == PR_MMA_WARP) {
        // one warp of each CTA of the pair allocates the same columns in both
        asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_holder)),
                     "r"(512u));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;");
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    // the peer's barriers are initialised before any copy or arrival targets them
    cluster_sync();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tmem = *tmem_holder;
    pdl_wait();
    pdl_trigger();

    if (warp < PR_NPROD) {
        // ---------------- TMA producers (slot s belongs to warp s % PR_NPROD) ----------------
        if (elect_one()) {
            asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&amap) : "memory");
            asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&bmap) : "memory");
            if (VARN) asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&bmap64) : "memory");
            if (SC) asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&bmap2) : "memory");
        }
        __syncwarp();
        const uint32_t full_even = mapa_shared(smem_u32(full), 0u);
        int it = 0;
        bool ok = true;
        for (int k = 0; k < n_units && ok; ++k) {
            if (__any_sync(0xffffffffu, *abort_flag)) break;
            const int u = unit_at(us, k, cid, ncl);
            const bool sc = SC && u >= n1;
            const PairUnit pu = pair_unit_sc<VARN, SC>(u, n1, g, g2);
            const int n_kb = sc ? g2.n_kb : g.n_kb;
            const bool hu = VARN && pu.narrow;                    // 128 channels
            const int m_pair = pu.item / (sc ? g2.n_tiles : g.n_tiles);
            const int m0 = (2 * m_pair + (int)crank) * BM;       // past M: rows that are never stored
            const int nimg = m0 / g.PQ, rem = m0 % g.PQ;
            const int p = rem / g.Q, q = rem % g.Q;
            // A coordinates: this layer's geometry (a shortcut reads its centre tap)
            const int w0 = q * g.stride - g.pad, h0 = p * g.stride - g.pad;
            for (int kb = 0; kb < n_kb; ++kb, ++it) {
                const int s = it % PR_STAGES;
                if (s % PR_NPROD != warp) continue;
                if (!warp_wait(smem_u32(&empty[s]), ((uint32_t)(it / PR_STAGES) & 1u) ^ 1u, a.err, 1u)) { ok = false; break; }
                if (elect_one()) {
                    const uint32_t fb = full_even + (uint32_t)(s * 8);
                    if (leader)
                        mbar_arrive_expect_tx(smem_u32(&full[s]), 2u * (A_BYTES + (hu ? PR_BH_BYTES / 2 : PR_BH_BYTES)));
                    const int tap = tap_of(kb / g.cpb, g.ctr_tap);
                    const int c0 = (kb % g.cpb) * BK;
                    const int r = tap / g.S, sx = tap % g.S;
                    tma_load_im2col_pair(smem_u32(As + s * A_BYTES), &amap, fb, c0, w0, h0, nimg, (uint16_t)sx,
                                         (uint16_t)r);
                    if (hu)
                        tma_load_2d_pair(smem_u32(Bs + s * PR_BH_BYTES), &bmap64, fb, tap * g.C + c0,
                                         pu.nb + (int)crank * (BM / 2));
                    else if (sc)
                        tma_load_2d_pair(smem_u32(Bs + s * PR_BH_BYTES), &bmap2, fb, c0, pu.nb + (int)crank * BM);
                    else
                        tma_load_2d_pair(smem_u32(Bs + s * PR_BH_BYTES), &bmap, fb, tap * g.C + c0,
                                         pu.nb + (int)crank * BM);
                }
                __syncwarp();
            }
        }
        if (!ok && lane == 0) *abort_flag = 1;
    } else if (warp == PR_MMA_WARP) {
        // ---------------- MMA issuer: the even CTA, one elected lane ----------------
        if (leader) {
            int it = 0;
            for (int lt = 0; lt < n_units; ++lt) {
                if (__any_sync(0xffffffffu, *abort_flag)) break;
                const int u = unit_at(us, lt, cid, ncl);
                const int n_kb = (SC && u >= n1) ? g2.n_kb : g.n_kb;
                const bool hu = VARN && pair_unit_sc<VARN, SC>(u, n1, g, g2).narrow;
                const uint32_t idesc = idesc_f16(2 * BM, hu ? BN / 2 : BN);
                const int ab = lt & 1;
                if (!warp_wait(smem_u32(&pair_empty[ab]), ((uint32_t)(lt >> 1) & 1u) ^ 1u, a.err, 8u)) {
                    if (lane == 0) *abort_flag = 1;
                    break;
                }
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                bool ok = true;
                for (int kb = 0; kb < n_kb; ++kb, ++it) {
                    const int s = it % PR_STAGES;
                    if (!warp_wait(smem_u32(&full[s]), (uint32_t)(it / PR_STAGES) & 1u, a.err, 2u)) { ok = false; break; }
                    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                    if (elect_one()) {
                        const uint32_t d = tmem + (uint32_t)(ab * BN);
                        const uint64_t ad0 = smem_desc_sw128(smem_u32(As + s * A_BYTES));
                        const uint64_t bd0 = smem_desc_sw128(smem_u32(Bs + s * PR_BH_BYTES));
#pragma unroll
                        for (int k16 = 0; k16 < BK / 16; ++k16)
                            umma_f16_pair(d, ad0 + 2 * k16, bd0 + 2 * k16, idesc, (kb > 0 || k16 > 0) ? 1u : 0u);
                        umma_commit_pair_mc(smem_u32(&empty[s]), (uint16_t)3u);
                    }
                    __syncwarp();
                }
                if (!ok) { if (lane == 0) *abort_flag = 1; break; }
                if (elect_one()) umma_commit_pair_mc(smem_u32(&acc_full[ab]), (uint16_t)3u);
                __syncwarp();
            }
            // fires in both CTAs once every MMA issued above has completed
            if (elect_one()) umma_commit_pair_mc(smem_u32(mma_done), (uint16_t)3u);
            __syncwarp();
        }
    } else {
        // ---------------- epilogue: 8 warps, this CTA's 128 rows ----------------
        const int ep = warp - PR_EPI_WARP0;
        const int quad = warp & 3;
        const int half = ep >> 2;
        const int row = quad * 32 + lane;
        const uint32_t pair_empty_even = mapa_shared(smem_u32(pair_empty), 0u);
        const int et = threadIdx.x - 32 * PR_EPI_WARP0;
        const bool bias_sm = SC ? stage_bias2(bias_s, a.bias, a2.bias, g.K, et, 32 * N_EPI_WARPS)
                                : stage_bias(bias_s, a.bias, g.K, et, 32 * N_EPI_WARPS);
        for (int lt = 0; lt < n_units; ++lt) {
            const int u = unit_at(us, lt, cid, ncl);
            const bool sc = SC && u >= n1;
            const ConvArgs &A = sc ? a2 : a;       // this unit's layer
            const TcGeom &G = sc ? g2 : g;
            const float *bias_l = bias_s + (sc ? G.K : 0);
            const __half *x = static_cast<const __half *>(A.x);
            const FaultDelta fd = A.fd;
            const float coef = __half2float(__ushort_as_half(G.coef_h));
            const int ctr_r = G.ctr_tap / G.S, ctr_s = G.ctr_tap % G.S;
            const bool has_res = A.res != nullptr, relu = A.relu != 0;
            const PairUnit pu = pair_unit_sc<VARN, SC>(u, n1, g, g2);
            const bool hu = VARN && pu.narrow;
            const int m_pair = pu.item / G.n_tiles;
            const int m0 = (2 * m_pair + (int)crank) * BM;
            const int m = m0 + row;
            const bool valid = m < G.M;
            const int mm = valid ? m : 0;
            const int nimg = mm / G.PQ, rem = mm % G.PQ, p = rem / G.Q, q = rem % G.Q;
            const bool do_cs = half == 0 && A.cs_out != nullptr && pu.nb == 0;
            // this warp's channels: cols [cw, cw + ncw) of the accumulator,
            // output channels nw + (0 .. ncw)
            const int ncw = hu ? BN / 4 : BN / 2;
            const int cw = half * ncw;
            const int nw = pu.nb + cw;
            Res16 rs[BN / 32];
#pragma unroll
            for (int c = 0; c < BN / 32; ++c)
                rs[c] = (valid && 16 * c < ncw) ? load_res16(A, G.K, (size_t)m, nw + 16 * c)
                                                : Res16{make_uint4(0u, 0u, 0u, 0u), make_uint4(0u, 0u, 0u, 0u)};
            CsIn csv{0.f, 0, 0};
            // carry-through column: coef * sum of the C channels of the centre-tap pixel
            float ctv = 0.f;
            if (do_cs && valid) {
                csv = load_cs_inputs(A, G, m, nimg, p, q);
                if (G.ct_mode != CT_NONE_) {
                    const int h = p * G.stride + ctr_r - G.pad, w = q * G.stride + ctr_s - G.pad;
                    if (h >= 0 && h < A.H && w >= 0 && w < A.W) {
                        const uint4 *src = reinterpret_cast<const uint4 *>(x + (((size_t)nimg * A.H + h) * A.W + w) * G.C);
                        float acc[4] = {0.f, 0.f, 0.f, 0.f};
                        for (int c8 = 0; c8 < G.C / 8; ++c8) {
                            const uint4 u = __ldg(src + c8);
                            const __half2 *hh = reinterpret_cast<const __half2 *>(&u);
#pragma unroll
                            for (int i = 0; i < 4; ++i) {
                                const float2 f = __half22float2(hh[i]);
                                acc[i] += f.x;
                                acc[i] += f.y;
                            }
                        }
                        ctv = coef * ((acc[0] + acc[1]) + (acc[2] + acc[3]));
                    }
                }
            }
            const int ab = lt & 1;
            const uint32_t aph = (uint32_t)(lt >> 1) & 1u;
            bool ok = mbar_wait(smem_u32(&acc_full[ab]), aph, A.err, 4u) && !*abort_flag;
            ok = __all_sync(0xffffffffu, ok);      // tcgen05.ld below is warp-collective
            if (!ok) break;
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            const uint32_t trow = tmem + (uint32_t)(ab * BN) + ((uint32_t)(quad * 32) << 16);
            float fsrc = 0.f;
            if (fd.active) {
                const int h = p * G.stride + fd.r - G.pad, w = q * G.stride + fd.s - G.pad;
                if (h >= 0 && h < A.H && w >= 0 && w < A.W) {
                    if (fd.cin < G.C) fsrc = ldh(x, (((size_t)nimg * A.H + h) * A.W + w) * G.C + fd.cin);
                    else if (A.cs_in) fsrc = ldh(static_cast<const __half *>(A.cs_in), ((size_t)nimg * A.H + h) * A.W + w);
                }
            }
            if (!fd.active && !has_res) {
                // whole lines: per 64 channels the lanes of each group of four
                // swap their 16-channel pieces (all lanes take part; stores of
                // pixels past M are skipped)
#pragma unroll
                for (int c0 = 0; c0 < BN / 2; c0 += 64) {
                    if (c0 >= ncw) break;
                    uint32_t pk[4][8];
#pragma unroll
                    for (int c = 0; c < 4; ++c) {
                        float v[16];
                        tmem_ld16(trow + cw + c0 + 16 * c, v);
                        pack16(v, bias16_at(bias_l, A.bias, bias_sm, nw + c0 + 16 * c), relu, pk[c]);
                    }
                    transpose4_pieces(pk, lane & 3);
#pragma unroll
                    for (int k = 0; k < 4; ++k) {
                        const int mk = m0 + quad * 32 + (lane & ~3) + k;
                        if (mk < G.M)
                            st_global_v8(static_cast<__half *>(A.y) + (size_t)mk * G.K + nw + c0 + 16 * (lane & 3),
                                         pk[k]);
                    }
                }
            } else {
#pragma unroll
            for (int c = 0; c < BN / 2; c += 16) {
                if (c >= ncw) break;
                float v[16];
                tmem_ld16(trow + cw + c, v);
                if (valid && fd.active) store_chunk_pre(v, rs[c / 16], A, G.K, (size_t)m, nw + c, fsrc);
                else if (valid)
                    store16_fast(v, bias16_at(bias_l, A.bias, bias_sm, nw + c), rs[c / 16], has_res, relu,
                                 static_cast<__half *>(A.y) + (size_t)m * G.K + nw + c);
            }
            }
            if (do_cs && valid) store_checksum_pre(ctv, csv, A, G, m, fsrc);
            asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
            __syncwarp();
            if (lane == 0) mbar_arrive_cluster(pair_empty_even + (uint32_t)(ab * 8));
        }
    }
    // every MMA of the pair has completed before TMEM is freed in either CTA
    if (warp == PR_MMA_WARP) warp_wait(smem_u32(mma_done), 0u, a.err, 16u);
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    // no CTA leaves while its peer may still read its shared memory or
    // arrive on its barriers
    cluster_sync();
    if (warp == PR_MMA_WARP) {
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(512u));
    }
}

// ---------------------------------------------------------------------------
// First layers with at most 4 input channels (the image): the input is
// stored NHWC with its channels padded to 4 (8 bytes per pixel) and the GEMM
// K index runs over (tap, channel of 4), 16 taps per 64-wide K block.  TMA
// im2col cannot fetch 8-byte pixels, so four producer warps build the A tile
// in shared memory: each thread owns one output pixel, loads one 8-byte
// input pixel per tap and writes the 128-byte swizzled row the MMA reads.
// Output channels: 64.  The carry-through row is coef at the centre tap's
// real channels: 16 constant rows after the 64 weight rows of every B stage,
// used (N = 80) on the centre tap's K block, which the loop visits first.
// Persistent, double-buffered accumulators, as above.
// ---------------------------------------------------------------------------
constexpr int SM_THREADS = 288;     // warps 0-3 producers, 4 MMA, 5-8 epilogue
constexpr int SM_STAGES = 8;
constexpr int SM_BN = 64;

struct TcGeomS {
    int M, PQ, Q, stride, pad, C, H, W, R, S;
    int n_kb, kb_ct, col_ct, ct;
    int tmem_cols, m_tiles;
    uint16_t coef_h;
};

__global__ void __launch_bounds__(SM_THREADS, 1)
conv_tc_small_kernel(const __grid_constant__ CUtensorMap bmap, const ConvArgs a, const TcGeomS g) {
    constexpr int B_ROWS = SM_BN + 16;
    constexpr int B_BYTES_STAGE = B_ROWS * BK * 2;
    constexpr int B_TMA_BYTES = SM_BN * BK * 2;
    constexpr int NCH = 4;                                // accumulator chains (see conv_tc_kernel)
    constexpr int CH = SM_BN + 16;
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint8_t *As = smem;
    uint8_t *Bs = As + SM_STAGES * A_BYTES;
    uint64_t *full = (uint64_t *)(Bs + SM_STAGES * B_BYTES_STAGE);
    uint64_t *empty = full + SM_STAGES;
    uint64_t *acc_full = empty + SM_STAGES;
    uint64_t *acc_empty = acc_full + 1;
    uint32_t *tmem_holder = (uint32_t *)(acc_empty + 1);
    volatile uint32_t *abort_flag = tmem_holder + 1;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int s = 0; s < SM_STAGES; ++s) {
            mbar_init(smem_u32(&full[s]), 128);
            mbar_init(smem_u32(&empty[s]), 1);
        }
        mbar_init(smem_u32(acc_full), 1);
        mbar_init(smem_u32(acc_empty), 4);
        *abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 4) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_holder)),
                     "r"((uint32_t)g.tmem_cols));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    if (warp >= 5) {
        // constant rows 64..79 of every B stage: row 64 = coef at the centre
        // tap's real channels (columns col_ct .. col_ct + C - 1), the rest 0;
        // rows whose index is a multiple of 8 are not permuted by the swizzle
        const int t = threadIdx.x - 160;
        const __half ch = __ushort_as_half(g.coef_h);
        for (int s = 0; s < SM_STAGES; ++s) {
            __half *rows = (__half *)(Bs + s * B_BYTES_STAGE + SM_BN * BK * 2);
            for (int i = t; i < 16 * BK; i += 128)
                rows[i] = (g.ct && i >= g.col_ct && i < g.col_ct + g.C) ? ch : __ushort_as_half((unsigned short)0);
        }
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tmem = *tmem_holder;
    // the previous kernel's outputs (and any fault flip) are visible from here
    pdl_wait();
    pdl_trigger();
    const __half *x = static_cast<const __half *>(a.x);

    if (warp < 4) {
        // ---------------- software im2col producers ----------------
        const int row = threadIdx.x;
        if (row == 0) asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&bmap) : "memory");
        const int taps = g.R * g.S;
        int it = 0;
        for (int tile = blockIdx.x; tile < g.m_tiles && !*abort_flag; tile += gridDim.x) {
            const int m = tile * BM + row;
            const bool valid = m < g.M;
            const int mm = valid ? m : 0;
            const int nimg = mm / g.PQ, rem = mm % g.PQ, p = rem / g.Q, q = rem % g.Q;
            const int h0 = p * g.stride - g.pad, w0 = q * g.stride - g.pad;
            const __half *ximg = x + (size_t)nimg * g.H * g.W * 4;
            for (int i = 0; i < g.n_kb; ++i, ++it) {
                const int kb = (i + g.kb_ct) % g.n_kb;
                // all 16 taps of this K block are fetched before any shared-memory
                // store, so their global-load latencies overlap
                uint2 v[16];
                int r = (kb * 16) / g.S, sx = (kb * 16) % g.S;
#pragma unroll
                for (int u = 0; u < 16; ++u) {
                    v[u] = make_uint2(0u, 0u);
                    const int h = h0 + r, w = w0 + sx;
                    if (valid && kb * 16 + u < taps && h >= 0 && h < g.H && w >= 0 && w < g.W)
                        v[u] = __ldg(reinterpret_cast<const uint2 *>(ximg + ((size_t)h * g.W + w) * 4));
                    if (++sx == g.S) { sx = 0; ++r; }
                }
                const int s = it % SM_STAGES;
                const uint32_t ph = (uint32_t)(it / SM_STAGES) & 1u;
                if (!mbar_wait(smem_u32(&empty[s]), ph ^ 1u, a.err, 1u)) { *abort_flag = 1; break; }
                const uint32_t fb = smem_u32(&full[s]);
                if (row == 0) {
                    mbar_expect_tx_only(fb, B_TMA_BYTES);
                    tma_load_2d(smem_u32(Bs + s * B_BYTES_STAGE), &bmap, fb, kb * BK, 0);
                }
                uint8_t *arow = As + s * A_BYTES + row * 128;
#pragma unroll
                for (int j = 0; j < 8; ++j)
                    *reinterpret_cast<uint4 *>(arow + ((j ^ (row & 7)) << 4)) =
                        make_uint4(v[2 * j].x, v[2 * j].y, v[2 * j + 1].x, v[2 * j + 1].y);
                asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                mbar_arrive(fb);
            }
        }
    } else if (warp == 4) {
        // ---------------- MMA issuer (whole warp, one lane issues) ----------------
        const uint32_t id_main = idesc_f16(BM, SM_BN);
        const uint32_t id_merged = idesc_f16(BM, SM_BN + 16);
        int it = 0, lt = 0;
        for (int tile = blockIdx.x; tile < g.m_tiles; tile += gridDim.x, ++lt) {
            if (__any_sync(0xffffffffu, *abort_flag)) break;
            if (!warp_wait(smem_u32(acc_empty), ((uint32_t)lt & 1u) ^ 1u, a.err, 8u)) {
                if (lane == 0) *abort_flag = 1;
                break;
            }
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            bool ok = true;
            for (int i = 0; i < g.n_kb; ++i, ++it) {
                const uint32_t d = tmem + (uint32_t)((i % NCH) * CH);
                const int s = it % SM_STAGES;
                const uint32_t ph = (uint32_t)(it / SM_STAGES) & 1u;
                if (!warp_wait(smem_u32(&full[s]), ph, a.err, 2u)) { ok = false; break; }
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                const uint32_t a_base = smem_u32(As + s * A_BYTES);
                const uint32_t b_base = smem_u32(Bs + s * B_BYTES_STAGE);
                const bool leader = elect_one();
#pragma unroll
                for (int k16 = 0; k16 < BK / 16; ++k16) {
                    const uint64_t ad = smem_desc_sw128(a_base + k16 * 32);
                    const uint64_t bd = smem_desc_sw128(b_base + k16 * 32);
                    const uint32_t acc = (i >= NCH || k16 > 0) ? 1u : 0u;   // first use of the chain
                    if (leader) umma_f16(d, ad, bd, (i == 0 && g.ct) ? id_merged : id_main, acc);
                }
                if (leader) umma_commit(smem_u32(&empty[s]));
                __syncwarp();
            }
            if (!ok) { if (lane == 0) *abort_flag = 1; break; }
            if (elect_one()) umma_commit(smem_u32(acc_full));
            __syncwarp();
        }
    } else {
        // ---------------- epilogue: warps 5..8 ----------------
        const int quad = warp & 3;
        const int row = quad * 32 + lane;
        const FaultDelta fd = a.fd;
        const int chains = min(NCH, g.n_kb);
        int lt = 0;
        for (int tile = blockIdx.x; tile < g.m_tiles; tile += gridDim.x, ++lt) {
            bool ok = mbar_wait(smem_u32(acc_full), (uint32_t)lt & 1u, a.err, 4u) && !*abort_flag;
            ok = __all_sync(0xffffffffu, ok);
            if (!ok) break;
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            const uint32_t trow = tmem + ((uint32_t)(quad * 32) << 16);
            float vals[SM_BN];
#pragma unroll
            for (int c = 0; c < SM_BN; c += 16) {
                tmem_ld16(trow + c, vals + c);
                for (int ch = 1; ch < chains; ++ch) {
                    float t[16];
                    tmem_ld16(trow + ch * CH + c, t);
#pragma unroll
                    for (int i = 0; i < 16; ++i) vals[c + i] += t[i];
                }
            }
            const float ctv = (a.cs_out != nullptr && g.ct) ? tmem_ld1(trow + SM_BN) : 0.f;   // chain 0 only
            asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(acc_empty));
            const int m = tile * BM + row;
            if (m < g.M) {
                const int nimg = m / g.PQ, rem = m % g.PQ, p = rem / g.Q, q = rem % g.Q;
                float fsrc = 0.f;
                if (fd.active) {
                    const int h = p * g.stride + fd.r - g.pad, w = q * g.stride + fd.s - g.pad;
                    if (fd.cin < g.C && h >= 0 && h < g.H && w >= 0 && w < g.W)
                        fsrc = ldh(x, (((size_t)nimg * g.H + h) * g.W + w) * 4 + fd.cin);
                }
#pragma unroll
                for (int c = 0; c < SM_BN; c += 16) store_chunk(vals + c, a, SM_BN, (size_t)m, c, fsrc);
                if (a.cs_out != nullptr) {
                    float o = (a.role == CT_ROLE_CT) ? ctv : 0.f;
                    if (fd.active && fd.kout == SM_BN) o += fd.dv * fsrc;
                    if (a.relu) o = relu_keep_nan(o);
                    static_cast<__half *>(a.cs_out)[m] = __float2half_rn(o);
                }
            }
        }
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (warp == 4) {
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"((uint32_t)g.tmem_cols));
    }
}

// ---------------------------------------------------------------------------
// Stride-1 3x3 convolutions from a halo tile.  An output tile of 16 rows x
// 8 columns (M = 128) needs an 18 x 10 pixel patch of its input; one tiled
// TMA per 64-channel block copies it to shared memory (128-byte rows,
// 128-byte swizzle, zero fill outside the image), and the nine taps are
// nine views of that patch: the A descriptor of tap (r, s) starts r patch
// rows and s pixels into it, and its 8-row groups (one output row each) are
// one patch row (1280 bytes) apart.  The 128-byte swizzle follows the
// absolute shared-memory address, so shifted starts read the rows the TMA
// wrote.  Each input pixel thus crosses L2 -> SM once per tile instead of
// once per tap (im2col).  B (64 x BN per tap and channel block) streams
// through its own ring, or stays resident for the whole kernel when the
// layer has one channel block and one N tile (C = K = 64).  The
// carry-through row is merged into the centre tap's MMAs as in
// conv_tc_kernel; two TMEM accumulators alternate between tiles.
// ---------------------------------------------------------------------------
constexpr int HT_TH = 16, HT_TW = 8;                    // output tile
constexpr int HT_PH = HT_TH + 2, HT_PW = HT_TW + 2;     // input patch with a one-pixel halo
constexpr int HT_A_BYTES = HT_PH * HT_PW * BK * 2;      // 23040
constexpr int HT_A_STAGE = 23 * 1024;                   // stage pitch (1024-byte aligned)
constexpr int HT_ROW = HT_PW * BK * 2;                  // 1280: one patch row, the A group stride

struct HaloGeom {
    int N, H, W, C, K;
    int ncb, n_tiles, ty_tiles, tx_tiles;
    int ct;
    int tmem_cols;
    int res, csin, rescs;       // epilogue operands fetched by TMA into the R ring
    uint16_t coef_h;
};

__device__ __forceinline__ uint64_t smem_desc_sw128_sbo(uint32_t addr, uint32_t sbo) {
    uint64_t d = 0;
    d |= (uint64_t)((addr >> 4) & 0x3FFF);
    d |= (uint64_t)1 << 16;
    d |= (uint64_t)((sbo >> 4) & 0x3FFF) << 32;
    d |= (uint64_t)1 << 46;
    d |= (uint64_t)2 << 61;
    return d;
}

__device__ __forceinline__ void tma_load_4d(uint32_t dst, const CUtensorMap *map, uint32_t bar, int c, int x,
                                            int y, int n) {
    asm volatile(
        "cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3, %4, %5}], [%6];" ::"r"(dst),
        "l"((uint64_t)map), "r"(c), "r"(x), "r"(y), "r"(n), "r"(bar)
        : "memory");
}

__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap *map, uint32_t bar, int x, int y, int n) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(dst),
        "l"((uint64_t)map), "r"(x), "r"(y), "r"(n), "r"(bar)
        : "memory");
}

struct HaloTile {
    int n, y0, x0, nt;
};
__device__ __forceinline__ HaloTile halo_tile(int t, const HaloGeom &hg) {
    HaloTile h;
    h.nt = t % hg.n_tiles;
    const int r1 = t / hg.n_tiles;
    h.x0 = (r1 % hg.tx_tiles) * HT_TW;
    const int r2 = r1 / hg.tx_tiles;
    h.y0 = (r2 % hg.ty_tiles) * HT_TH;
    h.n = r2 / hg.ty_tiles;
    return h;
}

// tensor maps of one halo plan: patch (A), weights (B), and the epilogue
// operands: residual tile [16 x 8 x BN], incoming and residual checksum
// planes [16 x 8]
struct HaloMaps {
    CUtensorMap amap, bmap, rmap, cmap, qmap;
};

// Epilogue operand ring (R): per tile, the residual tile and the incoming /
// residual checksum values of its pixels, fetched by the producer warp with
// TMA several tiles ahead so that the epilogue reads them from shared
// memory.  The residual is BN / 64 blocks of [128 pixels][64 channels], each
// copied with the 128-byte swizzle (16-byte chunk c of pixel r at chunk
// c ^ (r & 7)): the epilogue lane of pixel r reads 16 bytes of its own
// 128-byte row, and without the swizzle the 32 lanes of a warp would all hit
// the same four banks.
template <int BN>
struct HaloR {
    static constexpr int RES = 128 * BN * 2;
    static constexpr int CS = 128 * 2;
    static constexpr int STAGE = (RES + 2 * CS + 1023) / 1024 * 1024;   // swizzle atoms stay 1024-byte aligned
};

// Resident weights (one channel block, one N tile): tap visit i (the centre
// tap first) at offset halo_bres_off(i); only the centre tap is followed by
// the 16 constant carry-through rows.
template <int BN>
__host__ __device__ constexpr int halo_bres_off(int i) {
    return i == 0 ? 0 : (BN + 16) * BK * 2 + (i - 1) * BN * BK * 2;
}

// POOL: the 2 x 2 stride-2 max-pool that follows the convolution is applied
// in the epilogue (data and checksum alike); a.y / a.cs_out are then the
// pooled tensor [N, H / 2, W / 2, K] and its checksum plane.
template <int BN, bool BRES, int NA, int NB, int NR, bool POOL>
__global__ void __launch_bounds__(NTHREADS, 1)
conv_tc_halo_kernel(const __grid_constant__ HaloMaps maps, const ConvArgs a, const HaloGeom hg, const TcGeom g) {
    constexpr int B_ROWS = BN + 16;                       // 16 constant carry-through rows
    constexpr int B_STAGE = B_ROWS * BK * 2;
    constexpr int B_TMA = BN * BK * 2;
    constexpr int NBS = BRES ? 9 : NB;
    constexpr int B_AREA = BRES ? halo_bres_off<BN>(9) : NB * B_STAGE;
    constexpr int CH = BN + 16;
    using R = HaloR<BN>;
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint8_t *As = smem;
    uint8_t *Bs = As + NA * HT_A_STAGE;
    uint8_t *Rs = Bs + B_AREA;
    uint64_t *a_full = (uint64_t *)(Rs + NR * R::STAGE);
    uint64_t *a_empty = a_full + NA;
    uint64_t *b_full = a_empty + NA;
    uint64_t *b_empty = b_full + NBS;
    uint64_t *r_full = b_empty + NBS;
    uint64_t *r_empty = r_full + NR;
    uint64_t *acc_full = r_empty + NR;
    uint64_t *acc_empty = acc_full + 2;
    uint32_t *tmem_holder = (uint32_t *)(acc_empty + 2);
    volatile uint32_t *abort_flag = tmem_holder + 1;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int num_tiles = hg.N * hg.ty_tiles * hg.tx_tiles * hg.n_tiles;
    const bool ring = hg.res || hg.csin || hg.rescs;
    const uint32_t r_bytes = (hg.res ? R::RES : 0) + (hg.csin ? R::CS : 0) + (hg.rescs ? R::CS : 0);

    if (threadIdx.x == 0) {
        for (int s = 0; s < NA; ++s) {
            mbar_init(smem_u32(&a_full[s]), 1);
            mbar_init(smem_u32(&a_empty[s]), 1);
        }
        for (int s = 0; s < NBS; ++s) {
            mbar_init(smem_u32(&b_full[s]), 1);
            mbar_init(smem_u32(&b_empty[s]), 1);
        }
        for (int s = 0; s < NR; ++s) {
            mbar_init(smem_u32(&r_full[s]), 1);
            mbar_init(smem_u32(&r_empty[s]), N_EPI_WARPS);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(smem_u32(&acc_full[b]), 1);
            mbar_init(smem_u32(&acc_empty[b]), N_EPI_WARPS);
        }
        *abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_holder)),
                     "r"((uint32_t)hg.tmem_cols));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    if (warp >= 2) {
        // constant carry-through rows after the BN weight rows of every B stage:
        // row 0 = coef, rows 1..15 = 0 (swizzle-invariant)
        const uint32_t coef2 = (uint32_t)hg.coef_h | ((uint32_t)hg.coef_h << 16);
        const int t = threadIdx.x - 64;
        for (int sb = 0; sb < (BRES ? 1 : NBS); ++sb) {
            uint32_t *rows = (uint32_t *)(Bs + sb * B_STAGE + BN * BK * 2);
            for (int i = t; i < 16 * BK / 2; i += 32 * N_EPI_WARPS) rows[i] = (i < BK / 2) ? coef2 : 0u;
        }
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tmem = *tmem_holder;
    // the previous kernel's outputs (and any fault flip) are visible from here
    pdl_wait();
    pdl_trigger();

    if (warp == 0) {
        // ---------------- TMA producer (whole warp, one lane issues) ----------------
        if (elect_one()) {
            asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&maps.amap) : "memory");
            asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&maps.bmap) : "memory");
            if (BRES) {
                for (int i = 0; i < 9; ++i) {
                    mbar_arrive_expect_tx(smem_u32(&b_full[i]), B_TMA);
                    tma_load_2d(smem_u32(Bs + halo_bres_off<BN>(i)), &maps.bmap, smem_u32(&b_full[i]),
                                tap_of(i, 4) * hg.C, 0);
                }
            }
        }
        __syncwarp();
        int ai = 0, bi = 0, ri = 0;
        bool ok = true;
        for (int tile = blockIdx.x; tile < num_tiles && ok; tile += gridDim.x) {
            if (__any_sync(0xffffffffu, *abort_flag)) break;
            const HaloTile ht = halo_tile(tile, hg);
            for (int cb = 0; cb < hg.ncb && ok; ++cb) {
                const int as = ai % NA;
                if (!warp_wait(smem_u32(&a_empty[as]), ((uint32_t)(ai / NA) & 1u) ^ 1u, a.err, 1u)) { ok = false; break; }
                if (elect_one()) {
                    mbar_arrive_expect_tx(smem_u32(&a_full[as]), HT_A_BYTES);
                    tma_load_4d(smem_u32(As + as * HT_A_STAGE), &maps.amap, smem_u32(&a_full[as]), cb * BK, ht.x0 - 1,
                                ht.y0 - 1, ht.n);
                }
                __syncwarp();
                ++ai;
                if (cb == 0 && ring) {
                    // epilogue operands of this tile, behind its first patch
                    const int rs = ri % NR;
                    if (!warp_wait(smem_u32(&r_empty[rs]), ((uint32_t)(ri / NR) & 1u) ^ 1u, a.err, 1u)) { ok = false; break; }
                    if (elect_one()) {
                        const uint32_t rb = smem_u32(&r_full[rs]);
                        uint8_t *st = Rs + rs * R::STAGE;
                        mbar_arrive_expect_tx(rb, r_bytes);
                        if (hg.res)
                            for (int cb = 0; cb < BN / 64; ++cb)
                                tma_load_4d(smem_u32(st + cb * 128 * 128), &maps.rmap, rb, ht.nt * BN + cb * 64, ht.x0,
                                            ht.y0, ht.n);
                        if (hg.csin) tma_load_3d(smem_u32(st + R::RES), &maps.cmap, rb, ht.x0, ht.y0, ht.n);
                        if (hg.rescs) tma_load_3d(smem_u32(st + R::RES + R::CS), &maps.qmap, rb, ht.x0, ht.y0, ht.n);
                    }
                    __syncwarp();
                    ++ri;
                }
                if (!BRES) {
                    for (int i = 0; i < 9; ++i) {
                        const int bs = bi % NBS;
                        if (!warp_wait(smem_u32(&b_empty[bs]), ((uint32_t)(bi / NBS) & 1u) ^ 1u, a.err, 1u)) {
                            ok = false;
                            break;
                        }
                        if (elect_one()) {
                            mbar_arrive_expect_tx(smem_u32(&b_full[bs]), B_TMA);
                            tma_load_2d(smem_u32(Bs + bs * B_STAGE), &maps.bmap, smem_u32(&b_full[bs]),
                                        tap_of(i, 4) * hg.C + cb * BK, ht.nt * BN);
                        }
                        __syncwarp();
                        ++bi;
                    }
                }
            }
        }
        if (!ok && lane == 0) *abort_flag = 1;
    } else if (warp == 1) {
        // ---------------- MMA issuer (whole warp, one lane issues) ----------------
        const uint32_t id_main = idesc_f16(BM, BN);
        const uint32_t id_merged = idesc_f16(BM, BN + 16);
        int ai = 0, bi = 0, lt = 0;
        bool ok = true;
        if (BRES) {
            // resident weights: wait for all nine tiles once
            for (int i = 0; i < 9 && ok; ++i) ok = warp_wait(smem_u32(&b_full[i]), 0u, a.err, 2u);
        }
        for (int tile = blockIdx.x; tile < num_tiles && ok; tile += gridDim.x, ++lt) {
            if (__any_sync(0xffffffffu, *abort_flag)) break;
            const HaloTile ht = halo_tile(tile, hg);
            const bool ct_here = hg.ct && ht.nt == 0;
            const int ab = lt & 1;
            if (!warp_wait(smem_u32(&acc_empty[ab]), ((uint32_t)(lt >> 1) & 1u) ^ 1u, a.err, 8u)) { ok = false; break; }
            const uint32_t d = tmem + (uint32_t)(ab * CH);
            for (int cb = 0; cb < hg.ncb && ok; ++cb) {
                const int as = ai % NA;
                if (!warp_wait(smem_u32(&a_full[as]), (uint32_t)(ai / NA) & 1u, a.err, 2u)) { ok = false; break; }
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                const uint32_t a_base = smem_u32(As + as * HT_A_STAGE);
                if constexpr (BRES) {
                    // all 36 MMAs of the tile in one burst from one lane
                    if (elect_one()) {
                        const uint32_t b0 = smem_u32(Bs);
#pragma unroll
                        for (int i = 0; i < 9; ++i) {
                            const int tap = tap_of(i, 4);
                            const uint32_t a_tap = a_base + (uint32_t)(((tap / 3) * HT_PW + tap % 3) * BK * 2);
                            const uint32_t b_base = b0 + (uint32_t)halo_bres_off<BN>(i);
#pragma unroll
                            for (int k16 = 0; k16 < BK / 16; ++k16) {
                                const uint64_t ad = smem_desc_sw128_sbo(a_tap + k16 * 32, HT_ROW);
                                const uint64_t bd = smem_desc_sw128(b_base + k16 * 32);
                                const uint32_t acc = (cb > 0 || i > 0 || k16 > 0) ? 1u : 0u;
                                umma_f16(d, ad, bd, (ct_here && i == 0) ? id_merged : id_main, acc);
                            }
                        }
                        umma_commit(smem_u32(&a_empty[as]));
                    }
                    __syncwarp();
                    ++ai;
                } else {
                for (int i = 0; i < 9; ++i) {
                    const int bs = BRES ? i : bi % NBS;
                    const uint32_t bph = BRES ? 0u : (uint32_t)(bi / NBS) & 1u;
                    if (!warp_wait(smem_u32(&b_full[bs]), bph, a.err, 2u)) { ok = false; break; }
                    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                    const int tap = tap_of(i, 4);
                    const uint32_t a_tap = a_base + (uint32_t)(((tap / 3) * HT_PW + tap % 3) * BK * 2);
                    const uint32_t b_base = smem_u32(Bs + bs * B_STAGE);
                    const bool merged = ct_here && i == 0;
                    if (elect_one()) {
#pragma unroll
                        for (int k16 = 0; k16 < BK / 16; ++k16) {
                            const uint64_t ad = smem_desc_sw128_sbo(a_tap + k16 * 32, HT_ROW);
                            const uint64_t bd = smem_desc_sw128(b_base + k16 * 32);
                            const uint32_t acc = (cb > 0 || i > 0 || k16 > 0) ? 1u : 0u;
                            umma_f16(d, ad, bd, merged ? id_merged : id_main, acc);
                        }
                        if (!BRES) umma_commit(smem_u32(&b_empty[bs]));
                    }
                    __syncwarp();
                    if (!BRES) ++bi;
                }
                if (!ok) break;
                if (elect_one()) umma_commit(smem_u32(&a_empty[as]));
                __syncwarp();
                ++ai;
                }
            }
            if (!ok) break;
            if (elect_one()) umma_commit(smem_u32(&acc_full[ab]));   // fires when the tile's MMAs have completed
            __syncwarp();
        }
        if (!ok && lane == 0) *abort_flag = 1;
    } else {
        // ---------------- epilogue: warps 2..9 ----------------
        const int ep = warp - 2;
        const int quad = warp & 3;
        const int half = ep >> 2;
        const int row = quad * 32 + lane;
        const __half *x = static_cast<const __half *>(a.x);
        const FaultDelta fd = a.fd;
        const bool has_res = hg.res != 0, relu = a.relu != 0;
        // one N tile: this thread's channels are the same in every tile
        constexpr int NBIAS = BN <= 64 ? BN / 32 : 1;
        Bias16 bias_r[NBIAS];
#pragma unroll
        for (int c = 0; c < NBIAS; ++c) bias_r[c] = load_bias16(a.bias, half * (BN / 2) + 16 * c);
        int lt = 0;
        for (int tile = blockIdx.x; tile < num_tiles; tile += gridDim.x, ++lt) {
            const HaloTile ht = halo_tile(tile, hg);
            const int ab = lt & 1;
            const int p = ht.y0 + row / HT_TW, q = ht.x0 + row % HT_TW;
            const bool valid = p < hg.H && q < hg.W;
            const int m = valid ? (ht.n * hg.H + p) * hg.W + q : 0;
            const int n0 = ht.nt * BN + half * (BN / 2);
            const bool do_cs = half == 0 && a.cs_out != nullptr && ht.nt == 0;
            bool ok = mbar_wait(smem_u32(&acc_full[ab]), (uint32_t)(lt >> 1) & 1u, a.err, 4u) && !*abort_flag;
            const int rsl = lt % NR;
            if (ring) ok = ok && mbar_wait(smem_u32(&r_full[rsl]), (uint32_t)(lt / NR) & 1u, a.err, 4u);
            ok = __all_sync(0xffffffffu, ok);
            if (!ok) break;
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            const uint32_t trow = tmem + (uint32_t)(ab * CH) + ((uint32_t)(quad * 32) << 16);
            // all of the tile's TMEM loads in flight, one wait
            float vals[BN / 2];
            uint32_t rr[BN / 32][16], rc = 0;
            const bool want_ct = do_cs && hg.ct;                      // warp-uniform
#pragma unroll
            for (int c = 0; c < BN / 2; c += 16) tmem_ld16_nw(trow + half * (BN / 2) + c, rr[c / 16]);
            if (want_ct) tmem_ld1_nw(trow + BN, rc);
            tmem_wait_ld();
#pragma unroll
            for (int c = 0; c < BN / 2; c += 16) tmem_done16(rr[c / 16], vals + c);
            const float ctv = want_ct ? tmem_done(rc) : 0.f;
            asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&acc_empty[ab]));
            // epilogue operands from the R ring
            const uint8_t *rst = Rs + rsl * R::STAGE;
            Res16 rs[BN / 32];
#pragma unroll
            for (int c = 0; c < BN / 32; ++c) {
                if (hg.res) {
                    // channels ch .. ch + 15: 64-channel block ch / 64, chunks (ch % 64) / 8 and the next
                    const int ch = half * (BN / 2) + 16 * c;
                    const uint8_t *rrow = rst + (ch / 64) * 128 * 128 + row * 128;
                    const int ck = (ch % 64) / 8, sw = row & 7;
                    rs[c].r0 = *reinterpret_cast<const uint4 *>(rrow + ((ck ^ sw) << 4));
                    rs[c].r1 = *reinterpret_cast<const uint4 *>(rrow + (((ck + 1) ^ sw) << 4));
                } else {
                    rs[c].r0 = rs[c].r1 = make_uint4(0u, 0u, 0u, 0u);
                }
            }
            CsIn csv{0.f, 0, 0};
            if (do_cs) {
                if (hg.csin) csv.cin_h = reinterpret_cast<const unsigned short *>(rst + R::RES)[row];
                if (hg.rescs) csv.rcs_h = reinterpret_cast<const unsigned short *>(rst + R::RES + R::CS)[row];
            }
            if (ring) {
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(&r_empty[rsl]));
            }
            if (POOL) {
                // every lane computes its pixel (the shuffles need the whole warp);
                // the window's top-left lane stores the pooled pixel
                float fsrc = 0.f;
                if (fd.active && valid) {
                    const int h = p + fd.r - 1, w = q + fd.s - 1;
                    if (h >= 0 && h < hg.H && w >= 0 && w < hg.W) {
                        if (fd.cin < hg.C) fsrc = ldh(x, (((size_t)ht.n * hg.H + h) * hg.W + w) * hg.C + fd.cin);
                        else if (a.cs_in) fsrc = ldh(static_cast<const __half *>(a.cs_in), ((size_t)ht.n * hg.H + h) * hg.W + w);
                    }
                }
                const bool writer = valid && (row & 1) == 0 && (row & 8) == 0;
                const size_t mp = ((size_t)ht.n * (hg.H / 2) + p / 2) * (hg.W / 2) + q / 2;
#pragma unroll
                for (int c = 0; c < BN / 2; c += 16) {
                    float t[16];
                    epi16_vals(vals + c, BN <= 64 ? bias_r[(c / 16) % NBIAS] : load_bias16(a.bias, n0 + c), rs[c / 16],
                               has_res, relu, fd, n0 + c, fsrc, t);
                    uint32_t pk[8];
#pragma unroll
                    for (int i = 0; i < 8; ++i)
                        pk[i] = cvt_h2(pool2x2_lanes(t[2 * i]), pool2x2_lanes(t[2 * i + 1]), false);
                    if (writer) st_global_v8(static_cast<__half *>(a.y) + mp * hg.K + n0 + c, pk);
                }
                if (do_cs) {
                    const float o = pool2x2_lanes(checksum_value(ctv, csv, a, g, fsrc));
                    if (writer) static_cast<__half *>(a.cs_out)[mp] = __float2half_rn(o);
                }
            } else if (valid) {
                float fsrc = 0.f;
                if (fd.active) {
                    const int h = p + fd.r - 1, w = q + fd.s - 1;
                    if (h >= 0 && h < hg.H && w >= 0 && w < hg.W) {
                        if (fd.cin < hg.C) fsrc = ldh(x, (((size_t)ht.n * hg.H + h) * hg.W + w) * hg.C + fd.cin);
                        else if (a.cs_in) fsrc = ldh(static_cast<const __half *>(a.cs_in), ((size_t)ht.n * hg.H + h) * hg.W + w);
                    }
                }
                if (fd.active) {
#pragma unroll
                    for (int c = 0; c < BN / 2; c += 16)
                        store_chunk_pre(vals + c, rs[c / 16], a, hg.K, (size_t)m, n0 + c, fsrc);
                } else {
                    __half *yrow = static_cast<__half *>(a.y) + (size_t)m * hg.K + n0;
#pragma unroll
                    for (int c = 0; c < BN / 2; c += 16)
                        store16_fast(vals + c, BN <= 64 ? bias_r[(c / 16) % NBIAS] : load_bias16(a.bias, n0 + c),
                                     rs[c / 16], has_res, relu, yrow + c);
                }
                if (do_cs) store_checksum_pre(ctv, csv, a, g, m, fsrc);
            }
        }
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (warp == 1) {
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"((uint32_t)hg.tmem_cols));
    }
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------

PFN_cuTensorMapEncodeTiled_v12000 g_encode_tiled = nullptr;
PFN_cuTensorMapEncodeIm2col_v12000 g_encode_im2col = nullptr;
std::once_flag g_once;

bool load_encoders() {
    std::call_once(g_once, [] {
        cudaDriverEntryPointQueryResult q;
        void *p = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess && q == cudaDriverEntryPointSuccess)
            g_encode_tiled = (PFN_cuTensorMapEncodeTiled_v12000)p;
        p = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeIm2col", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess && q == cudaDriverEntryPointSuccess)
            g_encode_im2col = (PFN_cuTensorMapEncodeIm2col_v12000)p;
    });
    return g_encode_tiled && g_encode_im2col;
}

template <int BN, int STAGES, int SUB>
size_t smem_bytes() {
    return 1024 + (size_t)STAGES * SUB * (A_BYTES + (BN + 16) * BK * 2) + 16 * BK * 2 + 2 * BM * 4 +
           8 * (2 * STAGES + 6) + 16 + 16 + 4 * BIAS_SMEM;
}

uint16_t coef_half_bits(float c) {
    __half h = __float2half_rn(c);        // exact: coefficients are powers of two
    uint16_t b;
    memcpy(&b, &h, 2);
    return b;
}

int sm_count() { return device_sm_count(); }

}  // namespace

int device_sm_count() {
    int dev = 0, n = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n < 1)
        return 148;
    return n;
}

struct TcPlan {
    CUtensorMap amap;
    CUtensorMap bmap;
    TcGeom g;
    int BN, n_tiles, sms;
    size_t smem;
    CUtensorMap bmap_pair;       // N = 256 over CTA pairs: 128-row weight halves
    CUtensorMap bmap_pair64;     // 128-channel half tiles: 64-row weight quarters
    int pair_clusters;           // resident CTA pairs (0: no pair variant)
    size_t pair_smem;
    // launches that also run a shortcut: splits of the shortcut's items
    // for the last few batch sizes (batch, items, s0, x; batch 0: empty)
    int sc_cache[8][4];
    int sc_next;
};

bool tc_supported(int C, int K, int R, int S, int stride, int pad, std::string *why) {
    if (C % BK != 0) { if (why) *why = "input channels not a multiple of 64"; return false; }
    if (!(K == 64 || K == 128 || K % 256 == 0)) { if (why) *why = "output channels"; return false; }
    if (R != S || R > 7 || stride < 1 || stride > 2 || pad > 3 || pad > R / 2 + 1) {
        if (why) *why = "filter geometry";
        return false;
    }
    return true;
}

TcPlan *tc_plan_create(const ConvArgs &a, int max_batch, const void *w_dev, const void *x_dev, std::string *why) {
    if (!load_encoders()) { if (why) *why = "tensor-map encoders unavailable"; return nullptr; }
    TcPlan *pl = new TcPlan();
    memset(pl, 0, sizeof(*pl));
    pl->BN = a.K <= 256 ? a.K : 256;
    pl->n_tiles = a.K / pl->BN;
    pl->sms = sm_count();
    TcGeom &g = pl->g;
    g.PQ = a.P * a.Q; g.Q = a.Q; g.stride = a.stride; g.pad = a.pad; g.C = a.C; g.K = a.K;
    g.RSC = a.R * a.S * a.C; g.S = a.S;
    g.cpb = a.C / BK;
    g.n_kb = a.R * a.S * g.cpb;
    g.ctr_tap = ((a.R - 1) / 2) * a.S + (a.S - 1) / 2;
    g.ct_mode = a.role != CT_ROLE_CT ? CT_NONE_ : (pl->BN + 16 <= 256 && pl->n_tiles == 1 ? CT_MERGED : CT_SEPARATE);
    g.tmem_cols = 512;
    g.n_tiles = pl->n_tiles;
    g.coef_h = coef_half_bits(a.coef);
    // A: im2col view of the NHWC input [max_batch, H, W, C]
    cuuint64_t gdim[4] = {(cuuint64_t)a.C, (cuuint64_t)a.W, (cuuint64_t)a.H, (cuuint64_t)max_batch};
    cuuint64_t gstr[3] = {(cuuint64_t)a.C * 2, (cuuint64_t)a.W * a.C * 2, (cuuint64_t)a.H * a.W * a.C * 2};
    int lower[2] = {-a.pad, -a.pad};
    int upper[2] = {a.pad - (a.S - 1), a.pad - (a.R - 1)};
    cuuint32_t estr[4] = {1, (cuuint32_t)a.stride, (cuuint32_t)a.stride, 1};
    // a strided 1x1 convolution reads every other pixel: 256-byte L2
    // promotion would also fetch the pixels it skips (64 channels = 128 bytes)
    const CUtensorMapL2promotion apromo =
        (a.R == 1 && a.stride > 1) ? CU_TENSOR_MAP_L2_PROMOTION_L2_128B : CU_TENSOR_MAP_L2_PROMOTION_L2_256B;
    CUresult r = g_encode_im2col(&pl->amap, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 4, const_cast<void *>(x_dev), gdim, gstr,
                                 lower, upper, BK, BM, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                                 CU_TENSOR_MAP_SWIZZLE_128B, apromo, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) { if (why) *why = "im2col tensor map"; delete pl; return nullptr; }
    // B: weights [K, R*S*C] fp16, K-major rows
    cuuint64_t bdim[2] = {(cuuint64_t)g.RSC, (cuuint64_t)a.K};
    cuuint64_t bstr[1] = {(cuuint64_t)g.RSC * 2};
    cuuint32_t box[2] = {BK, (cuuint32_t)pl->BN};
    cuuint32_t bes[2] = {1, 1};
    r = g_encode_tiled(&pl->bmap, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void *>(w_dev), bdim, bstr, box, bes,
                       CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                       CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) { if (why) *why = "weight tensor map"; delete pl; return nullptr; }
    cudaError_t e;
    if (pl->BN == 64) {
        pl->smem = smem_bytes<64, 4, 2>();
        e = cudaFuncSetAttribute(conv_tc_kernel<64, 4, 2, 4, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)pl->smem);
    } else if (pl->BN == 128) {
        pl->smem = smem_bytes<128, 3, 2>();
        e = cudaFuncSetAttribute(conv_tc_kernel<128, 3, 2, 1, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)pl->smem);
        if (e == cudaSuccess)
            e = cudaFuncSetAttribute(conv_tc_kernel<128, 3, 2, 1, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)pl->smem);
    } else {
        pl->smem = smem_bytes<256, 4, 1>();
        e = cudaFuncSetAttribute(conv_tc_kernel<256, 4, 1, 1, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)pl->smem);
    }
    if (e != cudaSuccess) { if (why) *why = "shared memory attribute"; delete pl; return nullptr; }
    // N = 256 over CTA pairs (cta_group::2): each CTA copies half of the
    // tile's weight rows.  (128-channel layers stay on the single-CTA
    // kernel: on CTA pairs they ran 10-30% slower, measured.)
    pl->pair_clusters = 0;
    if (pl->BN == 256) {
        cuuint32_t box_h[2] = {BK, (cuuint32_t)BM};
        r = g_encode_tiled(&pl->bmap_pair, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void *>(w_dev), bdim, bstr,
                           box_h, bes, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                           CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
        cuuint32_t box_q[2] = {BK, (cuuint32_t)(BM / 2)};
        if (r == CUDA_SUCCESS)
            r = g_encode_tiled(&pl->bmap_pair64, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void *>(w_dev), bdim,
                               bstr, box_q, bes, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                               CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
        pl->pair_smem = pair_smem_bytes();
        cudaError_t pe = cudaSuccess;
        for (auto kern : {conv_tc_pair_kernel<false, false>, conv_tc_pair_kernel<true, false>,
                          conv_tc_pair_kernel<false, true>, conv_tc_pair_kernel<true, true>})
            if (pe == cudaSuccess)
                pe = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)pl->pair_smem);
        if (r == CUDA_SUCCESS && pe == cudaSuccess) {
            cudaLaunchConfig_t cfg = {};
            cfg.gridDim = dim3(2 * 64);
            cfg.blockDim = dim3(PR_THREADS);
            cfg.dynamicSmemBytes = pl->pair_smem;
            cudaLaunchAttribute at[1];
            at[0].id = cudaLaunchAttributeClusterDimension;
            at[0].val.clusterDim.x = 2;
            at[0].val.clusterDim.y = 1;
            at[0].val.clusterDim.z = 1;
            cfg.attrs = at;
            cfg.numAttrs = 1;
            int n = 0;
            if (cudaOccupancyMaxActiveClusters(&n, conv_tc_pair_kernel<false, false>, &cfg) == cudaSuccess && n > 0)
                pl->pair_clusters = n;
        }
        cudaGetLastError();
    }
    return pl;
}

namespace {

// Estimated cost of a work unit, in K-block times: its K blocks or, when
// more, the time its epilogue takes to store the tile (measured by clock
// traces: about 4 K blocks for a 128 x 128 tile, 12 for the 256 x 256 tile
// of a CTA pair), plus one for the accumulator hand-over.
constexpr double EPI_KB_SINGLE = 4.0, EPI_KB_PAIR = 12.0, UNIT_OVERHEAD_KB = 1.0;
double unit_cost(double kb, double epi) { return std::max(kb, epi) + UNIT_OVERHEAD_KB; }

// Split of the shortcut's n2 items (UnitSeq: CTAs 0 .. s0 - 1 share items
// 0 .. x - 1, the others the rest) that minimises the largest estimated
// load, given each CTA's load of the first layer's units and the cost c2
// of one shortcut item.  s0 is tried at the CTAs where that load changes
// (round-robin units give a few levels) and at both ends; for each, the
// best x balances the two groups' largest loads (the first grows with x,
// the second shrinks).
struct ScSplit {
    int s0, x;
};
ScSplit shortcut_split(const std::vector<double> &load, int n2, double c2) {
    const int ncl = (int)load.size();
    auto share = [&](int c, int s0, int x) -> long long {
        if (c < s0) return (c + 1) * (long long)x / s0 - c * (long long)x / s0;
        const long long nc = ncl - s0, r = n2 - x;
        return (c - s0 + 1) * r / nc - (c - s0) * r / nc;
    };
    auto group_max = [&](int c_lo, int c_hi, int s0, int x) {
        double mx = 0.0;
        for (int c = c_lo; c < c_hi; ++c) mx = std::max(mx, load[c] + (double)share(c, s0, x) * c2);
        return mx;
    };
    ScSplit best{0, 0};
    double best_max = 1e300;
    for (int s0 = 0; s0 <= ncl; ++s0) {
        if (s0 > 0 && s0 < ncl && load[s0] == load[s0 - 1]) continue;
        int x = s0 == 0 ? 0 : n2;
        if (s0 > 0 && s0 < ncl) {
            int lo = 0, hi = n2;
            while (lo < hi) {
                const int mid = (lo + hi) / 2;
                if (group_max(0, s0, s0, mid) >= group_max(s0, ncl, s0, mid)) hi = mid;
                else lo = mid + 1;
            }
            x = lo;
        }
        for (int xc = x; xc >= std::max(0, x - 1); --xc) {
            if ((s0 == 0 && xc != 0) || (s0 == ncl && xc != n2)) continue;
            const double mx = std::max(group_max(0, s0, s0, xc), group_max(s0, ncl, s0, xc));
            if (mx < best_max) {
                best_max = mx;
                best = ScSplit{s0, xc};
            }
        }
    }
    return best;
}

// The split for (batch, n2) from the plan's cache, else made by make() and
// cached (the oldest of the entries is replaced).
template <typename F>
ScSplit cached_split(TcPlan *pl, int batch, int n2, F &&make) {
    for (auto &e : pl->sc_cache)
        if (e[0] == batch && e[1] == n2) return ScSplit{e[2], e[3]};
    const ScSplit sp = make();
    int *e = pl->sc_cache[pl->sc_next];
    pl->sc_next = (pl->sc_next + 1) % 8;
    e[0] = batch;
    e[1] = n2;
    e[2] = sp.s0;
    e[3] = sp.x;
    return sp;
}

// Geometry of one launch of plan pl: output tiles, K split, CTA pairs.
TcGeom tc_launch_geom(const ConvArgs &a, const TcPlan *pl, bool *pairs) {
    TcGeom g = pl->g;
    g.M = a.N * a.P * a.Q;
    g.m_tiles = (g.M + BM - 1) / BM;
    const int tiles = g.m_tiles * g.n_tiles;
    // split K when the output tiles leave most SMs idle (at least 4 K blocks
    // per split; about half the SMs busy: more splits cost more in partial
    // sums than they gain, measured on 4-16 image batches)
    g.ws_ld = (g.K + 1 + 3) & ~3;
    g.splits = (a.K % 8 == 0) ? splitk_choose(tiles, g.n_kb, 4, pl->sms / 2, g.M, g.ws_ld, a.ws ? a.ws_bytes : 0) : 1;
    g.kps = (g.n_kb + g.splits - 1) / g.splits;
    g.sc_items = 0;
    g.sc_s0 = 0;
    g.sc_x = 0;
    *pairs = pl->pair_clusters > 0 && g.splits == 1 && g.m_tiles >= 2;
    return g;
}

}  // namespace

bool tc_shortcut_fits(const ConvArgs &a, const void *plan, const void *plan2) {
    const TcPlan *pl = static_cast<const TcPlan *>(plan);
    const TcPlan *pl2 = static_cast<const TcPlan *>(plan2);
    if (!pl || !pl2) return false;
    bool pairs = false;
    const TcGeom g = tc_launch_geom(a, pl, &pairs);
    // both layers whole (unsplit) N = 128 tiles on single CTAs, or N = 256
    // tiles on CTA pairs; the shortcut's K blocks are the centre tap's
    return g.splits == 1 && pl2->BN == pl->BN && pl2->n_tiles == pl->n_tiles && pl2->g.n_kb == pl->g.cpb &&
           ((pl->BN == 128 && !pairs) || (pl->BN == 256 && pairs));
}

cudaError_t launch_conv_tc(const ConvArgs &a, const void *plan, cudaStream_t st, int *n_kernels, const ConvArgs *a2,
                           const void *plan2, bool *merged) {
    TcPlan *pl = static_cast<TcPlan *>(const_cast<void *>(plan));
    const TcPlan *pl2 = static_cast<const TcPlan *>(plan2);
    if (merged) *merged = false;
    bool pairs = false;
    TcGeom g = tc_launch_geom(a, pl, &pairs);
    const int tiles = g.m_tiles * g.n_tiles;
    // a 1x1 shortcut of the same input (a2, plan2) joins this launch when the
    // tiles allow; the caller launches it on its own otherwise
    const bool sc = a2 && tc_shortcut_fits(a, plan, plan2);
    TcGeom g2 = sc ? pl2->g : g;
    if (sc) {
        g2.M = g.M;
        g2.m_tiles = g.m_tiles;
        g2.ws_ld = g.ws_ld;
        g2.splits = 1;
        g2.kps = g2.n_kb;
        g2.t_first = g2.units = 0;
        g2.sc_items = g2.sc_s0 = g2.sc_x = 0;
    }
    const ConvArgs &b = sc ? *a2 : a;
    const CUtensorMap &bm2 = sc ? (pairs ? pl2->bmap_pair : pl2->bmap) : (pairs ? pl->bmap_pair : pl->bmap);
    if (pairs) {
        // tiles over CTA pairs: 256 pixels x 256 channels per pair
        const int items = ((g.m_tiles + 1) / 2) * g.n_tiles;
        const int P = pl->pair_clusters;
        // last round of 256-channel tiles: rem tiles on P pairs; as 2 * rem
        // half tiles when they fit in one round (it then takes half a tile time)
        const int rem = items % P;
        const bool halves = rem > 0 && 2 * rem <= P;
        g.t_first = halves ? items - rem : items;
        g.units = halves ? items + rem : items;
        const int n2 = sc ? ((g.m_tiles + 1) / 2) * g2.n_tiles : 0;
        const int ncl = g.units + n2 < P ? g.units + n2 : P;
        if (sc) {
            g.sc_items = n2;
            const ScSplit sp = cached_split(pl, a.N, n2, [&] {
                std::vector<double> load(ncl, 0.0);
                for (int u = 0; u < g.units; ++u) {
                    const bool narrow = halves && u < g.units - g.t_first;
                    // a 128-channel half costs ~0.92 of a whole tile's K block (measured)
                    load[u % ncl] += unit_cost((narrow ? 0.92 : 1.0) * g.n_kb, EPI_KB_PAIR);
                }
                return shortcut_split(load, n2, unit_cost(g2.n_kb, EPI_KB_PAIR));
            });
            g.sc_s0 = sp.s0;
            g.sc_x = sp.x;
        }
        if (halves && sc)
            pdl_launch_cluster(conv_tc_pair_kernel<true, true>, dim3(2 * ncl), PR_THREADS, pl->pair_smem, st, 2,
                               pl->amap, pl->bmap_pair, pl->bmap_pair64, a, g, bm2, b, g2);
        else if (sc)
            pdl_launch_cluster(conv_tc_pair_kernel<false, true>, dim3(2 * ncl), PR_THREADS, pl->pair_smem, st, 2,
                               pl->amap, pl->bmap_pair, pl->bmap_pair64, a, g, bm2, b, g2);
        else if (halves)
            pdl_launch_cluster(conv_tc_pair_kernel<true, false>, dim3(2 * ncl), PR_THREADS, pl->pair_smem, st, 2,
                               pl->amap, pl->bmap_pair, pl->bmap_pair64, a, g, bm2, b, g2);
        else
            pdl_launch_cluster(conv_tc_pair_kernel<false, false>, dim3(2 * ncl), PR_THREADS, pl->pair_smem, st, 2,
                               pl->amap, pl->bmap_pair, pl->bmap_pair64, a, g, bm2, b, g2);
    } else {
        const int items = tiles * g.splits;
        const int n2 = sc ? g2.m_tiles * g2.n_tiles : 0;
        const int ncl = items + n2 < pl->sms ? items + n2 : pl->sms;
        dim3 grid(ncl);
        if (sc) {
            g.sc_items = n2;
            const ScSplit sp = cached_split(pl, a.N, n2, [&] {
                std::vector<double> load(ncl, 0.0);
                for (int u = 0; u < items; ++u) load[u % ncl] += unit_cost(g.n_kb, EPI_KB_SINGLE);
                return shortcut_split(load, n2, unit_cost(g2.n_kb, EPI_KB_SINGLE));
            });
            g.sc_s0 = sp.s0;
            g.sc_x = sp.x;
            pdl_launch(conv_tc_kernel<128, 3, 2, 1, true>, grid, tc_threads(128, 3), pl->smem, st, pl->amap, pl->bmap,
                       a, g, bm2, b, g2);
        } else if (pl->BN == 64) {
            pdl_launch(conv_tc_kernel<64, 4, 2, 4, false>, grid, tc_threads(64, 4), pl->smem, st, pl->amap, pl->bmap, a,
                       g, bm2, b, g2);
        } else if (pl->BN == 128) {
            pdl_launch(conv_tc_kernel<128, 3, 2, 1, false>, grid, tc_threads(128, 3), pl->smem, st, pl->amap, pl->bmap,
                       a, g, bm2, b, g2);
        } else {
            pdl_launch(conv_tc_kernel<256, 4, 1, 1, false>, grid, tc_threads(256, 4), pl->smem, st, pl->amap, pl->bmap,
                       a, g, bm2, b, g2);
        }
    }
    cudaError_t e = cudaGetLastError();
    if (n_kernels) *n_kernels = 1;
    if (e == cudaSuccess && merged) *merged = sc;
    if (e != cudaSuccess || g.splits == 1) return e;
    if (n_kernels) *n_kernels = 2;
    return launch_splitk_reduce(a, g.splits, g.ws_ld, true, st);
}

bool tc_small_supported(int C, int K, int R, int S, int stride, int pad) {
    return C >= 1 && C <= 4 && K == SM_BN && R == S && R <= 7 && stride >= 1 && stride <= 2 && pad <= 3;
}

int tc_small_kpad(int R, int S) { return ((R * S * 4 + BK - 1) / BK) * BK; }

struct TcSmallPlan {
    CUtensorMap bmap;
    TcGeomS g;
    int sms;
    size_t smem;
};

TcSmallPlan *tc_small_plan_create(const ConvArgs &a, const void *w_dev, std::string *why) {
    if (!load_encoders()) { if (why) *why = "tensor-map encoders unavailable"; return nullptr; }
    TcSmallPlan *pl = new TcSmallPlan();
    memset(pl, 0, sizeof(*pl));
    pl->sms = sm_count();
    TcGeomS &g = pl->g;
    g.PQ = a.P * a.Q; g.Q = a.Q; g.stride = a.stride; g.pad = a.pad; g.C = a.C;
    g.H = a.H; g.W = a.W; g.R = a.R; g.S = a.S;
    const int kp = tc_small_kpad(a.R, a.S);
    g.n_kb = kp / BK;
    const int ctr_tap = ((a.R - 1) / 2) * a.S + (a.S - 1) / 2;
    g.kb_ct = (ctr_tap * 4) / BK;
    g.col_ct = (ctr_tap * 4) % BK;
    g.ct = a.role == CT_ROLE_CT ? 1 : 0;
    g.tmem_cols = 512;
    g.coef_h = coef_half_bits(a.coef);
    cuuint64_t bdim[2] = {(cuuint64_t)kp, (cuuint64_t)SM_BN};
    cuuint64_t bstr[1] = {(cuuint64_t)kp * 2};
    cuuint32_t box[2] = {BK, (cuuint32_t)SM_BN};
    cuuint32_t bes[2] = {1, 1};
    CUresult r = g_encode_tiled(&pl->bmap, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void *>(w_dev), bdim, bstr,
                                box, bes, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                                CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) { if (why) *why = "weight tensor map"; delete pl; return nullptr; }
    pl->smem = 1024 + (size_t)SM_STAGES * (A_BYTES + (SM_BN + 16) * BK * 2) + 8 * (2 * SM_STAGES + 2) + 16;
    if (cudaFuncSetAttribute(conv_tc_small_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)pl->smem) !=
        cudaSuccess) {
        if (why) *why = "shared memory attribute";
        delete pl;
        return nullptr;
    }
    return pl;
}

void tc_small_plan_destroy(TcSmallPlan *p) { delete p; }

cudaError_t launch_conv_tc_small(const ConvArgs &a, const TcSmallPlan *pl, cudaStream_t st) {
    TcGeomS g = pl->g;
    g.M = a.N * a.P * a.Q;
    g.m_tiles = (g.M + BM - 1) / BM;
    dim3 grid(g.m_tiles < pl->sms ? g.m_tiles : pl->sms);
    pdl_launch(conv_tc_small_kernel, grid, SM_THREADS, pl->smem, st, pl->bmap, a, g);
    return cudaGetLastError();
}

void tc_plan_destroy(TcPlan *p) { delete p; }

// ---------------------------------------------------------------------------
// halo-tile plans
// ---------------------------------------------------------------------------
struct HaloPlan {
    HaloMaps maps;
    HaloGeom hg;
    TcGeom g;
    int BN, kind, pool, sms;
    size_t smem;
    const void *res, *csin, *rescs;   // tensors the R-ring maps point at
};

template <int BN, bool BRES, int NA, int NB, int NR, bool POOL>
size_t halo_smem() {
    const int nbs = BRES ? 9 : NB;
    const size_t b_area = BRES ? (size_t)halo_bres_off<BN>(9) : (size_t)NB * (BN + 16) * BK * 2;
    return 1024 + (size_t)NA * HT_A_STAGE + b_area + (size_t)NR * HaloR<BN>::STAGE +
           8 * (2 * NA + 2 * nbs + 2 * NR + 4) + 16;
}

// halo kernel variants <BN, resident weights, patch stages, weight stages,
// operand-ring stages>; each also with the fused 2 x 2 max-pool
#define HK0 64, true, 4, 0, 3
#define HK1 64, false, 3, 6, 3
#define HK2 128, false, 3, 4, 2

// Tiles that overhang the image waste MMA rows: require whole 8-column tiles
// and at most one partly filled row of tiles on a tall image.
bool halo_supported(int C, int K, int R, int S, int stride, int pad, int H, int W) {
    return R == 3 && S == 3 && stride == 1 && pad == 1 && C % BK == 0 && (K == 64 || K == 128) && W % HT_TW == 0 &&
           (H % HT_TH == 0 || H >= 3 * HT_TH);
}

static bool encode_plane_map(CUtensorMap *map, const void *plane, int N, int H, int W) {
    // [N, H, W] fp16 plane as boxes of 8 x 16 pixels
    cuuint64_t dim[3] = {(cuuint64_t)W, (cuuint64_t)H, (cuuint64_t)N};
    cuuint64_t str[2] = {(cuuint64_t)W * 2, (cuuint64_t)H * W * 2};
    cuuint32_t box[3] = {HT_TW, HT_TH, 1};
    cuuint32_t es[3] = {1, 1, 1};
    return g_encode_tiled(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 3, const_cast<void *>(plane), dim, str, box, es,
                          CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_NONE,
                          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

HaloPlan *halo_plan_create(const ConvArgs &a, int max_batch, const void *w_dev, const void *x_dev, const void *res_dev,
                           const void *csin_dev, const void *rescs_dev, bool pool, std::string *why) {
    if (!halo_supported(a.C, a.K, a.R, a.S, a.stride, a.pad, a.H, a.W)) { if (why) *why = "shape"; return nullptr; }
    if (pool && (a.H % 2 || a.W % 2)) { if (why) *why = "pooled shape"; return nullptr; }
    if (!load_encoders()) { if (why) *why = "tensor-map encoders unavailable"; return nullptr; }
    HaloPlan *pl = new HaloPlan();
    memset(pl, 0, sizeof(*pl));
    pl->BN = a.K;
    pl->sms = sm_count();
    pl->res = res_dev; pl->csin = csin_dev; pl->rescs = rescs_dev;
    HaloGeom &hg = pl->hg;
    hg.H = a.H; hg.W = a.W; hg.C = a.C; hg.K = a.K;
    hg.ncb = a.C / BK;
    hg.n_tiles = 1;
    hg.ty_tiles = (a.H + HT_TH - 1) / HT_TH;
    hg.tx_tiles = (a.W + HT_TW - 1) / HT_TW;
    hg.ct = a.role == CT_ROLE_CT ? 1 : 0;
    hg.tmem_cols = 2 * (pl->BN + 16) <= 256 ? 256 : 512;
    hg.coef_h = coef_half_bits(a.coef);
    hg.res = res_dev != nullptr; hg.csin = csin_dev != nullptr; hg.rescs = rescs_dev != nullptr;
    // geometry the shared epilogue helpers read
    TcGeom &g = pl->g;
    g.PQ = a.P * a.Q; g.Q = a.Q; g.stride = 1; g.pad = 1; g.C = a.C; g.K = a.K; g.S = 3; g.ctr_tap = 4;
    // A: the NHWC input [max_batch, H, W, C] as tiles of 64 channels x 10 x 18 pixels
    cuuint64_t gdim[4] = {(cuuint64_t)a.C, (cuuint64_t)a.W, (cuuint64_t)a.H, (cuuint64_t)max_batch};
    cuuint64_t gstr[3] = {(cuuint64_t)a.C * 2, (cuuint64_t)a.W * a.C * 2, (cuuint64_t)a.H * a.W * a.C * 2};
    cuuint32_t abox[4] = {BK, HT_PW, HT_PH, 1};
    cuuint32_t aes[4] = {1, 1, 1, 1};
    CUresult r = g_encode_tiled(&pl->maps.amap, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 4, const_cast<void *>(x_dev), gdim,
                                gstr, abox, aes, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                                CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) { if (why) *why = "patch tensor map"; delete pl; return nullptr; }
    const int RSC = 9 * a.C;
    cuuint64_t bdim[2] = {(cuuint64_t)RSC, (cuuint64_t)a.K};
    cuuint64_t bstr[1] = {(cuuint64_t)RSC * 2};
    cuuint32_t box[2] = {BK, (cuuint32_t)pl->BN};
    cuuint32_t bes[2] = {1, 1};
    r = g_encode_tiled(&pl->maps.bmap, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void *>(w_dev), bdim, bstr, box,
                       bes, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                       CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) { if (why) *why = "weight tensor map"; delete pl; return nullptr; }
    if (res_dev) {
        // residual [max_batch, H, W, K]: boxes of 64 channels x 8 x 16 pixels, pixel-major, 128-byte swizzle
        cuuint64_t rdim[4] = {(cuuint64_t)a.K, (cuuint64_t)a.W, (cuuint64_t)a.H, (cuuint64_t)max_batch};
        cuuint64_t rstr[3] = {(cuuint64_t)a.K * 2, (cuuint64_t)a.W * a.K * 2, (cuuint64_t)a.H * a.W * a.K * 2};
        cuuint32_t rbox[4] = {64, HT_TW, HT_TH, 1};
        if (g_encode_tiled(&pl->maps.rmap, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 4, const_cast<void *>(res_dev), rdim, rstr,
                           rbox, aes, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                           CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS) {
            if (why) *why = "residual tensor map";
            delete pl;
            return nullptr;
        }
    }
    if ((csin_dev && !encode_plane_map(&pl->maps.cmap, csin_dev, max_batch, a.H, a.W)) ||
        (rescs_dev && !encode_plane_map(&pl->maps.qmap, rescs_dev, max_batch, a.H, a.W))) {
        if (why) *why = "checksum tensor map";
        delete pl;
        return nullptr;
    }
    cudaError_t e;
    pl->pool = pool ? 1 : 0;
    pl->kind = (pl->BN == 64 && hg.ncb == 1) ? 0 : pl->BN == 64 ? 1 : 2;
#define HALO_ATTR(P, ...)                                                                                        \
    (pl->smem = halo_smem<__VA_ARGS__, P>(),                                                                       \
     cudaFuncSetAttribute(conv_tc_halo_kernel<__VA_ARGS__, P>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)pl->smem))
    if (pl->kind == 0) e = pool ? HALO_ATTR(true, HK0) : HALO_ATTR(false, HK0);
    else if (pl->kind == 1) e = pool ? HALO_ATTR(true, HK1) : HALO_ATTR(false, HK1);
    else e = pool ? HALO_ATTR(true, HK2) : HALO_ATTR(false, HK2);
#undef HALO_ATTR
    if (e != cudaSuccess) { cudaGetLastError(); if (why) *why = "shared memory attribute"; delete pl; return nullptr; }
    return pl;
}

int halo_tiles(const HaloPlan *pl, int batch) { return batch * pl->hg.ty_tiles * pl->hg.tx_tiles * pl->hg.n_tiles; }
int halo_sms(const HaloPlan *pl) { return pl->sms; }

cudaError_t launch_conv_tc_halo(const ConvArgs &a, const HaloPlan *pl, cudaStream_t st) {
    // the R-ring maps were encoded for these tensors
    if (a.res != pl->res || (a.cs_out && a.cs_in != pl->csin) || (a.cs_out && a.res_cs != pl->rescs))
        return cudaErrorInvalidValue;
    HaloGeom hg = pl->hg;
    hg.N = a.N;
    if (!a.cs_out) hg.csin = hg.rescs = 0;
    TcGeom g = pl->g;
    g.M = a.N * a.P * a.Q;
    const int tiles = halo_tiles(pl, a.N);
    dim3 grid(tiles < pl->sms ? tiles : pl->sms);
#define HALO_LAUNCH(P, ...) \
    pdl_launch(conv_tc_halo_kernel<__VA_ARGS__, P>, grid, NTHREADS, pl->smem, st, pl->maps, a, hg, g)
    if (pl->kind == 0) pl->pool ? HALO_LAUNCH(true, HK0) : HALO_LAUNCH(false, HK0);
    else if (pl->kind == 1) pl->pool ? HALO_LAUNCH(true, HK1) : HALO_LAUNCH(false, HK1);
    else pl->pool ? HALO_LAUNCH(true, HK2) : HALO_LAUNCH(false, HK2);
#undef HALO_LAUNCH
    return cudaGetLastError();
}

void halo_plan_destroy(HaloPlan *p) { delete p; }

}  // namespace ct
