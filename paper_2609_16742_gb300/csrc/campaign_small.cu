// Whole-network kernel for small networks (the LeNet-5 shape), used two ways:
// inference of a batch (ct_infer on such a model: one launch instead of one
// per layer, with any armed fault applied inside the kernel), and the
// batched fault-injection campaign of Sec. III-A (ct_campaign_batched: one
// launch evaluates many single-bit faults).  CTA (f, y) runs fault f on images
// y * ipc .. y * ipc + ipc - 1 of a fixed batch through the whole protected
// network in shared memory: conv -> ReLU -> 2x2 max-pool -> conv -> ReLU ->
// 2x2 max-pool -> FC -> ReLU -> FC -> ReLU -> FC (the LeNet-5 shape), FP32,
// widened construction (checksum planes beside the data channels).
//
// Fault model as in ct_inject: a weight flip changes one stored word of a
// convolution (this CTA's shared-memory copy of the weights is flipped, so
// every CTA carries its own fault), or, for an element of the construction
// that is not stored (carry-through row, zero checksum slice), adds
// dv * source to one output channel in the epilogue; an activation flip
// changes one word of the second convolution's input (the first max-pool's
// output, checksum plane included) for one image, and only that image's CTA
// runs.  FC weights are never faulted and are read from global memory.
//
// Arithmetic follows the per-layer kernels: each convolution output is an
// FFMA chain over the K index (r, s, c) in that order, then + bias, fault
// delta, ReLU; the carry-through channel is coef * (sum of the centre-tap
// input channels + incoming checksum); max-pool propagates NaN; each FC
// neuron is a dot product (warp-parallel here, so its summation order
// differs from the FC kernel's), the carry-through neuron coef * (sum of
// data inputs + sum of checksum inputs); the verdict is NOT(|S - r| <= tau).
#include "ct_internal.h"

namespace ct {

namespace {

__device__ __forceinline__ float relu_nan(float v) { return v < 0.f ? 0.f : v; }
__device__ __forceinline__ void vmax_nan(float &m, float v) { m = (v > m || v != v) ? v : m; }

__device__ __forceinline__ float flip_f32(float v, int bit) {
    return __uint_as_float(__float_as_uint(v) ^ (1u << bit));
}

// warp dot product of w[0..n) and x[0..n); every lane returns the sum
__device__ __forceinline__ float warp_dot(const float *__restrict__ w, const float *x, int n, int lane) {
    float s = 0.f;
    for (int i = lane; i < n; i += 32) s = fmaf(__ldg(w + i), x[i], s);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    return s;
}

__device__ __forceinline__ float warp_sum(const float *x, int n, int lane) {
    float s = 0.f;
    for (int i = lane; i < n; i += 32) s += x[i];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    return s;
}

// shared-memory layout (floats), from the shapes
struct SmLayout {
    int w1, w2, img, a1, c1, p1, q1, a2, c2, p2, q2, f1, f2, f3, total;
};
__host__ __device__ inline SmLayout sm_layout(const SmallNet &g) {
    SmLayout L;
    int o = 0;
    auto take = [&](int n) { int at = o; o += (n + 3) & ~3; return at; };
    L.w1 = take(g.K1 * g.R1 * g.R1 * g.C0);
    L.w2 = take(g.K2 * g.R2 * g.R2 * g.K1);
    L.img = take(g.C0 * g.H0 * g.W0);
    L.a1 = take(g.K1 * g.H1 * g.W1);
    L.c1 = take(g.H1 * g.W1);
    L.p1 = take(g.K1 * g.Hp1 * g.Wp1);
    L.q1 = take(g.Hp1 * g.Wp1);
    L.a2 = take(g.K2 * g.H2 * g.W2);
    L.c2 = take(g.H2 * g.W2);
    L.p2 = take(g.NIN1);                 // NHWC flatten order: (h, w, c)
    L.q2 = take(g.Hp2 * g.Wp2);
    L.f1 = take(g.N1 + 1);               // data neurons, then the carry-through neuron
    L.f2 = take(g.N2 + 1);
    L.f3 = take(g.N3 + 1);               // logits, then S
    L.total = o;
    return L;
}

// faults == null: inference -- one fault, `single` (kind 2: none), and every
// image of the batch is computed (an activation fault changes only its
// image); rows B .. B + rr.n - 1 are the re-run list: image rr.idx[j] of
// rr.x, whose logits and S go to row rr.idx[j] of rr.logits / rr.S (no
// flag).  logits_out, top1_out may be null.  Without protection
// (g.protect == 0) no checksum channel or neuron is computed, S is NaN and
// the flag 0, as for the per-layer kernels.
__global__ void __launch_bounds__(1024) campaign_small_kernel(const SmallNet g, const CampFault *faults,
                                                               const CampFault single, int ipc, float *S_out,
                                                               int32_t *top1_out, uint8_t *flag_out, float *logits_out,
                                                               const SmallRerun rr) {
    pdl_wait();
    pdl_trigger();
    const CampFault f = faults ? faults[blockIdx.x] : single;
    const bool campaign = faults != nullptr;
    const int pc = g.protect ? 1 : 0;            // checksum channels / neurons
    const int n_lo = blockIdx.y * ipc, n_hi = min(g.B + (campaign ? 0 : rr.n), n_lo + ipc);
    // a campaign's activation fault: only the hit image's CTA works
    if (campaign && f.kind == 1 && (f.img < n_lo || f.img >= n_hi)) return;
    extern __shared__ __align__(16) float sm[];
    const SmLayout L = sm_layout(g);
    float *w1 = sm + L.w1, *w2 = sm + L.w2, *img = sm + L.img, *a1 = sm + L.a1, *c1 = sm + L.c1;
    float *p1 = sm + L.p1, *q1 = sm + L.q1, *a2 = sm + L.a2, *c2 = sm + L.c2, *p2 = sm + L.p2, *q2 = sm + L.q2;
    float *f1 = sm + L.f1, *f2 = sm + L.f2, *f3 = sm + L.f3;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int nw1 = g.K1 * g.R1 * g.R1 * g.C0, nw2 = g.K2 * g.R2 * g.R2 * g.K1;
    for (int i = tid; i < nw1; i += blockDim.x) w1[i] = g.w1[i];
    for (int i = tid; i < nw2; i += blockDim.x) w2[i] = g.w2[i];
    __syncthreads();
    if (tid == 0 && f.kind == 0 && f.word >= 0) {
        float *w = f.layer == 0 ? w1 : w2;
        w[f.word] = flip_f32(w[f.word], f.bit);
    }
    const bool fd1 = f.kind == 0 && f.layer == 0 && f.fd.active;
    const bool fd2 = f.kind == 0 && f.layer == 1 && f.fd.active;
    __syncthreads();
    const int n_first = (campaign && f.kind == 1) ? f.img : n_lo;
    const int n_last = (campaign && f.kind == 1) ? f.img + 1 : n_hi;
    const int ctr1 = (g.R1 - 1) / 2, ctr2 = (g.R2 - 1) / 2;
    const int HW0 = g.H0 * g.W0, HW1 = g.H1 * g.W1, HWp1 = g.Hp1 * g.Wp1, HW2 = g.H2 * g.W2, HWp2 = g.Hp2 * g.Wp2;
    for (int n = n_first; n < n_last; ++n) {
        // ---- image [C0][H0][W0] ----
        const bool rerun = n >= g.B;             // a row of the re-run list
        const int src_n = rerun ? rr.idx[n - g.B] : n;
        const float *xn = rerun ? rr.x + (size_t)src_n * g.C0 * HW0
                        : (g.x2 && n >= g.n_split) ? g.x2 + (size_t)(n - g.n_split) * g.C0 * HW0
                                                   : g.x + (size_t)n * g.C0 * HW0;
        for (int i = tid; i < g.C0 * HW0; i += blockDim.x) img[i] = __ldg(xn + i);
        __syncthreads();
        // ---- conv1 + ReLU, its carry-through channel ----
        for (int e = tid; e < (g.K1 + pc) * HW1; e += blockDim.x) {
            const int k = e / HW1, pq = e % HW1, p = pq / g.W1, q = pq % g.W1;
            float o;
            if (k < g.K1) {
                float acc = 0.f;
                const float *wk = w1 + k * g.R1 * g.R1 * g.C0;
                for (int r = 0; r < g.R1; ++r)
                    for (int s = 0; s < g.R1; ++s)
                        for (int c = 0; c < g.C0; ++c)
                            acc = fmaf(img[(c * g.H0 + p + r) * g.W0 + q + s], wk[(r * g.R1 + s) * g.C0 + c], acc);
                o = acc + __ldg(g.b1 + k);
            } else {
                float cs = 0.f;
                for (int c = 0; c < g.C0; ++c) cs += img[(c * g.H0 + p + ctr1) * g.W0 + q + ctr1];
                o = g.coef1 * cs;                       // the image carries no checksum
            }
            if (fd1 && f.fd.kout == k && f.fd.cin < g.C0)
                o += f.fd.dv * img[(f.fd.cin * g.H0 + p + f.fd.r) * g.W0 + q + f.fd.s];
            o = relu_nan(o);
            if (k < g.K1) a1[k * HW1 + pq] = o; else c1[pq] = o;
        }
        __syncthreads();
        // ---- 2x2 max-pool (data and checksum); an activation flip of this image ----
        for (int e = tid; e < (g.K1 + pc) * HWp1; e += blockDim.x) {
            const int k = e / HWp1, pq = e % HWp1, p = pq / g.Wp1, q = pq % g.Wp1;
            const float *src = k < g.K1 ? a1 + k * HW1 : c1;
            float mx = -INFINITY;
            for (int i = 0; i < 2; ++i)
                for (int j = 0; j < 2; ++j) vmax_nan(mx, src[(2 * p + i) * g.W1 + 2 * q + j]);
            if (f.kind == 1 && n == f.img && f.act_c == k && f.act_hw == pq) mx = flip_f32(mx, f.bit);
            if (k < g.K1) p1[k * HWp1 + pq] = mx; else q1[pq] = mx;
        }
        __syncthreads();
        // ---- conv2 + ReLU (the checksum input is skipped by data filters),
        // carry-through channel over data and checksum inputs ----
        for (int e = tid; e < (g.K2 + pc) * HW2; e += blockDim.x) {
            const int k = e / HW2, pq = e % HW2, p = pq / g.W2, q = pq % g.W2;
            float o;
            if (k < g.K2) {
                float acc = 0.f;
                const float *wk = w2 + k * g.R2 * g.R2 * g.K1;
                for (int r = 0; r < g.R2; ++r)
                    for (int s = 0; s < g.R2; ++s)
                        for (int c = 0; c < g.K1; ++c)
                            acc = fmaf(p1[(c * g.Hp1 + p + r) * g.Wp1 + q + s], wk[(r * g.R2 + s) * g.K1 + c], acc);
                o = acc + __ldg(g.b2 + k);
            } else {
                float cs = 0.f;
                for (int c = 0; c < g.K1; ++c) cs += p1[(c * g.Hp1 + p + ctr2) * g.Wp1 + q + ctr2];
                o = g.coef2 * (cs + q1[(p + ctr2) * g.Wp1 + q + ctr2]);
            }
            if (fd2 && f.fd.kout == k) {
                const int h = p + f.fd.r, w = q + f.fd.s;
                o += f.fd.dv * (f.fd.cin < g.K1 ? p1[(f.fd.cin * g.Hp1 + h) * g.Wp1 + w] : q1[h * g.Wp1 + w]);
            }
            o = relu_nan(o);
            if (k < g.K2) a2[k * HW2 + pq] = o; else c2[pq] = o;
        }
        __syncthreads();
        // ---- 2x2 max-pool into the FC input: data in (h, w, c) order, checksum plane ----
        for (int e = tid; e < (g.K2 + pc) * HWp2; e += blockDim.x) {
            const int k = e / HWp2, pq = e % HWp2, p = pq / g.Wp2, q = pq % g.Wp2;
            const float *src = k < g.K2 ? a2 + k * HW2 : c2;
            float mx = -INFINITY;
            for (int i = 0; i < 2; ++i)
                for (int j = 0; j < 2; ++j) vmax_nan(mx, src[(2 * p + i) * g.W2 + 2 * q + j]);
            if (k < g.K2) p2[pq * g.K2 + k] = mx; else q2[pq] = mx;
        }
        __syncthreads();
        // ---- FC1 + ReLU; carry-through neuron ----
        for (int j = warp; j < g.N1 + pc; j += blockDim.x / 32) {
            float o;
            if (j < g.N1) o = warp_dot(g.wf1 + (size_t)j * g.NIN1, p2, g.NIN1, lane) + __ldg(g.bf1 + j);
            else o = g.coeff1 * (warp_sum(p2, g.NIN1, lane) + warp_sum(q2, HWp2, lane));
            if (lane == 0) f1[j] = relu_nan(o);
        }
        __syncthreads();
        // ---- FC2 + ReLU; carry-through neuron ----
        for (int j = warp; j < g.N2 + pc; j += blockDim.x / 32) {
            float o;
            if (j < g.N2) o = warp_dot(g.wf2 + (size_t)j * g.N1, f1, g.N1, lane) + __ldg(g.bf2 + j);
            else o = g.coeff2 * (warp_sum(f1, g.N1, lane) + f1[g.N1]);
            if (lane == 0) f2[j] = relu_nan(o);
        }
        __syncthreads();
        // ---- classifier; accumulated-checksum neuron S ----
        for (int j = warp; j < g.N3 + pc; j += blockDim.x / 32) {
            float o;
            if (j < g.N3) o = warp_dot(g.wf3 + (size_t)j * g.N2, f2, g.N2, lane) + __ldg(g.bf3 + j);
            else o = g.coeff3 * (warp_sum(f2, g.N2, lane) + f2[g.N2]);
            if (lane == 0) f3[j] = o;
        }
        __syncthreads();
        const size_t o = (size_t)blockIdx.x * g.B + n;
        if (rerun) {
            for (int j = tid; j < g.N3; j += blockDim.x) rr.logits[(size_t)src_n * g.N3 + j] = f3[j];
            if (tid == 0 && rr.S) rr.S[src_n] = g.protect ? f3[g.N3] : __int_as_float(0x7fc00000);
            __syncthreads();
            continue;
        }
        if (logits_out)
            for (int j = tid; j < g.N3; j += blockDim.x) logits_out[o * g.N3 + j] = f3[j];
        if (tid == 0) {
            // top-1: a NaN logit gives -1; ties go to the lowest index
            int best = 0;
            bool nan = false;
            for (int j = 0; j < g.N3; ++j) {
                if (f3[j] != f3[j]) nan = true;
                else if (f3[j] > f3[best]) best = j;
            }
            const float S = g.protect ? f3[g.N3] : __int_as_float(0x7fc00000);
            if (S_out) S_out[o] = S;
            if (top1_out) top1_out[o] = nan ? -1 : best;
            const uint8_t fv = g.protect ? !(fabs((double)S - g.ref) <= g.tau) : 0;
            if (flag_out) flag_out[o] = fv;
            if (!campaign && g.flag2) g.flag2[n] = fv;
        }
        __syncthreads();
    }
}

}  // namespace

size_t campaign_small_smem(const SmallNet &g) { return sizeof(float) * (size_t)sm_layout(g).total; }

cudaError_t launch_campaign_small(const SmallNet &g, const CampFault *faults, int n_faults, float *S, int32_t *top1,
                                  uint8_t *flag, cudaStream_t st) {
    if (n_faults <= 0) return cudaSuccess;
    constexpr int IPC = 8;
    const size_t smem = campaign_small_smem(g);
    if (smem > 48 * 1024) {
        cudaError_t e = cudaFuncSetAttribute(campaign_small_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)smem);
        if (e != cudaSuccess) return e;
    }
    dim3 grid(n_faults, (g.B + IPC - 1) / IPC);
    CampFault none{};
    none.kind = 2;
    SmallRerun rr{};
    pdl_launch(campaign_small_kernel, grid, 256, smem, st, g, faults, none, IPC, S, top1, flag, (float *)nullptr, rr);
    return cudaGetLastError();
}

cudaError_t launch_small_infer(const SmallNet &g, const CampFault &fault, float *logits, float *S, uint8_t *flag,
                               const SmallRerun &rr, cudaStream_t st) {
    const size_t smem = campaign_small_smem(g);
    if (smem > 48 * 1024) {
        cudaError_t e = cudaFuncSetAttribute(campaign_small_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)smem);
        if (e != cudaSuccess) return e;
    }
    // one image per CTA of 1024 threads: the images of a batch (and the
    // re-run list) run side by side
    dim3 grid(1, g.B + rr.n);
    pdl_launch(campaign_small_kernel, grid, 1024, smem, st, g, (const CampFault *)nullptr, fault, 1, S,
               (int32_t *)nullptr, flag, logits, rr);
    return cudaGetLastError();
}

}  // namespace ct
