// Fused image stem: input conversion, 7x7 stride-2 convolution with the
// carry-through filter on the tensor cores (tcgen05, FP32 accumulation in
// TMEM), bias, ReLU, and the 3x3 stride-2 max-pool that follows it, in one
// persistent kernel.  Only the pooled tensor and its checksum plane reach
// HBM; the unpooled convolution output and the FP16 copy of the image are
// never stored.  Rounding to FP16 before the max-pool and after it give the
// same result (rounding is monotone), so this equals conv -> store -> pool.
//
// GEMM view of one convolution output row (n, p): M = 128 output columns q
// (Q <= 128; rows q >= Q are computed and dropped), N = 64 filters plus the
// carry-through row, K = 7 filter rows x 2 steps x 16.  Step 0 of filter row
// r covers taps s = 0..3 and step 1 taps s = 3..6 (the weight of tap 3 is 0
// in step 1), each tap with 4 channels (the image's C <= 4 channels, then
// zeros).
//
// No im2col tile is built.  Image rows arrive by bulk copies (one per
// channel row) in a staging ring, two rows per producer warp in flight;
// the producer warps convert them from FP32 NCHW to FP16 pixels of 4
// channels (8 bytes) in a ring of shared-memory rows.  With stride 2, output column q reads input pixels 2q + s - 3, so in
// such a row the A operand of one step is a strided view: A row q starts
// 16 bytes after row q - 1 and each 8-element K chunk (2 taps) 16 bytes after
// the previous one.  That is a no-swizzle K-major UMMA descriptor with row
// pitch 16, LBO = 16 and SBO = 128 over overlapping rows.  Step 0 reads copy
// E of the row (pixel x at byte 8 (x + 3)), step 1 reads copy O (pixel x at
// byte 8 (x + 4)), so that both start on a 16-byte boundary.
//
// Work unit: one pooled output row (n, i), which takes convolution rows
// 2i - 1, 2i, 2i + 1.  Each CTA owns a contiguous range of units and computes
// their convolution rows in order, so a row shared by two units is computed
// once (plus one row at the start of each CTA's range in an image).  Each
// epilogue thread keeps the vertical maximum of its output column in
// registers; when a convolution row completes a pooled row, those column
// maxima go through a shared-memory row buffer for the 3-wide horizontal
// maximum and the pooled row is written.
//
// Warp roles (512 threads): warps 0-5 fill ring rows (entry e goes to warp
// e % 6), warps 6 and 7 issue tcgen05.mma (one elected lane each, for
// alternate convolution rows: issuing one row's 14 MMAs and 3 commits takes
// a thread about 900 cycles, so one issuer left the tensor core idle half the
// time, measured), warp 6 also allocates TMEM, warps 8-15 are the epilogue:
// each TMEM lane quadrant is read by two warps, each taking 32 of the 64
// channels.  Four TMEM accumulators rotate over
// consecutive convolution rows, so the MMAs run up to three rows ahead of
// the epilogue.  Every mbarrier wait is bounded; on
// expiry the kernel records an error code, stops and frees TMEM.
#include "ct_internal.h"
#include "tc_common.cuh"

namespace ct {

namespace {

using namespace tc;

constexpr int ST_K = 64;                     // filters
constexpr int ST_NB = ST_K + 16;             // B rows: filters, carry-through row, 15 zero rows
constexpr int ST_R = 7;                      // filter rows and columns
constexpr int ST_KSTEPS = 2 * ST_R;          // K16 steps
constexpr int ST_KLEN = 16 * ST_KSTEPS;      // 224: weight row length
constexpr int ST_RP = 264;                   // ring row pitch in pixels (8 bytes each)
constexpr int ST_ROW_BYTES = ST_RP * 8;      // one copy of one input row
constexpr int ST_SLOT_BYTES = 2 * ST_ROW_BYTES;
constexpr int ST_NSLOT = 24;                 // ring rows: the producers run up to ~8 convolution rows ahead
constexpr int ST_B_STEP = ST_NB * 32;        // B bytes per K16 step (two core-matrix columns)
constexpr int ST_B_LBO = ST_NB * 16;         // between the two K chunks of a step
constexpr int ST_PIX_H = 72;                 // halves per pixel in the epilogue row buffer (144 B)
constexpr int ST_NPROD = 6;                  // ring producer warps
constexpr int ST_NMMA = 2;                   // MMA warps: convolution rows alternate between them
constexpr int ST_MMA_WARP = ST_NPROD;        // the first also allocates TMEM
constexpr int ST_EPI0 = 32 * (ST_NPROD + ST_NMMA);   // first epilogue thread
constexpr int ST_THREADS = ST_EPI0 + 256;
constexpr int ST_EPI = 256;                  // epilogue threads
constexpr int ST_NACC = 4;                   // TMEM accumulators (rows in flight between MMA and epilogue)
constexpr int ST_TMEM_COLS = 128 * ST_NACC;

constexpr size_t ST_OFF_B = (size_t)ST_NSLOT * ST_SLOT_BYTES;
constexpr size_t ST_OFF_ROW = ST_OFF_B + (size_t)ST_KSTEPS * ST_B_STEP;
constexpr size_t ST_OFF_CS = ST_OFF_ROW + 2ull * 128 * ST_PIX_H * 2;
// staging of FP32 image rows (bulk copies): ST_STG_W per producer warp, up
// to 4 channels of 256 pixels each.  Shared memory goes to ring depth first:
// the producer, MMA and epilogue stages only overlap when the ring holds
// several convolution rows beyond the 7-row window (16 slots: 275 us at 256
// images, 24: 238 us; deeper staging gained nothing)
constexpr int ST_STG_W = 2;                  // staging slots per producer warp
constexpr int ST_NSTG = ST_NPROD * ST_STG_W;
constexpr int ST_STG_BYTES = 4 * 256 * 4;
constexpr size_t ST_OFF_STG = ST_OFF_CS + 2ull * 128 * 2;
constexpr size_t ST_OFF_BAR = ST_OFF_STG + (size_t)ST_NSTG * ST_STG_BYTES;
constexpr size_t ST_SMEM = 1024 + ST_OFF_BAR + 8 * (2 * ST_NSLOT + 2 * ST_NACC + ST_NMMA + ST_NSTG) + 16;

struct StemGeom {
    int N, C, H, W, P, Q, P2, Q2;
    int ct;              // carry-through column computed
    uint16_t coef_h;
};

// Walks the convolution rows of one CTA's unit range [u, u_end) in order.
struct StemJobs {
    int u, u_end;
    int n, p, p_end;
    bool seg_start;      // first row of a run within one image

    __device__ bool start_seg(const StemGeom &g) {
        if (u >= u_end) return false;
        n = u / g.P2;
        const int ia = u % g.P2;
        const int ib = min(g.P2 - 1, u_end - 1 - n * g.P2);
        p = ia == 0 ? 0 : 2 * ia - 1;
        p_end = min(2 * ib + 1, g.P - 1);
        u = (n + 1) * g.P2;
        seg_start = true;
        return true;
    }
    __device__ bool first(int u0, int u1, const StemGeom &g) {
        u = u0;
        u_end = u1;
        return start_seg(g);
    }
    __device__ bool next(const StemGeom &g) {
        if (p < p_end) {
            ++p;
            seg_start = false;
            return true;
        }
        return start_seg(g);
    }
};

// barrier among the epilogue warps that also ORs one predicate over them
__device__ __forceinline__ bool epi_bar_or(bool pred) {
    uint32_t r;
    asm volatile(
        "{\n\t.reg .pred p, q;\n\t"
        "setp.ne.u32 p, %1, 0;\n\t"
        "barrier.red.or.pred q, 1, %2, p;\n\t"
        "selp.u32 %0, 1, 0, q;\n\t}"
        : "=r"(r)
        : "r"((uint32_t)pred), "n"(ST_EPI)
        : "memory");
    return r != 0;
}

// two FP32 values to an FP16 pair (round to nearest) with ReLU in one
// conversion: negative values become 0, NaN stays NaN
__device__ __forceinline__ uint32_t cvt_relu_h2(float lo, float hi) {
    uint32_t r;
    asm("cvt.rn.relu.f16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
    return r;
}

__device__ __forceinline__ uint32_t hmax2u(uint32_t a, uint32_t b) {
    __half2 r = __hmax2_nan(*reinterpret_cast<__half2 *>(&a), *reinterpret_cast<__half2 *>(&b));
    return *reinterpret_cast<uint32_t *>(&r);
}

// image n of the batch: images n >= n_split come from the second input
// (re-executed images appended to a batch), directly or through the index
// list x2_idx
__device__ __forceinline__ const float *image_base(const ConvArgs &a, const StemGeom &g, int n) {
    const size_t chw = (size_t)g.C * g.H * g.W;
    if (a.x2 && n >= a.n_split) {
        const int i = a.x2_idx ? a.x2_idx[n - a.n_split] : n - a.n_split;
        return static_cast<const float *>(a.x2) + (size_t)i * chw;
    }
    return static_cast<const float *>(a.x) + (size_t)n * chw;
}

__device__ __forceinline__ float image_half(const float *img, const StemGeom &g, int c, int h, int w) {
    if (c >= g.C || h < 0 || h >= g.H || w < 0 || w >= g.W) return 0.f;
    return __half2float(__float2half_rn(img[((size_t)c * g.H + h) * g.W + w]));
}

// The ring entries in production order: a CTA's convolution rows each need
// the input rows not already in the ring (7 at the start of a run within an
// image, then 2).  Entry e is produced by warp e % ST_NPROD.
struct RowIter {
    StemJobs jb;
    bool have;
    int ecount, t, n_new, y0;
    int n_of_last;        // image of the entry last returned

    __device__ void set_job() {
        n_new = jb.seg_start ? 7 : 2;
        y0 = jb.seg_start ? 2 * jb.p - 3 : 2 * jb.p + 2;
    }
    __device__ void init(int u0, int u1, const StemGeom &g) {
        have = jb.first(u0, u1, g);
        ecount = 0;
        t = 0;
        n_of_last = 0;
        if (have) set_job();
    }
    // next entry of warp w: its index e and input row y
    __device__ bool next(int w, int &e, int &y, const StemGeom &g) {
        while (have) {
            while (t < n_new) {
                const int ee = ecount + t, tt = t;
                ++t;
                if (ee % ST_NPROD == w) {
                    e = ee;
                    y = y0 + tt;
                    n_of_last = jb.n;
                    return true;
                }
            }
            ecount += n_new;
            t = 0;
            have = jb.next(g);
            if (have) set_job();
        }
        return false;
    }
};

__global__ void __launch_bounds__(ST_THREADS, 1)
stem_pool_kernel(const ConvArgs a, const StemGeom g) {
    pdl_wait();
    pdl_trigger();
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint8_t *ring = smem;
    uint8_t *Bs = smem + ST_OFF_B;
    __half *rowbuf = (__half *)(smem + ST_OFF_ROW);
    __half *csbuf = (__half *)(smem + ST_OFF_CS);
    uint64_t *full = (uint64_t *)(smem + ST_OFF_BAR);
    uint64_t *empty = full + ST_NSLOT;
    uint64_t *acc_full = empty + ST_NSLOT;
    uint64_t *acc_empty = acc_full + ST_NACC;
    uint64_t *mma_done = acc_empty + ST_NACC;                // [ST_NMMA]
    uint64_t *stg_full = mma_done + ST_NMMA;                 // [ST_NSTG]
    float *stg = (float *)(smem + ST_OFF_STG);
    uint32_t *tmem_holder = (uint32_t *)(stg_full + ST_NSTG);
    volatile uint32_t *abort_flag = tmem_holder + 1;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int units = g.N * g.P2;
    const int u0 = (int)((long long)blockIdx.x * units / gridDim.x);
    const int u1 = (int)((long long)(blockIdx.x + 1) * units / gridDim.x);

    // ---- set-up: zero the ring (its padding columns stay zero), weights to
    // the canonical no-swizzle layout, the carry-through row ----
    for (int i = threadIdx.x; i < (int)(ST_OFF_B / 16); i += ST_THREADS)
        reinterpret_cast<uint4 *>(ring)[i] = make_uint4(0u, 0u, 0u, 0u);
    {
        const __half *w = static_cast<const __half *>(a.w);
        const __half coef = __ushort_as_half(g.coef_h);
        const __half zero = __ushort_as_half((unsigned short)0);
        for (int i = threadIdx.x; i < ST_NB * (ST_KLEN / 8); i += ST_THREADS) {
            const int nrow = i / (ST_KLEN / 8), k8 = i % (ST_KLEN / 8);
            uint4 v = make_uint4(0u, 0u, 0u, 0u);
            if (nrow < ST_K) {
                v = *reinterpret_cast<const uint4 *>(w + (size_t)nrow * ST_KLEN + k8 * 8);
            } else if (nrow == ST_K && g.ct) {
                // centre tap (r = 3, s = 3) lies in step 0 of filter row 3:
                // K index 3 * 32 + 3 * 4 + c
                __half h[8];
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    const int k = k8 * 8 + e;
                    h[e] = (k >= 108 && k < 108 + g.C) ? coef : zero;
                }
                v = *reinterpret_cast<uint4 *>(h);
            }
            const int t = k8 / 2, kc = k8 % 2;
            *reinterpret_cast<uint4 *>(Bs + t * ST_B_STEP + kc * ST_B_LBO + (nrow / 8) * 128 + (nrow % 8) * 16) = v;
        }
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    if (threadIdx.x == 0) {
        for (int s = 0; s < ST_NSLOT; ++s) {
            mbar_init(smem_u32(&full[s]), 32);
            mbar_init(smem_u32(&empty[s]), ST_NMMA);      // one release per MMA warp
        }
        for (int b = 0; b < ST_NACC; ++b) {
            mbar_init(smem_u32(&acc_full[b]), 1);
            mbar_init(smem_u32(&acc_empty[b]), ST_EPI / 32);
        }
        for (int w = 0; w < ST_NMMA; ++w) mbar_init(smem_u32(&mma_done[w]), 1);
        for (int s = 0; s < ST_NSTG; ++s) mbar_init(smem_u32(&stg_full[s]), 1);
        *abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == ST_MMA_WARP) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_holder)),
                     "r"((uint32_t)ST_TMEM_COLS));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tmem = *tmem_holder;

    if (warp < ST_NPROD) {
        // ---------------- ring producers ----------------
        // Each warp produces every ST_NPROD-th ring entry.  Its next ST_STG_W
        // entries' image rows are in flight as bulk copies (one per channel
        // row of W FP32 values) into its own staging slots; the warp then
        // converts a landed row to the two FP16 copies of its ring slot.
        // Rows outside the image are not copied (their slot reads as zero).
        RowIter ri;
        ri.init(u0, u1, g);
        int ent_e[ST_STG_W], ent_y[ST_STG_W];
        int k_issue = 0, k_done = 0;
        bool ok = true, more = true;
        const uint32_t row_bytes = (uint32_t)g.W * 4u;
        while (ok) {
            // keep ST_STG_W entries in flight
            while (more && k_issue - k_done < ST_STG_W) {
                int e, y;
                more = ri.next(warp, e, y, g);
                if (!more) break;
                const int i = k_issue % ST_STG_W, sl = warp * ST_STG_W + i;
                ent_e[i] = e; ent_y[i] = y;
                if (lane == 0) {
                    const uint32_t bar = smem_u32(&stg_full[sl]);
                    if (y >= 0 && y < g.H) {
                        const float *img = image_base(a, g, ri.n_of_last);
                        mbar_arrive_expect_tx(bar, row_bytes * (uint32_t)g.C);
                        for (int c = 0; c < g.C; ++c)
                            bulk_load(smem_u32(stg + (size_t)sl * (ST_STG_BYTES / 4) + c * g.W),
                                      img + ((size_t)c * g.H + y) * g.W, row_bytes, bar);
                    } else {
                        mbar_arrive(bar);
                    }
                }
                ++k_issue;
            }
            if (k_done == k_issue) break;
            if (__any_sync(0xffffffffu, *abort_flag)) { ok = false; break; }
            const int i = k_done % ST_STG_W, sl = warp * ST_STG_W + i;
            if (!warp_wait(smem_u32(&stg_full[sl]), (uint32_t)(k_done / ST_STG_W) & 1u, a.err, 1u)) { ok = false; break; }
            const int e = ent_e[i], y = ent_y[i];
            const int slot = e % ST_NSLOT;
            if (!warp_wait(smem_u32(&empty[slot]), ((uint32_t)(e / ST_NSLOT) & 1u) ^ 1u, a.err, 1u)) { ok = false; break; }
            const bool row_ok = y >= 0 && y < g.H;
            const float *sr = stg + (size_t)sl * (ST_STG_BYTES / 4);
            uint8_t *E = ring + slot * ST_SLOT_BYTES;
            uint8_t *O = E + ST_ROW_BYTES;
#pragma unroll
            for (int it = 0; it < 8; ++it) {
                const int col = lane + 32 * it;
                if (col < g.W) {
                    float v[4];
#pragma unroll
                    for (int c = 0; c < 4; ++c) v[c] = (row_ok && c < g.C) ? sr[c * g.W + col] : 0.f;
                    __half2 lo = __floats2half2_rn(v[0], v[1]);
                    __half2 hi = __floats2half2_rn(v[2], v[3]);
                    const uint2 pk = make_uint2(*reinterpret_cast<uint32_t *>(&lo), *reinterpret_cast<uint32_t *>(&hi));
                    *reinterpret_cast<uint2 *>(E + (col + 3) * 8) = pk;
                    *reinterpret_cast<uint2 *>(O + (col + 4) * 8) = pk;
                }
            }
            // the staging slot is refilled by a bulk copy (async proxy) after these reads
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            __syncwarp();
            mbar_arrive(smem_u32(&full[slot]));
            ++k_done;
        }
        if (!ok) {
            if (lane == 0) *abort_flag = 1;
            // copies still in flight land before the CTA leaves
            for (int k = k_done; k < k_issue; ++k)
                warp_wait(smem_u32(&stg_full[warp * ST_STG_W + k % ST_STG_W]), (uint32_t)(k / ST_STG_W) & 1u,
                          a.err, 1u);
        }
    } else if (warp < ST_MMA_WARP + ST_NMMA) {
        // ---------------- MMA issuers: job j goes to MMA warp j % ST_NMMA ----------------
        // One elected lane issues a job's 14 MMAs; the issue of one job and
        // the barrier waits of the next overlap across the two warps.  A ring
        // row is released once by each MMA warp, in row order, as soon as
        // none of that warp's later jobs reads it: after its job j, the rows
        // below the window of its next job j + 2 (all remaining rows after its
        // last job).  The release is a commit, so it also waits for the MMAs.
        const int mw = warp - ST_MMA_WARP;
        const uint32_t id64 = idesc_f16(128, ST_K);
        const uint32_t id80 = idesc_f16(128, ST_NB);
        const uint32_t ring_base = smem_u32(ring), b_base = smem_u32(Bs);
        // descriptors: the weights' are fixed; a ring row's is the ring base
        // descriptor plus the row's offset in 16-byte units (the start
        // address field of a no-swizzle descriptor is addr >> 4)
        uint64_t bd[ST_KSTEPS];
#pragma unroll
        for (int t = 0; t < ST_KSTEPS; ++t) bd[t] = smem_desc_noswz(b_base + t * ST_B_STEP, ST_B_LBO, 128);
        const uint64_t ad_base = smem_desc_noswz(ring_base, 16, 128);
        // window starts of jobs j, j + 1, j + 2 (scanned ahead of the issue)
        StemJobs scan;
        bool scan_have = scan.first(u0, u1, g);
        int scan_ec = 0;                       // ring entries of the jobs scanned so far
        int ws[3];
        bool hv[3];
        auto scan_one = [&](int &w, bool &h) {
            h = scan_have;
            w = 0;
            if (scan_have) {
                w = scan.seg_start ? scan_ec : scan_ec - 5;
                scan_ec += scan.seg_start ? 7 : 2;
                scan_have = scan.next(g);
            }
        };
        scan_one(ws[0], hv[0]);
        scan_one(ws[1], hv[1]);
        scan_one(ws[2], hv[2]);
        int j = 0, waited = 0, rel = 0;
        bool issued = false, ok = true;
        while (hv[0]) {
            if (j % ST_NMMA == mw) {
                if (__any_sync(0xffffffffu, *abort_flag)) { ok = false; break; }
                const int wstart = ws[0];
                const int ab = j % ST_NACC;
                const uint32_t use = (uint32_t)(j / ST_NACC) & 1u;
                ok = warp_wait(smem_u32(&acc_empty[ab]), use ^ 1u, a.err, 8u);
                // the rows of the window this warp has not waited for
                for (int e = max(waited, wstart); e < wstart + ST_R && ok; ++e)
                    ok = warp_wait(smem_u32(&full[e % ST_NSLOT]), (uint32_t)(e / ST_NSLOT) & 1u, a.err, 2u);
                if (!ok) { if (lane == 0) *abort_flag = 1; break; }
                waited = wstart + ST_R;
                const int rel_end = hv[ST_NMMA] ? ws[ST_NMMA] : scan_ec;
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                if (elect_one()) {
                    const uint32_t d = tmem + (uint32_t)(ab * 128);
                    int slot = wstart % ST_NSLOT;
                    uint64_t ad[ST_R];
#pragma unroll
                    for (int r = 0; r < ST_R; ++r) {
                        ad[r] = ad_base + (uint64_t)((slot * ST_SLOT_BYTES) >> 4);
                        slot = slot + 1 == ST_NSLOT ? 0 : slot + 1;
                    }
#pragma unroll
                    for (int i = 0; i < ST_R; ++i) {
                        const int r = i == 0 ? 3 : (i <= 3 ? i - 1 : i);    // centre row first
                        // the first MMA (centre row) writes all 80 columns when the
                        // carry-through row is present
                        umma_f16(d, ad[r], bd[2 * r], (i == 0 && g.ct) ? id80 : id64, i > 0 ? 1u : 0u);
                        umma_f16(d, ad[r] + (uint64_t)((ST_ROW_BYTES + 32) >> 4), bd[2 * r + 1], id64, 1u);
                    }
                    umma_commit(smem_u32(&acc_full[ab]));
                    for (int e = rel; e < rel_end; ++e) umma_commit(smem_u32(&empty[e % ST_NSLOT]));
                }
                __syncwarp();
                rel = max(rel, rel_end);
                issued = true;
            }
            ws[0] = ws[1]; hv[0] = hv[1];
            ws[1] = ws[2]; hv[1] = hv[2];
            scan_one(ws[2], hv[2]);
            ++j;
        }
        // a warp with no job after some rows (or none at all) still releases them
        if (ok && rel < scan_ec) {
            if (elect_one())
                for (int e = rel; e < scan_ec; ++e) umma_commit(smem_u32(&empty[e % ST_NSLOT]));
            __syncwarp();
        }
        // every issued MMA has completed before TMEM can be freed
        if (issued) {
            if (elect_one()) umma_commit(smem_u32(&mma_done[mw]));
            __syncwarp();
            warp_wait(smem_u32(&mma_done[mw]), 0u, a.err, 16u);
        }
    } else {
        // ---------------- epilogue: warps 8..15 ----------------
        const int et = threadIdx.x - ST_EPI0;
        const int quad = warp & 3;
        const int half_id = (warp - ST_MMA_WARP - ST_NMMA) >> 2;     // channels 32 * half_id ..
        const int q = quad * 32 + lane;                 // output column of this thread
        const int k0 = 32 * half_id;
        const FaultDelta fd = a.fd;
        float bias[32];
#pragma unroll
        for (int i = 0; i < 32; ++i) bias[i] = __ldg(a.bias + k0 + i);
        const bool has_cs = a.cs_out != nullptr;
        // pooling role: column jj, channels 8 cq .. 8 cq + 7 and 32 + 8 cq ..
        // 32 + 8 cq + 7 (16-byte chunks cq and cq + 4 of a 128-byte pixel):
        // with the 144-byte row-buffer pitch and stride-2 columns, the 32
        // lanes of a warp then start on every 16-byte bank group equally
        // often (contiguous 32-byte quarters would use half the banks)
        const int jj = et >> 2, cq = et & 3;
        const bool pool_data = jj < g.Q2;
        const bool pool_cs = has_cs && et < g.Q2;
        const bool want_ct = has_cs && g.ct && half_id == 0;      // warp-uniform
        const bool keep_cs = has_cs && half_id == 0;
        // vertical max-pool state of this thread's column q, carried across
        // convolution rows: after an odd row p it holds row p (shared with
        // the next pooled row), after an even row the maximum of rows p - 1
        // and p
        uint32_t vs[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) vs[i] = 0xFC00FC00u;
        __half vs_cs = __ushort_as_half((unsigned short)0xFC00);
        bool acc_valid = false, has_carry = false;
        int n_st = 0;                                   // pooled rows written: row-buffer parity
        StemJobs jb;
        bool have = jb.first(u0, u1, g);
        int j = 0;
        while (have) {
            const int ab = j % ST_NACC;
            const uint32_t use = (uint32_t)(j / ST_NACC) & 1u;
            bool ok = mbar_wait(smem_u32(&acc_full[ab]), use, a.err, 4u);
            ok = __all_sync(0xffffffffu, ok) && !*abort_flag;
            const int p = jb.p;
            const bool close_even = (p & 1) == 0 && p == g.P - 1;
            if (jb.seg_start) { acc_valid = false; has_carry = false; }
            // this row completes pooled row i2 (uniform over the epilogue)
            const bool store = (p & 1) ? acc_valid : close_even;
            __half *rb = rowbuf + (size_t)(n_st & 1) * 128 * ST_PIX_H;
            __half *cb = csbuf + (n_st & 1) * 128;
            if (ok) {
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                const uint32_t trow = tmem + (uint32_t)(ab * 128) + ((uint32_t)(quad * 32) << 16);
                // all of the row's TMEM loads in flight, one wait
                float v[32];
                uint32_t r0[16], r1[16], rc = 0;
                tmem_ld16_nw(trow + k0, r0);
                tmem_ld16_nw(trow + k0 + 16, r1);
                if (want_ct) tmem_ld1_nw(trow + ST_K, rc);
                tmem_wait_ld();
                tmem_done16(r0, v);
                tmem_done16(r1, v + 16);
                const float ctv = want_ct ? tmem_done(rc) : 0.f;
                asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(&acc_empty[ab]));
                // bias, ReLU, FP16: one conversion per channel pair on the
                // common path
                uint32_t u[16];
                float o_cs = (a.role == CT_ROLE_CT) ? ctv : 0.f;
                if (!fd.active) {
                    if (a.relu) {
#pragma unroll
                        for (int i = 0; i < 16; ++i) u[i] = cvt_relu_h2(v[2 * i] + bias[2 * i], v[2 * i + 1] + bias[2 * i + 1]);
                    } else {
#pragma unroll
                        for (int i = 0; i < 16; ++i) {
                            __half2 hh = __floats2half2_rn(v[2 * i] + bias[2 * i], v[2 * i + 1] + bias[2 * i + 1]);
                            u[i] = *reinterpret_cast<uint32_t *>(&hh);
                        }
                    }
                } else {
                    const float fsrc = q < g.Q
                        ? image_half(image_base(a, g, jb.n), g, fd.cin, 2 * p + fd.r - 3, 2 * q + fd.s - 3) : 0.f;
#pragma unroll
                    for (int i = 0; i < 32; i += 2) {
                        float o[2];
#pragma unroll
                        for (int t = 0; t < 2; ++t) {
                            float s = v[i + t] + bias[i + t];
                            if (fd.kout == k0 + i + t) s += fd.dv * fsrc;
                            if (a.relu) s = relu_keep_nan(s);
                            o[t] = s;
                        }
                        __half2 hh = __floats2half2_rn(o[0], o[1]);
                        u[i / 2] = *reinterpret_cast<uint32_t *>(&hh);
                    }
                    if (fd.kout == ST_K) o_cs += fd.dv * fsrc;
                }
                if (a.relu) o_cs = relu_keep_nan(o_cs);
                const __half u_cs = __float2half_rn(o_cs);
                // vertical pooling in registers
                uint32_t out[16];
                __half out_cs = u_cs;
                if (p & 1) {
#pragma unroll
                    for (int i = 0; i < 16; ++i) { out[i] = hmax2u(vs[i], u[i]); vs[i] = u[i]; }
                    out_cs = __hmax_nan(vs_cs, u_cs);
                    vs_cs = u_cs;
                } else {
#pragma unroll
                    for (int i = 0; i < 16; ++i) { vs[i] = has_carry ? hmax2u(vs[i], u[i]) : u[i]; out[i] = vs[i]; }
                    vs_cs = has_carry ? __hmax_nan(vs_cs, u_cs) : u_cs;
                    out_cs = vs_cs;
                }
                if (store && q < g.Q) {
                    uint4 *dst = reinterpret_cast<uint4 *>(rb + q * ST_PIX_H + k0);
#pragma unroll
                    for (int i = 0; i < 4; ++i) dst[i] = make_uint4(out[4 * i], out[4 * i + 1], out[4 * i + 2], out[4 * i + 3]);
                    if (keep_cs) cb[q] = out_cs;
                }
            }
            if (epi_bar_or(!ok)) {
                if (et == 0) *abort_flag = 1;
                break;
            }
            // ---- a completed pooled row: column max over 2jj - 1 .. 2jj + 1 ----
            if (store) {
                const int i2 = (p & 1) ? (p - 1) / 2 : p / 2;
                if (pool_data) {
                    uint32_t h[8];
#pragma unroll
                    for (int i = 0; i < 8; ++i) h[i] = 0xFC00FC00u;
#pragma unroll
                    for (int dc = -1; dc <= 1; ++dc) {
                        const int col = 2 * jj + dc;
                        if (col < 0 || col >= g.Q) continue;
                        const uint4 *src = reinterpret_cast<const uint4 *>(rb + col * ST_PIX_H + 8 * cq);
                        const uint4 s0 = src[0], s1 = src[4];
                        h[0] = hmax2u(h[0], s0.x); h[1] = hmax2u(h[1], s0.y);
                        h[2] = hmax2u(h[2], s0.z); h[3] = hmax2u(h[3], s0.w);
                        h[4] = hmax2u(h[4], s1.x); h[5] = hmax2u(h[5], s1.y);
                        h[6] = hmax2u(h[6], s1.z); h[7] = hmax2u(h[7], s1.w);
                    }
                    uint4 *dst = reinterpret_cast<uint4 *>(static_cast<__half *>(a.y) +
                                                            (((size_t)jb.n * g.P2 + i2) * g.Q2 + jj) * ST_K + 8 * cq);
                    dst[0] = make_uint4(h[0], h[1], h[2], h[3]);
                    dst[4] = make_uint4(h[4], h[5], h[6], h[7]);
                }
                if (pool_cs) {
                    __half h = __ushort_as_half((unsigned short)0xFC00);
                    for (int dc = -1; dc <= 1; ++dc) {
                        const int col = 2 * et + dc;
                        if (col >= 0 && col < g.Q) h = __hmax_nan(h, cb[col]);
                    }
                    static_cast<__half *>(a.cs_out)[((size_t)jb.n * g.P2 + i2) * g.Q2 + et] = h;
                }
                ++n_st;
            }
            if (p & 1) { acc_valid = false; has_carry = true; }
            else { acc_valid = !close_even; }
            have = jb.next(g);
            ++j;
        }
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (warp == ST_MMA_WARP) {
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"((uint32_t)ST_TMEM_COLS));
    }
}

}  // namespace

struct StemPlan {
    StemGeom g;
    int sms;
};

int stem_kidx(int r, int s, int c) { return r * 32 + (s <= 3 ? s * 4 : 16 + (s - 3) * 4) + c; }
int stem_klen() { return ST_KLEN; }

bool stem_pool_supported(int C, int K, int R, int S, int stride, int pad, int H, int W) {
    if (C < 1 || C > 4 || K != ST_K || R != ST_R || S != ST_R || stride != 2 || pad != 3) return false;
    const int P = (H + 2 * pad - R) / stride + 1, Q = (W + 2 * pad - S) / stride + 1;
    // W % 4: image rows are bulk-copied, which needs 16-byte multiples
    return P >= 2 && Q >= 2 && Q <= 128 && W + 4 <= ST_RP && W <= 256 && W % 4 == 0;
}

StemPlan *stem_plan_create(const ConvArgs &a, std::string *why) {
    if (!stem_pool_supported(a.C, a.K, a.R, a.S, a.stride, a.pad, a.H, a.W)) {
        if (why) *why = "shape not supported by the fused stem";
        return nullptr;
    }
    StemPlan *pl = new (std::nothrow) StemPlan();
    if (!pl) return nullptr;
    StemGeom &g = pl->g;
    g.C = a.C; g.H = a.H; g.W = a.W; g.P = a.P; g.Q = a.Q;
    g.P2 = (g.P + 2 - 3) / 2 + 1;
    g.Q2 = (g.Q + 2 - 3) / 2 + 1;
    g.ct = a.role == CT_ROLE_CT;
    __half h = __float2half_rn(a.coef);          // exact: coefficients are powers of two
    memcpy(&g.coef_h, &h, 2);
    pl->sms = device_sm_count();
    if (cudaFuncSetAttribute(stem_pool_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)ST_SMEM) !=
        cudaSuccess) {
        cudaGetLastError();
        if (why) *why = "cannot reserve shared memory for the fused stem";
        delete pl;
        return nullptr;
    }
    return pl;
}

void stem_plan_destroy(StemPlan *p) { delete p; }

cudaError_t launch_stem_pool(const ConvArgs &a, const StemPlan *pl, cudaStream_t st) {
    StemGeom g = pl->g;
    g.N = a.N;
    const int units = g.N * g.P2;
    const int grid = std::min(pl->sms, units);
    pdl_launch(stem_pool_kernel, grid, ST_THREADS, ST_SMEM, st, a, g);
    return cudaGetLastError();
}

}  // namespace ct
