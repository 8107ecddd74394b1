// Internal structures of libct (not part of the ABI).
#pragma once

#include <cuda_runtime.h>
#include <cuda_fp16.h>
#include <stdint.h>

#include <string>
#include <utility>
#include <vector>

#include "../../include/ct.h"

namespace ct {

// Implicit weight of the carry-through construction hit by a fault: output
// channel `kout` (== K for the checksum output) gains dv * input[cin] at tap
// (r, s), where cin == C means the incoming checksum plane.
struct FaultDelta {
    int active;
    int kout, cin, r, s;
    float dv;
};

// Arguments of every convolution kernel.  Activations are NHWC, the checksum
// plane is [N, H, W]; weights are KRSC (C innermost).
struct ConvArgs {
    const void *x;        // [N, H, W, C]
    const void *cs_in;    // [N, H, W] or null
    const void *w;        // [K, R, S, C]
    const float *bias;    // [K]
    const void *res;      // [N, P, Q, K] or null
    const void *res_cs;   // [N, P, Q] or null
    void *y;              // [N, P, Q, K]
    void *cs_out;         // [N, P, Q] or null
    int N, H, W, C, K, R, S, stride, pad, P, Q;
    int role;             // ct_role after ds_mode is applied
    int relu;
    float coef;           // carry-through coefficient 2^-ct_shift
    FaultDelta fd;
    uint32_t *err;        // device error word
    int cs_rowsum;        // > 0: an FC layer run as a 1x1 convolution; its checksum input
                          // is the sum of cs_in[m * cs_rowsum .. m * cs_rowsum + cs_rowsum)
    float *ws;            // split-K workspace (null: never split)
    size_t ws_bytes;
    const void *x2;       // first layer only: images n >= n_split are image n - n_split of x2
    int n_split;          // (null x2: every image comes from x)
    const int32_t *x2_idx;  // non-null: image n >= n_split is image x2_idx[n - n_split] of x2
                            // (device-visible: mapped host memory)
};

// Batched campaign on a LeNet-shaped FP32 network (campaign_small.cu):
// shapes, the model's device weights (convolutions KRSC, FC rows with
// columns in the NHWC flatten order), coefficients and threshold.
struct SmallNet {
    int B, C0, H0, W0;
    int protect;                          // widened construction (0: the network alone)
    const float *x2;                      // images n >= n_split are image n - n_split of x2 (null: none)
    int n_split;
    uint8_t *flag2;                       // inference: a second copy of the flags (host-mapped) or null
    int K1, R1, H1, W1, Hp1, Wp1;
    int K2, R2, H2, W2, Hp2, Wp2;
    int NIN1, N1, N2, N3;
    const float *x;                       // [B, C0, H0, W0] FP32 images
    const float *w1, *b1, *w2, *b2, *wf1, *bf1, *wf2, *bf2, *wf3, *bf3;
    float coef1, coef2, coeff1, coeff2, coeff3;
    double ref, tau;
};

// One fault of a batched campaign, resolved on the host.
struct CampFault {
    int kind;            // 0 weight, 1 activation, 2 none
    int layer;           // weight: 0 first convolution, 1 second
    long long word;      // weight: stored word to flip (-1: use fd)
    int bit;
    FaultDelta fd;       // weight: element of the construction that is not stored
    int img, act_c, act_hw;   // activation: image, channel (K1 = checksum), pixel of the first pool's output
};

bool dw_supported(int C, int K, bool half);
cudaError_t launch_conv_dw(const ConvArgs &a, bool half, cudaStream_t st);

size_t campaign_small_smem(const SmallNet &g);
cudaError_t launch_campaign_small(const SmallNet &g, const CampFault *faults, int n_faults, float *S, int32_t *top1,
                                  uint8_t *flag, cudaStream_t st);
// Re-run list of a whole-network inference: images idx[0 .. n) of x, their
// logits and S written to those rows of logits / S.
constexpr int SMALL_MAX_RERUN = 128;
struct SmallRerun {
    const float *x;
    float *logits, *S;
    int n;
    int idx[SMALL_MAX_RERUN];
};
// Inference of g.B images with the whole-network kernel: logits [B, N3],
// S [B] and flags [B] (each may be null), with `fault` (kind 2: none)
// applied, plus the fault-free re-run list rr (rr.n = 0: none).
cudaError_t launch_small_infer(const SmallNet &g, const CampFault &fault, float *logits, float *S, uint8_t *flag,
                               const SmallRerun &rr, cudaStream_t st);

struct FcArgs {
    const void *x;        // [B, n_in] data features
    const void *xcs;      // [B, n_cs] checksum features or null
    const void *w;        // [n_out, n_in]
    const float *bias;    // [n_out]
    void *y;              // [B, n_out]  (final: float logits)
    void *ycs;            // [B] carry-through neuron (hidden) or null
    float *S;             // final: [B] or null
    uint8_t *flag;        // final: [B] or null
    uint8_t *flag2;       // final: a second copy of the flags (host-mapped memory) or null
    int B, n_in, n_cs, n_out;
    int relu, final_layer, protect;
    float coef;
    double ref, tau;
    float *ws;            // split-K workspace (null: never split)
    size_t ws_bytes;
    // final layer with re-run rows: rows b >= rr_split are re-executed images
    // of an earlier batch; their logits and S go to row rr_idx[b - rr_split]
    // of rr_y / rr_S (rr_S may be null) and their flags are not written
    // (rr_idx null: every row is a row of this batch)
    int rr_split;
    const int32_t *rr_idx;
    float *rr_y;
    float *rr_S;
};

struct PoolArgs {
    const void *x; const void *cs_in;
    void *y; void *cs_out;
    int N, H, W, C, P, Q, k, stride, pad;
};

enum Family { FAM_TC = 0, FAM_SIMT = 1, FAM_FC = 2, FAM_POOL = 3, FAM_OTHER = 4, FAM_COUNT = 5 };

// Programmatic dependent launch: every kernel is launched so that it may
// start while the previous kernel in the stream finishes; it calls
// pdl_wait() before its first access to global memory (which returns once
// the previous kernel has completed and its writes are visible) and
// pdl_trigger() to let the next kernel start early.  Only prologues that
// touch no global memory (barrier set-up, TMEM allocation) overlap.
#ifdef __CUDACC__
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
#endif

template <typename... KArgs, typename... Args>
inline cudaError_t pdl_launch(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                              Args &&...args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// pdl_launch for a kernel launched in clusters of cluster_x CTAs
template <typename... KArgs, typename... Args>
inline cudaError_t pdl_launch_cluster(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                                      int cluster_x, Args &&...args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = (unsigned)cluster_x;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// kernel launchers; each returns cudaGetLastError()
// conv launchers report in *n_kernels (may be null) how many kernels they
// launched: 2 when K is split (the conv kernel and the split-K reduction)
cudaError_t launch_conv_simt(const ConvArgs &a, bool half, cudaStream_t st, int *n_kernels);
// a2 / tc_plan2: a 1x1 shortcut convolution of the same input at the same
// stride whose pixel is the first layer's centre tap; it runs in the same
// launch when both layers' tiles allow (*merged tells whether it did; if
// not, the caller launches it itself)
cudaError_t launch_conv_tc(const ConvArgs &a, const void *tc_plan, cudaStream_t st, int *n_kernels,
                           const ConvArgs *a2 = nullptr, const void *tc_plan2 = nullptr, bool *merged = nullptr);
// whether launch_conv_tc(a, tc_plan, ..., a2, tc_plan2) runs both layers in one launch
bool tc_shortcut_fits(const ConvArgs &a, const void *tc_plan, const void *tc_plan2);
// Split-K: number of K splits for `tiles` output tiles over n_kblocks K
// blocks (1 = no split); partial sums [splits][M][ws_ld] must fit ws_bytes.
int splitk_choose(int tiles, int n_kblocks, int min_kb_per_split, int target_ctas, int M, int ws_ld,
                  size_t ws_bytes);
// Adds the partials in a.ws and applies the conv epilogue (data and checksum).
cudaError_t launch_splitk_reduce(const ConvArgs &a, int splits, int ws_ld, bool half, cudaStream_t st);
cudaError_t launch_fc(const FcArgs &a, bool half, bool x_float, cudaStream_t st, int *n_kernels);
cudaError_t launch_maxpool(const PoolArgs &a, bool half, cudaStream_t st);
cudaError_t launch_gap(const PoolArgs &a, bool half, cudaStream_t st);
// idx non-null: row n of out is image idx[n] of in (device-visible idx)
cudaError_t launch_convert_input(const float *in, void *out, int N, int C, int Cp, int H, int W, bool half,
                                 cudaStream_t st, const int32_t *idx = nullptr);
cudaError_t launch_xor_bit(void *base, int64_t word, int bit, int word_bytes, cudaStream_t st);
cudaError_t launch_gather_images(const float *in, float *out, const int32_t *idx, int n,
                                 int64_t per_image, cudaStream_t st);
cudaError_t launch_scatter_rows(const float *src, float *dst, const int32_t *idx, int n, int row,
                                cudaStream_t st);

// Model facts and a fault-free inference for code outside ct_api.cu.
struct ModelInfo {
    int device, in_c, in_h, in_w, n_classes, max_batch, protect;
};
ct_status model_info(const ct_model *m, ModelInfo *out);
// ct_infer on device buffers with any armed fault left armed for the next ct_infer.
ct_status infer_fault_free(ct_model *m, const float *input, int batch, float *logits, float *S,
                           uint8_t *flag, cudaStream_t st);
// The re-execution gather and scatter launched for model m: counted by
// ct_kernel_count and timed under ct_profile_enable like every kernel of m.
cudaError_t reexec_gather(ct_model *m, const float *in, float *out, const int32_t *idx, int n, int64_t per_image,
                          cudaStream_t st);
cudaError_t reexec_scatter(ct_model *m, const float *src, float *dst, const int32_t *idx, int n, int row,
                           cudaStream_t st);
// Looks up, with `device` current, the device address of the static scratch
// of ct_reexecute_noalloc (loading its module commits the array); ct_build
// calls it so that no request-serving call does.
ct_status noalloc_scratch_setup(int device);

// number of SMs of the current device (148 if the query fails)
int device_sm_count();

// tensor-core conv plan (opaque outside conv_tc.cu)
struct TcPlan;
TcPlan *tc_plan_create(const ConvArgs &shape_args, int max_batch, const void *w_dev, const void *x_dev,
                       std::string *why);
void tc_plan_destroy(TcPlan *p);
bool tc_supported(int C, int K, int R, int S, int stride, int pad, std::string *why);

// tensor-core conv for first layers with at most 4 input channels (input
// stored NHWC with 4 channels; weights [64][tc_small_kpad] with K index
// tap * 4 + channel)
struct TcSmallPlan;
bool tc_small_supported(int C, int K, int R, int S, int stride, int pad);
int tc_small_kpad(int R, int S);
TcSmallPlan *tc_small_plan_create(const ConvArgs &shape_args, const void *w_dev, std::string *why);
void tc_small_plan_destroy(TcSmallPlan *p);
cudaError_t launch_conv_tc_small(const ConvArgs &a, const TcSmallPlan *plan, cudaStream_t st);

// Stride-1 3x3 convolution (C a multiple of 64, K = 64 or 128) from halo
// tiles of 16 x 8 output pixels: one patch load per tile and channel block.
struct HaloPlan;
bool halo_supported(int C, int K, int R, int S, int stride, int pad, int H, int W);
// res_dev / csin_dev / rescs_dev: residual tensor, incoming and residual
// checksum planes the layer reads (null if none); launches must pass them.
// pool: the layer's 2 x 2 stride-2 max-pool is applied in the epilogue (even
// H and W); launches then pass the pooled tensor and plane as y / cs_out.
HaloPlan *halo_plan_create(const ConvArgs &shape_args, int max_batch, const void *w_dev, const void *x_dev,
                           const void *res_dev, const void *csin_dev, const void *rescs_dev, bool pool,
                           std::string *why);
void halo_plan_destroy(HaloPlan *p);
int halo_tiles(const HaloPlan *p, int batch);
int halo_sms(const HaloPlan *p);
cudaError_t launch_conv_tc_halo(const ConvArgs &a, const HaloPlan *p, cudaStream_t st);

// Fused image stem (7x7 stride-2 convolution, C <= 4, 64 filters, followed
// by a 3x3 stride-2 padding-1 max-pool): reads the FP32 NCHW image, writes
// the pooled NHWC tensor and its checksum plane.  Weights [64][stem_klen()]
// with K index stem_kidx(r, s, c).
struct StemPlan;
bool stem_pool_supported(int C, int K, int R, int S, int stride, int pad, int H, int W);
int stem_kidx(int r, int s, int c);
int stem_klen();
StemPlan *stem_plan_create(const ConvArgs &shape_args, std::string *why);
void stem_plan_destroy(StemPlan *p);
cudaError_t launch_stem_pool(const ConvArgs &a, const StemPlan *p, cudaStream_t st);

}  // namespace ct
