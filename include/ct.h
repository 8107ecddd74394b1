/*
 * ct.h -- C ABI of the carry-through checksum inference library (libct.so).
 *
 * The library runs CNN inference in which convolutional layers carry the
 * carry-through filter of Sec. II-A (an extra output filter with a single 1
 * at the kernel centre over every input channel), propagates the resulting
 * checksum channel through bias, activation, pooling and the classifier,
 * sums it in the accumulated-checksum neuron of Sec. II-B, and flags every
 * image whose neuron deviates from a reference by more than a threshold.
 * A bit-flip injector (Sec. III-A) and re-execution of flagged images
 * (Sec. II-B, last paragraph) complete the path.
 *
 * Conventions shared by every entry point:
 *   - Status codes only; nothing is thrown across the ABI.
 *   - "_dev" pointers are CUDA device pointers on the model's device; the
 *     caller owns them and keeps them valid until the stream work that uses
 *     them has finished.  "_host" pointers are host memory.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *     stream).  Calls are asynchronous on that stream unless stated.
 *   - The library owns all weights, activation workspaces and scratch.
 *   - A model is not thread-safe: one host thread at a time per model.
 */
#ifndef CT_H
#define CT_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    CT_OK = 0,
    CT_EINVAL = 1,       /* bad argument or malformed description */
    CT_ENOMEM = 2,       /* device or host allocation failed */
    CT_ECUDA = 3,        /* a CUDA runtime/driver call failed */
    CT_ESTATE = 4,       /* call not valid in the model's current state */
    CT_ERANGE = 5,       /* index, batch or bit outside the allowed range */
    CT_EUNSUPPORTED = 6, /* shape the kernels do not implement */
    CT_EDEVICE = 7       /* a kernel reported a device-side error (bounded wait expired) */
} ct_status;

typedef enum { CT_FP32 = 0, CT_FP16 = 1 } ct_precision;

typedef enum { CT_OP_CONV = 0, CT_OP_MAXPOOL = 1, CT_OP_GAP = 2, CT_OP_FC = 3 } ct_op;

/* Role of a convolution in the scheme (Sec. II-A):
 *   CT_ROLE_CT   carries a carry-through filter (new last output channel);
 *   CT_ROLE_NONE carries none: the first convolution of a residual block,
 *                whose input is also the block's shortcut (Sec. II-A, last
 *                paragraph);
 *   CT_ROLE_PASS a 1x1 downsample shortcut: its checksum output is the
 *                incoming checksum at the sampled position (or nothing when
 *                the model is built with CT_DS_ZERO);
 *   CT_ROLE_AUTO derived from the network graph by the residual rule (see
 *                ct_resolve_roles). */
typedef enum { CT_ROLE_CT = 0, CT_ROLE_NONE = 1, CT_ROLE_PASS = 2, CT_ROLE_AUTO = 3 } ct_role;

typedef enum { CT_BUF_WEIGHT = 0, CT_BUF_ACT = 1 } ct_buf_kind;

typedef enum { CT_DS_PASS = 0, CT_DS_ZERO = 1 } ct_ds_mode;

/* One operation over numbered tensor slots; slot 0 is the network input.
 *   CONV    y = act(conv(x[src]) * BN + res[res]) with kernel k x k, stride,
 *           pad; res = -1 for none; weights OIHW [cout, cin, k, k].
 *   MAXPOOL k x k window, stride, pad (padding never wins).
 *   GAP     global average pool to a vector of cin features.
 *   FC      y = act(W x + b), W [cout, cin] with cin counted in the
 *           PyTorch flatten order (C, H, W) of the data channels; `final`
 *           marks the classifier, which gets the accumulated-checksum neuron.
 * ct_shift: the layer's carry-through coefficients are 2^-ct_shift instead
 * of 1 (keeps an FP16 checksum neuron inside the FP16 range). */
typedef struct {
    int32_t op, src, dst, res;
    int32_t cin, cout, k, stride, pad;
    int32_t role;
    int32_t bn, relu, final;
    int32_t ct_shift;
    int32_t groups;   /* CONV: 1 (dense) or cin == cout (depthwise; weights
                         [cout, 1, k, k]).  The paper constructs the
                         carry-through filter for dense convolutions; in a
                         depthwise layer the checksum is one more group, whose
                         filter sees only the incoming checksum channel, so it
                         passes the checksum through at the centre tap (role
                         CT or PASS; nothing when the input carries no
                         checksum).  Its literal weight layout is
                         [cout (+1), 1, k, k].  Not with CT_PROTECT_REPLACE. */
} ct_layer_desc;

typedef struct {
    int32_t n_layers;
    const ct_layer_desc *layers;
    int32_t in_c, in_h, in_w;     /* input image shape (NCHW without N) */
    int32_t n_classes;
    double bn_eps;                /* epsilon of Eq. 1 */
} ct_model_desc;

/* Weight pointers: `weights[6*i + j]` for layer i, host FP32, read-only,
 * copied by ct_build:
 *   j = 0  conv: W [cout, cin, k, k] (OIHW); fc: W [cout, cin]
 *   j = 1  bias [cout] or NULL (zero)
 *   j = 2..5  BatchNorm gamma, beta, running mean, running var [cout]
 *          (conv with bn = 1 only; otherwise NULL). */
#define CT_WEIGHTS_PER_LAYER 6

/* flags for ct_build_opts.flags */
#define CT_FLAG_SIMT_ONLY 1u      /* use the CUDA-core conv kernels everywhere */
#define CT_FLAG_LAYERWISE 2u      /* one kernel per layer even where the whole network
                                     fits one kernel (the LeNet-5 shape, FP32) or a
                                     shortcut could share its block's first launch */

/* ct_build_opts.protect: how the scheme of Sec. II-A is built in.
 *   CT_PROTECT_NONE     the network as described (the unprotected baseline);
 *   CT_PROTECT_WIDEN    every carry-through filter is an EXTRA output channel
 *                       (kept beside the tensor as a checksum plane) and every
 *                       hidden FC layer gets an extra neuron: the data path is
 *                       the unprotected one, bit for bit;
 *   CT_PROTECT_REPLACE  the paper's construction: in every tensor the least
 *                       important channel is pruned and the carry-through
 *                       filter (or neuron) takes its place as the LAST
 *                       channel, so widths and costs are those of the
 *                       unprotected network.  Importance: the combined L1 norm
 *                       of the channel's filters (before BatchNorm folding) in
 *                       its writers and of its slices in its readers, summed
 *                       over tensors tied by a residual add or a pooling; the
 *                       smallest, lowest index on ties.  A residual block's
 *                       first convolution gets an all-zero last channel, the
 *                       1x1 shortcut a pass-through one (CT_DS_ZERO: zero);
 *                       the slices of the incoming checksum are zero weights
 *                       that are multiplied like any other.  No fine-tuning.
 *                       The classifier keeps its classes and gets the
 *                       accumulated-checksum neuron (sum of all its inputs,
 *                       the checksum channel's features included).
 * Faults (ct_inject) address the stored tensors: for CT_PROTECT_REPLACE the
 * literal layout is the original shape. */
#define CT_PROTECT_NONE 0
#define CT_PROTECT_WIDEN 1
#define CT_PROTECT_REPLACE 2

typedef struct {
    int32_t precision;   /* ct_precision: storage type of weights and activations */
    int32_t protect;     /* CT_PROTECT_NONE / _WIDEN / _REPLACE (see above) */
    int32_t ds_mode;     /* ct_ds_mode */
    int32_t device;      /* CUDA device ordinal */
    int32_t max_batch;   /* workspaces are sized for this many images */
    uint32_t flags;
} ct_build_opts;

typedef struct ct_model ct_model;

/* ct_resolve_roles -- Sec. II-A residual rule, host only (no device is
 * touched).  A convolution whose input tensor is also read by another layer
 * (as the `src` of another layer or as a `res` operand: the shortcut of a
 * residual block) must not carry a carry-through filter: that tensor's
 * checksum already reaches the block's residual add along the shortcut, and
 * a filter on the other path would count it twice.  roles[i] (one per layer,
 * written for every layer) receives the effective role of convolution i, -1
 * for other layers.  CT_ROLE_AUTO resolves to CT_ROLE_CT for a convolution
 * whose input has no other reader; otherwise to CT_ROLE_PASS when its
 * output goes to nothing but a residual add (the shortcut), else to
 * CT_ROLE_NONE.  Explicit roles are kept.
 * Errors: CT_EINVAL for a malformed description or a CT_ROLE_CT
 * convolution that the rule forbids. */
ct_status ct_resolve_roles(const ct_model_desc *desc, int32_t *roles);

/* ct_build -- Sec. II-A/II-B construction.  Folds BatchNorm (Eq. 1) into the
 * convolutions in double precision with the identity (scale exactly 1, bias
 * 0) on every checksum channel; appends a carry-through filter to every
 * CT_ROLE_CT convolution; leaves the checksum input out of every data filter
 * (its zero slice is structural); adds one all-ones neuron to every hidden
 * FC layer and the accumulated-checksum neuron to the final one; rounds to
 * the storage precision; converts to the device layouts and uploads.
 * With FP16 storage, a first 7x7 stride-2 convolution on an image of at most
 * 4 channels with 64 filters, followed by a 3x3 stride-2 padding-1 max-pool
 * that is its only reader, runs as one fused kernel: the FP16 copy of the
 * image and the unpooled convolution output are then never stored.
 * An FP32 network of the LeNet-5 shape (conv, 2x2 max-pool, conv, 2x2
 * max-pool, three FC layers; widened or unprotected) runs as ONE kernel
 * whose CTAs take one image each through the whole network in shared
 * memory; an armed fault is applied inside it (its intermediate tensors are
 * then not stored, and a fault in the image is rejected with CT_ERANGE).
 * CT_FLAG_LAYERWISE keeps one kernel per layer.
 * With FP16 storage, a 1x1 shortcut convolution listed right after its
 * block's first convolution, reading the same tensor at the same stride
 * (the shortcut's pixel is that convolution's centre tap), runs in the same
 * launch on the tensor cores whenever both are whole N = 128 or N = 256
 * tiles (unless CT_FLAG_LAYERWISE); its outputs are the same bits.
 * With FP16 storage, a stride-1 3x3 convolution followed by a 2x2 stride-2
 * max-pool that is its only reader applies the pool in its epilogue (data
 * and checksum channels together) whenever it runs on halo tiles (batches
 * that fill the GPU with them): its unpooled output is then not stored.
 * Roles are resolved and checked by the rule of ct_resolve_roles first,
 * before any device is touched.
 * Synchronous.  On success *out owns device memory until ct_destroy.
 * Errors: CT_EINVAL (malformed description, or a carry-through filter that
 * the residual rule forbids), CT_EUNSUPPORTED, CT_ENOMEM, CT_ECUDA.  Nothing
 * is allocated on failure. */
ct_status ct_build(const ct_model_desc *desc, const float *const *weights,
                   const ct_build_opts *opts, ct_model **out);

/* ct_set_threshold -- Sec. II-B detection rule: an image is flagged when
 * NOT(|S - reference| <= tau), so a NaN or infinite S is always flagged.
 * tau must be >= 0 (CT_EINVAL otherwise).  A new model has tau = +inf. */
ct_status ct_set_threshold(ct_model *m, double reference, double tau);
ct_status ct_get_threshold(const ct_model *m, double *reference, double *tau);

/* ct_infer -- Sec. II-B.  Runs `batch` images through the network.
 *   input_dev  FP32 NCHW [batch, in_c, in_h, in_w], read-only.
 *   logits_dev FP32 [batch, n_classes], written.
 *   S_dev      FP32 [batch]: the accumulated-checksum neuron (NULL allowed;
 *              NaN for an unprotected model).
 *   flag_dev   uint8 [batch]: 1 = flagged (NULL allowed; 0 when unprotected).
 * An armed fault (ct_inject) is applied during this call and disarmed:
 * a weight fault flips the stored word before the layer runs and flips it
 * back after; an activation fault flips the stored word of the layer's
 * input tensor after its producer wrote it and before any reader.
 * Errors: CT_ERANGE if batch < 1 or batch > max_batch; CT_ECUDA. */
ct_status ct_infer(ct_model *m, const float *input_dev, int32_t batch, float *logits_dev,
                   float *S_dev, uint8_t *flag_dev, void *stream);

/* ct_inject -- Sec. III-A fault model: arms ONE transient single-bit flip
 * for the next ct_infer.  `layer` indexes desc->layers and must be a CONV.
 * `element` is a flat index into the literal layout of the protected
 * network, where the checksum is the last channel:
 *   CT_BUF_WEIGHT: [C_out_tot, C_in_tot, k, k] of that layer (carry-through
 *     row and zero checksum slice included);
 *   CT_BUF_ACT:    [batch, C_tot, H, W] of that layer's input tensor, for
 *     the batch of the next ct_infer.
 * `bit` is in [0, 32) for FP32 and [0, 16) for FP16 storage.
 * Errors: CT_EINVAL (not a conv layer, bad kind), CT_ERANGE (element or bit
 * out of range, or an activation tensor that is not stored: the image of a
 * model with a fused stem; an activation element is range-checked again by
 * ct_infer against its batch). */
ct_status ct_inject(ct_model *m, int32_t kind, int32_t layer, int64_t element, int32_t bit);
ct_status ct_clear_faults(ct_model *m);

/* ct_reexecute -- Sec. II-B mitigation.  Re-runs, fault-free, only the
 * images whose flag_dev entry is non-zero and overwrites their rows of
 * logits_dev and S_dev (the re-run's own flags are ignored; flag_dev is not
 * modified).  Synchronises `stream` once to read the flags.  *n_rerun
 * (host) receives the number of images re-run.  Same buffers as ct_infer.
 * The re-run batch is padded to the next power of two (or to max_batch when
 * that is smaller) by repeating the last flagged image.  Its inference is
 * captured into a CUDA graph on a model-owned stream the first time that
 * padded size occurs (that call is slower; ct_reexecute_prepare captures
 * them ahead of time) and replayed afterwards; with profiling on
 * (ct_profile_enable) the kernels are launched one by one instead.  A re-run row equals a fault-free
 * ct_infer of the padded batch; because small batches split K differently,
 * it can differ from the same image's row of a full batch by summation
 * order.  An armed fault stays armed for the next ct_infer. */
ct_status ct_reexecute(ct_model *m, const float *input_dev, int32_t batch,
                       const uint8_t *flag_dev, float *logits_dev, float *S_dev,
                       int32_t *n_rerun, void *stream);

/* ct_reexecute_prepare -- captures, ahead of time, the re-execution graphs
 * ct_reexecute replays (Sec. II-B mitigation): one per padded re-run size
 * (1, 2, 4, ... up to the first power of two >= max_images, capped at
 * max_batch), so that no later ct_reexecute pays a capture.  Synchronous;
 * launches nothing.  Errors: CT_EINVAL (null model), CT_ERANGE (max_images
 * outside 1..max_batch), CT_ECUDA (capture or instantiation failed). */
ct_status ct_reexecute_prepare(ct_model *m, int32_t max_images);

/* ct_infer_reexec -- ct_infer of `batch` new images (input_dev, logits_dev,
 * S_dev, flag_dev as for ct_infer) that also carries out the Sec. II-B
 * re-execution of a PREVIOUS inference's flagged images, deferred into this
 * one: the images of prev_input_dev [prev_batch, C, H, W] whose
 * prev_flag_dev entry is non-zero are appended as extra rows of this
 * inference (the same kernels over batch + n images), and their re-run
 * logits and S overwrite their rows of prev_logits_dev / prev_S_dev
 * (prev_S_dev may be NULL).  The re-run's flags are ignored and
 * prev_flag_dev is not modified.  A flagged image thus costs one more image
 * of a large batch instead of a separate small-batch pass.  Within one
 * inference every image's row is computed independently of the others, so
 * the re-run rows equal those of a fault-free ct_infer of the same images
 * at a batch size with the same tiling.
 *   - prev_input_dev NULL (or prev_batch 0): exactly ct_infer; *n_rerun = 0.
 *   - Synchronises `stream` once to read prev_flag_dev, like ct_reexecute.
 *   - The combined batch must fit max_batch: when batch + n > max_batch, or
 *     when a fault is armed (a re-run must be fault-free), the previous
 *     batch is re-executed first exactly as by ct_reexecute and then this
 *     batch is inferred as by ct_infer (the armed fault goes to it).
 *   - The previous batch's buffers must stay valid until the stream reaches
 *     this call's kernels; none of them may alias this call's outputs.
 *   - *n_rerun (host, may be NULL): images of the previous batch re-run.
 * Errors: CT_EINVAL (null model, input or logits; prev_input_dev given
 * without prev_flag_dev or prev_logits_dev), CT_ERANGE (batch or prev_batch
 * outside 1..max_batch), CT_ECUDA, and those of ct_infer. */
ct_status ct_infer_reexec(ct_model *m, const float *input_dev, int32_t batch, float *logits_dev,
                          float *S_dev, uint8_t *flag_dev, const float *prev_input_dev,
                          int32_t prev_batch, const uint8_t *prev_flag_dev, float *prev_logits_dev,
                          float *prev_S_dev, int32_t *n_rerun, void *stream);

/* One fault of a batched campaign: the arguments of ct_inject. */
typedef struct {
    int32_t kind;        /* ct_buf_kind */
    int32_t layer;       /* index into desc->layers of a convolution */
    int64_t element;     /* literal-layout element, as for ct_inject */
    int32_t bit;
} ct_fault;

/* ct_campaign_batched -- Sec. III-A fault-injection campaign, many faults
 * in ONE launch: for fault f and image n of the batch input_dev
 * [batch, C, H, W] (FP32, device), the result of ct_inject(faults[f]) +
 * ct_infer of that batch, without re-execution:
 *   S_dev[f * batch + n] (FP32), top1_dev[f * batch + n] (int32: argmax of
 *   the logits, lowest index on ties, -1 if any logit is NaN),
 *   flag_dev[f * batch + n] (uint8: NOT(|S - reference| <= tau)).
 * A weight fault (CT_BUF_WEIGHT, a convolution's literal weight layout)
 * touches every image, so all `batch` entries of its row are written.  An
 * activation fault (CT_BUF_ACT, element of [batch, C_tot, H, W] of the
 * second convolution's input) touches one image: only that image's entry is
 * written, the rest of the row is left as it was.
 * Each CTA holds its own copy of the convolution weights in shared memory,
 * flipped for its fault, and runs the whole network for its images; the
 * model's weights are never modified.  Supported networks: FP32, widened
 * (CT_PROTECT_WIDEN), the LeNet-5 shape -- an unpadded stride-1
 * convolution with a carry-through filter, 2x2 stride-2 max-pool, the same
 * again, then FC, FC, classifier, with ReLU after every convolution and
 * hidden FC -- small enough for one CTA's shared memory; CT_EUNSUPPORTED
 * otherwise.  The first convolution's input (the image) is not a fault site.
 * `faults` is host memory, read before the call returns.  Asynchronous on
 * `stream` after one synchronisation (the previous call's fault list).
 * Errors: CT_EINVAL, CT_ERANGE (batch, layer, element or bit out of range),
 * CT_EUNSUPPORTED, CT_ENOMEM, CT_ECUDA. */
ct_status ct_campaign_batched(ct_model *m, const float *input_dev, int32_t batch,
                              const ct_fault *faults, int32_t n_faults, float *S_dev,
                              int32_t *top1_dev, uint8_t *flag_dev, void *stream);

/* ct_reexecute_noalloc -- the same re-execution as ct_reexecute, for callers
 * that must not allocate device memory while they run: real-time loops whose
 * device memory is fixed at start-up so that a request can never fail for
 * want of memory, and plug-ins whose host application owns the device
 * allocator and forbids allocations behind its back.  (The paper has no
 * counterpart; this is a deployment variant of the mitigation step.)
 *
 * It allocates nothing.  ct_reexecute keeps its scratch (the gather index
 * list and the compacted batch of flagged images with their logits, S and
 * flags) in buffers made by ct_build; this entry point keeps that scratch
 * in one static device array of CT_NOALLOC_SCRATCH_BYTES that every GPU
 * loading the library holds until the process exits.  The model's weights
 * and activation workspaces are the ones ct_build allocated.
 *   - The scratch must hold the compacted batch: 256-byte aligned parts of
 *     4*n (indices), 4*n*in_c*in_h*in_w (images), 4*n*n_classes (logits),
 *     4*n (S) and n (flags) bytes for n flagged images.  If it does not,
 *     or batch > 65536, the call returns CT_ERANGE and runs nothing.
 *   - ct_build looks up the array's device address (cudaGetSymbolAddress)
 *     with the model's device current.  That lookup loads the array's
 *     module, which commits its CT_NOALLOC_SCRATCH_BYTES on the device, so
 *     the memory is taken when a model is built, never by this call.
 *   - *n_rerun is the number of images re-run: 0 when the call returns
 *     CT_ERANGE (nothing ran).
 *   - Every call on a device shares the one array and it keeps the last
 *     call's contents; calls that can overlap on the GPU race on it, so
 *     serialise them (one stream, or a wait between streams).  Host-side
 *     flag and index lists are static too: one host thread at a time.
 * Arguments, results and synchronisation are those of ct_reexecute. */
#define CT_NOALLOC_SCRATCH_BYTES (16u * 1024u * 1024u)
ct_status ct_reexecute_noalloc(ct_model *m, const float *input_dev, int32_t batch,
                               const uint8_t *flag_dev, float *logits_dev, float *S_dev,
                               int32_t *n_rerun, void *stream);

/* ct_infer_batches -- Sec. II-B over a list of batches resident on the
 * device: inference and verification of each batch, and re-execution of
 * every flagged image, deferred by two batches (Sec. II-B, last paragraph:
 * re-execute flagged inferences once, ignore the re-run's flag).  Step i
 * infers batch i and re-runs, as extra rows of that same inference, the
 * flagged images of batch i - 2, whose flags the library copied to pinned
 * host memory when that batch's inference ended; the host waits only for
 * that copy, which the device finished while it went on with batch i - 1,
 * so the device never idles for a flag read-back.  The last two batches'
 * flagged images are re-run on their own at the end.
 *   - input_dev[i], logits_dev[i], S_dev[i], flag_dev[i]: host arrays of
 *     n_batches device pointers (FP32 NCHW [batch, C, H, W]; FP32
 *     [batch, n_classes]; FP32 [batch]; uint8 [batch]), as for ct_infer.
 *     Every one must stay valid for the whole call; a re-run row overwrites
 *     its image's logits and S; the flags are the first run's.
 *   - The re-run rows must fit max_batch (batch + flagged images); when they
 *     do not, or a fault is armed, that batch's flagged images are re-run as
 *     by ct_reexecute instead (the armed fault goes to the next inference).
 *   - Returns after every result is final (the call synchronises `stream`).
 *   - *n_rerun (host, may be NULL): images re-run in all.
 * Errors: CT_EINVAL (null arrays or entries), CT_ERANGE (batch outside
 * 1..max_batch), CT_ENOMEM (first call: pinned host memory), CT_ECUDA. */
ct_status ct_infer_batches(ct_model *m, int32_t n_batches, int32_t batch, const float *const *input_dev,
                           float *const *logits_dev, float *const *S_dev, uint8_t *const *flag_dev,
                           int32_t *n_rerun, void *stream);

/* ct_run_host_batches -- ct_infer_batches for callers whose inputs and
 * results live in HOST memory: batch i's input (input_host[i], FP32 NCHW) is
 * copied into one of six library-owned device slots on a library copy
 * stream while the device still works on earlier batches, and its logits
 * (logits_host[i]), S (S_host[i]) and flags (flag_host[i]) are copied back
 * once its re-run rows are written (two batches later).  S_host and
 * flag_host, or any of their entries, may be NULL (not copied back).  With
 * pinned host buffers the copies overlap the inferences; pageable buffers
 * work, serialised.  The first call allocates the device slots (6 x
 * max_batch images and their results) and pinned flag buffers; they live
 * until ct_destroy.  Returns after every result is in host memory.
 * Errors as for ct_infer_batches. */
ct_status ct_run_host_batches(ct_model *m, int32_t n_batches, int32_t batch, const float *const *input_host,
                              float *const *logits_host, float *const *S_host, uint8_t *const *flag_host,
                              int32_t *n_rerun, void *stream);

/* ct_run_host -- end-to-end call for callers with host buffers: copies the
 * input from host memory, runs ct_infer and ct_reexecute, and copies
 * logits, S and flags back.  Returns after the results are in host memory.
 * Pinned host memory gives asynchronous copies; pageable memory works. */
ct_status ct_run_host(ct_model *m, const float *input_host, int32_t batch, float *logits_host,
                      float *S_host, uint8_t *flag_host, int32_t *n_rerun, void *stream);

/* ct_calibrate -- Sec. II-C distribution-based threshold, host arithmetic:
 * reference = mean of the n fault-free S values, tau = the nearest-rank
 * ceil((1 - alpha) * n)-th smallest |S - reference|.  CT_EINVAL for n < 1,
 * alpha outside [0, 1) or a non-finite S. */
ct_status ct_calibrate(const float *S_host, int64_t n, double alpha, double *reference,
                       double *tau);

/* ct_fi_threshold -- Sec. II-C FI-based threshold, host arithmetic: from a
 * fault-injection campaign on calibration inputs, with S_host[i] the
 * accumulated-checksum neuron of image trial i and critical[i] != 0 when
 * the fault changed its top-1 class, tau = the nearest-rank
 * ceil((1 - alpha) * m)-th smallest |S - reference| over the m non-critical
 * trials (a non-finite S counts as an infinite deviation), so that at most
 * alpha of them are flagged.  CT_EINVAL for n < 1, alpha outside [0, 1) or
 * no non-critical trial. */
ct_status ct_fi_threshold(const float *S_host, const uint8_t *critical, int64_t n, double reference,
                          double alpha, double *tau);

/* Fault-able buffers of the protected network for a given batch, in the
 * order used by campaign drivers: every conv weight tensor, then every
 * distinct tensor read by a convolution (the network input excluded),
 * addressed by the first convolution that reads it. */
ct_status ct_buffer_count(const ct_model *m, int32_t batch, int32_t *n);
ct_status ct_buffer_info(const ct_model *m, int32_t batch, int32_t i, int32_t *kind,
                         int32_t *layer, int64_t *n_elements, int32_t *bits);

/* Per-launch kernel timing with CUDA events recorded on the launch stream
 * (off by default).  ct_profile_read returns, for one kernel family, the
 * launches, milliseconds and algorithmic FLOPs accumulated since the last
 * read of that family, then resets it.  It synchronises on the recorded
 * events.  Families: 0 = tensor-core conv, 1 = CUDA-core conv, 2 = FC,
 * 3 = pooling, 4 = other. */
ct_status ct_profile_enable(ct_model *m, int32_t on);
ct_status ct_profile_read(ct_model *m, int32_t family, int64_t *launches, double *ms,
                          double *flops);

/* Number of library kernels the most recent inference of this model
 * launched (fault-injection bit flips not counted); a layer whose K
 * dimension is split across CTAs (small batches) launches two.  Before the
 * first inference: the count without split K. */
ct_status ct_launches_per_infer(const ct_model *m, int32_t *n);

/* ct_kernel_count -- number of library kernels launched for this model since
 * the previous call (directly, or as nodes of the re-execution graphs that
 * ct_reexecute replays), fault-injection bit flips included; resets the
 * count.  Host bookkeeping only: no synchronisation. */
ct_status ct_kernel_count(ct_model *m, int64_t *n);

/* ct_copy_activation -- diagnostic read of an intermediate tensor of the
 * last ct_infer on `stream`: slot `slot` (0 = converted input; the `dst` of
 * a layer otherwise) for the first `batch` images.  data_host receives the
 * data channels in the device layout, NHWC [batch, H, W, C] (FP32 features
 * [batch, C] after a global average pool, [batch, n] after a hidden FC), in
 * the slot's storage type (FP32, or FP16 words as uint16); cs_host (may be
 * NULL) receives the checksum plane [batch, H, W] in the same type.
 * When the first convolution runs on the tensor-core path for images with at
 * most 4 channels, slot 0 is stored with 4 channels (the extra ones zero)
 * and *C reports 4.
 * *C, *H, *W, *has_cs and *elem_bytes describe the slot (any may be NULL; call
 * first with data_host = NULL to query).  Synchronous.  CT_ERANGE for a slot
 * that is not kept (the classifier output) or batch > max_batch; CT_ESTATE
 * for a tensor that a fused kernel computes without storing (slot 0 and the
 * unpooled stem output of a model with a fused stem; the unpooled output of
 * a convolution whose max-pool ran in its kernel in the last inference). */
ct_status ct_copy_activation(ct_model *m, int32_t slot, int32_t batch, void *data_host, void *cs_host,
                             int32_t *C, int32_t *H, int32_t *W, int32_t *has_cs,
                             int32_t *elem_bytes, void *stream);

/* Reads and clears the model's device-side error word (set by a kernel whose
 * bounded wait expired).  Synchronises the model's device. */
ct_status ct_device_error(ct_model *m, uint32_t *code);

void ct_destroy(ct_model *m);
const char *ct_strerror(ct_status s);

#ifdef __cplusplus
}
#endif
#endif /* CT_H */
