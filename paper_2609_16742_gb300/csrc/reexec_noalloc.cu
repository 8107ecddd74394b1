// Re-execution of flagged images without any allocation at call time.
//
// ct_reexecute keeps its gather index list and the compacted batch (input
// images, logits, S, flags of the re-run) in buffers the library allocates
// in ct_build.  ct_reexecute_noalloc does the same work, but that scratch is
// one file-scope device array, g_reexec_scratch, of CT_NOALLOC_SCRATCH_BYTES.
// It is meant for callers that must not allocate device memory while they
// serve requests: real-time loops whose device memory is fixed up front so
// that no request can fail for want of memory, and plug-ins whose host
// application owns the device allocator.  The model itself (weights,
// activation workspaces) is still the one ct_build allocated.
//
// Host code must not pass g_reexec_scratch to a kernel: on the host the name
// stands for a host-side shadow, not a device address.  The device address is
// looked up once per device with cudaGetSymbolAddress, with that device
// current, by ct_build (noalloc_scratch_setup).  The lookup loads this file's
// module, which commits the array on that device; doing it in ct_build keeps
// that commitment out of the calls that serve requests.
#include <string.h>

#include "ct_internal.h"

namespace {

static __device__ __align__(256) unsigned char g_reexec_scratch[CT_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
constexpr int kMaxBatch = 65536;              // host-side flag and index lists
unsigned char *g_scratch_dev[kMaxDevices];    // device address per device, set up once
bool g_scratch_ready[kMaxDevices];
uint8_t g_host_flags[kMaxBatch];
int32_t g_host_idx[kMaxBatch];

size_t up256(size_t x) { return (x + 255) & ~(size_t)255; }

// device address of the array on the current device, looked up once
ct_status lookup(int device) {
    if (g_scratch_ready[device]) return CT_OK;
    void *p = nullptr;
    if (cudaGetSymbolAddress(&p, g_reexec_scratch) != cudaSuccess || p == nullptr) {
        cudaGetLastError();
        return CT_ECUDA;
    }
    g_scratch_dev[device] = static_cast<unsigned char *>(p);
    g_scratch_ready[device] = true;
    return CT_OK;
}

}  // namespace

namespace ct {

ct_status noalloc_scratch_setup(int device) {
    if (device < 0 || device >= kMaxDevices) return CT_EINVAL;
    return lookup(device);
}

}  // namespace ct

extern "C" ct_status ct_reexecute_noalloc(ct_model *m, const float *input_dev, int32_t batch,
                                          const uint8_t *flag_dev, float *logits_dev, float *S_dev,
                                          int32_t *n_rerun, void *stream) {
    if (n_rerun) *n_rerun = 0;
    if (!m || !input_dev || !flag_dev || !logits_dev) return CT_EINVAL;
    ct::ModelInfo mi;
    ct_status s = ct::model_info(m, &mi);
    if (s != CT_OK) return s;
    if (batch < 1 || batch > mi.max_batch || batch > kMaxBatch) return CT_ERANGE;
    if (mi.device < 0 || mi.device >= kMaxDevices) return CT_EINVAL;
    int prev = -1;
    if (cudaGetDevice(&prev) != cudaSuccess) return CT_ECUDA;
    if (prev != mi.device && cudaSetDevice(mi.device) != cudaSuccess) return CT_ECUDA;
    struct Restore {
        int dev, prev;
        ~Restore() { if (prev >= 0 && prev != dev) cudaSetDevice(prev); }
    } restore{mi.device, prev};

    // ct_build looked the address up for this device; the lookup here only
    // runs if that failed to happen (it is a no-op otherwise)
    if ((s = lookup(mi.device)) != CT_OK) return s;
    unsigned char *base = g_scratch_dev[mi.device];
    cudaStream_t st = (cudaStream_t)stream;

    // which images to re-run (host compaction, as in ct_reexecute)
    if (cudaMemcpyAsync(g_host_flags, flag_dev, batch, cudaMemcpyDeviceToHost, st) != cudaSuccess ||
        cudaStreamSynchronize(st) != cudaSuccess)
        return CT_ECUDA;
    int n = 0;
    for (int i = 0; i < batch; ++i)
        if (g_host_flags[i]) g_host_idx[n++] = i;
    if (n == 0) return CT_OK;

    // scratch layout: index list | compacted images | logits | S | flags
    const int64_t per = (int64_t)mi.in_c * mi.in_h * mi.in_w;
    const size_t off_idx = 0;
    const size_t off_in = up256(off_idx + sizeof(int32_t) * n);
    const size_t off_lg = up256(off_in + sizeof(float) * per * n);
    const size_t off_S = up256(off_lg + sizeof(float) * (size_t)mi.n_classes * n);
    const size_t off_fl = up256(off_S + sizeof(float) * n);
    const size_t need = off_fl + (size_t)n;
    if (need > (size_t)CT_NOALLOC_SCRATCH_BYTES) return CT_ERANGE;
    if (n_rerun) *n_rerun = n;
    int32_t *idx = reinterpret_cast<int32_t *>(base + off_idx);
    float *cin = reinterpret_cast<float *>(base + off_in);
    float *clg = reinterpret_cast<float *>(base + off_lg);
    float *cS = reinterpret_cast<float *>(base + off_S);
    uint8_t *cfl = reinterpret_cast<uint8_t *>(base + off_fl);

    if (cudaMemcpyAsync(idx, g_host_idx, sizeof(int32_t) * n, cudaMemcpyHostToDevice, st) != cudaSuccess)
        return CT_ECUDA;
    if (ct::reexec_gather(m, input_dev, cin, idx, n, per, st) != cudaSuccess) return CT_ECUDA;
    s = ct::infer_fault_free(m, cin, n, clg, cS, cfl, st);
    if (s != CT_OK) return s;
    if (ct::reexec_scatter(m, clg, logits_dev, idx, n, mi.n_classes, st) != cudaSuccess) return CT_ECUDA;
    if (S_dev && ct::reexec_scatter(m, cS, S_dev, idx, n, 1, st) != cudaSuccess) return CT_ECUDA;
    return CT_OK;
}
