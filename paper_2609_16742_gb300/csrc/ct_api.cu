// libct C ABI: model construction (Sec. II-A/II-B), inference orchestration,
// fault injection (Sec. III-A), re-execution (Sec. II-B) and calibration
// (Sec. II-C).  Every arithmetic step of inference runs in this library's
// CUDA kernels; the host only builds weights and launches.
#include <math.h>
#include <string.h>

#include <algorithm>
#include <memory>
#include <new>
#include <vector>

#include "ct_internal.h"

using namespace ct;

namespace {

// ---------------------------------------------------------------------------
// storage rounding (host)
// ---------------------------------------------------------------------------

// IEEE binary64 -> binary16, round to nearest even, directly (no float step).
uint16_t double_to_half_bits(double d) {
    uint64_t u;
    memcpy(&u, &d, 8);
    const uint16_t sign = (uint16_t)((u >> 48) & 0x8000u);
    const uint64_t mag = u & 0x7FFFFFFFFFFFFFFFull;
    if (mag >= 0x7FF0000000000000ull) return sign | (mag > 0x7FF0000000000000ull ? 0x7E00 : 0x7C00);
    const int e = (int)(mag >> 52) - 1023;
    if (e == -1023) return sign;                                // binary64 subnormal: below half's range
    const uint64_t full = (mag & ((1ull << 52) - 1)) | (1ull << 52);   // 53-bit significand
    if (e >= 16) return sign | 0x7C00;
    if (e >= -14) {                                             // half normal range
        uint64_t hm = full >> 42, rem = full & ((1ull << 42) - 1), hlf = 1ull << 41;
        int ee = e;
        if (rem > hlf || (rem == hlf && (hm & 1))) ++hm;
        if (hm == 2048) { hm = 1024; ++ee; }
        if (ee >= 16) return sign | 0x7C00;
        return (uint16_t)(sign | ((ee + 15) << 10) | (hm & 0x3FF));
    }
    const int shift = 28 - e;                                   // value / 2^-24 = full >> shift
    if (shift >= 54) return sign;
    uint64_t m = full >> shift, rem = full & ((1ull << shift) - 1), hlf = 1ull << (shift - 1);
    if (rem > hlf || (rem == hlf && (m & 1))) ++m;
    return (uint16_t)(sign | m);                               // m == 1024 encodes 2^-14
}

float half_bits_to_float(uint16_t h) {
    const uint32_t sign = (uint32_t)(h & 0x8000) << 16;
    const uint32_t e = (h >> 10) & 0x1F, m = h & 0x3FF;
    uint32_t bits;
    if (e == 0x1F) bits = sign | 0x7F800000u | (m << 13);
    else if (e == 0) {
        if (m == 0) bits = sign;
        else {
            float v = ldexpf((float)m, -24);
            memcpy(&bits, &v, 4);
            bits |= sign;
        }
    } else bits = sign | ((e + 112) << 23) | (m << 13);
    float f;
    memcpy(&f, &bits, 4);
    return f;
}

uint32_t float_bits(float f) { uint32_t u; memcpy(&u, &f, 4); return u; }
float bits_float(uint32_t u) { float f; memcpy(&f, &u, 4); return f; }

// ---------------------------------------------------------------------------
// model
// ---------------------------------------------------------------------------

struct Slot {
    int C = 0, H = 0, W = 0;
    int cp = 0;                  // channel pitch of the NHWC data (C, or 4 for a padded image)
    bool has_cs = false;
    bool is_float = false;       // GAP output: fp32 features whatever the precision
    bool stored = true;          // false: computed inside a fused kernel, never in HBM
    bool skipped_last = false;   // the last inference computed its reader (a fused max-pool) without storing it
    void *data = nullptr;
    void *cs = nullptr;
};

struct LayerRT {
    ct_layer_desc d{};
    int role = CT_ROLE_NONE;     // effective role (protect / ds_mode applied)
    // conv
    int C = 0, K = 0, R = 0, S = 0, H = 0, W = 0, P = 0, Q = 0;
    bool cs_in = false, cs_out = false;
    float coef = 1.f;
    void *w = nullptr;
    float *bias = nullptr;
    bool tc = false;
    TcPlan *plan = nullptr;
    HaloPlan *hplan = nullptr;   // stride-1 3x3 layers: halo tiles when the batch fills the GPU
    bool tc_small = false;       // first layer with <= 4 input channels on the tensor cores
    TcSmallPlan *splan = nullptr;
    bool stem = false;           // fused image stem: this conv and the max-pool after it
    StemPlan *stplan = nullptr;
    bool fused = false;          // max-pool computed by the preceding fused stem
    bool pool_fuse = false;      // conv: its halo kernel applies the 2 x 2 max-pool that follows (layer + 1)
    bool sc_next = false;        // conv: layer + 1 is a 1x1 shortcut of the same input that may run in this
                                 // layer's launch (its A operand is this layer's centre tap)
    int w_ld = 0, c_stride = 0;  // weight row length and channel stride within a tap
    // fc
    int n_in = 0, n_cs = 0, n_out = 0;
    bool x_float = false;
    bool fc_tc = false;          // hidden FC run on the tensor-core conv kernel as a 1x1 conv
    bool dw = false;             // depthwise convolution: weights [R*S][C]
};

// input channels a filter of this convolution spans in the literal layout
int weight_in_channels(const LayerRT &l) { return l.dw ? 1 : l.C + (l.cs_in ? 1 : 0); }

struct EvRec { int fam; int ev; double flops; int nk; };

// split-K workspace of a model (FP32 partial sums of one layer at a time)
constexpr size_t SPLITK_WS_BYTES = 32ull << 20;

}  // namespace

struct ct_model {
    int device = 0;
    int prec = CT_FP32;
    bool protect = true;         // widened construction: checksum planes beside the tensors
    bool replace = false;        // replace construction: checksum inside the pruned tensors
    int ds_mode = CT_DS_PASS;
    int max_batch = 0;
    uint32_t flags = 0;
    int in_c = 0, in_h = 0, in_w = 0, n_classes = 0;
    std::vector<LayerRT> L;
    std::vector<Slot> slots;
    double ref = 0.0, tau = INFINITY;
    // armed fault
    bool armed = false;
    int f_kind = 0, f_layer = 0, f_bit = 0;
    int64_t f_elem = 0;
    // scratch owned by the library
    float *re_input = nullptr, *re_logits = nullptr, *re_S = nullptr;
    uint8_t *re_flag = nullptr;
    int32_t *re_idx = nullptr;
    uint8_t *h_flags = nullptr;
    int32_t *h_idx = nullptr;          // host memory mapped for the device
    int32_t *h_idx_d = nullptr;        // its device address
    // batched campaign: resolved faults (device) and their pinned staging
    CampFault *camp_d = nullptr, *camp_h = nullptr;
    int camp_cap = 0;
    float *rh_input = nullptr, *rh_logits = nullptr, *rh_S = nullptr;
    uint8_t *rh_flag = nullptr;
    uint32_t *d_err = nullptr;
    float *ws = nullptr;         // split-K partial sums
    // re-execution: one captured inference graph per power-of-two batch
    cudaStream_t cap_stream = nullptr;
    std::vector<cudaGraphExec_t> re_graph;
    std::vector<int> re_graph_nk;        // kernels in each graph
    int64_t kernels_total = 0;           // kernels launched since the last ct_kernel_count
    int n_kernels_last = -1;     // kernels launched by the last inference
    bool small = false;          // the whole network runs as one kernel (LeNet-5 shape)
    uint8_t *flag_mirror = nullptr;   // set by run_batches: the final kernel also writes the flags here
    double small_flops = 0;      // its convolutions' multiply-adds per image
    int n_kernels_run = 0;
    std::vector<void *> dev_allocs;
    // ct_infer_batches / ct_run_host_batches: per pipeline slot a pinned copy
    // of the batch's flags, a pinned index list, events; a copy stream and
    // (host buffers) device slots for inputs and results; made on first use
    static constexpr int PIPE = 6;
    uint8_t *pipe_flags_h = nullptr;      // [PIPE][max_batch], host memory mapped for the device
    uint8_t *pipe_flags_d = nullptr;      // its device address
    int32_t *pipe_idx_h = nullptr;        // [PIPE + 2][max_batch], host memory mapped for the device
    int32_t *pipe_idx_d = nullptr;        // its device address
    cudaEvent_t pipe_ev_flags[PIPE] = {}, pipe_ev_step[PIPE] = {}, pipe_ev_in[PIPE] = {}, pipe_ev_out[PIPE] = {};
    cudaEvent_t pipe_ev_tail = nullptr;
    bool pipe_ready = false;
    cudaStream_t pipe_copy = nullptr;     // input copies
    cudaStream_t pipe_copy_out = nullptr; // result copies
    float *pipe_in_d = nullptr, *pipe_lg_d = nullptr, *pipe_S_d = nullptr;
    uint8_t *pipe_fl_d = nullptr;
    // profiling
    bool prof = false;
    std::vector<std::pair<cudaEvent_t, cudaEvent_t>> ev_pool;
    std::vector<int> ev_free;
    std::vector<EvRec> recs;

    size_t esz() const { return prec == CT_FP16 ? 2 : 4; }
};

namespace {

#define CUDA_TRY(x)                                   \
    do {                                              \
        cudaError_t e__ = (x);                        \
        if (e__ != cudaSuccess) return CT_ECUDA;      \
    } while (0)

struct DeviceGuard {
    int prev = -1;
    explicit DeviceGuard(int dev) {
        if (cudaGetDevice(&prev) != cudaSuccess) prev = -1;
        cudaSetDevice(dev);
    }
    ~DeviceGuard() { if (prev >= 0) cudaSetDevice(prev); }
};

ct_status dalloc(ct_model *m, void **p, size_t bytes) {
    if (bytes == 0) bytes = 16;
    if (cudaMalloc(p, bytes) != cudaSuccess) { cudaGetLastError(); return CT_ENOMEM; }
    m->dev_allocs.push_back(*p);
    return CT_OK;
}

void free_all(ct_model *m) {
    for (auto &l : m->L) {
        if (l.plan) tc_plan_destroy(l.plan);
        if (l.splan) tc_small_plan_destroy(l.splan);
        if (l.stplan) stem_plan_destroy(l.stplan);
        if (l.hplan) halo_plan_destroy(l.hplan);
    }
    for (void *p : m->dev_allocs) cudaFree(p);
    m->dev_allocs.clear();
    if (m->h_flags) cudaFreeHost(m->h_flags);
    if (m->camp_h) cudaFreeHost(m->camp_h);
    if (m->camp_d) cudaFree(m->camp_d);
    if (m->h_idx) cudaFreeHost(m->h_idx);
    for (auto &e : m->ev_pool) { cudaEventDestroy(e.first); cudaEventDestroy(e.second); }
    m->ev_pool.clear();
    for (cudaGraphExec_t g : m->re_graph)
        if (g) cudaGraphExecDestroy(g);
    m->re_graph.clear();
    if (m->cap_stream) cudaStreamDestroy(m->cap_stream);
    m->cap_stream = nullptr;
    if (m->pipe_flags_h) cudaFreeHost(m->pipe_flags_h);
    if (m->pipe_idx_h) cudaFreeHost(m->pipe_idx_h);
    m->pipe_flags_h = nullptr;
    m->pipe_idx_h = nullptr;
    m->pipe_idx_d = nullptr;
    for (int i = 0; i < ct_model::PIPE; ++i)
        for (cudaEvent_t *e : {&m->pipe_ev_flags[i], &m->pipe_ev_step[i], &m->pipe_ev_in[i], &m->pipe_ev_out[i]})
            if (*e) { cudaEventDestroy(*e); *e = nullptr; }
    if (m->pipe_ev_tail) cudaEventDestroy(m->pipe_ev_tail);
    m->pipe_ev_tail = nullptr;
    if (m->pipe_copy) cudaStreamDestroy(m->pipe_copy);
    if (m->pipe_copy_out) cudaStreamDestroy(m->pipe_copy_out);
    m->pipe_copy = m->pipe_copy_out = nullptr;
}

// store a double as the storage word (fp32 or fp16) into a byte buffer
void put(std::vector<uint8_t> &buf, size_t i, double v, int prec) {
    if (prec == CT_FP16) {
        uint16_t h = double_to_half_bits(v);
        memcpy(&buf[i * 2], &h, 2);
    } else {
        float f = (float)v;
        memcpy(&buf[i * 4], &f, 4);
    }
}

// value of a storage word after flipping `bit`, as float
float flipped(double stored, int bit, int prec) {
    if (prec == CT_FP16) return half_bits_to_float((uint16_t)(double_to_half_bits(stored) ^ (1u << bit)));
    return bits_float(float_bits((float)stored) ^ (1u << bit));
}

// stored word of data-filter weight (k, r, s, c) in the device weight array
int64_t weight_word(const LayerRT &l, int k, int r, int s, int c) {
    if (l.dw) return ((int64_t)r * l.S + s) * l.C + k;      // c is 0: the filter's one channel
    if (l.stem) return (int64_t)k * l.w_ld + stem_kidx(r, s, c);
    return (int64_t)k * l.w_ld + ((int64_t)r * l.S + s) * l.c_stride + c;
}

// ---------------------------------------------------------------------------
// profiling helpers
// ---------------------------------------------------------------------------

// fault-injection bit flip (counted, not timed)
cudaError_t xor_bit(ct_model *m, void *base, int64_t word, int bit, int word_bytes, cudaStream_t st) {
    ++m->kernels_total;
    return launch_xor_bit(base, word, bit, word_bytes, st);
}

template <typename F>
cudaError_t launch(ct_model *m, int fam, double flops, cudaStream_t st, F &&fn, const int *nk = nullptr) {
    if (!m->prof) {
        cudaError_t e = fn();
        m->n_kernels_run += nk ? *nk : 1;
        m->kernels_total += nk ? *nk : 1;
        return e;
    }
    int ev;
    if (!m->ev_free.empty()) { ev = m->ev_free.back(); m->ev_free.pop_back(); }
    else {
        cudaEvent_t a, b;
        if (cudaEventCreate(&a) != cudaSuccess) return cudaErrorMemoryAllocation;
        if (cudaEventCreate(&b) != cudaSuccess) { cudaEventDestroy(a); return cudaErrorMemoryAllocation; }
        m->ev_pool.push_back({a, b});
        ev = (int)m->ev_pool.size() - 1;
    }
    cudaEventRecord(m->ev_pool[ev].first, st);
    cudaError_t e = fn();
    cudaEventRecord(m->ev_pool[ev].second, st);
    const int n = nk ? *nk : 1;
    m->recs.push_back({fam, ev, flops, n});
    m->n_kernels_run += n;
    m->kernels_total += n;
    return e;
}

// ---------------------------------------------------------------------------
// build
// ---------------------------------------------------------------------------

// Replace construction (Sec. II-A): per slot, the output channel pruned to
// make room for the carry-through filter (-1: none).  Slots tied by a
// residual add, a max-pool or the global average pool form one stream with
// one index: the channel whose combined L1 norm over the stream's writers
// (their output filters, before BatchNorm folding) and readers (their input
// slices; an FC reader's H*W columns of the channel) is smallest, the lowest
// such index on ties.  The network input and the classifier output are not
// pruned.
std::vector<int> replace_prune_index(const ct_model_desc *desc, const float *const *wts, int n_slots) {
    const int nL = desc->n_layers;
    std::vector<int> parent(n_slots);
    for (int i = 0; i < n_slots; ++i) parent[i] = i;
    auto find = [&](int a) {
        while (parent[a] != a) a = parent[a] = parent[parent[a]];
        return a;
    };
    auto unite = [&](int a, int b) {
        a = find(a); b = find(b);
        if (a != b) parent[std::max(a, b)] = std::min(a, b);
    };
    std::vector<int> ch(n_slots, 0), hw(n_slots, 1);
    ch[0] = desc->in_c;
    std::vector<int> H(n_slots, 0), W(n_slots, 0);
    H[0] = desc->in_h; W[0] = desc->in_w;
    int final_dst = -1;
    for (int i = 0; i < nL; ++i) {
        const ct_layer_desc &d = desc->layers[i];
        if (d.op == CT_OP_CONV) {
            ch[d.dst] = d.cout;
            H[d.dst] = (H[d.src] + 2 * d.pad - d.k) / d.stride + 1;
            W[d.dst] = (W[d.src] + 2 * d.pad - d.k) / d.stride + 1;
            if (d.res >= 0) unite(d.dst, d.res);
        } else if (d.op == CT_OP_MAXPOOL) {
            ch[d.dst] = ch[d.src];
            H[d.dst] = (H[d.src] + 2 * d.pad - d.k) / d.stride + 1;
            W[d.dst] = (W[d.src] + 2 * d.pad - d.k) / d.stride + 1;
            unite(d.dst, d.src);
        } else if (d.op == CT_OP_GAP) {
            ch[d.dst] = ch[d.src]; H[d.dst] = W[d.dst] = 1;
            unite(d.dst, d.src);
        } else {
            ch[d.dst] = d.cout; H[d.dst] = W[d.dst] = 1;
            if (d.final) final_dst = d.dst;
        }
    }
    std::vector<std::vector<double>> score(n_slots);
    auto add = [&](int slot, int c, double v) {
        const int r = find(slot);
        if (r == find(0) || (final_dst >= 0 && r == find(final_dst))) return;
        if ((int)score[r].size() < ch[slot]) score[r].resize(ch[slot], 0.0);
        score[r][c] += v;
    };
    for (int i = 0; i < nL; ++i) {
        const ct_layer_desc &d = desc->layers[i];
        const float *w = wts[CT_WEIGHTS_PER_LAYER * i];
        if (!w) continue;
        if (d.op == CT_OP_CONV) {
            if (d.groups > 1) continue;
            const int RS = d.k * d.k;
            for (int k = 0; k < d.cout; ++k)
                for (int c = 0; c < d.cin; ++c) {
                    double a = 0.0;
                    for (int t = 0; t < RS; ++t) a += fabs((double)w[((size_t)k * d.cin + c) * RS + t]);
                    add(d.dst, k, a);
                    add(d.src, c, a);
                }
        } else if (d.op == CT_OP_FC) {
            const int C = ch[d.src], P = H[d.src] * W[d.src];
            for (int j = 0; j < d.cout; ++j)
                for (int c = 0; c < C; ++c) {
                    double a = 0.0;
                    for (int p = 0; p < P; ++p) a += fabs((double)w[(size_t)j * d.cin + (size_t)c * P + p]);
                    if (!d.final) add(d.dst, j, a);
                    add(d.src, c, a);
                }
        }
    }
    std::vector<int> out(n_slots, -1);
    for (int sl = 0; sl < n_slots; ++sl) {
        const std::vector<double> &v = score[find(sl)];
        if (v.empty()) continue;
        int best = 0;
        for (int c = 1; c < (int)v.size(); ++c)
            if (v[c] < v[best]) best = c;
        out[sl] = best;
    }
    return out;
}

// Sec. II-A, residual networks: a convolution whose input tensor is also
// read by another layer (the shortcut of a residual block) gets no
// carry-through filter, because that tensor's checksum already reaches the
// block's residual add along the shortcut; a filter on the other path would
// add it a second time.  Resolves CT_ROLE_AUTO per convolution into roles[i]
// (one whose input has another reader: the shortcut, PASS, if its output
// goes to nothing but a residual add, else NONE; otherwise CT) and rejects
// an explicit CT_ROLE_CT that the rule forbids.  roles[i] is -1 for layers
// that are not convolutions.
ct_status resolve_roles(const ct_model_desc *desc, int32_t *roles) {
    const int nL = desc->n_layers;
    int max_slot = 0;
    for (int i = 0; i < nL; ++i) {
        const ct_layer_desc &d = desc->layers[i];
        if (d.src < 0 || d.dst <= 0 || d.res < -1) return CT_EINVAL;
        max_slot = std::max(max_slot, std::max(std::max(d.dst, d.src), d.res));
    }
    std::vector<int> readers(max_slot + 1, 0), is_res(max_slot + 1, 0);
    for (int i = 0; i < nL; ++i) {
        const ct_layer_desc &d = desc->layers[i];
        ++readers[d.src];
        if (d.res >= 0) { ++readers[d.res]; is_res[d.res] = 1; }
    }
    for (int i = 0; i < nL; ++i) {
        const ct_layer_desc &d = desc->layers[i];
        roles[i] = -1;
        if (d.op != CT_OP_CONV) continue;
        const bool shared_input = readers[d.src] > 1;
        int r = d.role;
        if (r == CT_ROLE_AUTO)
            r = !shared_input ? CT_ROLE_CT : (is_res[d.dst] && readers[d.dst] == 1) ? CT_ROLE_PASS : CT_ROLE_NONE;
        if (r < CT_ROLE_CT || r > CT_ROLE_PASS) return CT_EINVAL;
        if (r == CT_ROLE_CT && shared_input) return CT_EINVAL;
        roles[i] = r;
    }
    return CT_OK;
}

static bool small_net_of(const ct_model *m, SmallNet *g);

ct_status build_impl(ct_model *m, const ct_model_desc *desc, const float *const *wts) {
    const int nL = desc->n_layers;
    int max_slot = 0;
    for (int i = 0; i < nL; ++i) {
        const ct_layer_desc &d = desc->layers[i];
        if (d.src < 0 || d.dst <= 0) return CT_EINVAL;
        max_slot = std::max(max_slot, std::max(d.dst, d.src));
    }
    std::vector<int> defined(max_slot + 1, 0);
    m->slots.assign(max_slot + 1, Slot());
    Slot &in = m->slots[0];
    in.C = desc->in_c; in.H = desc->in_h; in.W = desc->in_w;
    defined[0] = 1;
    const int prec = m->prec;
    const size_t esz = m->esz();
    const int B = m->max_batch;
    int n_final = 0;
    // replace construction: pruned channel per slot (-1 elsewhere and in the other
    // modes).  Its scores read every weight as a dense [cout, cin, k, k] array, so
    // grouped convolutions are rejected before any weight is read.
    if (m->replace)
        for (int i = 0; i < nL; ++i)
            if (desc->layers[i].op == CT_OP_CONV && desc->layers[i].groups > 1) return CT_EUNSUPPORTED;
    const std::vector<int> pj = m->replace ? replace_prune_index(desc, wts, max_slot + 1)
                                           : std::vector<int>(max_slot + 1, -1);
    std::vector<int32_t> roles(nL);
    if (resolve_roles(desc, roles.data()) != CT_OK) return CT_EINVAL;

    for (int i = 0; i < nL; ++i) {
        const ct_layer_desc &d = desc->layers[i];
        if (!defined[d.src] || defined[d.dst]) return CT_EINVAL;
        if (d.res >= 0 && (d.res > max_slot || !defined[d.res])) return CT_EINVAL;
        Slot &src = m->slots[d.src];
        Slot &dst = m->slots[d.dst];
        LayerRT l;
        l.d = d;
        if (d.op == CT_OP_CONV) l.d.role = roles[i];
        const float *W = wts[CT_WEIGHTS_PER_LAYER * i + 0];
        const float *bias = wts[CT_WEIGHTS_PER_LAYER * i + 1];
        if (d.op == CT_OP_CONV) {
            if (src.is_float || d.cin != src.C || d.k < 1 || d.stride < 1 || d.pad < 0 || d.cout < 1 || !W)
                return CT_EINVAL;
            const int groups = d.groups < 1 ? 1 : d.groups;
            l.dw = groups > 1;
            if (l.dw && (groups != d.cin || groups != d.cout || m->replace || !dw_supported(d.cin, d.cout, prec == CT_FP16)))
                return CT_EUNSUPPORTED;
            int role = m->protect ? l.d.role : CT_ROLE_NONE;
            if (role == CT_ROLE_PASS && m->ds_mode == CT_DS_ZERO && !l.dw) role = CT_ROLE_NONE;
            if (role < CT_ROLE_CT || role > CT_ROLE_PASS) return CT_EINVAL;
            // depthwise: the checksum group passes the incoming checksum through
            if (l.dw) role = (role != CT_ROLE_NONE && src.has_cs) ? CT_ROLE_PASS : CT_ROLE_NONE;
            l.role = role;
            l.C = d.cin; l.K = d.cout; l.R = l.S = d.k;
            l.H = src.H; l.W = src.W;
            l.P = (src.H + 2 * d.pad - d.k) / d.stride + 1;
            l.Q = (src.W + 2 * d.pad - d.k) / d.stride + 1;
            if (l.P < 1 || l.Q < 1) return CT_EINVAL;
            l.cs_in = src.has_cs;
            const bool res_cs = d.res >= 0 && m->slots[d.res].has_cs;
            if (d.res >= 0) {
                const Slot &r = m->slots[d.res];
                if (r.C != l.K || r.H != l.P || r.W != l.Q || r.is_float) return CT_EINVAL;
            }
            l.cs_out = role == CT_ROLE_CT || role == CT_ROLE_PASS || res_cs;
            l.coef = ldexpf(1.f, -d.ct_shift);
            dst.C = l.K; dst.H = l.P; dst.W = l.Q; dst.has_cs = l.cs_out;
            // ---- weights: BN fold in double (Eq. 1); the checksum channel keeps
            // scale 1 and bias 0 because its filter is never folded ----
            const int RSC = l.R * l.S * l.C;
            std::string why;
            l.tc = !l.dw && prec == CT_FP16 && !(m->flags & CT_FLAG_SIMT_ONLY) &&
                   tc_supported(l.C, l.K, l.R, l.S, d.stride, d.pad, &why);
            if (!l.dw && prec == CT_FP16 && !(m->flags & CT_FLAG_SIMT_ONLY) && d.src == 0 && d.res < 0 && i + 1 < nL &&
                stem_pool_supported(l.C, l.K, l.R, l.S, d.stride, d.pad, l.H, l.W)) {
                // the image and the unpooled output must have no other reader
                const ct_layer_desc &nx = desc->layers[i + 1];
                int readers_in = 0, readers_mid = 0;
                for (int j = 0; j < nL; ++j) {
                    readers_in += (desc->layers[j].src == 0) + (desc->layers[j].res == 0);
                    readers_mid += (desc->layers[j].src == d.dst) + (desc->layers[j].res == d.dst);
                }
                l.stem = nx.op == CT_OP_MAXPOOL && nx.src == d.dst && nx.k == 3 && nx.stride == 2 &&
                         nx.pad == 1 && readers_in == 1 && readers_mid == 1;
                if (l.stem) { src.stored = false; dst.stored = false; }
            }
            if (!l.dw && !l.stem && prec == CT_FP16 && !(m->flags & CT_FLAG_SIMT_ONLY) && d.src == 0 &&
                tc_small_supported(l.C, l.K, l.R, l.S, d.stride, d.pad)) {
                int readers = 0;               // the padded image must have no other reader
                for (int j = 0; j < nL; ++j)
                    readers += (desc->layers[j].src == 0) + (desc->layers[j].res == 0);
                l.tc_small = readers == 1;
            }
            if (l.stem) l.tc = false;
            l.w_ld = l.dw ? l.R * l.S : l.stem ? stem_klen() : l.tc_small ? tc_small_kpad(l.R, l.S) : RSC;
            l.c_stride = l.tc_small ? 4 : l.C;
            if (l.tc_small) src.cp = 4;
            std::vector<uint8_t> hw((size_t)l.K * l.w_ld * esz, 0);
            std::vector<float> hb(l.K, 0.f);
            // replace construction: stored output channel kk holds original
            // channel kk (+1 past the pruned one); the last holds the
            // carry-through filter (zero for a block's first convolution,
            // pass-through for the shortcut); stored input channel cc likewise,
            // the last (the incoming checksum) being a zero slice
            const int jo = pj[d.dst], ji = pj[d.src];
            if (jo >= 0) {
                const int ctr = (l.R - 1) / 2;
                const int kk = l.K - 1;
                for (int cc = 0; cc < l.C; ++cc) {
                    double v = 0.0;
                    if (l.d.role == CT_ROLE_CT) v = l.coef;
                    else if (l.d.role == CT_ROLE_PASS && m->ds_mode == CT_DS_PASS && cc == l.C - 1 && ji >= 0) v = 1.0;
                    if (v != 0.0) put(hw, (size_t)weight_word(l, kk, ctr, ctr, cc), v, prec);
                }
            }
            for (int kk = 0; kk < l.K - (jo >= 0 ? 1 : 0); ++kk) {
                const int k = (jo >= 0 && kk >= jo) ? kk + 1 : kk;
                double scale = 1.0, shift = bias ? (double)bias[k] : 0.0;
                if (d.bn) {
                    const float *g = wts[CT_WEIGHTS_PER_LAYER * i + 2], *be = wts[CT_WEIGHTS_PER_LAYER * i + 3];
                    const float *mu = wts[CT_WEIGHTS_PER_LAYER * i + 4], *var = wts[CT_WEIGHTS_PER_LAYER * i + 5];
                    if (!g || !be || !mu || !var) return CT_EINVAL;
                    scale = (double)g[k] / sqrt((double)var[k] + desc->bn_eps);
                    double t = (shift - (double)mu[k]) * scale;
                    shift = t + (double)be[k];
                }
                hb[kk] = (float)shift;
                if (l.dw) {
                    for (int r = 0; r < l.R; ++r)
                        for (int s = 0; s < l.S; ++s)
                            put(hw, (size_t)weight_word(l, kk, r, s, 0),
                                (double)W[((size_t)k * l.R + r) * l.S + s] * scale, prec);
                    continue;
                }
                for (int cc = 0; cc < l.C - (ji >= 0 ? 1 : 0); ++cc) {
                    const int c = (ji >= 0 && cc >= ji) ? cc + 1 : cc;
                    for (int r = 0; r < l.R; ++r)
                        for (int s = 0; s < l.S; ++s) {
                            double v = (double)W[(((size_t)k * l.C + c) * l.R + r) * l.S + s] * scale;
                            put(hw, (size_t)weight_word(l, kk, r, s, cc), v, prec);
                        }
                }
            }
            ct_status st;
            if ((st = dalloc(m, &l.w, hw.size())) != CT_OK) return st;
            if ((st = dalloc(m, (void **)&l.bias, sizeof(float) * l.K)) != CT_OK) return st;
            CUDA_TRY(cudaMemcpy(l.w, hw.data(), hw.size(), cudaMemcpyHostToDevice));
            CUDA_TRY(cudaMemcpy(l.bias, hb.data(), sizeof(float) * l.K, cudaMemcpyHostToDevice));
        } else if (d.op == CT_OP_MAXPOOL) {
            if (src.is_float || d.k < 1 || d.stride < 1 || d.pad < 0 || d.pad >= d.k) return CT_EINVAL;
            l.fused = !m->L.empty() && m->L.back().stem && m->L.back().d.dst == d.src;
            dst.C = src.C;
            dst.H = (src.H + 2 * d.pad - d.k) / d.stride + 1;
            dst.W = (src.W + 2 * d.pad - d.k) / d.stride + 1;
            dst.has_cs = src.has_cs;
            if (dst.H < 1 || dst.W < 1) return CT_EINVAL;
        } else if (d.op == CT_OP_GAP) {
            if (src.is_float) return CT_EINVAL;
            dst.C = src.C; dst.H = dst.W = 1; dst.has_cs = src.has_cs; dst.is_float = true;
        } else if (d.op == CT_OP_FC) {
            const int HW = src.H * src.W;
            if (d.cin != src.C * HW || d.cout < 1 || !W) return CT_EINVAL;
            l.n_in = d.cin; l.n_out = d.cout;
            l.n_cs = src.has_cs ? HW : 0;
            l.x_float = src.is_float;
            l.coef = ldexpf(1.f, -d.ct_shift);
            if (d.final) { ++n_final; if (d.cout != desc->n_classes || i != nL - 1) return CT_EINVAL; }
            dst.C = l.n_out; dst.H = dst.W = 1;
            dst.has_cs = m->protect && !d.final;
            std::string why;
            l.fc_tc = prec == CT_FP16 && !(m->flags & CT_FLAG_SIMT_ONLY) && !d.final && !src.is_float &&
                      tc_supported(l.n_in, l.n_out, 1, 1, 1, 0, &why);
            // weights: columns permuted from (c, h, w) to the NHWC flatten (h, w, c)
            std::vector<uint8_t> hw((size_t)l.n_out * l.n_in * esz, 0);
            std::vector<float> hb(l.n_out, 0.f);
            // replace construction: neuron jj holds original neuron jj (+1 past
            // the pruned one), the last a carry-through neuron of weight coef;
            // input channel cc likewise, the last (checksum) zero in every
            // normal neuron.  The classifier keeps its neurons; its
            // accumulated-checksum neuron is computed by the FC kernel.
            const int jo = d.final ? -1 : pj[d.dst], ji = pj[d.src];
            if (jo >= 0)
                for (int q = 0; q < l.n_in; ++q) put(hw, (size_t)(l.n_out - 1) * l.n_in + q, l.coef, prec);
            for (int jj = 0; jj < l.n_out - (jo >= 0 ? 1 : 0); ++jj) {
                const int j = (jo >= 0 && jj >= jo) ? jj + 1 : jj;
                hb[jj] = bias ? bias[j] : 0.f;
                for (int cc = 0; cc < src.C - (ji >= 0 ? 1 : 0); ++cc) {
                    const int c = (ji >= 0 && cc >= ji) ? cc + 1 : cc;
                    for (int p = 0; p < HW; ++p)
                        put(hw, (size_t)jj * l.n_in + (size_t)p * src.C + cc,
                            (double)W[(size_t)j * l.n_in + (size_t)c * HW + p], prec);
                }
            }
            ct_status st;
            if ((st = dalloc(m, &l.w, hw.size())) != CT_OK) return st;
            if ((st = dalloc(m, (void **)&l.bias, sizeof(float) * l.n_out)) != CT_OK) return st;
            CUDA_TRY(cudaMemcpy(l.w, hw.data(), hw.size(), cudaMemcpyHostToDevice));
            CUDA_TRY(cudaMemcpy(l.bias, hb.data(), sizeof(float) * l.n_out, cudaMemcpyHostToDevice));
        } else {
            return CT_EINVAL;
        }
        defined[d.dst] = 1;
        m->L.push_back(l);
    }
    if (n_final != 1) return CT_EINVAL;
    // ---- activation slots ----
    for (size_t s = 0; s < m->slots.size(); ++s) {
        Slot &sl = m->slots[s];
        if (!defined[s] || !sl.stored) continue;
        bool is_final_out = false;
        for (auto &l : m->L) if (l.d.op == CT_OP_FC && l.d.final && l.d.dst == (int)s) is_final_out = true;
        if (is_final_out) continue;
        const size_t e = sl.is_float ? 4 : esz;
        if (sl.cp < sl.C) sl.cp = sl.C;
        ct_status st;
        if ((st = dalloc(m, &sl.data, (size_t)B * sl.H * sl.W * sl.cp * e)) != CT_OK) return st;
        if (sl.has_cs && (st = dalloc(m, &sl.cs, (size_t)B * sl.H * sl.W * e)) != CT_OK) return st;
    }
    // ---- tensor-core plans ----
    for (auto &l : m->L) {
        if (l.stem) {
            ConvArgs a{};
            a.N = B; a.H = l.H; a.W = l.W; a.C = l.C; a.K = l.K; a.R = l.R; a.S = l.S;
            a.stride = l.d.stride; a.pad = l.d.pad; a.P = l.P; a.Q = l.Q; a.role = l.role; a.coef = l.coef;
            std::string why;
            l.stplan = stem_plan_create(a, &why);
            if (!l.stplan) return CT_ECUDA;
            continue;
        }
        if (l.tc_small) {
            ConvArgs a{};
            a.N = B; a.H = l.H; a.W = l.W; a.C = l.C; a.K = l.K; a.R = l.R; a.S = l.S;
            a.stride = l.d.stride; a.pad = l.d.pad; a.P = l.P; a.Q = l.Q; a.role = l.role; a.coef = l.coef;
            std::string why;
            l.splan = tc_small_plan_create(a, l.w, &why);
            if (!l.splan) return CT_ECUDA;
            continue;
        }
        if (l.fc_tc) {
            ConvArgs a{};
            a.N = B; a.H = a.W = 1; a.C = l.n_in; a.K = l.n_out; a.R = a.S = 1;
            a.stride = 1; a.pad = 0; a.P = a.Q = 1;
            a.role = m->protect ? CT_ROLE_CT : CT_ROLE_NONE; a.coef = l.coef;
            std::string why;
            l.plan = tc_plan_create(a, B, l.w, m->slots[l.d.src].data, &why);
            if (!l.plan) return CT_ECUDA;
            continue;
        }
        if (!l.tc) continue;
        ConvArgs a{};
        a.N = B; a.H = l.H; a.W = l.W; a.C = l.C; a.K = l.K; a.R = l.R; a.S = l.S;
        a.stride = l.d.stride; a.pad = l.d.pad; a.P = l.P; a.Q = l.Q; a.role = l.role; a.coef = l.coef;
        std::string why;
        l.plan = tc_plan_create(a, B, l.w, m->slots[l.d.src].data, &why);
        if (!l.plan) return CT_ECUDA;
        if (halo_supported(l.C, l.K, l.R, l.S, l.d.stride, l.d.pad, l.H, l.W) && m->slots[l.d.src].cp == l.C) {
            const Slot &sx = m->slots[l.d.src];
            const Slot *sr = l.d.res >= 0 ? &m->slots[l.d.res] : nullptr;
            const bool cs_out = l.cs_out;
            // a 2 x 2 stride-2 max-pool that is the only reader of this output
            // runs in the halo kernel's epilogue
            const size_t li = (size_t)(&l - m->L.data());
            if (li + 1 < m->L.size() && l.P % 2 == 0 && l.Q % 2 == 0) {
                const ct_layer_desc &nx = m->L[li + 1].d;
                int readers = 0;
                for (auto &o : m->L) readers += (o.d.src == l.d.dst) + (o.d.res == l.d.dst);
                l.pool_fuse = nx.op == CT_OP_MAXPOOL && nx.src == l.d.dst && nx.k == 2 && nx.stride == 2 &&
                              nx.pad == 0 && readers == 1;
            }
            l.hplan = halo_plan_create(a, B, l.w, sx.data, sr ? sr->data : nullptr,
                                       (cs_out && sx.has_cs) ? sx.cs : nullptr,
                                       (cs_out && sr && sr->has_cs) ? sr->cs : nullptr, l.pool_fuse, &why);
            if (!l.hplan) return CT_ECUDA;
        }
    }
    // ---- 1x1 shortcuts that run in the launch of the convolution before them ----
    // Layer i + 1 reads the same tensor as layer i at the same stride, and
    // its pixel (p * stride, q * stride) is layer i's centre tap (pad =
    // (R - 1) / 2): its GEMM operand A is layer i's centre-tap K blocks.
    for (size_t i = 0; i + 1 < m->L.size() && !(m->flags & CT_FLAG_LAYERWISE); ++i) {
        LayerRT &l = m->L[i];
        const LayerRT &n = m->L[i + 1];
        l.sc_next = l.tc && l.plan && n.tc && n.plan && !l.stem && !n.stem && l.d.op == CT_OP_CONV &&
                    n.d.op == CT_OP_CONV && n.d.src == l.d.src && n.R == 1 && n.S == 1 && n.d.pad == 0 &&
                    n.d.stride == l.d.stride && l.R == l.S && l.d.pad == (l.R - 1) / 2 && n.C == l.C &&
                    n.K == l.K && n.d.res < 0 && (l.K == 128 || l.K % 256 == 0);
    }
    // ---- the LeNet-5 shape runs as one whole-network kernel ----
    {
        SmallNet g;
        m->small = !(m->flags & CT_FLAG_LAYERWISE) && small_net_of(m, &g);
        if (m->small)
            m->small_flops = (double)g.K1 * g.H1 * g.W1 * g.R1 * g.R1 * g.C0 + (double)g.K2 * g.H2 * g.W2 * g.R2 * g.R2 * g.K1;
    }
    // ---- scratch for re-execution and host runs ----
    const size_t per_img = (size_t)m->in_c * m->in_h * m->in_w;
    ct_status st;
    if ((st = dalloc(m, (void **)&m->re_input, sizeof(float) * per_img * B)) != CT_OK) return st;
    if ((st = dalloc(m, (void **)&m->re_logits, sizeof(float) * m->n_classes * B)) != CT_OK) return st;
    if ((st = dalloc(m, (void **)&m->re_S, sizeof(float) * B)) != CT_OK) return st;
    if ((st = dalloc(m, (void **)&m->re_flag, B)) != CT_OK) return st;
    if ((st = dalloc(m, (void **)&m->re_idx, sizeof(int32_t) * B)) != CT_OK) return st;
    if ((st = dalloc(m, (void **)&m->rh_input, sizeof(float) * per_img * B)) != CT_OK) return st;
    if ((st = dalloc(m, (void **)&m->rh_logits, sizeof(float) * m->n_classes * B)) != CT_OK) return st;
    if ((st = dalloc(m, (void **)&m->rh_S, sizeof(float) * B)) != CT_OK) return st;
    if ((st = dalloc(m, (void **)&m->rh_flag, B)) != CT_OK) return st;
    if ((st = dalloc(m, (void **)&m->d_err, sizeof(uint32_t))) != CT_OK) return st;
    if ((st = dalloc(m, (void **)&m->ws, SPLITK_WS_BYTES)) != CT_OK) return st;
    CUDA_TRY(cudaMemset(m->d_err, 0, sizeof(uint32_t)));
    if (cudaMallocHost((void **)&m->h_flags, B) != cudaSuccess) return CT_ENOMEM;
    if (cudaHostAlloc((void **)&m->h_idx, sizeof(int32_t) * B, cudaHostAllocMapped) != cudaSuccess ||
        cudaHostGetDevicePointer((void **)&m->h_idx_d, m->h_idx, 0) != cudaSuccess)
        return CT_ENOMEM;
    CUDA_TRY(cudaDeviceSynchronize());
    return CT_OK;
}

// ---------------------------------------------------------------------------
// fault resolution
// ---------------------------------------------------------------------------

struct WeightFault {
    bool explicit_word = false;   // XOR a device word
    int64_t word = 0;
    FaultDelta fd{};
};

// Map a literal weight element [K_tot, C_tot, R, S] of conv layer l to the
// device representation: an explicit stored word (a data filter weight), or
// an implicit weight of the construction (zero checksum slice, carry-through
// or pass-through row), whose flipped value enters the epilogue as
// dv * input, dv = flipped - stored.
WeightFault resolve_weight_fault(const ct_model *m, const LayerRT &l, int64_t e, int bit) {
    const int Ct = weight_in_channels(l);
    const int RS = l.R * l.S;
    const int k = (int)(e / ((int64_t)Ct * RS));
    const int c = (int)((e / RS) % Ct);
    const int r = (int)((e / l.S) % l.R), s = (int)(e % l.S);
    const bool centre = r == (l.R - 1) / 2 && s == (l.S - 1) / 2;
    WeightFault f;
    if (k < l.K && (l.dw || c < l.C)) {
        f.explicit_word = true;
        f.word = weight_word(l, k, r, s, c);
        return f;
    }
    double stored = 0.0;                      // zero slice and off-centre taps
    if (k == l.K && l.role == CT_ROLE_CT && centre) stored = l.coef;
    if (k == l.K && l.role == CT_ROLE_PASS && centre && (l.dw || c == l.C)) stored = 1.0;
    const float v = flipped(stored, bit, m->prec);
    f.fd.active = 1;
    f.fd.kout = k;
    f.fd.cin = c;
    f.fd.r = r;
    f.fd.s = s;
    f.fd.dv = v - (float)stored;
    return f;
}

ct_status act_fault_word(const ct_model *m, int slot, int batch, int64_t e, void **base, int64_t *word) {
    const Slot &sl = m->slots[slot];
    const int Ct = sl.C + (sl.has_cs ? 1 : 0);
    const int64_t HW = (int64_t)sl.H * sl.W;
    if (!sl.stored || e < 0 || e >= (int64_t)batch * Ct * HW) return CT_ERANGE;
    const int64_t n = e / (Ct * HW);
    const int c = (int)((e / HW) % Ct);
    const int64_t hw = e % HW;
    if (c < sl.C) { *base = sl.data; *word = (n * HW + hw) * sl.cp + c; }
    else { *base = sl.cs; *word = n * HW + hw; }
    return CT_OK;
}

// ---------------------------------------------------------------------------
// inference
// ---------------------------------------------------------------------------

// The LeNet shape the whole-network kernel runs (FP32, widened or
// unprotected): conv -> pool -> conv -> pool -> fc -> fc -> fc, with ReLU
// after every conv and hidden FC, 2x2 stride-2 pools, unpadded stride-1
// convolutions with a carry-through filter (widened).
static bool small_net_of(const ct_model *m, SmallNet *g) {
    if (m->prec != CT_FP32 || m->replace || m->L.size() != 7) return false;
    const LayerRT &c1 = m->L[0], &p1 = m->L[1], &c2 = m->L[2], &p2 = m->L[3];
    const LayerRT &f1 = m->L[4], &f2 = m->L[5], &f3 = m->L[6];
    const int want_role = m->protect ? CT_ROLE_CT : CT_ROLE_NONE;
    auto conv_ok = [&](const LayerRT &l) {
        return l.d.op == CT_OP_CONV && l.d.stride == 1 && l.d.pad == 0 && l.d.relu && l.d.res < 0 &&
               l.role == want_role && l.R == l.S && l.w_ld == l.R * l.S * l.C && l.c_stride == l.C && !l.dw;
    };
    auto pool_ok = [](const LayerRT &l) { return l.d.op == CT_OP_MAXPOOL && l.d.k == 2 && l.d.stride == 2 && l.d.pad == 0; };
    if (!conv_ok(c1) || !pool_ok(p1) || !conv_ok(c2) || !pool_ok(p2)) return false;
    if (c1.d.src != 0 || p1.d.src != c1.d.dst || c2.d.src != p1.d.dst || p2.d.src != c2.d.dst) return false;
    if (f1.d.op != CT_OP_FC || f2.d.op != CT_OP_FC || f3.d.op != CT_OP_FC || !f1.d.relu || !f2.d.relu ||
        !f3.d.final || f1.d.src != p2.d.dst || f2.d.src != f1.d.dst || f3.d.src != f2.d.dst)
        return false;
    if (c1.cs_in || c2.cs_in != m->protect || f1.x_float || f1.fc_tc || f2.fc_tc) return false;
    const Slot &s1 = m->slots[p1.d.dst], &s2 = m->slots[p2.d.dst];
    SmallNet &n = *g;
    memset(&n, 0, sizeof(n));
    n.protect = m->protect ? 1 : 0;
    n.C0 = c1.C; n.H0 = c1.H; n.W0 = c1.W;
    n.K1 = c1.K; n.R1 = c1.R; n.H1 = c1.P; n.W1 = c1.Q; n.Hp1 = s1.H; n.Wp1 = s1.W;
    n.K2 = c2.K; n.R2 = c2.R; n.H2 = c2.P; n.W2 = c2.Q; n.Hp2 = s2.H; n.Wp2 = s2.W;
    n.NIN1 = f1.n_in; n.N1 = f1.n_out; n.N2 = f2.n_out; n.N3 = f3.n_out;
    if (n.NIN1 != n.K2 * n.Hp2 * n.Wp2 || f1.n_cs != (m->protect ? n.Hp2 * n.Wp2 : 0) || f2.n_in != n.N1 ||
        f3.n_in != n.N2)
        return false;
    n.w1 = (const float *)c1.w; n.b1 = c1.bias; n.w2 = (const float *)c2.w; n.b2 = c2.bias;
    n.wf1 = (const float *)f1.w; n.bf1 = f1.bias; n.wf2 = (const float *)f2.w; n.bf2 = f2.bias;
    n.wf3 = (const float *)f3.w; n.bf3 = f3.bias;
    n.coef1 = c1.coef; n.coef2 = c2.coef; n.coeff1 = f1.coef; n.coeff2 = f2.coef; n.coeff3 = f3.coef;
    n.ref = m->ref; n.tau = m->tau;
    return campaign_small_smem(n) <= 200 * 1024;
}

// input2 / n_split: images n >= n_split of the batch are image n - n_split
// of input2 (re-executed images appended to a batch); the rest of the
// network is unaware of it
// Re-executed images appended to an inference as rows n_split .. batch - 1:
// image idx[j] of the earlier batch's input (input2), whose logits and S
// rows they write.  idx is device-visible (mapped host memory).
struct RerunRows {
    const int32_t *idx;
    float *logits, *S;
};

ct_status infer_impl(ct_model *m, const float *input, int batch, float *logits, float *S,
                     uint8_t *flag, cudaStream_t st, const float *input2 = nullptr, int n_split = 0,
                     const SmallRerun *rerun = nullptr, const RerunRows *rows = nullptr) {
    const bool half = m->prec == CT_FP16;
    const int wb = half ? 2 : 4;
    if (m->small) {
        // the whole network in one kernel; an armed fault is applied inside it
        SmallNet g;
        small_net_of(m, &g);
        g.B = batch;
        g.x = input;
        g.x2 = input2;
        g.n_split = input2 ? n_split : batch;
        g.ref = m->ref;
        g.tau = m->tau;
        g.flag2 = m->flag_mirror;
        CampFault f{};
        f.kind = 2;
        if (m->armed) {
            const LayerRT &l = m->L[m->f_layer];
            f.kind = m->f_kind;
            f.bit = m->f_bit;
            f.word = -1;
            if (m->f_kind == CT_BUF_WEIGHT) {
                f.layer = m->f_layer == 0 ? 0 : 1;
                const WeightFault wf = resolve_weight_fault(m, l, m->f_elem, m->f_bit);
                if (wf.explicit_word) f.word = wf.word;
                else f.fd = wf.fd;
            } else {
                const int per_img = (g.K1 + (g.protect ? 1 : 0)) * g.Hp1 * g.Wp1;
                if (m->f_layer != 2 || m->f_elem < 0 || m->f_elem >= (int64_t)batch * per_img) return CT_ERANGE;
                f.img = (int)(m->f_elem / per_img);
                const int within = (int)(m->f_elem % per_img);
                f.act_c = within / (g.Hp1 * g.Wp1);
                f.act_hw = within % (g.Hp1 * g.Wp1);
            }
        }
        m->armed = false;
        m->n_kernels_run = 0;
        for (auto &sl : m->slots) sl.skipped_last = true;
        m->slots[0].skipped_last = false;
        SmallRerun none{};
        const SmallRerun &rr = rerun ? *rerun : none;
        CUDA_TRY(launch(m, FAM_SIMT, 2.0 * (batch + rr.n) * m->small_flops, st,
                        [&] { return launch_small_infer(g, f, logits, S, flag, rr, st); }));
        m->n_kernels_last = m->n_kernels_run;
        return CT_OK;
    }
    for (auto &sl : m->slots) sl.skipped_last = false;
    const bool armed = m->armed;
    m->armed = false;
    m->n_kernels_run = 0;
    int act_slot = -1;
    void *act_base = nullptr;
    int64_t act_word = 0;
    if (armed && m->f_kind == CT_BUF_ACT) {
        act_slot = m->L[m->f_layer].d.src;
        if (act_fault_word(m, act_slot, batch, m->f_elem, &act_base, &act_word) != CT_OK) return CT_ERANGE;
    }
    Slot &s0 = m->slots[0];
    const int n_first = input2 ? n_split : batch;
    if (s0.stored) {
        CUDA_TRY(launch(m, FAM_OTHER, 0, st, [&] {
            return launch_convert_input(input, s0.data, n_first, s0.C, s0.cp, s0.H, s0.W, half, st);
        }));
        if (input2) {
            void *dst2 = static_cast<uint8_t *>(s0.data) + (size_t)n_split * s0.H * s0.W * s0.cp * wb;
            CUDA_TRY(launch(m, FAM_OTHER, 0, st, [&] {
                return launch_convert_input(input2, dst2, batch - n_split, s0.C, s0.cp, s0.H, s0.W, half, st,
                                            rows ? rows->idx : nullptr);
            }));
        }
    }
    if (act_slot == 0) CUDA_TRY(xor_bit(m, act_base, act_word, m->f_bit, wb, st));
    size_t pool_done = (size_t)-1;               // a max-pool applied by the preceding conv kernel
    size_t sc_done = (size_t)-1;                 // a shortcut run by the preceding conv's launch
    // arguments of convolution layer li; a weight fault armed on it is
    // resolved into wf (an explicit word is flipped by the caller around the
    // launch, an implicit one rides in the epilogue as a delta)
    auto conv_args = [&](size_t li, ConvArgs &a, WeightFault &wf) -> bool {
        const LayerRT &l = m->L[li];
        const ct_layer_desc &d = l.d;
        const Slot &src = m->slots[d.src];
        const Slot &dst = m->slots[d.dst];
        a = ConvArgs{};
        a.x = src.data; a.cs_in = src.has_cs ? src.cs : nullptr; a.w = l.w; a.bias = l.bias;
        if (d.res >= 0) {
            a.res = m->slots[d.res].data;
            a.res_cs = m->slots[d.res].has_cs ? m->slots[d.res].cs : nullptr;
        }
        a.y = dst.data; a.cs_out = dst.has_cs ? dst.cs : nullptr;
        a.N = batch; a.H = l.H; a.W = l.W; a.C = l.C; a.K = l.K; a.R = l.R; a.S = l.S;
        a.stride = d.stride; a.pad = d.pad; a.P = l.P; a.Q = l.Q;
        a.role = l.role; a.relu = d.relu; a.coef = l.coef; a.err = m->d_err;
        a.ws = m->ws; a.ws_bytes = SPLITK_WS_BYTES;
        const bool wfault = armed && m->f_kind == CT_BUF_WEIGHT && m->f_layer == (int)li;
        if (wfault) {
            wf = resolve_weight_fault(m, l, m->f_elem, m->f_bit);
            if (!wf.explicit_word) a.fd = wf.fd;
        }
        return wfault;
    };
    auto conv_flops = [&](const LayerRT &l) { return 2.0 * batch * l.P * l.Q * (double)l.K * l.R * l.S * l.C; };
    for (size_t i = 0; i < m->L.size(); ++i) {
        LayerRT &l = m->L[i];
        const ct_layer_desc &d = l.d;
        Slot &src = m->slots[d.src];
        Slot &dst = m->slots[d.dst];
        if (i == sc_done) {
            // computed by the launch of the convolution before it
        } else if (d.op == CT_OP_CONV) {
            ConvArgs a;
            WeightFault wf;
            const bool wfault = conv_args(i, a, wf);
            if (wfault && wf.explicit_word) CUDA_TRY(xor_bit(m, l.w, wf.word, m->f_bit, wb, st));
            const double flops = conv_flops(l);
            if (l.stem) {
                // the fused kernel reads the FP32 image and writes the max-pool's output
                const Slot &po = m->slots[m->L[i + 1].d.dst];
                a.x = input;
                a.x2 = input2;
                a.n_split = n_first;
                a.x2_idx = rows ? rows->idx : nullptr;
                a.y = po.data;
                a.cs_out = po.has_cs ? po.cs : nullptr;
                CUDA_TRY(launch(m, FAM_TC, flops, st, [&] { return launch_stem_pool(a, l.stplan, st); }));
            } else if (l.dw) {
                const double dw_flops = 2.0 * batch * l.P * l.Q * (double)l.K * l.R * l.S;
                CUDA_TRY(launch(m, FAM_OTHER, dw_flops, st, [&] { return launch_conv_dw(a, half, st); }));
            } else if (l.tc_small) {
                CUDA_TRY(launch(m, FAM_TC, flops, st, [&] { return launch_conv_tc_small(a, l.splan, st); }));
            } else {
                int nk = 1;
                const bool halo = l.hplan && halo_tiles(l.hplan, batch) >= halo_sms(l.hplan);
                dst.skipped_last = halo && l.pool_fuse;
                if (halo && l.pool_fuse) {
                    // the kernel writes the max-pool's output; this output is never stored
                    const Slot &po = m->slots[m->L[i + 1].d.dst];
                    a.y = po.data;
                    a.cs_out = po.has_cs ? po.cs : nullptr;
                    pool_done = i + 1;
                }
                const LayerRT *ln = l.sc_next ? &m->L[i + 1] : nullptr;
                ConvArgs a2;
                WeightFault wf2;
                bool wfault2 = false;
                if (ln) wfault2 = conv_args(i + 1, a2, wf2);
                if (halo) {
                    CUDA_TRY(launch(m, FAM_TC, flops, st, [&] { return launch_conv_tc_halo(a, l.hplan, st); }));
                } else if (ln && tc_shortcut_fits(a, l.plan, ln->plan)) {
                    // the shortcut (layer i + 1) runs in this launch
                    if (wfault2 && wf2.explicit_word) CUDA_TRY(xor_bit(m, ln->w, wf2.word, m->f_bit, wb, st));
                    bool merged = false;
                    CUDA_TRY(launch(m, FAM_TC, flops + conv_flops(*ln), st,
                                    [&] { return launch_conv_tc(a, l.plan, st, &nk, &a2, ln->plan, &merged); }, &nk));
                    if (!merged) return CT_ECUDA;
                    if (wfault2 && wf2.explicit_word) CUDA_TRY(xor_bit(m, ln->w, wf2.word, m->f_bit, wb, st));
                    sc_done = i + 1;
                } else if (l.tc) {
                    CUDA_TRY(launch(m, FAM_TC, flops, st, [&] { return launch_conv_tc(a, l.plan, st, &nk); }, &nk));
                } else {
                    CUDA_TRY(launch(m, FAM_SIMT, flops, st, [&] { return launch_conv_simt(a, half, st, &nk); }, &nk));
                }
            }
            if (wfault && wf.explicit_word) CUDA_TRY(xor_bit(m, l.w, wf.word, m->f_bit, wb, st));
        } else if (l.fused || i == pool_done) {
            // computed by the fused stem, or by the halo kernel of the conv before it
        } else if (d.op == CT_OP_MAXPOOL || d.op == CT_OP_GAP) {
            PoolArgs a{};
            a.x = src.data; a.cs_in = src.has_cs ? src.cs : nullptr;
            a.y = dst.data; a.cs_out = dst.has_cs ? dst.cs : nullptr;
            a.N = batch; a.H = src.H; a.W = src.W; a.C = src.C; a.P = dst.H; a.Q = dst.W;
            a.k = d.k; a.stride = d.stride; a.pad = d.pad;
            if (d.op == CT_OP_MAXPOOL) CUDA_TRY(launch(m, FAM_POOL, 0, st, [&] { return launch_maxpool(a, half, st); }));
            else CUDA_TRY(launch(m, FAM_POOL, 0, st, [&] { return launch_gap(a, half, st); }));
        } else if (l.fc_tc) {
            // hidden FC as a 1x1 convolution over [batch, 1, 1, n_in]: the carry-through
            // neuron is the kernel's carry-through column plus the sum of the incoming
            // checksum features
            ConvArgs a{};
            a.x = src.data; a.cs_in = src.has_cs ? src.cs : nullptr; a.w = l.w; a.bias = l.bias;
            a.y = dst.data; a.cs_out = dst.has_cs ? dst.cs : nullptr;
            a.N = batch; a.H = a.W = 1; a.C = l.n_in; a.K = l.n_out; a.R = a.S = 1;
            a.stride = 1; a.pad = 0; a.P = a.Q = 1;
            a.role = m->protect ? CT_ROLE_CT : CT_ROLE_NONE; a.relu = d.relu; a.coef = l.coef;
            a.err = m->d_err; a.cs_rowsum = l.n_cs;
            a.ws = m->ws; a.ws_bytes = SPLITK_WS_BYTES;
            const double flops = 2.0 * batch * (double)l.n_in * l.n_out;
            int nk = 1;
            CUDA_TRY(launch(m, FAM_FC, flops, st, [&] { return launch_conv_tc(a, l.plan, st, &nk); }, &nk));
        } else {
            FcArgs a{};
            a.x = src.data; a.xcs = src.has_cs ? src.cs : nullptr; a.w = l.w; a.bias = l.bias;
            a.B = batch; a.n_in = l.n_in; a.n_cs = l.n_cs; a.n_out = l.n_out;
            a.relu = d.relu; a.final_layer = d.final; a.coef = l.coef;
            // replace construction: the classifier's accumulated-checksum neuron
            // sums every input feature (the checksum channel is one of them)
            a.protect = m->protect || (m->replace && d.final);
            a.ref = m->ref; a.tau = m->tau;
            if (d.final) {
                a.y = logits; a.S = S; a.flag = flag; a.flag2 = m->flag_mirror;
                if (rows) { a.rr_split = n_split; a.rr_idx = rows->idx; a.rr_y = rows->logits; a.rr_S = rows->S; }
            }
            else { a.y = dst.data; a.ycs = dst.has_cs ? dst.cs : nullptr; }
            a.ws = m->ws; a.ws_bytes = SPLITK_WS_BYTES;
            const double flops = 2.0 * batch * (double)l.n_in * l.n_out;
            int nk = 1;
            CUDA_TRY(launch(m, FAM_FC, flops, st, [&] { return launch_fc(a, half, l.x_float, st, &nk); }, &nk));
        }
        if (act_slot == d.dst) CUDA_TRY(xor_bit(m, act_base, act_word, m->f_bit, wb, st));
    }
    m->n_kernels_last = m->n_kernels_run;
    return CT_OK;
}

// Fault-free inference of the first `bucket` images of the re-execution
// scratch, replayed from a graph captured on first use of this batch size:
// one graph launch instead of one host launch per kernel.  Falls back to
// direct launches if capture or instantiation fails.
cudaGraphExec_t reexec_graph(ct_model *m, int bucket) {
    int slot = 0;
    while ((1 << slot) < bucket) ++slot;
    if ((int)m->re_graph.size() <= slot) {
        m->re_graph.resize(slot + 1, nullptr);
        m->re_graph_nk.resize(slot + 1, 0);
    }
    if (m->re_graph[slot]) return m->re_graph[slot];
    if (!m->cap_stream && cudaStreamCreateWithFlags(&m->cap_stream, cudaStreamNonBlocking) != cudaSuccess) {
        cudaGetLastError();
        return nullptr;
    }
    if (cudaStreamBeginCapture(m->cap_stream, cudaStreamCaptureModeThreadLocal) != cudaSuccess) {
        cudaGetLastError();
        return nullptr;
    }
    const int64_t before = m->kernels_total;
    uint8_t *const mirror = m->flag_mirror;      // a re-run never writes a batch's flag copy
    m->flag_mirror = nullptr;
    const ct_status s = infer_impl(m, m->re_input, bucket, m->re_logits, m->re_S, m->re_flag, m->cap_stream);
    m->flag_mirror = mirror;
    m->re_graph_nk[slot] = (int)(m->kernels_total - before);
    m->kernels_total = before;           // captured, not launched
    cudaGraph_t g = nullptr;
    const cudaError_t e = cudaStreamEndCapture(m->cap_stream, &g);
    cudaGraphExec_t ex = nullptr;
    if (s == CT_OK && e == cudaSuccess && g && cudaGraphInstantiate(&ex, g, 0) != cudaSuccess) ex = nullptr;
    if (g) cudaGraphDestroy(g);
    cudaGetLastError();
    m->re_graph[slot] = ex;
    return ex;
}

// Re-execution of the images whose host-side flag is set (Sec. II-B, last
// paragraph): gather them into a batch of their own, padded to a power of
// two (at most max_batch) by repeating the last one, run it fault-free
// (graph replay, or direct launches when profiling) and scatter the first n
// rows back.  idx_host: a pinned index buffer of max_batch entries that no
// copy still in flight reads.
ct_status reexec_rows(ct_model *m, const float *input, int batch, const uint8_t *flags_host, float *logits,
                      float *S, int *n_rerun, int32_t *idx_host, cudaStream_t st) {
    int n = 0;
    for (int i = 0; i < batch; ++i)
        if (flags_host[i]) idx_host[n++] = i;
    if (n_rerun) *n_rerun = n;
    if (n == 0) return CT_OK;
    // each bucket size has its own graph slot (ceil log2); max_batch is the
    // only size in the last slot
    int bucket = 1;
    while (bucket < n) bucket <<= 1;
    if (bucket > m->max_batch) bucket = m->max_batch;
    for (int i = n; i < bucket; ++i) idx_host[i] = idx_host[n - 1];
    CUDA_TRY(cudaMemcpyAsync(m->re_idx, idx_host, sizeof(int32_t) * bucket, cudaMemcpyHostToDevice, st));
    const int64_t per = (int64_t)m->in_c * m->in_h * m->in_w;
    CUDA_TRY(launch(m, FAM_OTHER, 0, st, [&] { return launch_gather_images(input, m->re_input, m->re_idx, bucket, per, st); }));
    // fault-free re-run: an armed fault stays armed for the next ct_infer;
    // it writes no batch's flag copy
    const bool armed = m->armed;
    m->armed = false;
    uint8_t *const mirror = m->flag_mirror;
    m->flag_mirror = nullptr;
    ct_status s = CT_OK;
    cudaGraphExec_t ex = m->prof ? nullptr : reexec_graph(m, bucket);
    if (ex) {
        int slot = 0;
        while ((1 << slot) < bucket) ++slot;
        if (cudaGraphLaunch(ex, st) != cudaSuccess) s = CT_ECUDA;
        else m->kernels_total += m->re_graph_nk[slot];
    } else {
        s = infer_impl(m, m->re_input, bucket, m->re_logits, m->re_S, m->re_flag, st);
    }
    m->armed = armed;
    m->flag_mirror = mirror;
    if (s != CT_OK) return s;
    CUDA_TRY(launch(m, FAM_OTHER, 0, st, [&] { return launch_scatter_rows(m->re_logits, logits, m->re_idx, n, m->n_classes, st); }));
    if (S) CUDA_TRY(launch(m, FAM_OTHER, 0, st, [&] { return launch_scatter_rows(m->re_S, S, m->re_idx, n, 1, st); }));
    return CT_OK;
}

// the device flags of a finished inference, read on the host (one stream synchronisation)
ct_status read_flags(ct_model *m, const uint8_t *flag, int batch, cudaStream_t st) {
    CUDA_TRY(cudaMemcpyAsync(m->h_flags, flag, batch, cudaMemcpyDeviceToHost, st));
    CUDA_TRY(cudaStreamSynchronize(st));
    return CT_OK;
}

ct_status reexec_impl(ct_model *m, const float *input, int batch, const uint8_t *flag, float *logits,
                      float *S, int *n_rerun, cudaStream_t st) {
    ct_status s = read_flags(m, flag, batch, st);
    if (s != CT_OK) return s;
    return reexec_rows(m, input, batch, m->h_flags, logits, S, n_rerun, m->h_idx, st);
}

// Inference of `batch` new images with the flagged images of a previous
// batch (host-side flags) re-executed as extra rows of the same launch
// sequence (Sec. II-B): their cost is that of the extra images, not of a
// separate small-batch pass.  Falls back to reexec_rows + infer_impl when a
// fault is armed (the re-run must be fault-free) or the rows do not fit
// max_batch.  idx_host as for reexec_rows.
ct_status infer_with_reruns(ct_model *m, const float *input, int batch, float *logits, float *S, uint8_t *flag,
                            const float *prev_input, int prev_batch, const uint8_t *prev_flags_host,
                            float *prev_logits, float *prev_S, int *n_rerun, int32_t *idx_host, cudaStream_t st,
                            const int32_t *idx_dev = nullptr) {
    if (n_rerun) *n_rerun = 0;
    int n = 0;
    for (int i = 0; i < prev_batch; ++i)
        if (prev_flags_host[i]) idx_host[n++] = i;
    if (n == 0) return infer_impl(m, input, batch, logits, S, flag, st);
    if (m->armed || batch + n > m->max_batch) {
        int nr = 0;
        ct_status s = reexec_rows(m, prev_input, prev_batch, prev_flags_host, prev_logits, prev_S, &nr, idx_host, st);
        if (s != CT_OK) return s;
        if (n_rerun) *n_rerun = nr;
        return infer_impl(m, input, batch, logits, S, flag, st);
    }
    if (n_rerun) *n_rerun = n;
    if (m->small && n <= SMALL_MAX_RERUN) {
        // the whole-network kernel reads the re-run images and writes their rows itself
        SmallRerun rr{};
        rr.x = prev_input;
        rr.logits = prev_logits;
        rr.S = prev_S;
        rr.n = n;
        for (int j = 0; j < n; ++j) rr.idx[j] = idx_host[j];
        return infer_impl(m, input, batch, logits, S, flag, st, nullptr, 0, &rr);
    }
    if (idx_dev) {
        // the first layer reads the re-run images through the index list and
        // the final FC writes their rows to the earlier batch's outputs: no
        // gather, copy or scatter around the inference
        const RerunRows rows{idx_dev, prev_logits, prev_S};
        return infer_impl(m, input, batch + n, logits, S, flag, st, prev_input, batch, nullptr, &rows);
    }
    CUDA_TRY(cudaMemcpyAsync(m->re_idx, idx_host, sizeof(int32_t) * n, cudaMemcpyHostToDevice, st));
    const int64_t per = (int64_t)m->in_c * m->in_h * m->in_w;
    CUDA_TRY(launch(m, FAM_OTHER, 0, st, [&] { return launch_gather_images(prev_input, m->re_input, m->re_idx, n, per, st); }));
    const int tot = batch + n;
    ct_status s = infer_impl(m, input, tot, m->re_logits, m->re_S, m->re_flag, st, m->re_input, batch);
    if (s != CT_OK) return s;
    // rows < batch: this batch; rows >= batch: the re-run, whose flag is ignored
    CUDA_TRY(cudaMemcpyAsync(logits, m->re_logits, sizeof(float) * m->n_classes * batch, cudaMemcpyDeviceToDevice, st));
    if (S) CUDA_TRY(cudaMemcpyAsync(S, m->re_S, sizeof(float) * batch, cudaMemcpyDeviceToDevice, st));
    if (flag) CUDA_TRY(cudaMemcpyAsync(flag, m->re_flag, batch, cudaMemcpyDeviceToDevice, st));
    CUDA_TRY(launch(m, FAM_OTHER, 0, st, [&] {
        return launch_scatter_rows(m->re_logits + (size_t)batch * m->n_classes, prev_logits, m->re_idx, n, m->n_classes, st);
    }));
    if (prev_S) CUDA_TRY(launch(m, FAM_OTHER, 0, st, [&] { return launch_scatter_rows(m->re_S + batch, prev_S, m->re_idx, n, 1, st); }));
    return CT_OK;
}

ct_status infer_reexec_impl(ct_model *m, const float *input, int batch, float *logits, float *S, uint8_t *flag,
                            const float *prev_input, int prev_batch, const uint8_t *prev_flag, float *prev_logits,
                            float *prev_S, int *n_rerun, cudaStream_t st) {
    if (n_rerun) *n_rerun = 0;
    if (!prev_input || prev_batch == 0) return infer_impl(m, input, batch, logits, S, flag, st);
    ct_status s = read_flags(m, prev_flag, prev_batch, st);
    if (s != CT_OK) return s;
    return infer_with_reruns(m, input, batch, logits, S, flag, prev_input, prev_batch, m->h_flags, prev_logits, prev_S,
                             n_rerun, m->h_idx, st, m->h_idx_d);
}

// Re-execution of the flagged images of nb <= 2 batches (host flags) as one
// padded batch: each batch's images are gathered after the previous ones'
// and their rows scattered back to that batch's outputs.  idx_host holds
// 2 * max_batch entries that no copy in flight reads.  When the combined
// count exceeds max_batch, each batch is re-run on its own.
template <typename In, typename Fl, typename Lg, typename Sv>
ct_status reexec_rows_of(ct_model *m, int nb, In in, Fl fl, Lg lg, Sv Sp, int batch, int *n_rerun, int32_t *idx_host,
                         cudaStream_t st) {
    int tot = 0;
    for (int j = 0; j < nb; ++j)
        for (int i = 0; i < batch; ++i) tot += fl(j)[i] ? 1 : 0;
    if (n_rerun) *n_rerun = tot;
    if (tot == 0) return CT_OK;
    if (nb == 1 || tot > m->max_batch) {
        for (int j = 0; j < nb; ++j) {
            int nr = 0;
            ct_status s = reexec_rows(m, in(j), batch, fl(j), lg(j), Sp(j), &nr, idx_host + (size_t)j * m->max_batch, st);
            if (s != CT_OK) return s;
        }
        return CT_OK;
    }
    int bucket = 1;
    while (bucket < tot) bucket <<= 1;
    if (bucket > m->max_batch) bucket = m->max_batch;
    // gather lists: per batch its own flagged indices, then the padded combined list
    const int64_t per = (int64_t)m->in_c * m->in_h * m->in_w;
    int32_t *lists = idx_host;                     // [nb][<= batch] flagged indices
    int off = 0;
    std::vector<int> cnt(nb);
    for (int j = 0; j < nb; ++j) {
        int c = 0;
        for (int i = 0; i < batch; ++i)
            if (fl(j)[i]) lists[off + c++] = i;
        cnt[j] = c;
        off += c;
    }
    CUDA_TRY(cudaMemcpyAsync(m->re_idx, lists, sizeof(int32_t) * tot, cudaMemcpyHostToDevice, st));
    // rows [o_j, o_j + cnt_j) of the re-run batch: batch j's images; padding repeats the last one
    for (int j = 0, o = 0; j < nb; o += cnt[j], ++j) {
        if (!cnt[j]) continue;
        const int c = cnt[j];
        float *dst = m->re_input + (size_t)o * per;
        CUDA_TRY(launch(m, FAM_OTHER, 0, st, [&] { return launch_gather_images(in(j), dst, m->re_idx + o, c, per, st); }));
    }
    for (int r = tot; r < bucket; ++r)           // padding: copies of the last gathered image
        CUDA_TRY(cudaMemcpyAsync(m->re_input + (size_t)r * per, m->re_input + (size_t)(tot - 1) * per,
                                 sizeof(float) * per, cudaMemcpyDeviceToDevice, st));
    const bool armed = m->armed;
    m->armed = false;
    uint8_t *const mirror = m->flag_mirror;
    m->flag_mirror = nullptr;
    ct_status s = CT_OK;
    cudaGraphExec_t ex = m->prof ? nullptr : reexec_graph(m, bucket);
    if (ex) {
        int slot = 0;
        while ((1 << slot) < bucket) ++slot;
        if (cudaGraphLaunch(ex, st) != cudaSuccess) s = CT_ECUDA;
        else m->kernels_total += m->re_graph_nk[slot];
    } else {
        s = infer_impl(m, m->re_input, bucket, m->re_logits, m->re_S, m->re_flag, st);
    }
    m->armed = armed;
    m->flag_mirror = mirror;
    if (s != CT_OK) return s;
    for (int j = 0, o = 0; j < nb; o += cnt[j], ++j) {
        if (!cnt[j]) continue;
        const int c = cnt[j];
        float *L = lg(j), *Sj = Sp(j);
        CUDA_TRY(launch(m, FAM_OTHER, 0, st, [&] {
            return launch_scatter_rows(m->re_logits + (size_t)o * m->n_classes, L, m->re_idx + o, c, m->n_classes, st);
        }));
        if (Sj) CUDA_TRY(launch(m, FAM_OTHER, 0, st, [&] { return launch_scatter_rows(m->re_S + o, Sj, m->re_idx + o, c, 1, st); }));
    }
    return CT_OK;
}

// Pipeline resources of ct_infer_batches / ct_run_host_batches, made on the
// first call (host slots only for the host-buffer call).
ct_status pipe_setup(ct_model *m, bool host) {
    if (!m->pipe_ready) {
        const size_t B = (size_t)m->max_batch;
        if (cudaHostAlloc((void **)&m->pipe_flags_h, ct_model::PIPE * B, cudaHostAllocMapped) != cudaSuccess ||
            cudaHostGetDevicePointer((void **)&m->pipe_flags_d, m->pipe_flags_h, 0) != cudaSuccess ||
            cudaHostAlloc((void **)&m->pipe_idx_h, sizeof(int32_t) * (ct_model::PIPE + 2) * B, cudaHostAllocMapped) !=
                cudaSuccess ||
            cudaHostGetDevicePointer((void **)&m->pipe_idx_d, m->pipe_idx_h, 0) != cudaSuccess) {
            cudaGetLastError();
            return CT_ENOMEM;
        }
        for (int i = 0; i < ct_model::PIPE; ++i)
            for (cudaEvent_t *e : {&m->pipe_ev_flags[i], &m->pipe_ev_step[i], &m->pipe_ev_in[i], &m->pipe_ev_out[i]})
                CUDA_TRY(cudaEventCreateWithFlags(e, cudaEventDisableTiming));
        CUDA_TRY(cudaEventCreateWithFlags(&m->pipe_ev_tail, cudaEventDisableTiming));
        CUDA_TRY(cudaStreamCreateWithFlags(&m->pipe_copy, cudaStreamNonBlocking));
        CUDA_TRY(cudaStreamCreateWithFlags(&m->pipe_copy_out, cudaStreamNonBlocking));
        m->pipe_ready = true;
    }
    if (host && !m->pipe_in_d) {
        const size_t B = (size_t)m->max_batch, per = (size_t)m->in_c * m->in_h * m->in_w;
        ct_status st;
        if ((st = dalloc(m, (void **)&m->pipe_in_d, sizeof(float) * ct_model::PIPE * B * per)) != CT_OK ||
            (st = dalloc(m, (void **)&m->pipe_lg_d, sizeof(float) * ct_model::PIPE * B * m->n_classes)) != CT_OK ||
            (st = dalloc(m, (void **)&m->pipe_S_d, sizeof(float) * ct_model::PIPE * B)) != CT_OK ||
            (st = dalloc(m, (void **)&m->pipe_fl_d, ct_model::PIPE * B)) != CT_OK)
            return st;
    }
    return CT_OK;
}

// Buffers of one call of ct_infer_batches (device) or ct_run_host_batches (host).
struct BatchIO {
    const float *const *in;
    float *const *lg;
    float *const *S;
    uint8_t *const *fl;
};

// n batches of `batch` images with the re-execution of Sec. II-B deferred by
// two batches: step i infers batch i and re-runs, as extra rows of the same
// inference, the flagged images of batch i - 2.  The flags of every batch
// are copied to pinned host memory when its inference ends, and the host
// waits for batch i - 2's copy before it launches step i; the device is then
// working on batch i - 1, so the wait does not idle it, and the host stays
// at most two batches ahead.  Host buffers: batch i's input is copied into
// device slot i % PIPE on a copy stream (overlapping the device's work on
// earlier batches) and batch i's results are copied back once its re-run
// rows are written (after step i + 2).  The last two batches' flagged
// images are re-run on their own at the end.  Returns after every result is
// final (and, for host buffers, copied back).
ct_status run_batches(ct_model *m, int n, int batch, const BatchIO &io, bool host, int *n_rerun, cudaStream_t st) {
    constexpr int P = ct_model::PIPE;
    const size_t B = (size_t)m->max_batch, per = (size_t)m->in_c * m->in_h * m->in_w, nc = (size_t)m->n_classes;
    const cudaStream_t cs = m->pipe_copy, co = m->pipe_copy_out;   // inputs in, results out
    int reruns = 0;
    auto dev_in = [&](int i) -> const float * { return host ? m->pipe_in_d + (size_t)(i % P) * B * per : io.in[i]; };
    auto dev_lg = [&](int i) -> float * { return host ? m->pipe_lg_d + (size_t)(i % P) * B * nc : io.lg[i]; };
    auto dev_S = [&](int i) -> float * { return host ? m->pipe_S_d + (size_t)(i % P) * B : io.S[i]; };
    auto dev_fl = [&](int i) -> uint8_t * { return host ? m->pipe_fl_d + (size_t)(i % P) * B : io.fl[i]; };
    auto copy_out = [&](int i) -> ct_status {       // host: results of batch i (co waits for them first)
        const int q = i % P;
        CUDA_TRY(cudaMemcpyAsync(io.lg[i], dev_lg(i), sizeof(float) * nc * batch, cudaMemcpyDeviceToHost, co));
        if (io.S && io.S[i]) CUDA_TRY(cudaMemcpyAsync(io.S[i], dev_S(i), sizeof(float) * batch, cudaMemcpyDeviceToHost, co));
        if (io.fl && io.fl[i]) CUDA_TRY(cudaMemcpyAsync(io.fl[i], dev_fl(i), batch, cudaMemcpyDeviceToHost, co));
        CUDA_TRY(cudaEventRecord(m->pipe_ev_out[q], co));
        return CT_OK;
    };
    for (int i = 0; i < n; ++i) {
        const int s = i % P;
        if (host) {
            // slot s last held batch i - P: its input was last read by step i - P + 2
            // (the re-run gather) and its results were copied out after that step
            if (i >= P) CUDA_TRY(cudaStreamWaitEvent(cs, m->pipe_ev_step[(i - P + 2) % P], 0));
            CUDA_TRY(cudaMemcpyAsync(const_cast<float *>(dev_in(i)), io.in[i], sizeof(float) * per * batch,
                                     cudaMemcpyHostToDevice, cs));
            CUDA_TRY(cudaEventRecord(m->pipe_ev_in[s], cs));
            CUDA_TRY(cudaStreamWaitEvent(st, m->pipe_ev_in[s], 0));
            if (i >= P) CUDA_TRY(cudaStreamWaitEvent(st, m->pipe_ev_out[s], 0));
        }
        ct_status r;
        int nr = 0;
        // the final kernel writes this batch's flags to the mapped host ring too
        m->flag_mirror = m->pipe_flags_d + (size_t)s * B;
        if (i >= 2) {
            const int q = (i - 2) % P;
            CUDA_TRY(cudaEventSynchronize(m->pipe_ev_flags[q]));
            r = infer_with_reruns(m, dev_in(i), batch, dev_lg(i), dev_S(i), dev_fl(i), dev_in(i - 2), batch,
                                  m->pipe_flags_h + (size_t)q * B, dev_lg(i - 2), dev_S(i - 2), &nr,
                                  m->pipe_idx_h + (size_t)s * B, st, m->pipe_idx_d + (size_t)s * B);
        } else {
            r = infer_impl(m, dev_in(i), batch, dev_lg(i), dev_S(i), dev_fl(i), st);
        }
        m->flag_mirror = nullptr;
        if (r != CT_OK) return r;
        reruns += nr;
        CUDA_TRY(cudaEventRecord(m->pipe_ev_flags[s], st));
        CUDA_TRY(cudaEventRecord(m->pipe_ev_step[s], st));
        if (host && i >= 2) {
            CUDA_TRY(cudaStreamWaitEvent(co, m->pipe_ev_step[s], 0));
            ct_status c = copy_out(i - 2);
            if (c != CT_OK) return c;
        }
    }
    // the last two batches: their flagged images re-run together, one batch
    const int k0 = n >= 2 ? n - 2 : 0;
    for (int k = k0; k < n; ++k) CUDA_TRY(cudaEventSynchronize(m->pipe_ev_flags[k % P]));
    int nr = 0;
    ct_status r = reexec_rows_of(m, n - k0, [&](int j) { return dev_in(k0 + j); },
                                 [&](int j) { return (const uint8_t *)(m->pipe_flags_h + (size_t)((k0 + j) % P) * B); },
                                 [&](int j) { return dev_lg(k0 + j); }, [&](int j) { return dev_S(k0 + j); }, batch, &nr,
                                 m->pipe_idx_h + (size_t)P * B, st);
    if (r != CT_OK) return r;
    reruns += nr;
    if (host) {
        CUDA_TRY(cudaEventRecord(m->pipe_ev_tail, st));
        CUDA_TRY(cudaStreamWaitEvent(co, m->pipe_ev_tail, 0));
        for (int k = k0; k < n; ++k) {
            ct_status c = copy_out(k);
            if (c != CT_OK) return c;
        }
        CUDA_TRY(cudaStreamSynchronize(cs));
        CUDA_TRY(cudaStreamSynchronize(co));
    }
    CUDA_TRY(cudaStreamSynchronize(st));
    if (n_rerun) *n_rerun = reruns;
    return CT_OK;
}

}  // namespace

namespace ct {

ct_status model_info(const ct_model *m, ModelInfo *out) {
    if (!m || !out) return CT_EINVAL;
    out->device = m->device;
    out->in_c = m->in_c; out->in_h = m->in_h; out->in_w = m->in_w;
    out->n_classes = m->n_classes;
    out->max_batch = m->max_batch;
    out->protect = m->protect ? 1 : 0;
    return CT_OK;
}

ct_status infer_fault_free(ct_model *m, const float *input, int batch, float *logits, float *S,
                           uint8_t *flag, cudaStream_t st) {
    if (!m || batch < 1 || batch > m->max_batch) return CT_ERANGE;
    const bool armed = m->armed;
    m->armed = false;
    ct_status s = infer_impl(m, input, batch, logits, S, flag, st);
    m->armed = armed;
    return s;
}

cudaError_t reexec_gather(ct_model *m, const float *in, float *out, const int32_t *idx, int n, int64_t per_image,
                          cudaStream_t st) {
    return launch(m, FAM_OTHER, 0, st, [&] { return launch_gather_images(in, out, idx, n, per_image, st); });
}

cudaError_t reexec_scatter(ct_model *m, const float *src, float *dst, const int32_t *idx, int n, int row,
                           cudaStream_t st) {
    return launch(m, FAM_OTHER, 0, st, [&] { return launch_scatter_rows(src, dst, idx, n, row, st); });
}

}  // namespace ct

// ===========================================================================
// C ABI
// ===========================================================================

extern "C" {

ct_status ct_resolve_roles(const ct_model_desc *desc, int32_t *roles) {
    if (!desc || !roles || desc->n_layers < 1 || !desc->layers) return CT_EINVAL;
    return resolve_roles(desc, roles);
}

ct_status ct_build(const ct_model_desc *desc, const float *const *weights, const ct_build_opts *opts,
                   ct_model **out) {
    if (!desc || !weights || !opts || !out || desc->n_layers < 1 || !desc->layers) return CT_EINVAL;
    if (opts->precision != CT_FP32 && opts->precision != CT_FP16) return CT_EINVAL;
    if (opts->protect < CT_PROTECT_NONE || opts->protect > CT_PROTECT_REPLACE) return CT_EINVAL;
    if (opts->max_batch < 1 || desc->in_c < 1 || desc->in_h < 1 || desc->in_w < 1 || desc->n_classes < 1)
        return CT_EINVAL;
    *out = nullptr;
    {
        // the description is checked against the residual rule before any device work
        std::vector<int32_t> roles(desc->n_layers);
        if (resolve_roles(desc, roles.data()) != CT_OK) return CT_EINVAL;
    }
    int ndev = 0;
    if (cudaGetDeviceCount(&ndev) != cudaSuccess || opts->device < 0 || opts->device >= ndev) {
        cudaGetLastError();
        return CT_ECUDA;
    }
    DeviceGuard g(opts->device);
    ct_model *m = new (std::nothrow) ct_model();
    if (!m) return CT_ENOMEM;
    m->device = opts->device;
    m->prec = opts->precision;
    m->protect = opts->protect == CT_PROTECT_WIDEN;
    m->replace = opts->protect == CT_PROTECT_REPLACE;
    m->ds_mode = opts->ds_mode;
    m->max_batch = opts->max_batch;
    m->flags = opts->flags;
    m->in_c = desc->in_c; m->in_h = desc->in_h; m->in_w = desc->in_w;
    m->n_classes = desc->n_classes;
    ct_status s = build_impl(m, desc, weights);
    // the static scratch of ct_reexecute_noalloc is committed here, not on
    // its first call
    if (s == CT_OK) s = noalloc_scratch_setup(m->device);
    if (s != CT_OK) {
        free_all(m);
        delete m;
        return s;
    }
    *out = m;
    return CT_OK;
}

ct_status ct_set_threshold(ct_model *m, double reference, double tau) {
    if (!m || !(tau >= 0.0) || reference != reference) return CT_EINVAL;
    m->ref = reference;
    m->tau = tau;
    return CT_OK;
}

ct_status ct_get_threshold(const ct_model *m, double *reference, double *tau) {
    if (!m || !reference || !tau) return CT_EINVAL;
    *reference = m->ref;
    *tau = m->tau;
    return CT_OK;
}

ct_status ct_infer(ct_model *m, const float *input_dev, int32_t batch, float *logits_dev, float *S_dev,
                   uint8_t *flag_dev, void *stream) {
    if (!m || !input_dev || !logits_dev) return CT_EINVAL;
    if (batch < 1 || batch > m->max_batch) return CT_ERANGE;
    DeviceGuard g(m->device);
    return infer_impl(m, input_dev, batch, logits_dev, S_dev, flag_dev, (cudaStream_t)stream);
}

ct_status ct_inject(ct_model *m, int32_t kind, int32_t layer, int64_t element, int32_t bit) {
    if (!m || layer < 0 || layer >= (int)m->L.size()) return CT_EINVAL;
    const LayerRT &l = m->L[layer];
    if (l.d.op != CT_OP_CONV) return CT_EINVAL;
    if (kind != CT_BUF_WEIGHT && kind != CT_BUF_ACT) return CT_EINVAL;
    const int bits = m->prec == CT_FP16 ? 16 : 32;
    if (bit < 0 || bit >= bits) return CT_ERANGE;
    if (kind == CT_BUF_WEIGHT) {
        const int Kt = l.K + ((l.role == CT_ROLE_CT || l.role == CT_ROLE_PASS) ? 1 : 0);
        const int Ct = weight_in_channels(l);
        if (element < 0 || element >= (int64_t)Kt * Ct * l.R * l.S) return CT_ERANGE;
    } else {
        const Slot &sl = m->slots[l.d.src];
        const int Ct = sl.C + (sl.has_cs ? 1 : 0);
        if (!sl.stored || element < 0 || element >= (int64_t)m->max_batch * Ct * sl.H * sl.W) return CT_ERANGE;
    }
    m->armed = true;
    m->f_kind = kind; m->f_layer = layer; m->f_elem = element; m->f_bit = bit;
    return CT_OK;
}

ct_status ct_clear_faults(ct_model *m) {
    if (!m) return CT_EINVAL;
    m->armed = false;
    return CT_OK;
}

ct_status ct_reexecute(ct_model *m, const float *input_dev, int32_t batch, const uint8_t *flag_dev,
                       float *logits_dev, float *S_dev, int32_t *n_rerun, void *stream) {
    if (!m || !input_dev || !flag_dev || !logits_dev) return CT_EINVAL;
    if (batch < 1 || batch > m->max_batch) return CT_ERANGE;
    DeviceGuard g(m->device);
    int n = 0;
    ct_status s = reexec_impl(m, input_dev, batch, flag_dev, logits_dev, S_dev, &n, (cudaStream_t)stream);
    if (n_rerun) *n_rerun = n;
    return s;
}

ct_status ct_reexecute_prepare(ct_model *m, int32_t max_images) {
    if (!m) return CT_EINVAL;
    if (max_images < 1 || max_images > m->max_batch) return CT_ERANGE;
    DeviceGuard g(m->device);
    // the same buckets reexec_impl uses: powers of two, the last one capped at max_batch
    for (int b = 1;; b <<= 1) {
        const int bucket = b > m->max_batch ? m->max_batch : b;
        if (!reexec_graph(m, bucket)) return CT_ECUDA;
        if (b >= max_images) break;
    }
    return CT_OK;
}

ct_status ct_infer_reexec(ct_model *m, const float *input_dev, int32_t batch, float *logits_dev, float *S_dev,
                          uint8_t *flag_dev, const float *prev_input_dev, int32_t prev_batch,
                          const uint8_t *prev_flag_dev, float *prev_logits_dev, float *prev_S_dev, int32_t *n_rerun,
                          void *stream) {
    if (!m || !input_dev || !logits_dev) return CT_EINVAL;
    if (batch < 1 || batch > m->max_batch) return CT_ERANGE;
    if (prev_input_dev) {
        if (!prev_flag_dev || !prev_logits_dev) return CT_EINVAL;
        if (prev_batch < 1 || prev_batch > m->max_batch) return CT_ERANGE;
    }
    DeviceGuard g(m->device);
    int n = 0;
    ct_status s = infer_reexec_impl(m, input_dev, batch, logits_dev, S_dev, flag_dev, prev_input_dev,
                                    prev_input_dev ? prev_batch : 0, prev_flag_dev, prev_logits_dev, prev_S_dev, &n,
                                    (cudaStream_t)stream);
    if (n_rerun) *n_rerun = n;
    return s;
}

ct_status ct_campaign_batched(ct_model *m, const float *input_dev, int32_t batch, const ct_fault *faults,
                              int32_t n_faults, float *S_dev, int32_t *top1_dev, uint8_t *flag_dev, void *stream) {
    if (!m || !input_dev || (n_faults > 0 && (!faults || !S_dev || !top1_dev || !flag_dev)) || n_faults < 0)
        return CT_EINVAL;
    if (batch < 1 || batch > m->max_batch) return CT_ERANGE;
    SmallNet g;
    if (!m->protect || !small_net_of(m, &g)) return CT_EUNSUPPORTED;
    if (n_faults == 0) return CT_OK;
    g.B = batch;
    g.x = input_dev;
    DeviceGuard dg(m->device);
    cudaStream_t st = (cudaStream_t)stream;
    // resolve every fault on the host, as ct_inject + ct_infer would
    if (n_faults > m->camp_cap) {
        CUDA_TRY(cudaStreamSynchronize(st));
        if (m->camp_h) cudaFreeHost(m->camp_h);
        if (m->camp_d) cudaFree(m->camp_d);
        m->camp_h = nullptr; m->camp_d = nullptr; m->camp_cap = 0;
        if (cudaMallocHost((void **)&m->camp_h, sizeof(CampFault) * n_faults) != cudaSuccess ||
            cudaMalloc((void **)&m->camp_d, sizeof(CampFault) * n_faults) != cudaSuccess) {
            cudaGetLastError();
            return CT_ENOMEM;
        }
        m->camp_cap = n_faults;
    } else {
        CUDA_TRY(cudaStreamSynchronize(st));        // the staging of the previous call was copied
    }
    const int per_img = (g.K1 + 1) * g.Hp1 * g.Wp1;
    for (int i = 0; i < n_faults; ++i) {
        const ct_fault &fi = faults[i];
        CampFault &cf = m->camp_h[i];
        memset(&cf, 0, sizeof(cf));
        cf.kind = fi.kind;
        cf.bit = fi.bit;
        cf.word = -1;
        if (fi.bit < 0 || fi.bit >= 32) return CT_ERANGE;
        if (fi.kind == CT_BUF_WEIGHT) {
            if (fi.layer != 0 && fi.layer != 2) return CT_ERANGE;
            const LayerRT &l = m->L[fi.layer];
            const int64_t n_el = (int64_t)(l.K + 1) * (l.C + (l.cs_in ? 1 : 0)) * l.R * l.S;
            if (fi.element < 0 || fi.element >= n_el) return CT_ERANGE;
            cf.layer = fi.layer == 0 ? 0 : 1;
            const WeightFault wf = resolve_weight_fault(m, l, fi.element, fi.bit);
            if (wf.explicit_word) cf.word = wf.word;
            else cf.fd = wf.fd;
        } else if (fi.kind == CT_BUF_ACT) {
            // the second convolution's input; the network input is not a fault site
            if (fi.layer != 2 || fi.element < 0 || fi.element >= (int64_t)batch * per_img) return CT_ERANGE;
            cf.img = (int)(fi.element / per_img);
            const int within = (int)(fi.element % per_img);
            cf.act_c = within / (g.Hp1 * g.Wp1);
            cf.act_hw = within % (g.Hp1 * g.Wp1);
        } else {
            return CT_EINVAL;
        }
    }
    CUDA_TRY(cudaMemcpyAsync(m->camp_d, m->camp_h, sizeof(CampFault) * n_faults, cudaMemcpyHostToDevice, st));
    CUDA_TRY(launch(m, FAM_OTHER, 0, st, [&] {
        return launch_campaign_small(g, m->camp_d, n_faults, S_dev, top1_dev, flag_dev, st);
    }));
    return CT_OK;
}

ct_status ct_infer_batches(ct_model *m, int32_t n_batches, int32_t batch, const float *const *input_dev,
                           float *const *logits_dev, float *const *S_dev, uint8_t *const *flag_dev, int32_t *n_rerun,
                           void *stream) {
    if (n_rerun) *n_rerun = 0;
    if (!m || n_batches < 0 || (n_batches > 0 && (!input_dev || !logits_dev || !S_dev || !flag_dev))) return CT_EINVAL;
    if (batch < 1 || batch > m->max_batch) return CT_ERANGE;
    for (int i = 0; i < n_batches; ++i)
        if (!input_dev[i] || !logits_dev[i] || !S_dev[i] || !flag_dev[i]) return CT_EINVAL;
    if (n_batches == 0) return CT_OK;
    DeviceGuard g(m->device);
    ct_status s = pipe_setup(m, false);
    if (s != CT_OK) return s;
    int nr = 0;
    s = run_batches(m, n_batches, batch, BatchIO{input_dev, logits_dev, S_dev, flag_dev}, false, &nr,
                    (cudaStream_t)stream);
    if (n_rerun) *n_rerun = nr;
    return s;
}

ct_status ct_run_host_batches(ct_model *m, int32_t n_batches, int32_t batch, const float *const *input_host,
                              float *const *logits_host, float *const *S_host, uint8_t *const *flag_host,
                              int32_t *n_rerun, void *stream) {
    if (n_rerun) *n_rerun = 0;
    if (!m || n_batches < 0 || (n_batches > 0 && (!input_host || !logits_host))) return CT_EINVAL;
    if (batch < 1 || batch > m->max_batch) return CT_ERANGE;
    for (int i = 0; i < n_batches; ++i)
        if (!input_host[i] || !logits_host[i]) return CT_EINVAL;
    if (n_batches == 0) return CT_OK;
    DeviceGuard g(m->device);
    ct_status s = pipe_setup(m, true);
    if (s != CT_OK) return s;
    int nr = 0;
    s = run_batches(m, n_batches, batch, BatchIO{input_host, logits_host, S_host, flag_host}, true, &nr,
                    (cudaStream_t)stream);
    if (n_rerun) *n_rerun = nr;
    return s;
}

ct_status ct_run_host(ct_model *m, const float *input_host, int32_t batch, float *logits_host,
                      float *S_host, uint8_t *flag_host, int32_t *n_rerun, void *stream) {
    if (!m || !input_host || !logits_host) return CT_EINVAL;
    if (batch < 1 || batch > m->max_batch) return CT_ERANGE;
    DeviceGuard g(m->device);
    cudaStream_t st = (cudaStream_t)stream;
    const size_t per = (size_t)m->in_c * m->in_h * m->in_w;
    CUDA_TRY(cudaMemcpyAsync(m->rh_input, input_host, sizeof(float) * per * batch, cudaMemcpyHostToDevice, st));
    ct_status s = infer_impl(m, m->rh_input, batch, m->rh_logits, m->rh_S, m->rh_flag, st);
    if (s != CT_OK) return s;
    int n = 0;
    if (m->protect) {
        s = reexec_impl(m, m->rh_input, batch, m->rh_flag, m->rh_logits, m->rh_S, &n, st);
        if (s != CT_OK) return s;
    }
    if (n_rerun) *n_rerun = n;
    CUDA_TRY(cudaMemcpyAsync(logits_host, m->rh_logits, sizeof(float) * m->n_classes * batch,
                             cudaMemcpyDeviceToHost, st));
    if (S_host) CUDA_TRY(cudaMemcpyAsync(S_host, m->rh_S, sizeof(float) * batch, cudaMemcpyDeviceToHost, st));
    if (flag_host) CUDA_TRY(cudaMemcpyAsync(flag_host, m->rh_flag, batch, cudaMemcpyDeviceToHost, st));
    CUDA_TRY(cudaStreamSynchronize(st));
    return CT_OK;
}

ct_status ct_calibrate(const float *S_host, int64_t n, double alpha, double *reference, double *tau) {
    if (!S_host || n < 1 || !(alpha >= 0.0 && alpha < 1.0) || !reference || !tau) return CT_EINVAL;
    double sum = 0.0;
    for (int64_t i = 0; i < n; ++i) {
        if (!isfinite(S_host[i])) return CT_EINVAL;
        sum += (double)S_host[i];
    }
    const double r = sum / (double)n;
    std::vector<double> dev(n);
    for (int64_t i = 0; i < n; ++i) dev[i] = fabs((double)S_host[i] - r);
    std::sort(dev.begin(), dev.end());
    int64_t rank = (int64_t)ceil((1.0 - alpha) * (double)n);
    rank = std::min<int64_t>(std::max<int64_t>(rank, 1), n);
    *reference = r;
    *tau = dev[rank - 1];
    return CT_OK;
}

ct_status ct_fi_threshold(const float *S_host, const uint8_t *critical, int64_t n, double reference,
                          double alpha, double *tau) {
    if (!S_host || !critical || n < 1 || !(alpha >= 0.0 && alpha < 1.0) || !tau) return CT_EINVAL;
    std::vector<double> dev;
    dev.reserve((size_t)n);
    for (int64_t i = 0; i < n; ++i) {
        if (critical[i]) continue;
        const double d = fabs((double)S_host[i] - reference);
        dev.push_back(d == d ? d : INFINITY);    // a non-finite S deviates without bound
    }
    if (dev.empty()) return CT_EINVAL;
    std::sort(dev.begin(), dev.end());
    const int64_t m = (int64_t)dev.size();
    int64_t rank = (int64_t)ceil((1.0 - alpha) * (double)m);
    rank = std::min<int64_t>(std::max<int64_t>(rank, 1), m);
    *tau = dev[rank - 1];
    return CT_OK;
}

ct_status ct_buffer_count(const ct_model *m, int32_t batch, int32_t *n) {
    if (!m || !n || batch < 1) return CT_EINVAL;
    int cnt = 0;
    std::vector<int> seen;
    for (auto &l : m->L)
        if (l.d.op == CT_OP_CONV) ++cnt;
    for (auto &l : m->L)
        if (l.d.op == CT_OP_CONV && l.d.src != 0 &&
            std::find(seen.begin(), seen.end(), l.d.src) == seen.end()) {
            seen.push_back(l.d.src);
            ++cnt;
        }
    *n = cnt;
    return CT_OK;
}

ct_status ct_buffer_info(const ct_model *m, int32_t batch, int32_t i, int32_t *kind, int32_t *layer,
                         int64_t *n_elements, int32_t *bits) {
    if (!m || batch < 1 || !kind || !layer || !n_elements || !bits) return CT_EINVAL;
    const int b = m->prec == CT_FP16 ? 16 : 32;
    int idx = 0;
    for (size_t li = 0; li < m->L.size(); ++li) {
        const LayerRT &l = m->L[li];
        if (l.d.op != CT_OP_CONV) continue;
        if (idx++ == i) {
            const int Kt = l.K + ((l.role == CT_ROLE_CT || l.role == CT_ROLE_PASS) ? 1 : 0);
            const int Ct = weight_in_channels(l);
            *kind = CT_BUF_WEIGHT; *layer = (int)li; *n_elements = (int64_t)Kt * Ct * l.R * l.S; *bits = b;
            return CT_OK;
        }
    }
    std::vector<int> seen;
    for (size_t li = 0; li < m->L.size(); ++li) {
        const LayerRT &l = m->L[li];
        if (l.d.op != CT_OP_CONV || l.d.src == 0) continue;
        if (std::find(seen.begin(), seen.end(), l.d.src) != seen.end()) continue;
        seen.push_back(l.d.src);
        if (idx++ == i) {
            const Slot &sl = m->slots[l.d.src];
            *kind = CT_BUF_ACT; *layer = (int)li;
            *n_elements = (int64_t)batch * (sl.C + (sl.has_cs ? 1 : 0)) * sl.H * sl.W;
            *bits = b;
            return CT_OK;
        }
    }
    return CT_ERANGE;
}

ct_status ct_profile_enable(ct_model *m, int32_t on) {
    if (!m) return CT_EINVAL;
    m->prof = on != 0;
    return CT_OK;
}

ct_status ct_profile_read(ct_model *m, int32_t family, int64_t *launches, double *ms, double *flops) {
    if (!m || family < 0 || family >= FAM_COUNT || !launches || !ms) return CT_EINVAL;
    DeviceGuard g(m->device);
    int64_t n = 0;
    double t = 0.0, f = 0.0;
    std::vector<EvRec> keep;
    for (const EvRec &r : m->recs) {
        if (r.fam != family) { keep.push_back(r); continue; }
        float e = 0.f;
        CUDA_TRY(cudaEventSynchronize(m->ev_pool[r.ev].second));
        CUDA_TRY(cudaEventElapsedTime(&e, m->ev_pool[r.ev].first, m->ev_pool[r.ev].second));
        t += e;
        f += r.flops;
        n += r.nk;
        m->ev_free.push_back(r.ev);
    }
    m->recs.swap(keep);
    *launches = n;
    *ms = t;
    if (flops) *flops = f;
    return CT_OK;
}

ct_status ct_kernel_count(ct_model *m, int64_t *n) {
    if (!m || !n) return CT_EINVAL;
    *n = m->kernels_total;
    m->kernels_total = 0;
    return CT_OK;
}

ct_status ct_launches_per_infer(const ct_model *m, int32_t *n) {
    if (!m || !n) return CT_EINVAL;
    if (m->n_kernels_last >= 0) { *n = m->n_kernels_last; return CT_OK; }
    int cnt = m->slots[0].stored ? 1 : 0;
    for (auto &l : m->L) cnt += l.fused ? 0 : 1;
    *n = cnt;
    return CT_OK;
}

ct_status ct_copy_activation(ct_model *m, int32_t slot, int32_t batch, void *data_host, void *cs_host,
                             int32_t *C, int32_t *H, int32_t *W, int32_t *has_cs, int32_t *elem_bytes,
                             void *stream) {
    if (!m) return CT_EINVAL;
    if (slot < 0 || slot >= (int)m->slots.size() || batch < 1 || batch > m->max_batch) return CT_ERANGE;
    const Slot &sl = m->slots[slot];
    if (!sl.stored || sl.skipped_last) return CT_ESTATE;
    if (!sl.data) return CT_ERANGE;
    const size_t e = sl.is_float ? 4 : m->esz();
    if (C) *C = sl.cp;
    if (H) *H = sl.H;
    if (W) *W = sl.W;
    if (has_cs) *has_cs = sl.has_cs ? 1 : 0;
    if (elem_bytes) *elem_bytes = (int32_t)e;
    if (!data_host) return CT_OK;
    DeviceGuard g(m->device);
    cudaStream_t st = (cudaStream_t)stream;
    const size_t hw = (size_t)batch * sl.H * sl.W;
    CUDA_TRY(cudaMemcpyAsync(data_host, sl.data, hw * sl.cp * e, cudaMemcpyDeviceToHost, st));
    if (cs_host && sl.has_cs) CUDA_TRY(cudaMemcpyAsync(cs_host, sl.cs, hw * e, cudaMemcpyDeviceToHost, st));
    CUDA_TRY(cudaStreamSynchronize(st));
    return CT_OK;
}

ct_status ct_device_error(ct_model *m, uint32_t *code) {
    if (!m || !code) return CT_EINVAL;
    DeviceGuard g(m->device);
    CUDA_TRY(cudaDeviceSynchronize());
    CUDA_TRY(cudaMemcpy(code, m->d_err, sizeof(uint32_t), cudaMemcpyDeviceToHost));
    CUDA_TRY(cudaMemset(m->d_err, 0, sizeof(uint32_t)));
    return CT_OK;
}

void ct_destroy(ct_model *m) {
    if (!m) return;
    DeviceGuard g(m->device);
    cudaDeviceSynchronize();
    free_all(m);
    delete m;
}

const char *ct_strerror(ct_status s) {
    switch (s) {
        case CT_OK: return "ok";
        case CT_EINVAL: return "invalid argument or model description";
        case CT_ENOMEM: return "out of memory";
        case CT_ECUDA: return "CUDA call failed";
        case CT_ESTATE: return "invalid state";
        case CT_ERANGE: return "index, batch or bit out of range";
        case CT_EUNSUPPORTED: return "unsupported shape";
        case CT_EDEVICE: return "device-side error (bounded wait expired)";
    }
    return "unknown status";
}

}  // extern "C"
