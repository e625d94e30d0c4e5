// C ABI of the QUASAR reconstruction library: argument validation, kernel
// selection and launch configuration.  Declarations and contracts are in
// include/quasar.h.
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdint>
#include <cstdlib>
#include <cstring>
#include <mutex>

#include "params.h"
#include "quasar.h"

namespace quasar {
// integer-code kernels: one entry per (8-candidate chunks, clamp-set size)
#define QUASAR_INT_ENTRY(n, s) const void* int_kernel_nch##n##_ss##s(int epl, bool batch, bool adam, bool var);
QUASAR_INT_ENTRY(1, 8) QUASAR_INT_ENTRY(1, 4) QUASAR_INT_ENTRY(1, 3) QUASAR_INT_ENTRY(1, 2)
QUASAR_INT_ENTRY(1, 1)
QUASAR_INT_ENTRY(2, 4) QUASAR_INT_ENTRY(2, 2) QUASAR_INT_ENTRY(2, 1)
QUASAR_INT_ENTRY(4, 4) QUASAR_INT_ENTRY(4, 2) QUASAR_INT_ENTRY(4, 1)
#undef QUASAR_INT_ENTRY
const void* nvfp4_kernel(int nch, bool batch);
const void* amax_kernel(bool batch);
const void* amax_init_kernel(bool batch);
const void* amax_to_scale_kernel(bool batch);
const void* lut_kernel();
const void* adamw_amax_kernel();
const void* sym_kernel(int epl);
}  // namespace quasar

// Per-device status word (bit 0: a kernel timed out on a wait).
__device__ unsigned int g_quasar_status_word;

namespace {

using namespace quasar;

// 8 warps per CTA: with two 5 KB tiles and the 4 KB transpose scratch per
// warp, two CTAs fit in an SM's shared memory (16 resident warps, at 128
// registers a thread the whole register file).
constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
// The AdamW-fused integer kernel also stages m (14 instead of 10 bytes a
// weight): 6 warps per CTA keep two CTAs in an SM's shared memory.
constexpr int kAdamWarps = 6;
constexpr uint64_t kDefaultTimeoutNs = 1000000000ull;  // 1 s per wait

std::atomic<int64_t> g_force_timeout_ns{0};
std::atomic<unsigned int*> g_stats{nullptr};
std::atomic<int> g_hoist{-1};  // -1: the environment's choice (tuning().hoist)

// The error bounds' defaults are the smallest values their derivations allow
// (the summation-depth bound of the candidate errors, the NVFP4 direct-sum
// bound, the fit error that triggers the compensated fit): an environment
// value below one is raised to it, so a setting can make the careful paths
// run more often but never skip one that correctness needs.  Larger values
// are capped where a float overflow would start to matter.
constexpr float kTieKappaMin = 16.0f;
constexpr float kTieScaleMin = 1.0f;
constexpr float kFitUlpsMin = 8.0f;

struct Tuning {
    int stages = 0;            // 0: chosen from the shared-memory budget
    int smem_budget = 100 * 1024;
    float tie_kappa = kTieKappaMin;  // NVFP4 tie bound, in ulps
    float tie_scale = kTieScaleMin;  // multiplier of the integer kernel's summation-depth bound
    float fit_ulps = kFitUlpsMin;
    int hoist = 1;             // 0: the integer kernel's code-clamp sets hold one candidate
};

// A float from the environment, clamped to [lo, hi] (non-numbers give lo).
float env_float(const char* s, float lo, float hi)
{
    const double x = std::atof(s);
    return !(x >= lo) ? lo : (x > hi ? hi : (float)x);
}

const Tuning& tuning()
{
    static const Tuning t = [] {
        Tuning x;
        if (const char* s = std::getenv("QUASAR_STAGES")) x.stages = std::min(std::max(std::atoi(s), 0), 8);
        if (const char* s = std::getenv("QUASAR_SMEM_BUDGET")) x.smem_budget = std::atoi(s);
        if (const char* s = std::getenv("QUASAR_TIE_KAPPA")) x.tie_kappa = env_float(s, kTieKappaMin, 1e4f);
        if (const char* s = std::getenv("QUASAR_TIE_SCALE")) x.tie_scale = env_float(s, kTieScaleMin, 1e3f);
        if (const char* s = std::getenv("QUASAR_FIT_ULPS")) x.fit_ulps = env_float(s, kFitUlpsMin, 1e4f);
        if (const char* s = std::getenv("QUASAR_HOIST")) x.hoist = std::atoi(s);
        return x;
    }();
    return t;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

bool overlaps(const void* a, size_t na, const void* b, size_t nb)
{
    if (!a || !b || na == 0 || nb == 0) return false;
    const uintptr_t x = reinterpret_cast<uintptr_t>(a), y = reinterpret_cast<uintptr_t>(b);
    return x < y + nb && y < x + na;
}

size_t dtype_size(quasar_dtype d) { return d == QUASAR_BF16 ? 2 : 4; }

bool valid_dtype(quasar_dtype d) { return d == QUASAR_F32 || d == QUASAR_BF16; }

// Checks shared by both reconstruction entry points.  On success fills n.
quasar_status check_common(const float* w, const void* g, quasar_dtype g_dtype, const float* v,
                           float beta2, const float* clip, int n_clip, int64_t rows, int64_t cols,
                           const void* r, quasar_dtype r_dtype, int64_t* n)
{
    if (rows < 0 || cols < 0) return QUASAR_ERR_INVALID_ARG;
    if (rows != 0 && cols > (int64_t(1) << 62) / rows) return QUASAR_ERR_INVALID_ARG;
    *n = rows * cols;
    if (!(beta2 >= 0.0f && beta2 < 1.0f)) return QUASAR_ERR_INVALID_ARG;
    if (!clip || n_clip < 1 || n_clip > kMaxClip) return QUASAR_ERR_INVALID_ARG;
    for (int k = 0; k < n_clip; ++k)
        if (!(clip[k] > 0.0f && clip[k] <= 1.0f)) return QUASAR_ERR_INVALID_ARG;
    if (!valid_dtype(r_dtype) || (g && !valid_dtype(g_dtype))) return QUASAR_ERR_INVALID_ARG;
    if (*n == 0) return QUASAR_OK;
    if (!w || !v || !r) return QUASAR_ERR_INVALID_ARG;
    if (!aligned16(w) || !aligned16(v) || !aligned16(r) || (g && !aligned16(g)))
        return QUASAR_ERR_INVALID_ARG;
    return QUASAR_OK;
}

// Output byte ranges must not overlap w, g or v.
bool outputs_alias_inputs(const float* w, const void* g, quasar_dtype g_dtype, const float* v,
                          int64_t n, const void* const* outs, const size_t* out_bytes, int n_out)
{
    const size_t nb = (size_t)n;
    for (int i = 0; i < n_out; ++i) {
        if (overlaps(outs[i], out_bytes[i], w, nb * 4)) return true;
        if (overlaps(outs[i], out_bytes[i], v, nb * 4)) return true;
        if (g && overlaps(outs[i], out_bytes[i], g, nb * dtype_size(g_dtype))) return true;
    }
    return false;
}

void fill_clip(const float* clip, int n_clip, float* f, float* invf)
{
    for (int k = 0; k < kMaxClip; ++k) {
        const float fk = clip[std::min(k, n_clip - 1)];
        f[k] = fk;
        invf[k] = (float)(1.0 / (double)fk);
    }
}

// Code clamps of the integer kernel.  A set of consecutive candidate slots
// shares one clamp when some tau has J f_max (1 + 1e-3) <= tau <= (J + 1)
// f_min (1 - 1e-3), J = (qmax - 1) / 2: then min(|d|, tau range / qmax) P_k
// has the code min(floor(|d| P_k), J) for every slot k of the set (a capped
// |d| gives cap P_k ~ tau / f_k in [J, J + 1), and below the cap
// |d| P_k < J + 1).  The margin covers the fp32 roundings of the cap, of R
// and of P.  The largest set size of 4, 2, 1 whose sets all qualify is taken
// (a set of one always does), and no larger than max_size; every slot holds
// its set's tau / qmax.  Also the centre factor of each 8-candidate chunk.
void fill_caps(IntParams* p, int max_size, bool single_chunk = false)
{
    const int J = p->qmax >> 1;
    // the sets of a size: consecutive runs of `size` slots; 3: the runs 3, 3,
    // 2 of every 8 slots (3 and 8: with a single chunk only)
    auto first_of = [](int size, int k) { return size == 3 ? 8 * (k / 8) + 3 * ((k % 8) / 3) : k - k % size; };
    auto len_of = [](int size, int k0) { return size == 3 ? (k0 % 8 == 6 ? 2 : 3) : size; };
    auto cap_of = [&](int k0, int n, double* tau) {
        double fmax = 0.0, fmin = 2.0;
        for (int k = k0; k < k0 + n; ++k) {
            fmax = std::max(fmax, (double)p->f[k]);
            fmin = std::min(fmin, (double)p->f[k]);
        }
        const double lo = J * fmax * (1.0 + 1e-3), hi = (J + 1) * fmin * (1.0 - 1e-3);
        *tau = 0.5 * (lo + hi);
        return lo < hi;
    };
    int size = 1;
    for (int cand : {8, 4, 3, 2}) {
        if ((cand == 3 || cand == 8) ? (!single_chunk || max_size < 4) : cand > max_size) continue;
        bool ok = true;
        double tau;
        for (int k0 = 0; k0 < kMaxClip && ok; k0 += len_of(cand, k0)) ok = cap_of(k0, len_of(cand, k0), &tau);
        if (ok) {
            size = cand;
            break;
        }
    }
    p->set_size = size;
    for (int k = 0; k < kMaxClip; ++k) {
        const int k0 = first_of(size, k);
        double tau = 0.0;
        cap_of(k0, len_of(size, k0), &tau);
        p->cap[k] = (float)(tau / p->qmax);
    }
    for (int c = 0; c < kMaxClip / 8; ++c) {
        double lo = 1e300, hi = 0.0;
        for (int k = 8 * c; k < 8 * c + 8 && k < std::max(p->n_clip, 8 * c + 1); ++k) {
            lo = std::min(lo, 1.0 / (double)p->f[k]);
            hi = std::max(hi, 1.0 / (double)p->f[k]);
        }
        p->invfc[c] = (float)(0.5 * (lo + hi));
    }
}

int nch_for(int n_clip) { return n_clip <= 8 ? 1 : (n_clip <= 16 ? 2 : 4); }

struct Launch {
    int stages;
    uint32_t stage_bytes;
    size_t smem;
};

// Shared memory per CTA: for each of its warps, `stages` tiles of
// unit_bytes, a scratch area, and stages + 1 mbarriers.
Launch plan(uint32_t unit_bytes, uint32_t scratch_bytes, int warps = kWarps)
{
    const Tuning& t = tuning();
    Launch L;
    L.stage_bytes = (unit_bytes + 127u) & ~127u;
    auto total = [&](int s) {
        return (size_t)warps * s * L.stage_bytes + (size_t)warps * scratch_bytes +
               (size_t)warps * (s + 1) * 8;
    };
    int s = t.stages;
    if (s <= 0) {
        s = 2;
        while (s < 4 && total(s + 1) <= (size_t)t.smem_budget) ++s;
    }
    L.stages = s;
    L.smem = total(s);
    return L;
}

// Per-device facts looked up once: SM count and the status word's address.
constexpr int kMaxDevices = 64;
struct DeviceInfo {
    std::atomic<int> ready{0};
    int nsm = 0;
    unsigned int* status = nullptr;
};
DeviceInfo g_dev[kMaxDevices];
std::mutex g_mu;

// Launch configuration of one kernel at one shared-memory size, per device.
struct KernelConfig {
    const void* fn = nullptr;
    size_t smem = 0;
    int dev = -1;
    int occupancy = 0;
};
constexpr int kMaxConfigs = 256;
KernelConfig g_cfg[kMaxConfigs];
int g_ncfg = 0;
// Kernels whose dynamic shared-memory limit was raised, per device.  The
// limit is always set to the device's opt-in maximum, so it never has to be
// raised again or lowered for another size (a full table only repeats the
// same setting).
struct SmemLimit {
    const void* fn = nullptr;
    int dev = -1;
};
constexpr int kMaxLimits = 256;
SmemLimit g_limit[kMaxLimits];
int g_nlimit = 0;

quasar_status device_info(int* dev_out, const DeviceInfo** info)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return QUASAR_ERR_CUDA;
    if (dev < 0 || dev >= kMaxDevices) return QUASAR_ERR_UNSUPPORTED;
    DeviceInfo& d = g_dev[dev];
    if (!d.ready.load(std::memory_order_acquire)) {
        std::lock_guard<std::mutex> lock(g_mu);
        if (!d.ready.load(std::memory_order_relaxed)) {
            void* ptr = nullptr;
            if (cudaDeviceGetAttribute(&d.nsm, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
                return QUASAR_ERR_CUDA;
            if (cudaGetSymbolAddress(&ptr, g_quasar_status_word) != cudaSuccess)
                return QUASAR_ERR_CUDA;
            d.status = static_cast<unsigned int*>(ptr);
            d.ready.store(1, std::memory_order_release);
        }
    }
    *dev_out = dev;
    *info = &d;
    return QUASAR_OK;
}

quasar_status status_ptr(unsigned int** p)
{
    int dev;
    const DeviceInfo* info;
    const quasar_status st = device_info(&dev, &info);
    if (st != QUASAR_OK) return st;
    *p = info->status;
    return QUASAR_OK;
}

// Resident CTAs per SM for (fn, smem) on device dev.  The kernel's dynamic
// shared-memory limit is set once per device, to the device's opt-in
// maximum, so every configuration cached earlier stays launchable.
quasar_status occupancy(const void* fn, size_t smem, int threads, int dev, int* occ)
{
    std::lock_guard<std::mutex> lock(g_mu);
    for (int i = 0; i < g_ncfg; ++i)
        if (g_cfg[i].fn == fn && g_cfg[i].dev == dev && g_cfg[i].smem == smem) {
            *occ = g_cfg[i].occupancy;
            return QUASAR_OK;
        }
    bool raised = false;
    for (int i = 0; i < g_nlimit && !raised; ++i) raised = g_limit[i].fn == fn && g_limit[i].dev == dev;
    if (!raised) {
        int optin = 0;
        if (cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess)
            return QUASAR_ERR_CUDA;
        if (smem > (size_t)optin) return QUASAR_ERR_UNSUPPORTED;
        if (cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, optin) != cudaSuccess)
            return QUASAR_ERR_CUDA;
        if (g_nlimit < kMaxLimits) g_limit[g_nlimit++] = SmemLimit{fn, dev};
    }
    int o = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&o, fn, threads, smem) != cudaSuccess)
        return QUASAR_ERR_CUDA;
    if (g_ncfg < kMaxConfigs) g_cfg[g_ncfg++] = KernelConfig{fn, smem, dev, o};
    *occ = o;
    return QUASAR_OK;
}

// Persistent launch: at most (#SMs x resident CTAs) CTAs of `warps` warps,
// no more than there are units of work for the warps.
quasar_status launch_persistent(const void* fn, void* params, size_t smem, int64_t n_units,
                                cudaStream_t stream, int warps = kWarps)
{
    int dev = 0, occ = 0;
    const DeviceInfo* info = nullptr;
    quasar_status st = device_info(&dev, &info);
    if (st != QUASAR_OK) return st;
    if ((st = occupancy(fn, smem, warps * 32, dev, &occ)) != QUASAR_OK) return st;
    if (occ < 1) return QUASAR_ERR_UNSUPPORTED;
    const int64_t want = (n_units + warps - 1) / warps;
    const int grid = (int)std::max<int64_t>(1, std::min<int64_t>((int64_t)info->nsm * occ, want));
    void* args[] = {params};
    if (cudaLaunchKernel(fn, dim3(grid), dim3(warps * 32), args, smem, stream) != cudaSuccess)
        return QUASAR_ERR_CUDA;
    return QUASAR_OK;
}


// Variant options of a call (quasar_options; NULL means the defaults).
struct Opts {
    int h_mode = kSalEma;
    bool packed = false;
    bool symmetric = false;
};

quasar_status read_options(const quasar_options* o, Opts* out)
{
    *out = Opts{};
    if (!o) return QUASAR_OK;
    if (o->saliency != QUASAR_SALIENCY_EMA && o->saliency != QUASAR_SALIENCY_EMA_SQUARED &&
        o->saliency != QUASAR_SALIENCY_UNIFORM)
        return QUASAR_ERR_INVALID_ARG;
    if (o->codes_layout != QUASAR_CODES_U8 && o->codes_layout != QUASAR_CODES_PACKED)
        return QUASAR_ERR_INVALID_ARG;
    if (o->grid != QUASAR_GRID_ASYMMETRIC && o->grid != QUASAR_GRID_SYMMETRIC)
        return QUASAR_ERR_INVALID_ARG;
    out->symmetric = o->grid == QUASAR_GRID_SYMMETRIC;
    out->h_mode = o->saliency == QUASAR_SALIENCY_EMA_SQUARED ? kSalEmaSquared
                  : o->saliency == QUASAR_SALIENCY_UNIFORM   ? kSalUniform
                                                             : kSalEma;
    out->packed = o->codes_layout == QUASAR_CODES_PACKED;
    return QUASAR_OK;
}


// Validation of one tensor of an integer-code call; fills its descriptor
// (unit0 is set by the caller).
quasar_status int_tensor(const float* w, const void* g, quasar_dtype g_dtype, float* v,
                         float beta2, const float* clip, int n_clip, int64_t rows, int64_t cols,
                         void* r, quasar_dtype r_dtype, uint8_t* codes, float* a, float* b,
                         uint8_t* cand_idx, int group_size, IntTensor* T, int bits = 8,
                         bool packed = false)
{
    int64_t n = 0;
    quasar_status st = check_common(w, g, g_dtype, v, beta2, clip, n_clip, rows, cols, r, r_dtype, &n);
    if (st != QUASAR_OK) return st;
    if (group_size <= 0 || cols % group_size != 0) return QUASAR_ERR_INVALID_ARG;
    const int64_t n_groups = n / group_size;
    if (n > 0) {
        if (!a || !b) return QUASAR_ERR_INVALID_ARG;
        if (codes && !aligned16(codes)) return QUASAR_ERR_INVALID_ARG;
        const void* outs[] = {r, codes, a, b, cand_idx};
        const size_t code_bytes = packed ? (size_t)n / 8 * (size_t)bits : (size_t)n;
        const size_t bytes[] = {(size_t)n * dtype_size(r_dtype), codes ? code_bytes : 0,
                                (size_t)n_groups * 4, (size_t)n_groups * 4,
                                cand_idx ? (size_t)n_groups : 0};
        if (outputs_alias_inputs(w, g, g_dtype, v, n, outs, bytes, 5)) return QUASAR_ERR_INVALID_ARG;
    }
    *T = IntTensor{w, g, v, nullptr, r, codes, a, b, cand_idx, n_groups, 0};
    return QUASAR_OK;
}

// Settings shared by the tensors of an integer-code call (no CUDA calls).
quasar_status int_check(int bits, int group_size)
{
    if (bits < 1 || bits > 8) return QUASAR_ERR_INVALID_ARG;
    if (group_size <= 0) return QUASAR_ERR_INVALID_ARG;
    if (group_size != 32 && group_size != 64 && group_size != 128 && group_size != 256)
        return QUASAR_ERR_UNSUPPORTED;
    return QUASAR_OK;
}

// Hyper-parameters of the fused AdamW step (validated by the caller).
struct AdamHp {
    float lr, beta1, eps, weight_decay;
    int64_t step;
};

// Stage bytes of one unit of the symmetric-code kernel: w, v, g.
uint32_t int_unit_bytes(int group_size, int g_kind, bool adam)
{
    const int gbytes = g_kind == 2 ? 2 : (g_kind == 1 ? 4 : 0);
    return (uint32_t)(kGroupsPerUnit * group_size * ((adam ? 12 : 8) + gbytes));
}

// Shared memory of the asymmetric integer kernel's CTA ring: S slots of one
// unit tile each (w, v, m for the fused AdamW step, then the gradient
// region, which is also the transpose scratch and so at least
// kIntXposeBytes), S + 1 mbarriers and S sequence words.  S is one slot a
// warp plus `extra` slots in flight (QUASAR_STAGES, default 2).
Launch plan_ring(int group_size, int g_kind, bool adam, int warps)
{
    const uint32_t gbytes = g_kind == 2 ? 2u : (g_kind == 1 ? 4u : 0u);
    const uint32_t unit = (uint32_t)(kIntGroups * group_size);
    const uint32_t tile = unit * (adam ? 12u : 8u) + std::max(unit * gbytes, kIntXposeBytes);
    Launch L;
    L.stage_bytes = (tile + 127u) & ~127u;
    auto total = [&](int s) {
        return (size_t)s * L.stage_bytes + (size_t)(s + 1) * 8 + (size_t)s * 4;
    };
    int extra = tuning().stages;
    if (extra <= 0) {
        // two slots in flight, one if that keeps two CTAs on an SM (each
        // CTA's share of the SM's 228 KB, less the 1 KB the system keeps);
        // one if two would exceed the 227 KB a CTA may have
        constexpr size_t kTwoCtas = 113 * 1024, kOneCta = 227 * 1024;
        extra = 2;
        if ((total(warps + 2) > kTwoCtas && total(warps + 1) <= kTwoCtas) || total(warps + 2) > kOneCta)
            extra = 1;
    }
    L.stages = warps + extra;
    L.smem = total(L.stages);
    return L;
}

// Parameters shared by the tensors of an integer-code call (adam: the
// AdamW-fused variant's step, else nullptr).
quasar_status int_params(quasar_dtype g_dtype, bool has_g, float beta2, int bits, int group_size,
                         const float* clip, int n_clip, quasar_dtype r_dtype, IntParams* p,
                         const AdamHp* adam = nullptr, const Opts& opt = Opts{})
{
    quasar_status st0 = int_check(bits, group_size);
    if (st0 != QUASAR_OK) return st0;
    *p = IntParams{};
    p->g_kind = has_g ? (g_dtype == QUASAR_BF16 ? 2 : 1) : 0;
    p->r_bf16 = r_dtype == QUASAR_BF16;
    p->h_mode = opt.h_mode;
    p->codes_packed = opt.packed;
    p->bits = bits;
    p->qmax = (1 << bits) - 1;
    p->n_clip = n_clip;
    p->beta2 = beta2;
    p->c1 = 1.0f - beta2;
    // each candidate sum is accumulated over at most G/8 (asymmetric kernel:
    // 4 lanes a group) or G/16 (symmetric: 8 lanes) terms a packed half, plus
    // the halves' sum and the lane tree (2 or 3 levels); the terms' own
    // roundings and those that form N, D and E make up the rest
    p->tie_kappa = tuning().tie_scale * (float)(group_size / (opt.symmetric ? 16 : 8) + 8);
    p->fit_ulps = tuning().fit_ulps;
    p->timeout_ns = kDefaultTimeoutNs;
    p->force_timeout_ns = (uint64_t)std::max<int64_t>(0, g_force_timeout_ns.load());
    p->stats = g_stats.load();
    fill_clip(clip, n_clip, p->f, p->invf);
    fill_caps(p, 4);
    p->monotone = 1;
    for (int k = 1; k < n_clip; ++k) p->monotone &= p->invf[k] >= p->invf[k - 1] ? 1 : 0;
    quasar_status st;
    if ((st = status_ptr(&p->status)) != QUASAR_OK) return st;
    if (adam) {
        // fp32 constants of the step, formed in double from the fp32
        // hyper-parameters: w' = w - (w*lr*wd + step_size * m' / den),
        // den = sqrt(v') / sqrt(1 - beta2^t) + eps
        const double t = (double)adam->step;
        p->beta1 = adam->beta1;
        p->c1b = 1.0f - adam->beta1;
        p->lr_wd = (float)((double)adam->lr * (double)adam->weight_decay);
        p->step_size = (float)((double)adam->lr / (1.0 - std::pow((double)adam->beta1, t)));
        p->isbc2 = (float)(1.0 / std::sqrt(1.0 - std::pow((double)beta2, t)));
        p->eps = adam->eps;
    }
    return QUASAR_OK;
}

// Number the tensors' units consecutively and launch over all of them.
template <int MAXT>
quasar_status int_launch(IntLaunch<MAXT>& Lp, int group_size, int n_clip, cudaStream_t stream,
                         bool adam = false, bool symmetric = false)
{
    // units: 8 groups for the asymmetric kernel, 4 for the symmetric one
    const int per_unit = symmetric ? kGroupsPerUnit : kIntGroups;
    int64_t units = 0;
    for (int i = 0; i < Lp.n_t; ++i) {
        Lp.t[i].unit0 = units;
        units += (Lp.t[i].n_groups + per_unit - 1) / per_unit;
    }
    Lp.n_units = units;
    if (units == 0) return QUASAR_OK;
    const int warps = adam ? kAdamWarps : kWarps;
    const Launch L = symmetric ? plan(int_unit_bytes(group_size, Lp.p.g_kind, adam), kIntScratchBytes, warps)
                               : plan_ring(group_size, Lp.p.g_kind, adam, warps);
    Lp.p.stages = L.stages;
    Lp.p.stage_bytes = L.stage_bytes;
    const int epl = group_size / (symmetric ? kLanesPerGroup : kIntLanes);
    const int nch = nch_for(n_clip);
    const bool batch = MAXT > 1;
    const bool var = Lp.p.h_mode != kSalEma || Lp.p.codes_packed;
    // clamp sets: as large as the factors allow, unless switched off (sets of
    // one); the option variants are built with sets of one, the fused AdamW
    // step with sets of four or one
    const int hoist_on = g_hoist.load() < 0 ? tuning().hoist : g_hoist.load();
    // (sets of 8 or 3-3-2 with a single chunk, not for the fused AdamW step)
    fill_caps(&Lp.p, (!hoist_on || var) ? 1 : 4, nch == 1 && !adam);
    if (adam && Lp.p.set_size == 2) fill_caps(&Lp.p, 1);
    using Entry = const void* (*)(int, bool, bool, bool);
    static const Entry table[3][5] = {
        {int_kernel_nch1_ss8, int_kernel_nch1_ss4, int_kernel_nch1_ss3, int_kernel_nch1_ss2, int_kernel_nch1_ss1},
        {nullptr, int_kernel_nch2_ss4, nullptr, int_kernel_nch2_ss2, int_kernel_nch2_ss1},
        {nullptr, int_kernel_nch4_ss4, nullptr, int_kernel_nch4_ss2, int_kernel_nch4_ss1}};
    const int ci = nch == 1 ? 0 : (nch == 2 ? 1 : 2);
    const int ss = Lp.p.set_size;
    const int si = ss == 8 ? 0 : (ss == 4 ? 1 : (ss == 3 ? 2 : (ss == 2 ? 3 : 4)));
    if (!table[ci][si]) return QUASAR_ERR_UNSUPPORTED;
    const void* fn = symmetric ? (MAXT > 1 ? sym_kernel(epl) : nullptr)
                               : table[ci][si](epl, batch, adam, var);
    if (!fn) return QUASAR_ERR_UNSUPPORTED;
    return launch_persistent(fn, &Lp, L.smem, units, stream, warps);
}

// Validation of one tensor of an NVFP4 call; fills its descriptor and its
// absmax/scale item (unit0 is set later).
quasar_status nvfp4_tensor(const float* w, const void* g, quasar_dtype g_dtype, float* v,
                           float beta2, const float* clip, int n_clip, int64_t rows, int64_t cols,
                           const float* tensor_amax, void* r, quasar_dtype r_dtype, uint8_t* codes,
                           uint8_t* block_scale, float* tensor_scale, uint8_t* cand_idx,
                           Nvfp4Tensor* T, AmaxItem* A, bool packed = false)
{
    int64_t n = 0;
    quasar_status st = check_common(w, g, g_dtype, v, beta2, clip, n_clip, rows, cols, r, r_dtype, &n);
    if (st != QUASAR_OK) return st;
    if (cols % 16 != 0) return QUASAR_ERR_INVALID_ARG;
    if (!tensor_scale || (reinterpret_cast<uintptr_t>(tensor_scale) & 3u) != 0)
        return QUASAR_ERR_INVALID_ARG;
    if (tensor_amax && (reinterpret_cast<uintptr_t>(tensor_amax) & 3u) != 0)
        return QUASAR_ERR_INVALID_ARG;
    const int64_t n_blocks = n / 16;
    if (n > 0) {
        if (!block_scale) return QUASAR_ERR_INVALID_ARG;
        if (codes && !aligned16(codes)) return QUASAR_ERR_INVALID_ARG;
        const void* outs[] = {r, codes, block_scale, tensor_scale, cand_idx};
        const size_t bytes[] = {(size_t)n * dtype_size(r_dtype),
                                codes ? (packed ? (size_t)n / 2 : (size_t)n) : 0, (size_t)n_blocks, 4,
                                cand_idx ? (size_t)n_blocks : 0};
        if (outputs_alias_inputs(w, g, g_dtype, v, n, outs, bytes, 5)) return QUASAR_ERR_INVALID_ARG;
        if (tensor_amax && overlaps(tensor_amax, 4, tensor_scale, 4)) return QUASAR_ERR_INVALID_ARG;
    }
    *T = Nvfp4Tensor{w, g, v, r, codes, block_scale, cand_idx, tensor_scale, n_blocks, 0};
    *A = AmaxItem{w, n, tensor_scale, tensor_amax};
    return QUASAR_OK;
}

quasar_status nvfp4_params(bool has_g, quasar_dtype g_dtype, float beta2, const float* clip,
                           int n_clip, quasar_dtype r_dtype, Nvfp4Params* p,
                           const Opts& opt = Opts{})
{
    *p = Nvfp4Params{};
    p->g_kind = has_g ? (g_dtype == QUASAR_BF16 ? 2 : 1) : 0;
    p->r_bf16 = r_dtype == QUASAR_BF16;
    p->h_mode = opt.h_mode;
    p->codes_packed = opt.packed;
    p->n_clip = n_clip;
    p->beta2 = beta2;
    p->c1 = 1.0f - beta2;
    p->tie_kappa = tuning().tie_kappa;
    p->timeout_ns = kDefaultTimeoutNs;
    p->force_timeout_ns = (uint64_t)std::max<int64_t>(0, g_force_timeout_ns.load());
    p->stats = g_stats.load();
    fill_clip(clip, n_clip, p->f, p->invf);
    return status_ptr(&p->status);
}

// The absmax slots of a batch set to 0 (those of the tensors whose amax is
// computed, or all of them), in one launch.
template <int MAXT>
quasar_status zero_amax_slots(const AmaxBatch<MAXT>& B, bool all, cudaStream_t s)
{
    int flag = all ? 1 : 0;
    void* args[] = {(void*)&B, (void*)&flag};
    if (cudaLaunchKernel(amax_init_kernel(MAXT > 1), dim3(1), dim3(256), args, 0, s) != cudaSuccess)
        return QUASAR_ERR_CUDA;
    return QUASAR_OK;
}

// Absmax of the tensors whose amax is not supplied, into their scale slots
// (zeroed first by the caller of each slot), then every slot := s_T.
template <int MAXT>
quasar_status launch_amax(const AmaxBatch<MAXT>& B, cudaStream_t s)
{
    int dev = 0;
    const DeviceInfo* info = nullptr;
    const quasar_status st = device_info(&dev, &info);
    if (st != QUASAR_OK) return st;
    int64_t nmax = 0;
    for (int i = 0; i < B.n_t; ++i)
        if (!B.t[i].amax_in) nmax = std::max(nmax, B.t[i].n);
    if (nmax == 0) return QUASAR_OK;
    const int64_t want = (nmax / 4 + kThreads - 1) / kThreads;
    const int64_t per_sm = std::max<int64_t>(1, (int64_t)info->nsm * 8 / B.n_t);
    const int gx = (int)std::max<int64_t>(1, std::min<int64_t>(per_sm, want));
    void* args[] = {(void*)&B};
    if (cudaLaunchKernel(amax_kernel(MAXT > 1), dim3(gx, B.n_t), dim3(kThreads), args, 0, s) !=
        cudaSuccess)
        return QUASAR_ERR_CUDA;
    return QUASAR_OK;
}

// amax_done: the slots already hold each tensor's absmax (the fused AdamW
// step took it), so only the scale pass and the reconstruction remain.
template <int MAXT>
quasar_status nvfp4_run(Nvfp4Launch<MAXT>& Lp, AmaxBatch<MAXT>& B, int n_clip, cudaStream_t s,
                        bool amax_done = false)
{
    quasar_status st;
    if (!amax_done) {
        // scale slots of tensors whose amax is computed start at 0
        bool any = false;
        for (int i = 0; i < B.n_t; ++i) any |= !B.t[i].amax_in;
        if (any && (st = zero_amax_slots(B, false, s)) != QUASAR_OK) return st;
        if ((st = launch_amax(B, s)) != QUASAR_OK) return st;
    }
    {
        void* args[] = {(void*)&B};
        if (cudaLaunchKernel(amax_to_scale_kernel(MAXT > 1), dim3(1), dim3(256), args, 0, s) !=
            cudaSuccess)
            return QUASAR_ERR_CUDA;
    }
    int64_t units = 0;
    for (int i = 0; i < Lp.n_t; ++i) {
        Lp.t[i].unit0 = units;
        units += (Lp.t[i].n_blocks + kBlocksPerUnit - 1) / kBlocksPerUnit;
    }
    Lp.n_units = units;
    if (units == 0) return QUASAR_OK;
    const int gbytes = Lp.p.g_kind == 2 ? 2 : (Lp.p.g_kind == 1 ? 4 : 0);
    const Launch L = plan((uint32_t)(kBlocksPerUnit * 16 * (8 + gbytes)), 0);
    Lp.p.stages = L.stages;
    Lp.p.stage_bytes = L.stage_bytes;
    const void* fn = nvfp4_kernel(nch_for(n_clip), MAXT > 1);
    if (!fn) return QUASAR_ERR_UNSUPPORTED;
    return launch_persistent(fn, &Lp, L.smem, units, s);
}

}  // namespace

extern "C" {

quasar_status quasar_recon_int(const float* w, const void* g, quasar_dtype g_dtype, float* v,
                               float beta2, int bits, int group_size, const float* clip,
                               int n_clip, int64_t rows, int64_t cols, void* r,
                               quasar_dtype r_dtype, uint8_t* codes, float* a, float* b,
                               uint8_t* cand_idx, quasar_stream_t stream)
{
    IntLaunch<1> Lp;
    quasar_status st = int_tensor(w, g, g_dtype, v, beta2, clip, n_clip, rows, cols, r, r_dtype,
                                  codes, a, b, cand_idx, group_size > 0 ? group_size : 1, &Lp.t[0]);
    if (st != QUASAR_OK) return st;
    if ((st = int_check(bits, group_size)) != QUASAR_OK) return st;
    if (Lp.t[0].n_groups == 0) return QUASAR_OK;  // empty: no-op
    if ((st = int_params(g_dtype, g != nullptr, beta2, bits, group_size, clip, n_clip, r_dtype,
                         &Lp.p)) != QUASAR_OK)
        return st;
    Lp.n_t = 1;
    return int_launch(Lp, group_size, n_clip, reinterpret_cast<cudaStream_t>(stream));
}

quasar_status quasar_recon_int_batch(const quasar_int_tensor* tensors, int n_tensors,
                                     quasar_dtype g_dtype, float beta2, int bits, int group_size,
                                     const float* clip, int n_clip, quasar_dtype r_dtype,
                                     quasar_stream_t stream)
{
    return quasar_recon_int_batch_ex(tensors, n_tensors, g_dtype, beta2, bits, group_size, clip,
                                     n_clip, r_dtype, nullptr, stream);
}

quasar_status quasar_recon_int_batch_ex(const quasar_int_tensor* tensors, int n_tensors,
                                        quasar_dtype g_dtype, float beta2, int bits,
                                        int group_size, const float* clip, int n_clip,
                                        quasar_dtype r_dtype, const quasar_options* options,
                                        quasar_stream_t stream)
{
    Opts opt;
    if (read_options(options, &opt) != QUASAR_OK) return QUASAR_ERR_INVALID_ARG;
    if (n_tensors < 0 || (n_tensors > 0 && !tensors)) return QUASAR_ERR_INVALID_ARG;
    if (opt.symmetric && bits < 2) return QUASAR_ERR_INVALID_ARG;  // Q = 2^(bits-1) - 1 >= 1
    if (n_tensors == 0) return QUASAR_OK;
    // all non-empty tensors carry a gradient, or none does
    int with_g = 0, non_empty = 0;
    for (int i = 0; i < n_tensors; ++i)
        if (tensors[i].rows != 0 && tensors[i].cols != 0) {
            ++non_empty;
            with_g += tensors[i].g != nullptr;
        }
    if (with_g != 0 && with_g != non_empty) return QUASAR_ERR_INVALID_ARG;
    const bool has_g = with_g != 0;
    static thread_local IntLaunch<kMaxBatch> Lp;  // 20 KB: kept off the stack
    quasar_status st = int_check(bits, group_size);
    if (st != QUASAR_OK) return st;
    // validate every tensor before launching anything
    int64_t total = 0;
    for (int i = 0; i < n_tensors; ++i) {
        const quasar_int_tensor& x = tensors[i];
        IntTensor T;
        if ((st = int_tensor(x.w, x.g, g_dtype, x.v, beta2, clip, n_clip, x.rows, x.cols, x.r,
                             r_dtype, x.codes, x.a, x.b, x.cand_idx, group_size, &T, bits,
                             opt.packed)) != QUASAR_OK)
            return st;
        total += T.n_groups;
    }
    if (total == 0) return QUASAR_OK;
    if ((st = int_params(g_dtype, has_g, beta2, bits, group_size, clip, n_clip, r_dtype, &Lp.p,
                         nullptr, opt)) != QUASAR_OK)
        return st;
    const cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    for (int i0 = 0; i0 < n_tensors; i0 += kMaxBatch) {
        Lp.n_t = std::min(kMaxBatch, n_tensors - i0);
        for (int i = 0; i < Lp.n_t; ++i) {
            const quasar_int_tensor& x = tensors[i0 + i];
            int_tensor(x.w, x.g, g_dtype, x.v, beta2, clip, n_clip, x.rows, x.cols, x.r, r_dtype,
                       x.codes, x.a, x.b, x.cand_idx, group_size, &Lp.t[i], bits, opt.packed);
        }
        if ((st = int_launch(Lp, group_size, n_clip, s, false, opt.symmetric)) != QUASAR_OK) return st;
    }
    return QUASAR_OK;
}

quasar_status quasar_adamw_recon_int_batch(const quasar_adamw_tensor* tensors, int n_tensors,
                                           quasar_dtype g_dtype, float lr, float beta1,
                                           float beta2, float eps, float weight_decay,
                                           int64_t step, int bits, int group_size,
                                           const float* clip, int n_clip, quasar_dtype r_dtype,
                                           const quasar_options* options, quasar_stream_t stream)
{
    Opts opt;
    if (read_options(options, &opt) != QUASAR_OK) return QUASAR_ERR_INVALID_ARG;
    if (opt.symmetric) return QUASAR_ERR_UNSUPPORTED;  // no fused AdamW kernel for symmetric codes
    if (n_tensors < 0 || (n_tensors > 0 && !tensors)) return QUASAR_ERR_INVALID_ARG;
    if (!(std::isfinite(lr) && lr >= 0.0f) || !(beta1 >= 0.0f && beta1 < 1.0f) ||
        !(std::isfinite(eps) && eps > 0.0f) ||
        !(std::isfinite(weight_decay) && weight_decay >= 0.0f) || step < 1)
        return QUASAR_ERR_INVALID_ARG;
    if (n_tensors == 0) return QUASAR_OK;
    static thread_local IntLaunch<kMaxBatch> Lp;
    quasar_status st = int_check(bits, group_size);
    if (st != QUASAR_OK) return st;
    // one tensor's descriptor; checks beyond those of the reconstruction:
    // g and m present, and w, g, m, v pairwise disjoint
    auto describe = [&](const quasar_adamw_tensor& x, IntTensor* T) {
        quasar_status s1 = int_tensor(x.w, x.g, g_dtype, x.v, beta2, clip, n_clip, x.rows, x.cols,
                                      x.r, r_dtype, x.codes, x.a, x.b, x.cand_idx, group_size, T,
                                      bits, opt.packed);
        if (s1 != QUASAR_OK) return s1;
        T->m = x.m;
        if (T->n_groups == 0) return QUASAR_OK;
        if (!x.g || !x.m || !aligned16(x.m)) return QUASAR_ERR_INVALID_ARG;
        const size_t n = (size_t)(x.rows * x.cols);
        const void* outs[] = {x.r, x.codes, x.a, x.b, x.cand_idx};
        const size_t bytes[] = {n * dtype_size(r_dtype), x.codes ? (opt.packed ? n / 8 * bits : n) : 0,
                                (size_t)T->n_groups * 4, (size_t)T->n_groups * 4,
                                x.cand_idx ? (size_t)T->n_groups : 0};
        for (int i = 0; i < 5; ++i)
            if (overlaps(outs[i], bytes[i], x.m, n * 4)) return QUASAR_ERR_INVALID_ARG;
        const void* state[] = {x.w, x.g, x.m, x.v};
        const size_t sbytes[] = {n * 4, n * dtype_size(g_dtype), n * 4, n * 4};
        for (int i = 0; i < 4; ++i)
            for (int j = i + 1; j < 4; ++j)
                if (overlaps(state[i], sbytes[i], state[j], sbytes[j])) return QUASAR_ERR_INVALID_ARG;
        return QUASAR_OK;
    };
    int64_t total = 0;
    for (int i = 0; i < n_tensors; ++i) {
        IntTensor T;
        if ((st = describe(tensors[i], &T)) != QUASAR_OK) return st;
        total += T.n_groups;
    }
    if (total == 0) return QUASAR_OK;
    const AdamHp hp{lr, beta1, eps, weight_decay, step};
    if ((st = int_params(g_dtype, true, beta2, bits, group_size, clip, n_clip, r_dtype, &Lp.p,
                         &hp, opt)) != QUASAR_OK)
        return st;
    const cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    for (int i0 = 0; i0 < n_tensors; i0 += kMaxBatch) {
        Lp.n_t = std::min(kMaxBatch, n_tensors - i0);
        for (int i = 0; i < Lp.n_t; ++i) describe(tensors[i0 + i], &Lp.t[i]);
        if ((st = int_launch(Lp, group_size, n_clip, s, true)) != QUASAR_OK) return st;
    }
    return QUASAR_OK;
}

quasar_status quasar_tensor_amax(const float* w, int64_t n, float* amax_out, quasar_stream_t stream)
{
    if (n < 0 || !amax_out) return QUASAR_ERR_INVALID_ARG;
    if (n > 0 && (!w || !aligned16(w))) return QUASAR_ERR_INVALID_ARG;
    if ((reinterpret_cast<uintptr_t>(amax_out) & 3u) != 0) return QUASAR_ERR_INVALID_ARG;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    if (cudaMemsetAsync(amax_out, 0, sizeof(float), s) != cudaSuccess) return QUASAR_ERR_CUDA;
    if (n == 0) return QUASAR_OK;
    AmaxBatch<1> B;
    B.n_t = 1;
    B.t[0] = AmaxItem{w, n, amax_out, nullptr};
    return launch_amax(B, s);
}

quasar_status quasar_recon_nvfp4(const float* w, const void* g, quasar_dtype g_dtype, float* v,
                                 float beta2, const float* clip, int n_clip, int64_t rows,
                                 int64_t cols, const float* tensor_amax, void* r,
                                 quasar_dtype r_dtype, uint8_t* codes, uint8_t* block_scale,
                                 float* tensor_scale, uint8_t* cand_idx, quasar_stream_t stream)
{
    Nvfp4Launch<1> Lp;
    AmaxBatch<1> B;
    quasar_status st = nvfp4_tensor(w, g, g_dtype, v, beta2, clip, n_clip, rows, cols, tensor_amax, r,
                                    r_dtype, codes, block_scale, tensor_scale, cand_idx, &Lp.t[0],
                                    &B.t[0]);
    if (st != QUASAR_OK) return st;
    Lp.n_t = B.n_t = 1;
    if ((st = nvfp4_params(g != nullptr, g_dtype, beta2, clip, n_clip, r_dtype, &Lp.p)) != QUASAR_OK)
        return st;
    return nvfp4_run(Lp, B, n_clip, reinterpret_cast<cudaStream_t>(stream));
}

quasar_status quasar_recon_nvfp4_batch(const quasar_nvfp4_tensor* tensors, int n_tensors,
                                       quasar_dtype g_dtype, float beta2, const float* clip,
                                       int n_clip, quasar_dtype r_dtype, quasar_stream_t stream)
{
    return quasar_recon_nvfp4_batch_ex(tensors, n_tensors, g_dtype, beta2, clip, n_clip, r_dtype,
                                       nullptr, stream);
}

quasar_status quasar_recon_nvfp4_batch_ex(const quasar_nvfp4_tensor* tensors, int n_tensors,
                                          quasar_dtype g_dtype, float beta2, const float* clip,
                                          int n_clip, quasar_dtype r_dtype,
                                          const quasar_options* options, quasar_stream_t stream)
{
    Opts opt;
    if (read_options(options, &opt) != QUASAR_OK) return QUASAR_ERR_INVALID_ARG;
    if (opt.symmetric) return QUASAR_ERR_INVALID_ARG;  // an integer-code option
    if (n_tensors < 0 || (n_tensors > 0 && !tensors)) return QUASAR_ERR_INVALID_ARG;
    if (n_tensors == 0) return QUASAR_OK;
    int with_g = 0, non_empty = 0;
    for (int i = 0; i < n_tensors; ++i)
        if (tensors[i].rows != 0 && tensors[i].cols != 0) {
            ++non_empty;
            with_g += tensors[i].g != nullptr;
        }
    if (with_g != 0 && with_g != non_empty) return QUASAR_ERR_INVALID_ARG;
    const bool has_g = with_g != 0;
    static thread_local Nvfp4Launch<kMaxBatch> Lp;  // kept off the stack
    static thread_local AmaxBatch<kMaxBatch> B;
    quasar_status st;
    for (int i = 0; i < n_tensors; ++i) {  // validate everything first
        const quasar_nvfp4_tensor& x = tensors[i];
        Nvfp4Tensor T;
        AmaxItem A;
        if ((st = nvfp4_tensor(x.w, x.g, g_dtype, x.v, beta2, clip, n_clip, x.rows, x.cols,
                               x.tensor_amax, x.r, r_dtype, x.codes, x.block_scale, x.tensor_scale,
                               x.cand_idx, &T, &A, opt.packed)) != QUASAR_OK)
            return st;
    }
    if ((st = nvfp4_params(has_g, g_dtype, beta2, clip, n_clip, r_dtype, &Lp.p, opt)) != QUASAR_OK)
        return st;
    const cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    for (int i0 = 0; i0 < n_tensors; i0 += kMaxBatch) {
        Lp.n_t = B.n_t = std::min(kMaxBatch, n_tensors - i0);
        for (int i = 0; i < Lp.n_t; ++i) {
            const quasar_nvfp4_tensor& x = tensors[i0 + i];
            nvfp4_tensor(x.w, x.g, g_dtype, x.v, beta2, clip, n_clip, x.rows, x.cols, x.tensor_amax,
                         x.r, r_dtype, x.codes, x.block_scale, x.tensor_scale, x.cand_idx, &Lp.t[i],
                         &B.t[i], opt.packed);
        }
        if ((st = nvfp4_run(Lp, B, n_clip, s)) != QUASAR_OK) return st;
    }
    return QUASAR_OK;
}

quasar_status quasar_recon_lut_batch(const quasar_lut_tensor* tensors, int n_tensors,
                                     quasar_dtype g_dtype, float beta2, const float* clip,
                                     int n_clip, quasar_dtype r_dtype, const quasar_options* options,
                                     quasar_stream_t stream)
{
    Opts opt;
    if (read_options(options, &opt) != QUASAR_OK) return QUASAR_ERR_INVALID_ARG;
    if (opt.symmetric) return QUASAR_ERR_INVALID_ARG;  // an integer-code option
    if (n_tensors < 0 || (n_tensors > 0 && !tensors)) return QUASAR_ERR_INVALID_ARG;
    if (n_tensors == 0) return QUASAR_OK;
    int with_g = 0, non_empty = 0;
    for (int i = 0; i < n_tensors; ++i)
        if (tensors[i].rows != 0 && tensors[i].cols != 0) {
            ++non_empty;
            with_g += tensors[i].g != nullptr;
        }
    if (with_g != 0 && with_g != non_empty) return QUASAR_ERR_INVALID_ARG;
    const bool has_g = with_g != 0;
    // one tensor's checks; fills its descriptor (unit0 set later)
    auto describe = [&](const quasar_lut_tensor& x, LutTensor* T) {
        int64_t n = 0;
        quasar_status s1 = check_common(x.w, x.g, g_dtype, x.v, beta2, clip, n_clip, x.rows, x.cols,
                                        x.r, r_dtype, &n);
        if (s1 != QUASAR_OK) return s1;
        if (x.rows % kLutRows != 0 || x.cols % kLutCols != 0) return QUASAR_ERR_INVALID_ARG;
        const int64_t n_blocks = n / kLutBlock;
        if (n_blocks > (int64_t)UINT32_MAX) return QUASAR_ERR_INVALID_ARG;  // 32-bit block indices
        if (n > 0) {
            if (!x.book || !aligned16(x.book)) return QUASAR_ERR_INVALID_ARG;
            if (x.codes && !aligned16(x.codes)) return QUASAR_ERR_INVALID_ARG;
            const void* outs[] = {x.r, x.codes, x.book, x.cand_idx};
            const size_t bytes[] = {(size_t)n * dtype_size(r_dtype),
                                    x.codes ? (opt.packed ? (size_t)n / 8 * 3 : (size_t)n) : 0,
                                    (size_t)n_blocks * 8, x.cand_idx ? (size_t)n_blocks : 0};
            if (outputs_alias_inputs(x.w, x.g, g_dtype, x.v, n, outs, bytes, 4))
                return QUASAR_ERR_INVALID_ARG;
        }
        *T = LutTensor{x.w, x.g, x.v, x.r, x.codes, x.book, x.cand_idx, x.cols, n_blocks, 0};
        return QUASAR_OK;
    };
    static thread_local LutLaunch<kMaxBatch> Lp;
    int64_t total = 0;
    quasar_status st;
    for (int i = 0; i < n_tensors; ++i) {
        LutTensor T;
        if ((st = describe(tensors[i], &T)) != QUASAR_OK) return st;
        total += T.n_blocks;
    }
    if (total == 0) return QUASAR_OK;
    LutParams& p = Lp.p;
    p = LutParams{};
    p.g_kind = has_g ? (g_dtype == QUASAR_BF16 ? 2 : 1) : 0;
    p.r_bf16 = r_dtype == QUASAR_BF16;
    p.h_mode = opt.h_mode;
    p.codes_packed = opt.packed;
    p.n_clip = n_clip;
    p.beta2 = beta2;
    p.c1 = 1.0f - beta2;
    // summation depth of the per-index sums: 8 per packed half, the fold,
    // 8 per reader accumulator and two combining levels, plus margin
    p.tie_kappa = 24.0f * tuning().tie_scale;
    p.timeout_ns = kDefaultTimeoutNs;
    p.force_timeout_ns = (uint64_t)std::max<int64_t>(0, g_force_timeout_ns.load());
    p.stats = g_stats.load();
    fill_clip(clip, n_clip, p.f, p.invf);
    if ((st = status_ptr(&p.status)) != QUASAR_OK) return st;
    const int gbytes = p.g_kind == 2 ? 2 : (p.g_kind == 1 ? 4 : 0);
    const Launch L = plan((uint32_t)(kLutBlock * (8 + gbytes)), kLutScratchBytes);
    p.stages = L.stages;
    p.stage_bytes = L.stage_bytes;
    const cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    for (int i0 = 0; i0 < n_tensors; i0 += kMaxBatch) {
        Lp.n_t = std::min(kMaxBatch, n_tensors - i0);
        int64_t units = 0;
        for (int i = 0; i < Lp.n_t; ++i) {
            describe(tensors[i0 + i], &Lp.t[i]);
            Lp.t[i].unit0 = units;
            units += Lp.t[i].n_blocks;
        }
        Lp.n_units = units;
        if (units == 0) continue;
        if ((st = launch_persistent(lut_kernel(), &Lp, L.smem, units, s)) != QUASAR_OK) return st;
    }
    return QUASAR_OK;
}

quasar_status quasar_adamw_recon_nvfp4_batch(const quasar_adamw_nvfp4_tensor* tensors,
                                             int n_tensors, quasar_dtype g_dtype, float lr,
                                             float beta1, float beta2, float eps,
                                             float weight_decay, int64_t step, const float* clip,
                                             int n_clip, quasar_dtype r_dtype,
                                             const quasar_options* options, quasar_stream_t stream)
{
    Opts opt;
    if (read_options(options, &opt) != QUASAR_OK) return QUASAR_ERR_INVALID_ARG;
    if (opt.symmetric) return QUASAR_ERR_INVALID_ARG;  // an integer-code option
    if (n_tensors < 0 || (n_tensors > 0 && !tensors)) return QUASAR_ERR_INVALID_ARG;
    if (!(std::isfinite(lr) && lr >= 0.0f) || !(beta1 >= 0.0f && beta1 < 1.0f) ||
        !(std::isfinite(eps) && eps > 0.0f) ||
        !(std::isfinite(weight_decay) && weight_decay >= 0.0f) || step < 1 || !valid_dtype(g_dtype))
        return QUASAR_ERR_INVALID_ARG;
    if (n_tensors == 0) return QUASAR_OK;
    // one tensor: the reconstruction's checks (without a gradient: v is
    // updated by the AdamW pass), plus g and m present and w, g, m, v
    // pairwise disjoint
    auto describe = [&](const quasar_adamw_nvfp4_tensor& x, Nvfp4Tensor* T, AmaxItem* A,
                        AdamwItem* W) {
        quasar_status s1 = nvfp4_tensor(x.w, nullptr, g_dtype, x.v, beta2, clip, n_clip, x.rows,
                                        x.cols, nullptr, x.r, r_dtype, x.codes, x.block_scale,
                                        x.tensor_scale, x.cand_idx, T, A, opt.packed);
        if (s1 != QUASAR_OK) return s1;
        const int64_t n = x.rows * x.cols;
        *W = AdamwItem{x.w, x.g, x.m, x.v, n, x.tensor_scale};
        if (n == 0) return QUASAR_OK;
        if (!x.g || !x.m || !aligned16(x.g) || !aligned16(x.m)) return QUASAR_ERR_INVALID_ARG;
        const size_t nb = (size_t)n;
        const void* outs[] = {x.r, x.codes, x.block_scale, x.tensor_scale, x.cand_idx};
        const size_t bytes[] = {nb * dtype_size(r_dtype), x.codes ? (opt.packed ? nb / 2 : nb) : 0,
                                nb / 16, 4, x.cand_idx ? nb / 16 : 0};
        for (int i = 0; i < 5; ++i)
            if (overlaps(outs[i], bytes[i], x.m, nb * 4) ||
                overlaps(outs[i], bytes[i], x.g, nb * dtype_size(g_dtype)))
                return QUASAR_ERR_INVALID_ARG;
        const void* state[] = {x.w, x.g, x.m, x.v};
        const size_t sbytes[] = {nb * 4, nb * dtype_size(g_dtype), nb * 4, nb * 4};
        for (int i = 0; i < 4; ++i)
            for (int j = i + 1; j < 4; ++j)
                if (overlaps(state[i], sbytes[i], state[j], sbytes[j])) return QUASAR_ERR_INVALID_ARG;
        return QUASAR_OK;
    };
    static thread_local Nvfp4Launch<kMaxBatch> Lp;
    static thread_local AmaxBatch<kMaxBatch> B;
    static thread_local AdamwBatch<kMaxBatch> Ad;
    quasar_status st;
    for (int i = 0; i < n_tensors; ++i) {
        Nvfp4Tensor T;
        AmaxItem A;
        AdamwItem W;
        if ((st = describe(tensors[i], &T, &A, &W)) != QUASAR_OK) return st;
    }
    if ((st = nvfp4_params(false, g_dtype, beta2, clip, n_clip, r_dtype, &Lp.p, opt)) != QUASAR_OK)
        return st;
    {
        const double t = (double)step;
        AdamwHp& hp = Ad.hp;
        hp.g_kind = g_dtype == QUASAR_BF16 ? 2 : 1;
        hp.beta1 = beta1;
        hp.c1b = 1.0f - beta1;
        hp.beta2 = beta2;
        hp.c1 = 1.0f - beta2;
        hp.lr_wd = (float)((double)lr * (double)weight_decay);
        hp.step_size = (float)((double)lr / (1.0 - std::pow((double)beta1, t)));
        hp.isbc2 = (float)(1.0 / std::sqrt(1.0 - std::pow((double)beta2, t)));
        hp.eps = eps;
    }
    int dev = 0;
    const DeviceInfo* info = nullptr;
    if ((st = device_info(&dev, &info)) != QUASAR_OK) return st;
    const cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    for (int i0 = 0; i0 < n_tensors; i0 += kMaxBatch) {
        Lp.n_t = B.n_t = Ad.n_t = std::min(kMaxBatch, n_tensors - i0);
        int64_t nmax = 0;
        for (int i = 0; i < Lp.n_t; ++i) {
            describe(tensors[i0 + i], &Lp.t[i], &B.t[i], &Ad.t[i]);
            nmax = std::max(nmax, Ad.t[i].n);
        }
        if ((st = zero_amax_slots(B, true, s)) != QUASAR_OK) return st;
        if (nmax > 0) {
            const int64_t want = (nmax / 4 + kThreads - 1) / kThreads;
            const int64_t per = std::max<int64_t>(1, (int64_t)info->nsm * 8 / Ad.n_t);
            const int gx = (int)std::max<int64_t>(1, std::min<int64_t>(per, want));
            void* args[] = {(void*)&Ad};
            if (cudaLaunchKernel(adamw_amax_kernel(), dim3(gx, Ad.n_t), dim3(kThreads), args, 0, s) !=
                cudaSuccess)
                return QUASAR_ERR_CUDA;
        }
        if ((st = nvfp4_run(Lp, B, n_clip, s, true)) != QUASAR_OK) return st;
    }
    return QUASAR_OK;
}

quasar_status quasar_get_device_status(quasar_stream_t stream)
{
    if (cudaStreamSynchronize(reinterpret_cast<cudaStream_t>(stream)) != cudaSuccess)
        return QUASAR_ERR_CUDA;
    unsigned int word = 0;
    if (cudaMemcpyFromSymbol(&word, g_quasar_status_word, sizeof(word)) != cudaSuccess)
        return QUASAR_ERR_CUDA;
    if (word == 0) return QUASAR_OK;
    const unsigned int zero = 0;
    if (cudaMemcpyToSymbol(g_quasar_status_word, &zero, sizeof(zero)) != cudaSuccess)
        return QUASAR_ERR_CUDA;
    return (word & kStatusTimeout) ? QUASAR_ERR_TIMEOUT : QUASAR_OK;
}

void quasar_debug_force_timeout(int64_t nanoseconds) { g_force_timeout_ns.store(nanoseconds); }

void quasar_debug_set_stats(unsigned int* device_counters) { g_stats.store(device_counters); }

void quasar_debug_set_hoist(int enable) { g_hoist.store(enable ? 1 : 0); }

const char* quasar_status_string(quasar_status status)
{
    switch (status) {
    case QUASAR_OK: return "QUASAR_OK";
    case QUASAR_ERR_INVALID_ARG: return "QUASAR_ERR_INVALID_ARG";
    case QUASAR_ERR_UNSUPPORTED: return "QUASAR_ERR_UNSUPPORTED";
    case QUASAR_ERR_CUDA: return "QUASAR_ERR_CUDA";
    case QUASAR_ERR_TIMEOUT: return "QUASAR_ERR_TIMEOUT";
    default: return "QUASAR_ERR_UNKNOWN";
    }
}

int quasar_version(void) { return 100; }

}  // extern "C"
