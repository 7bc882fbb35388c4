// espace_api.cu -- the C ABI declared in include/espace.h: argument checks, handles and
// their device memory, the host side of calibration and projection building, and dispatch
// of the forward pass to the tcgen05 or the streaming kernels.
#include <cuda_runtime.h>
#include <math.h>
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include <algorithm>
#include <cmath>
#include <atomic>
#include <functional>
#include <mutex>
#include <string>
#include <vector>

#include "../../include/espace.h"
#include "kernels.h"

namespace espace {
int host_eigh(const double* A, int64_t n, double* w, double* V, int threads);
int host_eigh_select(const double* A, int64_t n, double* w,
                     const std::function<std::vector<int64_t>(const std::vector<double>&)>& order_sel,
                     std::vector<double>& V, int threads);
}

using namespace espace;

// ============================================================================ errors

namespace {

thread_local std::string g_last_error;

int fail(int code, const char* fmt, ...)
{
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof(buf), fmt, ap);
    va_end(ap);
    g_last_error = buf;
    return code;
}

int fail_cuda(cudaError_t e, const char* what)
{
    return fail(ESPACE_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

#define CUDA_TRY(expr, what)                        \
    do {                                            \
        cudaError_t _e = (expr);                    \
        if (_e != cudaSuccess) return fail_cuda(_e, what); \
    } while (0)

// As CUDA_TRY, running `cleanup` before returning the error.
#define CUDA_TRY_OR(expr, what, cleanup)            \
    do {                                            \
        cudaError_t _e = (expr);                    \
        if (_e != cudaSuccess) {                    \
            const int _rc = fail_cuda(_e, what);    \
            cleanup;                                \
            return _rc;                             \
        }                                           \
    } while (0)

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

std::atomic<uint64_t> g_wait_limit_ns{4000000000ull};
thread_local cudaEvent_t g_phase_event = nullptr;

// Makes `device` current for the lifetime of the guard.
struct DeviceGuard {
    int prev = -1;
    bool ok = true;
    explicit DeviceGuard(int device)
    {
        if (cudaGetDevice(&prev) != cudaSuccess) prev = -1;
        if (device >= 0 && device != prev) ok = cudaSetDevice(device) == cudaSuccess;
    }
    ~DeviceGuard()
    {
        int cur = -1;
        if (prev >= 0 && cudaGetDevice(&cur) == cudaSuccess && cur != prev) cudaSetDevice(prev);
    }
};

// bf16 bits of the value nearest to x, ties to even, in one rounding from fp64: x is first
// narrowed to fp32 with rounding to odd, which keeps the later fp32 -> bf16 rounding to
// nearest correct (Boldo & Melquiond, "Emulation of FMA and correctly rounded sums: proved
// algorithms using rounding to odd", IEEE TC 2008).
uint16_t bf16_from_double(double x)
{
    if (x != x) return 0x7fc0;
    float f = static_cast<float>(x);
    if (static_cast<double>(f) != x && !__builtin_isinf(f)) {
        // truncate towards zero, then force the last bit to one (round to odd)
        if (fabs(static_cast<double>(f)) > fabs(x)) f = nextafterf(f, 0.0f);
        uint32_t b;
        memcpy(&b, &f, 4);
        b |= 1u;
        memcpy(&f, &b, 4);
    }
    uint32_t b;
    memcpy(&b, &f, 4);
    if ((b & 0x7f800000u) == 0x7f800000u) return static_cast<uint16_t>(b >> 16);   // inf
    b += 0x7fffu + ((b >> 16) & 1u);
    return static_cast<uint16_t>(b >> 16);
}

int64_t round_up(int64_t v, int64_t m) { return (v + m - 1) / m * m; }

// The build's eigen-solve: all K eigenvalues of C (K x K, row-major) in the projection's
// order into w, and the first L eigenvectors in that order as the columns of P (K x L,
// row-major). The order is decreasing eigenvalue, or decreasing |eigenvalue| (ties keep the
// signed order) when by_magnitude is set or C is not positive semidefinite (smallest
// eigenvalue below -1e-6 of the largest magnitude), as the paper orders an indefinite C.
// Only those L eigenvectors are formed.
int principal_eigenvectors(const double* C, int64_t K, int64_t L, bool by_magnitude, std::vector<double>& w,
                           std::vector<double>& P)
{
    std::vector<double> desc(K);
    std::vector<int64_t> order;
    auto sel = [&](const std::vector<double>& wd) {
        order.resize(K);
        for (int64_t i = 0; i < K; ++i) order[i] = i;
        const double wmax = std::max(std::fabs(wd[0]), std::fabs(wd[K - 1]));
        if (by_magnitude || wd[K - 1] < -1e-6 * wmax)
            std::stable_sort(order.begin(), order.end(),
                             [&](int64_t a, int64_t b) { return std::fabs(wd[a]) > std::fabs(wd[b]); });
        return std::vector<int64_t>(order.begin(), order.begin() + L);
    };
    const int rc = host_eigh_select(C, K, desc.data(), sel, P, 0);
    if (rc != ESPACE_OK) return rc;
    w.resize(K);
    for (int64_t i = 0; i < K; ++i) w[i] = desc[order[i]];
    return ESPACE_OK;
}

}  // namespace

// ============================================================================ device state

namespace espace {

int device_info(DeviceInfo** out)
{
    static std::mutex mu;
    static std::vector<DeviceInfo*> infos;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return fail_cuda(e, "cudaGetDevice");
    std::lock_guard<std::mutex> lock(mu);
    if (dev >= static_cast<int>(infos.size())) infos.resize(dev + 1, nullptr);
    if (infos[dev] == nullptr) {
        DeviceInfo* d = new DeviceInfo();
        d->device = dev;
        e = cudaDeviceGetAttribute(&d->num_sms, cudaDevAttrMultiProcessorCount, dev);
        if (e != cudaSuccess) {
            delete d;
            return fail_cuda(e, "cudaDeviceGetAttribute");
        }
        int major = 0, minor = 0;
        cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
        if (major != 10 || minor != 3) {
            delete d;
            return fail(ESPACE_ERR_STATE,
                        "device %d is sm_%d%d; this library is built for sm_103a only", dev,
                        major, minor);
        }
        e = cudaMalloc(&d->status, sizeof(int));
        if (e != cudaSuccess) {
            delete d;
            return fail_cuda(e, "cudaMalloc(status)");
        }
        e = cudaMemset(d->status, 0, sizeof(int));
        if (e != cudaSuccess) {
            cudaFree(d->status);
            delete d;
            return fail_cuda(e, "cudaMemset(status)");
        }
        infos[dev] = d;
    }
    *out = infos[dev];
    return ESPACE_OK;
}

uint64_t wait_limit_ns() { return g_wait_limit_ns.load(std::memory_order_relaxed); }

}  // namespace espace

// ============================================================================ handles

struct espace_calib_s {
    int64_t K = 0;
    int device = 0;
    float* S = nullptr;            // [K][K] fp32, upper triangle valid
    int* sched = nullptr;          // the SYRK's wave and exit counters (zeroed; left zero)
    int64_t n = 0;
    int mode = 0;                  // 0 unset, 1 plain, 2 normalized (Cor. 1), 3 NL-MSE (Thm. 2),
                                   // 4 NL-MSE with L2-normalized tokens and gradients
    void* xn = nullptr;            // scratch for normalized tokens
    int64_t xn_tokens = 0;
    void* gn = nullptr;            // scratch for normalized gradients (NL-MSE)
    int64_t gn_tokens = 0;
    float* nl_f32 = nullptr;       // NL-MSE scratch: two K x K fp32 autocorrelations
    void* nl_bf = nullptr;         //   and four bf16 halves (hi / lo of each), Kp x K, zero rows past K
};

struct espace_proj_s {
    int64_t K = 0, M = 0, L = 0, Lp = 0;
    int device = 0;
    uint16_t* PT = nullptr;        // [Lp][K] bf16, rows >= L zero
    uint16_t* WfT = nullptr;       // [M][Lp] bf16, columns >= L zero
    std::vector<double> evals;     // K eigenvalues, decreasing (if calibrated)
    uint16_t* Z = nullptr;         // [zcap][Lp] bf16 scratch for the rank-L intermediate
    int64_t zcap = 0;
    unsigned int* bar = nullptr;   // grid barrier counter of the decode kernel (zeroed)
    int* ready = nullptr;          // fused forward: ceil(zcap / 256) readiness counters, ticket, exit counter (zeroed)
    float* part = nullptr;         // split reductions of the few-token products (fp32)
    int64_t part_cap = 0;
    // tensor-parallel layer (tp_kind != 0): Lp = tp * L is the width of Z. COLUMN: PT is
    // [tp L][K] (rank r's P_r^T in rows r L ..), WfT is [M][L] (rank r's W'_r^T in rows
    // r M/tp ..). ROW: PT is [tp L][K/tp], WfT is [M][tp L] (rank r's in columns r L ..).
    int tp = 1;
    int tp_kind = 0;
    // host-buffer forward: device staging of X and Y, copy streams and per-chunk events
    uint16_t* hx = nullptr;
    uint16_t* hy = nullptr;
    int64_t h_cap = 0;
    cudaStream_t s_in = nullptr, s_out = nullptr;
    cudaEvent_t ev[2 * 16 + 2] = {};
    // training view: backward scratch, grown on demand
    uint16_t* dz = nullptr;        // [dz_cap][Lp] bf16: dY W'^T
    int64_t dz_cap = 0;
    float* dwp32 = nullptr;        // [Lp][M] fp32: Z^T dY
    uint16_t* dwp16 = nullptr;     // [Lp][M] bf16
    std::mutex mu;                 // guards scratch growth
};

// A device allocation freed when it goes out of scope.
struct DevBuf {
    void* ptr = nullptr;
    ~DevBuf()
    {
        if (ptr) cudaFree(ptr);
    }
    template <typename T>
    T* as() const
    {
        return static_cast<T*>(ptr);
    }
};

extern "C" {

int espace_version(void) { return 100; }

const char* espace_last_error(void) { return g_last_error.c_str(); }

int espace_set_phase_event(void* event)
{
    g_phase_event = static_cast<cudaEvent_t>(event);
    return ESPACE_OK;
}

int espace_set_wait_limit_ns(uint64_t ns)
{
    g_wait_limit_ns.store(ns == 0 ? 4000000000ull : ns);
    return ESPACE_OK;
}

int espace_host_eigh(const double* A_host, int64_t K, double* w, double* V, int threads)
{
    if (A_host == nullptr || w == nullptr) return fail(ESPACE_ERR_ARG, "espace_host_eigh: null pointer");
    if (K < 1 || K > 65536) return fail(ESPACE_ERR_SHAPE, "espace_host_eigh: K=%lld out of range", (long long)K);
    const int rc = host_eigh(A_host, K, w, V, threads);
    if (rc != ESPACE_OK) return fail(rc, "espace_host_eigh: QR iteration did not converge");
    return ESPACE_OK;
}

// ---------------------------------------------------------------------------- calibration

int espace_calib_create(int64_t K, espace_calib_t* out)
{
    if (out == nullptr) return fail(ESPACE_ERR_ARG, "espace_calib_create: out is null");
    *out = nullptr;
    if (K < 8 || K > 65536 || K % 8 != 0)
        return fail(ESPACE_ERR_SHAPE, "espace_calib_create: K=%lld must be a multiple of 8 in [8, 65536]", (long long)K);
    DeviceInfo* dev = nullptr;
    int rc = device_info(&dev);
    if (rc != ESPACE_OK) return rc;
    espace_calib_s* h = new espace_calib_s();
    h->K = K;
    h->device = dev->device;
    cudaError_t e = cudaMalloc(&h->S, sizeof(float) * K * K);
    if (e != cudaSuccess) {
        delete h;
        return fail(ESPACE_ERR_NOMEM, "espace_calib_create: cudaMalloc of %lld bytes: %s",
                    (long long)(sizeof(float) * K * K), cudaGetErrorString(e));
    }
    e = cudaMemset(h->S, 0, sizeof(float) * K * K);
    if (e == cudaSuccess) e = cudaMalloc(&h->sched, 64);
    if (e == cudaSuccess) e = cudaMemset(h->sched, 0, 64);
    if (e != cudaSuccess) {
        cudaFree(h->S);
        if (h->sched) cudaFree(h->sched);
        delete h;
        return fail_cuda(e, "espace_calib_create: scratch");
    }
    *out = h;
    return ESPACE_OK;
}

static int calib_accumulate_impl(espace_calib_t h, const void* X, int64_t N, void* stream,
                                 int mode)
{
    if (h == nullptr) return fail(ESPACE_ERR_ARG, "calib_accumulate: null handle");
    if (N < 0) return fail(ESPACE_ERR_SHAPE, "calib_accumulate: N=%lld < 0", (long long)N);
    if (N == 0) return ESPACE_OK;
    if (X == nullptr) return fail(ESPACE_ERR_ARG, "calib_accumulate: X is null");
    if (!aligned16(X)) return fail(ESPACE_ERR_ALIGN, "calib_accumulate: X not 16-byte aligned");
    if (N > (int64_t(1) << 31) - 64) return fail(ESPACE_ERR_SHAPE, "calib_accumulate: N=%lld too large for one call", (long long)N);
    if (h->mode != 0 && h->mode != mode)
        return fail(ESPACE_ERR_STATE, "calib_accumulate: plain and normalized accumulation mixed on one handle");
    DeviceGuard g(h->device);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const void* src = X;
    if (mode == 2) {
        if (h->xn_tokens < N) {
            CUDA_TRY(cudaStreamSynchronize(st), "calib_accumulate_normalized: sync");
            if (h->xn) cudaFree(h->xn);
            h->xn = nullptr;
            h->xn_tokens = 0;
            cudaError_t e = cudaMalloc(&h->xn, sizeof(uint16_t) * N * h->K);
            if (e != cudaSuccess) return fail(ESPACE_ERR_NOMEM, "calib_accumulate_normalized: scratch: %s", cudaGetErrorString(e));
            h->xn_tokens = N;
        }
        CUDA_TRY(launch_normalize_rows(X, N, static_cast<int>(h->K), h->xn, st), "normalize_rows launch");
        src = h->xn;
    }
    CUDA_TRY(launch_syrk_upper(src, N, static_cast<int>(h->K), h->S, st, h->sched), "syrk launch");
    h->mode = mode;
    h->n += N;
    return ESPACE_OK;
}

int espace_calib_accumulate(espace_calib_t h, const void* X_dev, int64_t N, void* stream)
{
    return calib_accumulate_impl(h, X_dev, N, stream, 1);
}

int espace_calib_accumulate_normalized(espace_calib_t h, const void* X_dev, int64_t N, void* stream)
{
    return calib_accumulate_impl(h, X_dev, N, stream, 2);
}

// Grows a bf16 token scratch of the calibration handle to `tokens` rows (synchronously).
static int grow_token_scratch(espace_calib_t h, void** buf, int64_t* cap, int64_t tokens, cudaStream_t st)
{
    if (*cap >= tokens) return ESPACE_OK;
    CUDA_TRY(cudaStreamSynchronize(st), "calibration scratch: sync");
    if (*buf) cudaFree(*buf);
    *buf = nullptr;
    *cap = 0;
    cudaError_t e = cudaMalloc(buf, sizeof(uint16_t) * tokens * h->K);
    if (e != cudaSuccess) return fail(ESPACE_ERR_NOMEM, "calibration scratch: %s", cudaGetErrorString(e));
    *cap = tokens;
    return ESPACE_OK;
}

int espace_calib_accumulate_nl(espace_calib_t h, const void* X_dev, const void* G_dev, int64_t T, int normalized,
                               void* stream)
{
    if (h == nullptr) return fail(ESPACE_ERR_ARG, "espace_calib_accumulate_nl: null handle");
    if (X_dev == nullptr || G_dev == nullptr) return fail(ESPACE_ERR_ARG, "espace_calib_accumulate_nl: null pointer");
    if (T < 1 || T > (int64_t(1) << 31) - 64)
        return fail(ESPACE_ERR_SHAPE, "espace_calib_accumulate_nl: T=%lld tokens", (long long)T);
    if (!aligned16(X_dev) || !aligned16(G_dev))
        return fail(ESPACE_ERR_ALIGN, "espace_calib_accumulate_nl: X / G not 16-byte aligned");
    const int mode = normalized ? 4 : 3;
    if (h->mode != 0 && h->mode != mode)
        return fail(ESPACE_ERR_STATE, "espace_calib_accumulate_nl: mixed with another accumulation on one handle");
    DeviceGuard g(h->device);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const int64_t K = h->K, kk = K * K;
    if (normalized) {
        // the L2-normalized variant: x / |x| and g / |g| for every token (Sec. 3.3)
        int rc = grow_token_scratch(h, &h->xn, &h->xn_tokens, T, st);
        if (rc == ESPACE_OK) rc = grow_token_scratch(h, &h->gn, &h->gn_tokens, T, st);
        if (rc != ESPACE_OK) return rc;
        CUDA_TRY(launch_normalize_rows(X_dev, T, static_cast<int>(K), h->xn, st), "accumulate_nl: normalize X");
        CUDA_TRY(launch_normalize_rows(G_dev, T, static_cast<int>(K), h->gn, st), "accumulate_nl: normalize G");
        X_dev = h->xn;
        G_dev = h->gn;
    }
    // the bf16 halves of A and B as four blocks of Kp = ceil(K / 64) * 64 rows; the rows past
    // K stay zero, so that every block is a whole number of 64-row k-blocks
    const int64_t Kp = (K + 63) / 64 * 64, blk = Kp * K;
    if (h->nl_f32 == nullptr) {
        cudaError_t e = cudaMalloc(&h->nl_f32, sizeof(float) * 2 * kk);
        if (e == cudaSuccess) e = cudaMalloc(&h->nl_bf, sizeof(uint16_t) * 4 * blk);
        if (e == cudaSuccess) e = cudaMemsetAsync(h->nl_bf, 0, sizeof(uint16_t) * 4 * blk, st);
        if (e != cudaSuccess) {
            if (h->nl_f32) cudaFree(h->nl_f32);
            if (h->nl_bf) cudaFree(h->nl_bf);
            h->nl_f32 = nullptr;
            h->nl_bf = nullptr;
            return fail(ESPACE_ERR_NOMEM, "espace_calib_accumulate_nl: scratch: %s", cudaGetErrorString(e));
        }
    }
    float* a32 = h->nl_f32;
    float* b32 = h->nl_f32 + kk;
    uint16_t* a_hi = static_cast<uint16_t*>(h->nl_bf);
    uint16_t* a_lo = a_hi + blk;
    uint16_t* b_hi = a_lo + blk;
    uint16_t* b_lo = b_hi + blk;
    const int k = static_cast<int>(K);
    // A = X^T X / T and B = G^T G / T (upper triangles on the tensor cores, then the full
    // symmetric matrices split into bf16 hi + lo)
    CUDA_TRY(launch_syrk_upper_two(X_dev, G_dev, T, k, a32, b32, true, st), "accumulate_nl: X^T X and G^T G");
    CUDA_TRY(launch_sym_split_bf16(a32, K, 1.0f / static_cast<float>(T), a_hi, a_lo, st), "accumulate_nl: split A");
    CUDA_TRY(launch_sym_split_bf16(b32, K, 1.0f / static_cast<float>(T), b_hi, b_lo, st), "accumulate_nl: split B");
    // S += (A B + B A), upper triangle: A B ~ A_hi B_hi + A_hi B_lo + A_lo B_hi and the same
    // for B A; A and B are symmetric, so S += U^T V with U, V one of them each is S += U V,
    // and the six products are one reduction over six K-row segments of the four blocks
    const int r = static_cast<int>(Kp);
    const int seg_u[6] = {0, 0, r, 2 * r, 2 * r, 3 * r};       // A_hi A_hi A_lo B_hi B_hi B_lo
    const int seg_v[6] = {2 * r, 3 * r, 2 * r, 0, r, 0};       // B_hi B_lo B_hi A_hi A_lo A_hi
    CUDA_TRY(launch_syrk_segments_upper(h->nl_bf, 4 * Kp, k, r, 6, seg_u, seg_v, h->S, st), "accumulate_nl: products");
    h->mode = mode;
    h->n += 1;
    return ESPACE_OK;
}

static int read_sum(espace_calib_t h, std::vector<float>& S, void* stream)
{
    DeviceGuard g(h->device);
    CUDA_TRY(cudaStreamSynchronize(static_cast<cudaStream_t>(stream)), "calib read: sync");
    S.resize(static_cast<size_t>(h->K * h->K));
    CUDA_TRY(cudaMemcpy(S.data(), h->S, sizeof(float) * S.size(), cudaMemcpyDeviceToHost), "calib read: copy");
    return ESPACE_OK;
}

static void mirror_scaled(const std::vector<float>& S, int64_t K, double scale, double* C)
{
    for (int64_t i = 0; i < K; ++i)
        for (int64_t j = 0; j < K; ++j) {
            const int64_t a = std::min(i, j), b = std::max(i, j);
            C[i * K + j] = static_cast<double>(S[a * K + b]) * scale;
        }
}

int espace_calib_read(espace_calib_t h, double* C_host, int64_t* n_out, void* stream)
{
    if (h == nullptr) return fail(ESPACE_ERR_ARG, "espace_calib_read: null handle");
    if (n_out) *n_out = h->n;
    if (C_host == nullptr) {
        DeviceGuard g(h->device);
        CUDA_TRY(cudaStreamSynchronize(static_cast<cudaStream_t>(stream)), "calib read: sync");
        return ESPACE_OK;
    }
    if (h->n == 0) return fail(ESPACE_ERR_STATE, "espace_calib_read: no tokens accumulated");
    std::vector<float> S;
    int rc = read_sum(h, S, stream);
    if (rc != ESPACE_OK) return rc;
    mirror_scaled(S, h->K, 1.0 / static_cast<double>(h->n), C_host);
    return ESPACE_OK;
}

int espace_calib_export(espace_calib_t h, float* S_host, int64_t* n_out, void* stream)
{
    if (h == nullptr || S_host == nullptr) return fail(ESPACE_ERR_ARG, "espace_calib_export: null pointer");
    std::vector<float> S;
    int rc = read_sum(h, S, stream);
    if (rc != ESPACE_OK) return rc;
    memcpy(S_host, S.data(), sizeof(float) * S.size());
    if (n_out) *n_out = h->n;
    return ESPACE_OK;
}

int espace_calib_import(espace_calib_t h, const float* S_host, int64_t n, void* stream)
{
    if (h == nullptr || S_host == nullptr) return fail(ESPACE_ERR_ARG, "espace_calib_import: null pointer");
    if (n < 0) return fail(ESPACE_ERR_ARG, "espace_calib_import: n < 0");
    DeviceGuard g(h->device);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    CUDA_TRY(cudaStreamSynchronize(st), "calib import: sync");
    CUDA_TRY(cudaMemcpy(h->S, S_host, sizeof(float) * h->K * h->K, cudaMemcpyHostToDevice), "calib import: copy");
    h->n = n;
    return ESPACE_OK;
}

int espace_calib_reset(espace_calib_t h, void* stream)
{
    if (h == nullptr) return fail(ESPACE_ERR_ARG, "espace_calib_reset: null handle");
    DeviceGuard g(h->device);
    CUDA_TRY(launch_zero_f32(h->S, h->K * h->K, static_cast<cudaStream_t>(stream)), "calib reset");
    h->n = 0;
    h->mode = 0;
    return ESPACE_OK;
}

void espace_calib_destroy(espace_calib_t h)
{
    if (h == nullptr) return;
    DeviceGuard g(h->device);
    cudaDeviceSynchronize();
    if (h->S) cudaFree(h->S);
    if (h->sched) cudaFree(h->sched);
    if (h->xn) cudaFree(h->xn);
    if (h->nl_f32) cudaFree(h->nl_f32);
    if (h->nl_bf) cudaFree(h->nl_bf);
    if (h->gn) cudaFree(h->gn);
    delete h;
}

// ---------------------------------------------------------------------------- projection

static int proj_create(int64_t K, int64_t M, int64_t L, espace_proj_s** out)
{
    DeviceInfo* dev = nullptr;
    int rc = device_info(&dev);
    if (rc != ESPACE_OK) return rc;
    espace_proj_s* p = new espace_proj_s();
    p->K = K;
    p->M = M;
    p->L = L;
    p->Lp = round_up(L, 64);
    p->device = dev->device;
    cudaError_t e = cudaMalloc(&p->PT, sizeof(uint16_t) * p->Lp * K);
    if (e == cudaSuccess) e = cudaMalloc(&p->WfT, sizeof(uint16_t) * M * p->Lp);
    if (e == cudaSuccess) e = cudaMalloc(&p->bar, 64);
    if (e == cudaSuccess) e = cudaMemset(p->bar, 0, 64);
    if (e != cudaSuccess) {
        if (p->PT) cudaFree(p->PT);
        if (p->WfT) cudaFree(p->WfT);
        if (p->bar) cudaFree(p->bar);
        delete p;
        return fail(ESPACE_ERR_NOMEM, "projection: cudaMalloc: %s", cudaGetErrorString(e));
    }
    *out = p;
    return ESPACE_OK;
}

static int check_proj_shape(int64_t K, int64_t M, int64_t L)
{
    if (K < 8 || K % 8 != 0 || K > 65536)
        return fail(ESPACE_ERR_SHAPE, "K=%lld must be a multiple of 8 in [8, 65536]", (long long)K);
    if (M < 8 || M % 8 != 0 || M > (int64_t(1) << 30))
        return fail(ESPACE_ERR_SHAPE, "M=%lld must be a positive multiple of 8", (long long)M);
    if (L < 1 || L > K) return fail(ESPACE_ERR_SHAPE, "L=%lld must be in [1, K=%lld]", (long long)L, (long long)K);
    return ESPACE_OK;
}

// Uploads P (fp64 [K][L] row-major) as bf16 P^T [Lp][K] and folds W'^T = W P on the GPU.
static int proj_upload_and_fold(espace_proj_s* p, const double* P, const void* W, cudaStream_t st)
{
    const int64_t K = p->K, L = p->L, Lp = p->Lp;
    std::vector<uint16_t> pt(static_cast<size_t>(Lp * K), 0);
    for (int64_t l = 0; l < L; ++l)
        for (int64_t k = 0; k < K; ++k) pt[l * K + k] = bf16_from_double(P[k * L + l]);
    CUDA_TRY(cudaStreamSynchronize(st), "projection: sync");
    CUDA_TRY(cudaMemcpy(p->PT, pt.data(), sizeof(uint16_t) * pt.size(), cudaMemcpyHostToDevice), "projection: upload P");
    CUDA_TRY(launch_gemm_tn(W, K, p->PT, K, static_cast<int>(p->M), static_cast<int>(Lp),
                            static_cast<int>(K), p->WfT, Lp, st),
             "projection: fold launch");
    CUDA_TRY(cudaStreamSynchronize(st), "projection: fold");
    return ESPACE_OK;
}

int espace_proj_from_host(int64_t K, int64_t M, int64_t L, const double* P_host, const void* W_dev,
                          void* stream, espace_proj_t* out)
{
    if (out == nullptr || P_host == nullptr || W_dev == nullptr)
        return fail(ESPACE_ERR_ARG, "espace_proj_from_host: null pointer");
    *out = nullptr;
    int rc = check_proj_shape(K, M, L);
    if (rc != ESPACE_OK) return rc;
    if (!aligned16(W_dev)) return fail(ESPACE_ERR_ALIGN, "espace_proj_from_host: W not 16-byte aligned");
    espace_proj_s* p = nullptr;
    rc = proj_create(K, M, L, &p);
    if (rc != ESPACE_OK) return rc;
    rc = proj_upload_and_fold(p, P_host, W_dev, static_cast<cudaStream_t>(stream));
    if (rc != ESPACE_OK) {
        espace_proj_destroy(p);
        return rc;
    }
    *out = p;
    return ESPACE_OK;
}

int espace_build_projection_go(espace_calib_t h, const void* W_dev, int64_t M, int64_t L, void* stream,
                               espace_proj_t* out)
{
    if (out == nullptr || h == nullptr || W_dev == nullptr)
        return fail(ESPACE_ERR_ARG, "espace_build_projection_go: null pointer");
    *out = nullptr;
    const int64_t K = h->K;
    int rc = check_proj_shape(K, M, L);
    if (rc != ESPACE_OK) return rc;
    if (!aligned16(W_dev)) return fail(ESPACE_ERR_ALIGN, "espace_build_projection_go: W not 16-byte aligned");
    if (h->n == 0) return fail(ESPACE_ERR_STATE, "espace_build_projection_go: no calibration tokens");
    if (h->mode > 2) return fail(ESPACE_ERR_STATE, "espace_build_projection_go: needs an activation autocorrelation");
    DeviceGuard g(h->device);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const size_t kk = static_cast<size_t>(K * K);
    DevBuf cw_upper, cx, cw, t;
    cudaError_t e = cudaMalloc(&cw_upper.ptr, sizeof(float) * kk);
    if (e == cudaSuccess) e = cudaMalloc(&cx.ptr, sizeof(double) * kk);
    if (e == cudaSuccess) e = cudaMalloc(&cw.ptr, sizeof(double) * kk);
    if (e == cudaSuccess) e = cudaMalloc(&t.ptr, sizeof(double) * kk);
    if (e != cudaSuccess) return fail(ESPACE_ERR_NOMEM, "espace_build_projection_go: %s", cudaGetErrorString(e));
    // C_W = W^T W / M: the calibration SYRK with the M weight rows as its tokens
    CUDA_TRY(launch_zero_f32(cw_upper.as<float>(), static_cast<int64_t>(kk), st), "build_projection_go: clear");
    CUDA_TRY(launch_syrk_upper(W_dev, M, static_cast<int>(K), cw_upper.as<float>(), st), "build_projection_go: C_W");
    CUDA_TRY(launch_sym_full_f64(h->S, K, 1.0 / static_cast<double>(h->n), cx.as<double>(), st),
             "build_projection_go: C_X");
    CUDA_TRY(launch_sym_full_f64(cw_upper.as<float>(), K, 1.0 / static_cast<double>(M), cw.as<double>(), st),
             "build_projection_go: C_W full");
    // T = C_X C_W in fp64; C = T + T^T = C_X C_W + C_W C_X (both factors symmetric)
    CUDA_TRY(launch_gemm_f64(cx.as<double>(), cw.as<double>(), static_cast<int>(K), t.as<double>(), st),
             "build_projection_go: product");
    std::vector<double> T(kk), C(kk), wo, P;
    CUDA_TRY(cudaStreamSynchronize(st), "build_projection_go: sync");
    CUDA_TRY(cudaMemcpy(T.data(), t.ptr, sizeof(double) * kk, cudaMemcpyDeviceToHost), "build_projection_go: read");
    for (int64_t i = 0; i < K; ++i)
        for (int64_t j = 0; j < K; ++j) C[i * K + j] = T[i * K + j] + T[j * K + i];
    // C may be indefinite: order by |eigenvalue|, largest first (ties keep the signed order)
    rc = principal_eigenvectors(C.data(), K, L, true, wo, P);
    if (rc != ESPACE_OK) return fail(rc, "espace_build_projection_go: eigen-solver did not converge");
    espace_proj_s* p = nullptr;
    rc = proj_create(K, M, L, &p);
    if (rc != ESPACE_OK) return rc;
    p->evals = wo;
    rc = proj_upload_and_fold(p, P.data(), W_dev, st);
    if (rc != ESPACE_OK) {
        espace_proj_destroy(p);
        return rc;
    }
    *out = p;
    return ESPACE_OK;
}

int espace_proj_from_device(int64_t K, int64_t M, int64_t L, const void* PT_dev, const void* W_dev, void* stream,
                            espace_proj_t* out)
{
    if (out == nullptr || PT_dev == nullptr || W_dev == nullptr)
        return fail(ESPACE_ERR_ARG, "espace_proj_from_device: null pointer");
    *out = nullptr;
    int rc = check_proj_shape(K, M, L);
    if (rc != ESPACE_OK) return rc;
    if (!aligned16(W_dev) || !aligned16(PT_dev))
        return fail(ESPACE_ERR_ALIGN, "espace_proj_from_device: P^T and W must be 16-byte aligned");
    espace_proj_s* p = nullptr;
    rc = proj_create(K, M, L, &p);
    if (rc != ESPACE_OK) return rc;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    // rows L .. Lp-1 of the handle's P^T are zero
    CUDA_TRY_OR(cudaMemcpyAsync(p->PT, PT_dev, sizeof(uint16_t) * L * K, cudaMemcpyDeviceToDevice, st),
                "espace_proj_from_device: copy P^T", espace_proj_destroy(p));
    if (p->Lp > L)
        CUDA_TRY_OR(cudaMemsetAsync(p->PT + L * K, 0, sizeof(uint16_t) * (p->Lp - L) * K, st),
                    "espace_proj_from_device: clear padding", espace_proj_destroy(p));
    CUDA_TRY_OR(launch_gemm_tn(W_dev, K, p->PT, K, static_cast<int>(M), static_cast<int>(p->Lp), static_cast<int>(K),
                               p->WfT, p->Lp, st),
                "espace_proj_from_device: fold launch", espace_proj_destroy(p));
    CUDA_TRY_OR(cudaStreamSynchronize(st), "espace_proj_from_device: fold", espace_proj_destroy(p));
    *out = p;
    return ESPACE_OK;
}

int espace_build_projection(espace_calib_t h, const void* W_dev, int64_t M, int64_t L, void* stream,
                            espace_proj_t* out)
{
    if (out == nullptr || h == nullptr || W_dev == nullptr)
        return fail(ESPACE_ERR_ARG, "espace_build_projection: null pointer");
    *out = nullptr;
    const int64_t K = h->K;
    int rc = check_proj_shape(K, M, L);
    if (rc != ESPACE_OK) return rc;
    if (!aligned16(W_dev)) return fail(ESPACE_ERR_ALIGN, "espace_build_projection: W not 16-byte aligned");
    if (h->n == 0) return fail(ESPACE_ERR_STATE, "espace_build_projection: no calibration tokens");
    DeviceGuard g(h->device);
    std::vector<float> S;
    rc = read_sum(h, S, stream);
    if (rc != ESPACE_OK) return rc;
    std::vector<double> C(static_cast<size_t>(K * K)), w, P;
    mirror_scaled(S, K, 1.0 / static_cast<double>(h->n), C.data());
    // decreasing eigenvalues; when C is not positive semidefinite (e.g. an NL-MSE matrix),
    // decreasing |eigenvalue| instead, as the paper does
    rc = principal_eigenvectors(C.data(), K, L, false, w, P);
    if (rc != ESPACE_OK) return fail(rc, "espace_build_projection: eigen-solver did not converge");
    espace_proj_s* p = nullptr;
    rc = proj_create(K, M, L, &p);
    if (rc != ESPACE_OK) return rc;
    p->evals = w;
    rc = proj_upload_and_fold(p, P.data(), W_dev, static_cast<cudaStream_t>(stream));
    if (rc != ESPACE_OK) {
        espace_proj_destroy(p);
        return rc;
    }
    *out = p;
    return ESPACE_OK;
}

// ---------------------------------------------------------------------------- tensor parallel

static int check_tp_shape(int kind, int tp, int64_t K, int64_t M, int64_t L)
{
    if (kind != ESPACE_TP_COLUMN && kind != ESPACE_TP_ROW) return fail(ESPACE_ERR_ARG, "tensor parallel: unknown kind %d", kind);
    if (tp < 1 || tp > 8) return fail(ESPACE_ERR_SHAPE, "tensor parallel: tp=%d must be in [1, 8]", tp);
    if (K < 8 || K % 8 != 0 || K > 65536) return fail(ESPACE_ERR_SHAPE, "tensor parallel: K=%lld", (long long)K);
    if (M < 8 || M % 8 != 0 || M > (int64_t(1) << 30)) return fail(ESPACE_ERR_SHAPE, "tensor parallel: M=%lld", (long long)M);
    if (L < 64 || L % 64 != 0) return fail(ESPACE_ERR_SHAPE, "tensor parallel: L=%lld must be a positive multiple of 64", (long long)L);
    if (kind == ESPACE_TP_COLUMN) {
        if (M % tp != 0 || (M / tp) % 8 != 0)
            return fail(ESPACE_ERR_SHAPE, "tensor parallel: M/tp must be a multiple of 8 (M=%lld, tp=%d)", (long long)M, tp);
        if (L > K) return fail(ESPACE_ERR_SHAPE, "tensor parallel: L=%lld > K=%lld", (long long)L, (long long)K);
    } else {
        if (K % tp != 0 || (K / tp) % 64 != 0)
            return fail(ESPACE_ERR_SHAPE, "tensor parallel: K/tp must be a multiple of 64 (K=%lld, tp=%d)", (long long)K, tp);
        if (L > K / tp) return fail(ESPACE_ERR_SHAPE, "tensor parallel: L=%lld > K/tp=%lld", (long long)L, (long long)(K / tp));
    }
    return ESPACE_OK;
}

// Allocates a tensor-parallel handle, uploads the tp projections (fp64 [tp][Kr][L]) as bf16
// P^T blocks and folds each rank's W'_r on the GPU.
static int tp_create_and_fold(int kind, int tp, int64_t K, int64_t M, int64_t L, const double* P, const void* W,
                              cudaStream_t st, espace_proj_s** out)
{
    DeviceInfo* dev = nullptr;
    int rc = device_info(&dev);
    if (rc != ESPACE_OK) return rc;
    const int64_t Kr = kind == ESPACE_TP_COLUMN ? K : K / tp, Mr = kind == ESPACE_TP_COLUMN ? M / tp : M;
    espace_proj_s* p = new espace_proj_s();
    p->K = K;
    p->M = M;
    p->L = L;
    p->Lp = tp * L;
    p->tp = tp;
    p->tp_kind = kind;
    p->device = dev->device;
    cudaError_t e = cudaMalloc(&p->PT, sizeof(uint16_t) * tp * L * Kr);
    if (e == cudaSuccess) e = cudaMalloc(&p->WfT, sizeof(uint16_t) * M * (kind == ESPACE_TP_COLUMN ? L : tp * L));
    if (e == cudaSuccess) e = cudaMalloc(&p->bar, 64);
    if (e == cudaSuccess) e = cudaMemset(p->bar, 0, 64);
    if (e != cudaSuccess) {
        espace_proj_destroy(p);
        return fail(ESPACE_ERR_NOMEM, "tensor parallel: cudaMalloc: %s", cudaGetErrorString(e));
    }
    std::vector<uint16_t> pt(static_cast<size_t>(tp * L * Kr));
    for (int r = 0; r < tp; ++r)
        for (int64_t l = 0; l < L; ++l)
            for (int64_t k = 0; k < Kr; ++k)
                pt[(r * L + l) * Kr + k] = bf16_from_double(P[(r * Kr + k) * L + l]);
    CUDA_TRY_OR(cudaStreamSynchronize(st), "tensor parallel: sync", espace_proj_destroy(p));
    CUDA_TRY_OR(cudaMemcpy(p->PT, pt.data(), sizeof(uint16_t) * pt.size(), cudaMemcpyHostToDevice),
                "tensor parallel: upload P", espace_proj_destroy(p));
    const uint16_t* Wb = static_cast<const uint16_t*>(W);
    for (int r = 0; r < tp; ++r) {
        cudaError_t f;
        if (kind == ESPACE_TP_COLUMN)   // W'_r^T [M/tp][L] = W_r [M/tp][K] P_r
            f = launch_gemm_tn(Wb + r * Mr * K, K, p->PT + r * L * K, K, static_cast<int>(Mr), static_cast<int>(L),
                               static_cast<int>(K), p->WfT + r * Mr * L, L, st);
        else                            // W'_r^T [M][L] = W[:, r K/tp ..] P_r, columns r L .. of WfT
            f = launch_gemm_tn(Wb + r * Kr, K, p->PT + r * L * Kr, Kr, static_cast<int>(M), static_cast<int>(L),
                               static_cast<int>(Kr), p->WfT + r * L, tp * L, st);
        CUDA_TRY_OR(f, "tensor parallel: fold launch", espace_proj_destroy(p));
    }
    CUDA_TRY_OR(cudaStreamSynchronize(st), "tensor parallel: fold", espace_proj_destroy(p));
    *out = p;
    return ESPACE_OK;
}

int espace_proj_tp_from_host(int kind, int tp, int64_t K, int64_t M, int64_t L, const double* P_host,
                             const void* W_dev, void* stream, espace_proj_t* out)
{
    if (out == nullptr || P_host == nullptr || W_dev == nullptr)
        return fail(ESPACE_ERR_ARG, "espace_proj_tp_from_host: null pointer");
    *out = nullptr;
    int rc = check_tp_shape(kind, tp, K, M, L);
    if (rc != ESPACE_OK) return rc;
    if (!aligned16(W_dev)) return fail(ESPACE_ERR_ALIGN, "espace_proj_tp_from_host: W not 16-byte aligned");
    espace_proj_s* p = nullptr;
    rc = tp_create_and_fold(kind, tp, K, M, L, P_host, W_dev, static_cast<cudaStream_t>(stream), &p);
    if (rc != ESPACE_OK) return rc;
    *out = p;
    return ESPACE_OK;
}

int espace_build_projection_tp(espace_calib_t h, const void* W_dev, int64_t M, int64_t L, int kind, int tp,
                               void* stream, espace_proj_t* out)
{
    if (out == nullptr || h == nullptr || W_dev == nullptr)
        return fail(ESPACE_ERR_ARG, "espace_build_projection_tp: null pointer");
    *out = nullptr;
    const int64_t K = h->K;
    if (kind == ESPACE_TP_COLUMN) {
        if (tp < 1 || tp > 8) return fail(ESPACE_ERR_SHAPE, "tensor parallel: tp=%d must be in [1, 8]", tp);
        // every column-parallel rank sees all K inputs: one eigen-solve, the plain layer
        return espace_build_projection(h, W_dev, M, L, stream, out);
    }
    int rc = check_tp_shape(kind, tp, K, M, L);
    if (rc != ESPACE_OK) return rc;
    if (!aligned16(W_dev)) return fail(ESPACE_ERR_ALIGN, "espace_build_projection_tp: W not 16-byte aligned");
    if (h->n == 0) return fail(ESPACE_ERR_STATE, "espace_build_projection_tp: no calibration tokens");
    if (h->mode > 2) return fail(ESPACE_ERR_STATE, "espace_build_projection_tp: needs an activation autocorrelation");
    DeviceGuard g(h->device);
    std::vector<float> S;
    rc = read_sum(h, S, stream);
    if (rc != ESPACE_OK) return rc;
    std::vector<double> C(static_cast<size_t>(K * K));
    mirror_scaled(S, K, 1.0 / static_cast<double>(h->n), C.data());
    const int64_t Kr = K / tp;
    std::vector<double> P(static_cast<size_t>(tp * Kr * L)), evals(static_cast<size_t>(K));
    std::vector<double> Cr(static_cast<size_t>(Kr * Kr)), w, Pr;
    for (int r = 0; r < tp; ++r) {
        // rank r's inputs are features r Kr .. (r+1) Kr: its autocorrelation is C's diagonal block
        for (int64_t i = 0; i < Kr; ++i)
            for (int64_t j = 0; j < Kr; ++j) Cr[i * Kr + j] = C[(r * Kr + i) * K + r * Kr + j];
        rc = principal_eigenvectors(Cr.data(), Kr, L, false, w, Pr);
        if (rc != ESPACE_OK) return fail(rc, "espace_build_projection_tp: eigen-solver did not converge");
        std::copy(Pr.begin(), Pr.end(), P.begin() + r * Kr * L);
        for (int64_t i = 0; i < Kr; ++i) evals[r * Kr + i] = w[i];
    }
    espace_proj_s* p = nullptr;
    rc = tp_create_and_fold(kind, tp, K, M, L, P.data(), W_dev, static_cast<cudaStream_t>(stream), &p);
    if (rc != ESPACE_OK) return rc;
    p->evals = evals;
    *out = p;
    return ESPACE_OK;
}

int espace_proj_tp_info(espace_proj_t p, int* kind, int* tp)
{
    if (p == nullptr) return fail(ESPACE_ERR_ARG, "espace_proj_tp_info: null handle");
    if (kind) *kind = p->tp_kind;
    if (tp) *tp = p->tp;
    return ESPACE_OK;
}

int espace_proj_shape(espace_proj_t p, int64_t* K, int64_t* M, int64_t* L)
{
    if (p == nullptr) return fail(ESPACE_ERR_ARG, "espace_proj_shape: null handle");
    if (K) *K = p->K;
    if (M) *M = p->M;
    if (L) *L = p->L;
    return ESPACE_OK;
}

int espace_proj_eigenvalues(espace_proj_t p, double* dst)
{
    if (p == nullptr || dst == nullptr) return fail(ESPACE_ERR_ARG, "espace_proj_eigenvalues: null pointer");
    if (p->evals.empty()) return fail(ESPACE_ERR_STATE, "espace_proj_eigenvalues: projection was not calibrated");
    memcpy(dst, p->evals.data(), sizeof(double) * p->evals.size());
    return ESPACE_OK;
}

int espace_proj_read_P(espace_proj_t p, uint16_t* P_host)
{
    if (p == nullptr || P_host == nullptr) return fail(ESPACE_ERR_ARG, "espace_proj_read_P: null pointer");
    DeviceGuard g(p->device);
    // plain: P^T is [Lp][K]; tensor parallel: tp blocks of L rows of Kr (K or K / tp)
    const int64_t nb = p->tp_kind != 0 ? p->tp : 1;
    const int64_t Kr = p->tp_kind == ESPACE_TP_ROW ? p->K / p->tp : p->K;
    const int64_t rows = p->tp_kind != 0 ? p->tp * p->L : p->Lp;
    std::vector<uint16_t> pt(static_cast<size_t>(rows * Kr));
    CUDA_TRY(cudaDeviceSynchronize(), "read_P: sync");
    CUDA_TRY(cudaMemcpy(pt.data(), p->PT, sizeof(uint16_t) * pt.size(), cudaMemcpyDeviceToHost), "read_P: copy");
    for (int64_t b = 0; b < nb; ++b)
        for (int64_t k = 0; k < Kr; ++k)
            for (int64_t l = 0; l < p->L; ++l) P_host[(b * Kr + k) * p->L + l] = pt[(b * p->L + l) * Kr + k];
    return ESPACE_OK;
}

int espace_proj_read_Wfold(espace_proj_t p, uint16_t* Wf_host)
{
    if (p == nullptr || Wf_host == nullptr) return fail(ESPACE_ERR_ARG, "espace_proj_read_Wfold: null pointer");
    if (p->tp_kind != 0) return fail(ESPACE_ERR_STATE, "espace_proj_read_Wfold: tensor-parallel handle");
    DeviceGuard g(p->device);
    std::vector<uint16_t> wt(static_cast<size_t>(p->M * p->Lp));
    CUDA_TRY(cudaDeviceSynchronize(), "read_Wfold: sync");
    CUDA_TRY(cudaMemcpy(wt.data(), p->WfT, sizeof(uint16_t) * wt.size(), cudaMemcpyDeviceToHost), "read_Wfold: copy");
    for (int64_t l = 0; l < p->L; ++l)
        for (int64_t m = 0; m < p->M; ++m) Wf_host[l * p->M + m] = wt[m * p->Lp + l];
    return ESPACE_OK;
}

int espace_proj_export(espace_proj_t p, uint16_t* PT_host, uint16_t* WfT_host, double* evals)
{
    if (p == nullptr || PT_host == nullptr || WfT_host == nullptr)
        return fail(ESPACE_ERR_ARG, "espace_proj_export: null pointer");
    if (p->tp_kind != 0) return fail(ESPACE_ERR_STATE, "espace_proj_export: tensor-parallel handle");
    DeviceGuard g(p->device);
    CUDA_TRY(cudaDeviceSynchronize(), "proj_export: sync");
    CUDA_TRY(cudaMemcpy(PT_host, p->PT, sizeof(uint16_t) * p->Lp * p->K, cudaMemcpyDeviceToHost), "proj_export: P");
    CUDA_TRY(cudaMemcpy(WfT_host, p->WfT, sizeof(uint16_t) * p->M * p->Lp, cudaMemcpyDeviceToHost), "proj_export: W'");
    if (evals) {
        for (int64_t i = 0; i < p->K; ++i) evals[i] = p->evals.empty() ? 0.0 : p->evals[i];
    }
    return ESPACE_OK;
}

int espace_proj_import(int64_t K, int64_t M, int64_t L, const uint16_t* PT_host, const uint16_t* WfT_host,
                       const double* evals, espace_proj_t* out)
{
    if (out == nullptr || PT_host == nullptr || WfT_host == nullptr)
        return fail(ESPACE_ERR_ARG, "espace_proj_import: null pointer");
    *out = nullptr;
    int rc = check_proj_shape(K, M, L);
    if (rc != ESPACE_OK) return rc;
    espace_proj_s* p = nullptr;
    rc = proj_create(K, M, L, &p);
    if (rc != ESPACE_OK) return rc;
    cudaError_t e = cudaMemcpy(p->PT, PT_host, sizeof(uint16_t) * p->Lp * K, cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMemcpy(p->WfT, WfT_host, sizeof(uint16_t) * M * p->Lp, cudaMemcpyHostToDevice);
    if (e != cudaSuccess) {
        espace_proj_destroy(p);
        return fail_cuda(e, "espace_proj_import: copy");
    }
    if (evals) p->evals.assign(evals, evals + K);
    *out = p;
    return ESPACE_OK;
}

void espace_proj_destroy(espace_proj_t p)
{
    if (p == nullptr) return;
    DeviceGuard g(p->device);
    cudaDeviceSynchronize();
    if (p->PT) cudaFree(p->PT);
    if (p->WfT) cudaFree(p->WfT);
    if (p->Z) cudaFree(p->Z);
    if (p->bar) cudaFree(p->bar);
    if (p->ready) cudaFree(p->ready);
    if (p->part) cudaFree(p->part);
    if (p->dz) cudaFree(p->dz);
    if (p->dwp32) cudaFree(p->dwp32);
    if (p->dwp16) cudaFree(p->dwp16);
    if (p->hx) cudaFree(p->hx);
    if (p->hy) cudaFree(p->hy);
    for (cudaEvent_t e : p->ev)
        if (e) cudaEventDestroy(e);
    if (p->s_in) cudaStreamDestroy(p->s_in);
    if (p->s_out) cudaStreamDestroy(p->s_out);
    delete p;
}

// ---------------------------------------------------------------------------- forward

// The fused kernel runs on CTA pairs with 256 x 256 tiles: worth it when both products
// have more than one tile row and column.
static bool fused_forward_applies(int n, int Lp, int M)
{
    return n > 128 && Lp > 128 && M > 128 && pair_kernel_enabled();
}

static int ensure_z(espace_proj_s* p, int64_t N, cudaStream_t st)
{
    std::lock_guard<std::mutex> lock(p->mu);
    if (p->zcap >= N) return ESPACE_OK;
    CUDA_TRY(cudaStreamSynchronize(st), "forward: sync before scratch growth");
    if (p->Z) cudaFree(p->Z);
    if (p->ready) cudaFree(p->ready);
    p->Z = nullptr;
    p->ready = nullptr;
    p->zcap = 0;
    const int64_t cap = std::max<int64_t>(N, 128);
    cudaError_t e = cudaMalloc(&p->Z, sizeof(uint16_t) * cap * p->Lp);
    // fused forward: one readiness counter per 256-row block of Z, then its work-item
    // ticket and exit counter
    const int64_t blocks = (cap + 255) / 256;
    if (e == cudaSuccess) e = cudaMalloc(&p->ready, sizeof(int) * (blocks + 2));
    if (e == cudaSuccess) e = cudaMemset(p->ready, 0, sizeof(int) * (blocks + 2));
    if (e != cudaSuccess) return fail(ESPACE_ERR_NOMEM, "forward: Z scratch of %lld tokens: %s", (long long)cap, cudaGetErrorString(e));
    p->zcap = cap;
    return ESPACE_OK;
}

// Workspace of the swapped products (phase 1: P^T against X; phase 2: W'^T against Z) for
// n tokens, grown when a plan needs more.
static int ensure_swap(espace_proj_s* p, int n, int num_sms, cudaStream_t st)
{
    const SwapPlan a = gemm_swap_plan(static_cast<int>(p->Lp), n, static_cast<int>(p->K), num_sms, true);
    const SwapPlan b = gemm_swap_plan(static_cast<int>(p->M), n, static_cast<int>(p->Lp), num_sms, true);
    const int64_t part = std::max(a.part_elems, b.part_elems);
    std::lock_guard<std::mutex> lock(p->mu);
    if (part == 0 || p->part_cap >= part) return ESPACE_OK;
    CUDA_TRY(cudaStreamSynchronize(st), "forward: sync before workspace growth");
    if (p->part) cudaFree(p->part);
    p->part = nullptr;
    p->part_cap = 0;
    cudaError_t e = cudaMalloc(&p->part, sizeof(float) * part);
    if (e != cudaSuccess) return fail(ESPACE_ERR_NOMEM, "forward: split workspace: %s", cudaGetErrorString(e));
    p->part_cap = part;
    return ESPACE_OK;
}

// Tensor-parallel layer: a dense product and a block-diagonal one (one block per rank), Z
// ([N][tp L]) through the scratch buffer.
static int tp_forward(espace_proj_s* p, const void* X, int n, void* Y, cudaStream_t st)
{
    DeviceGuard g(p->device);
    int rc = ensure_z(p, n, st);
    if (rc != ESPACE_OK) return rc;
    const int tp = p->tp, K = static_cast<int>(p->K), M = static_cast<int>(p->M), L = static_cast<int>(p->L);
    const int zw = tp * L;   // width of Z
    int ak0[8], c0[8], cw[8];
    cudaEvent_t mid = g_phase_event;
    g_phase_event = nullptr;
    if (p->tp_kind == ESPACE_TP_COLUMN) {
        CUDA_TRY(launch_gemm_tn(X, K, p->PT, K, n, zw, K, p->Z, zw, st), "tensor parallel: phase 1");
        if (mid) CUDA_TRY(cudaEventRecord(mid, st), "forward: phase event");
        for (int r = 0; r < tp; ++r) {
            ak0[r] = r * L;
            c0[r] = r * (M / tp);
            cw[r] = M / tp;
        }
        CUDA_TRY(launch_gemm_tn_blocks(p->Z, zw, zw, p->WfT, n, tp, ak0, c0, cw, L, Y, M, st), "tensor parallel: phase 2");
    } else {
        for (int r = 0; r < tp; ++r) {
            ak0[r] = r * (K / tp);
            c0[r] = r * L;
            cw[r] = L;
        }
        CUDA_TRY(launch_gemm_tn_blocks(X, K, K, p->PT, n, tp, ak0, c0, cw, K / tp, p->Z, zw, st), "tensor parallel: phase 1");
        if (mid) CUDA_TRY(cudaEventRecord(mid, st), "forward: phase event");
        CUDA_TRY(launch_gemm_tn(p->Z, zw, p->WfT, zw, n, M, zw, Y, M, st), "tensor parallel: phase 2");
    }
    return ESPACE_OK;
}

// Tokens served by the swapped tcgen05 products (between the decode kernel and the fused
// CTA-pair launch).
static bool swap_forward_applies(int n, int path) { return n <= SWAP_MAX_TOKENS && path != ESPACE_PATH_TENSOR_SPLIT; }

// Above SWAP_MAX_TOKENS, a rank-L product with fewer 256 x 256 tiles than a quarter of the
// SMs (small L and N, e.g. L = 512 at 2048 tokens: 16 tiles) leaves most CTA pairs of the
// fused launch idle while it runs. When it also holds most of the work (K >= 2 M, e.g. an
// FC2 layer) it takes the swapped product with its reduction split over the SMs instead,
// then the folded-weight product on CTA pairs (measured: GPT3-1.3B FC2 at 2048 tokens 56 ->
// 42 us); otherwise the fused launch, whose folded-weight tiles fill the idle pairs, stays
// faster (GPT3-1.3B QKV 41 against 47 us, GPT3-8B QKV 73 against 86 us).
static bool split_phase1_applies(int n, int K, int Lp, int M, int num_sms, int path)
{
    const int64_t tiles = ((static_cast<int64_t>(n) + 255) / 256) * ((Lp + 255) / 256);
    return n > SWAP_MAX_TOKENS && path != ESPACE_PATH_SMALL_N && tiles < num_sms / 4 &&
           static_cast<int64_t>(K) >= 2 * static_cast<int64_t>(M);
}

int espace_linear_forward_path(espace_proj_t p, const void* X_dev, int64_t N, void* Y_dev, void* stream,
                               int path)
{
    if (p == nullptr) return fail(ESPACE_ERR_ARG, "espace_linear_forward: null handle");
    if (N < 0) return fail(ESPACE_ERR_SHAPE, "espace_linear_forward: N=%lld < 0", (long long)N);
    if (N == 0) return ESPACE_OK;
    if (X_dev == nullptr || Y_dev == nullptr) return fail(ESPACE_ERR_ARG, "espace_linear_forward: null pointer");
    if (!aligned16(X_dev) || !aligned16(Y_dev)) return fail(ESPACE_ERR_ALIGN, "espace_linear_forward: X/Y not 16-byte aligned");
    if (N > (int64_t(1) << 31) - 256) return fail(ESPACE_ERR_SHAPE, "espace_linear_forward: N=%lld too large", (long long)N);
    if (path < 0 || path > 3) return fail(ESPACE_ERR_ARG, "espace_linear_forward: unknown path %d", path);
    const int K = static_cast<int>(p->K), M = static_cast<int>(p->M), Lp = static_cast<int>(p->Lp);
    const int n = static_cast<int>(N);
    if (p->tp_kind != 0) return tp_forward(p, X_dev, n, Y_dev, static_cast<cudaStream_t>(stream));
    DeviceInfo* dev = nullptr;
    {
        DeviceGuard g0(p->device);
        int rc0 = device_info(&dev);
        if (rc0 != ESPACE_OK) return rc0;
    }
    const bool small_ok = N <= DECODE_MAX_TOKENS && decode_supported(n, K, Lp, M, dev->num_sms);
    if (path == ESPACE_PATH_SMALL_N && !small_ok)
        return fail(ESPACE_ERR_SHAPE, "espace_linear_forward: N=%lld (K=%d, Lp=%d) beyond the small-N kernels", (long long)N, K, Lp);
    const bool small = path == ESPACE_PATH_SMALL_N || (path == ESPACE_PATH_AUTO && small_ok && N <= DECODE_AUTO_TOKENS);
    DeviceGuard g(p->device);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    int rc = ensure_z(p, N, st);
    if (rc != ESPACE_OK) return rc;
    cudaEvent_t mid = g_phase_event;
    g_phase_event = nullptr;
    if (small) {
        // one launch holds both products; the phase event marks its end
        CUDA_TRY(launch_decode_forward(p->PT, p->WfT, X_dev, p->Z, Y_dev, K, Lp, M, n, p->bar, st),
                 "forward: decode kernel");
        if (mid) CUDA_TRY(cudaEventRecord(mid, st), "forward: phase event");
    } else if (swap_forward_applies(n, path)) {
        // few tokens: the weights are the 128-row operand; phase 1 splits its reduction
        rc = ensure_swap(p, n, dev->num_sms, st);
        if (rc != ESPACE_OK) return rc;
        // both products start streaming the handle's weights (which no kernel of the stream
        // writes meanwhile) while the grid before them finishes
        CUDA_TRY(launch_gemm_swap(p->PT, K, X_dev, K, Lp, n, K, p->Z, Lp, p->part, st, mid == nullptr),
                 "forward: phase 1");
        if (mid) CUDA_TRY(cudaEventRecord(mid, st), "forward: phase event");
        CUDA_TRY(launch_gemm_swap(p->WfT, Lp, p->Z, Lp, M, n, Lp, Y_dev, M, p->part, st, mid == nullptr),
                 "forward: phase 2");
    } else if (split_phase1_applies(n, K, Lp, M, dev->num_sms, path)) {
        rc = ensure_swap(p, n, dev->num_sms, st);
        if (rc != ESPACE_OK) return rc;
        CUDA_TRY(launch_gemm_swap(p->PT, K, X_dev, K, Lp, n, K, p->Z, Lp, p->part, st, mid == nullptr),
                 "forward: phase 1");
        if (mid) CUDA_TRY(cudaEventRecord(mid, st), "forward: phase event");
        CUDA_TRY(launch_gemm_tn(p->Z, Lp, p->WfT, Lp, n, M, Lp, Y_dev, M, st), "forward: phase 2");
    } else if (path != ESPACE_PATH_TENSOR_SPLIT && fused_forward_applies(n, Lp, M)) {
        // one persistent launch holds both products; the phase event marks its start
        if (mid) CUDA_TRY(cudaEventRecord(mid, st), "forward: phase event");
        CUDA_TRY(launch_forward_fused(X_dev, p->PT, p->Z, p->WfT, Y_dev, n, K, Lp, M, p->ready,
                                      p->ready + (p->zcap + 255) / 256, st),
                 "forward: fused kernel");
    } else {
        CUDA_TRY(launch_gemm_tn(X_dev, K, p->PT, K, n, Lp, K, p->Z, Lp, st), "forward: phase 1");
        if (mid) CUDA_TRY(cudaEventRecord(mid, st), "forward: phase event");
        CUDA_TRY(launch_gemm_tn(p->Z, Lp, p->WfT, Lp, n, M, Lp, Y_dev, M, st), "forward: phase 2");
    }
    return ESPACE_OK;
}

int espace_linear_forward_launches(espace_proj_t p, int64_t N, int path)
{
    if (p == nullptr || N < 0 || path < 0 || path > 3) return -1;
    if (N == 0) return 0;
    DeviceInfo* dev = nullptr;
    {
        DeviceGuard g(p->device);
        if (device_info(&dev) != ESPACE_OK) return -1;
    }
    if (p->tp_kind != 0) return 2;
    const int n = static_cast<int>(N), K = static_cast<int>(p->K), M = static_cast<int>(p->M),
              Lp = static_cast<int>(p->Lp);
    const bool small_ok = N <= DECODE_MAX_TOKENS && decode_supported(n, K, Lp, M, dev->num_sms);
    if (path == ESPACE_PATH_SMALL_N || (path == ESPACE_PATH_AUTO && small_ok && N <= DECODE_AUTO_TOKENS))
        return small_ok ? 1 : -1;
    if (swap_forward_applies(n, path)) {
        // one launch per product, plus one per split reduction
        const int a = gemm_swap_plan(Lp, n, K, dev->num_sms, true).ksplit > 1 ? 2 : 1;
        const int b = gemm_swap_plan(M, n, Lp, dev->num_sms, true).ksplit > 1 ? 2 : 1;
        return a + b;
    }
    if (split_phase1_applies(n, K, Lp, M, dev->num_sms, path))
        return (gemm_swap_plan(Lp, n, K, dev->num_sms, true).ksplit > 1 ? 2 : 1) + 1;
    if (path != ESPACE_PATH_TENSOR_SPLIT && fused_forward_applies(n, Lp, M)) return 1;
    return 2;
}

int espace_linear_forward(espace_proj_t p, const void* X_dev, int64_t N, void* Y_dev, void* stream)
{
    return espace_linear_forward_path(p, X_dev, N, Y_dev, stream, ESPACE_PATH_AUTO);
}

// Chunks of the host-buffer forward: up to 8, each at least 512 tokens (multiples of 256).
// The host link (~0.2 TB/s each way, measured) is far slower than the products, so small
// chunks shorten the pipeline's fill and drain while their products stay off the critical
// path.
static int host_chunks(int64_t N, int64_t min_chunk, int64_t* chunk)
{
    int nc = static_cast<int>(std::min<int64_t>(8, std::max<int64_t>(1, N / min_chunk)));
    int64_t c = (N + nc - 1) / nc;
    c = (c + 255) / 256 * 256;
    nc = static_cast<int>((N + c - 1) / c);
    *chunk = c;
    return nc;
}

// The handle's copy streams, events and device staging for N tokens (created or grown on
// first need; growth synchronizes the caller's stream).
static int ensure_host_io(espace_proj_s* p, int64_t N, cudaStream_t st)
{
    std::lock_guard<std::mutex> lock(p->mu);
    if (p->s_in == nullptr) {
        cudaError_t e = cudaStreamCreateWithFlags(&p->s_in, cudaStreamNonBlocking);
        if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&p->s_out, cudaStreamNonBlocking);
        for (cudaEvent_t& ev : p->ev)
            if (e == cudaSuccess) e = cudaEventCreateWithFlags(&ev, cudaEventDisableTiming);
        if (e != cudaSuccess) {
            // release what was made, so that the next call starts over
            for (cudaEvent_t& ev : p->ev)
                if (ev) {
                    cudaEventDestroy(ev);
                    ev = nullptr;
                }
            if (p->s_out) cudaStreamDestroy(p->s_out);
            if (p->s_in) cudaStreamDestroy(p->s_in);
            p->s_in = p->s_out = nullptr;
            return fail_cuda(e, "espace_linear_forward_host: streams");
        }
    }
    if (p->h_cap < N) {
        CUDA_TRY(cudaStreamSynchronize(st), "espace_linear_forward_host: sync before staging growth");
        if (p->hx) cudaFree(p->hx);
        if (p->hy) cudaFree(p->hy);
        p->hx = p->hy = nullptr;
        p->h_cap = 0;
        cudaError_t e = cudaMalloc(&p->hx, sizeof(uint16_t) * N * p->K);
        if (e == cudaSuccess) e = cudaMalloc(&p->hy, sizeof(uint16_t) * N * p->M);
        if (e != cudaSuccess) return fail(ESPACE_ERR_NOMEM, "espace_linear_forward_host: staging: %s", cudaGetErrorString(e));
        p->h_cap = N;
    }
    return ESPACE_OK;
}

// Chunk boundaries (b[0] = 0 < ... < b[n] = N, n <= 11) of one layer's N tokens in the
// pipeline of several layers: up to 8 chunks of about 8192 tokens (at most, below 64K
// tokens); the pipeline's first layer leads with chunks of 2048 and 4096 tokens (its first
// product starts once 2048 tokens are in, and each next chunk is copied in while the one
// before computes), and its last layer ends with a 2048-token chunk (the last copy out is
// short), where N leaves room for them.
static int many_bounds(int64_t N, bool first, bool last, int64_t* b)
{
    if (N <= 0) return 0;
    int n = 0;
    b[0] = 0;
    int64_t lo = 0;
    const int64_t keep = 8192 + (last ? 2048 : 0);
    if (first)
        for (int64_t h : {int64_t(2048), int64_t(4096)})
            if (N - lo >= h + keep) {
                lo += h;
                b[++n] = lo;
            }
    const int64_t tail = (last && N - lo >= 2048 + 8192) ? 2048 : 0;
    const int64_t hi = N - tail;
    const int64_t k = std::min<int64_t>(8, (hi - lo + 8191) / 8192);
    int64_t c = (hi - lo + k - 1) / k;
    c = (c + 255) / 256 * 256;
    for (int64_t t = lo + c; t < hi; t += c) b[++n] = t;
    b[++n] = hi;
    if (tail > 0) b[++n] = N;
    return n;
}

// The host-buffer pipeline over `count` independent layers (distinct handles, validated by
// the caller): every copy in on the first handle's copy-in stream and every product on the
// caller's stream, both in layer order, each copy out on the first handle's copy-out stream
// once its chunk is computed, through layer i's staging and events. The layers' tokens go
// in the chunks of many_bounds (several_layers), else in chunks of at least min_chunk (up
// to 8). wait: return once every Y_host is filled; else the caller's stream is ordered after
// the last copy out and the call returns once queued.
static int host_pipeline(int count, espace_proj_s* const* layers, const void* const* X_host, const int64_t* N,
                         void* const* Y_host, cudaStream_t st, int64_t min_chunk, bool wait, bool several_layers)
{
    espace_proj_s* h0 = layers[0];
    DeviceGuard g(h0->device);
    for (int i = 0; i < count; ++i) {
        const int rc = ensure_host_io(layers[i], std::max<int64_t>(N[i], 1), st);
        if (rc != ESPACE_OK) return rc;
    }
    cudaStream_t s_in = h0->s_in, s_out = h0->s_out;
    cudaEvent_t start = h0->ev[32], end = h0->ev[33];
    // the copies start after the work already on the caller's stream
    CUDA_TRY(cudaEventRecord(start, st), "espace_linear_forward_host: order");
    CUDA_TRY(cudaStreamWaitEvent(s_in, start, 0), "espace_linear_forward_host: order");
    CUDA_TRY(cudaStreamWaitEvent(s_out, start, 0), "espace_linear_forward_host: order");
    // on an error after copies were queued, wait for them before returning, so that no copy
    // touches the caller's host buffers after the call
    struct Drain {
        cudaStream_t a, b, c;
        bool armed = true;
        ~Drain()
        {
            if (!armed) return;
            cudaStreamSynchronize(a);
            cudaStreamSynchronize(b);
            cudaStreamSynchronize(c);
        }
    } drain{s_in, st, s_out};
    int64_t bounds[ESPACE_HOST_MANY_MAX][12];
    int nchunks[ESPACE_HOST_MANY_MAX];
    for (int i = 0; i < count; ++i) {
        espace_proj_s* p = layers[i];
        if (several_layers) {
            nchunks[i] = many_bounds(N[i], i == 0, i == count - 1, bounds[i]);
        } else {
            int64_t c = 0;
            nchunks[i] = N[i] > 0 ? host_chunks(N[i], min_chunk, &c) : 0;
            for (int j = 0; j <= nchunks[i]; ++j) bounds[i][j] = std::min(j * c, N[i]);
        }
        const uint16_t* xh = static_cast<const uint16_t*>(X_host[i]);
        for (int j = 0; j < nchunks[i]; ++j) {
            const int64_t t0 = bounds[i][j], n = bounds[i][j + 1] - t0;
            CUDA_TRY(cudaMemcpyAsync(p->hx + t0 * p->K, xh + t0 * p->K, sizeof(uint16_t) * n * p->K,
                                     cudaMemcpyHostToDevice, s_in),
                     "espace_linear_forward_host: copy in");
            CUDA_TRY(cudaEventRecord(p->ev[j], s_in), "espace_linear_forward_host: event");   // chunk j in
        }
    }
    for (int i = 0; i < count; ++i) {
        espace_proj_s* p = layers[i];
        uint16_t* yh = static_cast<uint16_t*>(Y_host[i]);
        for (int j = 0; j < nchunks[i]; ++j) {
            const int64_t t0 = bounds[i][j], n = bounds[i][j + 1] - t0;
            // chunk j's product runs once its tokens are on the device, while other chunks'
            // tokens and outputs are copied
            CUDA_TRY(cudaStreamWaitEvent(st, p->ev[j], 0), "espace_linear_forward_host: order");
            int rc = espace_linear_forward_path(p, p->hx + t0 * p->K, n, p->hy + t0 * p->M, st, ESPACE_PATH_AUTO);
            if (rc != ESPACE_OK) return rc;
            CUDA_TRY(cudaEventRecord(p->ev[16 + j], st), "espace_linear_forward_host: event");   // chunk j done
            CUDA_TRY(cudaStreamWaitEvent(s_out, p->ev[16 + j], 0), "espace_linear_forward_host: order");
            CUDA_TRY(cudaMemcpyAsync(yh + t0 * p->M, p->hy + t0 * p->M, sizeof(uint16_t) * n * p->M,
                                     cudaMemcpyDeviceToHost, s_out),
                     "espace_linear_forward_host: copy out");
        }
    }
    CUDA_TRY(cudaEventRecord(end, s_out), "espace_linear_forward_host: event");
    CUDA_TRY(cudaStreamWaitEvent(st, end, 0), "espace_linear_forward_host: order");
    if (wait) CUDA_TRY(cudaEventSynchronize(end), "espace_linear_forward_host: wait");
    drain.armed = false;
    return ESPACE_OK;
}

// One layer through the pipeline. Chunks of at least 512 tokens for the synchronous form
// (one layer in flight: the copies overlap only its own chunks' products), of at least 8192
// for the asynchronous one (other layers in flight fill the gaps, and long chunks keep each
// product efficient: three 16,384-token layers on three streams took 10.3-10.6 ms per step
// in 2 chunks, 11.0-11.6 ms in 8).
static int forward_host(espace_proj_t p, const void* X_host, int64_t N, void* Y_host, void* stream, bool wait)
{
    if (p == nullptr) return fail(ESPACE_ERR_ARG, "espace_linear_forward_host: null handle");
    if (p->tp_kind != 0) return fail(ESPACE_ERR_STATE, "espace_linear_forward_host: tensor-parallel handle");
    if (N < 0 || N > (int64_t(1) << 31) - 256) return fail(ESPACE_ERR_SHAPE, "espace_linear_forward_host: N=%lld", (long long)N);
    if (N == 0) return ESPACE_OK;
    if (X_host == nullptr || Y_host == nullptr) return fail(ESPACE_ERR_ARG, "espace_linear_forward_host: null pointer");
    void* y = Y_host;
    return host_pipeline(1, &p, &X_host, &N, &y, static_cast<cudaStream_t>(stream), wait ? 512 : 8192, wait, false);
}

int espace_linear_forward_host_many(int count, const espace_proj_t* layers, const void* const* X_host,
                                    const int64_t* N, void* const* Y_host, void* stream)
{
    const char* what = "espace_linear_forward_host_many";
    if (count < 0 || count > ESPACE_HOST_MANY_MAX) return fail(ESPACE_ERR_ARG, "%s: count=%d", what, count);
    if (count == 0) return ESPACE_OK;
    if (layers == nullptr || X_host == nullptr || N == nullptr || Y_host == nullptr)
        return fail(ESPACE_ERR_ARG, "%s: null array", what);
    for (int i = 0; i < count; ++i) {
        espace_proj_s* p = layers[i];
        if (p == nullptr) return fail(ESPACE_ERR_ARG, "%s: null handle %d", what, i);
        if (p->tp_kind != 0) return fail(ESPACE_ERR_STATE, "%s: layer %d is a tensor-parallel handle", what, i);
        if (p->device != layers[0]->device) return fail(ESPACE_ERR_ARG, "%s: layers on different devices", what);
        if (N[i] < 0 || N[i] > (int64_t(1) << 31) - 256) return fail(ESPACE_ERR_SHAPE, "%s: N[%d]=%lld", what, i, (long long)N[i]);
        if (N[i] > 0 && (X_host[i] == nullptr || Y_host[i] == nullptr)) return fail(ESPACE_ERR_ARG, "%s: null buffer %d", what, i);
        for (int j = 0; j < i; ++j)
            if (layers[j] == p) return fail(ESPACE_ERR_ARG, "%s: handle %d repeated", what, i);
    }
    // the chunks of many_bounds: about 8192 tokens, shorter at the pipeline's two ends
    return host_pipeline(count, layers, X_host, N, Y_host, static_cast<cudaStream_t>(stream), 8192, true, true);
}

int espace_linear_forward_host(espace_proj_t p, const void* X_host, int64_t N, void* Y_host, void* stream)
{
    return forward_host(p, X_host, N, Y_host, stream, true);
}

int espace_linear_forward_host_async(espace_proj_t p, const void* X_host, int64_t N, void* Y_host, void* stream)
{
    return forward_host(p, X_host, N, Y_host, stream, false);
}

// Split workspace of the dense forward's few-token products, per device (dense calls on
// one device must be ordered on the GPU: the same stream, or streams that wait on each
// other).
struct DenseWs {
    float* part = nullptr;
    int64_t cap = 0;
    std::mutex mu;
};
static DenseWs g_dense_ws[64];

int espace_dense_forward(const void* X_dev, int64_t N, int64_t K, const void* W_dev, int64_t M, void* Y_dev,
                         void* stream)
{
    if (N < 0) return fail(ESPACE_ERR_SHAPE, "espace_dense_forward: N < 0");
    if (N == 0) return ESPACE_OK;
    if (X_dev == nullptr || W_dev == nullptr || Y_dev == nullptr) return fail(ESPACE_ERR_ARG, "espace_dense_forward: null pointer");
    if (!aligned16(X_dev) || !aligned16(W_dev) || !aligned16(Y_dev))
        return fail(ESPACE_ERR_ALIGN, "espace_dense_forward: pointers must be 16-byte aligned");
    if (K < 8 || K % 8 != 0 || K > 65536 || M < 8 || M % 8 != 0 || M > (int64_t(1) << 30) || N > (int64_t(1) << 31) - 256)
        return fail(ESPACE_ERR_SHAPE, "espace_dense_forward: unsupported shape N=%lld K=%lld M=%lld", (long long)N, (long long)K, (long long)M);
    DeviceInfo* dev = nullptr;
    int rc = device_info(&dev);
    if (rc != ESPACE_OK) return rc;
    // few tokens: stream W once through the decode kernel; otherwise the tcgen05 GEMM
    if (N <= DECODE_DENSE_AUTO_TOKENS &&
        decode_dense_supported(static_cast<int>(N), static_cast<int>(K), static_cast<int>(M), dev->num_sms)) {
        CUDA_TRY(launch_decode_dense(W_dev, X_dev, Y_dev, static_cast<int>(K), static_cast<int>(M), static_cast<int>(N),
                                     static_cast<cudaStream_t>(stream)),
                 "espace_dense_forward: decode launch");
        return ESPACE_OK;
    }
    if (N <= SWAP_MAX_TOKENS) {
        // few tokens: the weight rows span the grid, the reduction split over the SMs when
        // the tiles would leave SMs idle (partials in the device's dense workspace)
        float* part = nullptr;
        const SwapPlan pl = gemm_swap_plan(static_cast<int>(M), static_cast<int>(N), static_cast<int>(K), dev->num_sms, true);
        if (pl.part_elems > 0 && dev->device >= 0 && dev->device < 64) {
            DenseWs& ws = g_dense_ws[dev->device];
            std::lock_guard<std::mutex> lock(ws.mu);
            if (ws.cap < pl.part_elems) {
                CUDA_TRY(cudaStreamSynchronize(static_cast<cudaStream_t>(stream)), "espace_dense_forward: sync");
                if (ws.part) cudaFree(ws.part);
                ws.part = nullptr;
                ws.cap = 0;
                cudaError_t e = cudaMalloc(&ws.part, sizeof(float) * pl.part_elems);
                if (e != cudaSuccess) return fail(ESPACE_ERR_NOMEM, "espace_dense_forward: workspace: %s", cudaGetErrorString(e));
                ws.cap = pl.part_elems;
            }
            part = ws.part;
        }
        // like the projected layer's few-token products, it may start loading W while the
        // grid before it finishes (header: W must not be that grid's output)
        CUDA_TRY(launch_gemm_swap(W_dev, K, X_dev, K, static_cast<int>(M), static_cast<int>(N), static_cast<int>(K), Y_dev,
                                  M, part, static_cast<cudaStream_t>(stream), true),
                 "espace_dense_forward: launch");
        return ESPACE_OK;
    }
    CUDA_TRY(launch_gemm_tn(X_dev, K, W_dev, K, static_cast<int>(N), static_cast<int>(M), static_cast<int>(K), Y_dev, M,
                            static_cast<cudaStream_t>(stream)),
             "espace_dense_forward: launch");
    return ESPACE_OK;
}

// ---------------------------------------------------------------------------- training view

int espace_proj_refold(espace_proj_t p, const void* W_dev, void* stream)
{
    if (p == nullptr || W_dev == nullptr) return fail(ESPACE_ERR_ARG, "espace_proj_refold: null pointer");
    if (p->tp_kind != 0) return fail(ESPACE_ERR_STATE, "espace_proj_refold: tensor-parallel handle");
    if (!aligned16(W_dev)) return fail(ESPACE_ERR_ALIGN, "espace_proj_refold: W not 16-byte aligned");
    DeviceGuard g(p->device);
    CUDA_TRY(launch_gemm_tn(W_dev, p->K, p->PT, p->K, static_cast<int>(p->M), static_cast<int>(p->Lp),
                            static_cast<int>(p->K), p->WfT, p->Lp, static_cast<cudaStream_t>(stream)),
             "espace_proj_refold: launch");
    return ESPACE_OK;
}

// The fp32 accumulator of (dW P)^T ([Lp][M], zeroed) and its bf16 copy, made on first use.
static int ensure_grad_acc(espace_proj_s* p, cudaStream_t st)
{
    std::lock_guard<std::mutex> lock(p->mu);
    if (p->dwp32 != nullptr) return ESPACE_OK;
    const int64_t count = p->Lp * p->M;
    cudaError_t e = cudaMalloc(&p->dwp32, sizeof(float) * count);
    if (e == cudaSuccess) e = cudaMalloc(&p->dwp16, sizeof(uint16_t) * count);
    if (e == cudaSuccess) e = launch_zero_f32(p->dwp32, count, st);
    if (e != cudaSuccess) {
        if (p->dwp32) cudaFree(p->dwp32);
        if (p->dwp16) cudaFree(p->dwp16);
        p->dwp32 = nullptr;
        p->dwp16 = nullptr;
        return fail(ESPACE_ERR_NOMEM, "training view: gradient accumulator: %s", cudaGetErrorString(e));
    }
    return ESPACE_OK;
}

static int train_check(espace_proj_t p, int64_t N, const char* what)
{
    if (p == nullptr) return fail(ESPACE_ERR_ARG, "%s: null handle", what);
    if (p->tp_kind != 0) return fail(ESPACE_ERR_STATE, "%s: tensor-parallel handle", what);
    if (N < 0 || N > (int64_t(1) << 31) - 256) return fail(ESPACE_ERR_SHAPE, "%s: N=%lld", what, (long long)N);
    return ESPACE_OK;
}

int espace_train_forward(espace_proj_t p, const void* X_dev, int64_t N, void* Z_dev, void* Y_dev, void* stream)
{
    int rc = train_check(p, N, "espace_train_forward");
    if (rc != ESPACE_OK || N == 0) return rc;
    if (X_dev == nullptr || Z_dev == nullptr || Y_dev == nullptr) return fail(ESPACE_ERR_ARG, "espace_train_forward: null pointer");
    if (!aligned16(X_dev) || !aligned16(Z_dev) || !aligned16(Y_dev))
        return fail(ESPACE_ERR_ALIGN, "espace_train_forward: pointers must be 16-byte aligned");
    DeviceGuard g(p->device);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    rc = ensure_z(p, N, st);   // the fused launch's readiness counters
    if (rc != ESPACE_OK) return rc;
    const int n = static_cast<int>(N), K = static_cast<int>(p->K), M = static_cast<int>(p->M), Lp = static_cast<int>(p->Lp);
    if (fused_forward_applies(n, Lp, M)) {
        CUDA_TRY(launch_forward_fused(X_dev, p->PT, Z_dev, p->WfT, Y_dev, n, K, Lp, M, p->ready,
                                      p->ready + (p->zcap + 255) / 256, st),
                 "espace_train_forward: fused kernel");
    } else {
        CUDA_TRY(launch_gemm_tn(X_dev, K, p->PT, K, n, Lp, K, Z_dev, Lp, st), "espace_train_forward: Z");
        CUDA_TRY(launch_gemm_tn(Z_dev, Lp, p->WfT, Lp, n, M, Lp, Y_dev, M, st), "espace_train_forward: Y");
    }
    return ESPACE_OK;
}

int espace_train_backward(espace_proj_t p, const void* dY_dev, const void* Z_dev, int64_t N, void* dX_dev,
                          void* stream)
{
    int rc = train_check(p, N, "espace_train_backward");
    if (rc != ESPACE_OK || N == 0) return rc;
    if (dY_dev == nullptr || Z_dev == nullptr || dX_dev == nullptr)
        return fail(ESPACE_ERR_ARG, "espace_train_backward: null pointer");
    if (!aligned16(dY_dev) || !aligned16(Z_dev) || !aligned16(dX_dev))
        return fail(ESPACE_ERR_ALIGN, "espace_train_backward: pointers must be 16-byte aligned");
    DeviceGuard g(p->device);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const int64_t K = p->K, M = p->M, Lp = p->Lp;
    rc = ensure_grad_acc(p, st);
    if (rc != ESPACE_OK) return rc;
    {
        std::lock_guard<std::mutex> lock(p->mu);
        if (p->dz_cap < N) {
            CUDA_TRY(cudaStreamSynchronize(st), "espace_train_backward: sync before scratch growth");
            if (p->dz) cudaFree(p->dz);
            p->dz = nullptr;
            p->dz_cap = 0;
            cudaError_t e = cudaMalloc(&p->dz, sizeof(uint16_t) * N * Lp);
            if (e != cudaSuccess) return fail(ESPACE_ERR_NOMEM, "espace_train_backward: scratch: %s", cudaGetErrorString(e));
            p->dz_cap = N;
        }
    }
    const int n = static_cast<int>(N), k = static_cast<int>(K), m = static_cast<int>(M), lp = static_cast<int>(Lp);
    // dZ = dY W' (W' = P^T W: W'^T is [M][Lp], read M/N-major)
    CUDA_TRY(launch_gemm_nn(dY_dev, M, p->WfT, Lp, n, lp, m, p->dz, Lp, st), "espace_train_backward: dZ");
    // dX = dZ P^T (P^T is [Lp][K], read M/N-major)
    CUDA_TRY(launch_gemm_nn(p->dz, Lp, p->PT, K, n, k, lp, dX_dev, K, st), "espace_train_backward: dX");
    // (dW P)^T += Z^T dY over the tokens (the weight gradient waits for the step's end)
    CUDA_TRY(launch_gemm_tn_tokens_f32(Z_dev, lp, dY_dev, m, N, p->dwp32, M, st), "espace_train_backward: Z^T dY");
    return ESPACE_OK;
}

int espace_train_weight_grad(espace_proj_t p, float* dW_dev, void* stream)
{
    int rc = train_check(p, 0, "espace_train_weight_grad");
    if (rc != ESPACE_OK) return rc;
    if (dW_dev == nullptr) return fail(ESPACE_ERR_ARG, "espace_train_weight_grad: null pointer");
    if (!aligned16(dW_dev)) return fail(ESPACE_ERR_ALIGN, "espace_train_weight_grad: dW not 16-byte aligned");
    DeviceGuard g(p->device);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const int64_t K = p->K, M = p->M, Lp = p->Lp;
    rc = ensure_grad_acc(p, st);
    if (rc != ESPACE_OK) return rc;
    // dW = (dW P) P^T: the accumulated (dW P)^T rounded to bf16, reduced over the rank index
    CUDA_TRY(launch_f32_to_bf16(p->dwp32, Lp * M, p->dwp16, st), "espace_train_weight_grad: round");
    CUDA_TRY(launch_zero_f32(dW_dev, K * M, st), "espace_train_weight_grad: clear dW");
    CUDA_TRY(launch_gemm_tn_tokens_f32(p->dwp16, static_cast<int>(M), p->PT, static_cast<int>(K), Lp, dW_dev, K, st),
             "espace_train_weight_grad: dW");
    CUDA_TRY(launch_zero_f32(p->dwp32, Lp * M, st), "espace_train_weight_grad: reset");
    return ESPACE_OK;
}

int espace_dense_backward(const void* dY_dev, int64_t N, const void* X_dev, int64_t K, const void* W_dev, int64_t M,
                          void* dX_dev, float* dW_dev, int accumulate, void* stream)
{
    if (N < 0) return fail(ESPACE_ERR_SHAPE, "espace_dense_backward: N < 0");
    if (dW_dev == nullptr || W_dev == nullptr) return fail(ESPACE_ERR_ARG, "espace_dense_backward: null pointer");
    if (N > 0 && (dY_dev == nullptr || X_dev == nullptr || dX_dev == nullptr))
        return fail(ESPACE_ERR_ARG, "espace_dense_backward: null pointer");
    if (K < 8 || K % 8 != 0 || K > 65536 || M < 8 || M % 8 != 0 || M > (int64_t(1) << 30) || N > (int64_t(1) << 31) - 256)
        return fail(ESPACE_ERR_SHAPE, "espace_dense_backward: unsupported shape N=%lld K=%lld M=%lld", (long long)N, (long long)K,
                    (long long)M);
    if ((N > 0 && (!aligned16(dY_dev) || !aligned16(X_dev) || !aligned16(dX_dev))) || !aligned16(W_dev) || !aligned16(dW_dev))
        return fail(ESPACE_ERR_ALIGN, "espace_dense_backward: pointers must be 16-byte aligned");
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (!accumulate) CUDA_TRY(launch_zero_f32(dW_dev, K * M, st), "espace_dense_backward: clear dW");
    if (N == 0) return ESPACE_OK;
    // dX = dY W (W [M][K] read M/N-major), dW = dY^T X over the tokens
    CUDA_TRY(launch_gemm_nn(dY_dev, M, W_dev, K, static_cast<int>(N), static_cast<int>(K), static_cast<int>(M), dX_dev, K, st),
             "espace_dense_backward: dX");
    CUDA_TRY(launch_gemm_tn_tokens_f32(dY_dev, static_cast<int>(M), X_dev, static_cast<int>(K), N, dW_dev, K, st),
             "espace_dense_backward: dW");
    return ESPACE_OK;
}

int espace_debug_wait_timeout(uint64_t limit_ns, void* stream)
{
    if (limit_ns == 0 || limit_ns > 1000000000ull)
        return fail(ESPACE_ERR_ARG, "espace_debug_wait_timeout: limit must be in (0, 1e9] ns");
    CUDA_TRY(launch_wait_timeout(limit_ns, static_cast<cudaStream_t>(stream)), "espace_debug_wait_timeout");
    return ESPACE_OK;
}

int espace_debug_occupy(int ctas, uint64_t hold_ns, void* stream)
{
    DeviceInfo* dev = nullptr;
    int rc = device_info(&dev);
    if (rc != ESPACE_OK) return rc;
    if (ctas < 1 || ctas > dev->num_sms)
        return fail(ESPACE_ERR_ARG, "espace_debug_occupy: ctas must be in [1, %d]", dev->num_sms);
    if (hold_ns == 0 || hold_ns > 1000000000ull)
        return fail(ESPACE_ERR_ARG, "espace_debug_occupy: hold must be in (0, 1e9] ns");
    CUDA_TRY(launch_occupy(ctas, hold_ns, static_cast<cudaStream_t>(stream)), "espace_debug_occupy");
    return ESPACE_OK;
}

int espace_check(void* stream)
{
    DeviceInfo* dev = nullptr;
    int rc = device_info(&dev);
    if (rc != ESPACE_OK) return rc;
    CUDA_TRY(cudaStreamSynchronize(static_cast<cudaStream_t>(stream)), "espace_check: stream");
    int status = 0;
    CUDA_TRY(cudaMemcpy(&status, dev->status, sizeof(int), cudaMemcpyDeviceToHost), "espace_check: status");
    if (status != 0) {
        CUDA_TRY(cudaMemset(dev->status, 0, sizeof(int)), "espace_check: clear");
        return fail(status, "espace_check: a kernel gave up waiting (device status %d)", status);
    }
    return ESPACE_OK;
}

}  // extern "C"

// ============================================================================ internal views

namespace espace {

struct ProjView {
    int64_t K, M, L, Lp;
    int device;
    const void* PT;
    const void* WfT;
    unsigned int* bar;
};

int proj_view(espace_proj_t p, ProjView* out)
{
    if (p == nullptr || out == nullptr) return fail(ESPACE_ERR_ARG, "proj_view: null pointer");
    if (p->tp_kind != 0) return fail(ESPACE_ERR_STATE, "espace_linear_forward_noalloc: tensor-parallel handle");
    out->K = p->K;
    out->M = p->M;
    out->L = p->L;
    out->Lp = p->Lp;
    out->device = p->device;
    out->PT = p->PT;
    out->WfT = p->WfT;
    out->bar = p->bar;
    return ESPACE_OK;
}

void set_last_error(const char* msg) { g_last_error = msg; }

}  // namespace espace
