// runtime.cu -- host-side plumbing: error strings, launch checks, the device
// status word, SM count, and TMA tensor-map encoding.
#include <stdarg.h>
#include <stdio.h>

#include <atomic>
#include <mutex>

#include "internal.h"

namespace ff {

namespace {
thread_local char g_err[512] = "";

// One status word per device; kernels OR error bits into it.
__device__ int g_device_status;

constexpr int kMaxDevices = 64;
// Per-device caches, keyed by device ordinal: they hold the primary
// context's values and go stale after cudaDeviceReset.
std::atomic<int*> g_status_ptr[kMaxDevices] = {};
std::atomic<int> g_num_sms[kMaxDevices] = {};
std::mutex g_mu;

using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                   const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeTiledFn g_encode = nullptr;

int current_device() {
    int d = 0;
    if (cudaGetDevice(&d) != cudaSuccess || d < 0 || d >= kMaxDevices) return -1;
    return d;
}
}  // namespace

int set_error(int code, const char* fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, sizeof(g_err), fmt, ap);
    va_end(ap);
    return code;
}

const char* last_error() { return g_err; }

int check_launch(const char* what) {
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return set_error(FF_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
    return FF_OK;
}

int* device_status_ptr() {
    const int d = current_device();
    if (d < 0) return nullptr;
    int* p = g_status_ptr[d].load(std::memory_order_acquire);
    if (!p) {
        std::lock_guard<std::mutex> lk(g_mu);
        p = g_status_ptr[d].load(std::memory_order_relaxed);
        if (!p) {
            void* q = nullptr;
            if (cudaGetSymbolAddress(&q, g_device_status) != cudaSuccess) return nullptr;
            p = static_cast<int*>(q);
            g_status_ptr[d].store(p, std::memory_order_release);
        }
    }
    return p;
}

int num_sms() {
    const int d = current_device();
    if (d < 0) return 1;
    int n = g_num_sms[d].load(std::memory_order_relaxed);
    if (!n) {
        cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, d);
        if (n <= 0) n = 1;
        g_num_sms[d].store(n, std::memory_order_relaxed);
    }
    return n;
}

int make_tmap_f32_sw128(CUtensorMap* tm, const void* base, int64_t rows, int64_t cols, int64_t ld, int box_rows) {
    if (!g_encode) {
        CUtensorMap dummy;
        const int rc = make_tmap_bf16(&dummy, base, 1, 8, 8, 1);   // resolves the driver entry point
        if (rc) return rc;
    }
    if (!aligned16(base)) return set_error(FF_ERR_INVALID_ARG, "tensor map base not 16-byte aligned");
    if ((ld * 4) % 16) return set_error(FF_ERR_INVALID_ARG, "tensor map row pitch not a multiple of 16 bytes");
    const cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
    const cuuint64_t strides[1] = {static_cast<cuuint64_t>(ld) * 4};
    const cuuint32_t box[2] = {32, static_cast<cuuint32_t>(box_rows)};
    const cuuint32_t estr[2] = {1, 1};
    const CUresult r = g_encode(tm, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<void*>(base), dims, strides, box,
                                estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                                CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS)
        return set_error(FF_ERR_CUDA, "cuTensorMapEncodeTiled (fp32) failed (%d) rows=%lld cols=%lld ld=%lld", (int)r,
                         (long long)rows, (long long)cols, (long long)ld);
    return FF_OK;
}

int make_tmap_out(CUtensorMap* tm, const void* base, int64_t rows, int64_t cols, int64_t ld, bool f32) {
    if (!g_encode) {
        CUtensorMap dummy;
        const int rc = make_tmap_bf16(&dummy, base, 1, 8, 8, 1);   // resolves the driver entry point
        if (rc) return rc;
    }
    const int es = f32 ? 4 : 2;
    if (!aligned16(base)) return set_error(FF_ERR_INVALID_ARG, "tensor map base not 16-byte aligned");
    if ((ld * es) % 16) return set_error(FF_ERR_INVALID_ARG, "tensor map row pitch not a multiple of 16 bytes");
    const cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
    const cuuint64_t strides[1] = {static_cast<cuuint64_t>(ld) * es};
    const cuuint32_t box[2] = {32, 32};
    const cuuint32_t estr[2] = {1, 1};
    const CUresult r = g_encode(tm, f32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
                                const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                                f32 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B,
                                CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS)
        return set_error(FF_ERR_CUDA, "cuTensorMapEncodeTiled (output) failed (%d) rows=%lld cols=%lld ld=%lld",
                         (int)r, (long long)rows, (long long)cols, (long long)ld);
    return FF_OK;
}

int make_tmap_bf16(CUtensorMap* tm, const void* base, int64_t rows, int64_t cols, int64_t ld, int box_rows) {
    if (!g_encode) {
        std::lock_guard<std::mutex> lk(g_mu);
        if (!g_encode) {
            void* fn = nullptr;
            cudaDriverEntryPointQueryResult q;
            if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) !=
                    cudaSuccess ||
                q != cudaDriverEntryPointSuccess || !fn)
                return set_error(FF_ERR_CUDA, "cuTensorMapEncodeTiled not available from the driver");
            g_encode = reinterpret_cast<EncodeTiledFn>(fn);
        }
    }
    if (!aligned16(base)) return set_error(FF_ERR_INVALID_ARG, "tensor map base not 16-byte aligned");
    if ((ld * 2) % 16) return set_error(FF_ERR_INVALID_ARG, "tensor map row pitch not a multiple of 16 bytes");
    const cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
    const cuuint64_t strides[1] = {static_cast<cuuint64_t>(ld) * 2};
    const cuuint32_t box[2] = {64, static_cast<cuuint32_t>(box_rows)};
    const cuuint32_t estr[2] = {1, 1};
    const CUresult r = g_encode(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
                                estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                                CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS)
        return set_error(FF_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d) rows=%lld cols=%lld ld=%lld box=%d",
                         (int)r, (long long)rows, (long long)cols, (long long)ld, box_rows);
    return FF_OK;
}

}  // namespace ff

extern "C" {

const char* ff_last_error(void) { return ff::last_error(); }

int ff_version(void) { return 100; }

int ff_check_device_status(cudaStream_t stream, int* status_out) {
    if (!status_out) return ff::set_error(FF_ERR_INVALID_ARG, "status_out is null");
    int* p = ff::device_status_ptr();
    if (!p) return ff::set_error(FF_ERR_CUDA, "no device status word");
    if (cudaStreamSynchronize(stream) != cudaSuccess)
        return ff::set_error(FF_ERR_CUDA, "stream synchronise failed: %s", cudaGetErrorString(cudaGetLastError()));
    int v = 0;
    if (cudaMemcpy(&v, p, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess)
        return ff::set_error(FF_ERR_CUDA, "status read failed");
    const int zero = 0;
    if (cudaMemcpy(p, &zero, sizeof(int), cudaMemcpyHostToDevice) != cudaSuccess)
        return ff::set_error(FF_ERR_CUDA, "status clear failed");
    *status_out = v;
    return v ? ff::set_error(FF_ERR_DEVICE_CHECK, "device status 0x%x", v) : FF_OK;
}

}  // extern "C"

// ------------------------------------------------------------------ timing
namespace ff {
namespace {
struct ProfRecord {
    char name[48];
    double flops, bytes;
};
std::mutex g_prof_mu;
bool g_prof_on = false;
int g_prof_cap = 0;
int g_prof_n = 0;
cudaEvent_t* g_prof_ev = nullptr;   // 2 per record
ProfRecord* g_prof_rec = nullptr;

void prof_free() {
    if (g_prof_ev) {
        for (int i = 0; i < 2 * g_prof_cap; ++i) cudaEventDestroy(g_prof_ev[i]);
        delete[] g_prof_ev;
        delete[] g_prof_rec;
    }
    g_prof_ev = nullptr;
    g_prof_rec = nullptr;
    g_prof_cap = g_prof_n = 0;
    g_prof_on = false;
}
}  // namespace

ProfScope::ProfScope(cudaStream_t s, const char* name, double flops, double bytes) : slot(-1), stream(s) {
    if (!g_prof_on) return;
    std::lock_guard<std::mutex> lk(g_prof_mu);
    if (!g_prof_on || g_prof_n >= g_prof_cap) return;
    slot = g_prof_n++;
    snprintf(g_prof_rec[slot].name, sizeof(g_prof_rec[slot].name), "%s", name);
    g_prof_rec[slot].flops = flops;
    g_prof_rec[slot].bytes = bytes;
    cudaEventRecord(g_prof_ev[2 * slot], s);
}

ProfScope::~ProfScope() {
    if (slot >= 0) cudaEventRecord(g_prof_ev[2 * slot + 1], stream);
}

}  // namespace ff

extern "C" {

int ff_prof_enable(int max_records) {
    using namespace ff;
    if (max_records <= 0) return set_error(FF_ERR_INVALID_ARG, "max_records must be positive");
    std::lock_guard<std::mutex> lk(g_prof_mu);
    prof_free();
    g_prof_ev = new cudaEvent_t[2 * max_records];
    g_prof_rec = new ProfRecord[max_records];
    for (int i = 0; i < 2 * max_records; ++i) {
        if (cudaEventCreate(&g_prof_ev[i]) != cudaSuccess) {
            for (int j = 0; j < i; ++j) cudaEventDestroy(g_prof_ev[j]);
            delete[] g_prof_ev;
            delete[] g_prof_rec;
            g_prof_ev = nullptr;
            g_prof_rec = nullptr;
            return set_error(FF_ERR_CUDA, "cudaEventCreate failed");
        }
    }
    g_prof_cap = max_records;
    g_prof_n = 0;
    g_prof_on = true;
    return FF_OK;
}

int ff_prof_disable(void) {
    std::lock_guard<std::mutex> lk(ff::g_prof_mu);
    ff::g_prof_on = false;
    return FF_OK;
}

int ff_prof_reset(void) {
    std::lock_guard<std::mutex> lk(ff::g_prof_mu);
    ff::g_prof_n = 0;
    return FF_OK;
}

int ff_prof_count(int* n) {
    if (!n) return ff::set_error(FF_ERR_INVALID_ARG, "n is null");
    *n = ff::g_prof_n;
    return FF_OK;
}

int ff_prof_read(int i, char* name, int name_cap, float* ms, double* flops, double* bytes) {
    using namespace ff;
    if (i < 0 || i >= g_prof_n || !ms) return set_error(FF_ERR_INVALID_ARG, "record %d out of range", i);
    if (cudaEventSynchronize(g_prof_ev[2 * i + 1]) != cudaSuccess ||
        cudaEventElapsedTime(ms, g_prof_ev[2 * i], g_prof_ev[2 * i + 1]) != cudaSuccess)
        return set_error(FF_ERR_CUDA, "event timing failed for record %d", i);
    if (name && name_cap > 0) snprintf(name, name_cap, "%s", g_prof_rec[i].name);
    if (flops) *flops = g_prof_rec[i].flops;
    if (bytes) *bytes = g_prof_rec[i].bytes;
    return FF_OK;
}

}  // extern "C"
