// C ABI of the library: argument validation, workspace planning, dispatch.
// Declarations and the contract of every entry point: include/tla.h.
#include <string.h>

#include <algorithm>
#include <mutex>
#include <vector>

#include "common.cuh"
#include "internal.h"
#include "sm100.cuh"

namespace tla {

// Device error word for bounded waits (first failure wins; cleared on read).
__device__ int g_device_error = 0;

static size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

static bool aligned16(const void* x) { return ((uintptr_t)x & 15) == 0; }

static bool dims_ok(int d) { return d >= 16 && d <= 128 && d % 16 == 0; }

static tla_status validate(const tla_problem* p) {
    if (!p) return TLA_ERR_INVALID_ARG;
    if (p->B < 1 || p->T < 1 || p->H < 1 || p->E < 1) return TLA_ERR_INVALID_ARG;
    if (p->dtype != TLA_BF16 && p->dtype != TLA_FP32) return TLA_ERR_INVALID_ARG;
    if (p->out_dtype != TLA_BF16 && p->out_dtype != TLA_FP32) return TLA_ERR_INVALID_ARG;
    if (p->use_delta != 0 && p->use_delta != 1) return TLA_ERR_INVALID_ARG;
    if (!p->q || !p->k || !p->v || !p->q2 || !p->k2 || !p->g || !p->o) return TLA_ERR_INVALID_ARG;
    if (p->use_delta && !p->beta) return TLA_ERR_INVALID_ARG;
    if (p->chunk != kChunk) return TLA_ERR_UNSUPPORTED;
    if (!dims_ok(p->dk) || !dims_ok(p->dv) || p->E > 32) return TLA_ERR_UNSUPPORTED;
    if (p->E > 16 && p->dk > 64) return TLA_ERR_UNSUPPORTED;   // shared-memory state slab
    if (p->gate_per_head != 0 && p->gate_per_head != 1) return TLA_ERR_INVALID_ARG;
    if (p->H > 65535 || p->B > 65535) return TLA_ERR_UNSUPPORTED;
    const void* ptrs[] = {p->q, p->k, p->v, p->q2, p->k2, p->g, p->beta, p->h0, p->o, p->ht};
    for (const void* x : ptrs)
        if (!aligned16(x)) return TLA_ERR_INVALID_ARG;
    if (p->cu_seqlens) {   // packed documents: B = 1, offsets 0 = cu[0] <= ... <= cu[n_docs] = T
        if (p->B != 1 || p->n_docs < 1) return TLA_ERR_INVALID_ARG;
        if (p->n_docs > 65535) return TLA_ERR_UNSUPPORTED;
        if (p->cu_seqlens[0] != 0 || p->cu_seqlens[p->n_docs] != p->T) return TLA_ERR_INVALID_ARG;
        for (int d = 0; d < p->n_docs; ++d)
            if (p->cu_seqlens[d + 1] < p->cu_seqlens[d]) return TLA_ERR_INVALID_ARG;
    }
    return TLA_OK;
}


// Waits on a barrier that nothing arrives at: the bounded wait must give up after
// timeout_ns and leave its record in the error word.
static __global__ void selftest_wait_kernel(unsigned long long timeout_ns, int* err) {
    __shared__ __align__(8) uint64_t bar;
    if (threadIdx.x == 0) {
        sm100::mbar_init(&bar, 1);
        sm100::fence_barrier_init();
    }
    __syncthreads();
    const bool ok = sm100::mbar_wait(&bar, 0, timeout_ns);
    if (!ok && threadIdx.x == 0) record_device_error(err, TLA_ERR_TIMEOUT);
}

// Address of the error word on the current device, looked up once per device (a
// std::once_flag per device orders concurrent first calls); nullptr if the lookup
// failed, which every entry point reports as TLA_ERR_CUDA before launching anything.
constexpr int kMaxDevices = 64;
int* device_error_word() {
    static std::once_flag once[kMaxDevices];
    static int* ptr[kMaxDevices] = {nullptr};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
    std::call_once(once[dev], [dev]() {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_device_error) == cudaSuccess) ptr[dev] = (int*)p;
    });
    return ptr[dev];
}

// Value columns per CTA of the SIMT recurrences: the E x dk x tv fp32 slab
// stays within 64 KiB of shared memory.
static int simt_tv(const tla_problem& p) {
    for (int tv = 32; tv >= 8; tv >>= 1)
        if (p.dv % tv == 0 && (size_t)p.E * p.dk * tv * 4 <= 65536) return tv;
    return 8;
}

int chunk_count(const tla_problem& p) {
    if (!p.cu_seqlens) return (p.T + kChunk - 1) / kChunk;
    long long nc = 0;
    for (int d = 0; d < p.n_docs; ++d)
        nc += (p.cu_seqlens[d + 1] - p.cu_seqlens[d] + kChunk - 1) / kChunk;
    return (int)nc;
}

FwdPlan plan_fwd(const tla_problem& p, int save) {
    FwdPlan f;
    memset(&f, 0, sizeof(f));
    f.NT = chunk_count(p);
    f.nseq = p.cu_seqlens ? p.n_docs : p.B;
    f.tv = simt_tv(p);
    f.tc_tv = tc_fwd_tv(p);   // layout depends on shapes only
    const size_t tokE = (size_t)p.B * p.T * p.H * p.E * 4;
    const size_t mats = (size_t)p.B * p.H * f.NT * kChunk * kChunk * 4;
    const size_t tokV = (size_t)p.B * f.NT * kChunk * p.H * p.dv * 4;   // whole chunks (token tiles)
    size_t off = 0;
    f.G = off; off = align256(off + tokE);
    f.A = off; off = align256(off + mats);
    if (p.use_delta) { f.N = off; off = align256(off + mats); }
    if (f.tc_tv) {
        f.A2 = off; off = align256(off + 2 * mats);   // hi + lo 128 x 64 bf16 tiles
        f.coef = off;
        off = align256(off + (size_t)p.B * p.H * f.NT * (3 * kChunk * p.E + 16) * 4);
        f.tcb = (save && tc_bwd_ok(p, f.tc_tv)) ? 1 : 0;
        f.ck_tiles = (f.tcb && tc_grads_shape_ok(p)) ? 1 : 0;
        if (f.tcb) { f.BT = off; off = align256(off + 2 * mats); }
    }
    // A feeds the CUDA-core recurrences only: the forward without tensor cores, or the
    // backward recurrence when it cannot run on tensor cores
    f.need_A = (!f.tc_tv || (save && !f.tcb)) ? 1 : 0;
    if (save) {   // tile checkpoints keep 128 key rows (zero past d_k = 64)
        const size_t states = (size_t)p.B * p.H * f.NT * p.E * (f.ck_tiles ? 128 : p.dk) * p.dv * 4;
        f.S = off; off = align256(off + states);
        f.U = off; off = align256(off + tokV);
        if (p.use_delta || f.ck_tiles) { f.Res = off; off = align256(off + tokV); }
    }
    if (p.cu_seqlens) {
        f.ctab = off; off = align256(off + (size_t)f.NT * sizeof(int2));
        f.dtab = off; off = align256(off + (size_t)p.n_docs * sizeof(int4));
    }
    f.bytes = off;
    return f;
}

BwdPlan plan_bwd(const tla_problem& p) {
    BwdPlan b;
    memset(&b, 0, sizeof(b));
    const int NT = chunk_count(p);
    b.tv = simt_tv(p);
    const size_t tokV = (size_t)p.B * NT * kChunk * p.H * p.dv * 4;   // whole chunks (token tiles)
    // tile checkpoints (the forward plan's choice) keep 128 key rows (zero past d_k = 64)
    const int ck_rows = plan_fwd(p, 1).ck_tiles ? 128 : p.dk;
    const size_t states = (size_t)p.B * p.H * NT * p.E * ck_rows * p.dv * 4;
    size_t off = 0;
    b.dU = off; off = align256(off + tokV);
    b.dRes = off; off = align256(off + tokV);
    b.dS = off; off = align256(off + states);
    if (p.gate_per_head) { b.dgE = off; off = align256(off + (size_t)p.B * p.T * p.H * p.E * 4); }
    if (p.E > 8 && tc_grads_ok(p, plan_fwd(p, 1))) {
        b.gscr = off;
        off = align256(off + (size_t)p.B * p.H * NT * 3 * kChunk * p.E * 4);
    }
    b.bytes = off;
    return b;
}

static tla_status cuda_status(cudaError_t e) { return e == cudaSuccess ? TLA_OK : TLA_ERR_CUDA; }


// ---- kernel timing: a pool of event pairs, one per launch while enabled
struct ProfRecord {
    const char* name;
    cudaEvent_t a, b;
};
static std::mutex g_prof_mu;
static bool g_prof_on = false;
static std::vector<ProfRecord> g_prof;   // records of the current session
static std::vector<cudaEvent_t> g_pool;  // reusable events
static size_t g_pool_next = 0;

static cudaEvent_t pool_event() {
    if (g_pool_next == g_pool.size()) {
        cudaEvent_t e = nullptr;
        if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
        g_pool.push_back(e);
    }
    return g_pool[g_pool_next++];
}

void prof_before(const char* name, cudaStream_t s) {
    std::lock_guard<std::mutex> lk(g_prof_mu);
    if (!g_prof_on) return;
    ProfRecord r{name, pool_event(), pool_event()};
    if (!r.a || !r.b) return;
    cudaEventRecord(r.a, s);
    g_prof.push_back(r);
}

void prof_after(cudaStream_t s) {
    std::lock_guard<std::mutex> lk(g_prof_mu);
    if (!g_prof_on || g_prof.empty()) return;
    cudaEventRecord(g_prof.back().b, s);
}

}  // namespace tla

using namespace tla;

extern "C" {

size_t tla_fwd_workspace_bytes(const tla_problem* p, int save_for_bwd) {
    if (validate(p) != TLA_OK) return 0;
    return plan_fwd(*p, save_for_bwd ? 1 : 0).bytes;
}

size_t tla_bwd_workspace_bytes(const tla_problem* p) {
    if (validate(p) != TLA_OK) return 0;
    return plan_bwd(*p).bytes;
}

tla_status tla_chunk_fwd(const tla_problem* p, void* workspace, size_t workspace_bytes,
                         int save_for_bwd, void* stream) {
    tla_status st = validate(p);
    if (st != TLA_OK) return st;
    const int save = save_for_bwd ? 1 : 0;
    FwdPlan fp = plan_fwd(*p, save);
    if (!workspace || workspace_bytes < fp.bytes || ((uintptr_t)workspace & 255))
        return TLA_ERR_WORKSPACE;
    if (p->cu_seqlens && !fp.tc_tv) return TLA_ERR_UNSUPPORTED;   // packed: tensor-core path only
    int* err = device_error_word();
    if (!err) return TLA_ERR_CUDA;
    cudaStream_t s = (cudaStream_t)stream;
    char* ws = (char*)workspace;
    if (p->cu_seqlens) {   // packed documents: chunk and document tables
        std::vector<int2> ct(fp.NT);
        std::vector<int4> dt(p->n_docs);
        int g = 0;
        for (int d = 0; d < p->n_docs; ++d) {
            const int t0 = p->cu_seqlens[d], len = p->cu_seqlens[d + 1] - t0;
            const int nc = (len + kChunk - 1) / kChunk;
            dt[d] = make_int4(t0, nc, g, len);
            for (int c = 0; c < nc; ++c) ct[g++] = make_int2(t0 + c * kChunk, std::min(kChunk, len - c * kChunk));
        }
        cudaError_t ce = cudaMemcpyAsync(ws + fp.ctab, ct.data(), ct.size() * sizeof(int2),
                                         cudaMemcpyHostToDevice, s);
        if (ce == cudaSuccess)
            ce = cudaMemcpyAsync(ws + fp.dtab, dt.data(), dt.size() * sizeof(int4),
                                 cudaMemcpyHostToDevice, s);
        if (ce != cudaSuccess) return TLA_ERR_CUDA;
    }
    cudaError_t e = launch_gate_cumsum(*p, fp, ws, (float*)(ws + fp.G), s);
    if (e == cudaSuccess) {
        if (fp.tc_tv)
            e = launch_chunk_prep_tc(*p, fp, ws, err, s);
        else
            e = launch_chunk_prep(*p, (const float*)(ws + fp.G), (float*)(ws + fp.A),
                                  p->use_delta ? (float*)(ws + fp.N) : nullptr, s);
    }
    if (e == cudaSuccess) {
        if (fp.tc_tv)
            e = launch_fwd_recurrence_tc(*p, fp, ws, save, err, s);
        else e = launch_fwd_recurrence(*p, fp, ws, save, s);
    }
    return cuda_status(e);
}

tla_status tla_chunk_bwd(const tla_problem* p, const void* fwd_ws, size_t fwd_ws_bytes,
                         const void* dO, const float* dht, void* dq, void* dk, void* dv,
                         void* dq2, void* dk2, float* dbeta, float* dg, float* dh0,
                         void* workspace, size_t workspace_bytes, void* stream) {
    tla_status st = validate(p);
    if (st != TLA_OK) return st;
    if (!dO || !dq || !dk || !dv || !dq2 || !dk2 || !dg) return TLA_ERR_INVALID_ARG;
    {
        const void* ptrs[] = {dO, dht, dq, dk, dv, dq2, dk2, dbeta, dg, dh0};
        for (const void* x : ptrs)
            if (!aligned16(x)) return TLA_ERR_INVALID_ARG;
    }
    if ((p->beta != nullptr) != (dbeta != nullptr)) return TLA_ERR_INVALID_ARG;
    if ((p->h0 != nullptr) != (dh0 != nullptr)) return TLA_ERR_INVALID_ARG;
    FwdPlan fp = plan_fwd(*p, 1);
    BwdPlan bp = plan_bwd(*p);
    if (p->cu_seqlens && !(fp.tcb && tc_grads_ok(*p, fp))) return TLA_ERR_UNSUPPORTED;
    if (!fwd_ws || fwd_ws_bytes < fp.bytes || ((uintptr_t)fwd_ws & 255)) return TLA_ERR_WORKSPACE;
    if (!workspace || workspace_bytes < bp.bytes || ((uintptr_t)workspace & 255))
        return TLA_ERR_WORKSPACE;
    int* err = device_error_word();
    if (!err) return TLA_ERR_CUDA;
    cudaStream_t s = (cudaStream_t)stream;
    const char* fws = (const char*)fwd_ws;
    char* bws = (char*)workspace;
    float* dgs = p->gate_per_head ? (float*)(bws + bp.dgE) : dg;   // per-slice gate gradient
    cudaError_t e = fp.tcb ? launch_bwd_recurrence_tc(*p, fp, fws, bp, bws, dO, dht, dv, dh0,
                                                      err, s)
                           : launch_bwd_recurrence(*p, fp, fws, bp, bws, dO, dht, dv, dh0, s);
    if (e == cudaSuccess) {
        if (tc_grads_ok(*p, fp))
            e = launch_bwd_chunk_grads_tc(*p, fp, fws, bp, bws, dO, dq, dk, dq2, dk2, dbeta, dgs,
                                          err, s);
        else
            e = launch_bwd_chunk_grads(*p, fp, fws, bp, bws, dO, dq, dk, dq2, dk2, dbeta, dgs, s);
    }
    if (e == cudaSuccess && p->gate_per_head)
        e = launch_sum_slices(dgs, dg, (long long)p->B * p->T * p->H, p->E, s);
    return cuda_status(e);
}

tla_status tla_decode_step(int B, int H, int dk, int dv, int E, int use_delta, int dtype,
                           const void* q, const void* k, const void* v, const void* q2,
                           const void* k2, const float* g, const float* beta, float* state,
                           void* o, void* stream) {
    if (B < 1 || H < 1 || E < 1) return TLA_ERR_INVALID_ARG;
    if (dtype != TLA_BF16 && dtype != TLA_FP32) return TLA_ERR_INVALID_ARG;
    if (use_delta != 0 && use_delta != 1) return TLA_ERR_INVALID_ARG;
    if (!q || !k || !v || !q2 || !k2 || !g || !state || !o) return TLA_ERR_INVALID_ARG;
    if (use_delta && !beta) return TLA_ERR_INVALID_ARG;
    {
        const void* ptrs[] = {q, k, v, q2, k2, g, beta, state, o};
        for (const void* x : ptrs)
            if (!aligned16(x)) return TLA_ERR_INVALID_ARG;
    }
    if (!dims_ok(dk) || !dims_ok(dv) || E > 32 || E * dk > 2048) return TLA_ERR_UNSUPPORTED;
    if ((long long)B * H > 65535) return TLA_ERR_UNSUPPORTED;  // grid.y
    int* err = device_error_word();
    if (!err) return TLA_ERR_CUDA;
    return cuda_status(launch_decode_step(B, H, dk, dv, E, use_delta, dtype, q, k, v, q2, k2, g,
                                          beta, state, o, err, (cudaStream_t)stream));
}

const char* tla_status_string(int status) {
    switch (status) {
        case TLA_OK: return "TLA_OK";
        case TLA_ERR_INVALID_ARG: return "TLA_ERR_INVALID_ARG";
        case TLA_ERR_UNSUPPORTED: return "TLA_ERR_UNSUPPORTED";
        case TLA_ERR_CUDA: return "TLA_ERR_CUDA";
        case TLA_ERR_TIMEOUT: return "TLA_ERR_TIMEOUT";
        case TLA_ERR_WORKSPACE: return "TLA_ERR_WORKSPACE";
        default: return "TLA_UNKNOWN_STATUS";
    }
}

tla_status tla_selftest_bounded_wait(unsigned long long timeout_ns, void* stream) {
    if (timeout_ns < 1 || timeout_ns > 1000000000ull) return TLA_ERR_INVALID_ARG;
    int* err = device_error_word();
    if (!err) return TLA_ERR_CUDA;
    selftest_wait_kernel<<<1, 32, 0, (cudaStream_t)stream>>>(timeout_ns, err);
    return cudaGetLastError() == cudaSuccess ? TLA_OK : TLA_ERR_CUDA;
}

tla_status tla_last_device_status(void* stream) {
    cudaStream_t s = (cudaStream_t)stream;
    if (cudaStreamSynchronize(s) != cudaSuccess) return TLA_ERR_CUDA;
    int word = 0;
    if (cudaMemcpyFromSymbol(&word, g_device_error, sizeof(int)) != cudaSuccess) return TLA_ERR_CUDA;
    if (word != 0) {
        const int zero = 0;
        if (cudaMemcpyToSymbol(g_device_error, &zero, sizeof(int)) != cudaSuccess) return TLA_ERR_CUDA;
        return TLA_ERR_TIMEOUT;
    }
    return TLA_OK;
}

tla_status tla_profile_begin(void) {
    std::lock_guard<std::mutex> lk(g_prof_mu);
    g_prof.clear();
    g_pool_next = 0;
    g_prof_on = true;
    return TLA_OK;
}

int tla_profile_end(void* stream, char* names_out, int* launches_out, float* ms_out,
                    int max_kernels) {
    if (cudaStreamSynchronize((cudaStream_t)stream) != cudaSuccess) return TLA_ERR_CUDA;
    std::lock_guard<std::mutex> lk(g_prof_mu);
    g_prof_on = false;
    if (cudaDeviceSynchronize() != cudaSuccess) return TLA_ERR_CUDA;
    int nk = 0;
    std::vector<const char*> names;
    std::vector<int> cnt;
    std::vector<double> ms;
    for (const ProfRecord& r : g_prof) {
        float t = 0.f;
        if (cudaEventElapsedTime(&t, r.a, r.b) != cudaSuccess) return TLA_ERR_CUDA;
        int i = 0;
        while (i < nk && strcmp(names[i], r.name) != 0) ++i;
        if (i == nk) {
            names.push_back(r.name);
            cnt.push_back(0);
            ms.push_back(0.0);
            ++nk;
        }
        cnt[i] += 1;
        ms[i] += t;
    }
    g_prof.clear();
    int n = nk < max_kernels ? nk : max_kernels;
    for (int i = 0; i < n; ++i) {
        if (names_out) {
            strncpy(names_out + 64 * i, names[i], 63);
            names_out[64 * i + 63] = 0;
        }
        if (launches_out) launches_out[i] = cnt[i];
        if (ms_out) ms_out[i] = (float)ms[i];
    }
    return n;
}

const char* tla_version(void) { return "tla 0.1 sm_103a"; }

}  // extern "C"
