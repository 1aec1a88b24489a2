// C ABI of the SDM hot path: argument validation, workspace layout, kernel launches.
// Declarations and semantics: include/sdm.h.
#include "sdm_internal.h"
#include "sdm.h"

#include <stdarg.h>
#include <stdio.h>
#include <stddef.h>
#include <string.h>

#include <atomic>
#include <mutex>
#include <string>

static_assert(sizeof(sdm_shape) == 48, "sdm_shape layout is part of the ABI");
static_assert(offsetof(sdm_shape, N) == 24, "sdm_shape layout is part of the ABI");

namespace {

thread_local std::string g_last_error;

sdm_status fail(sdm_status st, const char* fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof(buf), fmt, ap);
    va_end(ap);
    g_last_error = buf;
    return st;
}

sdm_status ok() {
    g_last_error.clear();
    return SDM_OK;
}

sdm_status cuda_fail(cudaError_t e, const char* where) {
    return fail(SDM_ERR_CUDA, "%s: %s (%s)", where, cudaGetErrorString(e), cudaGetErrorName(e));
}

// Device status word followed by event counters (index 1..), one array per device; its
// address is looked up once per device.
__device__ int g_status_word[16];
constexpr int kMaxDevices = 64;
std::atomic<int*> g_status_addr[kMaxDevices];

sdm_status status_word(int** out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    if (dev < 0 || dev >= kMaxDevices) return fail(SDM_ERR_UNSUPPORTED, "device ordinal %d >= %d", dev, kMaxDevices);
    int* p = g_status_addr[dev].load(std::memory_order_acquire);
    if (p == nullptr) {
        e = cudaGetSymbolAddress(reinterpret_cast<void**>(&p), g_status_word);
        if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress(status word)");
        g_status_addr[dev].store(p, std::memory_order_release);
    }
    *out = p;
    return SDM_OK;
}

// Per-device side stream and fork/join events for the M0 broadcast that overlaps the
// addressing in sdm_forward_m0 (created on first use; the mutex orders the host-side
// enqueue of fork/join sequences from concurrent callers).
struct SideStream {
    cudaStream_t stream = nullptr;
    cudaEvent_t fork = nullptr, join = nullptr;
};
SideStream g_side[kMaxDevices];
std::mutex g_side_mutex[kMaxDevices];

sdm_status side_stream(int* dev_out, SideStream** out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    if (dev < 0 || dev >= kMaxDevices) return fail(SDM_ERR_UNSUPPORTED, "device ordinal %d >= %d", dev, kMaxDevices);
    SideStream& ss = g_side[dev];
    if (ss.stream == nullptr) {
        e = cudaStreamCreateWithFlags(&ss.stream, cudaStreamNonBlocking);
        if (e == cudaSuccess) e = cudaEventCreateWithFlags(&ss.fork, cudaEventDisableTiming);
        if (e == cudaSuccess) e = cudaEventCreateWithFlags(&ss.join, cudaEventDisableTiming);
        if (e != cudaSuccess) {
            ss = SideStream{};
            return cuda_fail(e, "side stream creation");
        }
    }
    *dev_out = dev;
    *out = &ss;
    return SDM_OK;
}

int64_t isqrt64(int64_t n) {
    if (n < 0) return -1;
    int64_t r = 0;
    while ((r + 1) * (r + 1) <= n) {
        int64_t step = 1;
        while ((r + 2 * step) * (r + 2 * step) <= n) step *= 2;
        r += step;
    }
    return r;
}

size_t elem_bytes(int dtype) { return dtype == SDM_F32 ? 4 : 2; }

size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

struct Range {
    const void* p;
    size_t n;
    const char* name;
};

bool overlaps(const Range& a, const Range& b) {
    if (!a.p || !b.p || !a.n || !b.n) return false;
    const uintptr_t a0 = reinterpret_cast<uintptr_t>(a.p), b0 = reinterpret_cast<uintptr_t>(b.p);
    return a0 < b0 + b.n && b0 < a0 + a.n;
}

// Common shape checks.  need_pkm: the call runs PKM addressing (N square, k <= sqrt(N), d_k bounds).
sdm_status check_shape(const sdm_shape* s, bool need_pkm, int64_t* S_out) {
    if (!s) return fail(SDM_ERR_INVALID_ARG, "shape is NULL");
    if (s->B < 0 || s->H < 0 || s->T < 0) return fail(SDM_ERR_INVALID_ARG, "B, H, T must be >= 0 (got %d, %d, %d)", s->B, s->H, s->T);
    if (s->dtype != SDM_F32 && s->dtype != SDM_BF16) return fail(SDM_ERR_INVALID_ARG, "unknown dtype %d", s->dtype);
    if (s->N < 1 || s->N > INT32_MAX) return fail(SDM_ERR_INVALID_ARG, "N must be in [1, 2^31-1] (got %lld)", (long long)s->N);
    if (s->d_v < 1) return fail(SDM_ERR_INVALID_ARG, "d_v must be >= 1 (got %d)", s->d_v);
    if ((static_cast<size_t>(s->d_v) * elem_bytes(s->dtype)) % 16 != 0)
        return fail(SDM_ERR_UNSUPPORTED, "d_v * element size must be a multiple of 16 bytes (d_v=%d)", s->d_v);
    if (s->k_write < 1 || s->k_read < 1 || s->k_write > 64 || s->k_read > 64)
        return fail(SDM_ERR_UNSUPPORTED, "k_write and k_read must be in [1, 64] (got %d, %d)", s->k_write, s->k_read);
    if (s->k_write > s->N || s->k_read > s->N) return fail(SDM_ERR_INVALID_ARG, "k exceeds N");
    if (need_pkm) {
        const int64_t S = isqrt64(s->N);
        if (S * S != s->N) return fail(SDM_ERR_INVALID_ARG, "N=%lld is not a perfect square", (long long)s->N);
        if (S > 46340) return fail(SDM_ERR_UNSUPPORTED, "sqrt(N) too large");
        if (s->k_write > S || s->k_read > S)
            return fail(SDM_ERR_INVALID_ARG, "k_write, k_read must be <= sqrt(N)=%lld", (long long)S);
        if (s->addr != SDM_ADDR_PROJECTED && s->addr != SDM_ADDR_DIRECT) return fail(SDM_ERR_INVALID_ARG, "unknown addr mode %d", s->addr);
        if (s->d_k < 1) return fail(SDM_ERR_INVALID_ARG, "d_k must be >= 1");
        if (s->addr == SDM_ADDR_DIRECT && s->d_k != 2 * S)
            return fail(SDM_ERR_INVALID_ARG, "DIRECT addressing needs d_k == 2*sqrt(N) (d_k=%d, sqrt(N)=%lld)", s->d_k, (long long)S);
        if (s->d_k > 256) return fail(SDM_ERR_UNSUPPORTED, "d_k > 256 is not supported");
        if (S_out) *S_out = S;
    }
    return SDM_OK;
}

struct Layout {
    size_t idx_w, w_w, idx_r, w_r, pnorm, part_v, part_i, queue, hz, firstw, total;
    sdm::AddrPlan plan;
};

// lazy: also the first-writer table of the copy-on-write initial memory ([B*H, N] int32).
Layout layout_for(const sdm_shape* s, int64_t S, bool lazy = false) {
    Layout L{};
    const size_t bht = static_cast<size_t>(s->B) * s->H * s->T;
    const int kmax = s->k_write > s->k_read ? s->k_write : s->k_read;
    L.plan = sdm::addr_plan(s->dtype, s->addr == SDM_ADDR_DIRECT, s->B, s->H, s->T, s->d_k, static_cast<int>(S), kmax);
    size_t off = 0;
    L.idx_w = off; off = align256(off + bht * s->k_write * 4);
    L.w_w = off;   off = align256(off + bht * s->k_write * 4);
    L.idx_r = off; off = align256(off + bht * s->k_read * 4);
    L.w_r = off;   off = align256(off + bht * s->k_read * 4);
    L.pnorm = off; off = align256(off + 2 * static_cast<size_t>(s->H) * 4);
    const size_t part = sdm::addr_partial_bytes(L.plan, s->B, s->H, s->T) / 2;
    L.part_v = off; off = align256(off + part);
    L.part_i = off; off = align256(off + part);
    L.queue = off;  off = align256(off + sdm::addr_queue_bytes(s->B, s->H, s->T));
    L.hz = off;     off = align256(off + sdm::rec_workspace_bytes(s->B, s->H, s->T, s->k_write, s->k_read));
    L.firstw = off;
    if (lazy) off = align256(off + static_cast<size_t>(s->B) * s->H * static_cast<size_t>(s->N) * 4);
    L.total = off;
    return L;
}

// |fp32 score - float64 score| <= c * sum_d |P_jd x_d| <= c * max_j ||P_j|| * ||x||.
//   FFMA path (sequential fp32 fused multiply-adds in d order): c = (d_k + 4) 2^-24, the
//   classical gamma_{d_k} bound with the float64 reference's own rounding as margin.
//   Tensor cores (tcgen05.mma kind::f16, bf16 operands, fp32 accumulation, K = 16 per
//   instruction): every product of two bf16 numbers is exact in fp32.  One instruction adds
//   16 products to the accumulator D; modelling it as an alignment of the 17 terms to the
//   largest exponent e with at least 24 significant bits kept (each term off by less than
//   2^(e-23) <= 2^-23 max|term|) and a rounding or truncation of the result to fp32 (off by
//   at most 2^-23 |D'|) bounds its error by 18 * 2^-23 (|D| + sum of the block's |products|).
//   |D| before block i is at most the sum of the earlier blocks' |products|, so over the
//   d_k / 16 instructions the error is at most 18 (d_k / 16) 2^-23 sum_d |P_jd x_d|, plus
//   2^-40 of slack for the float64 reference (d_k 2^-53).  The model allows more error than
//   round-to-nearest accumulation could make; the GPU test of the raw scores checks it.
double score_bound_constant(int dk, bool mma) {
    if (!mma) return (dk + 4) * 0x1p-24;
    return 18.0 * ((dk + 15) / 16) * 0x1p-23 + 0x1p-40;
}

// Addressing into the given (or workspace) index/weight buffers.
sdm_status run_address(const sdm_shape* s, int64_t S, const Layout& L, const void* P_q, const void* P_k, const void* q,
                       const void* k, int32_t* idx_w, float* w_w, int32_t* idx_r, float* w_r, char* ws,
                       int* err, cudaStream_t stream) {
    sdm::AddrArgs a{};
    const bool direct = s->addr == SDM_ADDR_DIRECT;
    a.P[0] = direct ? nullptr : P_q;
    a.P[1] = direct ? nullptr : P_k;
    a.X[0] = q;
    a.X[1] = k;
    a.idx[0] = idx_r; a.w[0] = w_r; a.kk[0] = s->k_read;
    a.idx[1] = idx_w; a.w[1] = w_w; a.kk[1] = s->k_write;
    a.B = s->B; a.H = s->H; a.T = s->T; a.dk = s->d_k; a.S = static_cast<int>(S);
    a.ncc = L.plan.ncc;
    a.cw = L.plan.cw;
    a.cbound = static_cast<float>(score_bound_constant(s->d_k, L.plan.mma));
    a.part_v = reinterpret_cast<float*>(ws + L.part_v);
    a.part_i = reinterpret_cast<int*>(ws + L.part_i);
    a.pnorm = reinterpret_cast<float*>(ws + L.pnorm);
    a.queue = sdm::addr_queue_bytes(s->B, s->H, s->T) ? reinterpret_cast<int*>(ws + L.queue) : nullptr;
    a.err = err;
    cudaError_t e = sdm::launch_address(s->dtype, L.plan, a, stream);
    if (e != cudaSuccess) return cuda_fail(e, "addressing launch");
    return SDM_OK;
}

sdm_status check_vec(const void* p, const char* name, size_t align) {
    if (!p) return fail(SDM_ERR_INVALID_ARG, "%s is NULL", name);
    if (!aligned(p, align)) return fail(SDM_ERR_INVALID_ARG, "%s is not %zu-byte aligned", name, align);
    return SDM_OK;
}

#define SDM_TRY(expr)                  \
    do {                               \
        sdm_status _st = (expr);       \
        if (_st != SDM_OK) return _st; \
    } while (0)

// Copy-on-write initial memory (sdm_forward_lazy): M0 and the chains' touched bitmaps.
struct LazyIn {
    const void* M0;
    uint32_t* touched;
};

sdm_status forward_impl(const char* who, const sdm_shape* s, const void* P_q, const void* P_k, const void* q,
                        const void* k, const void* v, const void* alpha, const void* beta, void* mem, void* y,
                        int32_t* idx_w, float* w_w, int32_t* idx_r, float* w_r, void* workspace,
                        size_t workspace_bytes, cudaStream_t stream, bool run_recurrence, const void* M0 = nullptr,
                        const LazyIn* lazy = nullptr) {
    int64_t S = 0;
    SDM_TRY(check_shape(s, true, &S));
    const size_t es = elem_bytes(s->dtype);
    const size_t bht = static_cast<size_t>(s->B) * s->H * s->T;
    if (bht == 0) return ok();
    if (s->addr == SDM_ADDR_PROJECTED) {
        SDM_TRY(check_vec(P_q, "P_q", es));
        SDM_TRY(check_vec(P_k, "P_k", es));
    }
    SDM_TRY(check_vec(q, "q", es));
    SDM_TRY(check_vec(k, "k", es));
    if (run_recurrence) {
        SDM_TRY(check_vec(v, "v", 16));
        SDM_TRY(check_vec(alpha, "alpha", es));
        SDM_TRY(check_vec(beta, "beta", es));
        SDM_TRY(check_vec(mem, "mem", 16));
        SDM_TRY(check_vec(y, "y", 16));
    } else {
        SDM_TRY(check_vec(idx_w, "idx_w", 4));
        SDM_TRY(check_vec(w_w, "w_w", 4));
        SDM_TRY(check_vec(idx_r, "idx_r", 4));
        SDM_TRY(check_vec(w_r, "w_r", 4));
    }
    const Layout L = layout_for(s, S, lazy != nullptr);
    if (!workspace) return fail(SDM_ERR_INVALID_ARG, "%s: workspace is NULL (need %zu bytes)", who, L.total);
    if (!aligned(workspace, 256)) return fail(SDM_ERR_INVALID_ARG, "%s: workspace must be 256-byte aligned", who);
    if (workspace_bytes < L.total)
        return fail(SDM_ERR_INVALID_ARG, "%s: workspace too small (%zu < %zu bytes)", who, workspace_bytes, L.total);
    const size_t rowb = static_cast<size_t>(s->d_v) * es;
    if (run_recurrence) {
        const Range rm{mem, static_cast<size_t>(s->B) * s->H * static_cast<size_t>(s->N) * rowb, "mem"};
        const Range others[] = {
            {P_q, s->addr == SDM_ADDR_PROJECTED ? static_cast<size_t>(s->H) * 2 * S * s->d_k * es : 0, "P_q"},
            {P_k, s->addr == SDM_ADDR_PROJECTED ? static_cast<size_t>(s->H) * 2 * S * s->d_k * es : 0, "P_k"},
            {q, bht * s->d_k * es, "q"}, {k, bht * s->d_k * es, "k"}, {v, bht * rowb, "v"},
            {alpha, bht * es, "alpha"}, {beta, bht * es, "beta"}, {y, bht * rowb, "y"},
            {idx_w, idx_w ? bht * s->k_write * 4 : 0, "idx_w"}, {w_w, w_w ? bht * s->k_write * 4 : 0, "w_w"},
            {idx_r, idx_r ? bht * s->k_read * 4 : 0, "idx_r"}, {w_r, w_r ? bht * s->k_read * 4 : 0, "w_r"},
            {workspace, L.total, "workspace"}};
        for (const Range& r : others)
            if (overlaps(rm, r)) return fail(SDM_ERR_INVALID_ARG, "%s: mem overlaps %s", who, r.name);
        const Range ry{y, bht * rowb, "y"};
        for (int i = 0; i < 7; ++i)
            if (overlaps(ry, others[i])) return fail(SDM_ERR_INVALID_ARG, "%s: y overlaps %s", who, others[i].name);
        if (M0 != nullptr) {
            SDM_TRY(check_vec(M0, "M0", 16));
            if (overlaps(rm, Range{M0, static_cast<size_t>(s->H) * static_cast<size_t>(s->N) * rowb, "M0"}))
                return fail(SDM_ERR_INVALID_ARG, "%s: mem overlaps M0", who);
        }
        if (lazy != nullptr) {
            SDM_TRY(check_vec(lazy->M0, "M0", 16));
            SDM_TRY(check_vec(lazy->touched, "touched", 4));
            const Range r0{lazy->M0, static_cast<size_t>(s->H) * static_cast<size_t>(s->N) * rowb, "M0"};
            const Range rt{lazy->touched, static_cast<size_t>(s->B) * s->H * static_cast<size_t>((s->N + 31) / 32) * 4,
                           "touched"};
            if (overlaps(rm, r0)) return fail(SDM_ERR_INVALID_ARG, "%s: mem overlaps M0", who);
            if (overlaps(rm, rt)) return fail(SDM_ERR_INVALID_ARG, "%s: mem overlaps touched", who);
            for (const Range& r : others)
                if (overlaps(rt, r)) return fail(SDM_ERR_INVALID_ARG, "%s: touched overlaps %s", who, r.name);
            if (overlaps(rt, r0)) return fail(SDM_ERR_INVALID_ARG, "%s: touched overlaps M0", who);
        }
    }
    char* ws = static_cast<char*>(workspace);
    int32_t* iw = idx_w ? idx_w : reinterpret_cast<int32_t*>(ws + L.idx_w);
    float* ww = w_w ? w_w : reinterpret_cast<float*>(ws + L.w_w);
    int32_t* ir = idx_r ? idx_r : reinterpret_cast<int32_t*>(ws + L.idx_r);
    float* wr = w_r ? w_r : reinterpret_cast<float*>(ws + L.w_r);
    int* err = nullptr;
    SDM_TRY(status_word(&err));
    std::unique_lock<std::mutex> side_lock;      // held until the recurrence has waited on the join
    cudaEvent_t mem_ready = nullptr;
    if (run_recurrence && M0 != nullptr) {
        // mem = M0 broadcast on the side stream, running beside the addressing (independent
        // data) and joined back before the recurrence.  The copy goes through the bulk-copy
        // engine from one thread per SM, so it takes almost nothing from the addressing
        // kernels (an SM-thread copy with one 256-thread CTA per SM measured 0.34 ms slower
        // per step at layer_1p4b; with more CTAs per SM, slower still).
        int dev = 0;
        SideStream* ss = nullptr;
        SDM_TRY(side_stream(&dev, &ss));
        side_lock = std::unique_lock<std::mutex>(g_side_mutex[dev]);
        cudaError_t e = cudaEventRecord(ss->fork, stream);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(ss->stream, ss->fork, 0);
        if (e == cudaSuccess)
            e = sdm::launch_init_bulk(M0, mem, static_cast<int64_t>(static_cast<size_t>(s->H) * s->N * rowb), s->B,
                                      err, ss->stream);
        if (e == cudaSuccess) e = cudaEventRecord(ss->join, ss->stream);
        if (e != cudaSuccess) return cuda_fail(e, "M0 broadcast on the side stream");
        SDM_TRY(run_address(s, S, L, P_q, P_k, q, k, iw, ww, ir, wr, ws, err, stream));
        mem_ready = ss->join;                     // joined after the hazard pass, before the recurrence
    } else {
        SDM_TRY(run_address(s, S, L, P_q, P_k, q, k, iw, ww, ir, wr, ws, err, stream));
    }
    if (run_recurrence) {
        sdm::RecArgs r{};
        r.idx_w = iw; r.w_w = ww; r.idx_r = ir; r.w_r = wr;
        r.v = v; r.alpha = alpha; r.beta = beta; r.mem = mem; r.y = y;
        r.B = s->B; r.H = s->H; r.T = s->T; r.dv = s->d_v; r.kw = s->k_write; r.kr = s->k_read;
        r.N = s->N;
        r.err = err;
        int32_t* firstw = nullptr;
        if (lazy != nullptr) {
            // first writer of every slot in this call, then the chains' bitmaps for the next
            // call; the recurrence gathers rows nobody has written from M0
            firstw = reinterpret_cast<int32_t*>(ws + L.firstw);
            const int64_t chains = static_cast<int64_t>(s->B) * s->H;
            cudaError_t e = sdm::launch_lazy_prepare(lazy->touched, firstw, iw, chains, s->T, s->k_write, s->N, stream);
            if (e == cudaSuccess) e = sdm::launch_lazy_bitmap(firstw, lazy->touched, chains, s->N, stream);
            if (e != cudaSuccess) return cuda_fail(e, "lazy initial memory launch");
            r.M0 = lazy->M0;
        }
        cudaError_t e = sdm::launch_recur(s->dtype, r, reinterpret_cast<int32_t*>(ws + L.hz), stream, firstw, mem_ready);
        if (e != cudaSuccess) return cuda_fail(e, "recurrence launch");
    }
    return ok();
}

// sdm_recur with an optional undo log (defined after the C entry points).
sdm_status recur_impl(const char* who, const sdm_shape* s, const int32_t* idx_w, const float* w_w,
                      const int32_t* idx_r, const float* w_r, const void* v, const void* alpha, const void* beta,
                      void* mem, void* y, void* undo, void* workspace, size_t workspace_bytes, sdm_stream_t stream,
                      long long wait_cycles = 0, int hold_handover = 0);

// sdm_recur_backward over a stored log (kind 0) or a quantised snapshot (kind 1, 2).
sdm_status backward_impl(const char* who, const sdm_shape* s, const int32_t* idx_w, const float* w_w,
                         const int32_t* idx_r, const float* w_r, const void* v, const void* alpha, const void* beta,
                         void* mem, int kind, const void* log, const float* scales, const void* dy, float* dv,
                         float* dalpha, float* dbeta, float* dw_w, float* dw_r, float* dM, sdm_stream_t stream);

}  // namespace

extern "C" {

int sdm_abi_version(void) { return SDM_ABI_VERSION; }

const char* sdm_last_error(void) { return g_last_error.c_str(); }

size_t sdm_workspace_bytes(const sdm_shape* shape) {
    int64_t S = 0;
    if (check_shape(shape, true, &S) != SDM_OK) return 0;
    return layout_for(shape, S).total;
}

sdm_status sdm_init_memory(const sdm_shape* s, const void* M0, void* mem, sdm_stream_t stream) {
    SDM_TRY(check_shape(s, false, nullptr));
    const size_t per_seq = static_cast<size_t>(s->H) * static_cast<size_t>(s->N) * s->d_v * elem_bytes(s->dtype);
    if (per_seq == 0 || s->B == 0) return ok();
    SDM_TRY(check_vec(M0, "M0", 16));
    SDM_TRY(check_vec(mem, "mem", 16));
    if (overlaps(Range{M0, per_seq, "M0"}, Range{mem, per_seq * s->B, "mem"}))
        return fail(SDM_ERR_INVALID_ARG, "sdm_init_memory: M0 overlaps mem");
    cudaError_t e = sdm::launch_init_memory(M0, mem, static_cast<int64_t>(per_seq), s->B, reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "init_memory launch");
    return ok();
}

sdm_status sdm_address(const sdm_shape* s, const void* P_q, const void* P_k, const void* q, const void* k,
                       int32_t* idx_w, float* w_w, int32_t* idx_r, float* w_r, void* workspace,
                       size_t workspace_bytes, sdm_stream_t stream) {
    return forward_impl("sdm_address", s, P_q, P_k, q, k, nullptr, nullptr, nullptr, nullptr, nullptr, idx_w, w_w,
                        idx_r, w_r, workspace, workspace_bytes, reinterpret_cast<cudaStream_t>(stream), false);
}

sdm_status sdm_forward(const sdm_shape* s, const void* P_q, const void* P_k, const void* q, const void* k,
                       const void* v, const void* alpha, const void* beta, void* mem, void* y, int32_t* idx_w,
                       float* w_w, int32_t* idx_r, float* w_r, void* workspace, size_t workspace_bytes,
                       sdm_stream_t stream) {
    return forward_impl("sdm_forward", s, P_q, P_k, q, k, v, alpha, beta, mem, y, idx_w, w_w, idx_r, w_r, workspace,
                        workspace_bytes, reinterpret_cast<cudaStream_t>(stream), true);
}

sdm_status sdm_forward_m0(const sdm_shape* s, const void* M0, const void* P_q, const void* P_k, const void* q,
                          const void* k, const void* v, const void* alpha, const void* beta, void* mem, void* y,
                          int32_t* idx_w, float* w_w, int32_t* idx_r, float* w_r, void* workspace,
                          size_t workspace_bytes, sdm_stream_t stream) {
    if (s != nullptr && s->B > 0 && s->H > 0 && s->T > 0 && M0 == nullptr)
        return fail(SDM_ERR_INVALID_ARG, "sdm_forward_m0: M0 is NULL");
    return forward_impl("sdm_forward_m0", s, P_q, P_k, q, k, v, alpha, beta, mem, y, idx_w, w_w, idx_r, w_r, workspace,
                        workspace_bytes, reinterpret_cast<cudaStream_t>(stream), true, M0);
}

size_t sdm_lazy_workspace_bytes(const sdm_shape* shape) {
    int64_t S = 0;
    if (check_shape(shape, true, &S) != SDM_OK) return 0;
    return layout_for(shape, S, true).total;
}

sdm_status sdm_forward_lazy(const sdm_shape* s, const void* M0, uint32_t* touched, const void* P_q, const void* P_k,
                            const void* q, const void* k, const void* v, const void* alpha, const void* beta, void* mem,
                            void* y, int32_t* idx_w, float* w_w, int32_t* idx_r, float* w_r, void* workspace,
                            size_t workspace_bytes, sdm_stream_t stream) {
    const LazyIn lz{M0, touched};
    return forward_impl("sdm_forward_lazy", s, P_q, P_k, q, k, v, alpha, beta, mem, y, idx_w, w_w, idx_r, w_r,
                        workspace, workspace_bytes, reinterpret_cast<cudaStream_t>(stream), true, nullptr, &lz);
}

sdm_status sdm_materialize(const sdm_shape* s, const void* M0, const uint32_t* touched, void* mem, sdm_stream_t stream) {
    SDM_TRY(check_shape(s, false, nullptr));
    const size_t rowb = static_cast<size_t>(s->d_v) * elem_bytes(s->dtype);
    const size_t per_seq = static_cast<size_t>(s->H) * static_cast<size_t>(s->N) * rowb;
    if (per_seq == 0 || s->B == 0) return ok();
    SDM_TRY(check_vec(M0, "M0", 16));
    SDM_TRY(check_vec(touched, "touched", 4));
    SDM_TRY(check_vec(mem, "mem", 16));
    const Range rm{mem, per_seq * s->B, "mem"};
    const Range rt{touched, static_cast<size_t>(s->B) * s->H * static_cast<size_t>((s->N + 31) / 32) * 4, "touched"};
    if (overlaps(rm, Range{M0, per_seq, "M0"})) return fail(SDM_ERR_INVALID_ARG, "sdm_materialize: M0 overlaps mem");
    if (overlaps(rm, rt)) return fail(SDM_ERR_INVALID_ARG, "sdm_materialize: touched overlaps mem");
    cudaError_t e = sdm::launch_materialize(M0, touched, mem, static_cast<int64_t>(s->B) * s->H, s->H, s->N,
                                            static_cast<int64_t>(rowb), reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "materialize launch");
    return ok();
}

sdm_status sdm_gates(const sdm_shape* s, int32_t d_model, const void* x, const void* W_a, const void* W_b,
                     const float* b_dt, const float* A, void* alpha, void* beta, sdm_stream_t stream) {
    SDM_TRY(check_shape(s, false, nullptr));
    const size_t es = elem_bytes(s->dtype);
    if (s->H > 32) return fail(SDM_ERR_UNSUPPORTED, "sdm_gates: H > 32 is not supported (H=%d)", s->H);
    if (d_model < 1 || (static_cast<size_t>(d_model) * es) % 16 != 0)
        return fail(SDM_ERR_UNSUPPORTED, "sdm_gates: d_model * element size must be a positive multiple of 16 bytes (d_model=%d)",
                    d_model);
    const size_t bt = static_cast<size_t>(s->B) * s->T;
    if (bt == 0 || s->H == 0) return ok();
    SDM_TRY(check_vec(x, "x", 16));
    SDM_TRY(check_vec(W_a, "W_a", 16));
    SDM_TRY(check_vec(W_b, "W_b", 16));
    SDM_TRY(check_vec(b_dt, "b_dt", 4));
    SDM_TRY(check_vec(A, "A", 4));
    SDM_TRY(check_vec(alpha, "alpha", es));
    SDM_TRY(check_vec(beta, "beta", es));
    const size_t gbytes = bt * s->H * es;
    const Range ra{alpha, gbytes, "alpha"}, rb{beta, gbytes, "beta"};
    const Range ins[] = {{x, bt * d_model * es, "x"}, {W_a, static_cast<size_t>(s->H) * d_model * es, "W_a"},
                         {W_b, static_cast<size_t>(s->H) * d_model * es, "W_b"}, {b_dt, s->H * 4u, "b_dt"},
                         {A, s->H * 4u, "A"}};
    for (const Range& r : ins)
        if (overlaps(ra, r) || overlaps(rb, r)) return fail(SDM_ERR_INVALID_ARG, "sdm_gates: a gate output overlaps %s", r.name);
    if (overlaps(ra, rb)) return fail(SDM_ERR_INVALID_ARG, "sdm_gates: alpha overlaps beta");
    cudaError_t e;
    if (sdm::gates_tc_supported(s->dtype, s->H, d_model)) {
        int* err = nullptr;
        SDM_TRY(status_word(&err));
        e = sdm::launch_gates_tc(x, W_a, W_b, b_dt, A, alpha, beta, s->B, s->T, s->H, d_model, err,
                                 reinterpret_cast<cudaStream_t>(stream));
    } else {
        e = sdm::launch_gates(s->dtype, x, W_a, W_b, b_dt, A, alpha, beta, s->B, s->T, s->H, d_model,
                              reinterpret_cast<cudaStream_t>(stream));
    }
    if (e != cudaSuccess) return cuda_fail(e, "gates launch");
    return ok();
}

int sdm_gates_tensor_cores(const sdm_shape* s, int32_t d_model) {
    return s != nullptr && sdm::gates_tc_supported(s->dtype, s->H, d_model) ? 1 : 0;
}

sdm_status sdm_head_mix(const sdm_shape* s, int32_t d_model, const void* z, const void* W_o, void* out,
                        sdm_stream_t stream) {
    SDM_TRY(check_shape(s, false, nullptr));
    if (s->dtype != SDM_BF16) return fail(SDM_ERR_UNSUPPORTED, "sdm_head_mix: bf16 storage only");
    const int64_t K = static_cast<int64_t>(s->H) * s->d_v;
    if (d_model <= 0 || d_model % 32 != 0)
        return fail(SDM_ERR_UNSUPPORTED, "sdm_head_mix: d_model must be a positive multiple of 32 (d_model=%d)", d_model);
    if (K % 8 != 0) return fail(SDM_ERR_UNSUPPORTED, "sdm_head_mix: H * d_v must be a multiple of 8");
    const size_t M = static_cast<size_t>(s->B) * s->T;
    if (M == 0) return ok();
    SDM_TRY(check_vec(z, "z", 16));
    SDM_TRY(check_vec(W_o, "W_o", 16));
    SDM_TRY(check_vec(out, "out", 16));
    const Range ro{out, M * d_model * 2, "out"};
    const Range ins[] = {{z, M * K * 2, "z"}, {W_o, static_cast<size_t>(d_model) * K * 2, "W_o"}};
    for (const Range& r : ins)
        if (overlaps(ro, r)) return fail(SDM_ERR_INVALID_ARG, "sdm_head_mix: out overlaps %s", r.name);
    int* err = nullptr;
    SDM_TRY(status_word(&err));
    cudaError_t e = sdm::launch_head_mix(z, W_o, out, static_cast<int64_t>(M), d_model, static_cast<int>(K), err,
                                         reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "head_mix launch");
    return ok();
}

sdm_status sdm_norm_gate(const sdm_shape* s, const void* y, const void* g, const float* gamma, float eps, void* z,
                         sdm_stream_t stream) {
    SDM_TRY(check_shape(s, false, nullptr));
    const size_t es = elem_bytes(s->dtype);
    if (static_cast<size_t>(s->d_v) * es > 1024)
        return fail(SDM_ERR_UNSUPPORTED, "sdm_norm_gate: d_v * element size must be <= 1024 bytes (d_v=%d)", s->d_v);
    if (!(eps >= 0.f)) return fail(SDM_ERR_INVALID_ARG, "sdm_norm_gate: eps must be >= 0");
    const size_t rows = static_cast<size_t>(s->B) * s->H * s->T;
    if (rows == 0) return ok();
    SDM_TRY(check_vec(y, "y", 16));
    SDM_TRY(check_vec(g, "g", 16));
    SDM_TRY(check_vec(gamma, "gamma", 4));
    SDM_TRY(check_vec(z, "z", 16));
    const size_t bytes = rows * s->d_v * es;
    const Range rz{z, bytes, "z"};
    const Range ins[] = {{y, bytes, "y"}, {g, bytes, "g"}, {gamma, s->d_v * 4u, "gamma"}};
    for (const Range& r : ins)
        if (overlaps(rz, r)) return fail(SDM_ERR_INVALID_ARG, "sdm_norm_gate: z overlaps %s", r.name);
    cudaError_t e = sdm::launch_norm_gate(s->dtype, y, g, gamma, eps, z, s->B, s->H, s->T, s->d_v,
                                          reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "norm_gate launch");
    return ok();
}

size_t sdm_access_stats_workspace_bytes(const sdm_shape* s) {
    if (check_shape(s, false, nullptr) != SDM_OK) return 0;
    return align256(static_cast<size_t>(2) * s->B * s->H * static_cast<size_t>((s->N + 31) / 32) * 4) + 256;
}

sdm_status sdm_access_stats(const sdm_shape* s, const int32_t* idx_w, const float* w_w, const int32_t* idx_r,
                            const float* w_r, double* out, void* workspace, size_t workspace_bytes,
                            sdm_stream_t stream) {
    SDM_TRY(check_shape(s, false, nullptr));
    SDM_TRY(check_vec(out, "out", 8));
    const size_t bht = static_cast<size_t>(s->B) * s->H * s->T;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    if (bht == 0) {
        cudaError_t e = cudaMemsetAsync(out, 0, static_cast<size_t>(4 + s->k_write + s->k_read) * sizeof(double), st);
        if (e != cudaSuccess) return cuda_fail(e, "sdm_access_stats");
        return ok();
    }
    SDM_TRY(check_vec(idx_w, "idx_w", 4));
    SDM_TRY(check_vec(w_w, "w_w", 4));
    SDM_TRY(check_vec(idx_r, "idx_r", 4));
    SDM_TRY(check_vec(w_r, "w_r", 4));
    const size_t need = align256(static_cast<size_t>(2) * s->B * s->H * static_cast<size_t>((s->N + 31) / 32) * 4);
    if (!workspace) return fail(SDM_ERR_INVALID_ARG, "sdm_access_stats: workspace is NULL (need %zu bytes)", need);
    if (!aligned(workspace, 256)) return fail(SDM_ERR_INVALID_ARG, "sdm_access_stats: workspace must be 256-byte aligned");
    if (workspace_bytes < need)
        return fail(SDM_ERR_INVALID_ARG, "sdm_access_stats: workspace too small (%zu < %zu bytes)", workspace_bytes, need);
    const Range ro{out, static_cast<size_t>(4 + s->k_write + s->k_read) * sizeof(double), "out"};
    if (overlaps(ro, Range{workspace, need, "workspace"}))
        return fail(SDM_ERR_INVALID_ARG, "sdm_access_stats: out overlaps workspace");
    cudaError_t e = sdm::launch_access_stats(idx_w, w_w, idx_r, w_r, static_cast<int64_t>(s->B) * s->H, s->T,
                                             s->k_write, s->k_read, s->N, static_cast<uint32_t*>(workspace), out, st);
    if (e != cudaSuccess) return cuda_fail(e, "access stats launch");
    return ok();
}

sdm_status sdm_decode_step(const sdm_shape* s, const void* P_q, const void* P_k, const void* q, const void* k,
                           const void* v, const void* alpha, const void* beta, void* mem, void* y, int32_t* idx_w,
                           float* w_w, int32_t* idx_r, float* w_r, void* workspace, size_t workspace_bytes,
                           sdm_stream_t stream) {
    if (s && s->T != 1) return fail(SDM_ERR_INVALID_ARG, "sdm_decode_step needs shape->T == 1 (got %d)", s->T);
    return forward_impl("sdm_decode_step", s, P_q, P_k, q, k, v, alpha, beta, mem, y, idx_w, w_w, idx_r, w_r,
                        workspace, workspace_bytes, reinterpret_cast<cudaStream_t>(stream), true);
}

size_t sdm_recur_workspace_bytes(const sdm_shape* s) {
    if (check_shape(s, false, nullptr) != SDM_OK) return 0;
    return align256(sdm::rec_workspace_bytes(s->B, s->H, s->T, s->k_write, s->k_read)) + 256;
}

sdm_status sdm_recur(const sdm_shape* s, const int32_t* idx_w, const float* w_w, const int32_t* idx_r,
                     const float* w_r, const void* v, const void* alpha, const void* beta, void* mem, void* y,
                     void* workspace, size_t workspace_bytes, sdm_stream_t stream) {
    return recur_impl("sdm_recur", s, idx_w, w_w, idx_r, w_r, v, alpha, beta, mem, y, nullptr, workspace,
                      workspace_bytes, stream);
}

sdm_status sdm_recur_chunkwise(const sdm_shape* s, const int32_t* idx_w, const float* w_w, const int32_t* idx_r,
                               const float* w_r, const void* v, const void* alpha, const void* beta, void* mem,
                               void* y, int32_t chunk, sdm_stream_t stream) {
    if (chunk < 1 || chunk > 32) return fail(SDM_ERR_INVALID_ARG, "sdm_recur_chunkwise: chunk must be in [1, 32] (got %d)", chunk);
    if (s != nullptr && s->d_v > 256)
        return fail(SDM_ERR_UNSUPPORTED, "sdm_recur_chunkwise: d_v > 256 is not supported (d_v=%d)", s->d_v);
    sdm::RecArgs r{};
    bool empty = false;
    SDM_TRY(sdm::recur_args("sdm_recur_chunkwise", s, idx_w, w_w, idx_r, w_r, v, alpha, beta, mem, y, &r, &empty));
    if (empty) return ok();
    cudaError_t e = sdm::launch_recur_chunkwise(s->dtype, r, chunk, reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "chunkwise recurrence launch");
    return ok();
}

size_t sdm_undo_log_bytes(const sdm_shape* s) {
    if (check_shape(s, false, nullptr) != SDM_OK) return 0;
    return static_cast<size_t>(s->B) * s->H * s->T * s->k_write * s->d_v * elem_bytes(s->dtype);
}

sdm_status sdm_recur_undo(const sdm_shape* s, const int32_t* idx_w, const float* w_w, const int32_t* idx_r,
                          const float* w_r, const void* v, const void* alpha, const void* beta, void* mem, void* y,
                          void* undo, void* workspace, size_t workspace_bytes, sdm_stream_t stream) {
    if (s != nullptr && static_cast<size_t>(s->B) * s->H * s->T > 0 && undo == nullptr)
        return fail(SDM_ERR_INVALID_ARG, "sdm_recur_undo: undo is NULL");
    return recur_impl("sdm_recur_undo", s, idx_w, w_w, idx_r, w_r, v, alpha, beta, mem, y, undo, workspace,
                      workspace_bytes, stream);
}

sdm_status sdm_recur_backward(const sdm_shape* s, const int32_t* idx_w, const float* w_w, const int32_t* idx_r,
                              const float* w_r, const void* v, const void* alpha, const void* beta, void* mem,
                              const void* undo, const void* dy, float* dv, float* dalpha, float* dbeta, float* dw_w,
                              float* dw_r, float* dM, sdm_stream_t stream) {
    return backward_impl("sdm_recur_backward", s, idx_w, w_w, idx_r, w_r, v, alpha, beta, mem, 0, undo, nullptr,
                         dy, dv, dalpha, dbeta, dw_w, dw_r, dM, stream);
}

size_t sdm_undo_code_bytes(const sdm_shape* s, int kind) {
    if (check_shape(s, false, nullptr) != SDM_OK || (kind != SDM_UNDO_FP8 && kind != SDM_UNDO_INT4)) return 0;
    const size_t rows = static_cast<size_t>(s->B) * s->H * s->T * s->k_write;
    return rows * (kind == SDM_UNDO_FP8 ? s->d_v : s->d_v / 2);
}

sdm_status sdm_undo_quantize(const sdm_shape* s, const void* undo, int kind, void* codes, float* scales,
                             sdm_stream_t stream) {
    SDM_TRY(check_shape(s, false, nullptr));
    if (kind != SDM_UNDO_FP8 && kind != SDM_UNDO_INT4)
        return fail(SDM_ERR_INVALID_ARG, "sdm_undo_quantize: kind must be SDM_UNDO_FP8 or SDM_UNDO_INT4 (kind=%d)", kind);
    if (s->d_v % 32 != 0 || s->d_v > 256)
        return fail(SDM_ERR_UNSUPPORTED, "sdm_undo_quantize: d_v must be a multiple of 32, at most 256 (d_v=%d)", s->d_v);
    const size_t rows = static_cast<size_t>(s->B) * s->H * s->T * s->k_write;
    if (rows == 0) return ok();
    const size_t es = elem_bytes(s->dtype);
    SDM_TRY(check_vec(undo, "undo", 16));
    SDM_TRY(check_vec(codes, "codes", 16));
    SDM_TRY(check_vec(scales, "scales", 4));
    const Range in{undo, rows * s->d_v * es, "undo"};
    const Range oc{codes, sdm_undo_code_bytes(s, kind), "codes"}, os{scales, rows * 4, "scales"};
    if (overlaps(oc, in) || overlaps(os, in) || overlaps(oc, os))
        return fail(SDM_ERR_INVALID_ARG, "sdm_undo_quantize: undo, codes and scales must not overlap");
    cudaError_t e = sdm::launch_undo_quantize(s->dtype, kind, undo, static_cast<int64_t>(rows), s->d_v, codes, scales,
                                              reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "undo quantize launch");
    return ok();
}

sdm_status sdm_recur_backward_q(const sdm_shape* s, const int32_t* idx_w, const float* w_w, const int32_t* idx_r,
                                const float* w_r, const void* v, const void* alpha, const void* beta, void* mem,
                                int kind, const void* codes, const float* scales, const void* dy, float* dv,
                                float* dalpha, float* dbeta, float* dw_w, float* dw_r, float* dM, sdm_stream_t stream) {
    if (kind != SDM_UNDO_FP8 && kind != SDM_UNDO_INT4)
        return fail(SDM_ERR_INVALID_ARG, "sdm_recur_backward_q: kind must be SDM_UNDO_FP8 or SDM_UNDO_INT4 (kind=%d)", kind);
    return backward_impl("sdm_recur_backward_q", s, idx_w, w_w, idx_r, w_r, v, alpha, beta, mem, kind, codes, scales,
                         dy, dv, dalpha, dbeta, dw_w, dw_r, dM, stream);
}

}  // extern "C"

namespace {

sdm_status backward_impl(const char* who, const sdm_shape* s, const int32_t* idx_w, const float* w_w,
                         const int32_t* idx_r, const float* w_r, const void* v, const void* alpha, const void* beta,
                         void* mem, int kind, const void* log, const float* scales, const void* dy, float* dv,
                         float* dalpha, float* dbeta, float* dw_w, float* dw_r, float* dM, sdm_stream_t stream) {
    SDM_TRY(check_shape(s, false, nullptr));
    if (s->d_v % 32 != 0 || s->d_v > 256)
        return fail(SDM_ERR_UNSUPPORTED, "%s: d_v must be a multiple of 32, at most 256 (d_v=%d)", who, s->d_v);
    if (s->k_write > 32 || s->k_read > 32)
        return fail(SDM_ERR_UNSUPPORTED, "%s: k_write and k_read must be at most 32 (%d, %d)", who, s->k_write, s->k_read);
    const size_t es = elem_bytes(s->dtype);
    const size_t bht = static_cast<size_t>(s->B) * s->H * s->T;
    if (bht == 0) return ok();
    SDM_TRY(check_vec(idx_w, "idx_w", 4));
    SDM_TRY(check_vec(w_w, "w_w", 4));
    SDM_TRY(check_vec(idx_r, "idx_r", 4));
    SDM_TRY(check_vec(w_r, "w_r", 4));
    SDM_TRY(check_vec(v, "v", es));
    SDM_TRY(check_vec(alpha, "alpha", es));
    SDM_TRY(check_vec(beta, "beta", es));
    SDM_TRY(check_vec(mem, "mem", 16));
    SDM_TRY(check_vec(log, kind == 0 ? "undo" : "codes", 16));
    if (kind != 0) SDM_TRY(check_vec(scales, "scales", 4));
    SDM_TRY(check_vec(dy, "dy", es));
    SDM_TRY(check_vec(dv, "dv", 4));
    SDM_TRY(check_vec(dalpha, "dalpha", 4));
    SDM_TRY(check_vec(dbeta, "dbeta", 4));
    SDM_TRY(check_vec(dw_w, "dw_w", 4));
    SDM_TRY(check_vec(dw_r, "dw_r", 4));
    SDM_TRY(check_vec(dM, "dM", 4));
    const size_t rowb = static_cast<size_t>(s->d_v) * es;
    const size_t memb = static_cast<size_t>(s->B) * s->H * static_cast<size_t>(s->N) * rowb;
    const size_t logb = kind == 0 ? bht * s->k_write * rowb : sdm_undo_code_bytes(s, kind);
    const Range outs[] = {{mem, memb, "mem"}, {dv, bht * s->d_v * 4, "dv"}, {dalpha, bht * 4, "dalpha"},
                          {dbeta, bht * 4, "dbeta"}, {dw_w, bht * s->k_write * 4, "dw_w"},
                          {dw_r, bht * s->k_read * 4, "dw_r"},
                          {dM, static_cast<size_t>(s->B) * s->H * static_cast<size_t>(s->N) * s->d_v * 4, "dM"}};
    const Range ins[] = {{idx_w, bht * s->k_write * 4, "idx_w"}, {w_w, bht * s->k_write * 4, "w_w"},
                         {idx_r, bht * s->k_read * 4, "idx_r"}, {w_r, bht * s->k_read * 4, "w_r"},
                         {v, bht * rowb, "v"}, {alpha, bht * es, "alpha"}, {beta, bht * es, "beta"},
                         {log, logb, kind == 0 ? "undo" : "codes"},
                         {scales, kind == 0 ? 0 : bht * s->k_write * 4, "scales"}, {dy, bht * rowb, "dy"}};
    for (size_t i = 0; i < sizeof(outs) / sizeof(outs[0]); ++i) {
        for (const Range& r : ins)
            if (overlaps(outs[i], r)) return fail(SDM_ERR_INVALID_ARG, "%s: %s overlaps %s", who, outs[i].name, r.name);
        for (size_t j = i + 1; j < sizeof(outs) / sizeof(outs[0]); ++j)
            if (overlaps(outs[i], outs[j]))
                return fail(SDM_ERR_INVALID_ARG, "%s: %s overlaps %s", who, outs[i].name, outs[j].name);
    }
    int* err = nullptr;
    SDM_TRY(status_word(&err));
    sdm::RecArgs r{};
    r.idx_w = idx_w; r.w_w = w_w; r.idx_r = idx_r; r.w_r = w_r;
    r.v = v; r.alpha = alpha; r.beta = beta; r.mem = mem;
    r.B = s->B; r.H = s->H; r.T = s->T; r.dv = s->d_v; r.kw = s->k_write; r.kr = s->k_read;
    r.N = s->N;
    r.err = err;
    cudaError_t e = sdm::launch_recur_backward(s->dtype, r, kind, kind == 0 ? log : nullptr, kind == 0 ? nullptr : log,
                                               scales, dy, dv, dalpha, dbeta, dw_w, dw_r, dM,
                                               reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "backward launch");
    return ok();
}

sdm_status recur_impl(const char* who, const sdm_shape* s, const int32_t* idx_w, const float* w_w,
                      const int32_t* idx_r, const float* w_r, const void* v, const void* alpha, const void* beta,
                      void* mem, void* y, void* undo, void* workspace, size_t workspace_bytes, sdm_stream_t stream,
                      long long wait_cycles, int hold_handover) {
    SDM_TRY(check_shape(s, false, nullptr));
    const size_t es = elem_bytes(s->dtype);
    const size_t bht = static_cast<size_t>(s->B) * s->H * s->T;
    if (bht == 0) return ok();
    SDM_TRY(check_vec(idx_w, "idx_w", 4));
    SDM_TRY(check_vec(w_w, "w_w", 4));
    SDM_TRY(check_vec(idx_r, "idx_r", 4));
    SDM_TRY(check_vec(w_r, "w_r", 4));
    SDM_TRY(check_vec(v, "v", 16));
    SDM_TRY(check_vec(alpha, "alpha", es));
    SDM_TRY(check_vec(beta, "beta", es));
    SDM_TRY(check_vec(mem, "mem", 16));
    SDM_TRY(check_vec(y, "y", 16));
    const size_t rowb = static_cast<size_t>(s->d_v) * es;
    const Range rm{mem, static_cast<size_t>(s->B) * s->H * static_cast<size_t>(s->N) * rowb, "mem"};
    const Range others[] = {{idx_w, bht * s->k_write * 4, "idx_w"}, {w_w, bht * s->k_write * 4, "w_w"},
                            {idx_r, bht * s->k_read * 4, "idx_r"},  {w_r, bht * s->k_read * 4, "w_r"},
                            {v, bht * rowb, "v"}, {alpha, bht * es, "alpha"}, {beta, bht * es, "beta"},
                            {y, bht * rowb, "y"}};
    for (const Range& r : others)
        if (overlaps(rm, r)) return fail(SDM_ERR_INVALID_ARG, "%s: mem overlaps %s", who, r.name);
    const size_t need = align256(sdm::rec_workspace_bytes(s->B, s->H, s->T, s->k_write, s->k_read));
    if (!workspace) return fail(SDM_ERR_INVALID_ARG, "%s: workspace is NULL (need %zu bytes)", who, need);
    if (!aligned(workspace, 256)) return fail(SDM_ERR_INVALID_ARG, "%s: workspace must be 256-byte aligned", who);
    if (workspace_bytes < need)
        return fail(SDM_ERR_INVALID_ARG, "%s: workspace too small (%zu < %zu bytes)", who, workspace_bytes, need);
    if (overlaps(rm, Range{workspace, need, "workspace"})) return fail(SDM_ERR_INVALID_ARG, "%s: mem overlaps workspace", who);
    if (undo != nullptr) {
        SDM_TRY(check_vec(undo, "undo", 16));
        const Range ru{undo, bht * s->k_write * rowb, "undo"};
        if (overlaps(ru, rm) || overlaps(ru, Range{workspace, need, "workspace"}))
            return fail(SDM_ERR_INVALID_ARG, "%s: undo overlaps mem or the workspace", who);
        for (const Range& r : others)
            if (overlaps(ru, r)) return fail(SDM_ERR_INVALID_ARG, "%s: undo overlaps %s", who, r.name);
    }
    int* err = nullptr;
    SDM_TRY(status_word(&err));
    sdm::RecArgs r{};
    r.idx_w = idx_w; r.w_w = w_w; r.idx_r = idx_r; r.w_r = w_r;
    r.v = v; r.alpha = alpha; r.beta = beta; r.mem = mem; r.y = y;
    r.B = s->B; r.H = s->H; r.T = s->T; r.dv = s->d_v; r.kw = s->k_write; r.kr = s->k_read;
    r.N = s->N;
    r.err = err;
    r.undo = undo;
    r.wait_cycles = wait_cycles;
    r.hold_handover = hold_handover;
    cudaError_t e = sdm::launch_recur(s->dtype, r, static_cast<int32_t*>(workspace), reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "recurrence launch");
    return ok();
}

}  // namespace

extern "C" {

sdm_status sdm_device_stats(uint32_t* counts, int n, sdm_stream_t stream) {
    if (!counts || n < 0 || n > 15) return fail(SDM_ERR_INVALID_ARG, "counts must be non-NULL and n in [0, 15]");
    if (n == 0) return ok();
    int* w = nullptr;
    SDM_TRY(status_word(&w));
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    cudaError_t e = cudaMemcpyAsync(counts, w + 1, sizeof(uint32_t) * n, cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e == cudaSuccess) e = cudaMemsetAsync(w + 1, 0, sizeof(uint32_t) * n, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return cuda_fail(e, "sdm_device_stats");
    return ok();
}

sdm_status sdm_device_status(int32_t* code, sdm_stream_t stream) {
    if (!code) return fail(SDM_ERR_INVALID_ARG, "code is NULL");
    int* w = nullptr;
    SDM_TRY(status_word(&w));
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    int host = 0;
    cudaError_t e = cudaMemcpyAsync(&host, w, sizeof(int), cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e == cudaSuccess) e = cudaMemsetAsync(w, 0, sizeof(int), st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return cuda_fail(e, "sdm_device_status");
    *code = host;
    if (host != 0)
        return fail((host & sdm::ERR_TIMEOUT) ? SDM_ERR_TIMEOUT : SDM_ERR_DEVICE,
                    "device status word = 0x%x (bit 0: slot index outside [0, N) skipped; "
                    "bit 1: slot list not strictly ascending; bit 2: bounded wait timed out; "
                    "bit 3: selection invariant failed)", host);
    return ok();
}

sdm_status sdm_test_scores(const sdm_shape* s, const void* P_q, const void* P_k, const void* q, const void* k,
                           float* scores, void* workspace, size_t workspace_bytes, sdm_stream_t stream) {
    int64_t S = 0;
    SDM_TRY(check_shape(s, true, &S));
    if (static_cast<size_t>(s->B) * s->H * s->T == 0) return ok();
    const Layout L = layout_for(s, S);
    if (!L.plan.mma) return fail(SDM_ERR_UNSUPPORTED, "sdm_test_scores: the shape does not take the tensor-core score path");
    SDM_TRY(check_vec(P_q, "P_q", 16));
    SDM_TRY(check_vec(P_k, "P_k", 16));
    SDM_TRY(check_vec(q, "q", 16));
    SDM_TRY(check_vec(k, "k", 16));
    SDM_TRY(check_vec(scores, "scores", 4));
    if (!workspace || !aligned(workspace, 256) || workspace_bytes < L.total)
        return fail(SDM_ERR_INVALID_ARG, "sdm_test_scores: workspace must be >= sdm_workspace_bytes and 256-byte aligned");
    int* err = nullptr;
    SDM_TRY(status_word(&err));
    char* ws = static_cast<char*>(workspace);
    sdm::AddrArgs a{};
    a.P[0] = P_q; a.P[1] = P_k; a.X[0] = q; a.X[1] = k;
    a.kk[0] = s->k_read; a.kk[1] = s->k_write;
    a.B = s->B; a.H = s->H; a.T = s->T; a.dk = s->d_k; a.S = static_cast<int>(S);
    a.ncc = L.plan.ncc; a.cw = L.plan.cw;
    a.part_v = reinterpret_cast<float*>(ws + L.part_v);
    a.part_i = reinterpret_cast<int*>(ws + L.part_i);
    a.err = err;
    a.raw = scores;
    cudaError_t e = sdm::launch_address_mma(L.plan, a, reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "sdm_test_scores launch");
    return ok();
}

sdm_status sdm_recur_plan(const sdm_shape* s, int32_t* out, int n) {
    SDM_TRY(check_shape(s, false, nullptr));
    if (!out || n < 0 || n > 6) return fail(SDM_ERR_INVALID_ARG, "sdm_recur_plan: out must be non-NULL and n in [0, 6]");
    const sdm::RecPlan p = sdm::rec_plan(s->dtype, s->B, s->H, s->T, s->d_v, s->k_write, s->k_read);
    const int32_t v[6] = {p.dch, p.nsplit, p.spt, p.la, p.w, p.p};
    for (int i = 0; i < n; ++i) out[i] = v[i];
    return ok();
}

sdm_status sdm_test_recur_wait_timeout(const sdm_shape* s, const int32_t* idx_w, const float* w_w,
                                       const int32_t* idx_r, const float* w_r, const void* v, const void* alpha,
                                       const void* beta, void* mem, void* y, void* workspace, size_t workspace_bytes,
                                       int64_t wait_cycles, sdm_stream_t stream) {
    SDM_TRY(check_shape(s, false, nullptr));
    if (wait_cycles < 1 || wait_cycles > (static_cast<int64_t>(1) << 32))
        return fail(SDM_ERR_INVALID_ARG, "sdm_test_recur_wait_timeout: wait_cycles must be in [1, 2^32]");
    const sdm::RecPlan p = sdm::rec_plan(s->dtype, s->B, s->H, s->T, s->d_v, s->k_write, s->k_read);
    if (p.w < 2 || static_cast<int64_t>(s->B) * s->H * s->T == 0)
        return fail(SDM_ERR_UNSUPPORTED, "sdm_test_recur_wait_timeout: the token-interleaved kernel does not serve this shape");
    return recur_impl("sdm_test_recur_wait_timeout", s, idx_w, w_w, idx_r, w_r, v, alpha, beta, mem, y, nullptr,
                      workspace, workspace_bytes, stream, static_cast<long long>(wait_cycles), 1);
}

}  // extern "C"

// Internal helpers for entry points defined in other translation units.
namespace sdm {

sdm_status api_error(sdm_status st, const char* msg) { return fail(st, "%s", msg); }

sdm_status api_ok() { return ok(); }

// The argument checks of sdm_recur without its workspace; fills `r` (including the status
// word) and sets *empty when B H T == 0 (nothing to launch).
sdm_status recur_args(const char* who, const sdm_shape* s, const int32_t* idx_w, const float* w_w,
                      const int32_t* idx_r, const float* w_r, const void* v, const void* alpha, const void* beta,
                      void* mem, void* y, RecArgs* r, bool* empty) {
    SDM_TRY(check_shape(s, false, nullptr));
    const size_t es = elem_bytes(s->dtype);
    const size_t bht = static_cast<size_t>(s->B) * s->H * s->T;
    *empty = bht == 0;
    if (*empty) return ok();
    SDM_TRY(check_vec(idx_w, "idx_w", 4));
    SDM_TRY(check_vec(w_w, "w_w", 4));
    SDM_TRY(check_vec(idx_r, "idx_r", 4));
    SDM_TRY(check_vec(w_r, "w_r", 4));
    SDM_TRY(check_vec(v, "v", 16));
    SDM_TRY(check_vec(alpha, "alpha", es));
    SDM_TRY(check_vec(beta, "beta", es));
    SDM_TRY(check_vec(mem, "mem", 16));
    SDM_TRY(check_vec(y, "y", 16));
    const size_t rowb = static_cast<size_t>(s->d_v) * es;
    const Range rm{mem, static_cast<size_t>(s->B) * s->H * static_cast<size_t>(s->N) * rowb, "mem"};
    const Range others[] = {{idx_w, bht * s->k_write * 4, "idx_w"}, {w_w, bht * s->k_write * 4, "w_w"},
                            {idx_r, bht * s->k_read * 4, "idx_r"},  {w_r, bht * s->k_read * 4, "w_r"},
                            {v, bht * rowb, "v"}, {alpha, bht * es, "alpha"}, {beta, bht * es, "beta"},
                            {y, bht * rowb, "y"}};
    for (const Range& q : others)
        if (overlaps(rm, q)) return fail(SDM_ERR_INVALID_ARG, "%s: mem overlaps %s", who, q.name);
    int* err = nullptr;
    SDM_TRY(status_word(&err));
    *r = RecArgs{};
    r->idx_w = idx_w; r->w_w = w_w; r->idx_r = idx_r; r->w_r = w_r;
    r->v = v; r->alpha = alpha; r->beta = beta; r->mem = mem; r->y = y;
    r->B = s->B; r->H = s->H; r->T = s->T; r->dv = s->d_v; r->kw = s->k_write; r->kr = s->k_read;
    r->N = s->N;
    r->err = err;
    return SDM_OK;
}

}  // namespace sdm
