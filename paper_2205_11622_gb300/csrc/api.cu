// C entry points of libslnr (declared in include/slnr.h): argument checks,
// workspace layout, and the launch sequence of each variant.
#include <cstdarg>
#include <cstdio>
#include <cstring>

#include "launch.h"

using namespace slnr;

namespace {

thread_local char g_last_error[512] = "";
thread_local long long g_wait_limit = 0;  // 0: kWaitCycles

slnr_status fail(slnr_status st, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_last_error, sizeof(g_last_error), fmt, ap);
  va_end(ap);
  return st;
}

// ---------------------------------------------------------------------------
// per-launch timing (slnr_timing_*): events recorded between launches

constexpr int kMaxTimed = 16;
struct Timing {
  bool on = false;
  bool created = false;
  int n = 0;
  const char* names[kMaxTimed] = {};
  cudaEvent_t ev[kMaxTimed + 1] = {};
};
thread_local Timing g_timing;
thread_local int32_t g_launches = 0;  // kernel launches of this thread's current call

void timing_begin() {
  g_timing.n = 0;
  g_launches = 0;
}

void timing_mark(const char* name, cudaStream_t s) {
  if (!g_timing.on || g_timing.n >= kMaxTimed) return;
  cudaEventRecord(g_timing.ev[g_timing.n], s);
  g_timing.names[g_timing.n++] = name;
}

void timing_end(cudaStream_t s) {
  if (g_timing.on && g_timing.n > 0) cudaEventRecord(g_timing.ev[g_timing.n], s);
}

#define SLNR_CUDA(expr)                                                                   \
  do {                                                                                    \
    cudaError_t e_ = (expr);                                                              \
    if (e_ != cudaSuccess) return fail(SLNR_ERR_CUDA, "%s: %s", #expr, cudaGetErrorString(e_)); \
  } while (0)

// Widths the specialised kernels take (powers of two in [4, 256]); any other
// multiple of 4 up to kWideMax goes to the run-time-width kernels (wide.cu).
bool pow2_dim(int32_t d) { return d >= 4 && d <= 256 && (d & (d - 1)) == 0; }
bool all_pow2(int32_t a, int32_t b, int32_t c = 4) { return pow2_dim(a) && pow2_dim(b) && pow2_dim(c); }
bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

// ---------------------------------------------------------------------------
// workspace layout (identical for the size query and the call)

struct Layout {
  size_t cur = sizeof(WsHeader);
  size_t take(size_t bytes) {
    cur = align256(cur);
    const size_t o = cur;
    cur += bytes;
    return o;
  }
  // heavy-row split of a CSR-shaped level
  size_t o_heavy = 0, o_chunks = 0, o_partial = 0;
  int max_heavy = 0, max_chunks = 0;
  void split(int64_t nrows, int64_t nnz, int width) {
    if (nnz > kLightMax) {
      int64_t mh = nnz / (kLightMax + 1);
      if (mh > nrows) mh = nrows;
      max_heavy = (int)mh;
      max_chunks = (int)(nnz / kChunk + mh + 1);
    }
    o_heavy = take(sizeof(HeavyRow) * (size_t)max_heavy);
    o_chunks = take(sizeof(Chunk) * (size_t)max_chunks);
    o_partial = take(sizeof(float) * (size_t)max_chunks * (size_t)width);
  }
  // MTTKRP units
  size_t o_su = 0, o_units = 0, o_upartial = 0, o_uparts = 0;
  int max_units = 0;
  void units(int64_t nslices, int64_t nnz, int width) {
    max_units = (int)(nnz / kUnitNnz + nslices + 1);
    o_su = take(sizeof(SliceUnits) * (size_t)nslices);
    o_units = take(sizeof(Unit) * (size_t)max_units);
    o_upartial = take(sizeof(float) * (size_t)max_units * (size_t)width);
    o_uparts = take(sizeof(float) * (size_t)max_units * (size_t)width);
  }
  // row segments of the tensor-core path (partials are A rows of the output width)
  size_t o_counts = 0, o_segs = 0;
  int max_segs = 0;
  void segs(int64_t nrows, int64_t nnz, int width) {
    int64_t mh = 0, mc = 0;
    if (nnz > kSegChunk) {
      mh = nnz / (kSegChunk + 1);
      if (mh > nrows) mh = nrows;
      mc = nnz / kSegChunk + mh + 1;
    }
    max_heavy = (int)mh;
    max_chunks = (int)mc;
    max_segs = (int)(nrows + mc);
    o_counts = take(sizeof(int) * kSegCounters * (size_t)seg_scan_blocks(nrows));
    o_segs = take(sizeof(int4) * (size_t)max_segs);
    o_heavy = take(sizeof(HeavyRow) * (size_t)mh);
    o_partial = take(sizeof(float) * (size_t)mc * (size_t)width);
  }
  size_t o_inter = 0, o_inter2 = 0;
  void inter(size_t bytes) { o_inter = take(bytes); }
  void inter2(size_t bytes) { o_inter2 = take(bytes); }
  size_t total() const { return align256(cur); }
};

SplitPlan split_plan(char* ws, const Layout& l) {
  return SplitPlan{reinterpret_cast<WsHeader*>(ws), reinterpret_cast<HeavyRow*>(ws + l.o_heavy),
                   reinterpret_cast<Chunk*>(ws + l.o_chunks), reinterpret_cast<float*>(ws + l.o_partial),
                   l.max_heavy, l.max_chunks};
}

SegPlan seg_plan(char* ws, const Layout& l) {
  return SegPlan{reinterpret_cast<WsHeader*>(ws), reinterpret_cast<int*>(ws + l.o_counts),
                 reinterpret_cast<int4*>(ws + l.o_segs), reinterpret_cast<HeavyRow*>(ws + l.o_heavy),
                 reinterpret_cast<float*>(ws + l.o_partial), l.max_segs, l.max_heavy, l.max_chunks};
}

// The heavy-row records and partial rows of a segment plan, as k_combine reads them.
SplitPlan combine_plan(const SegPlan& g) {
  return SplitPlan{g.hdr, g.heavy, nullptr, g.partial, g.max_heavy, g.max_chunks};
}

UnitPlan unit_plan(char* ws, const Layout& l) {
  return UnitPlan{reinterpret_cast<WsHeader*>(ws), reinterpret_cast<SliceUnits*>(ws + l.o_su),
                  reinterpret_cast<Unit*>(ws + l.o_units), reinterpret_cast<float*>(ws + l.o_upartial),
                  l.max_units, reinterpret_cast<float*>(ws + l.o_uparts)};
}

// ---------------------------------------------------------------------------
// argument checks

slnr_status check_opts(const slnr_opts* o) {
  if (!o) return fail(SLNR_ERR_NULL, "opts is NULL");
  if (o->variant != SLNR_FUSED && o->variant != SLNR_UNFUSED)
    return fail(SLNR_ERR_UNSUPPORTED, "unknown variant %d", (int)o->variant);
  if (o->reserved != 0) return fail(SLNR_ERR_UNSUPPORTED, "opts.reserved must be 0");
  return SLNR_OK;
}

slnr_status check_csr(const slnr_csr* B, bool need_ptrs) {
  if (!B) return fail(SLNR_ERR_NULL, "B is NULL");
  if (B->nrows < 0 || B->ncols < 0 || B->nnz < 0) return fail(SLNR_ERR_SHAPE, "negative size in B");
  if (B->nnz >= (int64_t(1) << 31)) return fail(SLNR_ERR_UNSUPPORTED, "nnz must be < 2^31");
  if (B->nnz > 0 && (B->nrows == 0 || B->ncols == 0)) return fail(SLNR_ERR_SHAPE, "nnz > 0 in an empty matrix");
  if (need_ptrs) {
    if (!B->pos) return fail(SLNR_ERR_NULL, "B.pos is NULL");
    if (B->nnz > 0 && (!B->crd || !B->vals)) return fail(SLNR_ERR_NULL, "B.crd or B.vals is NULL");
  }
  return SLNR_OK;
}

slnr_status check_csf(const slnr_csf3* B, bool need_ptrs) {
  if (!B) return fail(SLNR_ERR_NULL, "B is NULL");
  if (B->dim[0] < 0 || B->dim[1] < 0 || B->dim[2] < 0 || B->nnz < 0 || B->nslices < 0 || B->nfibers < 0)
    return fail(SLNR_ERR_SHAPE, "negative size in B");
  if (B->nnz >= (int64_t(1) << 31)) return fail(SLNR_ERR_UNSUPPORTED, "nnz must be < 2^31");
  if (B->nslices > B->dim[0] || (int64_t)B->nfibers > (int64_t)B->nslices * B->dim[1] ||
      B->nnz > (int64_t)B->nfibers * B->dim[2])
    return fail(SLNR_ERR_SHAPE, "counts of B exceed its dimensions");
  if (need_ptrs) {
    if (!B->pos1 || !B->pos2 || !B->pos3) return fail(SLNR_ERR_NULL, "a CSF position array is NULL");
    if (B->nslices > 0 && !B->crd1) return fail(SLNR_ERR_NULL, "B.crd1 is NULL");
    if (B->nfibers > 0 && !B->crd2) return fail(SLNR_ERR_NULL, "B.crd2 is NULL");
    if (B->nnz > 0 && (!B->crd3 || !B->vals)) return fail(SLNR_ERR_NULL, "B.crd3 or B.vals is NULL");
  }
  return SLNR_OK;
}

slnr_status check_dims(const char* what, int32_t d) {
  if (d <= 0) return fail(SLNR_ERR_SHAPE, "%s = %d must be positive", what, (int)d);
  if (!wide_dim(d))
    return fail(SLNR_ERR_UNSUPPORTED, "%s = %d: must be a multiple of 4 in [4, %d]", what, (int)d, kWideMax);
  return SLNR_OK;
}

slnr_status check_dense(const char* what, const void* p) {
  if (!p) return fail(SLNR_ERR_NULL, "%s is NULL", what);
  if (!aligned16(p)) return fail(SLNR_ERR_UNSUPPORTED, "%s must be 16-byte aligned", what);
  return SLNR_OK;
}

slnr_status check_ws(const slnr_opts* o, size_t need) {
  if (!o->workspace) return fail(SLNR_ERR_WORKSPACE, "workspace is NULL (needs %zu bytes)", need);
  if ((reinterpret_cast<uintptr_t>(o->workspace) & 255u) != 0)
    return fail(SLNR_ERR_WORKSPACE, "workspace must be 256-byte aligned");
  if (o->workspace_bytes < need)
    return fail(SLNR_ERR_WORKSPACE, "workspace has %zu bytes, needs %zu", o->workspace_bytes, need);
  return SLNR_OK;
}

// A kernel launch of the call: timing mark, then the launch, then its status.
#define SLNR_LAUNCH(name, expr) \
  do {                          \
    timing_mark(name, s);       \
    SLNR_CUDA(expr);            \
  } while (0)

#define SLNR_CHECK(expr)            \
  do {                              \
    slnr_status st_ = (expr);       \
    if (st_ != SLNR_OK) return st_; \
  } while (0)

// Zero the header, then (validate mode) run the device check and wait for it.
template <typename Launch>
slnr_status begin(char* ws, cudaStream_t s, bool validate, Launch launch_validate) {
  WsHeader* hdr = reinterpret_cast<WsHeader*>(ws);
  SLNR_CUDA(cudaMemsetAsync(hdr, 0, sizeof(WsHeader), s));
  if (validate) {
    SLNR_CUDA(launch_validate(hdr));
    int flag = 0;
    SLNR_CUDA(cudaMemcpyAsync(&flag, &hdr->error, sizeof(int), cudaMemcpyDeviceToHost, s));
    SLNR_CUDA(cudaStreamSynchronize(s));
    if (flag != 0) return fail(SLNR_ERR_INDEX, "malformed index arrays (flags 0x%x)", flag);
  }
  return SLNR_OK;
}

// End of a call.  In validate mode the call waits for its launches and reads
// the device flag word: a bounded wait that gave up returns SLNR_ERR_TIMEOUT,
// an inspector bound exceeded (positions inconsistent with nnz) returns
// SLNR_ERR_INDEX.  Otherwise the launches stay asynchronous.
slnr_status finish(char* ws, cudaStream_t s, bool validate) {
  timing_end(s);
  if (!validate) return SLNR_OK;
  WsHeader* hdr = reinterpret_cast<WsHeader*>(ws);
  int flag = 0;
  SLNR_CUDA(cudaMemcpyAsync(&flag, &hdr->error, sizeof(int), cudaMemcpyDeviceToHost, s));
  SLNR_CUDA(cudaStreamSynchronize(s));
  if (flag & kErrTimeout) return fail(SLNR_ERR_TIMEOUT, "a bounded device-side wait gave up (flags 0x%x)", flag);
  if (flag != 0) return fail(SLNR_ERR_INDEX, "the inspector found more work than the sizes allow (flags 0x%x)", flag);
  return SLNR_OK;
}

// ---------------------------------------------------------------------------
// layouts per operation

// The fused tensor-core path takes row segments; everything else splits heavy rows.
bool use_tc(const slnr_opts* o, int32_t K, int32_t L) { return o->allow_tf32 != 0 && tc_supported(K, L); }

// The fused tensor-core kernel (persistent CTAs, tensor memory, an inspector
// pass) pays a fixed cost of some tens of microseconds; below this many
// nonzeros the fused CUDA-core kernels finish first.
constexpr int64_t kTcFusedMinNnz = int64_t(1) << 14;
bool use_tc_fused(const slnr_opts* o, int32_t K, int32_t L, int64_t nnz) {
  return o->variant == SLNR_FUSED && use_tc(o, K, L) && nnz >= kTcFusedMinNnz;
}

Layout layout_spmm_gemm(const slnr_csr* B, int32_t K, int32_t L, const slnr_opts* o) {
  Layout l;
  if (use_tc_fused(o, K, L, B->nnz)) {
    l.segs(B->nrows, B->nnz, L);
  } else {
    l.split(B->nrows, B->nnz, K);
    if (o->variant == SLNR_UNFUSED) l.inter(sizeof(float) * (size_t)B->nrows * (size_t)K);
  }
  return l;
}

Layout layout_sddmm_spmm(const slnr_csr* B, int32_t L, int32_t K, int variant) {
  (void)L;
  Layout l;
  l.split(B->nrows, B->nnz, K);
  if (variant == SLNR_UNFUSED) l.inter(sizeof(float) * (size_t)B->nnz);
  return l;
}

Layout layout_mttkrp(const slnr_csf3* B, int32_t L, int variant) {
  Layout l;
  l.units(B->nslices, B->nnz, L);
  if (variant == SLNR_UNFUSED) {
    l.split(B->nfibers, B->nnz, L);
    l.inter(sizeof(float) * (size_t)B->nfibers * (size_t)L);
  }
  return l;
}

Layout layout_spttm_ttm(const slnr_csf3* B, int32_t L, int32_t M, const slnr_opts* o) {
  Layout l;
  if (use_tc_fused(o, L, M, B->nnz)) {
    l.segs(B->nfibers, B->nnz, M);
  } else {
    l.split(B->nfibers, B->nnz, L);
    if (o->variant == SLNR_UNFUSED) l.inter(sizeof(float) * (size_t)B->nfibers * (size_t)L);
  }
  return l;
}

// The fused <SDDMM,SpMM,GEMM> runs on the tensor-core kernel (sampled rows)
// when TF32 is allowed and the dot product and the temporary have one width.
bool use_tc_sampled(const slnr_opts* o, int32_t K, int32_t L, int32_t M, int64_t nnz) {
  return o->variant == SLNR_FUSED && o->allow_tf32 != 0 && tc_sampled_supported(K, L, M) && nnz >= kTcFusedMinNnz;
}

Layout layout_sddmm_spmm_gemm(const slnr_csr* B, int32_t K, int32_t L, int32_t M, const slnr_opts* o) {
  const int variant = o->variant;
  Layout l;
  if (use_tc_sampled(o, K, L, M, B->nnz)) {
    l.segs(B->nrows, B->nnz, M);
    return l;
  }
  l.split(B->nrows, B->nnz, L);
  if (variant == SLNR_UNFUSED) {
    l.inter(sizeof(float) * (size_t)B->nnz);                      // Y
    l.inter2(sizeof(float) * (size_t)B->nrows * (size_t)L);       // T = Y.F
  }
  return l;
}

Layout layout_mttkrp_gemm(const slnr_csf3* B, int32_t L, int variant) {
  Layout l;
  l.units(B->nslices, B->nnz, L);
  if (variant == SLNR_UNFUSED) {
    l.split(B->nfibers, B->nnz, L);
    l.inter(sizeof(float) * (size_t)B->nfibers * (size_t)L);      // per-fiber T
    l.inter2(sizeof(float) * (size_t)B->dim[0] * (size_t)L);      // the MTTKRP result
  }
  return l;
}

CsrView csr_view(const slnr_csr* B) { return CsrView{B->nrows, B->ncols, B->nnz, B->pos, B->crd, B->vals}; }
CsrView fiber_view(const slnr_csf3* B) {
  return CsrView{B->nfibers, B->dim[2], B->nnz, B->pos3, B->crd3, B->vals};
}

// ---------------------------------------------------------------------------
// widths outside the specialised kernels (wide.cu): the same schedules with
// the width chosen at run time

// <SpMM,GEMM> shape (also <SpTTM,SpTTM> over fibers and, with C2, <SpMMH,GEMM>):
// A = B . (C [.* C2]) . D, C2 NULL or the Hadamard partner of C
slnr_status wide_spmm_gemm(const CsrView& v, const float* C, const float* C2, int32_t K, const float* D, int32_t L,
                           float* A, char* ws, const Layout& l, int variant, bool tc, cudaStream_t s) {
  const SplitPlan sp = split_plan(ws, l);
  SLNR_LAUNCH("classify", launch_classify(v, sp, s));
  if (variant == SLNR_FUSED) {
    SLNR_LAUNCH("w_spmm_chunks", launch_w_spmm(K, v, C, C2, nullptr, sp, s));
    SLNR_LAUNCH("w_spmm_gemm_tiles", launch_w_spmm_gemm_tiles(K, L, v, C, C2, D, A, s));
    SLNR_LAUNCH("w_combine", launch_w_combine(K, sp, D, L, A, s));
  } else {
    float* T = reinterpret_cast<float*>(ws + l.o_inter);
    SLNR_LAUNCH("w_spmm", launch_w_spmm(K, v, C, C2, T, sp, s));
    SLNR_LAUNCH("w_combine", launch_w_combine(K, sp, nullptr, 0, T, s));
    if (tc)
      SLNR_LAUNCH("tc_dense_gemm", launch_tc_dense_gemm(v.nrows, K, L, T, D, A, sp.hdr, s));
    else
      SLNR_LAUNCH("w_dense_gemm", launch_w_dense_gemm(v.nrows, K, L, T, D, A, s));
  }
  return SLNR_OK;
}

// MTTKRP (E NULL) or <MTTKRP,GEMM> (times E, L x M); the units are already listed
slnr_status wide_mttkrp(const slnr_csf3* B, const float* C, const float* D, int32_t L, const float* E, int32_t M,
                        float* A, char* ws, const Layout& l, const UnitPlan& up, int variant, bool tc,
                        cudaStream_t s) {
  if (variant == SLNR_FUSED) {
    SLNR_LAUNCH("w_mttkrp_units", launch_w_mttkrp_units(L, *B, C, D, nullptr, up, s));
    SLNR_LAUNCH("w_mttkrp_combine", launch_w_mttkrp_combine(L, *B, up, E, M, A, s));
    return SLNR_OK;
  }
  const CsrView fv = fiber_view(B);
  const SplitPlan sp = split_plan(ws, l);
  float* T = reinterpret_cast<float*>(ws + l.o_inter);
  SLNR_LAUNCH("classify", launch_classify(fv, sp, s));
  SLNR_LAUNCH("w_spmm", launch_w_spmm(L, fv, D, nullptr, T, sp, s));
  SLNR_LAUNCH("w_combine", launch_w_combine(L, sp, nullptr, 0, T, s));
  SLNR_LAUNCH("w_mttkrp_units", launch_w_mttkrp_units(L, *B, C, nullptr, T, up, s));
  if (E == nullptr) {
    SLNR_LAUNCH("w_mttkrp_combine", launch_w_mttkrp_combine(L, *B, up, nullptr, 0, A, s));
    return SLNR_OK;
  }
  float* U = reinterpret_cast<float*>(ws + l.o_inter2);
  SLNR_LAUNCH("w_mttkrp_combine", launch_w_mttkrp_combine(L, *B, up, nullptr, 0, U, s));
  if (tc)
    SLNR_LAUNCH("tc_dense_gemm", launch_tc_dense_gemm(B->dim[0], L, M, U, E, A, sp.hdr, s));
  else
    SLNR_LAUNCH("w_dense_gemm", launch_w_dense_gemm(B->dim[0], L, M, U, E, A, s));
  return SLNR_OK;
}

}  // namespace

void slnr::set_last_error(const char* msg) { snprintf(g_last_error, sizeof(g_last_error), "%s", msg); }

long long slnr::wait_limit_cycles() { return g_wait_limit > 0 ? g_wait_limit : kWaitCycles; }

void slnr::note_launch() { ++g_launches; }

// ===========================================================================

extern "C" {

const char* slnr_status_string(slnr_status s) {
  switch (s) {
    case SLNR_OK: return "SLNR_OK";
    case SLNR_ERR_NULL: return "SLNR_ERR_NULL";
    case SLNR_ERR_SHAPE: return "SLNR_ERR_SHAPE";
    case SLNR_ERR_INDEX: return "SLNR_ERR_INDEX";
    case SLNR_ERR_WORKSPACE: return "SLNR_ERR_WORKSPACE";
    case SLNR_ERR_UNSUPPORTED: return "SLNR_ERR_UNSUPPORTED";
    case SLNR_ERR_CUDA: return "SLNR_ERR_CUDA";
    case SLNR_ERR_TIMEOUT: return "SLNR_ERR_TIMEOUT";
  }
  return "SLNR_ERR_UNKNOWN";
}

const char* slnr_last_error(void) { return g_last_error; }

const char* slnr_version(void) { return "slnr 0.2.0 (sm_103a)"; }

slnr_status slnr_peak_ffma(void* stream, double* tflops) {
  if (!tflops) return fail(SLNR_ERR_NULL, "tflops is NULL");
  SLNR_CUDA(peak_ffma(static_cast<cudaStream_t>(stream), tflops));
  return SLNR_OK;
}

slnr_status slnr_peak_tf32(void* stream, double* tflops) {
  if (!tflops) return fail(SLNR_ERR_NULL, "tflops is NULL");
  const cudaError_t e = peak_tf32(static_cast<cudaStream_t>(stream), tflops);
  if (e == cudaErrorLaunchTimeout) return fail(SLNR_ERR_TIMEOUT, "the TF32 peak kernel's wait gave up");
  SLNR_CUDA(e);
  return SLNR_OK;
}

slnr_status slnr_peak_gather(const float* table, int64_t rows, int width, void* stream, double* gbs) {
  if (!table || !gbs) return fail(SLNR_ERR_NULL, "table or gbs is NULL");
  if (rows < 1 || rows > INT32_MAX) return fail(SLNR_ERR_SHAPE, "rows must be in [1, 2^31)");
  if (width < 4 || width > 128 || (width & (width - 1)) != 0)
    return fail(SLNR_ERR_SHAPE, "width must be a power of two in [4, 128]");
  if (!aligned16(table)) return fail(SLNR_ERR_UNSUPPORTED, "table must be 16-byte aligned");
  SLNR_CUDA(peak_gather(table, rows, width, static_cast<cudaStream_t>(stream), gbs));
  return SLNR_OK;
}

slnr_status slnr_set_wait_limit(int64_t cycles) {
  if (cycles < 0) return fail(SLNR_ERR_SHAPE, "wait limit must be >= 0");
  g_wait_limit = cycles;
  return SLNR_OK;
}

slnr_status slnr_timing_enable(int32_t on) {
  if (on && !g_timing.created) {
    for (int i = 0; i <= kMaxTimed; ++i) SLNR_CUDA(cudaEventCreate(&g_timing.ev[i]));
    g_timing.created = true;
  }
  g_timing.on = on != 0;
  g_timing.n = 0;
  return SLNR_OK;
}

int32_t slnr_timing_count(void) { return g_timing.on ? g_timing.n : 0; }

int32_t slnr_timing_launches(void) { return g_launches; }

slnr_status slnr_timing_get(int32_t i, const char** name, float* ms) {
  if (!g_timing.on || i < 0 || i >= g_timing.n) return fail(SLNR_ERR_SHAPE, "no timed launch %d", (int)i);
  if (!name || !ms) return fail(SLNR_ERR_NULL, "name or ms is NULL");
  SLNR_CUDA(cudaEventSynchronize(g_timing.ev[g_timing.n]));
  SLNR_CUDA(cudaEventElapsedTime(ms, g_timing.ev[i], g_timing.ev[i + 1]));
  *name = g_timing.names[i];
  return SLNR_OK;
}

slnr_status slnr_spmm_gemm_workspace(const slnr_csr* B, int32_t K, int32_t L, const slnr_opts* opts,
                                     size_t* bytes) {
  SLNR_CHECK(check_opts(opts));
  SLNR_CHECK(check_csr(B, false));
  SLNR_CHECK(check_dims("K", K));
  SLNR_CHECK(check_dims("L", L));
  if (!bytes) return fail(SLNR_ERR_NULL, "bytes is NULL");
  *bytes = layout_spmm_gemm(B, K, L, opts).total();
  return SLNR_OK;
}

slnr_status slnr_sddmm_spmm_workspace(const slnr_csr* B, int32_t L, int32_t K, const slnr_opts* opts,
                                      size_t* bytes) {
  SLNR_CHECK(check_opts(opts));
  SLNR_CHECK(check_csr(B, false));
  SLNR_CHECK(check_dims("L", L));
  SLNR_CHECK(check_dims("K", K));
  if (!bytes) return fail(SLNR_ERR_NULL, "bytes is NULL");
  *bytes = layout_sddmm_spmm(B, L, K, opts->variant).total();
  return SLNR_OK;
}

slnr_status slnr_mttkrp_workspace(const slnr_csf3* B, int32_t L, const slnr_opts* opts, size_t* bytes) {
  SLNR_CHECK(check_opts(opts));
  SLNR_CHECK(check_csf(B, false));
  SLNR_CHECK(check_dims("L", L));
  if (!bytes) return fail(SLNR_ERR_NULL, "bytes is NULL");
  *bytes = layout_mttkrp(B, L, opts->variant).total();
  return SLNR_OK;
}

slnr_status slnr_spttm_ttm_workspace(const slnr_csf3* B, int32_t L, int32_t M, const slnr_opts* opts,
                                     size_t* bytes) {
  SLNR_CHECK(check_opts(opts));
  SLNR_CHECK(check_csf(B, false));
  SLNR_CHECK(check_dims("L", L));
  SLNR_CHECK(check_dims("M", M));
  if (!bytes) return fail(SLNR_ERR_NULL, "bytes is NULL");
  *bytes = layout_spttm_ttm(B, L, M, opts).total();
  return SLNR_OK;
}

slnr_status slnr_sddmm_spmm_gemm_workspace(const slnr_csr* B, int32_t K, int32_t L, int32_t M, const slnr_opts* opts,
                                           size_t* bytes) {
  SLNR_CHECK(check_opts(opts));
  SLNR_CHECK(check_csr(B, false));
  SLNR_CHECK(check_dims("K", K));
  SLNR_CHECK(check_dims("L", L));
  SLNR_CHECK(check_dims("M", M));
  if (!bytes) return fail(SLNR_ERR_NULL, "bytes is NULL");
  *bytes = layout_sddmm_spmm_gemm(B, K, L, M, opts).total();
  return SLNR_OK;
}

slnr_status slnr_mttkrp_gemm_workspace(const slnr_csf3* B, int32_t L, int32_t M, const slnr_opts* opts,
                                       size_t* bytes) {
  SLNR_CHECK(check_opts(opts));
  SLNR_CHECK(check_csf(B, false));
  SLNR_CHECK(check_dims("L", L));
  SLNR_CHECK(check_dims("M", M));
  if (!bytes) return fail(SLNR_ERR_NULL, "bytes is NULL");
  *bytes = layout_mttkrp_gemm(B, L, opts->variant).total();
  return SLNR_OK;
}

slnr_status slnr_spmmh_gemm_workspace(const slnr_csr* B, int32_t J, int32_t L, const slnr_opts* opts,
                                      size_t* bytes) {
  SLNR_CHECK(check_opts(opts));
  SLNR_CHECK(check_csr(B, false));
  SLNR_CHECK(check_dims("J", J));
  SLNR_CHECK(check_dims("L", L));
  if (!bytes) return fail(SLNR_ERR_NULL, "bytes is NULL");
  *bytes = layout_spmm_gemm(B, J, L, opts).total();
  return SLNR_OK;
}

slnr_status slnr_spmm_gemm(const slnr_csr* B, const float* C, int32_t K, const float* D, int32_t L, float* A,
                           const slnr_opts* opts) {
  g_last_error[0] = '\0';
  timing_begin();
  SLNR_CHECK(check_opts(opts));
  SLNR_CHECK(check_csr(B, true));
  SLNR_CHECK(check_dims("K", K));
  SLNR_CHECK(check_dims("L", L));
  SLNR_CHECK(check_dense("C", C));
  SLNR_CHECK(check_dense("D", D));
  SLNR_CHECK(check_dense("A", A));
  const Layout l = layout_spmm_gemm(B, K, L, opts);
  SLNR_CHECK(check_ws(opts, l.total()));
  if (B->nrows == 0) return SLNR_OK;
  cudaStream_t s = static_cast<cudaStream_t>(opts->stream);
  char* ws = static_cast<char*>(opts->workspace);
  SLNR_CHECK(begin(ws, s, opts->validate != 0,
                   [&](WsHeader* h) { return launch_validate_csr(*B, h, s); }));
  const CsrView v = csr_view(B);
  const bool tc = use_tc(opts, K, L);
  if (use_tc_fused(opts, K, L, B->nnz)) {
    const SegPlan gp = seg_plan(ws, l);
    SLNR_LAUNCH("seg_count", launch_seg_count(v, gp, s));
    SLNR_LAUNCH("seg_write", launch_seg_write(v, gp, s));
    SLNR_LAUNCH("tc_spmm_gemm", launch_tc_spmm_gemm(K, L, v, C, D, A, gp, s));
    SLNR_LAUNCH("combine", launch_combine(L, combine_plan(gp), nullptr, 0, A, s));
  } else if (!all_pow2(K, L)) {
    SLNR_CHECK(wide_spmm_gemm(v, C, nullptr, K, D, L, A, ws, l, opts->variant, tc, s));
  } else {
    const SplitPlan sp = split_plan(ws, l);
    SLNR_LAUNCH("classify", launch_classify(v, sp, s));
    SLNR_LAUNCH("spmm_chunks", launch_spmm_chunks(K, v, C, sp, s));
    if (opts->variant == SLNR_FUSED) {
      SLNR_LAUNCH("spmm_gemm_tiles", launch_spmm_gemm_tiles(K, L, v, C, D, A, 0, s));
      SLNR_LAUNCH("combine", launch_combine(K, sp, D, L, A, s));
    } else {
      float* T = reinterpret_cast<float*>(ws + l.o_inter);
      SLNR_LAUNCH("spmm_rows", launch_spmm_rows(K, v, C, T, s));
      SLNR_LAUNCH("combine", launch_combine(K, sp, nullptr, 0, T, s));
      if (tc)
        SLNR_LAUNCH("tc_dense_gemm", launch_tc_dense_gemm(B->nrows, K, L, T, D, A, sp.hdr, s));
      else
        SLNR_LAUNCH("dense_gemm", launch_dense_gemm(B->nrows, K, L, T, D, A, 0, s));
    }
  }
  return finish(ws, s, opts->validate != 0);
}

slnr_status slnr_sddmm_spmm(const slnr_csr* B, const float* C, const float* D, int32_t L, const float* E,
                            int32_t K, float* A, const slnr_opts* opts) {
  g_last_error[0] = '\0';
  timing_begin();
  SLNR_CHECK(check_opts(opts));
  SLNR_CHECK(check_csr(B, true));
  SLNR_CHECK(check_dims("L", L));
  SLNR_CHECK(check_dims("K", K));
  SLNR_CHECK(check_dense("C", C));
  SLNR_CHECK(check_dense("D", D));
  SLNR_CHECK(check_dense("E", E));
  SLNR_CHECK(check_dense("A", A));
  const Layout l = layout_sddmm_spmm(B, L, K, opts->variant);
  SLNR_CHECK(check_ws(opts, l.total()));
  if (B->nrows == 0) return SLNR_OK;
  cudaStream_t s = static_cast<cudaStream_t>(opts->stream);
  char* ws = static_cast<char*>(opts->workspace);
  SLNR_CHECK(begin(ws, s, opts->validate != 0,
                   [&](WsHeader* h) { return launch_validate_csr(*B, h, s); }));
  const CsrView v = csr_view(B);
  const SplitPlan sp = split_plan(ws, l);
  SLNR_LAUNCH("classify", launch_classify(v, sp, s));
  if (!all_pow2(L, K)) {
    if (opts->variant == SLNR_FUSED) {
      SLNR_LAUNCH("w_sddmm_spmm", launch_w_sddmm_spmm(v, C, D, L, E, K, A, nullptr, sp, s));
    } else {
      float* Y = reinterpret_cast<float*>(ws + l.o_inter);
      SLNR_LAUNCH("w_sddmm", launch_w_sddmm_spmm(v, C, D, L, nullptr, K, nullptr, Y, sp, s));
      CsrView vy = v;
      vy.vals = Y;
      SLNR_LAUNCH("w_spmm", launch_w_spmm(K, vy, E, nullptr, A, sp, s));
    }
    SLNR_LAUNCH("w_combine", launch_w_combine(K, sp, nullptr, 0, A, s));
  } else if (opts->variant == SLNR_FUSED) {
    SLNR_LAUNCH("sddmm_spmm_rows", launch_sddmm_spmm_rows(v, C, D, L, E, K, A, sp, s));
    SLNR_LAUNCH("combine", launch_combine(K, sp, nullptr, 0, A, s));
  } else {
    float* Y = reinterpret_cast<float*>(ws + l.o_inter);
    SLNR_LAUNCH("sddmm_rows", launch_sddmm_rows(v, C, D, L, Y, s));
    SLNR_LAUNCH("sddmm_chunks", launch_sddmm_chunks(v, C, D, L, Y, sp, s));
    CsrView vy = v;
    vy.vals = Y;
    SLNR_LAUNCH("spmm_chunks", launch_spmm_chunks(K, vy, E, sp, s));
    SLNR_LAUNCH("spmm_rows", launch_spmm_rows(K, vy, E, A, s));
    SLNR_LAUNCH("combine", launch_combine(K, sp, nullptr, 0, A, s));
  }
  return finish(ws, s, opts->validate != 0);
}

slnr_status slnr_mttkrp(const slnr_csf3* B, const float* C, const float* D, int32_t L, float* A,
                        const slnr_opts* opts) {
  g_last_error[0] = '\0';
  timing_begin();
  SLNR_CHECK(check_opts(opts));
  SLNR_CHECK(check_csf(B, true));
  SLNR_CHECK(check_dims("L", L));
  SLNR_CHECK(check_dense("C", C));
  SLNR_CHECK(check_dense("D", D));
  SLNR_CHECK(check_dense("A", A));
  const Layout l = layout_mttkrp(B, L, opts->variant);
  SLNR_CHECK(check_ws(opts, l.total()));
  if (B->dim[0] == 0) return SLNR_OK;
  cudaStream_t s = static_cast<cudaStream_t>(opts->stream);
  char* ws = static_cast<char*>(opts->workspace);
  SLNR_CHECK(begin(ws, s, opts->validate != 0,
                   [&](WsHeader* h) { return launch_validate_csf(*B, h, s); }));
  const UnitPlan up = unit_plan(ws, l);
  SLNR_LAUNCH("csf_units", launch_csf_units(*B, up, s));
  if (!pow2_dim(L)) {
    SLNR_CHECK(wide_mttkrp(B, C, D, L, nullptr, 0, A, ws, l, up, opts->variant, false, s));
    return finish(ws, s, opts->validate != 0);
  }
  if (opts->variant == SLNR_FUSED) {
    SLNR_LAUNCH("mttkrp_units", launch_mttkrp_units(L, *B, C, D, up, s));
  } else {
    const CsrView fv = fiber_view(B);
    const SplitPlan sp = split_plan(ws, l);
    float* T = reinterpret_cast<float*>(ws + l.o_inter);
    SLNR_LAUNCH("classify", launch_classify(fv, sp, s));
    SLNR_LAUNCH("spmm_chunks", launch_spmm_chunks(L, fv, D, sp, s));
    SLNR_LAUNCH("spmm_rows", launch_spmm_rows(L, fv, D, T, s));
    SLNR_LAUNCH("combine", launch_combine(L, sp, nullptr, 0, T, s));
    SLNR_LAUNCH("mttkrp_stage2_units", launch_mttkrp_stage2_units(L, *B, T, C, up, s));
  }
  SLNR_LAUNCH("mttkrp_combine", launch_mttkrp_combine(L, *B, up, nullptr, 0, A, s));
  return finish(ws, s, opts->validate != 0);
}

slnr_status slnr_spttm_ttm(const slnr_csf3* B, const float* C, int32_t L, const float* D, int32_t M,
                           int32_t* A_pos1, int32_t* A_crd1, int32_t* A_pos2, int32_t* A_crd2, float* A_vals,
                           const slnr_opts* opts) {
  g_last_error[0] = '\0';
  timing_begin();
  SLNR_CHECK(check_opts(opts));
  SLNR_CHECK(check_csf(B, true));
  SLNR_CHECK(check_dims("L", L));
  SLNR_CHECK(check_dims("M", M));
  SLNR_CHECK(check_dense("C", C));
  SLNR_CHECK(check_dense("D", D));
  if (!A_pos1 || !A_pos2 || (B->nslices > 0 && !A_crd1) || (B->nfibers > 0 && !A_crd2))
    return fail(SLNR_ERR_NULL, "an output index array of A is NULL");
  if (B->nfibers > 0) SLNR_CHECK(check_dense("A_vals", A_vals));
  const Layout l = layout_spttm_ttm(B, L, M, opts);
  SLNR_CHECK(check_ws(opts, l.total()));
  cudaStream_t s = static_cast<cudaStream_t>(opts->stream);
  char* ws = static_cast<char*>(opts->workspace);
  SLNR_CHECK(begin(ws, s, opts->validate != 0,
                   [&](WsHeader* h) { return launch_validate_csf(*B, h, s); }));
  // A's two compressed levels are B's (the (i,j) pattern is unchanged)
  SLNR_LAUNCH("copy_levels", launch_copy_levels(*B, A_pos1, A_crd1, A_pos2, A_crd2, s));
  if (B->nfibers == 0) return SLNR_OK;
  const CsrView fv = fiber_view(B);
  const bool tc = use_tc(opts, L, M);
  if (use_tc_fused(opts, L, M, B->nnz)) {
    const SegPlan gp = seg_plan(ws, l);
    SLNR_LAUNCH("seg_count", launch_seg_count(fv, gp, s));
    SLNR_LAUNCH("seg_write", launch_seg_write(fv, gp, s));
    SLNR_LAUNCH("tc_spmm_gemm", launch_tc_spmm_gemm(L, M, fv, C, D, A_vals, gp, s));
    SLNR_LAUNCH("combine", launch_combine(M, combine_plan(gp), nullptr, 0, A_vals, s));
  } else if (!all_pow2(L, M)) {
    SLNR_CHECK(wide_spmm_gemm(fv, C, nullptr, L, D, M, A_vals, ws, l, opts->variant, tc, s));
  } else {
    const SplitPlan sp = split_plan(ws, l);
    SLNR_LAUNCH("classify", launch_classify(fv, sp, s));
    SLNR_LAUNCH("spmm_chunks", launch_spmm_chunks(L, fv, C, sp, s));
    if (opts->variant == SLNR_FUSED) {
      SLNR_LAUNCH("spmm_gemm_tiles", launch_spmm_gemm_tiles(L, M, fv, C, D, A_vals, 0, s));
      SLNR_LAUNCH("combine", launch_combine(L, sp, D, M, A_vals, s));
    } else {
      float* T = reinterpret_cast<float*>(ws + l.o_inter);
      SLNR_LAUNCH("spmm_rows", launch_spmm_rows(L, fv, C, T, s));
      SLNR_LAUNCH("combine", launch_combine(L, sp, nullptr, 0, T, s));
      if (tc)
        SLNR_LAUNCH("tc_dense_gemm", launch_tc_dense_gemm(B->nfibers, L, M, T, D, A_vals, sp.hdr, s));
      else
        SLNR_LAUNCH("dense_gemm", launch_dense_gemm(B->nfibers, L, M, T, D, A_vals, 0, s));
    }
  }
  return finish(ws, s, opts->validate != 0);
}

slnr_status slnr_sddmm_spmm_gemm(const slnr_csr* B, const float* C, const float* D, int32_t K, const float* F,
                                 int32_t L, const float* W, int32_t M, float* A, const slnr_opts* opts) {
  g_last_error[0] = '\0';
  timing_begin();
  SLNR_CHECK(check_opts(opts));
  SLNR_CHECK(check_csr(B, true));
  SLNR_CHECK(check_dims("K", K));
  SLNR_CHECK(check_dims("L", L));
  SLNR_CHECK(check_dims("M", M));
  SLNR_CHECK(check_dense("C", C));
  SLNR_CHECK(check_dense("D", D));
  SLNR_CHECK(check_dense("F", F));
  SLNR_CHECK(check_dense("W", W));
  SLNR_CHECK(check_dense("A", A));
  const Layout l = layout_sddmm_spmm_gemm(B, K, L, M, opts);
  SLNR_CHECK(check_ws(opts, l.total()));
  if (B->nrows == 0) return SLNR_OK;
  cudaStream_t s = static_cast<cudaStream_t>(opts->stream);
  char* ws = static_cast<char*>(opts->workspace);
  SLNR_CHECK(begin(ws, s, opts->validate != 0,
                   [&](WsHeader* h) { return launch_validate_csr(*B, h, s); }));
  const CsrView v = csr_view(B);
  if (use_tc_sampled(opts, K, L, M, B->nnz)) {
    // T(i,:) built on chip by the producers, T.W on the TF32 tensor cores;
    // heavy rows' chunk rows of A are summed by the combine
    const SegPlan gp = seg_plan(ws, l);
    SLNR_LAUNCH("seg_count", launch_seg_count(v, gp, s));
    SLNR_LAUNCH("seg_write", launch_seg_write(v, gp, s));
    SLNR_LAUNCH("tc_sddmm_spmm_gemm", launch_tc_sddmm_spmm_gemm(v, C, D, F, L, W, M, A, gp, s));
    SLNR_LAUNCH("combine", launch_combine(M, combine_plan(gp), nullptr, 0, A, s));
    return finish(ws, s, opts->validate != 0);
  }
  const SplitPlan sp = split_plan(ws, l);
  SLNR_LAUNCH("classify", launch_classify(v, sp, s));
  if (!all_pow2(K, L, M)) {
    if (opts->variant == SLNR_FUSED) {
      SLNR_LAUNCH("w_sddmm_spmm_chunks", launch_w_sddmm_spmm(v, C, D, K, F, L, nullptr, nullptr, sp, s));
      SLNR_LAUNCH("w_sddmm_spmm_gemm_tiles", launch_w_sddmm_spmm_gemm_tiles(v, C, D, K, F, L, W, M, A, s));
      SLNR_LAUNCH("w_combine", launch_w_combine(L, sp, W, M, A, s));
    } else {
      float* Y = reinterpret_cast<float*>(ws + l.o_inter);
      float* T = reinterpret_cast<float*>(ws + l.o_inter2);
      SLNR_LAUNCH("w_sddmm", launch_w_sddmm_spmm(v, C, D, K, nullptr, L, nullptr, Y, sp, s));
      CsrView vy = v;
      vy.vals = Y;
      SLNR_LAUNCH("w_spmm", launch_w_spmm(L, vy, F, nullptr, T, sp, s));
      SLNR_LAUNCH("w_combine", launch_w_combine(L, sp, nullptr, 0, T, s));
      if (use_tc(opts, L, M))
        SLNR_LAUNCH("tc_dense_gemm", launch_tc_dense_gemm(B->nrows, L, M, T, W, A, sp.hdr, s));
      else
        SLNR_LAUNCH("w_dense_gemm", launch_w_dense_gemm(B->nrows, L, M, T, W, A, s));
    }
  } else if (opts->variant == SLNR_FUSED) {
    // heavy rows: partial T rows (width L), then their fixed-order sum times W
    SLNR_LAUNCH("sddmm_spmm_chunks", launch_sddmm_spmm_chunks(v, C, D, K, F, L, sp, s));
    SLNR_LAUNCH("sddmm_spmm_gemm_tiles", launch_sddmm_spmm_gemm_tiles(v, C, D, K, F, L, W, M, A, s));
    SLNR_LAUNCH("combine", launch_combine(L, sp, W, M, A, s));
  } else {
    float* Y = reinterpret_cast<float*>(ws + l.o_inter);
    float* T = reinterpret_cast<float*>(ws + l.o_inter2);
    SLNR_LAUNCH("sddmm_rows", launch_sddmm_rows(v, C, D, K, Y, s));
    SLNR_LAUNCH("sddmm_chunks", launch_sddmm_chunks(v, C, D, K, Y, sp, s));
    CsrView vy = v;
    vy.vals = Y;
    SLNR_LAUNCH("spmm_chunks", launch_spmm_chunks(L, vy, F, sp, s));
    SLNR_LAUNCH("spmm_rows", launch_spmm_rows(L, vy, F, T, s));
    SLNR_LAUNCH("combine", launch_combine(L, sp, nullptr, 0, T, s));
    if (use_tc(opts, L, M))
      SLNR_LAUNCH("tc_dense_gemm", launch_tc_dense_gemm(B->nrows, L, M, T, W, A, sp.hdr, s));
    else
      SLNR_LAUNCH("dense_gemm", launch_dense_gemm(B->nrows, L, M, T, W, A, 0, s));
  }
  return finish(ws, s, opts->validate != 0);
}

slnr_status slnr_mttkrp_gemm(const slnr_csf3* B, const float* C, const float* D, int32_t L, const float* E,
                             int32_t M, float* A, const slnr_opts* opts) {
  g_last_error[0] = '\0';
  timing_begin();
  SLNR_CHECK(check_opts(opts));
  SLNR_CHECK(check_csf(B, true));
  SLNR_CHECK(check_dims("L", L));
  SLNR_CHECK(check_dims("M", M));
  SLNR_CHECK(check_dense("C", C));
  SLNR_CHECK(check_dense("D", D));
  SLNR_CHECK(check_dense("E", E));
  SLNR_CHECK(check_dense("A", A));
  const Layout l = layout_mttkrp_gemm(B, L, opts->variant);
  SLNR_CHECK(check_ws(opts, l.total()));
  if (B->dim[0] == 0) return SLNR_OK;
  cudaStream_t s = static_cast<cudaStream_t>(opts->stream);
  char* ws = static_cast<char*>(opts->workspace);
  SLNR_CHECK(begin(ws, s, opts->validate != 0,
                   [&](WsHeader* h) { return launch_validate_csf(*B, h, s); }));
  const UnitPlan up = unit_plan(ws, l);
  SLNR_LAUNCH("csf_units", launch_csf_units(*B, up, s));
  if (!all_pow2(L, M)) {
    SLNR_CHECK(wide_mttkrp(B, C, D, L, E, M, A, ws, l, up, opts->variant, use_tc(opts, L, M), s));
  } else if (opts->variant == SLNR_FUSED) {
    SLNR_LAUNCH("mttkrp_units", launch_mttkrp_units(L, *B, C, D, up, s));
    SLNR_LAUNCH("mttkrp_combine", launch_mttkrp_combine(L, *B, up, E, M, A, s));
  } else {
    const CsrView fv = fiber_view(B);
    const SplitPlan sp = split_plan(ws, l);
    float* T = reinterpret_cast<float*>(ws + l.o_inter);
    float* U = reinterpret_cast<float*>(ws + l.o_inter2);
    SLNR_LAUNCH("classify", launch_classify(fv, sp, s));
    SLNR_LAUNCH("spmm_chunks", launch_spmm_chunks(L, fv, D, sp, s));
    SLNR_LAUNCH("spmm_rows", launch_spmm_rows(L, fv, D, T, s));
    SLNR_LAUNCH("combine", launch_combine(L, sp, nullptr, 0, T, s));
    SLNR_LAUNCH("mttkrp_stage2_units", launch_mttkrp_stage2_units(L, *B, T, C, up, s));
    SLNR_LAUNCH("mttkrp_combine", launch_mttkrp_combine(L, *B, up, nullptr, 0, U, s));
    if (use_tc(opts, L, M))
      SLNR_LAUNCH("tc_dense_gemm", launch_tc_dense_gemm(B->dim[0], L, M, U, E, A, sp.hdr, s));
    else
      SLNR_LAUNCH("dense_gemm", launch_dense_gemm(B->dim[0], L, M, U, E, A, 0, s));
  }
  return finish(ws, s, opts->validate != 0);
}

slnr_status slnr_spmmh_gemm(const slnr_csr* B, const float* C, const float* D, int32_t J, const float* E,
                            int32_t L, float* A, const slnr_opts* opts) {
  g_last_error[0] = '\0';
  timing_begin();
  SLNR_CHECK(check_opts(opts));
  SLNR_CHECK(check_csr(B, true));
  SLNR_CHECK(check_dims("J", J));
  SLNR_CHECK(check_dims("L", L));
  SLNR_CHECK(check_dense("C", C));
  SLNR_CHECK(check_dense("D", D));
  SLNR_CHECK(check_dense("E", E));
  SLNR_CHECK(check_dense("A", A));
  const Layout l = layout_spmm_gemm(B, J, L, opts);
  SLNR_CHECK(check_ws(opts, l.total()));
  if (B->nrows == 0) return SLNR_OK;
  cudaStream_t s = static_cast<cudaStream_t>(opts->stream);
  char* ws = static_cast<char*>(opts->workspace);
  SLNR_CHECK(begin(ws, s, opts->validate != 0,
                   [&](WsHeader* h) { return launch_validate_csr(*B, h, s); }));
  const CsrView v = csr_view(B);
  const bool tc = use_tc(opts, J, L);
  const bool tc_fused = use_tc_fused(opts, J, L, B->nnz);
  // the gathered row of column k is C(k,:) .* D(k,:); E is the consumer matrix
  if (tc_fused) {
    const SegPlan gp = seg_plan(ws, l);
    SLNR_LAUNCH("seg_count", launch_seg_count(v, gp, s));
    SLNR_LAUNCH("seg_write", launch_seg_write(v, gp, s));
    SLNR_LAUNCH("tc_spmmh_gemm", launch_tc_spmm_gemm(J, L, v, C, E, A, gp, s, D));
    SLNR_LAUNCH("combine", launch_combine(L, combine_plan(gp), nullptr, 0, A, s));
  } else if (!all_pow2(J, L)) {
    SLNR_CHECK(wide_spmm_gemm(v, C, D, J, E, L, A, ws, l, opts->variant, tc, s));
  } else {
    const SplitPlan sp = split_plan(ws, l);
    SLNR_LAUNCH("classify", launch_classify(v, sp, s));
    SLNR_LAUNCH("spmm_chunks", launch_spmm_chunks(J, v, C, sp, s, D));
    if (opts->variant == SLNR_FUSED) {
      SLNR_LAUNCH("spmm_gemm_tiles", launch_spmm_gemm_tiles(J, L, v, C, E, A, 0, s, D));
      SLNR_LAUNCH("combine", launch_combine(J, sp, E, L, A, s));
    } else {
      float* T = reinterpret_cast<float*>(ws + l.o_inter);
      SLNR_LAUNCH("spmm_rows", launch_spmm_rows(J, v, C, T, s, D));
      SLNR_LAUNCH("combine", launch_combine(J, sp, nullptr, 0, T, s));
      if (tc)
        SLNR_LAUNCH("tc_dense_gemm", launch_tc_dense_gemm(B->nrows, J, L, T, E, A, sp.hdr, s));
      else
        SLNR_LAUNCH("dense_gemm", launch_dense_gemm(B->nrows, J, L, T, E, A, 0, s));
    }
  }
  return finish(ws, s, opts->validate != 0);
}

}  // extern "C"
