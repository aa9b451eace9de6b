// Host side of libnmd: argument checks, CSR/CSC and panel-index construction,
// workspace layout, the block schedule of a sweep and the C ABI of nmd.h.
#include <math.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <algorithm>
#include <string>
#include <vector>

#include "nmd_internal.cuh"

using namespace nmd;

#define NMD_VERSION_STRING "libnmd 0.1 (sm_103a)"

namespace {

// ---------------------------------------------------------------------------
// Block order: SplitMix64 (S. Vigna's published generator) driving a
// Fisher-Yates shuffle.  State for (seed, sweep, side) is
// mix(seed) ^ mix((sweep << 1) | side); for i = K-1 down to 1 the block at i
// is swapped with the one at next() % (i + 1).
// ---------------------------------------------------------------------------
inline uint64_t sm64_mix(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

std::vector<int64_t> permutation(uint64_t seed, int64_t sweep, int side, int64_t K) {
  uint64_t state = sm64_mix(seed) ^ sm64_mix((((uint64_t)sweep) << 1) | (uint64_t)side);
  std::vector<int64_t> p(K);
  for (int64_t i = 0; i < K; ++i) p[i] = i;
  for (int64_t i = K - 1; i >= 1; --i) {
    state += 0x9E3779B97F4A7C15ull;
    uint64_t j = sm64_mix(state) % (uint64_t)(i + 1);
    std::swap(p[i], p[(int64_t)j]);
  }
  return p;
}

inline int64_t nblocks(int64_t N, int64_t b) { return (N + b - 1) / b; }

int pad_rank(int r) {
  if (r <= 16) return 16;
  if (r <= 32) return 32;
  if (r <= 64) return 64;
  if (r <= 128) return 128;
  return 256;
}

// ---------------------------------------------------------------------------
// Host copy of S: validated CSR of the positive entries and its transpose.
// ---------------------------------------------------------------------------
struct HostSparse {
  int64_t m = 0, n = 0;
  std::vector<int64_t> rowptr, colptr;
  std::vector<int32_t> col, row;
  std::vector<float> val, valT;
  double s_fro = 0.0;
};

nmd_status check_options(const nmd_options* o, std::string* why) {
  if (!o) { *why = "options pointer is NULL"; return NMD_ERR_INVALID; }
  if (o->block_rows < 1 || o->block_cols < 1) { *why = "block sizes must be >= 1"; return NMD_ERR_INVALID; }
  if (o->schedule != NMD_EXACT && o->schedule != NMD_STOCH) { *why = "unknown schedule"; return NMD_ERR_INVALID; }
  if (o->order != NMD_ALTERNATE && o->order != NMD_PHASED) { *why = "unknown order"; return NMD_ERR_INVALID; }
  if (!(o->eta > 0.0) || !isfinite(o->eta)) { *why = "eta must be a finite positive number"; return NMD_ERR_INVALID; }
  if (!(o->gamma >= 0.0 && o->gamma < 1.0)) { *why = "gamma must lie in [0, 1)"; return NMD_ERR_INVALID; }
  if (!(o->ridge >= 0.0) || !isfinite(o->ridge)) { *why = "ridge must be finite and >= 0"; return NMD_ERR_INVALID; }
  if (o->precision != NMD_BF16 && o->precision != NMD_FP32 && o->precision != NMD_SIMT) {
    *why = "unknown precision"; return NMD_ERR_INVALID;
  }
  if (o->epilogue != NMD_EPI_Z && o->epilogue != NMD_EPI_DELTA) { *why = "unknown epilogue"; return NMD_ERR_INVALID; }
  if (o->skip_zero_chunks < NMD_SKIP_NONE || o->skip_zero_chunks > NMD_SKIP_RANGE) {
    *why = "unknown chunk-skipping mode"; return NMD_ERR_INVALID;
  }
  return NMD_OK;
}

nmd_status build_sparse(int64_t m, int64_t n, int32_t r, const int64_t* row_ptr,
                        const int32_t* col_idx, const float* vals, HostSparse* S,
                        std::string* why) {
  if (m < 1 || n < 1 || m >= (int64_t(1) << 31) || n >= (int64_t(1) << 31)) {
    *why = "m and n must lie in [1, 2^31)"; return NMD_ERR_INVALID;
  }
  if (r < 1 || r > 256) { *why = "rank r must lie in [1, 256]"; return NMD_ERR_INVALID; }
  if (!row_ptr) { *why = "row_ptr is NULL"; return NMD_ERR_INVALID; }
  if (row_ptr[0] != 0) { *why = "row_ptr[0] must be 0"; return NMD_ERR_CSR; }
  for (int64_t i = 0; i < m; ++i)
    if (row_ptr[i + 1] < row_ptr[i]) {
      char b[96]; snprintf(b, sizeof b, "row_ptr decreases at row %lld", (long long)i);
      *why = b; return NMD_ERR_CSR;
    }
  int64_t nnz_in = row_ptr[m];
  if (nnz_in > 0 && (!col_idx || !vals)) { *why = "col_idx or vals is NULL"; return NMD_ERR_INVALID; }
  S->m = m; S->n = n;
  S->rowptr.assign(m + 1, 0);
  S->col.clear(); S->val.clear();
  S->col.reserve(nnz_in); S->val.reserve(nnz_in);
  double fro = 0.0;
  for (int64_t i = 0; i < m; ++i) {
    int64_t prev = -1;
    for (int64_t e = row_ptr[i]; e < row_ptr[i + 1]; ++e) {
      int64_t c = col_idx[e];
      float v = vals[e];
      if (c < 0 || c >= n) {
        char b[128]; snprintf(b, sizeof b, "column index %lld out of range at row %lld", (long long)c, (long long)i);
        *why = b; return NMD_ERR_CSR;
      }
      if (c <= prev) {
        char b[128]; snprintf(b, sizeof b, "columns not strictly increasing in row %lld", (long long)i);
        *why = b; return NMD_ERR_CSR;
      }
      if (!isfinite(v) || v < 0.0f) {
        char b[128]; snprintf(b, sizeof b, "negative or non-finite value in row %lld", (long long)i);
        *why = b; return NMD_ERR_CSR;
      }
      prev = c;
      if (v > 0.0f) {
        S->col.push_back((int32_t)c);
        S->val.push_back(v);
        fro += (double)v * (double)v;
      }
    }
    S->rowptr[i + 1] = (int64_t)S->col.size();
  }
  if (S->col.empty()) { *why = "S has no positive entry (||S||_F = 0)"; return NMD_ERR_CSR; }
  S->s_fro = sqrt(fro);
  // transpose (counting sort by column; rows stay ascending within a column)
  int64_t nnz = (int64_t)S->col.size();
  S->colptr.assign(n + 1, 0);
  for (int64_t e = 0; e < nnz; ++e) S->colptr[S->col[e] + 1]++;
  for (int64_t j = 0; j < n; ++j) S->colptr[j + 1] += S->colptr[j];
  S->row.resize(nnz); S->valT.resize(nnz);
  std::vector<int64_t> cur(S->colptr.begin(), S->colptr.end() - 1);
  for (int64_t i = 0; i < m; ++i)
    for (int64_t e = S->rowptr[i]; e < S->rowptr[i + 1]; ++e) {
      int64_t p = cur[S->col[e]]++;
      S->row[p] = (int32_t)i;
      S->valT[p] = S->val[e];
    }
  return NMD_OK;
}

// Split every block's rows (ascending) into short rows (len <= kShort), whole
// long rows (len <= seg) and slices of seg entries of the longer rows, with
// seg = the largest of kSegMax, kSegMax / 2, ... kSegMin whose segments of the
// block's long rows number at least kSegTarget (else kSegMin).
void finalize_panels(const std::vector<std::vector<PanelRow>>& per, PanelSet* P) {
  int64_t K = (int64_t)per.size();
  P->host.clear(); P->seg.clear(); P->multi.clear();
  P->row_ptr.assign(K + 1, 0);
  P->seg_ptr.assign(K + 1, 0);
  P->multi_ptr.assign(K + 1, 0);
  P->segd.assign(K, 0);
  P->max_segments = 0;
  for (int64_t k = 0; k < K; ++k) {
    P->row_ptr[k] = (int64_t)P->host.size();
    P->seg_ptr[k] = (int64_t)P->seg.size();
    P->multi_ptr[k] = (int64_t)P->multi.size();
    int64_t long_entries = 0;
    for (const PanelRow& pr : per[k])
      if (pr.len > kShort) long_entries += pr.len;
    int seg = kSegMax;
    while (seg > kSegMin && long_entries / seg < kSegTarget) seg /= 2;
    for (const PanelRow& pr : per[k]) {
      if (pr.len <= kShort) P->host.push_back(pr);
      else if (pr.len <= seg) P->seg.push_back(pr);
    }
    P->segd[k] = (int64_t)P->seg.size() - P->seg_ptr[k];
    const int64_t s0 = (int64_t)P->seg.size();
    for (const PanelRow& pr : per[k]) {
      if (pr.len <= seg) continue;
      int64_t first = (int64_t)P->seg.size() - s0;   // slot within the block's slices
      int32_t nseg = 0;
      for (int64_t off = 0; off < pr.len; off += seg, ++nseg)
        P->seg.push_back(PanelRow{pr.row, (int32_t)std::min<int64_t>(seg, pr.len - off), pr.beg + off});
      P->multi.push_back(PanelRow{pr.row, nseg, first});
    }
    P->max_segments = std::max<int64_t>(P->max_segments, (int64_t)P->seg.size() - s0);
  }
  P->row_ptr[K] = (int64_t)P->host.size();
  P->seg_ptr[K] = (int64_t)P->seg.size();
  P->multi_ptr[K] = (int64_t)P->multi.size();
}

// Panel lists.  Over a CSR-like (ptr, idx) with N rows: for each block of the
// *index* range (block size b over Nidx), the rows with entries in the block.
void build_stoch_panels(const std::vector<int64_t>& ptr, const std::vector<int32_t>& idx,
                        int64_t N, int64_t Nidx, int64_t b, PanelSet* P) {
  int64_t K = nblocks(Nidx, b);
  std::vector<std::vector<PanelRow>> per(K);
  for (int64_t i = 0; i < N; ++i) {
    int64_t e = ptr[i], end = ptr[i + 1];
    while (e < end) {
      int64_t blk = idx[e] / b;
      int64_t s = e;
      while (e < end && idx[e] / b == blk) ++e;
      per[blk].push_back(PanelRow{(int32_t)i, (int32_t)(e - s), s});
    }
  }
  finalize_panels(per, P);
  // every block's step updates all N rows
  P->flag_off.assign(K + 1, 0);
  P->flags.assign((size_t)K * N, 0);
  for (int64_t k = 0; k < K; ++k) {
    P->flag_off[k] = k * N;
    for (const PanelRow& pr : per[k]) P->flags[(size_t)k * N + pr.row] = 1;
  }
  P->flag_off[K] = K * N;
}

// Exact panels: block k of rows [k b, (k+1) b) with their complete rows.
void build_exact_panels(const std::vector<int64_t>& ptr, int64_t N, int64_t b, PanelSet* P) {
  int64_t K = nblocks(N, b);
  std::vector<std::vector<PanelRow>> per(K);
  for (int64_t k = 0; k < K; ++k) {
    int64_t i0 = k * b, i1 = std::min(N, (k + 1) * b);
    for (int64_t i = i0; i < i1; ++i) {
      int64_t len = ptr[i + 1] - ptr[i];
      if (len > 0) per[k].push_back(PanelRow{(int32_t)i, (int32_t)len, ptr[i]});
    }
  }
  finalize_panels(per, P);
  // block k's step updates its rows [k b, min(N, (k+1) b))
  P->flag_off.assign(K + 1, 0);
  P->flags.assign((size_t)N, 0);
  for (int64_t k = 0; k < K; ++k) {
    P->flag_off[k] = k * b;
    for (const PanelRow& pr : per[k]) P->flags[pr.row] = 1;
  }
  P->flag_off[K] = N;
}

void build_panels(const HostSparse& S, const nmd_options& o, PanelSet P[2][2]) {
  build_exact_panels(S.rowptr, S.m, o.block_rows, &P[NMD_ROW][NMD_EXACT]);
  build_exact_panels(S.colptr, S.n, o.block_cols, &P[NMD_COL][NMD_EXACT]);
  // COL/STOCH block J: all rows of S (M = W), entries with column in J
  build_stoch_panels(S.rowptr, S.col, S.m, S.n, o.block_cols, &P[NMD_COL][NMD_STOCH]);
  // ROW/STOCH block I: all columns of S (M = B), entries with row in I
  build_stoch_panels(S.colptr, S.row, S.n, S.m, o.block_rows, &P[NMD_ROW][NMD_STOCH]);
}

// ---------------------------------------------------------------------------
// Workspace layout
// ---------------------------------------------------------------------------
struct Carver {
  char* base;
  size_t off = 0;
  explicit Carver(void* b) : base((char*)b) {}
  template <class T>
  T* take(size_t count) {
    off = (off + 255) & ~size_t(255);
    T* p = base ? (T*)(base + off) : nullptr;
    off += count * sizeof(T);
    return p;
  }
};

// Words of the range-search mask of any step: per 128-row M tile one bit
// per Q chunk (chunks of at least 64 rows), words rounded up per tile.  A
// stochastic step has tiles over a whole factor and chunks over a block, an
// exact step the other way round; both are bounded by tiles(N) x words(N).
int64_t range_mask_words(int64_t m, int64_t n) {
  const int64_t N = std::max(m, n);
  return ((N + 127) / 128) * ((((N + 63) / 64) + 31) / 32);
}

void layout(Carver& c, int64_t m, int64_t n, int64_t nnz, int rp, int64_t npanels, int64_t maxseg,
            int64_t nflags, Workspace* w, Factor* W, Factor* B) {
  w->rowptr = c.take<int64_t>(m + 1);
  w->col = c.take<int32_t>(nnz);
  w->val = c.take<float>(nnz);
  w->colptr = c.take<int64_t>(n + 1);
  w->row = c.take<int32_t>(nnz);
  w->valT = c.take<float>(nnz);
  w->panels = c.take<PanelRow>(std::max<int64_t>(npanels, 1));
  for (Factor* f : {W, B}) {
    int64_t N = f == W ? m : n;
    f->rows = N;
    f->master = c.take<float>(N * rp);
    f->hi = c.take<bf16>(N * rp);
    f->lo = c.take<bf16>(N * rp);
    f->lo2 = c.take<bf16>(N * rp);
    f->E = c.take<float>(N * rp);
  }
  w->R = c.take<float>(std::max(m, n) * rp);
  w->R2 = c.take<float>(std::max(m, n) * rp);
  w->Rs = c.take<float>(std::max(m, n) * rp);
  w->Rs2 = c.take<float>(std::max(m, n) * rp);
  w->gram_part = c.take<float>((size_t)kGramParts * rp * rp);
  w->G = c.take<float>((size_t)rp * rp);
  w->Ginv = c.take<float>((size_t)rp * rp);
  w->G2 = c.take<float>((size_t)rp * rp);
  w->Ginv2 = c.take<float>((size_t)rp * rp);
  w->Gc = c.take<float>((size_t)rp * rp);
  w->Ginvc = c.take<float>((size_t)rp * rp);
  w->Gx = c.take<float>((size_t)rp * rp);
  w->Tm = c.take<float>((size_t)rp * rp);
  w->seg_partials = c.take<float>((size_t)std::max<int64_t>(maxseg, 1) * rp);
  w->flags = c.take<uint8_t>((size_t)std::max<int64_t>(nflags, 1));
  w->rpart = c.take<float>((size_t)kRpartRows * rp);
  const int64_t N = std::max(m, n);
  w->ball_m = c.take<float>((size_t)((N + 127) / 128) * rp);
  w->rad_m = c.take<float>((size_t)((N + 127) / 128));
  w->ball_q = c.take<float>((size_t)((N + 63) / 64) * rp);
  w->rad_q = c.take<float>((size_t)((N + 63) / 64));
  w->rmask = c.take<uint32_t>((size_t)range_mask_words(m, n));
  for (bf16*& g : w->gsplit) g = c.take<bf16>((size_t)2 * rp * split_stride(rp));
  for (Factor& g : w->gi) {
    g.rows = rp;
    g.master = c.take<float>((size_t)rp * rp);
    g.hi = c.take<bf16>((size_t)rp * rp);
    g.lo = c.take<bf16>((size_t)rp * rp);
    g.lo2 = c.take<bf16>((size_t)rp * rp);
  }
  w->loss_part = c.take<double>((size_t)kLossParts * 8);
  w->loss_out = c.take<double>(8);
  w->status = c.take<int>(kStatusWords);
  w->counters = c.take<int>(64);
  c.off = (c.off + 255) & ~size_t(255);
  w->bytes = c.off;
}

int64_t panel_total(PanelSet P[2][2]) {
  int64_t t = 0;
  for (int s = 0; s < 2; ++s)
    for (int k = 0; k < 2; ++k) t += (int64_t)(P[s][k].host.size() + P[s][k].seg.size() + P[s][k].multi.size());
  return t;
}

int64_t flag_total(PanelSet P[2][2]) {
  int64_t t = 0;
  for (int s = 0; s < 2; ++s)
    for (int k = 0; k < 2; ++k) t += (int64_t)P[s][k].flags.size();
  return t;
}

int64_t max_segments(PanelSet P[2][2]) {
  int64_t t = 0;
  for (int s = 0; s < 2; ++s)
    for (int k = 0; k < 2; ++k) t = std::max(t, P[s][k].max_segments);
  return t;
}

// Every call that takes a handle runs with the handle's device current and
// puts the caller's device back afterwards, so that kernels, per-device
// kernel attributes and the handle's streams all belong to the same device.
struct DeviceScope {
  int prev = -1;
  explicit DeviceScope(const nmd_handle* h) {
    int cur = -1;
    if (h && cudaGetDevice(&cur) == cudaSuccess && cur != h->device && cudaSetDevice(h->device) == cudaSuccess)
      prev = cur;
  }
  ~DeviceScope() {
    if (prev >= 0) cudaSetDevice(prev);
  }
};

// ---------------------------------------------------------------------------
// Error plumbing
// ---------------------------------------------------------------------------
nmd_status fail(nmd_handle* h, nmd_status s, const std::string& why) {
  if (h) h->last_error = why;
  return s;
}

nmd_status cuda_check(nmd_handle* h, cudaError_t e, const char* what) {
  if (e == cudaSuccess) return NMD_OK;
  std::string w = std::string(what) + ": " + cudaGetErrorString(e);
  return fail(h, NMD_ERR_CUDA, w);
}

#define CK(h, call)                                          \
  do {                                                       \
    nmd_status _s = cuda_check((h), (call), #call);          \
    if (_s != NMD_OK) return _s;                             \
  } while (0)

nmd_status after_launch(nmd_handle* h, const char* what) {
  return cuda_check(h, cudaGetLastError(), what);
}

const char* status_name(int s) {
  switch (s) {
    case NMD_OK: return "ok";
    case NMD_ERR_INVALID: return "invalid argument";
    case NMD_ERR_CSR: return "malformed CSR";
    case NMD_ERR_NOT_SPD: return "block Gram matrix is not positive definite";
    case NMD_ERR_DIVERGED: return "non-finite factor entry (diverged)";
    case NMD_ERR_TIMEOUT: return "device-side wait timed out";
    case NMD_ERR_CUDA: return "CUDA error";
    case NMD_ERR_WORKSPACE: return "workspace too small or misaligned";
    case NMD_ERR_UNSUPPORTED: return "unsupported configuration";
  }
  return "unknown status";
}

// Synchronise, then read and clear the sticky device status.
nmd_status sync_and_check(nmd_handle* h) {
  CK(h, cudaStreamSynchronize(h->stream));
  if (h->side) CK(h, cudaStreamSynchronize(h->side));
  if (h->side2) CK(h, cudaStreamSynchronize(h->side2));
  if (h->aux) CK(h, cudaStreamSynchronize(h->aux));
  if (h->hp) CK(h, cudaStreamSynchronize(h->hp));
  h->pend[0].active = h->pend[1].active = false;
  int st[kStatusWords];
  CK(h, cudaMemcpy(st, h->ws.status, sizeof st, cudaMemcpyDeviceToHost));
  if (st[0] != 0) {
    h->gcache_f = -1;   // a failed step may have left the cached Gram unusable
    CK(h, cudaMemset(h->ws.status, 0, sizeof st));
    char b[192];
    snprintf(b, sizeof b, "%s (device detail %d, at block step %d)", status_name(st[0]), st[1], st[2]);
    return fail(h, (nmd_status)st[0], b);
  }
  return NMD_OK;
}

// ---------------------------------------------------------------------------
// Kernel timing: an event pair around a launch when profiling is on
// ---------------------------------------------------------------------------
cudaEvent_t pool_event(nmd_handle* h) {
  if (!h->event_pool.empty()) {
    cudaEvent_t e = h->event_pool.back();
    h->event_pool.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  cudaEventCreate(&e);
  return e;
}

struct TimedScope {
  nmd_handle* h;
  int cls;
  cudaStream_t st;
  cudaEvent_t a = nullptr, b = nullptr;
  TimedScope(nmd_handle* h_, int c, cudaStream_t s_ = nullptr) : h(h_), cls(c), st(s_ ? s_ : h_->cur) {
    if (h->profiling) {
      a = pool_event(h);
      b = pool_event(h);
      cudaEventRecord(a, st);
    }
  }
  ~TimedScope() {
    if (a) {
      cudaEventRecord(b, st);
      h->timed.push_back({cls, a, b});
    }
  }
};

// With NMD_TRACE set to a file name, every timed launch is also appended to
// that file as "class start_ms end_ms", relative to the first launch of the
// batch (a timeline across the streams).
void collect_timing(nmd_handle* h) {
  static const char* names[5] = {"dense", "sparse", "gram", "update", "loss"};
  const char* path = getenv("NMD_TRACE");
  FILE* tf = (path && !h->timed.empty()) ? fopen(path, "a") : nullptr;
  for (auto& t : h->timed) {
    float ms = 0.f;
    if (cudaEventElapsedTime(&ms, t.a, t.b) == cudaSuccess) {
      h->prof_ms[t.cls] += ms;
      h->prof_launches[t.cls] += 1;
    }
    float t0 = 0.f, t1 = 0.f;
    if (tf && cudaEventElapsedTime(&t0, h->timed[0].a, t.a) == cudaSuccess &&
        cudaEventElapsedTime(&t1, h->timed[0].a, t.b) == cudaSuccess)
      fprintf(tf, "%s %.4f %.4f\n", names[t.cls], t0, t1);
    h->event_pool.push_back(t.a);
    h->event_pool.push_back(t.b);
  }
  if (tf) fclose(tf);
  h->timed.clear();
}

// ---------------------------------------------------------------------------
// One block step
// ---------------------------------------------------------------------------
struct Roles {
  Factor* fm;
  Factor* fq;
  int64_t m0, M, q0, K;
  const PanelSet* P;
  const int32_t* qidx;   // absolute Q-side index of each sparse entry
  const float* vals;
  int64_t pblock = 0;    // the block of P whose panel the step uses
  bool sub = false;      // the step takes only the panel's M-side rows [m0, m0 + M)
};

// The sparse work of one step: the sub-lists of a block's panel lists whose
// M-side rows lie in the step's range (all of them, unless Roles::sub).
struct Span {
  const PanelRow *rows, *whole, *seg, *multi;   // device pointers
  int64_t nrows, nwhole, nseg, nmulti;
  int64_t seg_first;                            // first slice, relative to the block's slices
  const uint8_t* flags;                         // one byte per M-side row of the step
  // host-side index ranges (for nmd_panel_traversal)
  int64_t hr0, hr1, hw0, hw1, hu0, hu1;
};

Span panel_span(const Roles& ro) {
  const PanelSet& P = *ro.P;
  const int64_t b = ro.pblock;
  const int64_t r0 = P.row_ptr[b], r1 = P.row_ptr[b + 1];
  const int64_t g0 = P.seg_ptr[b], gd = g0 + P.segd[b], g1 = P.seg_ptr[b + 1];
  const int64_t u0 = P.multi_ptr[b], u1 = P.multi_ptr[b + 1];
  Span sp;
  sp.hr0 = r0; sp.hr1 = r1; sp.hw0 = g0; sp.hw1 = gd; sp.hu0 = u0; sp.hu1 = u1;
  sp.seg_first = 0;
  int64_t s0 = 0, s1 = g1 - gd;
  if (ro.sub) {   // lists are ascending by row: cut them to [m0, m0 + M)
    auto lo = [](const std::vector<PanelRow>& v, int64_t a, int64_t z, int64_t row) {
      return (int64_t)(std::lower_bound(v.begin() + a, v.begin() + z, row,
                                        [](const PanelRow& p, int64_t x) { return p.row < x; }) - v.begin());
    };
    const int64_t m1 = ro.m0 + ro.M;
    sp.hr0 = lo(P.host, r0, r1, ro.m0); sp.hr1 = lo(P.host, r0, r1, m1);
    sp.hw0 = lo(P.seg, g0, gd, ro.m0); sp.hw1 = lo(P.seg, g0, gd, m1);
    sp.hu0 = lo(P.multi, u0, u1, ro.m0); sp.hu1 = lo(P.multi, u0, u1, m1);
    if (sp.hu1 > sp.hu0) {
      s0 = P.multi[sp.hu0].beg;
      s1 = P.multi[sp.hu1 - 1].beg + P.multi[sp.hu1 - 1].len;
    } else {
      s0 = s1 = 0;
    }
  }
  sp.rows = P.d + sp.hr0;
  sp.nrows = sp.hr1 - sp.hr0;
  sp.whole = P.d_seg + sp.hw0;
  sp.nwhole = sp.hw1 - sp.hw0;
  sp.seg = P.d_seg + gd + s0;
  sp.nseg = s1 - s0;
  sp.seg_first = s0;
  sp.multi = P.d_multi + sp.hu0;
  sp.nmulti = sp.hu1 - sp.hu0;
  // stochastic panels flag every row of the M side, exact ones the block's rows
  sp.flags = P.d_flags + P.flag_off[b] + (ro.sub ? ro.m0 : 0);
  return sp;
}

nmd_status launch_span(nmd_handle* h, const StepArgs& a, const Roles& ro, const Span& sp, float* Rs, cudaStream_t s) {
  h->launches += launch_sparse(a, sp.rows, sp.nrows, sp.whole, sp.nwhole, sp.seg, sp.nseg, sp.multi, sp.nmulti,
                               ro.qidx, ro.vals, Rs, h->ws.seg_partials, sp.seg_first, s);
  return NMD_OK;
}

nmd_status roles(nmd_handle* h, int side, int64_t block, int kind, Roles* R) {
  if (side != NMD_ROW && side != NMD_COL) return fail(h, NMD_ERR_INVALID, "side must be NMD_ROW or NMD_COL");
  if (kind != NMD_EXACT && kind != NMD_STOCH) return fail(h, NMD_ERR_INVALID, "kind must be NMD_EXACT or NMD_STOCH");
  int64_t b = side == NMD_ROW ? h->opt.block_rows : h->opt.block_cols;
  int64_t N = side == NMD_ROW ? h->m : h->n;
  int64_t K = nblocks(N, b);
  if (block < 0 || block >= K) {
    char s[128]; snprintf(s, sizeof s, "block %lld out of range [0, %lld)", (long long)block, (long long)K);
    return fail(h, NMD_ERR_INVALID, s);
  }
  int64_t i0 = block * b, i1 = std::min(N, (block + 1) * b);
  const PanelSet* P = &h->panels[side][kind];
  if (side == NMD_ROW && kind == NMD_EXACT) {        // W_I from all of B on S[I, :]
    *R = Roles{&h->W, &h->B, i0, i1 - i0, 0, h->n, P, h->ws.col, h->ws.val, block};
  } else if (side == NMD_COL && kind == NMD_EXACT) { // B_J from all of W on S[:, J]^T
    *R = Roles{&h->B, &h->W, i0, i1 - i0, 0, h->m, P, h->ws.row, h->ws.valT, block};
  } else if (side == NMD_COL) {                      // all of W from B_J on S[:, J]
    *R = Roles{&h->W, &h->B, 0, h->m, i0, i1 - i0, P, h->ws.col, h->ws.val, block};
  } else {                                           // all of B from W_I on S[I, :]^T
    *R = Roles{&h->B, &h->W, 0, h->n, i0, i1 - i0, P, h->ws.row, h->ws.valT, block};
  }
  return NMD_OK;
}

// Combined row and column sub-sampling (Sec. 4.1, the remark after eq.
// lsqA_sto): NMD_ROW updates W_I from B_J on S[I, J] (the column panel of J
// cut to the rows I), NMD_COL updates B_J from W_I on S[I, J]^T (the row panel
// of I cut to the columns J).
nmd_status roles_combined(nmd_handle* h, int side, int64_t row_block, int64_t col_block, Roles* R) {
  if (side != NMD_ROW && side != NMD_COL) return fail(h, NMD_ERR_INVALID, "side must be NMD_ROW or NMD_COL");
  const int64_t Kr = nblocks(h->m, h->opt.block_rows), Kc = nblocks(h->n, h->opt.block_cols);
  if (row_block < 0 || row_block >= Kr || col_block < 0 || col_block >= Kc) {
    char b[160];
    snprintf(b, sizeof b, "blocks (%lld, %lld) out of range [0, %lld) x [0, %lld)", (long long)row_block,
             (long long)col_block, (long long)Kr, (long long)Kc);
    return fail(h, NMD_ERR_INVALID, b);
  }
  const int64_t i0 = row_block * h->opt.block_rows, i1 = std::min(h->m, (row_block + 1) * h->opt.block_rows);
  const int64_t j0 = col_block * h->opt.block_cols, j1 = std::min(h->n, (col_block + 1) * h->opt.block_cols);
  if (side == NMD_ROW)
    *R = Roles{&h->W, &h->B, i0, i1 - i0, j0, j1 - j0, &h->panels[NMD_COL][NMD_STOCH], h->ws.col, h->ws.val,
               col_block, true};
  else
    *R = Roles{&h->B, &h->W, j0, j1 - j0, i0, i1 - i0, &h->panels[NMD_ROW][NMD_STOCH], h->ws.row, h->ws.valT,
               row_block, true};
  return NMD_OK;
}

int factor_id(const nmd_handle* h, const Factor* f) { return f == &h->W ? 0 : 1; }

bool overlaps(int64_t x0, int64_t x1, int64_t y0, int64_t y1) { return x0 < y1 && y0 < x1 && x0 < x1 && y0 < y1; }

// Order the main stream after the deferred update of factor f.
nmd_status wait_pending(nmd_handle* h, int f) {
  if (h->pend[f].active) {
    h->pend[f].active = false;
    CK(h, cudaStreamWaitEvent(h->cur, h->pend[f].ev, 0));
  }
  return NMD_OK;
}

nmd_status wait_all_pending(nmd_handle* h) {
  nmd_status st = wait_pending(h, 0);
  if (st == NMD_OK) st = wait_pending(h, 1);
  return st;
}

// The step that follows the current one within a sweep (lets the update
// defer the rows that step does not read).
struct NextUse {
  int side;
  int64_t block;
  int kind;
};

// bf16 mode at r_pad = 256: X = R G^{-1} costs 2 r^2 flops per row, more
// than the CUDA cores deliver at the update's memory rate, so it runs on the
// tensor cores (the update pass of the dense kernel; R and G^{-1} as two bf16
// pieces each, three products, fp32 accumulation)
bool tc_update(const nmd_handle* h) {
  return h->rp == 256 && h->opt.precision == NMD_BF16 && tc_supported(h->rp, h->opt.precision);
}

// the pieces of the G^{-1} buffer in use (by step parity, or the exact steps' cache)
const Factor* gi_of(const nmd_handle* h, const float* Ginv) {
  return Ginv == h->ws.Ginv ? &h->ws.gi[0] : Ginv == h->ws.Ginv2 ? &h->ws.gi[1] : &h->ws.gi[2];
}

// the transposed pieces of the same buffer (bf16 mode, r_pad <= 128)
bf16* gsplit_of(const nmd_handle* h, const float* Ginv) {
  if (h->opt.precision != NMD_BF16 || h->rp > 128) return nullptr;
  return Ginv == h->ws.Ginv ? h->ws.gsplit[0] : Ginv == h->ws.Ginv2 ? h->ws.gsplit[1] : h->ws.gsplit[2];
}

nmd_status launch_update_rows(nmd_handle* h, const StepArgs& a, const Roles& ro, float* R, float* Rs,
                              const uint8_t* flags, const float* Ginv, int64_t lo, int64_t hi, bool momentum,
                              cudaStream_t s) {
  if (hi <= lo) return NMD_OK;
  StepArgs sub = a;
  sub.m0 = ro.m0 + lo;
  sub.M = hi - lo;
  TimedScope ts(h, NMD_K_UPDATE, s);
  if (tc_update(h)) {
    const nmd_status st = launch_update_tc(sub, R + lo * h->rp, Rs + lo * h->rp, flags + lo, *gi_of(h, Ginv),
                                           (float)h->opt.eta, momentum ? (float)h->opt.gamma : 0.f, momentum,
                                           h->ws.status, h->num_sms, s);
    if (st != NMD_OK) return fail(h, st, "tensor-core update");
  } else {
    launch_update(sub, R + lo * h->rp, Rs + lo * h->rp, flags + lo, Ginv, gsplit_of(h, Ginv), (float)h->opt.eta,
                  momentum ? (float)h->opt.gamma : 0.f, momentum, h->ws.status, s);
  }
  h->launches++;
  return NMD_OK;
}

// step kinds beyond nmd_kind: a stochastic step on a (row block, column
// block) pair (combined sub-sampling)
constexpr int kCombined = 2;

// The range-search mask of a step (Sec. 4.3, eq. range-search): balls around
// the normalised rows of its 128-row M tiles and of its Q chunks, then one
// bit per (tile, chunk) pair whose balls are far enough apart that L <= 0
// on all of it.  Sets a->rmask and a->rwords.
void range_pass(nmd_handle* h, const Roles& ro, StepArgs* a, cudaStream_t s) {
  const int bn = panel_chunk_rows(h->rp, h->opt.precision);
  const int64_t ntiles = (ro.M + 127) / 128, nchunks = (ro.K + bn - 1) / bn, words = (nchunks + 31) / 32;
  launch_range_balls(ro.fm->master, ro.m0, ro.M, ro.fq->master, ro.q0, ro.K, bn, h->rp, h->ws.ball_m,
                     h->ws.rad_m, h->ws.ball_q, h->ws.rad_q, s);
  launch_range_mask(h->ws.ball_m, h->ws.rad_m, ntiles, h->ws.ball_q, h->ws.rad_q, nchunks, words, h->rp,
                    h->ws.rmask, s);
  h->launches += 2;
  a->rmask = h->ws.rmask;
  a->rwords = words;
}

bool range_on(const nmd_handle* h) {
  return h->opt.skip_zero_chunks == NMD_SKIP_RANGE && h->opt.epilogue == NMD_EPI_DELTA &&
         h->opt.precision != NMD_SIMT;
}

nmd_status run_step_roles(nmd_handle* h, const Roles& ro, int kind, bool do_update, const NextUse* next);

nmd_status run_step(nmd_handle* h, int side, int64_t block, int kind, bool do_update,
                    const NextUse* next = nullptr) {
  Roles ro;
  nmd_status st = roles(h, side, block, kind, &ro);
  if (st != NMD_OK) return st;
  return run_step_roles(h, ro, kind, do_update, next);
}

nmd_status run_step_roles(nmd_handle* h, const Roles& ro, int kind, bool do_update, const NextUse* next) {
  nmd_status st = NMD_OK;
  StepArgs a{ro.fm, ro.fq, ro.m0, ro.M, ro.q0, ro.K, h->r, h->rp, h->opt.precision, h->opt.epilogue, h->num_sms,
              h->opt.skip_zero_chunks == NMD_SKIP_VOTE};
  cudaStream_t s = h->cur;
  // wait for deferred updates of rows this step reads or writes, and for
  // those of two steps back (they read the copies of R and G^{-1} reused now)
  const int fm = factor_id(h, ro.fm), fq = factor_id(h, ro.fq);
  if ((st = wait_pending(h, fm)) != NMD_OK) return st;
  const nmd_handle::Pending& pq = h->pend[fq];
  if (pq.active && (overlaps(ro.q0, ro.q0 + ro.K, pq.a0, pq.a1) || overlaps(ro.q0, ro.q0 + ro.K, pq.b0, pq.b1)))
    if ((st = wait_pending(h, fq)) != NMD_OK) return st;
  if (h->pend[fq].active && h->pend[fq].step <= h->step_index - 2)
    if ((st = wait_pending(h, fq)) != NMD_OK) return st;
  const int par = (int)(h->step_index & 1);
  float* R = par ? h->ws.R2 : h->ws.R;
  float* Rs = par ? h->ws.Rs2 : h->ws.Rs;
  float* G = par ? h->ws.G2 : h->ws.G;
  float* Ginv = par ? h->ws.Ginv2 : h->ws.Ginv;
  // bf16 mode: the step's least-squares problem is solved for the bf16 pieces
  // of the factors throughout -- the dense term (tensor cores), the support
  // term and the Gram matrix G = Qt^T Qt all read the rounded rows Qt (and
  // Mt), so that the rounding of Q is not a coherent error between R and G
  // that the solve would amplify by the condition number of G; the update
  // is applied to the fp32 masters.  The other modes use the masters.
  const bool rounded = h->opt.precision == NMD_BF16;
  // an exact step's Q side is a whole factor: every block of a half-sweep has
  // the same G, computed once and kept until that factor changes
  bool need_gram = true;
  if (kind == NMD_EXACT) {
    G = h->ws.Gc;
    Ginv = h->ws.Ginvc;
    need_gram = !(h->gcache_f == fq && h->gcache_ver == h->fver[fq]);
    h->gcache_f = fq;
    h->gcache_ver = h->fver[fq];
  }
  h->cur_R = R;
  h->cur_Rs = Rs;
  h->cur_G = G;
  h->cur_Ginv = Ginv;
  // The side stream computes G = Q^T Q of the Q-side rows and G^{-1}, the
  // second side stream the support term Rs of R, the main stream the dense
  // term of R.  None reads what another writes, so they overlap; the update
  // joins them.
  // Gram partials over parts of 64 Q-side rows where there are at most
  // kGramParts of them, else over kGramParts equal parts
  const bool rows64 = (ro.K + 63) / 64 <= kGramParts;
  const int nparts = rows64 ? (int)((ro.K + 63) / 64) : kGramParts;
  const int64_t chunk = rows64 ? 64 : ((ro.K + nparts - 1) / nparts + 31) / 32 * 32;
  CK(h, cudaEventRecord(h->ev_fork, s));
  CK(h, cudaStreamWaitEvent(h->side, h->ev_fork, 0));
  CK(h, cudaStreamWaitEvent(h->side2, h->ev_fork, 0));
  if (need_gram) {
    TimedScope ts(h, NMD_K_GRAM, h->side);
    launch_gram(ro.fq, rounded, ro.q0, ro.K, h->r, h->rp, h->ws.gram_part, nparts, chunk, (float)h->opt.ridge, G,
                h->side);
    launch_chol_inv(G, h->r, h->rp, Ginv, gsplit_of(h, Ginv), h->ws.status, h->side);
    h->launches += 3;
    if (tc_update(h)) {   // the pieces of G^{-1} for the tensor-core update
      Factor gi = *gi_of(h, Ginv);
      launch_pack(Ginv, false, h->rp, h->rp, h->rp, gi, h->side);
      h->launches++;
    }
  }
  if ((st = after_launch(h, "gram/cholesky")) != NMD_OK) return st;
  // sparse correction over the block's support
  const Span sp = panel_span(ro);
  const uint8_t* flags = sp.flags;
  h->cur_flags = flags;
  {
    TimedScope ts(h, NMD_K_SPARSE, h->side2);
    launch_span(h, a, ro, sp, Rs, h->side2);
  }
  if ((st = after_launch(h, "sparse correction")) != NMD_OK) return st;
  CK(h, cudaEventRecord(h->ev_join, h->side));
  CK(h, cudaEventRecord(h->ev_join2, h->side2));
  // dense Z-panel contraction R = P(L) Q over every (M-side, Q-side) pair
  if (range_on(h)) range_pass(h, ro, &a, s);
  {
    TimedScope ts(h, NMD_K_DENSE);
    if (h->opt.precision == NMD_SIMT) {
      launch_panel_simt(a, R, s);
      h->launches++;
    } else {
      st = launch_panel_tc(a, R, h->ws.status, h->ws.counters, h->num_sms, s, &h->launches, nullptr, h->ws.rpart,
                           kRpartRows);
    }
  }
  if (st != NMD_OK) return fail(h, st, "no tensor-core kernel for this rank/precision on this device");
  if ((st = after_launch(h, "dense panel")) != NMD_OK) return st;
  CK(h, cudaStreamWaitEvent(s, h->ev_join, 0));
  CK(h, cudaStreamWaitEvent(s, h->ev_join2, 0));
  if (do_update) {
    const bool momentum = kind != NMD_EXACT;
    // rows [lo, hi) (relative to m0) are updated on the main stream; when the
    // next step reads only these rows of this factor and writes the other
    // factor, the rest are updated on the aux stream, overlapping it
    int64_t lo = 0, hi = ro.M;
    if (next) {
      Roles rn;
      if (roles(h, next->side, next->block, next->kind, &rn) == NMD_OK && rn.fq == ro.fm && rn.fm != ro.fm) {
        lo = std::min(std::max(rn.q0 - ro.m0, (int64_t)0), ro.M);
        hi = std::max(std::min(rn.q0 + rn.K - ro.m0, ro.M), lo);
      }
    }
    if ((st = launch_update_rows(h, a, ro, R, Rs, flags, Ginv, lo, hi, momentum, s)) != NMD_OK) return st;
    if (lo > 0 || hi < ro.M) {
      CK(h, cudaEventRecord(h->ev_prio, s));
      CK(h, cudaStreamWaitEvent(h->aux, h->ev_prio, 0));
      if ((st = launch_update_rows(h, a, ro, R, Rs, flags, Ginv, 0, lo, momentum, h->aux)) != NMD_OK) return st;
      if ((st = launch_update_rows(h, a, ro, R, Rs, flags, Ginv, hi, ro.M, momentum, h->aux)) != NMD_OK) return st;
      nmd_handle::Pending& pm = h->pend[fm];
      CK(h, cudaEventRecord(pm.ev, h->aux));
      pm.active = true;
      pm.step = h->step_index;
      pm.a0 = ro.m0;
      pm.a1 = ro.m0 + lo;
      pm.b0 = ro.m0 + hi;
      pm.b1 = ro.m0 + ro.M;
    }
    if ((st = after_launch(h, "update")) != NMD_OK) return st;
  }
  if (do_update) h->fver[fm]++;
  h->step_index++;
  return NMD_OK;
}

}  // namespace

nmd_handle::~nmd_handle() {
  if (side) cudaStreamSynchronize(side);
  if (side2) cudaStreamSynchronize(side2);
  if (aux) cudaStreamSynchronize(aux);
  if (!timed.empty()) cudaStreamSynchronize(stream);
  for (auto& t : timed) {
    cudaEventDestroy(t.a);
    cudaEventDestroy(t.b);
  }
  for (cudaEvent_t e : event_pool) cudaEventDestroy(e);
  if (ev_fork) cudaEventDestroy(ev_fork);
  if (ev_join) cudaEventDestroy(ev_join);
  if (ev_join2) cudaEventDestroy(ev_join2);
  if (side) cudaStreamDestroy(side);
  if (side2) cudaStreamDestroy(side2);
  if (ev_prio) cudaEventDestroy(ev_prio);
  for (auto& p : pend)
    if (p.ev) cudaEventDestroy(p.ev);
  if (aux) cudaStreamDestroy(aux);
  if (hp) {
    cudaStreamSynchronize(hp);
    cudaStreamDestroy(hp);
  }
  if (ev_in) cudaEventDestroy(ev_in);
  if (ev_out) cudaEventDestroy(ev_out);
}

// ===========================================================================
// C ABI
// ===========================================================================
extern "C" {

const char* nmd_version(void) { return NMD_VERSION_STRING; }

void nmd_default_options(nmd_options* o) {
  if (!o) return;
  memset(o, 0, sizeof *o);
  o->block_rows = 4096;
  o->block_cols = 4096;
  o->schedule = NMD_STOCH;
  o->order = NMD_ALTERNATE;
  o->eta = 1.0;
  o->gamma = 0.9;
  o->ridge = 0.0;
  o->precision = NMD_BF16;
  o->epilogue = NMD_EPI_Z;
  o->seed = 0;
}

const char* nmd_status_string(nmd_status s) { return status_name((int)s); }

const char* nmd_last_error(const nmd_handle* h) { return h ? h->last_error.c_str() : ""; }

int64_t nmd_launch_count(const nmd_handle* h) { return h ? h->launches : 0; }

nmd_status nmd_selftest_wait_timeout(nmd_handle* h, int64_t limit_ns) {
  if (!h || limit_ns < 1000 || limit_ns > 1000000000) return NMD_ERR_INVALID;
  DeviceScope dg(h);
  nmd_status st = sync_and_check(h);
  if (st != NMD_OK) return st;
  launch_wait_selftest(h->ws.status, (uint64_t)limit_ns, h->stream);
  h->launches++;
  if ((st = after_launch(h, "wait self-test")) != NMD_OK) return st;
  return sync_and_check(h);
}

nmd_status nmd_skip_count(nmd_handle* h, int64_t* skipped, int32_t reset) {
  if (!h || !skipped) return NMD_ERR_INVALID;
  DeviceScope dg(h);
  nmd_status st = sync_and_check(h);
  if (st != NMD_OK) return st;
  unsigned long long v = 0;
  CK(h, cudaMemcpy(&v, h->ws.counters, sizeof v, cudaMemcpyDeviceToHost));
  *skipped = (int64_t)v;
  if (reset) CK(h, cudaMemset(h->ws.counters, 0, sizeof v));
  return NMD_OK;
}

nmd_status nmd_workspace_bytes(int64_t m, int64_t n, int32_t r, const int64_t* row_ptr,
                               const int32_t* col_idx, const float* vals, const nmd_options* opts,
                               size_t* bytes) {
  std::string why;
  nmd_status st = check_options(opts, &why);
  if (st != NMD_OK) return st;
  if (!bytes) return NMD_ERR_INVALID;
  HostSparse S;
  if ((st = build_sparse(m, n, r, row_ptr, col_idx, vals, &S, &why)) != NMD_OK) return st;
  PanelSet P[2][2];
  build_panels(S, *opts, P);
  Carver c(nullptr);
  Workspace w;
  Factor W, B;
  layout(c, m, n, (int64_t)S.col.size(), pad_rank(r), panel_total(P), max_segments(P), flag_total(P), &w, &W, &B);
  *bytes = w.bytes;
  return NMD_OK;
}

nmd_status nmd_create(int64_t m, int64_t n, int32_t r, const int64_t* row_ptr,
                      const int32_t* col_idx, const float* vals, const nmd_options* opts,
                      void* d_workspace, size_t ws_bytes, void* stream, nmd_handle** out) {
  if (!out) return NMD_ERR_INVALID;
  *out = nullptr;
  nmd_handle* h = new nmd_handle();
  std::string why;
  nmd_status st = check_options(opts, &why);
  HostSparse S;
  if (st == NMD_OK) st = build_sparse(m, n, r, row_ptr, col_idx, vals, &S, &why);
  if (st != NMD_OK) {
    fprintf(stderr, "nmd_create: %s\n", why.c_str());
    delete h;
    return st;
  }
  h->m = m; h->n = n; h->r = r; h->rp = pad_rank(r);
  h->nnz = (int64_t)S.col.size();
  h->opt = *opts;
  h->stream = (cudaStream_t)stream;
  h->cur = h->stream;
  h->s_fro = S.s_fro;
  build_panels(S, h->opt, h->panels);
  Carver c(d_workspace);
  layout(c, m, n, h->nnz, h->rp, panel_total(h->panels), max_segments(h->panels), flag_total(h->panels), &h->ws,
         &h->W, &h->B);
  auto bail = [&](nmd_status s, const std::string& w) {
    fprintf(stderr, "nmd_create: %s\n", w.c_str());
    delete h;
    return s;
  };
  if (!d_workspace || ((uintptr_t)d_workspace & 255) != 0)
    return bail(NMD_ERR_WORKSPACE, "workspace pointer is NULL or not 256-byte aligned");
  if (ws_bytes < h->ws.bytes) {
    char b[160]; snprintf(b, sizeof b, "workspace has %zu bytes, needs %zu", ws_bytes, h->ws.bytes);
    return bail(NMD_ERR_WORKSPACE, b);
  }
  cudaError_t e = cudaGetDevice(&h->device);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&h->num_sms, cudaDevAttrMultiProcessorCount, h->device);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&h->cc_major, cudaDevAttrComputeCapabilityMajor, h->device);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&h->cc_minor, cudaDevAttrComputeCapabilityMinor, h->device);
  if (e != cudaSuccess) return bail(NMD_ERR_CUDA, std::string("device query: ") + cudaGetErrorString(e));
  if (h->cc_major != 10) {
    char b[128]; snprintf(b, sizeof b, "device has compute capability %d.%d; libnmd is built for sm_103a",
                          h->cc_major, h->cc_minor);
    return bail(NMD_ERR_UNSUPPORTED, b);
  }
  // panel lists, concatenated [ROW][EXACT], [ROW][STOCH], [COL][EXACT], [COL][STOCH]
  std::vector<PanelRow> all;
  for (int s2 = 0; s2 < 2; ++s2)
    for (int k = 0; k < 2; ++k) {
      PanelSet& P = h->panels[s2][k];
      P.d = h->ws.panels + all.size();
      all.insert(all.end(), P.host.begin(), P.host.end());
      P.d_seg = h->ws.panels + all.size();
      all.insert(all.end(), P.seg.begin(), P.seg.end());
      P.d_multi = h->ws.panels + all.size();
      all.insert(all.end(), P.multi.begin(), P.multi.end());
    }
  std::vector<uint8_t> allf;
  for (int s2 = 0; s2 < 2; ++s2)
    for (int k = 0; k < 2; ++k) {
      PanelSet& P = h->panels[s2][k];
      P.d_flags = h->ws.flags + allf.size();
      allf.insert(allf.end(), P.flags.begin(), P.flags.end());
    }
  cudaStream_t s = h->stream;
  struct Cp { void* d; const void* src; size_t n; } cps[] = {
      {h->ws.flags, allf.data(), allf.size()},
      {h->ws.rowptr, S.rowptr.data(), S.rowptr.size() * 8},
      {h->ws.col, S.col.data(), S.col.size() * 4},
      {h->ws.val, S.val.data(), S.val.size() * 4},
      {h->ws.colptr, S.colptr.data(), S.colptr.size() * 8},
      {h->ws.row, S.row.data(), S.row.size() * 4},
      {h->ws.valT, S.valT.data(), S.valT.size() * 4},
      {h->ws.panels, all.data(), all.size() * sizeof(PanelRow)},
  };
  for (auto& cp : cps)
    if (cp.n && (e = cudaMemcpyAsync(cp.d, cp.src, cp.n, cudaMemcpyHostToDevice, s)) != cudaSuccess)
      return bail(NMD_ERR_CUDA, std::string("copy-in: ") + cudaGetErrorString(e));
  // zero factors, momentum and the status words
  for (Factor* f : {&h->W, &h->B}) {
    e = cudaMemsetAsync(f->master, 0, f->rows * h->rp * 4, s);
    if (e == cudaSuccess) e = cudaMemsetAsync(f->hi, 0, f->rows * h->rp * 2, s);
    if (e == cudaSuccess) e = cudaMemsetAsync(f->lo, 0, f->rows * h->rp * 2, s);
    if (e == cudaSuccess) e = cudaMemsetAsync(f->lo2, 0, f->rows * h->rp * 2, s);
    if (e == cudaSuccess) e = cudaMemsetAsync(f->E, 0, f->rows * h->rp * 4, s);
    if (e != cudaSuccess) return bail(NMD_ERR_CUDA, std::string("memset: ") + cudaGetErrorString(e));
  }
  int least = 0, greatest = 0;
  e = cudaDeviceGetStreamPriorityRange(&least, &greatest);
  const int side_prio = greatest < least ? greatest + 1 : greatest;
  if (e == cudaSuccess) e = cudaStreamCreateWithPriority(&h->side, cudaStreamNonBlocking, side_prio);
  if (e == cudaSuccess) e = cudaStreamCreateWithPriority(&h->side2, cudaStreamNonBlocking, side_prio);
  if (e == cudaSuccess) e = cudaStreamCreateWithPriority(&h->hp, cudaStreamNonBlocking, greatest);
  if (e == cudaSuccess) e = cudaStreamCreateWithPriority(&h->aux, cudaStreamNonBlocking, least);
  if (e == cudaSuccess) e = cudaEventCreateWithFlags(&h->ev_fork, cudaEventDisableTiming);
  if (e == cudaSuccess) e = cudaEventCreateWithFlags(&h->ev_join, cudaEventDisableTiming);
  if (e == cudaSuccess) e = cudaEventCreateWithFlags(&h->ev_join2, cudaEventDisableTiming);
  if (e == cudaSuccess) e = cudaEventCreateWithFlags(&h->ev_in, cudaEventDisableTiming);
  if (e == cudaSuccess) e = cudaEventCreateWithFlags(&h->ev_out, cudaEventDisableTiming);
  if (e == cudaSuccess) e = cudaEventCreateWithFlags(&h->ev_prio, cudaEventDisableTiming);
  for (int f = 0; f < 2 && e == cudaSuccess; ++f) e = cudaEventCreateWithFlags(&h->pend[f].ev, cudaEventDisableTiming);
  if (e != cudaSuccess) return bail(NMD_ERR_CUDA, std::string("side stream: ") + cudaGetErrorString(e));
  e = cudaMemsetAsync(h->ws.status, 0, kStatusWords * sizeof(int), s);
  if (e == cudaSuccess) e = cudaMemsetAsync(h->ws.Rs, 0, std::max(m, n) * h->rp * sizeof(float), s);
  if (e == cudaSuccess) e = cudaMemsetAsync(h->ws.Rs2, 0, std::max(m, n) * h->rp * sizeof(float), s);
  if (e == cudaSuccess) e = cudaMemsetAsync(h->ws.counters, 0, 64 * sizeof(int), s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return bail(NMD_ERR_CUDA, std::string("create: ") + cudaGetErrorString(e));
  // the host copies of the panel lists are kept for nmd_panel_traversal
  *out = h;
  return NMD_OK;
}

// A copy of `bytes` in four pieces on the handle's four streams, so that
// several copy engines move it at once (a host <-> device copy on one
// engine stays well below what the link carries); ordered after the earlier
// work of `s`, which continues after all four pieces.  Used outside sweeps
// only (it borrows the sweep's streams and events).
nmd_status copy_split(nmd_handle* h, void* dst, const void* src, size_t bytes, cudaMemcpyKind kind, cudaStream_t s) {
  constexpr int kPieces = 4;
  if (bytes < ((size_t)8 << 20)) {
    CK(h, cudaMemcpyAsync(dst, src, bytes, kind, s));
    return NMD_OK;
  }
  cudaStream_t t[kPieces] = {s, h->side, h->side2, h->aux};
  cudaEvent_t done[kPieces] = {nullptr, h->ev_join, h->ev_join2, h->ev_prio};
  const size_t piece = (bytes / kPieces + 255) & ~(size_t)255;
  CK(h, cudaEventRecord(h->ev_fork, s));
  for (int q = 0; q < kPieces; ++q) {
    const size_t off = (size_t)q * piece;
    if (off >= bytes) break;
    if (q > 0) CK(h, cudaStreamWaitEvent(t[q], h->ev_fork, 0));
    CK(h, cudaMemcpyAsync((char*)dst + off, (const char*)src + off, std::min(piece, bytes - off), kind, t[q]));
    if (q > 0) {
      CK(h, cudaEventRecord(done[q], t[q]));
      CK(h, cudaStreamWaitEvent(s, done[q], 0));
    }
  }
  return NMD_OK;
}

nmd_status nmd_set_factors(nmd_handle* h, const float* W, const float* H, int on_device) {
  if (!h || !W || !H) return fail(h, NMD_ERR_INVALID, "NULL argument to nmd_set_factors");
  DeviceScope dg(h);
  h->fver[0]++;
  h->fver[1]++;
  cudaStream_t s = h->stream;
  cudaMemcpyKind kind = on_device ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice;
  // stage through R (max(m, n) x rp floats >= m x r and r x n)
  nmd_status cs = copy_split(h, h->ws.R, W, (size_t)h->m * h->r * 4, kind, s);
  if (cs != NMD_OK) return cs;
  launch_pack(h->ws.R, false, h->m, h->r, h->rp, h->W, s);
  h->launches++;
  // H goes to the second copy of R, so that its copy overlaps W's packing
  if ((cs = copy_split(h, h->ws.R2, H, (size_t)h->n * h->r * 4, kind, s)) != NMD_OK) return cs;
  launch_pack(h->ws.R2, true, h->n, h->r, h->rp, h->B, s);
  h->launches++;
  CK(h, cudaMemsetAsync(h->W.E, 0, (size_t)h->m * h->rp * 4, s));
  CK(h, cudaMemsetAsync(h->B.E, 0, (size_t)h->n * h->rp * 4, s));
  nmd_status st = after_launch(h, "pack factors");
  if (st != NMD_OK) return st;
  if (!on_device) CK(h, cudaStreamSynchronize(s));   // host buffers may be released after return
  return NMD_OK;
}

nmd_status nmd_get_factors(nmd_handle* h, float* W, float* H, int on_device) {
  if (!h) return NMD_ERR_INVALID;
  DeviceScope dg(h);
  nmd_status st = sync_and_check(h);
  cudaStream_t s = h->stream;
  cudaMemcpyKind kind = on_device ? cudaMemcpyDeviceToDevice : cudaMemcpyDeviceToHost;
  if (W) {
    launch_unpack(h->W.master, false, h->m, h->r, h->rp, h->ws.R, s);
    h->launches++;
    nmd_status cs = copy_split(h, W, h->ws.R, (size_t)h->m * h->r * 4, kind, s);
    if (cs != NMD_OK) return cs;
  }
  if (H) {
    launch_unpack(h->B.master, true, h->n, h->r, h->rp, h->ws.R2, s);
    h->launches++;
    nmd_status cs = copy_split(h, H, h->ws.R2, (size_t)h->n * h->r * 4, kind, s);
    if (cs != NMD_OK) return cs;
  }
  CK(h, cudaStreamSynchronize(s));
  return st;
}

nmd_status nmd_block_update(nmd_handle* h, int32_t side, int64_t block, int32_t kind) {
  if (!h) return NMD_ERR_INVALID;
  DeviceScope dg(h);
  return run_step(h, side, block, kind, true);
}

nmd_status nmd_block_update_combined(nmd_handle* h, int32_t side, int64_t row_block, int64_t col_block) {
  if (!h) return NMD_ERR_INVALID;
  DeviceScope dg(h);
  Roles ro;
  nmd_status st = roles_combined(h, side, row_block, col_block, &ro);
  if (st != NMD_OK) return st;
  return run_step_roles(h, ro, kCombined, true, nullptr);
}

nmd_status nmd_block_order(const nmd_handle* h, int64_t sweep, int32_t side, int64_t* perm, int64_t K) {
  if (!h || !perm || (side != NMD_ROW && side != NMD_COL) || sweep < 0) return NMD_ERR_INVALID;
  int64_t Kexp = side == NMD_ROW ? nblocks(h->m, h->opt.block_rows) : nblocks(h->n, h->opt.block_cols);
  if (K != Kexp) return NMD_ERR_INVALID;
  std::vector<int64_t> p = permutation(h->opt.seed, sweep, side, K);
  std::copy(p.begin(), p.end(), perm);
  return NMD_OK;
}

nmd_status nmd_sweep(nmd_handle* h) {
  if (!h) return NMD_ERR_INVALID;
  DeviceScope dg(h);
  int64_t Kr = nblocks(h->m, h->opt.block_rows), Kc = nblocks(h->n, h->opt.block_cols);
  std::vector<int64_t> pr = permutation(h->opt.seed, h->sweep_index, NMD_ROW, Kr);
  std::vector<int64_t> pc = permutation(h->opt.seed, h->sweep_index, NMD_COL, Kc);
  // the sweep's steps in order, so that each update knows the step after it
  std::vector<NextUse> steps;
  if (h->opt.schedule == NMD_EXACT) {
    for (int64_t t = 0; t < Kr; ++t) steps.push_back({NMD_ROW, pr[t], NMD_EXACT});
    for (int64_t t = 0; t < Kc; ++t) steps.push_back({NMD_COL, pc[t], NMD_EXACT});
  } else if (h->opt.order == NMD_PHASED) {
    for (int64_t t = 0; t < Kc; ++t) steps.push_back({NMD_COL, pc[t], NMD_STOCH});
    for (int64_t t = 0; t < Kr; ++t) steps.push_back({NMD_ROW, pr[t], NMD_STOCH});
  } else {
    for (int64_t t = 0; t < std::max(Kr, Kc); ++t) {
      if (t < Kc) steps.push_back({NMD_COL, pc[t], NMD_STOCH});
      if (t < Kr) steps.push_back({NMD_ROW, pr[t], NMD_STOCH});
    }
  }
  CK(h, cudaEventRecord(h->ev_in, h->stream));
  CK(h, cudaStreamWaitEvent(h->hp, h->ev_in, 0));
  h->cur = h->hp;
  nmd_status st = NMD_OK;
  for (size_t t = 0; t < steps.size() && st == NMD_OK; ++t)
    st = run_step(h, steps[t].side, steps[t].block, steps[t].kind, true,
                  t + 1 < steps.size() ? &steps[t + 1] : nullptr);
  // `stream` continues after every kernel of the sweep, deferred ones included
  nmd_status st2 = wait_all_pending(h);
  h->cur = h->stream;
  if (st == NMD_OK) st = st2;
  CK(h, cudaEventRecord(h->ev_out, h->hp));
  CK(h, cudaStreamWaitEvent(h->stream, h->ev_out, 0));
  if (st == NMD_OK) h->sweep_index++;
  return st;
}

nmd_status nmd_sync(nmd_handle* h) {
  if (!h) return NMD_ERR_INVALID;
  DeviceScope dg(h);
  return sync_and_check(h);
}

nmd_status nmd_loss(nmd_handle* h, nmd_loss_out* out) {
  if (!h || !out) return fail(h, NMD_ERR_INVALID, "NULL argument to nmd_loss");
  DeviceScope dg(h);
  nmd_status st = sync_and_check(h);
  if (st != NMD_OK) return st;
  cudaStream_t s = h->stream;
  int ndense = 0;
  {
    TimedScope ts(h, NMD_K_LOSS);
    if (h->opt.precision == NMD_SIMT) {
      ndense = launch_loss_dense_simt(h, h->ws.loss_part, kLossParts / 2, s);
      h->launches++;
    } else {
      st = launch_loss_dense_tc(h, h->ws.loss_part, kLossParts / 2, &ndense, h->ws.status, s, &h->launches);
    }
  }
  if (st != NMD_OK) return fail(h, st, "no tensor-core loss kernel for this rank/precision");
  if ((st = after_launch(h, "dense loss")) != NMD_OK) return st;
  int nsparse = kLossParts / 2;
  double* sp = h->ws.loss_part + (size_t)(kLossParts / 2) * 8;
  launch_loss_sparse(h, sp, nsparse, s);
  launch_loss_final(h->ws.loss_part, ndense, sp, nsparse, h->ws.loss_out, s);
  h->launches += 2;
  if ((st = after_launch(h, "loss")) != NMD_OK) return st;
  double v[8];
  CK(h, cudaMemcpyAsync(v, h->ws.loss_out, sizeof v, cudaMemcpyDeviceToHost, s));
  if ((st = sync_and_check(h)) != NMD_OK) return st;
  // v: [relu2, relu, sum_a, sum_b, sum_min, sum_max]: the dense sums cover
  // the entries off the support (SIMT: every entry, with the support part
  // subtracted again by the support pass)
  double zl2 = v[0] + v[2], err2 = v[0] + v[3];
  out->s_fro = h->s_fro;
  out->obj = sqrt(zl2 > 0 ? zl2 : 0.0) / h->s_fro;
  out->rmse = sqrt(err2 > 0 ? err2 : 0.0) / h->s_fro;
  double den = v[1] + v[5];
  out->wjd = den > 0 ? 1.0 - v[4] / den : 0.0;
  out->sum_relu2 = v[0];
  out->sum_relu = v[1];
  return NMD_OK;
}

nmd_status nmd_block_terms(nmd_handle* h, int32_t side, int64_t block, int32_t kind, float* R,
                           float* G, int64_t* rows) {
  if (!h) return NMD_ERR_INVALID;
  DeviceScope dg(h);
  Roles ro;
  nmd_status st = roles(h, side, block, kind, &ro);
  if (st != NMD_OK) return st;
  if ((st = run_step(h, side, block, kind, false)) != NMD_OK) return st;
  h->step_index--;
  launch_combine(h->cur_R, h->cur_Rs, h->cur_flags, ro.M, h->rp, h->cur);
  h->launches++;
  if ((st = after_launch(h, "combine")) != NMD_OK) return st;
  if ((st = sync_and_check(h)) != NMD_OK) return st;
  if (rows) *rows = ro.M;
  cudaStream_t s = h->stream;
  const float* Rout = h->cur_R;
  const float* Gout = h->cur_G;
  if (h->opt.precision == NMD_BF16) {
    // the bf16 mode solves X = R' Gt^{-1} for the rounded rows (R' = Z Qt,
    // Gt = Qt^T Qt); report the exact G of the fp32 rows and the right-hand
    // side that gives the same X with it: R' Gt^{-1} G
    float* other = h->cur_R == h->ws.R ? h->ws.R2 : h->ws.R;
    const int rp = h->rp;
    const int64_t np = std::min<int64_t>(kGramParts, std::max<int64_t>(1, (ro.K + 63) / 64));
    const int64_t ch = ((ro.K + np - 1) / np + 31) / 32 * 32;
    launch_gram(ro.fq, false, ro.q0, ro.K, h->r, rp, h->ws.gram_part, (int)np, ch, (float)h->opt.ridge, h->ws.Gx, s);
    launch_small_gemm(h->cur_Ginv, rp, h->ws.Gx, rp, h->ws.Tm, rp, rp, rp, rp, s);
    launch_small_gemm(h->cur_R, rp, h->ws.Tm, rp, other, rp, ro.M, rp, rp, s);
    h->launches += 4;
    if ((st = after_launch(h, "equivalent right-hand side")) != NMD_OK) return st;
    Rout = other;
    Gout = h->ws.Gx;
  }
  if (R) CK(h, cudaMemcpy2DAsync(R, h->r * 4, Rout, h->rp * 4, h->r * 4, ro.M, cudaMemcpyDeviceToHost, s));
  if (G) CK(h, cudaMemcpy2DAsync(G, h->r * 4, Gout, h->rp * 4, h->r * 4, h->r, cudaMemcpyDeviceToHost, s));
  CK(h, cudaStreamSynchronize(s));
  return NMD_OK;
}

nmd_status nmd_dense_products(nmd_handle* h, int32_t side, int64_t block, int32_t kind, float* d_L,
                              int64_t* rows, int64_t* cols) {
  if (!h || !d_L) return fail(h, NMD_ERR_INVALID, "NULL argument to nmd_dense_products");
  DeviceScope dg(h);
  Roles ro;
  nmd_status st = roles(h, side, block, kind, &ro);
  if (st != NMD_OK) return st;
  if (h->opt.precision == NMD_SIMT) return fail(h, NMD_ERR_UNSUPPORTED, "dense products hook needs a tensor-core precision");
  StepArgs a{ro.fm, ro.fq, ro.m0, ro.M, ro.q0, ro.K, h->r, h->rp, h->opt.precision, h->opt.epilogue, h->num_sms,
              h->opt.skip_zero_chunks == NMD_SKIP_VOTE};
  st = launch_panel_tc(a, h->ws.R, h->ws.status, h->ws.counters, h->num_sms, h->stream, &h->launches, d_L);
  if (st != NMD_OK) return fail(h, st, "no tensor-core kernel for this rank/precision on this device");
  if ((st = after_launch(h, "dense products")) != NMD_OK) return st;
  if ((st = sync_and_check(h)) != NMD_OK) return st;
  if (rows) *rows = ro.M;
  if (cols) *cols = ro.K;
  return NMD_OK;
}

nmd_status nmd_embed(nmd_handle* h, float* d_xi, float* d_sigma) {
  if (!h || !d_xi) return fail(h, NMD_ERR_INVALID, "NULL argument to nmd_embed");
  if (h->m != h->n) return fail(h, NMD_ERR_INVALID, "the cell embedding needs a square matrix (m == n)");
  if (h->r > embed_max_rank()) return fail(h, NMD_ERR_INVALID, "the cell embedding supports r <= 128");
  DeviceScope dg(h);
  nmd_status st = wait_all_pending(h);
  if (st != NMD_OK) return st;
  if ((int64_t)h->n * h->rp < 6 * (int64_t)h->r * h->r)   // the r x r work space lives in R
    return fail(h, NMD_ERR_INVALID, "the cell embedding needs at least 6 r cells");
  st = launch_embed(h->W, h->B, h->n, h->r, h->rp, h->ws.gram_part, h->ws.G, h->ws.G2, h->ws.R, h->ws.Gx,
                    h->ws.Tm, d_sigma ? d_sigma : h->ws.Ginv2, d_xi, h->num_sms, h->stream, &h->launches);
  if (st != NMD_OK) return fail(h, st, "cudaFuncSetAttribute(embed_rows_kernel)");
  return after_launch(h, "embedding");
}

nmd_status nmd_range_mask(nmd_handle* h, int32_t side, int64_t block, int32_t kind, uint32_t* mask,
                          int64_t capacity, int64_t* ntiles, int64_t* words, int64_t* chunk_rows) {
  if (!h || !ntiles || !words || !chunk_rows) return fail(h, NMD_ERR_INVALID, "NULL argument to nmd_range_mask");
  DeviceScope dg(h);
  Roles ro;
  nmd_status st = roles(h, side, block, kind, &ro);
  if (st != NMD_OK) return st;
  if (h->opt.precision == NMD_SIMT) return fail(h, NMD_ERR_UNSUPPORTED, "range mask hook needs a tensor-core precision");
  if ((st = wait_all_pending(h)) != NMD_OK) return st;
  StepArgs a{ro.fm, ro.fq, ro.m0, ro.M, ro.q0, ro.K, h->r, h->rp, h->opt.precision, h->opt.epilogue, h->num_sms};
  range_pass(h, ro, &a, h->stream);
  if ((st = after_launch(h, "range mask")) != NMD_OK) return st;
  if ((st = sync_and_check(h)) != NMD_OK) return st;
  *ntiles = (ro.M + 127) / 128;
  *words = a.rwords;
  *chunk_rows = panel_chunk_rows(h->rp, h->opt.precision);
  if (mask && capacity >= *ntiles * *words)
    CK(h, cudaMemcpy(mask, h->ws.rmask, (size_t)(*ntiles * *words) * sizeof(uint32_t), cudaMemcpyDeviceToHost));
  return NMD_OK;
}

nmd_status nmd_support_term(nmd_handle* h, int32_t side, int64_t block, int32_t kind, float* d_R, int64_t* rows) {
  if (!h || !d_R) return fail(h, NMD_ERR_INVALID, "NULL argument to nmd_support_term");
  DeviceScope dg(h);
  Roles ro;
  nmd_status st = roles(h, side, block, kind, &ro);
  if (st != NMD_OK) return st;
  if ((st = wait_all_pending(h)) != NMD_OK) return st;
  StepArgs a{ro.fm, ro.fq, ro.m0, ro.M, ro.q0, ro.K, h->r, h->rp, h->opt.precision, h->opt.epilogue, h->num_sms,
              h->opt.skip_zero_chunks == NMD_SKIP_VOTE};
  cudaStream_t s = h->stream;
  CK(h, cudaMemsetAsync(d_R, 0, (size_t)ro.M * h->rp * sizeof(float), s));
  {
    TimedScope ts(h, NMD_K_SPARSE, s);
    launch_span(h, a, ro, panel_span(ro), d_R, s);
  }
  if ((st = after_launch(h, "support term")) != NMD_OK) return st;
  if (rows) *rows = ro.M;
  return NMD_OK;
}

nmd_status nmd_panel_traversal(const nmd_handle* h, int32_t side, int64_t block, int32_t kind,
                               int64_t* rows_out, int64_t* q_out, int64_t cap, int64_t* count) {
  if (!h || !count) return NMD_ERR_INVALID;
  DeviceScope dg(h);
  Roles ro;
  nmd_status st = roles(const_cast<nmd_handle*>(h), side, block, kind, &ro);
  if (st != NMD_OK) return st;
  // host mirrors of the index arrays are not kept; rebuild q from the device copy
  const PanelSet& P = *ro.P;
  std::vector<PanelRow> list(P.host.begin() + P.row_ptr[block], P.host.begin() + P.row_ptr[block + 1]);
  const int64_t gs = P.seg_ptr[block] + P.segd[block];   // first slice of the split rows
  list.insert(list.end(), P.seg.begin() + P.seg_ptr[block], P.seg.begin() + gs);
  for (int64_t u = P.multi_ptr[block]; u < P.multi_ptr[block + 1]; ++u) {
    const PanelRow& mr = P.multi[u];
    const PanelRow& first = P.seg[gs + mr.beg];
    int64_t len = 0;
    for (int32_t q = 0; q < mr.len; ++q) len += P.seg[gs + mr.beg + q].len;
    list.push_back(PanelRow{mr.row, (int32_t)len, first.beg});
  }
  std::sort(list.begin(), list.end(), [](const PanelRow& a, const PanelRow& b) { return a.row < b.row; });
  int64_t total = 0;
  for (auto& pr : list) total += pr.len;
  *count = total;
  if (!rows_out || !q_out || cap <= 0) return NMD_OK;
  std::vector<int32_t> idx;
  int64_t w = 0;
  for (auto& pr : list) {
    idx.resize(pr.len);
    cudaError_t e = cudaMemcpy(idx.data(), ro.qidx + pr.beg, (size_t)pr.len * 4, cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_check(const_cast<nmd_handle*>(h), e, "traversal copy");
    for (int64_t k = 0; k < pr.len && w < cap; ++k, ++w) {
      rows_out[w] = pr.row - ro.m0;
      q_out[w] = idx[k] - ro.q0;
    }
  }
  return NMD_OK;
}

nmd_status nmd_get_state(nmd_handle* h, float* W, float* H, float* EW, float* EH, int64_t* sweep_index) {
  if (!h) return NMD_ERR_INVALID;
  DeviceScope dg(h);
  nmd_status st = nmd_get_factors(h, W, H, 0);
  if (st != NMD_OK) return st;
  cudaStream_t s = h->stream;
  if (EW) {
    launch_unpack(h->W.E, false, h->m, h->r, h->rp, h->ws.R, s);
    h->launches++;
    CK(h, cudaMemcpyAsync(EW, h->ws.R, (size_t)h->m * h->r * 4, cudaMemcpyDeviceToHost, s));
  }
  if (EH) {
    launch_unpack(h->B.E, true, h->n, h->r, h->rp, h->ws.R, s);
    h->launches++;
    CK(h, cudaMemcpyAsync(EH, h->ws.R, (size_t)h->n * h->r * 4, cudaMemcpyDeviceToHost, s));
  }
  CK(h, cudaStreamSynchronize(s));
  if (sweep_index) *sweep_index = h->sweep_index;
  return NMD_OK;
}

nmd_status nmd_set_state(nmd_handle* h, const float* W, const float* H, const float* EW, const float* EH,
                         int64_t sweep_index) {
  if (!h || !W || !H || !EW || !EH || sweep_index < 0) return fail(h, NMD_ERR_INVALID, "bad nmd_set_state argument");
  DeviceScope dg(h);
  nmd_status st = nmd_set_factors(h, W, H, 0);
  if (st != NMD_OK) return st;
  cudaStream_t s = h->stream;
  // momentum: pack into the master buffers' E (pack writes master/hi/lo of a
  // Factor, so pack into a temporary view whose master is E)
  Factor tw = h->W, tb = h->B;
  tw.master = h->W.E; tw.hi = nullptr; tw.lo = nullptr; tw.lo2 = nullptr;
  tb.master = h->B.E; tb.hi = nullptr; tb.lo = nullptr; tb.lo2 = nullptr;
  CK(h, cudaMemcpyAsync(h->ws.R, EW, (size_t)h->m * h->r * 4, cudaMemcpyHostToDevice, s));
  launch_pack(h->ws.R, false, h->m, h->r, h->rp, tw, s);
  CK(h, cudaMemcpyAsync(h->ws.R, EH, (size_t)h->n * h->r * 4, cudaMemcpyHostToDevice, s));
  launch_pack(h->ws.R, true, h->n, h->r, h->rp, tb, s);
  h->launches += 2;
  if ((st = after_launch(h, "set state")) != NMD_OK) return st;
  CK(h, cudaStreamSynchronize(s));
  h->sweep_index = sweep_index;
  return NMD_OK;
}

nmd_status nmd_profile(nmd_handle* h, int on) {
  if (!h) return NMD_ERR_INVALID;
  DeviceScope dg(h);
  CK(h, cudaStreamSynchronize(h->stream));
  collect_timing(h);
  for (int c = 0; c < 5; ++c) {
    h->prof_ms[c] = 0.0;
    h->prof_launches[c] = 0;
  }
  h->profiling = on != 0;
  return NMD_OK;
}

nmd_status nmd_profile_read(nmd_handle* h, int32_t kernel_class, double* ms, int64_t* launches) {
  if (!h || kernel_class < 0 || kernel_class > 4) return NMD_ERR_INVALID;
  DeviceScope dg(h);
  CK(h, cudaStreamSynchronize(h->stream));
  collect_timing(h);
  if (ms) *ms = h->prof_ms[kernel_class];
  if (launches) *launches = h->prof_launches[kernel_class];
  return NMD_OK;
}

void nmd_destroy(nmd_handle* h) {
  DeviceScope dg(h);
  delete h;
}

}  // extern "C"
