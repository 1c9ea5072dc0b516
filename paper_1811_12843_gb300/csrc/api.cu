// C ABI and host scheduler of the grid-iteration engine (declared in include/lipz.h).
//
// The grid owns two population snapshots per population (ping-pong A/B): an iteration reads
// snapshot `cur` (evaluation, selection, gradients) and writes every cell's new centre into
// snapshot 1 - cur, so no cell can see a neighbour's half-updated state. Work is enqueued on
// one CUDA stream, the kernels with programmatic dependent launch (each kernel's set-up
// overlaps the previous kernel's tail; its first global access waits for that kernel); the
// host waits only when the caller asks for host-side results.
#include <climits>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <string>
#include <vector>

#include "common.cuh"
#include "engine.h"
#include "bwd_tc.h"
#include "dcgan.h"
#include "fwd_tc.h"
#include "lipz.h"

using namespace lipz;

namespace {

enum Phase { PH_IDLE = 0, PH_EVALUATED = 1, PH_SELECTED = 2 };

thread_local std::string t_create_err;

struct Descs {
  // evaluation (per parity of the snapshot): generator layers over (cell, slot i),
  // discriminator layers over (cell, slot j)
  GemmDesc *g1, *g2, *g3, *d1, *d2;
  GemvDesc* d3;
  // training (per parity): forward of the selected pair and its backward
  GemmDesc *tg1, *tg2, *td1, *td2, *bw2d, *bd1, *bw1d, *ba3, *bw3g, *ba2, *bw2g, *ba1, *bw1g;
  GemvDesc* tgv;
  ColSumDesc *cb1d, *cb3g, *cb2g, *cb1g;  // bias gradients (D's b2 comes from k_dlogit)
};

}  // namespace

struct lipz_grid {
  int rows = 0, cols = 0, cells = 0;
  lipz_arch a{};
  uint64_t seed = 0;
  int64_t t = 0;
  bool bf = false;
  size_t esz = 4;
  Layout lg{}, ld{};
  int64_t PG = 0, PD = 0, PGs = 0, PDs = 0;
  int64_t e_cell = 0;  // elements per cell of the evaluation input E (6B rows)
  cudaStream_t st = nullptr;      // stream all work is enqueued on
  cudaStream_t own_st = nullptr;  // the grid's own non-blocking stream (the default)
  cudaStream_t copy_st = nullptr;  // host minibatch uploads, overlapping the generator forward
  cudaEvent_t ev_x = nullptr;      // the upload of the caller's minibatch has landed
  // lipz_iterate_batch_next: a second staging buffer (allocated on first use) and the
  // minibatch uploaded ahead into buffer pre_buf (0: xin, 1: xin2) from host address pre_host
  float* xin2 = nullptr;
  cudaEvent_t ev_x2 = nullptr;
  const float* pre_host = nullptr;
  int pre_buf = -1;
  int* hstat = nullptr;            // pinned host copies of the device error flags
  // lipz_iterate_batch_async: per call slot (alternating) a pinned copy of its iteration's
  // fitnesses and device status words (gathered on the device into `astage` first: one copy)
  // with the caller's result pointers, and an event at its end; per staging buffer an event
  // after the last iteration that read it (an upload into the buffer waits for it)
  float* astage = nullptr;         // device [2 cells 5 fitnesses][8 status words]
  float* hstat_a = nullptr;        // pinned [2 slots][the same]
  float* a_fit[2][2] = {};         // per slot: the caller's fit_g, fit_d
  cudaEvent_t ev_it[2] = {nullptr, nullptr};
  cudaEvent_t ev_buf[2] = {nullptr, nullptr};
  bool buf_read[2] = {false, false};
  int a_last = 1;                  // slot of the newest call
  bool a_pending = false;          // the newest call's status is still to be reported
  int device = 0;
  // population snapshots: ping-pong pair, or three in rotation with stale neighbours (the
  // snapshot being written must not be the one the stale neighbours are read from)
  PopView G[3]{}, D[3]{};
  int nsnap = 2;
  int cur = 0;
  int phase = PH_IDLE;
  bool use_tc = false;
  std::vector<void*> allocs;
  std::string err;

  // data and work buffers
  void* pool = nullptr;  // [pool_n][x_dim] in the population precision
  int64_t pool_n = 0, pool_cap = 0;
  float* xin = nullptr;  // caller-supplied minibatch staging [cells][B][x_dim]
  void *Z = nullptr, *E = nullptr, *H1g = nullptr, *H2g = nullptr, *H1d = nullptr, *H2d = nullptr;
  float *logits = nullptr, *LG = nullptr, *LD = nullptr, *fG = nullptr, *fD = nullptr;
  // neighbour tables [cells][5] of individual indices (snapshot * cells + cell) per snapshot
  // parity: every slot from the current snapshot, or (stale neighbours) slots 1..4 from the
  // other snapshot, which holds the previous iteration's centres
  int *nbr_cur[3]{}, *nbr_stale[3]{};
  // the same tables as work lists of the CTA-pair evaluation kernels (tensor-core path)
  TcPairs pairs_cur[3]{}, pairs_stale[3]{};
  bool prev_valid = false;  // the other snapshot holds the previous iteration's centres
  int *sel_g = nullptr, *sel_d = nullptr, *src_g = nullptr, *src_d = nullptr;
  float *lrn_g = nullptr, *lrn_d = nullptr;
  float4 *coef_g = nullptr, *coef_d = nullptr;  // per cell: lr, 1/bc1, 1/bc2, step + 1
  void *TH1 = nullptr, *TH2 = nullptr, *TX = nullptr, *TG1 = nullptr, *TG2 = nullptr;
  float* TL = nullptr;
  void *J2 = nullptr, *D1 = nullptr, *A3 = nullptr, *A2 = nullptr, *A1 = nullptr;
  float *gG = nullptr, *gD = nullptr;
  int* flag = nullptr;
  // generator-mixture weights [cells][5] (always held: part of the state), and with
  // arch.mixture the score's work buffers: row norms [cells][6B], per-row block sums
  // [cells][6B][mix_nh][6], block means [cells][6][6], scores [cells]; the CUDA-core path
  // stores the Gram matrices [cells][6B][6B] first
  float *mix = nullptr, *rnorm = nullptr, *mixP = nullptr, *mixS = nullptr, *mixScore = nullptr;
  float* gram = nullptr;
  GemmDesc* dgram = nullptr;
  int mix_nh = 1;
  bool mix_tc = false;
  Descs dsc[3]{}, dsc_stale[3]{};
  TcPlan* tc[3]{};
  TcbPlan* tcb[3]{};
  DcPlan* dc = nullptr;  // LIPZ_DCGAN64: the convolutional networks' plan
  bool dcgan = false;
  bool use_tcb = false;

  // tracing: event pairs per phase execution, resolved at lipz_profile_read
  bool prof = false;
  std::vector<cudaEvent_t> ev_free;
  struct Mark {
    int phase;
    cudaEvent_t a, b;
  };
  std::vector<Mark> marks;
  cudaEvent_t open_ev[LIPZ_N_PHASES]{};
  int64_t launches[LIPZ_N_PHASES]{};
  int64_t counts[LIPZ_N_PHASES]{};
};

namespace {

int fail(lipz_grid* g, int code, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  if (g) g->err = buf;
  else t_create_err = buf;
  return code;
}

#define CK(g, call)                                                                   \
  do {                                                                                \
    cudaError_t e_ = (call);                                                          \
    if (e_ != cudaSuccess)                                                            \
      return fail((g), e_ == cudaErrorMemoryAllocation ? LIPZ_ERR_OOM : LIPZ_ERR_CUDA, \
                  "%s failed: %s (%s:%d)", #call, cudaGetErrorString(e_), __FILE__,   \
                  __LINE__);                                                          \
  } while (0)

#define CKL(g)                                                                               \
  do {                                                                                       \
    cudaError_t e_ = cudaGetLastError();                                                     \
    if (e_ != cudaSuccess)                                                                   \
      return fail((g), LIPZ_ERR_CUDA, "kernel launch failed: %s (%s:%d)", cudaGetErrorString(e_), \
                  __FILE__, __LINE__);                                                       \
  } while (0)

template <typename T>
int dalloc(lipz_grid* g, T** p, size_t bytes) {
  void* q = nullptr;
  if (bytes == 0) bytes = 16;
  cudaError_t e = cudaMalloc(&q, bytes);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return fail(g, e == cudaErrorMemoryAllocation ? LIPZ_ERR_OOM : LIPZ_ERR_CUDA,
                "cudaMalloc(%zu bytes) failed: %s", bytes, cudaGetErrorString(e));
  }
  g->allocs.push_back(q);
  *p = (T*)q;
  return LIPZ_OK;
}

cudaEvent_t take_event(lipz_grid* g) {
  if (!g->ev_free.empty()) {
    cudaEvent_t e = g->ev_free.back();
    g->ev_free.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  if (cudaEventCreate(&e) != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  return e;
}

void phase_begin(lipz_grid* g, int ph) {
  if (!g->prof) return;
  cudaEvent_t e = take_event(g);
  if (e) cudaEventRecord(e, g->st);
  g->open_ev[ph] = e;
}

// Closes a phase: counts its kernel launches and, when tracing, records its stop event.
void phase_end(lipz_grid* g, int ph, int n_launches) {
  g->launches[ph] += n_launches;
  g->counts[ph] += 1;
  if (!g->prof || !g->open_ev[ph]) return;
  cudaEvent_t e = take_event(g);
  if (!e) return;
  cudaEventRecord(e, g->st);
  g->marks.push_back({ph, g->open_ev[ph], e});
  g->open_ev[ph] = nullptr;
}

int64_t round_up(int64_t v, int64_t m) { return (v + m - 1) / m * m; }

// Layouts (PyTorch Linear convention, W [out][in] row-major).
void make_layouts(lipz_grid* g) {
  const int64_t z = g->a.z_dim, h = g->a.hidden, x = g->a.x_dim;
  if (g->dcgan) {
    dc_layouts((int)z, g->a.ngf, g->a.ndf, &g->lg, &g->ld);
    g->PG = g->lg.off[g->lg.n];
    g->PD = g->ld.off[g->ld.n];
    g->PGs = round_up(g->PG, 64);
    g->PDs = round_up(g->PD, 64);
    return;
  }
  auto build = [](Layout& L, const int64_t shapes[6][2]) {
    L = Layout{};
    L.n = 6;
    L.off[0] = 0;
    for (int t = 0; t < 6; ++t) {
      L.off[t + 1] = L.off[t] + shapes[t][0] * shapes[t][1];
      L.bound[t] = (t % 2 == 0)
                       ? (float)std::sqrt(6.0 / (double)(shapes[t][0] + shapes[t][1]))
                       : 0.f;
    }
  };
  const int64_t gs[6][2] = {{h, z}, {1, h}, {h, h}, {1, h}, {x, h}, {1, x}};
  const int64_t ds[6][2] = {{h, x}, {1, h}, {h, h}, {1, h}, {1, h}, {1, 1}};
  build(g->lg, gs);
  build(g->ld, ds);
  g->PG = g->lg.off[6];
  g->PD = g->ld.off[6];
  g->PGs = round_up(g->PG, 64);
  g->PDs = round_up(g->PD, 64);
}

const void* act_w(const PopView& p) { return p.wb ? (const void*)p.wb : (const void*)p.w; }

char* eoff(const void* base, int64_t elems, size_t esz) {
  return (char*)base + elems * (int64_t)esz;
}

GemmDesc gd(const void* A, int64_t sam, int64_t sak, const void* B, int64_t sbk, int64_t sbn,
            void* C, int64_t scm, int64_t scn, int M, int N, int K) {
  GemmDesc d;
  memset(&d, 0, sizeof d);
  d.A = A;
  d.B = B;
  d.C = C;
  d.sam = sam;
  d.sak = sak;
  d.sbk = sbk;
  d.sbn = sbn;
  d.scm = scm;
  d.scn = scn;
  d.M = M;
  d.N = N;
  d.K = K;
  return d;
}

// Host -> device copy and memset in the order of the grid's stream (which need not be the
// legacy default stream); the copy returns once the host buffer may be reused.
int h2d(lipz_grid* g, void* dst, const void* src, size_t bytes) {
  CK(g, cudaMemcpyAsync(dst, src, bytes, cudaMemcpyHostToDevice, g->st));
  CK(g, cudaStreamSynchronize(g->st));
  return LIPZ_OK;
}
int dset(lipz_grid* g, void* dst, int value, size_t bytes) {
  CK(g, cudaMemsetAsync(dst, value, bytes, g->st));
  return LIPZ_OK;
}

template <typename T>
int upload(lipz_grid* g, T** dst, const std::vector<T>& v) {
  int rc = dalloc(g, dst, v.size() * sizeof(T));
  if (rc) return rc;
  return h2d(g, *dst, v.data(), v.size() * sizeof(T));
}

// Snapshot written by an iteration that reads snapshot p, and the one it read before p.
int snap_next(const lipz_grid* g, int p) { return (p + 1) % g->nsnap; }
int snap_prev(const lipz_grid* g, int p) { return (p + g->nsnap - 1) % g->nsnap; }

int build_descs(lipz_grid* g, int p) {
  const int C = g->cells, B = g->a.batch, z = g->a.z_dim, h = g->a.hidden, x = g->a.x_dim;
  const size_t es = g->esz;
  // both snapshots are one allocation: individual k of the index space is snapshot k / C
  const PopView &Gp = g->G[0], &Dp = g->D[0];
  const void* Gw = act_w(Gp);
  const void* Dw = act_w(Dp);
  const Layout &L = g->lg, &M = g->ld;
  std::vector<int> nbr(C * 5), cur(C * 5), stale(C * 5);
  for (int r = 0; r < g->rows; ++r)
    for (int q = 0; q < g->cols; ++q) {
      int* n = &nbr[(r * g->cols + q) * 5];
      n[0] = r * g->cols + q;
      n[1] = ((r - 1 + g->rows) % g->rows) * g->cols + q;
      n[2] = ((r + 1) % g->rows) * g->cols + q;
      n[3] = r * g->cols + (q - 1 + g->cols) % g->cols;
      n[4] = r * g->cols + (q + 1) % g->cols;
    }
  for (int i = 0; i < C * 5; ++i) {
    cur[i] = p * C + nbr[i];
    stale[i] = (i % 5 == 0 ? p : snap_prev(g, p)) * C + nbr[i];
  }
  if (g->dcgan) {
    int rc;
    if ((rc = upload(g, &g->nbr_cur[p], cur)) || (rc = upload(g, &g->nbr_stale[p], stale)))
      return rc;
    return LIPZ_OK;
  }
  // pair lists of both tables for the tensor-core evaluation
  auto pair_lists = [&](const std::vector<int>& tab, TcPairs& P) -> int {
    std::vector<int4> gp, dp;
    std::vector<int2> pl;
    tc_build_pairs(tab.data(), C, g->nsnap * C, B, &gp, &dp, &pl);
    int4 *dg = nullptr, *dd = nullptr;
    int2* dl = nullptr;
    int rc;
    if ((rc = upload(g, &dg, gp)) || (rc = upload(g, &dd, dp)) || (rc = upload(g, &dl, pl)))
      return rc;
    P = TcPairs{dg, (int)gp.size(), dd, (int)dp.size(), dl};
    return LIPZ_OK;
  };
  {
    int rc;
    if ((rc = pair_lists(cur, g->pairs_cur[p])) ||
        (g->a.stale_neighbors && (rc = pair_lists(stale, g->pairs_stale[p]))))
      return rc;
  }
  // evaluation descriptors of one neighbour table
  auto eval_descs = [&](const std::vector<int>& tab, Descs& D) -> int {
    std::vector<GemmDesc> g1, g2, g3, d1, d2;
    std::vector<GemvDesc> d3;
    for (int c = 0; c < C; ++c)
      for (int s = 0; s < 5; ++s) {
        const int k = tab[c * 5 + s];
        const int64_t pg = (int64_t)k * g->PGs, pd = (int64_t)k * g->PDs;
        const int64_t cs = (int64_t)c * 5 + s;
        GemmDesc a = gd(eoff(g->Z, (int64_t)c * B * z, es), z, 1, eoff(Gw, pg + L.off[0], es), 1, z,
                        eoff(g->H1g, cs * B * h, es), h, 1, B, h, z);
        a.bias = Gp.w + pg + L.off[1];
        g1.push_back(a);
        GemmDesc b = gd(eoff(g->H1g, cs * B * h, es), h, 1, eoff(Gw, pg + L.off[2], es), 1, h,
                        eoff(g->H2g, cs * B * h, es), h, 1, B, h, h);
        b.bias = Gp.w + pg + L.off[3];
        g2.push_back(b);
        GemmDesc e = gd(eoff(g->H2g, cs * B * h, es), h, 1, eoff(Gw, pg + L.off[4], es), 1, h,
                        eoff(g->E, (int64_t)c * g->e_cell + (int64_t)(1 + s) * B * x, es), x, 1, B,
                        x, h);
        e.bias = Gp.w + pg + L.off[5];
        g3.push_back(e);
        GemmDesc f = gd(eoff(g->E, (int64_t)c * g->e_cell, es), x, 1, eoff(Dw, pd + M.off[0], es), 1,
                        x, eoff(g->H1d, cs * 6 * B * h, es), h, 1, 6 * B, h, x);
        f.bias = Dp.w + pd + M.off[1];
        d1.push_back(f);
        GemmDesc q2 = gd(eoff(g->H1d, cs * 6 * B * h, es), h, 1, eoff(Dw, pd + M.off[2], es), 1, h,
                         eoff(g->H2d, cs * 6 * B * h, es), h, 1, 6 * B, h, h);
        q2.bias = Dp.w + pd + M.off[3];
        d2.push_back(q2);
        GemvDesc v;
        memset(&v, 0, sizeof v);
        v.X = eoff(g->H2d, cs * 6 * B * h, es);
        v.w = eoff(Dw, pd + M.off[4], es);
        v.bias = Dp.w + pd + M.off[5];
        v.out = g->logits + cs * 6 * B;
        v.ld = h;
        v.rows = 6 * B;
        v.K = h;
        d3.push_back(v);
      }
    int rc;
    if ((rc = upload(g, &D.g1, g1)) || (rc = upload(g, &D.g2, g2)) ||
        (rc = upload(g, &D.g3, g3)) || (rc = upload(g, &D.d1, d1)) ||
        (rc = upload(g, &D.d2, d2)) || (rc = upload(g, &D.d3, d3)))
      return rc;
    return LIPZ_OK;
  };
  {
    int rc;
    if ((rc = upload(g, &g->nbr_cur[p], cur)) || (rc = upload(g, &g->nbr_stale[p], stale)) ||
        (rc = eval_descs(cur, g->dsc[p])) ||
        (g->a.stale_neighbors && (rc = eval_descs(stale, g->dsc_stale[p]))))
      return rc;
  }
  Descs& D = g->dsc[p];
  int rc;

  // ---- training descriptors: weights of the selected individual (wsel = src_g / src_d)
  std::vector<GemmDesc> tg1, tg2, td1, td2, bw2d, bd1, bw1d, ba3, bw3g, ba2, bw2g, ba1, bw1g;
  std::vector<GemvDesc> tgv;
  std::vector<ColSumDesc> cb1d, cb3g, cb2g, cb1g;
  auto selg = [&](GemmDesc d, int c) {
    d.wsel = g->src_g;
    d.wsel_stride = g->PGs;
    d.wsel_op = 2;
    d.cell = c;
    return d;
  };
  auto seld = [&](GemmDesc d, int c) {
    d.wsel = g->src_d;
    d.wsel_stride = g->PDs;
    d.wsel_op = 2;
    d.cell = c;
    return d;
  };
  auto cs = [](const void* X, float* out, int64_t ld, int rows, int cols) {
    ColSumDesc d;
    d.X = X;
    d.out = out;
    d.ld = ld;
    d.rows = rows;
    d.cols = cols;
    return d;
  };
  for (int c = 0; c < C; ++c) {
    const void* Zc = eoff(g->Z, (int64_t)c * B * z, es);
    void* TH1c = eoff(g->TH1, (int64_t)c * B * h, es);
    void* TH2c = eoff(g->TH2, (int64_t)c * B * h, es);
    void* TXc = eoff(g->TX, (int64_t)c * 2 * B * x, es);
    void* TG1c = eoff(g->TG1, (int64_t)c * 2 * B * h, es);
    void* TG2c = eoff(g->TG2, (int64_t)c * 2 * B * h, es);
    void* J2c = eoff(g->J2, (int64_t)c * 3 * B * h, es);
    void* D1c = eoff(g->D1, (int64_t)c * 3 * B * h, es);
    void* A3c = eoff(g->A3, (int64_t)c * B * x, es);
    void* A2c = eoff(g->A2, (int64_t)c * B * h, es);
    void* A1c = eoff(g->A1, (int64_t)c * B * h, es);
    float* gGc = g->gG + (int64_t)c * g->PGs;
    float* gDc = g->gD + (int64_t)c * g->PDs;

    GemmDesc a = selg(gd(Zc, z, 1, eoff(Gw, L.off[0], es), 1, z, TH1c, h, 1, B, h, z), c);
    a.bias = Gp.w + L.off[1];
    tg1.push_back(a);
    a = selg(gd(TH1c, h, 1, eoff(Gw, L.off[2], es), 1, h, TH2c, h, 1, B, h, h), c);
    a.bias = Gp.w + L.off[3];
    tg2.push_back(a);
    a = seld(gd(TXc, x, 1, eoff(Dw, M.off[0], es), 1, x, TG1c, h, 1, 2 * B, h, x), c);
    a.bias = Dp.w + M.off[1];
    td1.push_back(a);
    a = seld(gd(TG1c, h, 1, eoff(Dw, M.off[2], es), 1, h, TG2c, h, 1, 2 * B, h, h), c);
    a.bias = Dp.w + M.off[3];
    td2.push_back(a);
    GemvDesc v;
    memset(&v, 0, sizeof v);
    v.X = TG2c;
    v.w = eoff(Dw, M.off[4], es);
    v.bias = Dp.w + M.off[5];
    v.out = g->TL + (int64_t)c * 2 * B;
    v.wsel = g->src_d;
    v.wsel_stride = g->PDs;
    v.cell = c;
    v.ld = h;
    v.rows = 2 * B;
    v.K = h;
    tgv.push_back(v);
    // discriminator backward
    bw2d.push_back(gd(J2c, 1, h, TG1c, h, 1, gDc + M.off[2], h, 1, h, h, 2 * B));
    a = seld(gd(J2c, h, 1, eoff(Dw, M.off[2], es), h, 1, D1c, h, 1, 2 * B, h, h), c);
    a.aux = TG1c;
    a.sxm = h;
    a.sxn = 1;
    bd1.push_back(a);
    a = seld(gd(eoff(J2c, 2 * (int64_t)B * h, es), h, 1, eoff(Dw, M.off[2], es), h, 1,
                eoff(D1c, 2 * (int64_t)B * h, es), h, 1, B, h, h), c);
    a.aux = eoff(TG1c, (int64_t)B * h, es);
    a.sxm = h;
    a.sxn = 1;
    bd1.push_back(a);
    bw1d.push_back(gd(D1c, 1, h, TXc, x, 1, gDc + M.off[0], x, 1, h, x, 2 * B));
    cb1d.push_back(cs(D1c, gDc + M.off[1], h, 2 * B, h));
    // generator backward: into the fakes through D's first layer, then through G
    a = seld(gd(eoff(D1c, 2 * (int64_t)B * h, es), h, 1, eoff(Dw, M.off[0], es), x, 1, A3c, x, 1,
                B, x, h), c);
    a.aux = eoff(TXc, (int64_t)B * x, es);
    a.sxm = x;
    a.sxn = 1;
    ba3.push_back(a);
    bw3g.push_back(gd(A3c, 1, x, TH2c, h, 1, gGc + L.off[4], h, 1, x, h, B));
    cb3g.push_back(cs(A3c, gGc + L.off[5], x, B, x));
    a = selg(gd(A3c, x, 1, eoff(Gw, L.off[4], es), h, 1, A2c, h, 1, B, h, x), c);
    a.aux = TH2c;
    a.sxm = h;
    a.sxn = 1;
    ba2.push_back(a);
    bw2g.push_back(gd(A2c, 1, h, TH1c, h, 1, gGc + L.off[2], h, 1, h, h, B));
    cb2g.push_back(cs(A2c, gGc + L.off[3], h, B, h));
    a = selg(gd(A2c, h, 1, eoff(Gw, L.off[2], es), h, 1, A1c, h, 1, B, h, h), c);
    a.aux = TH1c;
    a.sxm = h;
    a.sxn = 1;
    ba1.push_back(a);
    bw1g.push_back(gd(A1c, 1, h, Zc, z, 1, gGc + L.off[0], z, 1, h, z, B));
    cb1g.push_back(cs(A1c, gGc + L.off[1], h, B, h));
  }
  if ((rc = upload(g, &D.tg1, tg1)) || (rc = upload(g, &D.tg2, tg2)) ||
      (rc = upload(g, &D.td1, td1)) || (rc = upload(g, &D.td2, td2)) ||
      (rc = upload(g, &D.tgv, tgv)) || (rc = upload(g, &D.bw2d, bw2d)) ||
      (rc = upload(g, &D.bd1, bd1)) || (rc = upload(g, &D.bw1d, bw1d)) ||
      (rc = upload(g, &D.ba3, ba3)) || (rc = upload(g, &D.bw3g, bw3g)) ||
      (rc = upload(g, &D.ba2, ba2)) || (rc = upload(g, &D.bw2g, bw2g)) ||
      (rc = upload(g, &D.ba1, ba1)) || (rc = upload(g, &D.bw1g, bw1g)) ||
      (rc = upload(g, &D.cb1d, cb1d)) ||
      (rc = upload(g, &D.cb3g, cb3g)) || (rc = upload(g, &D.cb2g, cb2g)) ||
      (rc = upload(g, &D.cb1g, cb1g)))
    return rc;
  return LIPZ_OK;
}

// Grouped GEMM in the grid's precision; out_f32 selects an fp32 output (gradients).
void gemm(lipz_grid* g, const GemmDesc* d, int n, int M, int N, int epi, int act, bool out_f32) {
  const float sl = g->a.leaky_slope;
  if (g->bf) {
    if (out_f32) launch_gemm<bf16, float, EPI_STORE>(d, n, M, N, act, sl, g->st);
    else if (epi == EPI_BIAS_ACT) launch_gemm<bf16, bf16, EPI_BIAS_ACT>(d, n, M, N, act, sl, g->st);
    else launch_gemm<bf16, bf16, EPI_DACT>(d, n, M, N, act, sl, g->st);
  } else {
    if (out_f32 && epi == EPI_STORE) launch_gemm<float, float, EPI_STORE>(d, n, M, N, act, sl, g->st);
    else if (epi == EPI_BIAS_ACT) launch_gemm<float, float, EPI_BIAS_ACT>(d, n, M, N, act, sl, g->st);
    else launch_gemm<float, float, EPI_DACT>(d, n, M, N, act, sl, g->st);
  }
}

void gemv(lipz_grid* g, const GemvDesc* d, int n, int rows) {
  if (g->bf) launch_gemv<bf16>(d, n, rows, g->st);
  else launch_gemv<float>(d, n, rows, g->st);
}

void colsum_on(lipz_grid* g, const ColSumDesc* d, int n, int cols, cudaStream_t st) {
  if (g->bf) launch_colsum<bf16>(d, n, cols, st);
  else launch_colsum<float>(d, n, cols, st);
}

void colsum(lipz_grid* g, const ColSumDesc* d, int n, int cols) { colsum_on(g, d, n, cols, g->st); }

int check_arch(const lipz_arch* a) {
  if (!a) return fail(nullptr, LIPZ_ERR_INVALID, "arch is null");
  if (a->struct_size != sizeof(lipz_arch))
    return fail(nullptr, LIPZ_ERR_INVALID, "arch.struct_size is %u, expected %zu", a->struct_size,
                sizeof(lipz_arch));
  if (a->kind != LIPZ_MLP && a->kind != LIPZ_DCGAN64)
    return fail(nullptr, LIPZ_ERR_INVALID, "arch.kind must be LIPZ_MLP or LIPZ_DCGAN64");
  if (a->kind == LIPZ_DCGAN64 &&
      (a->x_dim != 3 * 64 * 64 || a->ngf < 1 || a->ndf < 1 || a->ngf > 512 || a->ndf > 512 ||
       a->train_steps != 1))
    return fail(nullptr, LIPZ_ERR_INVALID,
                "LIPZ_DCGAN64 needs x_dim == 12288, ngf and ndf in 1..512 and train_steps == 1");
  if (a->precision != LIPZ_FP32 && a->precision != LIPZ_BF16)
    return fail(nullptr, LIPZ_ERR_INVALID, "arch.precision must be LIPZ_FP32 or LIPZ_BF16");
  if (a->z_dim < 1 || a->hidden < 1 || a->x_dim < 1 || a->batch < 1 || a->hidden > 1024 ||
      a->batch > 4096 || a->z_dim > 65536 || a->x_dim > 65536)
    return fail(nullptr, LIPZ_ERR_INVALID, "arch sizes out of range");
  if (a->tournament_size < 1 || a->tournament_size > 5)
    return fail(nullptr, LIPZ_ERR_INVALID, "tournament_size must be in 1..5");
  if (a->replace_mode != LIPZ_REPLACE_IF_BETTER && a->replace_mode != LIPZ_REPLACE_ALWAYS)
    return fail(nullptr, LIPZ_ERR_INVALID, "bad replace_mode");
  if (!(a->lr >= 0.f) || !(a->beta1 >= 0.f && a->beta1 < 1.f) ||
      !(a->beta2 >= 0.f && a->beta2 < 1.f) || !(a->eps > 0.f) || !(a->lr_mut_prob >= 0.f) ||
      !(a->lr_mut_prob <= 1.f))
    return fail(nullptr, LIPZ_ERR_INVALID, "bad optimiser / mutation hyper-parameters");
  if (a->train_steps < 1 || a->train_steps > 65536)
    return fail(nullptr, LIPZ_ERR_INVALID, "train_steps must be in 1..65536");
  if (a->stale_neighbors != 0 && a->stale_neighbors != 1)
    return fail(nullptr, LIPZ_ERR_INVALID, "stale_neighbors must be 0 or 1");
  if (a->stale_neighbors && a->train_steps != 1)
    return fail(nullptr, LIPZ_ERR_INVALID, "stale_neighbors needs train_steps == 1");
  if ((a->mixture != 0 && a->mixture != 1) || !(a->mix_sigma >= 0.f))
    return fail(nullptr, LIPZ_ERR_INVALID, "mixture must be 0 or 1 and mix_sigma >= 0");
  return LIPZ_OK;
}

// All snapshots of one population in one allocation per array (snapshot s at s * cells
// individuals), so that an individual index k = snapshot * cells + cell addresses any of them.
// w, m and v are three equal parts of one allocation (m = w + n, v = w + 2n floats), so that
// one 4-D tensor map reaches all three at once (the backward's fused Adam moves a chunk of
// each with a single TMA load and a single store).
int alloc_pops(lipz_grid* g, PopView* p, int64_t Ps) {
  const size_t C = g->cells, S = g->nsnap, n = S * C * Ps;
  PopView& a = p[0];
  int rc;
  if ((rc = dalloc(g, &a.w, 3 * n * 4)) || (rc = dalloc(g, &a.step, S * C * 4)) ||
      (rc = dalloc(g, &a.lr, S * C * 4)))
    return rc;
  a.m = a.w + n;
  a.v = a.w + 2 * n;
  a.wb = nullptr;
  if (g->bf && (rc = dalloc(g, &a.wb, n * 2))) return rc;
  if ((rc = dset(g, a.w, 0, n * 4)) || (rc = dset(g, a.m, 0, n * 4)) ||
      (rc = dset(g, a.v, 0, n * 4)) || (rc = dset(g, a.step, 0, S * C * 4)) ||
      (a.wb && (rc = dset(g, a.wb, 0, n * 2))))
    return rc;
  for (size_t s = 1; s < S; ++s) {
    PopView& b = p[s];
    b.w = a.w + s * C * Ps;
    b.m = a.m + s * C * Ps;
    b.v = a.v + s * C * Ps;
    b.wb = a.wb ? a.wb + s * C * Ps : nullptr;
    b.step = a.step + s * C;
    b.lr = a.lr + s * C;
  }
  return LIPZ_OK;
}

void bias_ranges(lipz_grid* g, int p, AdamRanges* rg, AdamRanges* rd);

int create_impl(lipz_grid* g) {
  const int C = g->cells, B = g->a.batch, z = g->a.z_dim, h = g->a.hidden, x = g->a.x_dim;
  const size_t es = g->esz;
  int rc;
  CK(g, cudaGetDevice(&g->device));
  // the grid's own stream (lipz_set_stream may replace it)
  CK(g, cudaStreamCreateWithFlags(&g->own_st, cudaStreamNonBlocking));
  g->st = g->own_st;
  CK(g, cudaStreamCreateWithFlags(&g->copy_st, cudaStreamNonBlocking));
  CK(g, cudaEventCreateWithFlags(&g->ev_x, cudaEventDisableTiming));
  CK(g, cudaMallocHost(&g->hstat, 8 * sizeof(int)));
  g->dcgan = g->a.kind == LIPZ_DCGAN64;
  make_layouts(g);
  g->e_cell = (int64_t)6 * B * x;
  g->nsnap = g->a.stale_neighbors ? 3 : 2;
  if ((rc = alloc_pops(g, g->G, g->PGs)) || (rc = alloc_pops(g, g->D, g->PDs))) return rc;
  const size_t CB = (size_t)C * B;
  if ((rc = dalloc(g, &g->Z, CB * z * es)) || (rc = dalloc(g, &g->E, (size_t)C * g->e_cell * es)) ||
      (rc = dalloc(g, &g->H1g, CB * 5 * h * es)) || (rc = dalloc(g, &g->H2g, CB * 5 * h * es)) ||
      (rc = dalloc(g, &g->H1d, CB * 30 * h * es)) || (rc = dalloc(g, &g->H2d, CB * 30 * h * es)) ||
      (rc = dalloc(g, &g->logits, CB * 30 * 4)) || (rc = dalloc(g, &g->LG, C * 25 * 4)) ||
      (rc = dalloc(g, &g->LD, C * 25 * 4)) || (rc = dalloc(g, &g->fG, C * 5 * 4)) ||
      (rc = dalloc(g, &g->fD, C * 5 * 4)) || (rc = dalloc(g, &g->sel_g, C * 4)) ||
      (rc = dalloc(g, &g->sel_d, C * 4)) || (rc = dalloc(g, &g->src_g, C * 4)) ||
      (rc = dalloc(g, &g->src_d, C * 4)) || (rc = dalloc(g, &g->lrn_g, C * 4)) ||
      (rc = dalloc(g, &g->lrn_d, C * 4)) || (rc = dalloc(g, &g->coef_g, C * 16)) ||
      (rc = dalloc(g, &g->coef_d, C * 16)) || (rc = dalloc(g, &g->TH1, CB * h * es)) ||
      (rc = dalloc(g, &g->TH2, CB * h * es)) || (rc = dalloc(g, &g->TX, CB * 2 * x * es)) ||
      (rc = dalloc(g, &g->TG1, CB * 2 * h * es)) || (rc = dalloc(g, &g->TG2, CB * 2 * h * es)) ||
      (rc = dalloc(g, &g->TL, CB * 2 * 4)) || (rc = dalloc(g, &g->J2, CB * 3 * h * es)) ||
      (rc = dalloc(g, &g->D1, CB * 3 * h * es)) || (rc = dalloc(g, &g->A3, CB * x * es)) ||
      (rc = dalloc(g, &g->A2, CB * h * es)) || (rc = dalloc(g, &g->A1, CB * h * es)) ||
      (rc = dalloc(g, &g->gG, (size_t)C * g->PGs * 4)) ||
      (rc = dalloc(g, &g->gD, (size_t)C * g->PDs * 4)) || (rc = dalloc(g, &g->flag, 4)) ||
      (rc = dalloc(g, &g->xin, CB * x * 4)) || (rc = dalloc(g, &g->mix, C * 5 * 4)))
    return rc;
  {
    std::vector<float> w(C * 5, 0.2f);
    if ((rc = h2d(g, g->mix, w.data(), C * 5 * 4))) return rc;
  }
  if (g->a.mixture) {
    const size_t R = (size_t)6 * B;
    g->mix_tc = g->bf && !g->a.force_simt && tc_supported(z, h, x, B) && tc_gram_supported(B);
    g->mix_nh = g->mix_tc ? tc_gram_halves(B) : 1;
    if ((rc = dalloc(g, &g->rnorm, C * R * 4)) ||
        (rc = dalloc(g, &g->mixP, C * R * g->mix_nh * 6 * 4)) ||
        (rc = dalloc(g, &g->mixS, C * 36 * 4)) || (rc = dalloc(g, &g->mixScore, C * 4)) ||
        (rc = dset(g, g->mixS, 0, C * 36 * 4)) || (rc = dset(g, g->mixScore, 0, C * 4)))
      return rc;
    if (!g->mix_tc) {
      if ((rc = dalloc(g, &g->gram, C * R * R * 4))) return rc;
      std::vector<GemmDesc> dg;
      for (int c = 0; c < C; ++c)
        dg.push_back(gd(eoff(g->E, (int64_t)c * g->e_cell, es), x, 1,
                        eoff(g->E, (int64_t)c * g->e_cell, es), 1, x,
                        g->gram + (int64_t)c * R * R, (int64_t)R, 1, (int)R, (int)R, x));
      if ((rc = upload(g, &g->dgram, dg))) return rc;
    }
  }
  const int big = INT_MAX;
  if ((rc = dset(g, g->gG, 0, (size_t)C * g->PGs * 4)) ||
      (rc = dset(g, g->gD, 0, (size_t)C * g->PDs * 4)) || (rc = h2d(g, g->flag, &big, 4)))
    return rc;
  // step 1: random initialisation of snapshot 0
  launch_init_params(g->G[0].w, g->G[0].wb, g->PG, g->PGs, g->lg, C, g->seed, LIPZ_STREAM_INIT_G,
                     g->st);
  launch_init_params(g->D[0].w, g->D[0].wb, g->PD, g->PDs, g->ld, C, g->seed, LIPZ_STREAM_INIT_D,
                     g->st);
  CKL(g);
  std::vector<float> lr(C, g->a.lr);
  for (int p = 0; p < g->nsnap; ++p)
    if ((rc = h2d(g, g->G[p].lr, lr.data(), C * 4)) || (rc = h2d(g, g->D[p].lr, lr.data(), C * 4)) ||
        (rc = build_descs(g, p)))
      return rc;
  g->use_tc = !g->dcgan && g->bf && !g->a.force_simt && tc_supported(z, h, x, B);
  if (g->dcgan) {
    DcShape s{C, B, z, g->a.ngf, g->a.ndf, g->bf, g->a.leaky_slope, g->nsnap * C};
    DcBuffers b{};
    b.Gw = g->G[0].w;
    b.Gop = act_w(g->G[0]);
    b.Dw = g->D[0].w;
    b.Dop = act_w(g->D[0]);
    b.PGs = g->PGs;
    b.PDs = g->PDs;
    b.goff = g->lg.off;
    b.doff = g->ld.off;
    b.Z = g->Z;
    b.E = g->E;
    b.e_cell = g->e_cell;
    b.logits = g->logits;
    b.src_g = g->src_g;
    b.src_d = g->src_d;
    b.gG = g->gG;
    b.gD = g->gD;
    std::string msg;
    g->dc = dc_plan_create(s, b, &msg);
    if (!g->dc) return fail(g, LIPZ_ERR_OOM, "DCGAN plan: %s", msg.c_str());
  }
  if (g->use_tc) {
    for (int p = 0; p < g->nsnap; ++p) {
      TcShape s{C, B, z, h, x, g->a.leaky_slope, g->nsnap * C};
      TcBuffers b{};
      b.Z = g->Z;
      b.E = g->E;
      b.e_cell = g->e_cell;
      b.logits = g->logits;
      b.nbr = g->nbr_cur[p];
      b.indiv_off = p * C;
      b.Gwb = g->G[0].wb;
      b.Gw = g->G[0].w;
      b.PGs = g->PGs;
      b.goff = g->lg.off;
      b.Dwb = g->D[0].wb;
      b.Dw = g->D[0].w;
      b.PDs = g->PDs;
      b.doff = g->ld.off;
      b.sel_g = g->sel_g;
      b.src_g = g->src_g;
      b.src_d = g->src_d;
      b.rnorm = g->mix_tc ? g->rnorm : nullptr;
      b.gram_out = g->mix_tc ? g->mixP : nullptr;
      b.TH1 = g->TH1;
      b.TH2 = g->TH2;
      b.TG1 = g->TG1;
      b.TG2 = g->TG2;
      b.TL = g->TL;
      std::string msg;
      g->tc[p] = tc_plan_create(s, b, &msg);
      if (!g->tc[p]) return fail(g, LIPZ_ERR_CUDA, "tensor-core plan: %s", msg.c_str());
    }
    g->use_tcb = tcb_supported(z, h, x, B);
    for (int p = 0; p < g->nsnap && g->use_tcb; ++p) {
      TcbShape s{C, B, z, h, x, g->a.leaky_slope, g->nsnap * C};
      TcbBuffers b{};
      b.Z = g->Z;
      b.E = g->E;
      b.e_cell = g->e_cell;
      b.sel_g = g->sel_g;
      b.TH1 = g->TH1;
      b.TH2 = g->TH2;
      b.TG1 = g->TG1;
      b.J2 = g->J2;
      b.D1 = g->D1;
      b.A3 = g->A3;
      b.A2 = g->A2;
      b.A1 = g->A1;
      b.gG = g->gG;
      b.gD = g->gD;
      b.Gwb = g->G[0].wb;
      b.Dwb = g->D[0].wb;
      b.PGs = g->PGs;
      b.PDs = g->PDs;
      b.goff = g->lg.off;
      b.doff = g->ld.off;
      b.src_g = g->src_g;
      b.src_d = g->src_d;
      // without keep_grads the weight matrices take their Adam step inside the backward
      b.fuse_adam = g->a.keep_grads ? 0 : 1;
      // old state: any individual of any snapshot (the selection's source); new: the next
      // snapshot
      const int q1 = snap_next(g, p);
      const PopView* pops[2][2] = {{&g->G[0], &g->G[q1]}, {&g->D[0], &g->D[q1]}};
      TcbBuffers::AdamPop* ap[2] = {&b.adam_g, &b.adam_d};
      for (int q = 0; q < 2; ++q) {
        ap[q]->w = pops[q][0]->w;
        ap[q]->m = pops[q][0]->m;
        ap[q]->v = pops[q][0]->v;
        ap[q]->w_new = pops[q][1]->w;
        ap[q]->m_new = pops[q][1]->m;
        ap[q]->v_new = pops[q][1]->v;
        ap[q]->wb_new = pops[q][1]->wb;
      }
      b.adam_g.coef = g->coef_g;
      b.adam_d.coef = g->coef_d;
      b.beta1 = g->a.beta1;
      b.beta2 = g->a.beta2;
      b.eps = g->a.eps;
      AdamRanges rr[2];
      bias_ranges(g, p, &rr[0], &rr[1]);
      b.ranges = b.fuse_adam ? rr : nullptr;
      std::string msg;
      g->tcb[p] = tcb_plan_create(s, b, &msg);
      if (!g->tcb[p]) return fail(g, LIPZ_ERR_CUDA, "tensor-core backward plan: %s", msg.c_str());
    }
  }
  // the plans' set-up (allocations, flag resets) ran outside the grid's stream
  CK(g, cudaDeviceSynchronize());
  return LIPZ_OK;
}

SelectParams select_params(const lipz_grid* g);
SelectIO select_io(lipz_grid* g);

// Neighbour table of the current evaluation: stale neighbours (the other snapshot's
// individuals in slots 1..4) once the other snapshot holds the previous iteration's centres.
const int* eval_nbr(const lipz_grid* g) {
  return g->a.stale_neighbors && g->prev_valid ? g->nbr_stale[g->cur] : g->nbr_cur[g->cur];
}
const TcPairs* eval_pairs(const lipz_grid* g) {
  return g->a.stale_neighbors && g->prev_valid ? &g->pairs_stale[g->cur] : &g->pairs_cur[g->cur];
}

// Minibatch step `step` of the current iteration into E's real rows and Z (the real rows from
// xin_dev when given, else from the pool).
void draw_batch(lipz_grid* g, const float* xin_dev, uint32_t step, int parts, bool pdl) {
  const int C = g->cells, B = g->a.batch, x = g->a.x_dim, z = g->a.z_dim;
  if (g->bf)
    launch_draw_batch<bf16>((const bf16*)g->pool, g->pool_n, xin_dev, (bf16*)g->E, g->e_cell,
                            (bf16*)g->Z, C, B, x, z, g->seed, (uint32_t)g->t, step, parts, pdl,
                            g->st);
  else
    launch_draw_batch<float>((const float*)g->pool, g->pool_n, xin_dev, (float*)g->E, g->e_cell,
                             (float*)g->Z, C, B, x, z, g->seed, (uint32_t)g->t, step, parts, pdl,
                             g->st);
}

// Step 4 on the evaluation's rows (E: the real minibatch and the five slots' fakes): squared
// row norms, the Gaussian-kernel block sums (tensor-core Gram kernel, or a stored Gram matrix
// on the CUDA-core path), then every cell's ES-(1+1) step on its mixture weights.
int mixture_impl(lipz_grid* g) {
  const int C = g->cells, B = g->a.batch, x = g->a.x_dim, R = 6 * B;
  phase_begin(g, LIPZ_PHASE_MIXTURE);
  if (g->bf)
    launch_row_norms<bf16>((const bf16*)g->E, g->e_cell, C, R, x, g->rnorm, g->st);
  else
    launch_row_norms<float>((const float*)g->E, g->e_cell, C, R, x, g->rnorm, g->st);
  CKL(g);
  if (g->mix_tc) {
    std::string msg;
    if (tc_run_gram(g->tc[g->cur], g->st, &msg)) return fail(g, LIPZ_ERR_CUDA, "%s", msg.c_str());
  } else {
    gemm(g, g->dgram, C, R, R, EPI_STORE, ACT_NONE, true);
    launch_mix_partials(g->gram, g->rnorm, C, R, B, x, g->mixP, g->st);
  }
  CKL(g);
  launch_mix_es(g->mixP, g->mix_nh, C, R, B, g->mix, g->mixS, g->mixScore, g->seed,
                (uint32_t)g->t, g->a.mix_sigma, g->st);
  CKL(g);
  phase_end(g, LIPZ_PHASE_MIXTURE, g->mix_tc ? 3 : 4);
  return LIPZ_OK;
}

// Evaluation (minibatch, forwards, fitness); with `then_select` the selection runs in the
// fitness kernel (the caller reads nothing back in between). With `x_ready`, the caller's
// minibatch xin_dev is still being uploaded: the noise and the generator forward go first,
// the real rows are copied into place after the event.
int eval_impl(lipz_grid* g, const float* xin_dev, bool then_select,
              cudaEvent_t x_ready = nullptr) {
  const int C = g->cells, B = g->a.batch, h = g->a.hidden, x = g->a.x_dim, z = g->a.z_dim;
  if (!xin_dev && g->pool_n <= 0)
    return fail(g, LIPZ_ERR_STATE, "no real-data pool: call lipz_set_data first");
  const int p = g->cur;
  auto draw = [&](int parts, bool pdl) { draw_batch(g, xin_dev, 0, parts, pdl); };
  phase_begin(g, LIPZ_PHASE_BATCH);
  draw(x_ready ? DRAW_NOISE : DRAW_REAL | DRAW_NOISE, true);
  CKL(g);
  phase_end(g, LIPZ_PHASE_BATCH, 1);
  if (g->dcgan) {
    std::string msg;
    phase_begin(g, LIPZ_PHASE_G_FWD);
    // stale neighbours read the other snapshot too; otherwise only snapshot p's individuals
    const bool both = g->a.stale_neighbors && g->prev_valid;
    dc_set_indiv_range(g->dc, both ? 0 : p * C, both ? 0 : C);
    if (dc_eval_g(g->dc, eval_nbr(g), g->st, &msg))
      return fail(g, LIPZ_ERR_CUDA, "%s", msg.c_str());
    phase_end(g, LIPZ_PHASE_G_FWD, dc_eval_launches(g->dc, 0));
    if (x_ready) {
      CK(g, cudaStreamWaitEvent(g->st, x_ready, 0));
      draw(DRAW_REAL, false);
      CKL(g);
    }
    phase_begin(g, LIPZ_PHASE_D_FWD);
    if (dc_eval_d(g->dc, eval_nbr(g), g->st, &msg))
      return fail(g, LIPZ_ERR_CUDA, "%s", msg.c_str());
    phase_end(g, LIPZ_PHASE_D_FWD, dc_eval_launches(g->dc, 1));
  } else if (g->use_tc) {
    std::string msg;
    tc_set_nbr(g->tc[p], eval_nbr(g), eval_pairs(g));
    phase_begin(g, LIPZ_PHASE_G_FWD);
    if (tc_run_g(g->tc[p], g->st, &msg)) return fail(g, LIPZ_ERR_CUDA, "%s", msg.c_str());
    phase_end(g, LIPZ_PHASE_G_FWD, 1);
    if (x_ready) {
      CK(g, cudaStreamWaitEvent(g->st, x_ready, 0));
      draw(DRAW_REAL, false);
      CKL(g);
    }
    phase_begin(g, LIPZ_PHASE_D_FWD);
    if (tc_run_d(g->tc[p], g->st, &msg)) return fail(g, LIPZ_ERR_CUDA, "%s", msg.c_str());
    phase_end(g, LIPZ_PHASE_D_FWD, 1);
  } else {
    const Descs& D = g->a.stale_neighbors && g->prev_valid ? g->dsc_stale[p] : g->dsc[p];
    phase_begin(g, LIPZ_PHASE_G_FWD);
    gemm(g, D.g1, C * 5, B, h, EPI_BIAS_ACT, ACT_RELU, false);
    gemm(g, D.g2, C * 5, B, h, EPI_BIAS_ACT, ACT_RELU, false);
    gemm(g, D.g3, C * 5, B, x, EPI_BIAS_ACT, ACT_TANH, false);
    phase_end(g, LIPZ_PHASE_G_FWD, 3);
    if (x_ready) {
      CK(g, cudaStreamWaitEvent(g->st, x_ready, 0));
      draw(DRAW_REAL, false);
      CKL(g);
    }
    phase_begin(g, LIPZ_PHASE_D_FWD);
    gemm(g, D.d1, C * 5, 6 * B, h, EPI_BIAS_ACT, ACT_LRELU, false);
    gemm(g, D.d2, C * 5, 6 * B, h, EPI_BIAS_ACT, ACT_LRELU, false);
    gemv(g, D.d3, C * 5, 6 * B);
    phase_end(g, LIPZ_PHASE_D_FWD, 3);
  }
  CKL(g);
  phase_begin(g, LIPZ_PHASE_FITNESS);
  if (then_select)
    launch_fitness_select(g->logits, C, B, g->LG, g->LD, g->fG, g->fD, g->flag, eval_nbr(g),
                          select_params(g), select_io(g), g->st);
  else
    launch_fitness(g->logits, C, B, g->LG, g->LD, g->fG, g->fD, g->flag, g->st);
  CKL(g);
  phase_end(g, LIPZ_PHASE_FITNESS, 1);
  if (g->a.mixture) {
    int rc = mixture_impl(g);
    if (rc) return rc;
  }
  g->phase = then_select ? PH_SELECTED : PH_EVALUATED;
  return LIPZ_OK;
}

SelectParams select_params(const lipz_grid* g) {
  SelectParams sp;
  memset(&sp, 0, sizeof sp);
  sp.seed = g->seed;
  sp.t = (uint32_t)g->t;
  sp.tournament_size = g->a.tournament_size;
  sp.replace_always = g->a.replace_mode == LIPZ_REPLACE_ALWAYS;
  sp.lr_mutation = g->a.lr_mutation;
  sp.lr_mut_std = g->a.lr_mut_std;
  double thr = std::floor((double)g->a.lr_mut_prob * 4294967296.0);
  sp.lr_mut_thr = (uint64_t)(thr < 0 ? 0 : (thr > 4294967296.0 ? 4294967296.0 : thr));
  sp.beta1 = g->a.beta1;
  sp.beta2 = g->a.beta2;
  return sp;
}

SelectIO select_io(lipz_grid* g) {
  const int p = g->cur;
  SelectIO io;
  io.lr_old[0] = g->G[0].lr;
  io.lr_old[1] = g->D[0].lr;
  io.step_old[0] = g->G[0].step;
  io.step_old[1] = g->D[0].step;
  io.sel[0] = g->sel_g;
  io.sel[1] = g->sel_d;
  io.src[0] = g->src_g;
  io.src[1] = g->src_d;
  io.lr_new[0] = g->lrn_g;
  io.lr_new[1] = g->lrn_d;
  io.coef[0] = g->coef_g;
  io.coef[1] = g->coef_d;
  return io;
}

int select_impl(lipz_grid* g) {
  if (g->phase != PH_EVALUATED)
    return fail(g, LIPZ_ERR_STATE, "lipz_select_replace must follow lipz_eval_neighborhoods");
  phase_begin(g, LIPZ_PHASE_SELECT);
  launch_select(g->fG, g->fD, eval_nbr(g), g->cells, select_params(g), select_io(g), g->st);
  CKL(g);
  phase_end(g, LIPZ_PHASE_SELECT, 1);
  g->phase = PH_SELECTED;
  return LIPZ_OK;
}

// The Adam ranges left over when the weight matrices take their step inside the backward:
// the biases of both networks and D's output layer, from snapshot p into the next one.
void bias_ranges(lipz_grid* g, int p, AdamRanges* rg, AdamRanges* rd) {
  *rg = AdamRanges{};
  *rd = AdamRanges{};
  rg->old_p = g->G[0];
  rg->new_p = g->G[snap_next(g, p)];
  rg->grad = g->gG;
  rg->src = g->src_g;
  rg->coef = g->coef_g;
  rg->Ps = g->PGs;
  rd->old_p = g->D[0];
  rd->new_p = g->D[snap_next(g, p)];
  rd->grad = g->gD;
  rd->src = g->src_d;
  rd->coef = g->coef_d;
  rd->Ps = g->PDs;
  for (int k : {1, 3, 5}) {
    rg->off[rg->n] = g->lg.off[k];
    rg->len[rg->n++] = (int)(g->lg.off[k + 1] - g->lg.off[k]);
  }
  for (int k : {1, 3, 4, 5}) {
    rd->off[rd->n] = g->ld.off[k];
    rd->len[rd->n++] = (int)(g->ld.off[k + 1] - g->ld.off[k]);
  }
}

// One Adam step of every cell's chosen pair (sel/src/coef) from snapshot cur into the other
// snapshot, which becomes cur.
int train_once(lipz_grid* g) {
  const int C = g->cells, B = g->a.batch, h = g->a.hidden, x = g->a.x_dim, z = g->a.z_dim;
  const int p = g->cur;
  if (g->dcgan) {
    // forward and backward of the selected pairs (gradients into gG, gD), then Adam +
    // replacement into the next snapshot
    std::string msg;
    phase_begin(g, LIPZ_PHASE_TRAIN_BWD);
    // the selected individuals come from the evaluation's neighbour table
    const bool both = g->a.stale_neighbors && g->prev_valid;
    dc_set_indiv_range(g->dc, both ? 0 : p * C, both ? 0 : C);
    if (dc_train(g->dc, g->st, &msg)) return fail(g, LIPZ_ERR_CUDA, "%s", msg.c_str());
    phase_end(g, LIPZ_PHASE_TRAIN_BWD, dc_train_launches(g->dc));
    phase_begin(g, LIPZ_PHASE_ADAM);
    launch_adam(g->G[0], g->G[snap_next(g, p)], g->gG, g->src_g, g->coef_g, C, g->PG, g->PGs,
                g->a.beta1, g->a.beta2, g->a.eps, g->st);
    launch_adam(g->D[0], g->D[snap_next(g, p)], g->gD, g->src_d, g->coef_d, C, g->PD, g->PDs,
                g->a.beta1, g->a.beta2, g->a.eps, g->st);
    CKL(g);
    phase_end(g, LIPZ_PHASE_ADAM, 2);
    g->cur = snap_next(g, p);
    return LIPZ_OK;
  }
  const Descs& D = g->dsc[p];
  phase_begin(g, LIPZ_PHASE_TRAIN_FWD);
  // the CUDA-core kernels read the discriminator's training input as one array TX; the
  // tensor-core kernels read it from E in place
  int n_fwd = 0;
  if (!(g->use_tc && g->use_tcb)) {
    if (g->bf)
      launch_train_prep<bf16>((const bf16*)g->E, g->e_cell, g->sel_g, (bf16*)g->TX, C, B, x,
                              g->st);
    else
      launch_train_prep<float>((const float*)g->E, g->e_cell, g->sel_g, (float*)g->TX, C, B, x,
                               g->st);
    n_fwd = 1;
  }
  // forward of the selected pair
  if (g->use_tc) {
    std::string msg;
    if (tc_run_train_g(g->tc[p], g->st, &msg) || tc_run_train_d(g->tc[p], g->st, &msg))
      return fail(g, LIPZ_ERR_CUDA, "%s", msg.c_str());
    n_fwd += 2;
  } else {
    gemm(g, D.tg1, C, B, h, EPI_BIAS_ACT, ACT_RELU, false);
    gemm(g, D.tg2, C, B, h, EPI_BIAS_ACT, ACT_RELU, false);
    gemm(g, D.td1, C, 2 * B, h, EPI_BIAS_ACT, ACT_LRELU, false);
    gemm(g, D.td2, C, 2 * B, h, EPI_BIAS_ACT, ACT_LRELU, false);
    gemv(g, D.tgv, C, 2 * B);
    n_fwd += 5;
  }
  // logit deltas (and D's output-layer gradient)
  if (g->bf)
    launch_dlogit<bf16>(g->TL, (const bf16*)g->TG2, g->D[0].wb, g->PDs, g->ld.off[4], g->src_d, C,
                        B, h, g->a.leaky_slope, (bf16*)g->J2, g->gD, g->PDs, g->ld.off[4],
                        g->ld.off[5], g->ld.off[3], g->st);
  else
    launch_dlogit<float>(g->TL, (const float*)g->TG2, g->D[0].w, g->PDs, g->ld.off[4], g->src_d,
                         C, B, h, g->a.leaky_slope, (float*)g->J2, g->gD, g->PDs, g->ld.off[4],
                         g->ld.off[5], g->ld.off[3], g->st);
  CKL(g);
  phase_end(g, LIPZ_PHASE_TRAIN_FWD, n_fwd + 1);
  phase_begin(g, LIPZ_PHASE_TRAIN_BWD);
  if (g->use_tcb) {
    // the nine backward products of every cell in one launch (with Adam on the weight
    // matrices unless the gradients are kept; the bias gradients summed in its epilogue)
    std::string msg;
    if (tcb_run_cells(g->tcb[p], g->st, &msg)) return fail(g, LIPZ_ERR_CUDA, "%s", msg.c_str());
    CKL(g);
    phase_end(g, LIPZ_PHASE_TRAIN_BWD, 1);
    phase_begin(g, LIPZ_PHASE_ADAM);
    if (!g->a.keep_grads) {
      // every Adam step (weight matrices, biases, D's output layer) ran inside the backward
      phase_end(g, LIPZ_PHASE_ADAM, 0);
      g->cur = snap_next(g, p);
      return LIPZ_OK;
    }
  } else {
    gemm(g, D.bw2d, C, h, h, EPI_STORE, ACT_NONE, true);
    gemm(g, D.bd1, 2 * C, 2 * B, h, EPI_DACT, ACT_LRELU, false);
    gemm(g, D.bw1d, C, h, x, EPI_STORE, ACT_NONE, true);
    colsum(g, D.cb1d, C, h);
    // generator's backward through D
    gemm(g, D.ba3, C, B, x, EPI_DACT, ACT_TANH, false);
    gemm(g, D.bw3g, C, x, h, EPI_STORE, ACT_NONE, true);
    colsum(g, D.cb3g, C, x);
    gemm(g, D.ba2, C, B, h, EPI_DACT, ACT_RELU, false);
    gemm(g, D.bw2g, C, h, h, EPI_STORE, ACT_NONE, true);
    colsum(g, D.cb2g, C, h);
    gemm(g, D.ba1, C, B, h, EPI_DACT, ACT_RELU, false);
    gemm(g, D.bw1g, C, h, z, EPI_STORE, ACT_NONE, true);
    colsum(g, D.cb1g, C, h);
    CKL(g);
    phase_end(g, LIPZ_PHASE_TRAIN_BWD, 15);
    phase_begin(g, LIPZ_PHASE_ADAM);
  }
  // Adam + replacement into the other snapshot (after the bias sums on the tensor-core path)
  launch_adam(g->G[0], g->G[snap_next(g, p)], g->gG, g->src_g, g->coef_g, C, g->PG, g->PGs, g->a.beta1,
              g->a.beta2, g->a.eps, g->st);
  launch_adam(g->D[0], g->D[snap_next(g, p)], g->gD, g->src_d, g->coef_d, C, g->PD, g->PDs, g->a.beta1,
              g->a.beta2, g->a.eps, g->st);
  CKL(g);
  phase_end(g, LIPZ_PHASE_ADAM, 2);
  g->cur = snap_next(g, p);
  return LIPZ_OK;
}

// Minibatch step k >= 1 of the iteration: a fresh minibatch, every cell's own centre chosen
// again (same lr, next Adam step), the centres' fakes, then one Adam step.
int train_again(lipz_grid* g, uint32_t k) {
  const int C = g->cells, B = g->a.batch, h = g->a.hidden, x = g->a.x_dim;
  phase_begin(g, LIPZ_PHASE_BATCH);
  draw_batch(g, nullptr, k, DRAW_REAL | DRAW_NOISE, true);
  CKL(g);
  phase_end(g, LIPZ_PHASE_BATCH, 1);
  phase_begin(g, LIPZ_PHASE_SELECT);
  launch_centre_select(C, g->cur * C, select_params(g), select_io(g), g->st);
  CKL(g);
  phase_end(g, LIPZ_PHASE_SELECT, 1);
  phase_begin(g, LIPZ_PHASE_G_FWD);
  if (g->use_tc) {
    std::string msg;
    if (tc_run_g_centre(g->tc[g->cur], g->st, &msg))
      return fail(g, LIPZ_ERR_CUDA, "%s", msg.c_str());
    phase_end(g, LIPZ_PHASE_G_FWD, 1);
  } else {
    // the CUDA-core kernels run the generators of all five slots (slot 0 is the one used)
    const Descs& D = g->dsc[g->cur];
    gemm(g, D.g1, C * 5, B, h, EPI_BIAS_ACT, ACT_RELU, false);
    gemm(g, D.g2, C * 5, B, h, EPI_BIAS_ACT, ACT_RELU, false);
    gemm(g, D.g3, C * 5, B, x, EPI_BIAS_ACT, ACT_TANH, false);
    phase_end(g, LIPZ_PHASE_G_FWD, 3);
  }
  CKL(g);
  return train_once(g);
}

int train_impl(lipz_grid* g) {
  if (g->phase != PH_SELECTED)
    return fail(g, LIPZ_ERR_STATE, "lipz_train_step must follow lipz_select_replace");
  const int K = g->a.train_steps;
  if (K > 1 && g->pool_n <= 0)
    return fail(g, LIPZ_ERR_STATE, "train_steps > 1 draws its minibatches from the pool: call "
                                   "lipz_set_data first");
  int rc = train_once(g);
  for (int k = 1; k < K && !rc; ++k) rc = train_again(g, (uint32_t)k);
  if (rc) return rc;
  g->t += 1;
  g->phase = PH_IDLE;
  g->prev_valid = true;
  return LIPZ_OK;
}

// Waits for the grid's stream and reports a bounded wait that expired in a tensor-core kernel
// or a non-finite loss seen since the last check (one synchronisation: all flags are copied
// into pinned host memory first); the flags are reset.
// The device flags of every kernel that can stop early, and the non-finite-loss flag.
void flag_ptrs(lipz_grid* g, int* (&dev)[8]) {
  int* d[8] = {g->tc[0] ? tc_error_flag(g->tc[0]) : nullptr,
               g->tc[1] ? tc_error_flag(g->tc[1]) : nullptr,
               g->tc[2] ? tc_error_flag(g->tc[2]) : nullptr,
               g->tcb[0] ? tcb_error_flag(g->tcb[0]) : nullptr,
               g->tcb[1] ? tcb_error_flag(g->tcb[1]) : nullptr,
               g->tcb[2] ? tcb_error_flag(g->tcb[2]) : nullptr,
               g->dc ? dc_error_flag(g->dc) : nullptr, g->flag};
  for (int i = 0; i < 8; ++i) dev[i] = d[i];
}

// Status from pinned copies st[8] of the device flags (the queued work has completed): a
// raised flag is reset on the device and reported.
int flag_status(lipz_grid* g, int* const (&dev)[8], const int* st) {
  for (int i = 0; i < 7; ++i) {
    const int code = st[i];
    if (code) {
      CK(g, cudaMemsetAsync(dev[i], 0, 4, g->st));
      CK(g, cudaStreamSynchronize(g->st));
      return fail(g, LIPZ_ERR_TIMEOUT, "tensor-core kernel stopped: bounded wait %d expired", code);
    }
  }
  const int v = st[7];
  if (v != INT_MAX) {
    const int big = INT_MAX;
    int rc = h2d(g, g->flag, &big, 4);
    if (rc) return rc;
    return fail(g, LIPZ_ERR_NONFINITE, "non-finite loss in cell %d", v);
  }
  return LIPZ_OK;
}

// Completes a pending lipz_iterate_batch_async call: waits for its iteration and copies its
// fitnesses to the caller (its status is left to the device flags, which stay raised until a
// check reads and resets them).
int deliver_pending(lipz_grid* g) {
  if (!g->a_pending) return LIPZ_OK;
  g->a_pending = false;
  CK(g, cudaEventSynchronize(g->ev_it[g->a_last]));
  const size_t n5 = (size_t)g->cells * 5;
  const float* hp = g->hstat_a + g->a_last * (2 * n5 + 8);
  if (g->a_fit[g->a_last][0]) memcpy(g->a_fit[g->a_last][0], hp, n5 * 4);
  if (g->a_fit[g->a_last][1]) memcpy(g->a_fit[g->a_last][1], hp + n5, n5 * 4);
  return LIPZ_OK;
}

int check_flag(lipz_grid* g) {
  // a pending pipelined call completes first; the flags read here cover its iteration too
  int rc0 = deliver_pending(g);
  if (rc0) return rc0;
  int* dev[8];
  flag_ptrs(g, dev);
  for (int i = 0; i < 8; ++i) {
    g->hstat[i] = i < 7 ? 0 : INT_MAX;
    if (dev[i]) CK(g, cudaMemcpyAsync(&g->hstat[i], dev[i], 4, cudaMemcpyDeviceToHost, g->st));
  }
  CK(g, cudaStreamSynchronize(g->st));
  return flag_status(g, dev, g->hstat);
}

float bf16_bits_to_float(uint16_t b) {
  uint32_t u = (uint32_t)b << 16;
  float f;
  memcpy(&f, &u, 4);
  return f;
}

// Copies `rows` blocks of `n` activation elements (device pitch `pitch` elements) to fp32 host.
int act_to_host(lipz_grid* g, const void* src, int64_t pitch, int64_t rows, int64_t n, float* out) {
  std::vector<char> tmp((size_t)(rows * n * g->esz));
  CK(g, cudaMemcpy2DAsync(tmp.data(), n * g->esz, src, pitch * g->esz, n * g->esz, rows,
                          cudaMemcpyDeviceToHost, g->st));
  CK(g, cudaStreamSynchronize(g->st));
  if (g->bf) {
    const uint16_t* s = (const uint16_t*)tmp.data();
    for (int64_t i = 0; i < rows * n; ++i) out[i] = bf16_bits_to_float(s[i]);
  } else {
    memcpy(out, tmp.data(), (size_t)(rows * n * 4));
  }
  return LIPZ_OK;
}

}  // namespace

// =============================================================================================
// C ABI
// =============================================================================================
extern "C" {

int lipz_arch_default(lipz_arch* a) {
  if (!a) return LIPZ_ERR_INVALID;
  memset(a, 0, sizeof *a);
  a->struct_size = sizeof(lipz_arch);
  a->kind = LIPZ_MLP;
  a->precision = LIPZ_FP32;
  a->z_dim = 64;
  a->hidden = 256;
  a->x_dim = 784;
  a->batch = 100;
  a->lr = 2e-4f;
  a->beta1 = 0.5f;
  a->beta2 = 0.999f;
  a->eps = 1e-8f;
  a->tournament_size = 2;
  a->replace_mode = LIPZ_REPLACE_IF_BETTER;
  a->lr_mutation = 0;
  a->lr_mut_std = 1e-4f;
  a->lr_mut_prob = 0.5f;
  a->leaky_slope = 0.2f;
  a->keep_grads = 0;
  a->force_simt = 0;
  a->train_steps = 1;
  a->mixture = 0;
  a->mix_sigma = 0.01f;
  a->stale_neighbors = 0;
  a->ngf = 64;
  a->ndf = 64;
  return LIPZ_OK;
}

int lipz_grid_create(int rows, int cols, const lipz_arch* arch, uint64_t seed, lipz_grid** out) {
  t_create_err.clear();
  if (!out) return fail(nullptr, LIPZ_ERR_INVALID, "out is null");
  *out = nullptr;
  if (rows < 1 || cols < 1 || (int64_t)rows * cols > (1 << 20))
    return fail(nullptr, LIPZ_ERR_INVALID, "grid needs 1 <= rows, cols and rows*cols <= 2^20");
  int rc = check_arch(arch);
  if (rc) return rc;
  lipz_grid* g = new (std::nothrow) lipz_grid();
  if (!g) return fail(nullptr, LIPZ_ERR_OOM, "host allocation failed");
  g->rows = rows;
  g->cols = cols;
  g->cells = rows * cols;
  g->a = *arch;
  g->seed = seed;
  g->bf = arch->precision == LIPZ_BF16;
  g->esz = g->bf ? 2 : 4;
  rc = create_impl(g);
  if (rc) {
    t_create_err = g->err;
    lipz_grid_destroy(g);
    return rc;
  }
  *out = g;
  return LIPZ_OK;
}

int lipz_grid_destroy(lipz_grid* g) {
  if (!g) return LIPZ_OK;
  cudaStreamSynchronize(g->st);
  if (g->dc) dc_plan_destroy(g->dc);
  for (int p = 0; p < 3; ++p) {
    if (g->tc[p]) tc_plan_destroy(g->tc[p]);
    if (g->tcb[p]) tcb_plan_destroy(g->tcb[p]);
  }
  for (auto& m : g->marks) {
    cudaEventDestroy(m.a);
    cudaEventDestroy(m.b);
  }
  for (auto e : g->ev_free) cudaEventDestroy(e);
  for (auto e : g->open_ev)
    if (e) cudaEventDestroy(e);
  for (void* p : g->allocs) cudaFree(p);
  if (g->own_st) cudaStreamDestroy(g->own_st);
  if (g->copy_st) {
    cudaStreamSynchronize(g->copy_st);
    cudaStreamDestroy(g->copy_st);
  }
  if (g->ev_x) cudaEventDestroy(g->ev_x);
  if (g->ev_x2) cudaEventDestroy(g->ev_x2);
  if (g->hstat) cudaFreeHost(g->hstat);
  if (g->hstat_a) cudaFreeHost(g->hstat_a);
  for (int i = 0; i < 2; ++i) {
    if (g->ev_it[i]) cudaEventDestroy(g->ev_it[i]);
    if (g->ev_buf[i]) cudaEventDestroy(g->ev_buf[i]);
  }
  delete g;
  return LIPZ_OK;
}

int lipz_set_stream(lipz_grid* g, void* stream) {
  if (!g) return LIPZ_ERR_INVALID;
  CK(g, cudaStreamSynchronize(g->st));  // work already queued stays ordered before the switch
  g->st = stream ? (cudaStream_t)stream : g->own_st;
  return LIPZ_OK;
}

int lipz_synchronize(lipz_grid* g) {
  if (!g) return LIPZ_ERR_INVALID;
  CK(g, cudaStreamSynchronize(g->st));
  return check_flag(g);
}

int lipz_set_data(lipz_grid* g, const float* host_pool, int64_t n_rows, int32_t dim) {
  if (!g) return LIPZ_ERR_INVALID;
  if (!host_pool || n_rows < 1 || n_rows > 0xFFFFFFFFll || dim != g->a.x_dim)
    return fail(g, LIPZ_ERR_INVALID, "set_data needs a pool of 1..2^32-1 rows of x_dim=%d",
                g->a.x_dim);
  CK(g, cudaStreamSynchronize(g->st));
  const size_t n = (size_t)n_rows * dim;
  if (n_rows > g->pool_cap) {
    if (g->pool) {
      for (auto& p : g->allocs)
        if (p == g->pool) p = nullptr;
      cudaFree(g->pool);
      g->pool = nullptr;
      g->pool_cap = 0;
    }
    int rc = dalloc(g, &g->pool, n * (g->bf ? 2 : 4));
    if (rc) return rc;
    g->pool_cap = n_rows;
  }
  if (g->bf) {
    // rounded once here: a drawn row is then the same bf16 row the fp32 pool would give
    float* tmp = nullptr;
    CK(g, cudaMalloc(&tmp, n * 4));
    cudaError_t e = cudaMemcpyAsync(tmp, host_pool, n * 4, cudaMemcpyHostToDevice, g->st);
    if (e == cudaSuccess) {
      launch_to_bf16(tmp, (bf16*)g->pool, (int64_t)n, g->st);
      e = cudaGetLastError();
    }
    if (e == cudaSuccess) e = cudaStreamSynchronize(g->st);
    cudaFree(tmp);
    CK(g, e);
  } else {
    int rc = h2d(g, g->pool, host_pool, n * 4);
    if (rc) return rc;
  }
  g->pool_n = n_rows;
  return LIPZ_OK;
}

int lipz_eval_neighborhoods(lipz_grid* g, float* fit_g, float* fit_d, float* pair_lg,
                            float* pair_ld) {
  if (!g) return LIPZ_ERR_INVALID;
  int rc = eval_impl(g, nullptr, false);
  if (rc) return rc;
  if (fit_g || fit_d || pair_lg || pair_ld) {
    const size_t C = g->cells;
    if (fit_g) CK(g, cudaMemcpyAsync(fit_g, g->fG, C * 20, cudaMemcpyDeviceToHost, g->st));
    if (fit_d) CK(g, cudaMemcpyAsync(fit_d, g->fD, C * 20, cudaMemcpyDeviceToHost, g->st));
    if (pair_lg) CK(g, cudaMemcpyAsync(pair_lg, g->LG, C * 100, cudaMemcpyDeviceToHost, g->st));
    if (pair_ld) CK(g, cudaMemcpyAsync(pair_ld, g->LD, C * 100, cudaMemcpyDeviceToHost, g->st));
    CK(g, cudaStreamSynchronize(g->st));
    return check_flag(g);
  }
  return LIPZ_OK;
}

int lipz_select_replace(lipz_grid* g, int32_t* sel_g, int32_t* sel_d) {
  if (!g) return LIPZ_ERR_INVALID;
  int rc = select_impl(g);
  if (rc) return rc;
  if (sel_g || sel_d) {
    if (sel_g) CK(g, cudaMemcpyAsync(sel_g, g->sel_g, g->cells * 4, cudaMemcpyDeviceToHost, g->st));
    if (sel_d) CK(g, cudaMemcpyAsync(sel_d, g->sel_d, g->cells * 4, cudaMemcpyDeviceToHost, g->st));
    CK(g, cudaStreamSynchronize(g->st));
  }
  return LIPZ_OK;
}

int lipz_train_step(lipz_grid* g) {
  if (!g) return LIPZ_ERR_INVALID;
  return train_impl(g);
}

int lipz_iterate(lipz_grid* g, int n_iters) {
  if (!g) return LIPZ_ERR_INVALID;
  if (n_iters < 0) return fail(g, LIPZ_ERR_INVALID, "n_iters < 0");
  for (int i = 0; i < n_iters; ++i) {
    int rc;
    if ((rc = eval_impl(g, nullptr, true)) || (rc = train_impl(g))) return rc;
  }
  return LIPZ_OK;
}

int lipz_iterate_batch(lipz_grid* g, const float* x_host, float* fit_g, float* fit_d) {
  if (!g) return LIPZ_ERR_INVALID;
  if (!x_host) return fail(g, LIPZ_ERR_INVALID, "x_host is null");
  // a pipelined call's iteration may still read a staging buffer
  int rc0 = deliver_pending(g);
  if (rc0) return rc0;
  const size_t bytes = (size_t)g->cells * g->a.batch * g->a.x_dim * 4;
  g->pre_buf = -1;  // (a minibatch uploaded ahead into the same buffer is superseded)
  g->pre_host = nullptr;
  // the upload runs on the copy stream while the noise and the generator forward compute
  CK(g, cudaMemcpyAsync(g->xin, x_host, bytes, cudaMemcpyHostToDevice, g->copy_st));
  CK(g, cudaEventRecord(g->ev_x, g->copy_st));
  int rc;
  if ((rc = eval_impl(g, g->xin, true, g->ev_x)) || (rc = train_impl(g))) return rc;
  const size_t C = g->cells;
  if (fit_g) CK(g, cudaMemcpyAsync(fit_g, g->fG, C * 20, cudaMemcpyDeviceToHost, g->st));
  if (fit_d) CK(g, cudaMemcpyAsync(fit_d, g->fD, C * 20, cudaMemcpyDeviceToHost, g->st));
  return check_flag(g);  // one stream synchronisation for the results and the flags
}

int lipz_iterate_batch_next(lipz_grid* g, const float* x_host, const float* x_next,
                            float* fit_g, float* fit_d) {
  if (!g) return LIPZ_ERR_INVALID;
  if (!x_host) return fail(g, LIPZ_ERR_INVALID, "x_host is null");
  int rc0 = deliver_pending(g);
  if (rc0) return rc0;
  const size_t bytes = (size_t)g->cells * g->a.batch * g->a.x_dim * 4;
  if (!g->xin2) {
    int rc;
    if ((rc = dalloc(g, &g->xin2, bytes))) return rc;
    CK(g, cudaEventCreateWithFlags(&g->ev_x2, cudaEventDisableTiming));
  }
  float* const buf[2] = {g->xin, g->xin2};
  const cudaEvent_t ev[2] = {g->ev_x, g->ev_x2};
  // this iteration's minibatch: uploaded during the previous call, or now
  int cur;
  if (g->pre_buf >= 0 && g->pre_host == x_host) {
    cur = g->pre_buf;
  } else {
    cur = g->pre_buf >= 0 ? 1 - g->pre_buf : 0;
    CK(g, cudaMemcpyAsync(buf[cur], x_host, bytes, cudaMemcpyHostToDevice, g->copy_st));
    CK(g, cudaEventRecord(ev[cur], g->copy_st));
  }
  g->pre_buf = -1;
  g->pre_host = nullptr;
  // the next one into the other buffer, behind it on the copy stream, while this iteration
  // computes (the other buffer's last reader, the previous iteration, has finished: every call
  // returns after its iteration is complete)
  if (x_next) {
    const int nb = 1 - cur;
    CK(g, cudaMemcpyAsync(buf[nb], x_next, bytes, cudaMemcpyHostToDevice, g->copy_st));
    CK(g, cudaEventRecord(ev[nb], g->copy_st));
    g->pre_buf = nb;
    g->pre_host = x_next;
  }
  int rc;
  if ((rc = eval_impl(g, buf[cur], true, ev[cur])) || (rc = train_impl(g))) {
    g->pre_buf = -1;
    g->pre_host = nullptr;
    return rc;
  }
  const size_t C = g->cells;
  if (fit_g) CK(g, cudaMemcpyAsync(fit_g, g->fG, C * 20, cudaMemcpyDeviceToHost, g->st));
  if (fit_d) CK(g, cudaMemcpyAsync(fit_d, g->fD, C * 20, cudaMemcpyDeviceToHost, g->st));
  return check_flag(g);
}

int lipz_iterate_batch_async(lipz_grid* g, const float* x_host, const float* x_next,
                             float* fit_g, float* fit_d) {
  if (!g) return LIPZ_ERR_INVALID;
  if (!x_host) return fail(g, LIPZ_ERR_INVALID, "x_host is null");
  const size_t bytes = (size_t)g->cells * g->a.batch * g->a.x_dim * 4;
  if (!g->xin2) {
    int rc;
    if ((rc = dalloc(g, &g->xin2, bytes))) return rc;
    CK(g, cudaEventCreateWithFlags(&g->ev_x2, cudaEventDisableTiming));
  }
  const size_t C = g->cells, n5 = C * 5, stage_words = 2 * n5 + 8;
  if (!g->hstat_a) {
    int rc0;
    if ((rc0 = dalloc(g, &g->astage, stage_words * 4))) return rc0;
    CK(g, cudaMallocHost(&g->hstat_a, 2 * stage_words * 4));
    for (int i = 0; i < 2; ++i) {
      CK(g, cudaEventCreateWithFlags(&g->ev_it[i], cudaEventDisableTiming));
      CK(g, cudaEventCreateWithFlags(&g->ev_buf[i], cudaEventDisableTiming));
    }
  }
  float* const buf[2] = {g->xin, g->xin2};
  const cudaEvent_t ev[2] = {g->ev_x, g->ev_x2};
  // an upload into a staging buffer waits for the last iteration that read it (which may
  // still be running: this call does not wait for the previous one before enqueueing)
  auto upload = [&](int b, const float* src) -> int {
    if (g->buf_read[b]) CK(g, cudaStreamWaitEvent(g->copy_st, g->ev_buf[b], 0));
    CK(g, cudaMemcpyAsync(buf[b], src, bytes, cudaMemcpyHostToDevice, g->copy_st));
    CK(g, cudaEventRecord(ev[b], g->copy_st));
    return LIPZ_OK;
  };
  int rc, cur;
  if (g->pre_buf >= 0 && g->pre_host == x_host) {
    cur = g->pre_buf;
  } else {
    cur = g->pre_buf >= 0 ? 1 - g->pre_buf : 0;
    if ((rc = upload(cur, x_host))) return rc;
  }
  g->pre_buf = -1;
  g->pre_host = nullptr;
  if (x_next) {
    if ((rc = upload(1 - cur, x_next))) return rc;
    g->pre_buf = 1 - cur;
    g->pre_host = x_next;
  }
  if ((rc = eval_impl(g, buf[cur], true, ev[cur])) || (rc = train_impl(g))) {
    g->pre_buf = -1;
    g->pre_host = nullptr;
    return rc;
  }
  // this iteration's fitnesses and status words, gathered and copied into this call's slot
  const int slot = 1 - g->a_last;
  int* dev[8];
  flag_ptrs(g, dev);
  StatusFlags fl;
  for (int i = 0; i < 8; ++i) fl.p[i] = dev[i];
  launch_gather_status(g->fG, g->fD, (int)n5, fl, g->astage, true, g->st);
  CKL(g);
  float* hs = g->hstat_a + slot * stage_words;
  CK(g, cudaMemcpyAsync(hs, g->astage, stage_words * 4, cudaMemcpyDeviceToHost, g->st));
  g->a_fit[slot][0] = fit_g;
  g->a_fit[slot][1] = fit_d;
  CK(g, cudaEventRecord(g->ev_it[slot], g->st));
  // the staging buffer is free once the iteration and its small copies are done (an upload
  // started earlier would hold up those copies, and the next iteration behind them)
  CK(g, cudaEventRecord(g->ev_buf[cur], g->st));
  g->buf_read[cur] = true;
  const bool had = g->a_pending;
  const int prev = g->a_last;
  g->a_last = slot;
  g->a_pending = true;
  if (!had) return LIPZ_OK;
  // the previous call's iteration (and its copy) has completed once this returns
  CK(g, cudaEventSynchronize(g->ev_it[prev]));
  const float* hp = g->hstat_a + prev * stage_words;
  if (g->a_fit[prev][0]) memcpy(g->a_fit[prev][0], hp, n5 * 4);
  if (g->a_fit[prev][1]) memcpy(g->a_fit[prev][1], hp + n5, n5 * 4);
  rc = flag_status(g, dev, reinterpret_cast<const int*>(hp + 2 * n5));
  if (rc) {
    // the flags are sticky until reset: drain this call too, whose copies may repeat the
    // report, and leave nothing pending
    CK(g, cudaStreamSynchronize(g->st));
    g->a_pending = false;
  }
  return rc;
}

int lipz_state_bytes(const lipz_grid* g, size_t* bytes) {
  if (!g || !bytes) return LIPZ_ERR_INVALID;
  const size_t C = g->cells;
  *bytes = 64 + C * (size_t)(g->PG + g->PD) * 3 * 4 + C * 16 + C * 20;
  return LIPZ_OK;
}

int lipz_export_state(lipz_grid* g, void* host, size_t bytes) {
  if (!g) return LIPZ_ERR_INVALID;
  size_t need = 0;
  lipz_state_bytes(g, &need);
  if (!host || bytes != need)
    return fail(g, LIPZ_ERR_INVALID, "export_state needs a %zu-byte buffer", need);
  char* o = (char*)host;
  uint32_t hdr[10] = {0x5A50494Cu, 2u, (uint32_t)g->rows, (uint32_t)g->cols,
                      (uint32_t)g->a.z_dim, (uint32_t)g->a.hidden, (uint32_t)g->a.x_dim,
                      (uint32_t)g->a.batch, (uint32_t)g->a.precision, 0u};
  memset(o, 0, 64);
  memcpy(o, hdr, 40);
  memcpy(o + 40, &g->t, 8);
  memcpy(o + 48, &g->seed, 8);
  o += 64;
  CK(g, cudaStreamSynchronize(g->st));
  const int p = g->cur;
  const size_t C = g->cells;
  auto put = [&](const float* src, int64_t P, int64_t Ps) -> int {
    CK(g, cudaMemcpy2DAsync(o, P * 4, src, Ps * 4, P * 4, C, cudaMemcpyDeviceToHost, g->st));
    o += C * P * 4;
    return LIPZ_OK;
  };
  int rc;
  if ((rc = put(g->G[p].w, g->PG, g->PGs)) || (rc = put(g->G[p].m, g->PG, g->PGs)) ||
      (rc = put(g->G[p].v, g->PG, g->PGs)) || (rc = put(g->D[p].w, g->PD, g->PDs)) ||
      (rc = put(g->D[p].m, g->PD, g->PDs)) || (rc = put(g->D[p].v, g->PD, g->PDs)))
    return rc;
  CK(g, cudaMemcpyAsync(o, g->G[p].step, C * 4, cudaMemcpyDeviceToHost, g->st));
  o += C * 4;
  CK(g, cudaMemcpyAsync(o, g->D[p].step, C * 4, cudaMemcpyDeviceToHost, g->st));
  o += C * 4;
  CK(g, cudaMemcpyAsync(o, g->G[p].lr, C * 4, cudaMemcpyDeviceToHost, g->st));
  o += C * 4;
  CK(g, cudaMemcpyAsync(o, g->D[p].lr, C * 4, cudaMemcpyDeviceToHost, g->st));
  o += C * 4;
  CK(g, cudaMemcpyAsync(o, g->mix, C * 20, cudaMemcpyDeviceToHost, g->st));
  CK(g, cudaStreamSynchronize(g->st));
  return LIPZ_OK;
}

int lipz_import_state(lipz_grid* g, const void* host, size_t bytes) {
  if (!g) return LIPZ_ERR_INVALID;
  size_t need = 0;
  lipz_state_bytes(g, &need);
  if (!host || bytes != need) return fail(g, LIPZ_ERR_INVALID, "import_state needs %zu bytes", need);
  const char* s = (const char*)host;
  uint32_t hdr[10];
  memcpy(hdr, s, 40);
  if (hdr[0] != 0x5A50494Cu || hdr[1] != 2u)
    return fail(g, LIPZ_ERR_INVALID, "not a version-2 grid state");
  if ((int)hdr[2] != g->rows || (int)hdr[3] != g->cols || (int)hdr[4] != g->a.z_dim ||
      (int)hdr[5] != g->a.hidden || (int)hdr[6] != g->a.x_dim || (int)hdr[7] != g->a.batch)
    return fail(g, LIPZ_ERR_INVALID, "state shape does not match this grid");
  CK(g, cudaStreamSynchronize(g->st));
  int64_t t;
  uint64_t seed;
  memcpy(&t, s + 40, 8);
  memcpy(&seed, s + 48, 8);
  s += 64;
  const int p = g->cur;
  const size_t C = g->cells;
  auto get = [&](float* dst, int64_t P, int64_t Ps) -> int {
    CK(g, cudaMemcpy2DAsync(dst, Ps * 4, s, P * 4, P * 4, C, cudaMemcpyHostToDevice, g->st));
    s += C * P * 4;
    return LIPZ_OK;
  };
  int rc;
  if ((rc = get(g->G[p].w, g->PG, g->PGs)) || (rc = get(g->G[p].m, g->PG, g->PGs)) ||
      (rc = get(g->G[p].v, g->PG, g->PGs)) || (rc = get(g->D[p].w, g->PD, g->PDs)) ||
      (rc = get(g->D[p].m, g->PD, g->PDs)) || (rc = get(g->D[p].v, g->PD, g->PDs)))
    return rc;
  CK(g, cudaMemcpyAsync(g->G[p].step, s, C * 4, cudaMemcpyHostToDevice, g->st));
  s += C * 4;
  CK(g, cudaMemcpyAsync(g->D[p].step, s, C * 4, cudaMemcpyHostToDevice, g->st));
  s += C * 4;
  CK(g, cudaMemcpyAsync(g->G[p].lr, s, C * 4, cudaMemcpyHostToDevice, g->st));
  s += C * 4;
  CK(g, cudaMemcpyAsync(g->D[p].lr, s, C * 4, cudaMemcpyHostToDevice, g->st));
  s += C * 4;
  CK(g, cudaMemcpyAsync(g->mix, s, C * 20, cudaMemcpyHostToDevice, g->st));
  g->prev_valid = false;  // the other snapshot no longer holds this state's predecessor
  if (g->bf) {
    launch_to_bf16(g->G[p].w, g->G[p].wb, (int64_t)C * g->PGs, g->st);
    launch_to_bf16(g->D[p].w, g->D[p].wb, (int64_t)C * g->PDs, g->st);
    CKL(g);
  }
  CK(g, cudaStreamSynchronize(g->st));
  g->t = t;
  g->seed = seed;
  g->phase = PH_IDLE;
  return LIPZ_OK;
}

int lipz_get_iteration(const lipz_grid* g, int64_t* t) {
  if (!g || !t) return LIPZ_ERR_INVALID;
  *t = g->t;
  return LIPZ_OK;
}

int lipz_get_batch(lipz_grid* g, float* x, float* z) {
  if (!g) return LIPZ_ERR_INVALID;
  if (g->phase == PH_IDLE) return fail(g, LIPZ_ERR_STATE, "no evaluation since the last train step");
  const int64_t B = g->a.batch;
  int rc;
  if (x && (rc = act_to_host(g, g->E, g->e_cell, g->cells, B * g->a.x_dim, x))) return rc;
  if (z && (rc = act_to_host(g, g->Z, B * g->a.z_dim, g->cells, B * g->a.z_dim, z))) return rc;
  return LIPZ_OK;
}

int lipz_get_mixture(lipz_grid* g, float* weights, float* blocks, float* score) {
  if (!g) return LIPZ_ERR_INVALID;
  if ((blocks || score) && !g->a.mixture)
    return fail(g, LIPZ_ERR_STATE, "grid was created without mixture");
  const size_t C = g->cells;
  if (weights) CK(g, cudaMemcpyAsync(weights, g->mix, C * 20, cudaMemcpyDeviceToHost, g->st));
  if (blocks) CK(g, cudaMemcpyAsync(blocks, g->mixS, C * 144, cudaMemcpyDeviceToHost, g->st));
  if (score) CK(g, cudaMemcpyAsync(score, g->mixScore, C * 4, cudaMemcpyDeviceToHost, g->st));
  CK(g, cudaStreamSynchronize(g->st));
  return LIPZ_OK;
}

int lipz_get_logits(lipz_grid* g, float* logits) {
  if (!g || !logits) return LIPZ_ERR_INVALID;
  if (g->phase == PH_IDLE) return fail(g, LIPZ_ERR_STATE, "no evaluation since the last train step");
  CK(g, cudaMemcpyAsync(logits, g->logits, (size_t)g->cells * 30 * g->a.batch * 4,
                        cudaMemcpyDeviceToHost, g->st));
  CK(g, cudaStreamSynchronize(g->st));
  return LIPZ_OK;
}

int lipz_get_gradients(lipz_grid* g, float* grad_g, float* grad_d) {
  if (!g) return LIPZ_ERR_INVALID;
  if (!g->a.keep_grads) return fail(g, LIPZ_ERR_STATE, "grid was created without keep_grads");
  CK(g, cudaStreamSynchronize(g->st));
  const size_t C = g->cells;
  if (grad_g)
    CK(g, cudaMemcpy2D(grad_g, g->PG * 4, g->gG, g->PGs * 4, g->PG * 4, C, cudaMemcpyDeviceToHost));
  if (grad_d)
    CK(g, cudaMemcpy2D(grad_d, g->PD * 4, g->gD, g->PDs * 4, g->PD * 4, C, cudaMemcpyDeviceToHost));
  return LIPZ_OK;
}

int lipz_profile_enable(lipz_grid* g, int enable) {
  if (!g) return LIPZ_ERR_INVALID;
  g->prof = enable != 0;
  return LIPZ_OK;
}

int lipz_profile_read(lipz_grid* g, double* ms, int64_t* count, int64_t* launches, int n) {
  if (!g) return LIPZ_ERR_INVALID;
  if (n < 0 || n > LIPZ_N_PHASES) return fail(g, LIPZ_ERR_INVALID, "n must be in 0..%d", LIPZ_N_PHASES);
  CK(g, cudaStreamSynchronize(g->st));
  double acc[LIPZ_N_PHASES] = {0};
  for (auto& m : g->marks) {
    float t = 0.f;
    CK(g, cudaEventElapsedTime(&t, m.a, m.b));
    acc[m.phase] += t;
    g->ev_free.push_back(m.a);
    g->ev_free.push_back(m.b);
  }
  g->marks.clear();
  for (int i = 0; i < n; ++i) {
    if (ms) ms[i] = acc[i];
    if (count) count[i] = g->counts[i];
    if (launches) launches[i] = g->launches[i];
  }
  for (int i = 0; i < LIPZ_N_PHASES; ++i) g->counts[i] = g->launches[i] = 0;
  return LIPZ_OK;
}

const char* lipz_last_error(const lipz_grid* g) {
  return g ? g->err.c_str() : t_create_err.c_str();
}

const char* lipz_status_string(int status) {
  switch (status) {
    case LIPZ_OK: return "ok";
    case LIPZ_ERR_INVALID: return "invalid argument";
    case LIPZ_ERR_CUDA: return "CUDA error";
    case LIPZ_ERR_OOM: return "out of memory";
    case LIPZ_ERR_NONFINITE: return "non-finite loss";
    case LIPZ_ERR_TIMEOUT: return "device wait timed out";
    case LIPZ_ERR_STATE: return "call out of order";
    default: return "unknown status";
  }
}

}  // extern "C"
