// DCGAN evaluation and training steps of the grid on the CUDA-core kernels (conv_kernels.cu).
// Every layer of every problem of a phase is one grouped launch: the evaluation's problems are
// the (cell, slot) pairs, the training's the cells. Weights are read in place from the
// population (individual index from the neighbour table or the selection), activations are
// NCHW per sample.
#include "dcgan.h"

#include <cuda_bf16.h>

#include "conv_tc.h"

#include <algorithm>
#include <cstdlib>
#include <cstring>
#include <vector>

namespace lipz {

namespace {

int ilog2(int v) {
  int l = 0;
  while ((1 << l) < v) ++l;
  return l;
}

}  // namespace

void dc_layouts(int z, int ngf, int ndf, Layout* lg, Layout* ld) {
  const int64_t g = ngf, d = ndf;
  const int64_t gch[5] = {z, 8 * g, 4 * g, 2 * g, g};
  Layout L{};
  int t = 0;
  int64_t off = 0;
  auto add = [&](int64_t n, int init, float bound) {
    L.off[t] = off;
    L.init[t] = init;
    L.bound[t] = bound;
    off += n;
    ++t;
  };
  for (int i = 0; i < 4; ++i) {
    add(gch[i] * gch[i + 1] * 16, INIT_NORMAL, 0.02f);
    add(gch[i + 1], INIT_ONE_NORMAL, 0.02f);
    add(gch[i + 1], INIT_UNIFORM, 0.f);
  }
  add(g * 3 * 16, INIT_NORMAL, 0.02f);
  L.n = t;
  L.off[t] = off;
  *lg = L;
  Layout M{};
  const int64_t dch[5] = {3, d, 2 * d, 4 * d, 8 * d};
  L = M;
  t = 0;
  off = 0;
  for (int i = 0; i < 4; ++i) add(dch[i + 1] * dch[i] * 16, INIT_NORMAL, 0.02f);
  add(8 * d * 16, INIT_NORMAL, 0.02f);
  L.n = t;
  L.off[t] = off;
  *ld = L;
}

struct DcPlan {
  DcShape s;
  DcBuffers b;
  std::vector<void*> allocs;
  // evaluation: generator layers (problems cells * 5), discriminator layers (5 problems per
  // cell, launched cell by cell)
  ConvDesc* eg[5];
  BnDesc* ebn[4];
  ConvDesc* ed[4];
  LogitDesc* edl;
  // training (problems = cells)
  ConvDesc* tg[5];
  BnDesc* tbn[4];
  ConvDesc* td[4];
  LogitDesc* tdl;
  LogitDesc* tdl_back_d;  // D loss, 2B rows, with the output layer's gradient
  LogitDesc* tdl_back_g;  // G loss, fake rows
  ConvDesc* dw[4];        // discriminator weight gradients W4, W3, W2, W1
  ConvDesc* dd[3];        // D-loss deltas into layers 3, 2, 1
  ConvDesc* gd[4];        // G-loss deltas into layers 3, 2, 1 and the fakes
  ConvDesc* gw[5];        // generator weight gradients W5, W4, W3, W2, W1
  ConvDesc* gdh[4];       // generator deltas dh4, dh3, dh2, dh1
  BnDesc* gbn[4];         // batch-norm backward of layers 4, 3, 2, 1
  void* TX;               // [cells][2B][12288] discriminator training input (real, fakes)
  float* tlogits;         // [cells][2B]
  void *dl_d, *dl_g;
  float* part;
  int64_t part_floats;
  int splits_dw[4], splits_gw[5];
  int64_t pstride_dw[4], pstride_gw[5];
  int eval_launches, train_launches;
  // tensor-core discriminator evaluation (bf16, ndf a multiple of 64): weights re-laid out as
  // [out][ky][kx][in] for every individual, a TMA map per layer, channel-last activations
  bool tc = false;
  bf16* Dwt = nullptr;
  CUtensorMap mW[4];
  CtcParams cp[4];
  ConvTcDesc* tcd[4];
  RelayoutD rel;
  int* err = nullptr;
  int sms = 148;
  // tensor-core generator evaluation (bf16, ngf a multiple of 64): layers 2-5 by parity class
  // from class-major weight copies, channel-last activations and batch norm
  bool tcg = false, tct = false;
  float* bnpart = nullptr;
  unsigned* bncnt = nullptr;
  CtcParams tgp[4], tdp[4];
  ConvTcDesc *tgd[4], *tdd[4];
  // tensor-core input gradients: the discriminator's as parity-class transposed convolutions
  // (class-major copies of its weights), the generator's as convolutions ((tap, channel)
  // copies of its transposed-convolution weights)
  bf16 *Ddt = nullptr, *Gct = nullptr;
  int64_t ddt_ps = 0, gct_ps = 0;
  RelayoutG reld;
  RelayoutC relc;
  CUtensorMap mDd[4], mGc[4];
  CtcParams ddp[3], gdp[4], gcp[4];
  ConvTcDesc *ddd[3], *gdd[4], *gcd[4];
  LogitDesc *tdl_tc, *tdl_back_d_tc, *tdl_back_g_tc;
  bf16* Gwt = nullptr;
  int64_t gwt_ps = 0;
  // the generator's first layer on tcgen05: a (tap, o) copy of its weights inside Gwt
  bool g1tc = false;
  int64_t g1_off = 0;
  CUtensorMap mG1;
  // the generator's first-layer weight gradient on tcgen05: a (o, tap) copy of its deltas
  bool g1w = false;
  bf16* dc1t = nullptr;
  void* dcb = nullptr;  // the generator's batch-norm-backward deltas, [cells][B][gmax]
  int64_t dcb_cell = 0;
  CUtensorMap mG1w;
  // individuals whose weight copies the next calls need (dc_set_indiv_range): [rl_lo,
  // rl_lo + rl_n), all when rl_n <= 0
  int rl_lo = 0, rl_n = 0;
  // batch-norm statistics of generator layers 2-4 summed in their convolutions' epilogues
  float2* bnp = nullptr;
  int bn_slots_e[3] = {0, 0, 0}, bn_slots_t[3] = {0, 0, 0};
  RelayoutG relg;
  CUtensorMap mG[4];
  CtcParams gp[4];
  ConvTcDesc* gtd[4];
  // activation maps of the channel-last tensor-core launches (A rows by TMA): evaluation D
  // and G, training forwards, D-loss and G-loss input gradients, generator input gradients
  CUtensorMap aEd[4], aEg[4], aTg[4], aTd[4], aDd[3], aGd[4], aGc[4];
  // scatter mode (one GEMM over input pixels, see conv_tc.h) for the 64 -> 3 transposed
  // convolutions: the generator's output layer (evaluation egs, training tgs) and the
  // G-loss input gradient of discriminator layer 1 (gds)
  bool scg = false, scd = false;
  bf16 *Gs = nullptr, *Ds = nullptr;
  CUtensorMap mGs, mDs, aEgs, aTgs, aGds;
  CtcParams egs, tgs, gds;
  float* halo = nullptr;
  std::vector<ConvTcDesc> h_gtd5, h_tgd5, h_gdd1;
  // tensor-core weight gradients of the layers whose channel counts fill the tiles
  bool wtc_d[4] = {}, wtc_g[5] = {};
  WgtcParams wdp[4], wgp[5];
  WgtcDesc *wdd[4] = {}, *wgd[5] = {};
  CUtensorMap wdA[4], wdB[4], wgA[5], wgB[5];
  float* wpart = nullptr;
};

namespace {

template <typename T>
int dev_alloc(DcPlan* p, T** out, size_t bytes, std::string* msg) {
  void* q = nullptr;
  if (cudaMalloc(&q, bytes ? bytes : 16) != cudaSuccess) {
    cudaGetLastError();
    if (msg) *msg = "cudaMalloc of " + std::to_string(bytes) + " bytes failed";
    return 1;
  }
  p->allocs.push_back(q);
  *out = (T*)q;
  return 0;
}

template <typename T>
int upload(DcPlan* p, T** out, const std::vector<T>& v, std::string* msg) {
  if (dev_alloc(p, out, v.size() * sizeof(T), msg)) return 1;
  if (cudaMemcpy(*out, v.data(), v.size() * sizeof(T), cudaMemcpyHostToDevice) != cudaSuccess) {
    cudaGetLastError();
    if (msg) *msg = "descriptor upload failed";
    return 1;
  }
  return 0;
}

ConvDesc cdesc(const void* a, int n, int ca, int ha, const void* b, int co, int ho, int s,
               int pad, void* out) {
  ConvDesc d;
  memset(&d, 0, sizeof d);
  d.a = a;
  d.b = b;
  d.out = out;
  d.n = n;
  d.ca = ca;
  d.lha = d.lwa = ilog2(ha);
  d.co = co;
  d.lho = d.lwo = ilog2(ho);
  d.s = s;
  d.p = pad;
  return d;
}

// WGRAD splits: chunks of about 4096 of the K = n * Ha * Wa reduction
int wgrad_splits(const ConvDesc& d) {
  const int64_t K = (int64_t)d.n << (d.lha + d.lwa);
  return (int)std::max<int64_t>(1, std::min<int64_t>(64, K / 4096));
}

}  // namespace

DcPlan* dc_plan_create(const DcShape& s, const DcBuffers& b, std::string* msg) {
  DcPlan* p = new DcPlan();
  p->s = s;
  p->b = b;
  const int C = s.cells, B = s.B, g = s.ngf, d = s.ndf, z = s.z;
  const size_t es = s.bf ? 2 : 4;
  const int64_t X = 3 * 64 * 64;
  auto el = [es](const void* base, int64_t i) { return (const char*)base + i * (int64_t)es; };
  auto elw = [es](void* base, int64_t i) { return (char*)base + i * (int64_t)es; };
  // generator channels and sizes per layer (input of layer l: gc[l] x gs[l]^2)
  const int gc[6] = {z, 8 * g, 4 * g, 2 * g, g, 3};
  const int gs[6] = {1, 4, 8, 16, 32, 64};
  const int dc[6] = {3, d, 2 * d, 4 * d, 8 * d, 1};
  const int ds[6] = {64, 32, 16, 8, 4, 1};
  int64_t gsz[5], dsz[5];  // per-sample sizes of the generator outputs 1..4 / disc. outputs 1..4
  for (int l = 1; l <= 4; ++l) {
    gsz[l] = (int64_t)gc[l] * gs[l] * gs[l];
    dsz[l] = (int64_t)dc[l] * ds[l] * ds[l];
  }
  const int64_t gmax = gsz[4] > gsz[3] ? gsz[4] : gsz[3], dmax = dsz[1];
  int64_t gall = 0, dall = 0;
  for (int l = 1; l <= 4; ++l) {
    gall += gsz[l];
    dall += dsz[l];
  }
  int64_t goffs[5] = {0}, doffs[5] = {0};  // per-sample offsets of stored layers
  for (int l = 2; l <= 4; ++l) {
    goffs[l] = goffs[l - 1] + gsz[l - 1];
    doffs[l] = doffs[l - 1] + dsz[l - 1];
  }
  const int PE = C * 5;
  p->tcg = s.bf && g % 64 == 0;
  const bool tcd = s.bf && d % 64 == 0 && 8 * d <= 512;
  // tensor-core training forward (both networks' widths multiples of 64): channel-last
  // activations, read by the CUDA-core backward kernels in that layout
  const bool tct = tcd && p->tcg;
  // LIPZ_CONV_GATHER=1: the gather warps load every A tile and the activation maps stay
  // unused (the tests check that both ways of loading A give bit-identical results)
  const char* gather_env = getenv("LIPZ_CONV_GATHER");
  const bool gather_a = gather_env && gather_env[0] == '1';
  auto act_map = [&](CUtensorMap* m, CtcParams* q, const ConvTcDesc* descs, int n) {
    return ctc_make_act_map(m, q, descs, n, msg, !gather_a);
  };
  p->tct = tct;
  // ---- buffers
  float *ec, *emean, *einv, *tc, *tmean, *tinv, *dh;
  void *eh, *ex, *ey, *th, *ta, *P, *Q, *P2, *Q2, *dcb, *d5;
  int64_t stats = 15 * (int64_t)g;  // channels of the four batch-normalised layers
  if (dev_alloc(p, &ec, (size_t)PE * B * gmax * 4, msg) ||
      dev_alloc(p, &eh, (size_t)PE * B * gmax * es, msg) ||
      dev_alloc(p, &emean, (size_t)PE * stats * 4, msg) ||
      dev_alloc(p, &einv, (size_t)PE * stats * 4, msg) ||
      dev_alloc(p, &ex, (size_t)5 * 6 * B * dmax * es, msg) ||
      dev_alloc(p, &ey, (size_t)5 * 6 * B * dsz[2] * es, msg) ||
      dev_alloc(p, &tc, (size_t)C * B * gall * 4, msg) ||
      dev_alloc(p, &th, (size_t)C * B * gall * es, msg) ||
      dev_alloc(p, &tmean, (size_t)C * stats * 4, msg) ||
      dev_alloc(p, &tinv, (size_t)C * stats * 4, msg) ||
      dev_alloc(p, &p->TX, (size_t)C * 2 * B * X * es, msg) ||
      dev_alloc(p, &ta, (size_t)C * 2 * B * dall * es, msg) ||
      dev_alloc(p, &p->tlogits, (size_t)C * 2 * B * 4, msg) ||
      dev_alloc(p, &p->dl_d, (size_t)C * 2 * B * es, msg) ||
      dev_alloc(p, &p->dl_g, (size_t)C * B * es, msg) ||
      dev_alloc(p, &P, (size_t)C * 2 * B * dmax * es, msg) ||
      dev_alloc(p, &Q, (size_t)C * 2 * B * dmax * es, msg) ||
      dev_alloc(p, &P2, (size_t)C * B * dmax * es, msg) ||
      dev_alloc(p, &Q2, (size_t)C * B * dmax * es, msg) ||
      dev_alloc(p, &dh, (size_t)C * B * gmax * 4, msg) ||
      dev_alloc(p, &dcb, (size_t)C * B * gmax * es, msg) ||
      dev_alloc(p, &d5, (size_t)C * B * X * es, msg)) {
    dc_plan_destroy(p);
    return nullptr;
  }
  int64_t stat_off[5] = {0};  // per-problem offsets of each layer's statistics
  for (int l = 2; l <= 4; ++l) stat_off[l] = stat_off[l - 1] + gc[l - 1];
  const int64_t* go = b.goff;
  const int64_t* dof = b.doff;
  auto Wg = [&](int l) { return el(b.Gop, go[3 * (l - 1)]); };  // W1..W5 at 0, 3, 6, 9, 12
  auto Wd = [&](int l) { return el(b.Dop, dof[l - 1]); };
  std::vector<ConvDesc> v;
  std::vector<BnDesc> vb;
  auto bn = [&](const float* c, void* h, float* mean, float* inv, const int* wsel, int idx,
                int l, int n) {
    BnDesc q;
    memset(&q, 0, sizeof q);
    q.c = c;
    q.h = h;
    q.mean = mean;
    q.inv = inv;
    q.params = b.Gw;
    q.wsel = wsel;
    q.wsel_stride = b.PGs;
    q.wsel_idx = idx;
    q.off_gamma = go[3 * (l - 1) + 1];
    q.off_beta = go[3 * (l - 1) + 2];
    q.n = n;
    q.C = gc[l];
    q.lhw = 2 * ilog2(gs[l]);
    return q;
  };
  bool ok = true;
  // ---- evaluation: generator of every (cell, slot) on the cell's noise
  for (int l = 1; l <= 5; ++l) {
    v.clear();
    vb.clear();
    for (int c = 0; c < C; ++c)
      for (int sl = 0; sl < 5; ++sl) {
        const int pr = c * 5 + sl;
        const void* in = l == 1 ? el(b.Z, (int64_t)c * B * z) : el(eh, (int64_t)pr * B * gmax);
        void* out = l == 5 ? elw(b.E, (int64_t)c * b.e_cell + (int64_t)(1 + sl) * B * X)
                           : (void*)(ec + (int64_t)pr * B * gmax);
        ConvDesc q = cdesc(in, B, gc[l - 1], gs[l - 1], Wg(l), gc[l], gs[l], l == 1 ? 1 : 2,
                           l == 1 ? 0 : 1, out);
        q.wsel_stride = b.PGs;
        q.wsel_idx = pr;
        q.nhwc_out = (p->tcg && l == 1) ? 1 : 0;
        v.push_back(q);
        if (l <= 4)
          vb.push_back(bn(ec + (int64_t)pr * B * gmax, elw(eh, (int64_t)pr * B * gmax),
                          emean + pr * stats + stat_off[l], einv + pr * stats + stat_off[l],
                          nullptr, pr, l, B));
      }
    ok = ok && !upload(p, &p->eg[l - 1], v, msg);
    if (l <= 4) ok = ok && !upload(p, &p->ebn[l - 1], vb, msg);
  }
  // ---- evaluation: discriminator of every (cell, slot) on E[c] (6B rows), one cell per launch
  // (buffers ex / ey hold the five problems of one cell)
  for (int l = 1; l <= 4; ++l) {
    v.clear();
    for (int c = 0; c < C; ++c)
      for (int sl = 0; sl < 5; ++sl) {
        void* bufs[2] = {elw(ex, (int64_t)sl * 6 * B * dmax),
                         elw(ey, (int64_t)sl * 6 * B * dsz[2])};
        const void* in = l == 1 ? el(b.E, (int64_t)c * b.e_cell) : bufs[l % 2];
        void* out = bufs[(l + 1) % 2];
        ConvDesc q = cdesc(in, 6 * B, dc[l - 1], ds[l - 1], Wd(l), dc[l], ds[l], 2, 1, out);
        q.wsel_stride = b.PDs;
        q.wsel_idx = c * 5 + sl;
        v.push_back(q);
      }
    ok = ok && !upload(p, &p->ed[l - 1], v, msg);
  }
  {
    std::vector<LogitDesc> vl;
    for (int c = 0; c < C; ++c)
      for (int sl = 0; sl < 5; ++sl) {
        LogitDesc q;
        memset(&q, 0, sizeof q);
        q.a = elw(ey, (int64_t)sl * 6 * B * dsz[2]);  // layer 4's output (4 x 4 x 8d)
        q.w = Wd(5);
        q.wsel_stride = b.PDs;
        q.wsel_idx = c * 5 + sl;
        q.logits = b.logits + (int64_t)(c * 5 + sl) * 6 * B;
        q.rows = 6 * B;
        q.K = (int)dsz[4];
        vl.push_back(q);
      }
    ok = ok && !upload(p, &p->edl, vl, msg);
  }
  // ---- training forward: the selected generator on the cell's noise, fakes into TX rows
  // [B, 2B); the selected discriminator on TX (real rows copied in at run time)
  auto tgc = [&](int c, int l) { return tc + ((int64_t)c * B) * gall + (int64_t)B * goffs[l]; };
  auto tgh = [&](int c, int l) { return elw(th, (int64_t)c * B * gall + (int64_t)B * goffs[l]); };
  auto tda = [&](int c, int l) {
    return elw(ta, (int64_t)c * 2 * B * dall + (int64_t)2 * B * doffs[l]);
  };
  auto tx = [&](int c) { return elw(p->TX, (int64_t)c * 2 * B * X); };
  for (int l = 1; l <= 5; ++l) {
    v.clear();
    vb.clear();
    for (int c = 0; c < C; ++c) {
      const void* in = l == 1 ? el(b.Z, (int64_t)c * B * z) : (const void*)tgh(c, l - 1);
      void* out = l == 5 ? elw(tx(c), (int64_t)B * X) : (void*)tgc(c, l);
      ConvDesc q = cdesc(in, B, gc[l - 1], gs[l - 1], Wg(l), gc[l], gs[l], l == 1 ? 1 : 2,
                         l == 1 ? 0 : 1, out);
      q.wsel = b.src_g;
      q.wsel_stride = b.PGs;
      q.wsel_idx = c;
      q.nhwc_out = (tct && l == 1) ? 1 : 0;
      v.push_back(q);
      if (l <= 4)
        vb.push_back(bn(tgc(c, l), tgh(c, l), tmean + c * stats + stat_off[l],
                        tinv + c * stats + stat_off[l], b.src_g, c, l, B));
    }
    ok = ok && !upload(p, &p->tg[l - 1], v, msg);
    if (l <= 4) ok = ok && !upload(p, &p->tbn[l - 1], vb, msg);
  }
  for (int l = 1; l <= 4; ++l) {
    v.clear();
    for (int c = 0; c < C; ++c) {
      const void* in = l == 1 ? (const void*)tx(c) : (const void*)tda(c, l - 1);
      ConvDesc q = cdesc(in, 2 * B, dc[l - 1], ds[l - 1], Wd(l), dc[l], ds[l], 2, 1, tda(c, l));
      q.wsel = b.src_d;
      q.wsel_stride = b.PDs;
      q.wsel_idx = c;
      v.push_back(q);
    }
    ok = ok && !upload(p, &p->td[l - 1], v, msg);
  }
  {
    std::vector<LogitDesc> vl, vd, vg;
    for (int c = 0; c < C; ++c) {
      LogitDesc q;
      memset(&q, 0, sizeof q);
      q.a = tda(c, 4);
      q.w = Wd(5);
      q.wsel = b.src_d;
      q.wsel_stride = b.PDs;
      q.wsel_idx = c;
      q.logits = p->tlogits + (int64_t)c * 2 * B;
      q.rows = 2 * B;
      q.K = (int)dsz[4];
      vl.push_back(q);
      LogitDesc r = q;
      r.dl = elw(p->dl_d, (int64_t)c * 2 * B);
      r.da = elw(P, (int64_t)c * 2 * B * dmax);
      r.dw = b.gD + (int64_t)c * b.PDs + dof[4];
      vd.push_back(r);
      LogitDesc t = q;
      t.a = elw(tda(c, 4), (int64_t)B * dsz[4]);
      t.rows = B;
      t.dl = elw(p->dl_g, (int64_t)c * B);
      t.da = elw(P2, (int64_t)c * B * dmax);
      t.dw = nullptr;
      vg.push_back(t);
    }
    ok = ok && !upload(p, &p->tdl, vl, msg) && !upload(p, &p->tdl_back_d, vd, msg) &&
         !upload(p, &p->tdl_back_g, vg, msg);
  }
  // ---- discriminator backward (D loss, 2B rows): the delta of layer l's output is in P for
  // l = 4, 2 and in Q for l = 3, 1
  int64_t part_need = 0;
  for (int l = 4; l >= 1; --l) {
    v.clear();
    std::vector<ConvDesc> vd;
    for (int c = 0; c < C; ++c) {
      void* dout = elw((l % 2 == 0) ? P : Q, (int64_t)c * 2 * B * dmax);
      const void* prev = l == 1 ? (const void*)tx(c) : (const void*)tda(c, l - 1);
      // weight gradient: a = delta of the output (dc[l] x ds[l]^2), b = the layer's input
      ConvDesc w = cdesc(dout, 2 * B, dc[l], ds[l], prev, dc[l - 1], ds[l - 1], 2, 1,
                         b.gD + (int64_t)c * b.PDs + dof[l - 1]);
      w.a_hwc = tct;
      w.b_hwc = tct && l >= 2;
      v.push_back(w);
      if (l >= 2) {
        void* din = elw((l % 2 == 0) ? Q : P, (int64_t)c * 2 * B * dmax);
        ConvDesc q = cdesc(dout, 2 * B, dc[l], ds[l], Wd(l), dc[l - 1], ds[l - 1], 2, 1, din);
        q.wsel = b.src_d;
        q.wsel_stride = b.PDs;
        q.wsel_idx = c;
        q.aux = tda(c, l - 1);
        q.a_hwc = tct;
        q.nhwc_out = tct;
        vd.push_back(q);
      }
    }
    const int k = 4 - l;
    p->splits_dw[k] = wgrad_splits(v[0]);
    p->pstride_dw[k] = (int64_t)v[0].ca * v[0].co * 16;
    part_need = std::max<int64_t>(part_need, (int64_t)C * p->splits_dw[k] * p->pstride_dw[k]);
    ok = ok && !upload(p, &p->dw[k], v, msg);
    if (l >= 2) ok = ok && !upload(p, &p->dd[k], vd, msg);
  }
  // ---- generator loss through the discriminator (fake rows): deltas P2 (l = 4, 2), Q2
  // (l = 3, 1), then the fakes' delta times tanh' into d5
  for (int l = 4; l >= 1; --l) {
    v.clear();
    for (int c = 0; c < C; ++c) {
      void* dout = elw((l % 2 == 0) ? P2 : Q2, (int64_t)c * B * dmax);
      const bool last = l == 1;
      void* din = last ? elw(d5, (int64_t)c * B * X)
                       : elw((l % 2 == 0) ? Q2 : P2, (int64_t)c * B * dmax);
      ConvDesc q = cdesc(dout, B, dc[l], ds[l], Wd(l), dc[l - 1], ds[l - 1], 2, 1, din);
      q.wsel = b.src_d;
      q.wsel_stride = b.PDs;
      q.wsel_idx = c;
      q.aux = last ? elw(tx(c), (int64_t)B * X)
                   : elw(tda(c, l - 1), (int64_t)B * dsz[l - 1]);
      q.a_hwc = tct;
      q.nhwc_out = tct && !last;
      v.push_back(q);
    }
    ok = ok && !upload(p, &p->gd[4 - l], v, msg);
  }
  // ---- generator backward: weight gradient of layer l from its input (h_{l-1} or z) and the
  // delta of its output (d5, or dc_l in dcb); delta of its input dh_{l-1} (fp32), then the
  // batch normalisation of layer l - 1
  for (int l = 5; l >= 1; --l) {
    v.clear();
    std::vector<ConvDesc> vd;
    vb.clear();
    for (int c = 0; c < C; ++c) {
      const void* dout = l == 5 ? elw(d5, (int64_t)c * B * X) : elw(dcb, (int64_t)c * B * gmax);
      const void* in = l == 1 ? el(b.Z, (int64_t)c * B * z) : (const void*)tgh(c, l - 1);
      ConvDesc w = cdesc(in, B, gc[l - 1], gs[l - 1], dout, gc[l], gs[l], l == 1 ? 1 : 2,
                         l == 1 ? 0 : 1, b.gG + (int64_t)c * b.PGs + go[3 * (l - 1)]);
      w.a_hwc = tct;
      w.b_hwc = tct && l < 5;
      v.push_back(w);
      if (l >= 2) {
        ConvDesc q = cdesc(dout, B, gc[l], gs[l], Wg(l), gc[l - 1], gs[l - 1], 2, 1,
                           dh + (int64_t)c * B * gmax);
        q.wsel = b.src_g;
        q.wsel_stride = b.PGs;
        q.wsel_idx = c;
        q.a_hwc = tct && l < 5;
        q.nhwc_out = tct;
        vd.push_back(q);
        BnDesc r = bn(tgc(c, l - 1), tgh(c, l - 1), tmean + c * stats + stat_off[l - 1],
                      tinv + c * stats + stat_off[l - 1], b.src_g, c, l - 1, B);
        r.dh = dh + (int64_t)c * B * gmax;
        r.dc = elw(dcb, (int64_t)c * B * gmax);
        r.dparams = b.gG + (int64_t)c * b.PGs;
        r.hwc = tct;
        vb.push_back(r);
      }
    }
    const int k = 5 - l;
    p->splits_gw[k] = wgrad_splits(v[0]);
    p->pstride_gw[k] = (int64_t)v[0].ca * v[0].co * 16;
    part_need = std::max<int64_t>(part_need, (int64_t)C * p->splits_gw[k] * p->pstride_gw[k]);
    ok = ok && !upload(p, &p->gw[k], v, msg);
    if (l >= 2) {
      ok = ok && !upload(p, &p->gdh[k], vd, msg);
      ok = ok && !upload(p, &p->gbn[k], vb, msg);
    }
  }
  p->part_floats = part_need;
  ok = ok && !dev_alloc(p, &p->part, (size_t)part_need * 4, msg);
  // ---- tensor-core discriminator evaluation
  p->tc = ok && tcd;
  if (p->tc) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&p->sms, cudaDevAttrMultiProcessorCount, dev);
    ok = !dev_alloc(p, &p->Dwt, (size_t)s.n_indiv * b.PDs * 2, msg) &&
         !dev_alloc(p, &p->err, 4, msg) && ctc_prepare(msg);
    if (ok) ok = cudaMemset(p->err, 0, 4) == cudaSuccess;
    for (int l = 0; l < 6; ++l) p->rel.off[l] = dof[l];
    for (int l = 0; l < 5; ++l) p->rel.ci[l] = dc[l];
    p->rel.P = dof[5];
    for (int l = 1; l <= 4 && ok; ++l) {
      const int ci = dc[l - 1], co = dc[l];
      const int nbox = co < 256 ? co : 256;
      // the first layer's weights in their own [out][c][ky][kx] order, from the population
      const bf16* wbase = l == 1 ? (const bf16*)b.Dop + dof[0] : p->Dwt + dof[l - 1];
      ok = ctc_make_map(&p->mW[l - 1], wbase, (uint64_t)ci * 16, co, s.n_indiv, b.PDs, nbox, msg);
      CtcParams q;
      memset(&q, 0, sizeof q);
      q.rows = 6 * B;
      q.ci = ci;
      q.lhi = ilog2(ds[l - 1]);
      q.co = co;
      q.lho = ilog2(ds[l]);
      q.nchw_in = l == 1 ? 1 : 0;
      q.kchunks = (ci * 16 + 63) / 64;
      q.nj = (co + 255) / 256;
      q.nbox = nbox;
      q.mtiles = ((6 * B << (2 * q.lho)) + 127) / 128;
      q.n_tiles = 5 * q.mtiles;
      q.slope = s.slope;
      q.err = p->err;
      if (l == 4) {
        // the output layer in layer 4's epilogue: the logits straight into the fitness input
        q.out_mode = CTC_LRELU_LOGIT;
        q.logit_w = p->Dwt + dof[4];
        q.logit_ws = b.PDs;
      }
      p->cp[l - 1] = q;
      std::vector<ConvTcDesc> vt;
      for (int c = 0; c < C; ++c)
        for (int sl = 0; sl < 5; ++sl) {
          void* bx = elw(ex, (int64_t)sl * 6 * B * dmax);
          void* by = elw(ey, (int64_t)sl * 6 * B * dsz[2]);
          ConvTcDesc t;
          memset(&t, 0, sizeof t);
          t.in = (const bf16*)(l == 1 ? el(b.E, (int64_t)c * b.e_cell) : (l % 2 == 0 ? bx : by));
          t.out = (bf16*)(l % 2 == 1 ? bx : by);
          t.logits = b.logits + (int64_t)(c * 5 + sl) * 6 * B;
          t.wsel_idx = c * 5 + sl;
          vt.push_back(t);
        }
      ok = ok && !upload(p, &p->tcd[l - 1], vt, msg);
      // one map serves every cell: the chunk buffers are shared
      ok = ok && act_map(&p->aEd[l - 1], &p->cp[l - 1], vt.data(), 5);
      // the first layer stores its output by TMA (its gather needs no activation map)
      if (l == 1) ok = ok && ctc_make_out_map(&p->aEd[0], &p->cp[0], vt.data(), 5, msg);
      for (size_t k = 5; k < vt.size() && ok && l >= 2; ++k)
        if (vt[k].in != vt[k % 5].in) {
          if (msg) *msg = "DCGAN evaluation buffers differ between cells";
          ok = false;
        }
    }
  }
  // ---- tensor-core generator evaluation (layers 2-5)
  if (ok && p->tcg) {
    if (!p->tc) {
      int dev = 0;
      cudaGetDevice(&dev);
      cudaDeviceGetAttribute(&p->sms, cudaDevAttrMultiProcessorCount, dev);
      ok = !dev_alloc(p, &p->err, 4, msg) && ctc_prepare(msg) &&
           cudaMemset(p->err, 0, 4) == cudaSuccess;
    }
    RelayoutG& r = p->relg;
    memset(&r, 0, sizeof r);
    r.n = 4;
    int64_t off = 0;
    for (int i = 0; i < 4; ++i) {
      const int l = i + 2;
      r.src_off[i] = go[3 * (l - 1)];
      r.ci[i] = gc[l - 1];
      r.co[i] = gc[l];
      r.cls_rows[i] = l == 5 ? 16 : gc[l];
      r.dst_off[i] = off;
      off += (int64_t)4 * r.cls_rows[i] * 4 * gc[l - 1];
    }
    p->g1tc = dense1_tc_supported(B, s.z, gc[1]);
    if (p->g1tc) {
      p->g1_off = (off + 63) / 64 * 64;
      off = p->g1_off + (int64_t)16 * gc[1] * 128;
    }
    p->gwt_ps = (off + 63) / 64 * 64;
    ok = ok && !dev_alloc(p, &p->bnpart, (size_t)bn_hwc_part_floats(PE, 8 * g) * 4, msg);
    ok = ok && !dev_alloc(p, &p->bncnt, (size_t)bn_hwc_counters(PE, 8 * g) * 4, msg);
    if (ok) ok = cudaMemset(p->bncnt, 0, (size_t)bn_hwc_counters(PE, 8 * g) * 4) == cudaSuccess;
    ok = ok && !dev_alloc(p, &p->Gwt, (size_t)s.n_indiv * p->gwt_ps * 2, msg);
    if (ok) ok = cudaMemset(p->Gwt, 0, (size_t)s.n_indiv * p->gwt_ps * 2) == cudaSuccess;
    if (ok && p->g1tc)
      ok = ctc_make_map(&p->mG1, p->Gwt + p->g1_off, 128, (uint64_t)16 * gc[1], s.n_indiv,
                        p->gwt_ps, 256, msg);
    for (int i = 0; i < 4 && ok; ++i) {
      const int l = i + 2;
      const int ci = gc[l - 1], co = gc[l];
      const int nbox = l == 5 ? 16 : (co < 256 ? co : 256);
      ok = ctc_make_map(&p->mG[i], p->Gwt + r.dst_off[i], (uint64_t)4 * ci, 4 * r.cls_rows[i],
                        s.n_indiv, p->gwt_ps, nbox, msg);
      CtcParams q;
      memset(&q, 0, sizeof q);
      q.rows = B;
      q.ci = ci;
      q.lhi = ilog2(gs[l - 1]);
      q.co = co;
      q.lho = ilog2(gs[l]);
      q.kchunks = 4 * ci / 64;
      q.nj = l == 5 ? 1 : (co + 255) / 256;
      q.nbox = nbox;
      q.transposed = 1;
      q.out_mode = l == 5 ? CTC_TANH_CHW : CTC_F32_HWC;
      q.cls_rows = r.cls_rows[i];
      q.mtiles = ((B << (2 * (q.lho - 1))) + 127) / 128;
      q.n_tiles = PE * 4 * q.mtiles;
      q.slope = s.slope;
      q.err = p->err;
      p->gp[i] = q;
      std::vector<ConvTcDesc> vt;
      for (int c = 0; c < C; ++c)
        for (int sl = 0; sl < 5; ++sl) {
          const int pr = c * 5 + sl;
          ConvTcDesc t;
          memset(&t, 0, sizeof t);
          t.in = (const bf16*)el(eh, (int64_t)pr * B * gmax);
          t.out = l == 5 ? (bf16*)elw(b.E, (int64_t)c * b.e_cell + (int64_t)(1 + sl) * B * X)
                         : (bf16*)(ec + (int64_t)pr * B * gmax);
          t.wsel_idx = pr;
          vt.push_back(t);
        }
      ok = ok && !upload(p, &p->gtd[i], vt, msg);
      if (l == 5) p->h_gtd5 = vt;
      ok = ok && act_map(&p->aEg[i], &p->gp[i], vt.data(), PE);
    }
    // the fp32 layers (2-4) sum their batch-norm statistics in the epilogue: slots of
    // (tile, half, lane quarter), consecutive per problem
    int64_t bnmax = p->g1tc ? (int64_t)PE * 16 * gc[1] : 0;  // layer 1: a slot per tap
    for (int i = 0; i < 3; ++i) {
      const CtcParams& q = p->gp[i];
      bnmax = std::max(bnmax, (int64_t)q.n_tiles * (q.m2 ? 2 : 1) * 4 * q.co);
    }
    ok = ok && !dev_alloc(p, &p->bnp, (size_t)bnmax * sizeof(float2), msg);
    for (int i = 0; i < 3 && ok; ++i) {
      CtcParams& q = p->gp[i];
      q.bn_part = p->bnp;
      p->bn_slots_e[i] = q.n_tiles / PE * (q.m2 ? 2 : 1) * 4;
    }
  }
  // ---- tensor-core training forward (channel-last), and the output layer's descriptors in
  // the re-laid (tap, channel) order
  if (ok && tct) {
    for (int i = 0; i < 4 && ok; ++i) {
      const int l = i + 2;
      CtcParams q = p->gp[i];
      q.mtiles = ((B << (2 * (q.lho - 1))) + 127) / 128;
      q.n_tiles = C * 4 * q.mtiles;
      p->tgp[i] = q;
      std::vector<ConvTcDesc> vt;
      for (int c = 0; c < C; ++c) {
        ConvTcDesc t;
        memset(&t, 0, sizeof t);
        t.in = (const bf16*)tgh(c, l - 1);
        t.out = l == 5 ? (bf16*)elw(tx(c), (int64_t)B * X) : (bf16*)tgc(c, l);
        t.wsel_idx = c;
        vt.push_back(t);
      }
      ok = ok && !upload(p, &p->tgd[i], vt, msg);
      if (l == 5) p->h_tgd5 = vt;
      ok = ok && act_map(&p->aTg[i], &p->tgp[i], vt.data(), C);
      if (i < 3)
        p->bn_slots_t[i] = p->tgp[i].n_tiles / C * (p->tgp[i].m2 ? 2 : 1) * 4;
    }
    for (int l = 1; l <= 4 && ok; ++l) {
      CtcParams q = p->cp[l - 1];
      q.rows = 2 * B;
      q.mtiles = ((2 * B << (2 * q.lho)) + 127) / 128;
      q.n_tiles = C * q.mtiles;
      q.out_mode = CTC_LRELU_HWC;  // training keeps the activations (the backward reads them)
      q.logit_w = nullptr;
      p->tdp[l - 1] = q;
      std::vector<ConvTcDesc> vt;
      for (int c = 0; c < C; ++c) {
        ConvTcDesc t;
        memset(&t, 0, sizeof t);
        t.in = (const bf16*)(l == 1 ? (const void*)tx(c) : (const void*)tda(c, l - 1));
        t.out = (bf16*)tda(c, l);
        t.wsel_idx = c;
        vt.push_back(t);
      }
      ok = ok && !upload(p, &p->tdd[l - 1], vt, msg);
      ok = ok && act_map(&p->aTd[l - 1], &p->tdp[l - 1], vt.data(), C);
      if (l == 1) ok = ok && ctc_make_out_map(&p->aTd[0], &p->tdp[0], vt.data(), C, msg);
    }
    std::vector<LogitDesc> vl, vd, vg;
    for (int c = 0; c < C; ++c) {
      LogitDesc q;
      memset(&q, 0, sizeof q);
      q.a = tda(c, 4);
      q.w = p->Dwt + dof[4];
      q.wsel = b.src_d;
      q.wsel_stride = b.PDs;
      q.wsel_idx = c;
      q.logits = p->tlogits + (int64_t)c * 2 * B;
      q.rows = 2 * B;
      q.K = (int)dsz[4];
      q.hwc_c = 8 * d;
      vl.push_back(q);
      LogitDesc r = q;
      r.dl = elw(p->dl_d, (int64_t)c * 2 * B);
      r.da = elw(P, (int64_t)c * 2 * B * dmax);
      r.dw = b.gD + (int64_t)c * b.PDs + dof[4];
      vd.push_back(r);
      LogitDesc t = q;
      t.a = elw(tda(c, 4), (int64_t)B * dsz[4]);
      t.rows = B;
      t.dl = elw(p->dl_g, (int64_t)c * B);
      t.da = elw(P2, (int64_t)c * B * dmax);
      t.dw = nullptr;
      vg.push_back(t);
    }
    ok = ok && !upload(p, &p->tdl_tc, vl, msg) && !upload(p, &p->tdl_back_d_tc, vd, msg) &&
         !upload(p, &p->tdl_back_g_tc, vg, msg);
  }
  if (ok && tct) {
    // discriminator input gradients: layer l's transposed convolution (in dc[l], out dc[l-1])
    RelayoutG& r = p->reld;
    memset(&r, 0, sizeof r);
    r.n = 4;
    int64_t off = 0;
    for (int i = 0; i < 4; ++i) {
      const int l = 4 - i;
      r.src_off[i] = dof[l - 1];
      r.ci[i] = dc[l];
      r.co[i] = dc[l - 1];
      r.cls_rows[i] = l == 1 ? 16 : dc[l - 1];
      r.dst_off[i] = off;
      off += (int64_t)4 * r.cls_rows[i] * 4 * dc[l];
    }
    p->ddt_ps = (off + 63) / 64 * 64;
    ok = !dev_alloc(p, &p->Ddt, (size_t)s.n_indiv * p->ddt_ps * 2, msg) &&
         cudaMemset(p->Ddt, 0, (size_t)s.n_indiv * p->ddt_ps * 2) == cudaSuccess;
    for (int i = 0; i < 4 && ok; ++i) {
      const int l = 4 - i;
      const int nbox = l == 1 ? 16 : (dc[l - 1] < 256 ? dc[l - 1] : 256);
      ok = ctc_make_map(&p->mDd[l - 1], p->Ddt + r.dst_off[i], (uint64_t)4 * dc[l],
                        4 * r.cls_rows[i], s.n_indiv, p->ddt_ps, nbox, msg);
      for (int chain = 0; chain < 2 && ok; ++chain) {
        if (chain == 0 && l == 1) continue;  // the D loss needs no input gradient of layer 1
        const int rows = chain == 0 ? 2 * B : B;
        CtcParams q;
        memset(&q, 0, sizeof q);
        q.rows = rows;
        q.ci = dc[l];
        q.lhi = ilog2(ds[l]);
        q.co = dc[l - 1];
        q.lho = ilog2(ds[l - 1]);
        q.kchunks = 4 * dc[l] / 64;
        q.nj = l == 1 ? 1 : (dc[l - 1] + 255) / 256;
        q.nbox = nbox;
        q.transposed = 1;
        q.out_mode = l == 1 ? CTC_DTANH_CHW : CTC_DLRELU_HWC;
        q.cls_rows = r.cls_rows[i];
        q.mtiles = ((rows << (2 * (q.lho - 1))) + 127) / 128;
        q.n_tiles = C * 4 * q.mtiles;
        q.slope = s.slope;
        q.err = p->err;
        std::vector<ConvTcDesc> vt;
        for (int c = 0; c < C; ++c) {
          ConvTcDesc t;
          memset(&t, 0, sizeof t);
          t.wsel_idx = c;
          if (chain == 0) {
            t.in = (const bf16*)elw((l % 2 == 0) ? P : Q, (int64_t)c * 2 * B * dmax);
            t.out = (bf16*)elw((l % 2 == 0) ? Q : P, (int64_t)c * 2 * B * dmax);
            t.aux = (const bf16*)tda(c, l - 1);
          } else {
            t.in = (const bf16*)elw((l % 2 == 0) ? P2 : Q2, (int64_t)c * B * dmax);
            t.out = l == 1 ? (bf16*)elw(d5, (int64_t)c * B * X)
                           : (bf16*)elw((l % 2 == 0) ? Q2 : P2, (int64_t)c * B * dmax);
            t.aux = l == 1 ? (const bf16*)elw(tx(c), (int64_t)B * X)
                           : (const bf16*)elw(tda(c, l - 1), (int64_t)B * dsz[l - 1]);
          }
          vt.push_back(t);
        }
        if (chain == 0) {
          ok = act_map(&p->aDd[4 - l], &q, vt.data(), C);
          p->ddp[4 - l] = q;
          ok = !upload(p, &p->ddd[4 - l], vt, msg);
        } else {
          ok = act_map(&p->aGd[4 - l], &q, vt.data(), C);
          p->gdp[4 - l] = q;
          if (l == 1) p->h_gdd1 = vt;
          ok = !upload(p, &p->gdd[4 - l], vt, msg);
        }
      }
    }
    // generator input gradients: layer l's convolution (in gc[l] channels, out gc[l-1])
    RelayoutC& rc = p->relc;
    memset(&rc, 0, sizeof rc);
    rc.n = 4;
    off = 0;
    for (int i = 0; i < 4; ++i) {
      const int l = 5 - i;
      rc.src_off[i] = go[3 * (l - 1)];
      rc.o[i] = gc[l - 1];
      rc.c[i] = gc[l];
      rc.dst_off[i] = off;
      off += (int64_t)gc[l - 1] * gc[l] * 16;
    }
    p->gct_ps = (off + 63) / 64 * 64;
    ok = ok && !dev_alloc(p, &p->Gct, (size_t)s.n_indiv * p->gct_ps * 2, msg);
    for (int i = 0; i < 4 && ok; ++i) {
      const int l = 5 - i;
      const int co = gc[l - 1], nbox = co < 256 ? co : 256;
      // the output layer's input gradient reads 3-channel images: its weights in their own
      // [out][c][ky][kx] order, from the population (launch_relayout_c leaves them out)
      ok = gc[l] == 3
               ? ctc_make_map(&p->mGc[i], (const bf16*)b.Gop + go[3 * (l - 1)], 48, co,
                              s.n_indiv, b.PGs, nbox, msg)
               : ctc_make_map(&p->mGc[i], p->Gct + rc.dst_off[i], (uint64_t)16 * gc[l], co,
                              s.n_indiv, p->gct_ps, nbox, msg);
      CtcParams q;
      memset(&q, 0, sizeof q);
      q.rows = B;
      q.ci = gc[l];
      q.lhi = ilog2(gs[l]);
      q.co = co;
      q.lho = ilog2(gs[l - 1]);
      q.nchw_in = l == 5 ? 1 : 0;
      q.kchunks = (16 * gc[l] + 63) / 64;
      q.nj = (co + 255) / 256;
      q.nbox = nbox;
      q.out_mode = CTC_F32_HWC;
      q.mtiles = ((B << (2 * q.lho)) + 127) / 128;
      q.n_tiles = C * q.mtiles;
      q.slope = s.slope;
      q.err = p->err;
      p->gcp[i] = q;
      std::vector<ConvTcDesc> vt;
      for (int c = 0; c < C; ++c) {
        ConvTcDesc t;
        memset(&t, 0, sizeof t);
        t.in = l == 5 ? (const bf16*)elw(d5, (int64_t)c * B * X)
                      : (const bf16*)elw(dcb, (int64_t)c * B * gmax);
        t.out = (bf16*)(dh + (int64_t)c * B * gmax);
        t.wsel_idx = c;
        vt.push_back(t);
      }
      ok = ok && !upload(p, &p->gcd[i], vt, msg);
      ok = ok && act_map(&p->aGc[i], &p->gcp[i], vt.data(), C);
    }
    // weight gradients: a = the output's delta (discriminator) or the layer's input
    // (generator), M = its channels; b = the other operand, gathered per tap
    ok = ok && wgtc_prepare(msg);
    int64_t wneed = 0;
    auto wplan = [&](WgtcParams& q) {
      const int64_t Kp = (int64_t)q.rows << (2 * q.la);
      const int64_t chunks = (Kp + 63) / 64;
      const int64_t per = (int64_t)C * ((q.M + 127) / 128) * (q.b_chw ? 1 : q.N / 256);
      // the fewest splits whose wave fill is within 3 % of the best: every split adds an
      // M x N fp32 partial to write and read back
      const int sp_max = (int)std::min<int64_t>(64, std::max<int64_t>(1, chunks / 8));
      auto fill = [&](int sp) {
        const int64_t t = per * sp;
        return (double)t / ((double)((t + p->sms - 1) / p->sms) * p->sms);
      };
      double be = 0;
      for (int sp = 1; sp <= sp_max; ++sp) be = std::max(be, fill(sp));
      int best = 1;
      while (best < sp_max && fill(best) < 0.97 * be) ++best;
      q.kc = (chunks + best - 1) / best * 64;
      q.splits = (int)((Kp + q.kc - 1) / q.kc);
      q.n_tiles = (int)(per * q.splits);
      q.n_probs = C;
      q.err = p->err;
      wneed = std::max<int64_t>(wneed, (int64_t)C * q.splits * q.M * q.N);
    };
    for (int l = 4; l >= 1 && ok; --l) {
      const int k = 4 - l;
      // layer 1 reads the 3-channel channel-major images (b_chw)
      if (l == 1 ? dc[1] % 64 != 0 : (dc[l] % 128 != 0 || dc[l - 1] % 64 != 0)) continue;
      WgtcParams q;
      memset(&q, 0, sizeof q);
      q.rows = 2 * B;
      q.M = dc[l];
      q.Cb = dc[l - 1];
      q.b_chw = l == 1;
      q.N = l == 1 ? 64 : 16 * q.Cb;
      q.la = ilog2(ds[l]);
      q.lb = ilog2(ds[l - 1]);
      q.s = 2;
      q.p = 1;
      wplan(q);
      std::vector<WgtcDesc> vw;
      for (int c = 0; c < C; ++c) {
        WgtcDesc w;
        w.a = (const bf16*)elw((l % 2 == 0) ? P : Q, (int64_t)c * 2 * B * dmax);
        w.b = (const bf16*)(l == 1 ? (const void*)tx(c) : (const void*)tda(c, l - 1));
        w.dw = b.gD + (int64_t)c * b.PDs + dof[l - 1];
        vw.push_back(w);
      }
      ok = wgtc_make_maps(&p->wdA[k], &p->wdB[k], &q, vw.data(), C, msg);
      if (gather_a) q.a_tma = 0;
      p->wdp[k] = q;
      p->wtc_d[k] = true;
      ok = ok && !upload(p, &p->wdd[k], vw, msg);
    }
    for (int l = 5; l >= 2 && ok; --l) {
      const int k = 5 - l;
      // layer 5 gathers the 3-channel channel-major delta of the fakes (b_chw)
      if (l == 5 ? gc[4] % 64 != 0 : (gc[l - 1] % 128 != 0 || gc[l] % 64 != 0)) continue;
      WgtcParams q;
      memset(&q, 0, sizeof q);
      q.rows = B;
      q.M = gc[l - 1];
      q.Cb = gc[l];
      q.b_chw = l == 5;
      q.N = l == 5 ? 64 : 16 * q.Cb;
      q.la = ilog2(gs[l - 1]);
      q.lb = ilog2(gs[l]);
      q.s = 2;
      q.p = 1;
      wplan(q);
      std::vector<WgtcDesc> vw;
      for (int c = 0; c < C; ++c) {
        WgtcDesc w;
        w.a = (const bf16*)tgh(c, l - 1);
        w.b = (const bf16*)(l == 5 ? elw(d5, (int64_t)c * B * X) : elw(dcb, (int64_t)c * B * gmax));
        w.dw = b.gG + (int64_t)c * b.PGs + go[3 * (l - 1)];
        vw.push_back(w);
      }
      ok = wgtc_make_maps(&p->wgA[k], &p->wgB[k], &q, vw.data(), C, msg);
      if (gather_a) q.a_tma = 0;
      p->wgp[k] = q;
      p->wtc_g[k] = true;
      ok = ok && !upload(p, &p->wgd[k], vw, msg);
    }
    ok = ok && !dev_alloc(p, &p->wpart, (size_t)wneed * 4, msg);
    // generator layer 1: z^T times its deltas in (o, tap) order
    p->g1w = ok && dense1_tc_supported(B, s.z, gc[1]);
    if (p->g1w) {
      p->dcb = dcb;
      p->dcb_cell = (int64_t)B * gmax;
      ok = !dev_alloc(p, &p->dc1t, (size_t)C * B * 16 * gc[1] * 2, msg) &&
           dense1_wgrad_make_map(&p->mG1w, p->dc1t, B, gc[1], C, msg);
    }
  }
  // ---- scatter mode for the 64 -> 3 transposed convolutions (its A tiles always come by TMA:
  // it has no gathered form)
  p->scg = ok && p->tcg && g == 64;
  p->scd = ok && tct && d == 64;
  if (p->scg || p->scd) {
    auto scatter_params = [&](int rows, int n_probs, int out_mode) {
      CtcParams q;
      memset(&q, 0, sizeof q);
      q.rows = rows;
      q.ci = 64;
      q.lhi = 5;
      q.co = 3;
      q.lho = 6;
      q.kchunks = 1;
      q.nj = 1;
      q.nbox = 64;
      q.out_mode = out_mode;
      q.scatter = 1;
      q.mtiles = (rows << 10) / 128;
      q.n_tiles = n_probs * q.mtiles;
      q.slope = s.slope;
      q.err = p->err;
      return q;
    };
    ok = !dev_alloc(p, &p->halo, (size_t)std::max(PE, C) * B * 8 * 768 * 4, msg);
    if (ok && p->scg) {
      ok = !dev_alloc(p, &p->Gs, (size_t)s.n_indiv * 4096 * 2, msg) &&
           ctc_make_map(&p->mGs, p->Gs, 64, 64, s.n_indiv, 4096, 64, msg);
      p->egs = scatter_params(B, PE, CTC_TANH_CHW);
      p->egs.halo = p->halo;
      ok = ok && ctc_make_act_map(&p->aEgs, &p->egs, p->h_gtd5.data(), PE, msg);
      if (ok && tct) {
        p->tgs = scatter_params(B, C, CTC_TANH_CHW);
        p->tgs.halo = p->halo;
        ok = ctc_make_act_map(&p->aTgs, &p->tgs, p->h_tgd5.data(), C, msg);
      }
      if (ok && !(p->egs.a_tma && (!tct || p->tgs.a_tma))) p->scg = false;
    }
    if (ok && p->scd) {
      ok = !dev_alloc(p, &p->Ds, (size_t)s.n_indiv * 4096 * 2, msg) &&
           ctc_make_map(&p->mDs, p->Ds, 64, 64, s.n_indiv, 4096, 64, msg);
      p->gds = scatter_params(B, C, CTC_DTANH_CHW);
      p->gds.halo = p->halo;
      ok = ok && ctc_make_act_map(&p->aGds, &p->gds, p->h_gdd1.data(), C, msg);
      if (ok && !p->gds.a_tma) p->scd = false;
    }
  }
  if (!ok) {
    dc_plan_destroy(p);
    return nullptr;
  }
  p->eval_launches = 9 + 5 * C;
  p->train_launches = tct ? 60 + (p->scg ? 1 : 0) + (p->scd ? 2 : 0) : 50;
  return p;
}

void dc_plan_destroy(DcPlan* p) {
  if (!p) return;
  for (void* q : p->allocs) cudaFree(q);
  delete p;
}

namespace {
int no_variant(std::string* msg) {
  if (msg) *msg = "no tensor-core convolution variant for a layer's A kind and output mode";
  return 1;
}

int check(std::string* msg, const char* what) {
  cudaError_t e = cudaGetLastError();
  if (e == cudaSuccess) return 0;
  if (msg) *msg = std::string(what) + ": " + cudaGetErrorString(e);
  return 1;
}
}  // namespace

void dc_set_indiv_range(DcPlan* p, int lo, int n) {
  p->rl_lo = lo;
  p->rl_n = n;
}

int dc_eval_g(DcPlan* p, const int* nbr, cudaStream_t st, std::string* msg) {
  const DcShape& s = p->s;
  const int C = s.cells, B = s.B, g = s.ngf;
  const int gc[6] = {s.z, 8 * g, 4 * g, 2 * g, g, 3};
  const int gs[6] = {1, 4, 8, 16, 32, 64};
  const int PE = C * 5;
  if (p->tcg) {
    const int64_t lo = p->rl_n > 0 ? p->rl_lo : 0;
    const int nI = p->rl_n > 0 ? p->rl_n : s.n_indiv;
    const bf16* gop = (const bf16*)p->b.Gop + lo * p->b.PGs;
    launch_relayout_g(gop, p->b.PGs, p->Gwt + lo * p->gwt_ps, p->gwt_ps, nI, p->relg, st);
    if (p->g1tc) {
      launch_relayout_g1(gop, p->b.PGs, p->b.goff[0], p->Gwt + lo * p->gwt_ps + p->g1_off,
                         p->gwt_ps, s.z, gc[1], nI, st);
      // (its epilogue sums the batch-norm statistics: 16 slots, one per tap)
      launch_dense1_tc(p->mG1, p->eg[0], PE, nbr, B, s.z, gc[1], p->err, st, p->bnp);
      launch_bn_relu_hwc_part(p->ebn[0], PE, gc[1], nbr, p->bnp, 16, (int64_t)B * 16 * gc[1], st);
    } else {
      launch_conv(DENSE1_MODE, CEPI_NONE_, true, true, p->eg[0], PE, B, 16 * gc[1], nbr, 1,
                  nullptr, 0, s.slope, st);
      launch_bn_relu_hwc(p->ebn[0], PE, gc[1], nbr, p->bnpart, p->bncnt, (int64_t)B * 16 * gc[1],
                         st);
    }
    if (p->scg)
      launch_relayout_s(gop, p->b.PGs, p->b.goff[12], p->Gs + lo * 4096, nI, st);
    for (int i = 0; i < 4; ++i) {
      CtcParams q = p->gp[i];
      q.descs = p->gtd[i];
      q.wsel = nbr;
      if (i == 3 && p->scg) {
        q = p->egs;
        q.descs = p->gtd[i];
        q.wsel = nbr;
        if (!launch_conv_tc(p->mGs, p->aEgs, q, p->sms, st)) return no_variant(msg);
        launch_scatter_fix(p->gtd[i], p->halo, PE, B, CTC_TANH_CHW, st);
        continue;
      }
      if (!launch_conv_tc(p->mG[i], p->aEg[i], q, p->sms, st)) return no_variant(msg);
      if (i < 3)
        launch_bn_relu_hwc_part(p->ebn[i + 1], PE, gc[i + 2], nbr, p->bnp, p->bn_slots_e[i],
                                (int64_t)B * gs[i + 2] * gs[i + 2] * gc[i + 2], st);
    }
    return check(msg, "DCGAN generator evaluation (tensor cores)");
  }
  for (int l = 1; l <= 5; ++l) {
    if (l == 1)
      launch_conv(DENSE1_MODE, CEPI_NONE_, s.bf, true, p->eg[0], PE, B, 16 * gc[1], nbr, 1,
                  nullptr, 0, s.slope, st);
    else
      launch_conv(CONVT2_MODE, l == 5 ? CEPI_TANH_ : CEPI_NONE_, s.bf, l < 5, p->eg[l - 1], PE,
                  B * gs[l] * gs[l], gc[l], nbr, 1, nullptr, 0, s.slope, st);
    if (l <= 4) launch_bn_relu(s.bf, p->ebn[l - 1], PE, gc[l], nbr, st);
  }
  return check(msg, "DCGAN generator evaluation");
}

int dc_eval_d(DcPlan* p, const int* nbr, cudaStream_t st, std::string* msg) {
  const DcShape& s = p->s;
  const int C = s.cells, B = s.B, d = s.ndf;
  const int dc[5] = {3, d, 2 * d, 4 * d, 8 * d};
  const int ds[5] = {64, 32, 16, 8, 4};
  if (p->tc) {
    // weights in the layout the tensor-core convolution reads, for every individual (they
    // change after every training step)
    const int64_t lo = p->rl_n > 0 ? p->rl_lo : 0;
    const int nI = p->rl_n > 0 ? p->rl_n : s.n_indiv;
    launch_relayout_d((const bf16*)p->b.Dop + lo * p->b.PDs, p->Dwt + lo * p->b.PDs, nI,
                      p->b.PDs, p->rel, st);
    for (int c = 0; c < C; ++c) {
      for (int l = 1; l <= 4; ++l) {
        CtcParams q = p->cp[l - 1];
        q.descs = p->tcd[l - 1] + c * 5;
        q.wsel = nbr;
        if (!launch_conv_tc(p->mW[l - 1], p->aEd[l - 1], q, p->sms, st)) return no_variant(msg);
      }
    }
    return check(msg, "DCGAN discriminator evaluation (tensor cores)");
  }
  for (int c = 0; c < C; ++c) {
    for (int l = 1; l <= 4; ++l)
      launch_conv(CONV_FWD_MODE, CEPI_LRELU_, s.bf, false, p->ed[l - 1] + c * 5, 5,
                  6 * B * ds[l] * ds[l], dc[l], nbr, 1, nullptr, 0, s.slope, st);
    launch_logit_dot(s.bf, p->edl + c * 5, 5, 6 * B, nbr, st);
  }
  return check(msg, "DCGAN discriminator evaluation");
}

int dc_train(DcPlan* p, cudaStream_t st, std::string* msg) {
  const DcShape& s = p->s;
  const int C = s.cells, B = s.B, g = s.ngf, d = s.ndf;
  const size_t es = s.bf ? 2 : 4;
  const int64_t X = 3 * 64 * 64;
  const int gc[6] = {s.z, 8 * g, 4 * g, 2 * g, g, 3};
  const int gs[6] = {1, 4, 8, 16, 32, 64};
  const int dc[5] = {3, d, 2 * d, 4 * d, 8 * d};
  const int ds[5] = {64, 32, 16, 8, 4};
  // forward of the selected pair
  if (p->tct) {
    if (p->g1tc) {
      launch_dense1_tc(p->mG1, p->tg[0], C, nullptr, B, s.z, gc[1], p->err, st, p->bnp);
      launch_bn_relu_hwc_part(p->tbn[0], C, gc[1], nullptr, p->bnp, 16, (int64_t)B * 16 * gc[1],
                              st);
    } else {
      launch_conv(DENSE1_MODE, CEPI_NONE_, true, true, p->tg[0], C, B, 16 * gc[1], nullptr, 1,
                  nullptr, 0, s.slope, st);
      launch_bn_relu_hwc(p->tbn[0], C, gc[1], nullptr, p->bnpart, p->bncnt,
                         (int64_t)B * 16 * gc[1], st);
    }
    for (int i = 0; i < 4; ++i) {
      CtcParams q = p->tgp[i];
      q.descs = p->tgd[i];
      q.wsel = p->b.src_g;
      if (i == 3 && p->scg) {
        q = p->tgs;
        q.descs = p->tgd[i];
        q.wsel = p->b.src_g;
        if (!launch_conv_tc(p->mGs, p->aTgs, q, p->sms, st)) return no_variant(msg);
        launch_scatter_fix(p->tgd[i], p->halo, C, B, CTC_TANH_CHW, st);
        continue;
      }
      if (!launch_conv_tc(p->mG[i], p->aTg[i], q, p->sms, st)) return no_variant(msg);
      if (i < 3)
        launch_bn_relu_hwc_part(p->tbn[i + 1], C, gc[i + 2], nullptr, p->bnp, p->bn_slots_t[i],
                                (int64_t)B * gs[i + 2] * gs[i + 2] * gc[i + 2], st);
    }
  } else {
    for (int l = 1; l <= 5; ++l) {
      if (l == 1)
        launch_conv(DENSE1_MODE, CEPI_NONE_, s.bf, true, p->tg[0], C, B, 16 * gc[1], nullptr, 1,
                    nullptr, 0, s.slope, st);
      else
        launch_conv(CONVT2_MODE, l == 5 ? CEPI_TANH_ : CEPI_NONE_, s.bf, l < 5, p->tg[l - 1], C,
                    B * gs[l] * gs[l], gc[l], nullptr, 1, nullptr, 0, s.slope, st);
      if (l <= 4) launch_bn_relu(s.bf, p->tbn[l - 1], C, gc[l], nullptr, st);
    }
  }
  // the real rows of every cell's minibatch into TX rows [0, B)
  if (cudaMemcpy2DAsync(p->TX, 2 * B * X * es, p->b.E, p->b.e_cell * es, B * X * es, C,
                        cudaMemcpyDeviceToDevice, st) != cudaSuccess) {
    check(msg, "DCGAN training input copy");
    return 1;
  }
  if (p->tct) {
    for (int l = 1; l <= 4; ++l) {
      CtcParams q = p->tdp[l - 1];
      q.descs = p->tdd[l - 1];
      q.wsel = p->b.src_d;
      if (!launch_conv_tc(p->mW[l - 1], p->aTd[l - 1], q, p->sms, st)) return no_variant(msg);
    }
    launch_logit_dot(true, p->tdl_tc, C, 2 * B, nullptr, st);
  } else {
    for (int l = 1; l <= 4; ++l)
      launch_conv(CONV_FWD_MODE, CEPI_LRELU_, s.bf, false, p->td[l - 1], C,
                  2 * B * ds[l] * ds[l], dc[l], nullptr, 1, nullptr, 0, s.slope, st);
    launch_logit_dot(s.bf, p->tdl, C, 2 * B, nullptr, st);
  }
  launch_dc_dlogit(s.bf, p->tlogits, C, B, p->dl_d, p->dl_g, st);
  if (p->tct) {
    // weights in the layouts the tensor-core input gradients read
    const int64_t lo = p->rl_n > 0 ? p->rl_lo : 0;
    const int nI = p->rl_n > 0 ? p->rl_n : s.n_indiv;
    const bf16* dop = (const bf16*)p->b.Dop + lo * p->b.PDs;
    launch_relayout_g(dop, p->b.PDs, p->Ddt + lo * p->ddt_ps, p->ddt_ps, nI, p->reld, st);
    launch_relayout_c((const bf16*)p->b.Gop + lo * p->b.PGs, p->b.PGs, p->Gct + lo * p->gct_ps,
                      p->gct_ps, nI, p->relc, st);
    if (p->scd) launch_relayout_s(dop, p->b.PDs, p->b.doff[0], p->Ds + lo * 4096, nI, st);
  }
  // discriminator backward (D loss)
  launch_logit_back(s.bf, p->tct ? p->tdl_back_d_tc : p->tdl_back_d, C, (int)(8 * d * 16), true,
                    s.slope, st);
  for (int l = 4; l >= 1; --l) {
    const int k = 4 - l;
    if (p->wtc_d[k]) {
      WgtcParams q = p->wdp[k];
      q.descs = p->wdd[k];
      q.part = p->wpart;
      launch_wgrad_tc(p->wdA[k], p->wdB[k], q, p->sms, st);
    } else {
      launch_conv(WGRAD_MODE, CEPI_NONE_, s.bf, true, p->dw[k], C, dc[l], dc[l - 1] * 16,
                  nullptr, p->splits_dw[k], p->part, p->pstride_dw[k], s.slope, st);
    }
    if (l >= 2 && p->tct) {
      CtcParams q = p->ddp[k];
      q.descs = p->ddd[k];
      q.wsel = p->b.src_d;
      if (!launch_conv_tc(p->mDd[l - 1], p->aDd[k], q, p->sms, st)) return no_variant(msg);
    } else if (l >= 2) {
      launch_conv(CONVT2_MODE, CEPI_DLRELU_, s.bf, false, p->dd[k], C,
                  2 * B * ds[l - 1] * ds[l - 1], dc[l - 1], nullptr, 1, nullptr, 0, s.slope,
                  st);
    }
  }
  // the generator loss through the discriminator
  launch_logit_back(s.bf, p->tct ? p->tdl_back_g_tc : p->tdl_back_g, C, (int)(8 * d * 16),
                    false, s.slope, st);
  for (int l = 4; l >= 1; --l) {
    if (p->tct && l == 1 && p->scd) {
      CtcParams q = p->gds;
      q.descs = p->gdd[3];
      q.wsel = p->b.src_d;
      if (!launch_conv_tc(p->mDs, p->aGds, q, p->sms, st)) return no_variant(msg);
      launch_scatter_fix(p->gdd[3], p->halo, C, B, CTC_DTANH_CHW, st);
    } else if (p->tct) {
      CtcParams q = p->gdp[4 - l];
      q.descs = p->gdd[4 - l];
      q.wsel = p->b.src_d;
      if (!launch_conv_tc(p->mDd[l - 1], p->aGd[4 - l], q, p->sms, st)) return no_variant(msg);
    } else {
      launch_conv(CONVT2_MODE, l == 1 ? CEPI_DTANH_ : CEPI_DLRELU_, s.bf, false,
                  p->gd[4 - l], C, B * ds[l - 1] * ds[l - 1], dc[l - 1], nullptr, 1, nullptr, 0,
                  s.slope, st);
    }
  }
  // generator backward
  for (int l = 5; l >= 1; --l) {
    const int k = 5 - l;
    if (p->wtc_g[k]) {
      WgtcParams q = p->wgp[k];
      q.descs = p->wgd[k];
      q.part = p->wpart;
      launch_wgrad_tc(p->wgA[k], p->wgB[k], q, p->sms, st);
    } else if (l == 1 && p->g1w) {
      launch_dense1_wgrad_tc(p->mG1w, (const bf16*)p->b.Z, (int64_t)B * s.z, (const bf16*)p->dcb,
                             p->dcb_cell, p->dc1t, p->b.gG + p->b.goff[0], p->b.PGs, B, s.z,
                             gc[1], C, p->err, st);
    } else {
      launch_conv(WGRAD_MODE, CEPI_NONE_, s.bf, true, p->gw[k], C, gc[l - 1], gc[l] * 16,
                  nullptr, p->splits_gw[k], p->part, p->pstride_gw[k], s.slope, st);
    }
    if (l >= 2) {
      if (p->tct) {
        CtcParams q = p->gcp[k];
        q.descs = p->gcd[k];
        q.wsel = p->b.src_g;
        if (!launch_conv_tc(p->mGc[k], p->aGc[k], q, p->sms, st)) return no_variant(msg);
      } else {
        launch_conv(CONV_FWD_MODE, CEPI_NONE_, s.bf, true, p->gdh[k], C,
                    B * gs[l - 1] * gs[l - 1], gc[l - 1], nullptr, 1, nullptr, 0, s.slope, st);
      }
      if (p->tct)
        launch_bn_relu_backward_hwc(p->gbn[k], C, gc[l - 1], p->bnpart, p->bncnt,
                                    (int64_t)B * gs[l - 1] * gs[l - 1] * gc[l - 1], st);
      else
        launch_bn_relu_backward(s.bf, p->gbn[k], C, gc[l - 1], st);
    }
  }
  return check(msg, "DCGAN training step");
}

int dc_eval_launches(const DcPlan* p, int part) {
  if (part == 0) return p->tcg ? 14 + (p->scg ? 2 : 0) : 9;
  return p->eval_launches - 9 + (p->tc ? 1 - p->s.cells : 0);
}

int* dc_error_flag(DcPlan* p) { return p && (p->tc || p->tcg) ? p->err : nullptr; }
int dc_train_launches(const DcPlan* p) { return p->train_launches; }

}  // namespace lipz
