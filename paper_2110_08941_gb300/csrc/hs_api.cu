// C-ABI of libhs: context, Dynamic Partitioning (Algorithm 1) and the synchronous SGD step
// (Section 1, Eq. 1, Section 4.2) over M logical workers on one GPU.
#include <cmath>
#include <cstdlib>
#include <cstdio>
#include <cstring>
#include <string>
#include <vector>

#include "../../include/hs.h"
#include "../../include/hs_debug.h"
#include "common.cuh"
#include "gemm_tc.cuh"
#include "ctx.cuh"

using hs::DevStatus;
using namespace hs;

namespace {

thread_local std::string g_init_error;

hs_status validate_model(const hs_model_desc* m, std::vector<int32_t>* dims, std::string* why) {
  if (!m || !m->dims) { *why = "model or model->dims is NULL"; return HS_ERR_INVALID_ARG; }
  if (m->precision != HS_BF16 && m->precision != HS_FP32_CHECK) { *why = "unknown precision"; return HS_ERR_INVALID_ARG; }
  if (m->sync < HS_SYNC_MEAN || m->sync > HS_SYNC_CP_LITERAL) { *why = "unknown sync mode"; return HS_ERR_INVALID_ARG; }
  if (m->arch == HS_MLP) {
    if (m->n_layers < 1 || m->n_layers > 64) { *why = "n_layers must be in [1, 64]"; return HS_ERR_INVALID_ARG; }
    dims->assign(m->dims, m->dims + m->n_layers + 1);
    for (int32_t d : *dims)
      if (d < 1 || d > (1 << 20)) { *why = "layer widths must be in [1, 2^20]"; return HS_ERR_INVALID_ARG; }
    return HS_OK;
  }
  if (m->arch == HS_CNN) {
    dims->assign(m->dims, m->dims + 7);
    for (int32_t d : *dims)
      if (d < 1 || d > (1 << 16)) { *why = "CNN dims must be in [1, 65536]"; return HS_ERR_INVALID_ARG; }
    return HS_OK;
  }
  *why = "unknown arch";
  return HS_ERR_INVALID_ARG;
}

int64_t mlp_param_count(const std::vector<int32_t>& d) {
  int64_t p = 0;
  for (size_t l = 1; l < d.size(); ++l) p += (int64_t)d[l] * d[l - 1] + d[l];
  return p;
}

int64_t cnn_param_count(const std::vector<int32_t>& d) {
  int64_t p = 0, prev = d[0];
  for (int k = 3; k < 6; ++k) {
    p += (int64_t)d[k] * prev * 9 + d[k];
    prev = d[k];
  }
  p += (int64_t)d[6] * prev + d[6];
  return p;
}

// ------------------------------------------------------------------ tensor-core plans
hs_status build_tc_static(hs_ctx* c) {
  const char* why = nullptr;
  if (!hs::tc_init_driver(&why)) return fail(c, HS_ERR_CUDA, why);
  c->tc_fwd.assign(c->L, hs::TcGemmParams{});
  c->tc_dgrad.assign(c->L, hs::TcGemmParams{});
  for (int l = 0; l < c->L; ++l) {
    const Layer& ly = c->layers[l];
    const bool last = (l == c->L - 1);
    // forward: A = H_l [N, in] (K-major), B = W_l [out, in] (K-major)
    hs::TcGemmParams& f = c->tc_fwd[l];
    std::memset(&f, 0, sizeof(f));
    hs::TcOperand a{reinterpret_cast<const __nv_bfloat16*>(c->d_act[l]), c->N, ly.in, ly.in};
    hs::TcOperand b{c->d_shadow + ly.w_off, ly.out, ly.in, ly.in};
    if (!hs::tc_make_kmajor_map(&f.tmA[0], a, hs::kTcBoxA, &why) ||
        !hs::tc_make_kmajor_map(&f.tmB[0], b, hs::kTcBoxB, &why))
      return fail(c, HS_ERR_CUDA, why);
    f.num_kb[0] = (ly.in + hs::kTcBK - 1) / hs::kTcBK;
    f.groups = 1;
    f.Mdim = c->N;
    f.Ndim = ly.out;
    f.n_store = last ? c->Cp : ly.out;
    f.tiles_m = (c->N + hs::kTcBM - 1) / hs::kTcBM;
    f.tiles_n = (f.n_store + hs::kTcBN - 1) / hs::kTcBN;
    f.epi = last ? hs::kTcEpiBiasF32 : hs::kTcEpiBiasReluBf16;
    if (!last && c->d_relu_bits.size() > (size_t)(l + 1) && c->d_relu_bits[l + 1]) {
      f.relu_bits_out = c->d_relu_bits[l + 1];
      f.bits_ld = c->N;
    }
    f.ew = 4;
    f.D = last ? static_cast<void*>(c->d_logits) : c->d_act[l + 1];
    f.ldd = last ? c->Cp : ly.out;
    f.st = c->d_status;
    if (!hs::tc_make_store_map(&f.tmD[0], f.D, last, c->N, f.n_store, f.ldd, &why)) return fail(c, HS_ERR_CUDA, why);
    if (l == 0) continue;
    // input gradient of layer l: A = delta_l [N, out] (K-major), B = W_l [out, in] (MN-major)
    hs::TcGemmParams& d = c->tc_dgrad[l];
    std::memset(&d, 0, sizeof(d));
    hs::TcOperand da{reinterpret_cast<const __nv_bfloat16*>(c->delta_buf(l)), c->N, ly.out, c->delta_ld(l)};
    hs::TcOperand db{c->d_shadow + ly.w_off, ly.out, ly.in, ly.in};
    if (!hs::tc_make_kmajor_map(&d.tmA[0], da, hs::kTcBoxA, &why) || !hs::tc_make_mnmajor_map(&d.tmB[0], db, &why))
      return fail(c, HS_ERR_CUDA, why);
    d.num_kb[0] = (ly.out + hs::kTcBK - 1) / hs::kTcBK;
    d.groups = 1;
    d.Mdim = c->N;
    d.Ndim = ly.in;
    d.n_store = ly.in;
    d.tiles_m = (c->N + hs::kTcBM - 1) / hs::kTcBM;
    d.tiles_n = (ly.in + hs::kTcBN - 1) / hs::kTcBN;
    d.epi = hs::kTcEpiMaskBf16;
    d.a_mn = 0;
    d.b_mn = 1;
    d.ew = ly.out <= 2048 ? 8 : 4;   // short K: the epilogue outlasts the main loop
    d.D = c->delta_buf(l - 1);
    d.ldd = c->delta_ld(l - 1);
    d.Z = reinterpret_cast<const __nv_bfloat16*>(c->d_act[l]);
    d.ldz = ly.in;
    if (c->d_relu_bits.size() > (size_t)l && c->d_relu_bits[l]) {
      d.relu_bits_in = c->d_relu_bits[l];
      d.bits_ld = c->N;
    }
    d.st = c->d_status;
    if (!hs::tc_make_store_map(&d.tmD[0], d.D, false, c->N, d.n_store, d.ldd, &why)) return fail(c, HS_ERR_CUDA, why);
  }
  return HS_OK;
}

// MMA steps of 16 rows holding data in the last k-block of a K extent of n rows (1..3), or 0 when
// that k-block is full (all four steps, the kernels' straight-line path).
int32_t last_ksteps(int64_t n) {
  const int64_t r = n < 1 ? 0 : ((n - 1) % hs::kTcBK) / 16 + 1;
  return r == hs::kTcBK / 16 ? 0 : (int32_t)r;
}

// The slab-free formulation's weight gradients: one group over all N rows into slab 0.
hs_status build_tc_wgrad_fused(hs_ctx* c) {
  const char* why = nullptr;
  c->tc_wgrad_fused.assign(c->L, hs::TcGemmParams{});
  for (int l = 0; l < c->L; ++l) {
    const Layer& ly = c->layers[l];
    const int ldd_delta = c->delta_ld(l);
    const int out_cols = (l == c->L - 1) ? c->C : ly.out;
    hs::TcGemmParams& w = c->tc_wgrad_fused[l];
    std::memset(&w, 0, sizeof(w));
    hs::TcOperand a{reinterpret_cast<const __nv_bfloat16*>(c->delta_buf(l)), c->N, out_cols, ldd_delta};
    hs::TcOperand b{reinterpret_cast<const __nv_bfloat16*>(c->d_act[l]), c->N, ly.in, ly.in};
    if (!hs::tc_make_mnmajor_map(&w.tmA[0], a, &why) || !hs::tc_make_mnmajor_map(&w.tmB[0], b, &why) ||
        !hs::tc_make_store_map(&w.tmD[0], c->d_slabs + ly.w_off, true, out_cols, ly.in, ly.in, &why))
      return fail(c, HS_ERR_CUDA, why);
    w.num_kb[0] = (c->N + hs::kTcBK - 1) / hs::kTcBK;
    w.groups = 1;
    w.Mdim = out_cols;
    w.Ndim = ly.in;
    w.n_store = ly.in;
    w.epi = hs::kTcEpiStoreF32;
    w.a_mn = 1;
    w.b_mn = 1;
    w.D = c->d_slabs + ly.w_off;
    w.ldd = ly.in;
    w.st = c->d_status;
  }
  return HS_OK;
}

// Per-worker weight gradients depend on the segments, so they are rebuilt on repartition.
hs_status build_tc_wgrad(hs_ctx* c) {
  const char* why = nullptr;
  c->tc_wgrad.assign(c->L, {});
  for (int l = 0; l < c->L; ++l) {
    const Layer& ly = c->layers[l];
    const int ldd_delta = c->delta_ld(l);
    const int out_cols = (l == c->L - 1) ? c->C : ly.out;
    for (int g0 = 0; g0 < c->M; g0 += hs::kTcMaxGroups) {
      const int ng = std::min(hs::kTcMaxGroups, c->M - g0);
      c->tc_wgrad[l].emplace_back();
      hs::TcGemmParams& w = c->tc_wgrad[l].back();
      std::memset(&w, 0, sizeof(w));
      for (int g = 0; g < ng; ++g) {
        const int m = g0 + g;
        const int64_t off = c->offsets[m], n = c->counts[m];
        // A^T: delta_l rows of worker m as [n rows][out cols] (MN-major: out contiguous)
        hs::TcOperand a{reinterpret_cast<const __nv_bfloat16*>(c->delta_buf(l)) + off * ldd_delta, n, out_cols,
                        ldd_delta};
        // B: H_{l-1} rows of worker m as [n rows][in cols] (MN-major: in contiguous)
        hs::TcOperand b{reinterpret_cast<const __nv_bfloat16*>(c->d_act[l]) + off * ly.in, n, ly.in, ly.in};
        float* dg = c->d_slabs + (int64_t)m * c->Ps + ly.w_off;
        if (!hs::tc_make_mnmajor_map(&w.tmA[g], a, &why) || !hs::tc_make_mnmajor_map(&w.tmB[g], b, &why) ||
            !hs::tc_make_store_map(&w.tmD[g], dg, true, out_cols, ly.in, ly.in, &why))
          return fail(c, HS_ERR_CUDA, why);
        w.num_kb[g] = (int32_t)((n + hs::kTcBK - 1) / hs::kTcBK);
        w.last_ksteps[g] = last_ksteps(n);
      }
      w.groups = ng;
      w.Mdim = out_cols;
      w.Ndim = ly.in;
      w.n_store = ly.in;
      w.tiles_m = (out_cols + hs::kTcBM - 1) / hs::kTcBM;
      w.tiles_n = (ly.in + hs::kTcBN - 1) / hs::kTcBN;
      w.epi = hs::kTcEpiStoreF32;
      w.a_mn = 1;
      w.b_mn = 1;
      w.D = c->d_slabs + (int64_t)g0 * c->Ps + ly.w_off;
      w.ldd = ly.in;
      w.d_gstride = c->Ps;
      w.st = c->d_status;
    }
  }
  return HS_OK;
}

// The tile-averaged weight gradients: per layer one launch over all workers (groups), the update
// fused in (launch_tc_wgrad_avg), for layers with at least one 256 x 256 weight tile per SM pair
// (all layers with HS_TILE_AVERAGE=all).  Layers 2..L write their bf16 weights to the second shadow (their
// input-gradient products still read the first); layer 1 writes the first.  theta's maps are bound
// per step (bind_avg_theta).  A layer whose operands the kernel cannot take keeps the slab path.
hs_status build_tc_wgrad_avg(hs_ctx* c) {
  const char* why = nullptr;
  c->tc_wgrad_avg.assign(c->L, hs::TcGemmParams{});
  c->avg_ok.assign(c->L, 0);
  c->avg_theta = nullptr;
  if (!c->tile_avg || c->M > hs::kTcMaxGroups) return HS_OK;
  for (int l = 0; l < c->L; ++l) {
    const Layer& ly = c->layers[l];
    const int ldd_delta = c->delta_ld(l);
    const int out_cols = (l == c->L - 1) ? c->C : ly.out;
    hs::TcGemmParams& w = c->tc_wgrad_avg[l];
    std::memset(&w, 0, sizeof(w));
    bool ok = true;
    for (int m = 0; m < c->M && ok; ++m) {
      const int64_t off = c->offsets[m], n = c->counts[m];
      hs::TcOperand a{reinterpret_cast<const __nv_bfloat16*>(c->delta_buf(l)) + off * ldd_delta, n, out_cols,
                      ldd_delta};
      hs::TcOperand b{reinterpret_cast<const __nv_bfloat16*>(c->d_act[l]) + off * ly.in, n, ly.in, ly.in};
      ok = n >= 1 && hs::tc_make_mnmajor_map(&w.tmA[m], a, &why) && hs::tc_make_mnmajor_map(&w.tmB[m], b, &why);
      w.num_kb[m] = (int32_t)((n + hs::kTcBK - 1) / hs::kTcBK);
      w.last_ksteps[m] = last_ksteps(n);
    }
    ok = ok && c->d_shadow_next && c->d_shadow;
    // One SM pair per 256 x 256 tile of the layer's weights: with fewer tiles than pairs the
    // grouped slab launch (a tile per worker) keeps more of the GPU busy.
    const int64_t tiles = ((out_cols + 255) / 256) * (int64_t)((ly.in + 255) / 256);
    if (!c->tile_avg_all && tiles < c->num_sms / 2) ok = false;
    w.groups = c->M;
    w.Mdim = out_cols;
    w.Ndim = ly.in;
    w.n_store = ly.in;
    w.epi = hs::kTcEpiAvgUpdate;
    w.a_mn = 1;
    w.b_mn = 1;
    w.wavg = c->d_w;
    w.st = c->d_status;
    c->avg_ok[l] = ok ? 1 : 0;
  }
  return HS_OK;
}

// Point the tile-averaged launches' update maps at `params`, the bf16 copies and (with the
// momentum recipe) the momentum buffer, in the box shapes of the update in use (a layer whose
// weights TMA cannot address, e.g. not 16-byte aligned, falls back to the slab path).
void bind_avg_theta(hs_ctx* c, float* params) {
  const bool recipe = c->opt_recipe && c->d_mom;
  if (c->avg_theta == params && c->avg_recipe == recipe) return;
  const char* why = nullptr;
  for (int l = 0; l < c->L; ++l) {
    if (!c->avg_ok[l]) continue;
    const Layer& ly = c->layers[l];
    hs::TcGemmParams& w = c->tc_wgrad_avg[l];
    __nv_bfloat16* shadow = (l > 0 ? c->d_shadow_next : c->d_shadow) + ly.w_off;
    bool ok;
    if (recipe)
      ok = hs::tc_make_store_map_16(&w.tmT, params + ly.w_off, true, w.Mdim, ly.in, ly.in, &why) &&
           hs::tc_make_store_map_16(&w.tmM, c->d_mom + ly.w_off, true, w.Mdim, ly.in, ly.in, &why) &&
           hs::tc_make_store_map_16(&w.tmS, shadow, false, w.Mdim, ly.in, ly.in, &why);
    else
      ok = hs::tc_make_store_map(&w.tmT, params + ly.w_off, true, w.Mdim, ly.in, ly.in, &why) &&
           hs::tc_make_store_map_bf16_32(&w.tmS, shadow, w.Mdim, ly.in, ly.in, &why);
    if (!ok) c->avg_ok[l] = 0;
    w.recipe = recipe ? 1 : 0;
  }
  c->avg_theta = params;
  c->avg_recipe = recipe;
}

void compute_weights(hs_ctx* c) {
  c->weights.assign(c->M, 0.0);
  for (int m = 0; m < c->M; ++m) {
    if (c->sync == HS_SYNC_MEAN) c->weights[m] = 1.0 / c->M;
    else if (c->sync == HS_SYNC_CP_WEIGHTED) c->weights[m] = (double)c->counts[m] / (double)c->N;
    else c->weights[m] = c->cp_norm[m] / c->M;
  }
}

// Apply a new partition (sizes already validated) and push it to the device on `s`.
void invalidate_step_graphs(hs_ctx* c);

hs_status apply_partition(hs_ctx* c, const std::vector<int32_t>& sizes, const std::vector<double>& cpn,
                          int32_t* index_map_out, cudaStream_t s) {
  const bool changed = (sizes != c->counts);
  c->cp_norm = cpn;
  if (changed) {
    invalidate_step_graphs(c);   // the plans below change what a step enqueues
    c->counts = sizes;
    c->offsets.assign(c->M + 1, 0);
    for (int m = 0; m < c->M; ++m) c->offsets[m + 1] = c->offsets[m] + sizes[m];
    ++c->version;
  }
  compute_weights(c);
  std::vector<float> wf(c->weights.begin(), c->weights.end());
  HS_CUDA(c, cudaMemcpyAsync(c->d_w, wf.data(), sizeof(float) * c->M, cudaMemcpyHostToDevice, s));
  std::vector<int4> chunks;
  std::vector<int32_t> chunk_begin;
  if (changed) {
    HS_CUDA(c, cudaMemcpyAsync(c->d_offsets, c->offsets.data(), sizeof(int32_t) * (c->M + 1),
                               cudaMemcpyHostToDevice, s));
    const int R = hs::bias_grad_chunk_rows();
    for (int m = 0; m < c->M; ++m) {
      chunk_begin.push_back((int32_t)chunks.size());
      for (int r = c->offsets[m]; r < c->offsets[m + 1]; r += R)
        chunks.push_back(make_int4(m, r, std::min(r + R, c->offsets[m + 1]), 0));
    }
    chunk_begin.push_back((int32_t)chunks.size());
    c->n_bg_chunks = (int)chunks.size();
    HS_CUDA(c, cudaMemcpyAsync(c->d_bg_chunks, chunks.data(), sizeof(int4) * chunks.size(), cudaMemcpyHostToDevice, s));
    HS_CUDA(c, cudaMemcpyAsync(c->d_bg_chunk_begin, chunk_begin.data(), sizeof(int32_t) * chunk_begin.size(),
                               cudaMemcpyHostToDevice, s));
  }
  if (changed || index_map_out) {
    hs::launch_partition_scatter(c->d_offsets, c->M, c->N, c->d_index_map, c->d_scale, index_map_out, s);
    HS_CUDA(c, cudaGetLastError());
  }
  if (c->d_scale_fused) {
    hs::launch_scale_by_weight(c->d_index_map, c->d_scale, c->d_w, c->N, c->d_scale_fused, s);
    HS_CUDA(c, cudaGetLastError());
  }
  // the host vectors above are pageable: make sure the copies consumed them before they change
  HS_CUDA(c, cudaStreamSynchronize(s));
  if (changed && c->arch == HS_MLP && c->precision == HS_BF16) {
    hs_status st = build_tc_wgrad(c);
    if (st == HS_OK) st = build_tc_wgrad_avg(c);
    if (st != HS_OK) return st;
  }
  if (changed && c->arch == HS_CNN) {
    // per-layer row offsets (a sample is Ho*Wo rows of a conv product, one row of the fc product)
    for (int k = 0; k < 4; ++k) {
      const int64_t rps = c->cnn_chunks[k].rows_per_sample;
      // conv layers have many narrow rows: longer chunks keep the per-worker combine short
      const int R = rps > 1 ? 16 * hs::bias_grad_chunk_rows() : hs::bias_grad_chunk_rows();
      std::vector<int32_t> ro(c->M + 1), begin;
      std::vector<int4> chunks;
      for (int m = 0; m <= c->M; ++m) ro[m] = (int32_t)(c->offsets[m] * rps);
      for (int m = 0; m < c->M; ++m) {
        begin.push_back((int32_t)chunks.size());
        for (int64_t r = ro[m]; r < ro[m + 1]; r += R)
          chunks.push_back(make_int4(m, (int)r, (int)std::min<int64_t>(r + R, ro[m + 1]), 0));
      }
      begin.push_back((int32_t)chunks.size());
      c->cnn_chunks[k].n = (int)chunks.size();
      HS_CUDA(c, cudaMemcpy(c->d_row_off[k], ro.data(), sizeof(int32_t) * ro.size(), cudaMemcpyHostToDevice));
      HS_CUDA(c, cudaMemcpy(c->cnn_chunks[k].d_chunks, chunks.data(), sizeof(int4) * chunks.size(),
                            cudaMemcpyHostToDevice));
      HS_CUDA(c, cudaMemcpy(c->cnn_chunks[k].d_begin, begin.data(), sizeof(int32_t) * begin.size(),
                            cudaMemcpyHostToDevice));
    }
    if (c->precision == HS_BF16) {
      hs_status st = cnn_build_partition_plans(c);
      if (st != HS_OK) return st;
    }
  }
  return HS_OK;
}

void fill_partition_view(const hs_ctx* c, hs_partition_t* out) {
  if (!out) return;
  out->M = c->M;
  out->N = c->N;
  out->counts_host = c->counts.data();
  out->offsets_host = c->offsets.data();
  out->index_map_dev = c->d_index_map;
  out->weights_host = c->weights.data();
  out->cp_host = c->cp_norm.data();
  out->version = c->version;
}


void free_all(hs_ctx* c) {
  auto f = [](void* p) { if (p) cudaFree(p); };
  f(c->d_offsets); f(c->d_index_map); f(c->d_scale); f(c->d_w);
  f(c->d_bg_chunks); f(c->d_bg_chunk_begin); f(c->d_bg_partial);
  f(c->d_scale_fused); f(c->d_all_off); f(c->d_w_one); f(c->all_rows.d_chunks); f(c->all_rows.d_begin);
  for (int k = 0; k < 3; ++k) { f(c->d_col[k]); f(c->d_cact[k]); f(c->d_dA[k]); }
  f(c->d_pooled); f(c->d_dpooled); f(c->d_dcol);
  for (int k = 0; k < 3; ++k) f(c->d_wperm[k]);
  f(c->d_ones);
  for (int k = 0; k < 3; ++k) f(c->d_wsub[k]);
  for (int k = 0; k < 4; ++k) {
    f(c->d_row_off[k]); f(c->cnn_chunks[k].d_chunks); f(c->cnn_chunks[k].d_begin);
    f(c->cnn_wgrad[k].d_partial); f(c->cnn_wgrad[k].d_chunk_begin);
  }
  for (void* p : c->d_act) f(p);
  f(c->d_logits); f(c->d_delta[0]); f(c->d_delta[1]); f(c->d_ce); f(c->d_lm); f(c->d_status); f(c->d_ticket);
  for (uint64_t* b : c->d_relu_bits) f(b);
  f(c->d_slabs); f(c->d_shadow); f(c->d_shadow_next); f(c->d_gdebug); f(c->d_xstage); f(c->d_ystage); f(c->d_mom);
  if (c->h_status) cudaFreeHost(c->h_status);
  for (auto& r : c->pending) {
    cudaEventDestroy(r.a);
    cudaEventDestroy(r.b);
  }
  for (cudaEvent_t e : c->event_pool) cudaEventDestroy(e);
  for (int k = 0; k < 2; ++k) {
    f(c->d_xslot[k]); f(c->d_yslot[k]);
    if (c->slot_staged[k]) cudaEventDestroy(c->slot_staged[k]);
    if (c->slot_consumed[k]) cudaEventDestroy(c->slot_consumed[k]);
  }
  for (cudaEvent_t e : c->upd_ready) if (e) cudaEventDestroy(e);
  if (c->upd_done) cudaEventDestroy(c->upd_done);
  if (c->dgrad_done) cudaEventDestroy(c->dgrad_done);
  if (c->upd_stream) cudaStreamDestroy(c->upd_stream);
  f(c->d_lr);
  if (c->cap_stream) cudaStreamDestroy(c->cap_stream);
}

bool is_device_ptr(const void* p) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged;
}

// ------------------------------------------------------------------ the MLP step
hs_status mlp_step_fp32(hs_ctx* c, float* params, const float* x, const int32_t* y, cudaStream_t s) {
  const int L = c->L;
  std::vector<const float*> act(L);
  act[0] = x;
  for (int l = 1; l < L; ++l) act[l] = reinterpret_cast<const float*>(c->d_act[l]);
  {
    // per-worker forward: the segments share theta, so all rows go through one product per layer
    PhaseScope ph(c, HS_PHASE_FORWARD, s);
    for (int l = 0; l < L; ++l) {
      const Layer& ly = c->layers[l];
      const bool last = (l == L - 1);
      hs::GemmF32Args g{};
      g.A = act[l]; g.a_sm = ly.in; g.a_sk = 1;
      g.B = params + ly.w_off; g.b_sk = 1; g.b_sn = ly.in;
      g.C = last ? c->d_logits : reinterpret_cast<float*>(c->d_act[l + 1]);
      g.ldc = last ? c->Cp : ly.out;
      g.Mdim = c->N; g.Ndim = ly.out; g.Kdim = ly.in;
      g.epi = last ? hs::kEpiBias : hs::kEpiBiasRelu;
      g.bias = params + ly.b_off;
      hs::launch_gemm_f32(g, s);
      ph.launched();
    }
  }
  const bool loss_bias = !c->fused_sync && c->C <= hs::loss_bias_max_width();
  {
    PhaseScope ph(c, HS_PHASE_LOSS, s);
    hs::launch_softmax_xent(c->d_logits, c->Cp, y, c->fused_sync ? c->d_scale_fused : c->d_scale, c->N, c->C,
                            c->delta_buf(L - 1), c->Cp, false,
                            c->d_ce, c->d_status, s);
    hs::launch_loss_reduce(c->d_ce, c->d_offsets, c->M, c->d_w, c->d_lm, c->d_status, c->d_ticket, s);
    ph.launched(2);
  }
  for (int l = L - 1; l >= 0; --l) {
    const Layer& ly = c->layers[l];
    const int ldd = c->delta_ld(l);
    const float* delta = reinterpret_cast<const float*>(c->delta_buf(l));
    const int out_cols = (l == L - 1) ? c->C : ly.out;
    {
      // per-worker weight gradient G_m[W_l] = delta_l[seg_m]^T H_{l-1}[seg_m]
      PhaseScope ph(c, HS_PHASE_WGRAD, s);
      hs::GemmF32Args w{};
      w.A = delta; w.a_sm = 1; w.a_sk = ldd;
      w.B = act[l]; w.b_sk = ly.in; w.b_sn = 1;
      w.C = c->d_slabs + ly.w_off; w.ldc = ly.in;
      w.Mdim = out_cols; w.Ndim = ly.in; w.Kdim = 0;
      w.epi = hs::kEpiStore;
      w.k_offsets = c->fused_sync ? c->d_all_off : c->d_offsets;
      w.groups = c->fused_sync ? 1 : c->M;
      w.c_gstride = c->Ps;
      hs::launch_gemm_f32(w, s);
      ph.launched();
    }
    {
      PhaseScope ph(c, HS_PHASE_BIASGRAD, s);
      hs::launch_bias_grad(delta, false, ldd, out_cols, c->fused_sync ? c->d_all_off : c->d_offsets,
                           c->fused_sync ? 1 : c->M, c->d_slabs, c->Ps, ly.b_off, s);
      ph.launched();
    }
    if (l > 0) {
      PhaseScope ph(c, HS_PHASE_DGRAD, s);
      hs::GemmF32Args d{};
      d.A = delta; d.a_sm = ldd; d.a_sk = 1;
      d.B = params + ly.w_off; d.b_sk = ly.in; d.b_sn = 1;
      d.C = reinterpret_cast<float*>(c->delta_buf(l - 1)); d.ldc = c->delta_ld(l - 1);
      d.Mdim = c->N; d.Ndim = ly.in; d.Kdim = out_cols;
      d.epi = hs::kEpiMask; d.Z = act[l]; d.ldz = ly.in;
      hs::launch_gemm_f32(d, s);
      ph.launched();
    }
  }
  return HS_OK;
}

// theta <- theta - lr * sum_m w_m G_m over layer l's parameter range [W_l, b_l] (Section 1).
// The update of layer l's parameter range [W_l, b_l]; the new bf16 weights go to `shadow` (the
// step's shadow, or the second shadow while input-gradient products still read the first).
void update_layer_range(hs_ctx* c, float* params, int l, float lr, const float* lr_dev, cudaStream_t s,
                        int blocks_per_sm, __nv_bfloat16* shadow = nullptr) {
  const int64_t start = c->layers[l].w_off;
  const int64_t end = (l + 1 < c->L) ? c->layers[l + 1].w_off : c->P;
  if (!shadow) shadow = c->d_shadow;
  PhaseScope ph(c, HS_PHASE_UPDATE, s);
  hs::UpdateRecipe r{c->opt_recipe ? c->d_mom + start : nullptr, c->opt_momentum, c->opt_weight_decay,
                     c->mom_valid ? 0 : 1};
  hs::launch_reduce_update(params + start, c->d_slabs + start, c->Ps, c->fused_sync ? 1 : c->M,
                           c->fused_sync ? c->d_w_one : c->d_w, lr, end - start,
                           shadow + start, c->debug ? c->d_gdebug + start : nullptr, c->num_sms, s,
                           blocks_per_sm, c->opt_recipe ? &r : nullptr, lr_dev);
  ph.launched();
}

// theta <- theta - lr * sum_m w_m G_m over [start, end) of the slabs (the bias range of a layer whose
// weights the tile-averaged launch updated; the momentum recipe as in the rest of the update),
// bf16 copy into `shadow`.
void update_range(hs_ctx* c, float* params, int64_t start, int64_t end, float lr, const float* lr_dev,
                  cudaStream_t s, __nv_bfloat16* shadow) {
  PhaseScope ph(c, HS_PHASE_UPDATE, s);
  hs::UpdateRecipe r{c->opt_recipe ? c->d_mom + start : nullptr, c->opt_momentum, c->opt_weight_decay,
                     c->mom_valid ? 0 : 1};
  hs::launch_reduce_update(params + start, c->d_slabs + start, c->Ps, c->M, c->d_w, lr, end - start, shadow + start,
                           nullptr, c->num_sms, s, 1, c->opt_recipe ? &r : nullptr, lr_dev);
  ph.launched();
}

hs_status mlp_step_bf16(hs_ctx* c, float* params, const float* x, const int32_t* y, float lr, const float* lr_dev,
                        cudaStream_t s) {
  const int L = c->L;
  {
    PhaseScope ph(c, HS_PHASE_CAST, s);
    hs::launch_cast_f32_bf16(x, reinterpret_cast<__nv_bfloat16*>(c->d_act[0]), (int64_t)c->N * c->layers[0].in, s);
    ph.launched();
  }
  {
    PhaseScope ph(c, HS_PHASE_FORWARD, s);
    for (int l = 0; l < L; ++l) {
      hs::TcGemmParams& f = c->tc_fwd[l];
      f.bias = params + c->layers[l].b_off;
      cudaError_t e = hs::launch_tc_gemm(f, c->num_sms, s);
      if (e != cudaSuccess) return cuda_fail(c, e, "forward GEMM launch");
      ph.launched();
    }
  }
  const bool loss_bias = !c->fused_sync && c->C <= hs::loss_bias_max_width();
  {
    PhaseScope ph(c, HS_PHASE_LOSS, s);
    __nv_bfloat16* delta_out = reinterpret_cast<__nv_bfloat16*>(c->delta_buf(L - 1));
    if (loss_bias && hs::softmax_loss_bias_ok(c->C, c->Cp, c->delta_ld(L - 1))) {
      // softmax, loss reduction and the output layer's bias gradients in one launch
      hs::launch_softmax_loss_bias(c->d_logits, c->Cp, y, c->d_scale, c->C, delta_out, c->delta_ld(L - 1), c->d_ce,
                                   c->d_offsets, c->M, c->d_w, c->d_lm, c->d_status, c->d_ticket, c->d_slabs, c->Ps,
                                   c->layers[L - 1].b_off, s);
      ph.launched();
    } else {
      hs::launch_softmax_xent(c->d_logits, c->Cp, y, c->fused_sync ? c->d_scale_fused : c->d_scale, c->N, c->C,
                              c->delta_buf(L - 1), c->Cp, true,
                              c->d_ce, c->d_status, s);
      if (loss_bias)   // the output layer's bias gradients in the same launch
        hs::launch_loss_bias_reduce(c->d_ce, c->d_offsets, c->M, c->d_w, c->d_lm, c->d_status, c->d_ticket,
                                    delta_out, c->delta_ld(L - 1), c->C, c->d_slabs, c->Ps, c->layers[L - 1].b_off, s);
      else
        hs::launch_loss_reduce(c->d_ce, c->d_offsets, c->M, c->d_w, c->d_lm, c->d_status, c->d_ticket, s);
      ph.launched(2);
    }
  }
  // Per-worker weight gradients averaged tile by tile in tensor memory, the update fused in: the
  // default where the layer's operands allow it; debug read-back, the slab-free formulation and
  // the momentum recipe take the slab path.
  const bool avg = c->tile_avg && !c->fused_sync && !c->debug;
  if (avg) bind_avg_theta(c, params);
  c->tile_step = false;
  for (int l = 0; l < L && avg; ++l) c->tile_step = c->tile_step || c->avg_ok[l];
  bool side = false;   // work queued on the update stream this step
  for (int l = L - 1; l >= 0; --l) {
    const Layer& ly = c->layers[l];
    const bool tile = avg && c->avg_ok[l];
    __nv_bfloat16* shadow_l = (l > 0 && c->d_shadow_next) ? c->d_shadow_next : c->d_shadow;
    {
      PhaseScope ph(c, HS_PHASE_WGRAD, s);
      if (tile) {
        hs::TcGemmParams& w = c->tc_wgrad_avg[l];
        w.lr = lr;
        w.lr_dev = lr_dev;
        w.mu = c->opt_momentum;
        w.wd = c->opt_weight_decay;
        w.first = c->mom_valid ? 0 : 1;
        cudaError_t e = hs::launch_tc_wgrad_avg(w, c->num_sms, s);
        if (e != cudaSuccess) return cuda_fail(c, e, "weight-gradient GEMM launch");
        ph.launched();
      } else if (c->fused_sync) {
        cudaError_t e = hs::launch_tc_gemm(c->tc_wgrad_fused[l], c->num_sms, s);
        if (e != cudaSuccess) return cuda_fail(c, e, "weight-gradient GEMM launch");
        ph.launched();
      } else {
        for (const hs::TcGemmParams& w : c->tc_wgrad[l]) {
          cudaError_t e = hs::launch_tc_gemm(w, c->num_sms, s);
          if (e != cudaSuccess) return cuda_fail(c, e, "weight-gradient GEMM launch");
          ph.launched();
        }
      }
    }
    if (!(loss_bias && l == L - 1)) {
      PhaseScope ph(c, HS_PHASE_BIASGRAD, s);
      const int out_cols = (l == L - 1) ? c->C : ly.out;
      const hs::ChunkTable* ct = nullptr;
      hs::ChunkTable per_worker;
      per_worker.d_chunks = c->d_bg_chunks;
      per_worker.d_begin = c->d_bg_chunk_begin;
      per_worker.n = c->n_bg_chunks;
      ct = c->fused_sync ? &c->all_rows : &per_worker;
      hs::launch_bias_grad_bf16(reinterpret_cast<const __nv_bfloat16*>(c->delta_buf(l)), c->delta_ld(l), out_cols,
                                ct->d_chunks, ct->n, ct->d_begin, c->fused_sync ? 1 : c->M, c->d_bg_partial,
                                c->d_slabs, c->Ps, ly.b_off, s);
      ph.launched(2);
    }
    if (tile) {
      // the bias range's update (its weights were updated inside the weight-gradient launch)
      const int64_t end = (l + 1 < L) ? c->layers[l + 1].w_off : c->P;
      update_range(c, params, ly.b_off, end, lr, lr_dev, s, shadow_l);
    } else if (c->overlap_update) {
      // Layer l's slabs are complete: its update runs beside the remaining (tensor-core bound)
      // backward products.  Its input-gradient product (next, on the step's stream) still reads
      // W_l's bf16 weights, so layers 2..L write theirs to the second shadow, copied over the
      // first once the last input-gradient product is done; layer 1 has none and writes in place.
      HS_CUDA(c, cudaEventRecord(c->upd_ready[l], s));
      HS_CUDA(c, cudaStreamWaitEvent(c->upd_stream, c->upd_ready[l], 0));
      update_layer_range(c, params, l, lr, lr_dev, c->upd_stream, l == 0 ? 4 : 1, shadow_l);
      side = true;
    } else {
      update_layer_range(c, params, l, lr, lr_dev, s, 4, shadow_l);
    }
    if (l > 0) {
      PhaseScope ph(c, HS_PHASE_DGRAD, s);
      cudaError_t e = hs::launch_tc_gemm(c->tc_dgrad[l], c->num_sms, s);
      if (e != cudaSuccess) return cuda_fail(c, e, "input-gradient GEMM launch");
      ph.launched();
    }
    if (l == 1 && c->d_shadow_next) {
      // The last input-gradient product has read the first shadow: the second shadow's ranges
      // (layers 2..L) go over it, on the copy engine beside layer 1's weight gradient.
      const int64_t w1 = c->layers[1].w_off;
      HS_CUDA(c, cudaEventRecord(c->dgrad_done, s));
      HS_CUDA(c, cudaStreamWaitEvent(c->upd_stream, c->dgrad_done, 0));
      HS_CUDA(c, cudaMemcpyAsync(c->d_shadow + w1, c->d_shadow_next + w1, sizeof(__nv_bfloat16) * (c->P - w1),
                                 cudaMemcpyDeviceToDevice, c->upd_stream));
      side = true;
    }
  }
  if (side) {
    HS_CUDA(c, cudaEventRecord(c->upd_done, c->upd_stream));
    HS_CUDA(c, cudaStreamWaitEvent(s, c->upd_done, 0));
  }
  return HS_OK;
}

// The step's kernels after the input handling: per-worker forward and backward passes, the
// synchronisation and the update.  lr_dev: non-null when the learning rate is read from device
// memory (a step captured into a graph).
hs_status step_body(hs_ctx* c, float* params, const float* xd, const int32_t* yd, float lr, const float* lr_dev,
                    cudaStream_t s) {
  const bool mlp_bf16 = (c->arch == HS_MLP && c->precision == HS_BF16);
  hs_status st = c->arch == HS_CNN ? cnn_step(c, params, xd, yd, s)
                 : mlp_bf16        ? mlp_step_bf16(c, params, xd, yd, lr, lr_dev, s)
                                   : mlp_step_fp32(c, params, xd, yd, s);
  if (st != HS_OK) return st;
  if (hs::cnn_fused_update(c)) return hs::launch_cnn_update(c, params, lr, lr_dev, s);
  if (!mlp_bf16) {
    PhaseScope ph(c, HS_PHASE_UPDATE, s);
    hs::UpdateRecipe r{c->d_mom, c->opt_momentum, c->opt_weight_decay, c->mom_valid ? 0 : 1};
    hs::launch_reduce_update(params, c->d_slabs, c->Ps, c->fused_sync ? 1 : c->M,
                             c->fused_sync ? c->d_w_one : c->d_w, lr, c->P,
                             c->precision == HS_BF16 ? c->d_shadow : nullptr, c->debug ? c->d_gdebug : nullptr,
                             c->num_sms, s, 4, c->opt_recipe ? &r : nullptr, lr_dev);
    ph.launched();
  }
  return HS_OK;
}

constexpr size_t kMaxStepGraphs = 4;

void destroy_step_graph(hs_ctx::StepGraph& g) {
  if (g.exec) cudaGraphExecDestroy(g.exec);   // an in-flight replay is freed on completion
  if (g.graph) cudaGraphDestroy(g.graph);
  g.exec = nullptr;
  g.graph = nullptr;
}

// Every captured step is stale once plans, flags or the optimizer change.
void invalidate_step_graphs(hs_ctx* c) {
  for (auto& g : c->graphs) destroy_step_graph(g);
  c->graphs.clear();
  c->graph_warm = false;
}

void disable_step_graphs(hs_ctx* c) {
  invalidate_step_graphs(c);
  c->graph_on = false;
  cudaGetLastError();
}

// Capture the step for key `k` on the context's capture stream (nothing runs), instantiate it and
// note its launches per phase and its profile event nodes.  On any failure the context falls back
// to eager steps for good (returns false, *st = HS_OK) unless the step itself failed (*st).
bool capture_step(hs_ctx* c, hs_ctx::StepGraph& k, float* params, const float* xd, const int32_t* yd, float lr,
                  hs_status* st) {
  *st = HS_OK;
  if (!c->d_lr && dalloc(c, &c->d_lr, sizeof(float)) != HS_OK) return false;
  if (!c->cap_stream && cudaStreamCreateWithFlags(&c->cap_stream, cudaStreamNonBlocking) != cudaSuccess) return false;
  int64_t before[HS_PHASE_COUNT];
  for (int i = 0; i < HS_PHASE_COUNT; ++i) before[i] = c->launches[i];
  const size_t pend0 = c->pending.size();
  if (cudaStreamBeginCapture(c->cap_stream, cudaStreamCaptureModeRelaxed) != cudaSuccess) return false;
  c->capturing = true;
  hs_status body = step_body(c, params, xd, yd, lr, c->d_lr, c->cap_stream);
  c->capturing = false;
  cudaGraph_t graph = nullptr;
  const cudaError_t end = cudaStreamEndCapture(c->cap_stream, &graph);
  for (int i = 0; i < HS_PHASE_COUNT; ++i) {
    k.launches[i] = c->launches[i] - before[i];
    c->launches[i] = before[i];
  }
  std::vector<hs_ctx::Rec> recs(c->pending.begin() + (std::ptrdiff_t)pend0, c->pending.end());
  c->pending.resize(pend0);
  for (auto& r : recs) {   // nodes of the graph refer to them; replays swap in fresh events
    c->event_pool.push_back(r.a);
    c->event_pool.push_back(r.b);
  }
  if (body != HS_OK || end != cudaSuccess || !graph) {
    if (graph) cudaGraphDestroy(graph);
    *st = body;
    return false;
  }
  cudaGraphExec_t exec = nullptr;
  if (cudaGraphInstantiate(&exec, graph, 0) != cudaSuccess) {
    cudaGraphDestroy(graph);
    return false;
  }
  if (!recs.empty()) {
    size_t n = 0;
    cudaGraphGetNodes(graph, nullptr, &n);
    std::vector<cudaGraphNode_t> nodes(n);
    if (n) cudaGraphGetNodes(graph, nodes.data(), &n);
    std::vector<std::pair<cudaEvent_t, cudaGraphNode_t>> by_event;
    for (cudaGraphNode_t nd : nodes) {
      cudaGraphNodeType t;
      cudaEvent_t ev = nullptr;
      if (cudaGraphNodeGetType(nd, &t) == cudaSuccess && t == cudaGraphNodeTypeEventRecord &&
          cudaGraphEventRecordNodeGetEvent(nd, &ev) == cudaSuccess)
        by_event.push_back({ev, nd});
    }
    auto node_of = [&](cudaEvent_t e) -> cudaGraphNode_t {
      for (auto& pr : by_event)
        if (pr.first == e) return pr.second;
      return nullptr;
    };
    for (auto& r : recs) {
      cudaGraphNode_t a = node_of(r.a), b = node_of(r.b);
      if (!a || !b) {   // the profile would miss phases: replay without profile is not what was asked
        cudaGraphExecDestroy(exec);
        cudaGraphDestroy(graph);
        return false;
      }
      k.phase_nodes.push_back({r.phase, a, b});
    }
  }
  k.graph = graph;
  k.exec = exec;
  return true;
}

// One step through the graph cache: eager until a step has run since the last invalidation, then
// the key's graph (captured on first use), launched after the learning rate is written to d_lr.
hs_status step_via_graph(hs_ctx* c, float* params, const float* xd, const int32_t* yd, float lr, cudaStream_t s) {
  if (!c->graph_warm) {
    hs_status st = step_body(c, params, xd, yd, lr, nullptr, s);
    if (st == HS_OK) c->graph_warm = true;
    return st;
  }
  hs_ctx::StepGraph* g = nullptr;
  for (auto& e : c->graphs)
    if (e.params == params && e.x == xd && e.y == yd && e.mom_valid == c->mom_valid && e.profiling == c->profiling)
      g = &e;
  if (!g) {
    hs_ctx::StepGraph k;
    k.params = params;
    k.x = xd;
    k.y = yd;
    k.mom_valid = c->mom_valid;
    k.profiling = c->profiling;
    hs_status st = HS_OK;
    if (!capture_step(c, k, params, xd, yd, lr, &st)) {
      if (st != HS_OK) return st;
      disable_step_graphs(c);
      return step_body(c, params, xd, yd, lr, nullptr, s);
    }
    if (c->graphs.size() >= kMaxStepGraphs) {
      size_t lru = 0;
      for (size_t i = 1; i < c->graphs.size(); ++i)
        if (c->graphs[i].last_use < c->graphs[lru].last_use) lru = i;
      destroy_step_graph(c->graphs[lru]);
      c->graphs.erase(c->graphs.begin() + (std::ptrdiff_t)lru);
    }
    c->graphs.push_back(std::move(k));
    g = &c->graphs.back();
  }
  g->last_use = ++c->graph_clock;
  hs::launch_set_scalar(c->d_lr, lr, s);
  c->launches[HS_PHASE_UPDATE] += 1;
  for (auto& pn : g->phase_nodes) {
    cudaEvent_t a = c->take_event(), b = c->take_event();
    if (!a || !b) return fail(c, HS_ERR_CUDA, "profile events");
    HS_CUDA(c, cudaGraphExecEventRecordNodeSetEvent(g->exec, pn.a, a));
    HS_CUDA(c, cudaGraphExecEventRecordNodeSetEvent(g->exec, pn.b, b));
    c->pending.push_back({pn.phase, a, b});
  }
  HS_CUDA(c, cudaGraphLaunch(g->exec, s));
  for (int i = 0; i < HS_PHASE_COUNT; ++i) c->launches[i] += g->launches[i];
  return HS_OK;
}

}  // namespace

void hs::set_init_error(const char* msg) { g_init_error = msg ? msg : ""; }

// ====================================================================== C ABI
extern "C" {

const char* hs_status_string(hs_status s) {
  switch (s) {
    case HS_OK: return "HS_OK";
    case HS_ERR_INVALID_ARG: return "HS_ERR_INVALID_ARG";
    case HS_ERR_CUDA: return "HS_ERR_CUDA";
    case HS_ERR_OOM: return "HS_ERR_OOM";
    case HS_ERR_UNSUPPORTED: return "HS_ERR_UNSUPPORTED";
    case HS_ERR_DEVICE_CHECK: return "HS_ERR_DEVICE_CHECK";
  }
  return "HS_ERR_UNKNOWN";
}

const char* hs_last_error(const hs_ctx* ctx) { return ctx ? ctx->err.c_str() : ""; }
const char* hs_last_init_error(void) { return g_init_error.c_str(); }

hs_status hs_param_count(const hs_model_desc* model, int64_t* P) {
  std::vector<int32_t> dims;
  std::string why;
  if (!P) return HS_ERR_INVALID_ARG;
  hs_status st = validate_model(model, &dims, &why);
  if (st != HS_OK) return st;
  *P = model->arch == HS_MLP ? mlp_param_count(dims) : cnn_param_count(dims);
  return HS_OK;
}

hs_status hs_init(const hs_model_desc* model, int32_t M, const double* compute_weights, int32_t global_batch,
                  hs_ctx** out) {
  g_init_error.clear();
  if (!out) return fail(nullptr, HS_ERR_INVALID_ARG, "out is NULL");
  *out = nullptr;
  std::vector<int32_t> dims;
  std::string why;
  hs_status st = validate_model(model, &dims, &why);
  if (st != HS_OK) return fail(nullptr, st, why);
  if (M < 1 || M > hs::kMaxWorkers) return fail(nullptr, HS_ERR_INVALID_ARG, "M must be in [1, 1024]");
  if (global_batch < M) return fail(nullptr, HS_ERR_INVALID_ARG, "global_batch must be >= M");

  std::vector<double> cp(M, 1.0);
  if (compute_weights) cp.assign(compute_weights, compute_weights + M);
  std::vector<int32_t> sizes(M);
  std::vector<double> cpn(M);
  const char* pwhy = nullptr;
  st = hs::partition_sizes_impl(M, global_batch, cp.data(), sizes.data(), cpn.data(), &pwhy);
  if (st != HS_OK) return fail(nullptr, st, std::string("compute_weights: ") + pwhy);

  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail(nullptr, HS_ERR_CUDA, std::string("no CUDA device: ") + cudaGetErrorString(e));
  cudaDeviceProp prop;
  e = cudaGetDeviceProperties(&prop, dev);
  if (e != cudaSuccess) return fail(nullptr, HS_ERR_CUDA, cudaGetErrorString(e));
  if (!(prop.major == 10 && prop.minor == 3))
    return fail(nullptr, HS_ERR_UNSUPPORTED, "libhs is built for sm_103a (compute capability 10.3) only");

  hs_ctx* c = new hs_ctx();
  c->device = dev;
  c->num_sms = prop.multiProcessorCount;
  c->arch = model->arch;
  c->precision = model->precision;
  c->sync = model->sync;
  c->dims = dims;
  c->M = M;
  c->N = global_batch;
  c->L = model->arch == HS_MLP ? model->n_layers : 0;
  // The step's own graph pays where launches outlast the GPU work; a step of more than 1e11
  // parameter-samples (P * N: the 4096-8192-8192-1000 workload's 1.8e12 is 5.6 ms of GPU work for
  // about 0.1 ms of host launches) keeps eager launches.  HS_STEP_GRAPH=0 / =1 force either.
  const char* cf = getenv("HS_CNN_FUSED_UPDATE");
  c->cnn_fuse_update = !(cf && !strcmp(cf, "0"));
  const char* sp = getenv("HS_SUBPIXEL");
  c->subpixel_comb = !(sp && !strcmp(sp, "classes"));
  const char* fp = getenv("HS_CNN_FC_POOL");
  c->cnn_fc_pool = !(fp && !strcmp(fp, "0"));
  const char* sg = getenv("HS_STEP_GRAPH");
  c->graph_on = !(sg && !strcmp(sg, "0"));
  c->graph_force = sg && !strcmp(sg, "1");
  const bool bf16 = (c->precision == HS_BF16);
  if (c->arch == HS_MLP) {
    if (bf16) {
      for (int l = 0; l < c->L; ++l)
        if (dims[l] % 8 != 0) {
          delete c;
          return fail(nullptr, HS_ERR_UNSUPPORTED, "bf16 precision needs input and hidden widths divisible by 8");
        }
    }
    int64_t off = 0;
    for (int l = 0; l < c->L; ++l) {
      Layer ly{dims[l], dims[l + 1], 0, 0};
      ly.w_off = off;
      off += (int64_t)ly.in * ly.out;
      ly.b_off = off;
      off += ly.out;
      c->layers.push_back(ly);
    }
    c->P = off;
    c->C = dims[c->L];
    c->Cp = (int)round_up(c->C, 8);
    c->maxw = c->Cp;
    for (int l = 1; l < c->L; ++l) c->maxw = std::max(c->maxw, dims[l]);
    c->in_features = dims[0];
  } else {
    // Cin, H, W, c1, c2, c3, classes: 3x3 convs (padding 1, strides 1, 2, 2), pooling, fc
    if (bf16 && (dims[3] % 8 || dims[4] % 8 || dims[5] % 8)) {
      delete c;
      return fail(nullptr, HS_ERR_UNSUPPORTED, "bf16 precision needs conv widths divisible by 8");
    }
    const int strides[3] = {1, 2, 2};
    int64_t off = 0;
    int h = dims[1], w = dims[2], prev = dims[0];
    for (int k = 0; k < 3; ++k) {
      ConvLayer L{};
      L.cin = prev;
      L.cout = dims[3 + k];
      L.hin = h;
      L.win = w;
      L.stride = strides[k];
      L.hout = (h + 2 - 3) / L.stride + 1;
      L.wout = (w + 2 - 3) / L.stride + 1;
      L.K = prev * 9;
      L.Kp = bf16 ? (int)round_up(L.K + 1, 8) : L.K;   // bf16 rows carry a ones column at K
      L.w_off = off;
      off += (int64_t)L.cout * L.K;
      L.b_off = off;
      off += L.cout;
      L.rows = (int64_t)global_batch * L.hout * L.wout;
      // Implicit patch rows where the geometry allows (HS_CONV_IMPLICIT=0 materialises them all)
      const char* imp = getenv("HS_CONV_IMPLICIT");
      L.implicit = bf16 && k > 0 && !(imp && !strcmp(imp, "0")) &&
                   hs::tc_conv_implicit_ok(L.cin, L.hout, L.wout, L.stride);
      // ... and the input gradient as the sub-pixel product (HS_CONV_IMPLICIT=fwd keeps the
      // patch-space product and its gather)
      L.subpixel = L.implicit && !(imp && !strcmp(imp, "fwd")) && L.stride == 2 && L.hin == 2 * L.hout &&
                   L.win == 2 * L.wout && L.cout % 64 == 0 && hs::tc_grid_ok(L.hout, L.wout, 64) &&
                   hs::tc_grid_ok(L.hout, L.wout, 32);
      c->convs.push_back(L);
      h = L.hout;
      w = L.wout;
      prev = L.cout;
    }
    c->fc_w_off = off;
    off += (int64_t)dims[6] * prev;
    c->fc_b_off = off;
    off += dims[6];
    c->P = off;
    c->C = dims[6];
    c->Cp = (int)round_up(c->C, 8);
    c->maxw = std::max(c->Cp, std::max(dims[3], std::max(dims[4], dims[5])));
    c->in_features = (int64_t)dims[0] * dims[1] * dims[2];
  }
  c->Ps = round_up(c->P, 64);
  if (!c->graph_force && (double)c->P * (double)c->N > 1e11) c->graph_on = false;

  const size_t N = (size_t)c->N;
  const size_t es = c->act_elem();
  hs_status s2 = HS_OK;
  auto chk = [&](hs_status r) { if (r != HS_OK && s2 == HS_OK) s2 = r; };
  chk(dalloc(c, &c->d_offsets, sizeof(int32_t) * (M + 1)));
  chk(dalloc(c, &c->d_index_map, sizeof(int32_t) * N));
  chk(dalloc(c, &c->d_scale, sizeof(float) * N));
  chk(dalloc(c, &c->d_w, sizeof(float) * M));
  const int R = hs::bias_grad_chunk_rows();
  const int max_chunks = c->N / R + M + 1;
  chk(dalloc(c, &c->d_bg_chunks, sizeof(int4) * max_chunks));
  chk(dalloc(c, &c->d_bg_chunk_begin, sizeof(int32_t) * (M + 1)));
  size_t delta_elems = N * (size_t)c->maxw;
  size_t bg_partial = (size_t)max_chunks * (size_t)c->maxw;
  if (c->arch == HS_MLP) {
    c->d_act.assign(c->L, nullptr);
    for (int l = 0; l < c->L; ++l) {
      if (l == 0 && !bf16) continue;   // fp32 reads x in place
      chk(dalloc(c, &c->d_act[l], es * N * (size_t)dims[l]));
    }
    // ReLU' of the hidden activations as bits for the input-gradient products (HS_RELU_BITS=0: read
    // the bf16 activations instead)
    const char* rb = getenv("HS_RELU_BITS");
    if (bf16 && !(rb && !strcmp(rb, "0"))) {
      c->d_relu_bits.assign(c->L, nullptr);
      for (int l = 1; l < c->L; ++l)
        chk(dalloc(c, &c->d_relu_bits[l], sizeof(uint64_t) * N * (size_t)((dims[l] + 63) / 64)));
    }
    chk(dalloc(c, &c->d_scale_fused, sizeof(float) * N));
    chk(dalloc(c, &c->d_all_off, sizeof(int32_t) * 2));
    chk(dalloc(c, &c->d_w_one, sizeof(float)));
    chk(dalloc(c, &c->all_rows.d_chunks, sizeof(int4) * (size_t)(c->N / R + 2)));
    chk(dalloc(c, &c->all_rows.d_begin, sizeof(int32_t) * 2));
  } else {
    const int c3 = c->convs[2].cout;
    int64_t dcol = 0;
    for (int k = 0; k < 3; ++k) {
      const ConvLayer& L = c->convs[k];
      if (!L.implicit) chk(dalloc(c, &c->d_col[k], es * (size_t)L.rows * L.Kp));
      chk(dalloc(c, &c->d_cact[k], es * (size_t)L.rows * L.cout));
      chk(dalloc(c, &c->d_dA[k], es * (size_t)L.rows * L.cout));
      if (k > 0 && !L.subpixel) dcol = std::max<int64_t>(dcol, L.rows * L.K);
    }
    chk(dalloc(c, &c->d_pooled, es * N * c3));
    chk(dalloc(c, &c->d_dpooled, sizeof(float) * N * c3));
    if (dcol > 0) chk(dalloc(c, &c->d_dcol, sizeof(float) * (size_t)dcol));
    if (bf16) {
      for (int k = 0; k < 3; ++k)
        chk(dalloc(c, &c->d_wperm[k], sizeof(__nv_bfloat16) * (size_t)c->convs[k].cout * c->convs[k].Kp));
      chk(dalloc(c, &c->d_ones, sizeof(__nv_bfloat16) * 64 * 64));
      // ReLU' of the first two convolutions' activations as bits, where the next convolution's input
      // gradient is the sub-pixel product (it reads them at its class pixels; HS_RELU_BITS=0: the
      // activations themselves)
      const char* rb = getenv("HS_RELU_BITS");
      c->d_relu_bits.assign(3, nullptr);
      for (int k = 0; k < 2 && !(rb && !strcmp(rb, "0")); ++k)
        if (c->convs[k].cout % 64 == 0 && c->convs[k + 1].subpixel)
          chk(dalloc(c, &c->d_relu_bits[k], sizeof(uint64_t) * (size_t)c->convs[k].rows * (c->convs[k].cout / 64)));
      for (int k = 1; k < 3; ++k) {
        hs::ConvLayer& Lk = c->convs[k];
        Lk.comb = Lk.subpixel && c->subpixel_comb && Lk.cin % 64 == 0;
        if (!Lk.subpixel) continue;
        // combined: 16 blocks of Cout x Cin per shift and class, 7 of them zero for good
        const size_t n = (Lk.comb ? 16 : 9) * (size_t)Lk.cout * Lk.cin;
        chk(dalloc(c, &c->d_wsub[k], sizeof(__nv_bfloat16) * n));
        if (s2 == HS_OK && Lk.comb && cudaMemset(c->d_wsub[k], 0, sizeof(__nv_bfloat16) * n) != cudaSuccess)
          chk(HS_ERR_CUDA);
      }
    }
    delta_elems = N * (size_t)c->Cp;
    for (int k = 0; k < 4; ++k) {
      const bool fc = (k == 3);
      const int64_t rps = fc ? 1 : (int64_t)c->convs[k].hout * c->convs[k].wout;
      const int width = fc ? c->C : c->convs[k].cout;
      const int64_t chunks = (int64_t)c->N * rps / R + M + 1;
      chk(dalloc(c, &c->d_row_off[k], sizeof(int32_t) * (M + 1)));
      chk(dalloc(c, &c->cnn_chunks[k].d_chunks, sizeof(int4) * (size_t)chunks));
      chk(dalloc(c, &c->cnn_chunks[k].d_begin, sizeof(int32_t) * (M + 1)));
      c->cnn_chunks[k].rows_per_sample = (int)rps;
      bg_partial = std::max(bg_partial, (size_t)chunks * (size_t)width);
      if (bf16) {
        CnnWgrad& wg = c->cnn_wgrad[k];
        const int rows_out = width;
        const int kcols = fc ? c3 : c->convs[k].K + 1;
        const int tiles = ((rows_out + kTcBM - 1) / kTcBM) * ((kcols + kTcBN - 1) / kTcBN);
        const int64_t target = std::max<int64_t>(1, (2LL * c->num_sms + tiles - 1) / tiles);
        wg.partial_capacity = (target + M + 1) * rows_out * round_up(kcols, 4);
        chk(dalloc(c, &wg.d_partial, sizeof(float) * (size_t)wg.partial_capacity));
        chk(dalloc(c, &wg.d_chunk_begin, sizeof(int32_t) * (M + 1)));
      }
    }
  }
  chk(dalloc(c, &c->d_bg_partial, sizeof(float) * bg_partial));
  chk(dalloc(c, &c->d_logits, sizeof(float) * N * c->Cp));
  chk(dalloc(c, &c->d_delta[0], es * delta_elems));
  chk(dalloc(c, &c->d_delta[1], es * (c->arch == HS_MLP ? delta_elems : 8)));
  chk(dalloc(c, &c->d_ce, sizeof(float) * N));
  chk(dalloc(c, &c->d_lm, sizeof(float) * M));
  chk(dalloc(c, &c->d_status, sizeof(DevStatus)));
  chk(dalloc(c, &c->d_ticket, sizeof(unsigned int)));
  chk(dalloc(c, &c->d_slabs, sizeof(float) * (size_t)M * (size_t)c->Ps));
  if (c->precision == HS_BF16) chk(dalloc(c, &c->d_shadow, sizeof(__nv_bfloat16) * (size_t)c->Ps));
  if (s2 == HS_OK) {
    e = cudaMallocHost(reinterpret_cast<void**>(&c->h_status), sizeof(DevStatus));
    if (e != cudaSuccess) s2 = cuda_fail(c, e, "cudaMallocHost");
  }
  if (s2 == HS_OK) {
    e = cudaMemset(c->d_status, 0, sizeof(DevStatus));
    if (e == cudaSuccess) e = cudaMemset(c->d_ticket, 0, sizeof(unsigned int));
    if (e == cudaSuccess) e = cudaMemset(c->d_slabs, 0, sizeof(float) * (size_t)M * (size_t)c->Ps);
    if (e == cudaSuccess && c->d_shadow) e = cudaMemset(c->d_shadow, 0, sizeof(__nv_bfloat16) * (size_t)c->Ps);
    if (e == cudaSuccess) e = cudaMemset(c->d_delta[0], 0, es * delta_elems);
    if (e == cudaSuccess && c->arch == HS_MLP) e = cudaMemset(c->d_delta[1], 0, es * delta_elems);
    if (e != cudaSuccess) s2 = cuda_fail(c, e, "cudaMemset");
  }
  if (s2 == HS_OK && c->arch == HS_MLP) {
    // one-worker tables of the slab-free formulation
    const int32_t all_off[2] = {0, c->N};
    const float one = 1.0f;
    std::vector<int4> chunks;
    for (int r = 0; r < c->N; r += R) chunks.push_back(make_int4(0, r, std::min(r + R, c->N), 0));
    const int32_t begin[2] = {0, (int32_t)chunks.size()};
    c->all_rows.n = (int)chunks.size();
    e = cudaMemcpy(c->d_all_off, all_off, sizeof(all_off), cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMemcpy(c->d_w_one, &one, sizeof(one), cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMemcpy(c->all_rows.d_chunks, chunks.data(), sizeof(int4) * chunks.size(), cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMemcpy(c->all_rows.d_begin, begin, sizeof(begin), cudaMemcpyHostToDevice);
    if (e != cudaSuccess) s2 = cuda_fail(c, e, "slab-free tables");
  }
  if (s2 == HS_OK && bf16) s2 = c->arch == HS_MLP ? build_tc_static(c) : cnn_build_static(c);
  if (s2 == HS_OK && bf16 && c->arch == HS_MLP) s2 = build_tc_wgrad_fused(c);
  if (s2 == HS_OK && bf16 && c->arch == HS_MLP) {
    // HS_OVERLAP_UPDATE=0: slab-path updates on the step's stream instead of the update stream;
    // HS_TILE_AVERAGE=0: every layer on the slab path (per-worker gradients stored, then reduced);
    // =all: the tile-averaged launch also for layers with fewer weight tiles than SM pairs
    const char* ov = getenv("HS_OVERLAP_UPDATE");
    c->overlap_update = !(ov && !strcmp(ov, "0"));
    const char* ta = getenv("HS_TILE_AVERAGE");
    c->tile_avg = !(ta && !strcmp(ta, "0")) && c->M <= hs::kTcMaxGroups;
    c->tile_avg_all = ta && !strcmp(ta, "all");
    e = cudaStreamCreateWithFlags(&c->upd_stream, cudaStreamNonBlocking);
    c->upd_ready.assign(c->L, nullptr);
    for (int l = 0; l < c->L && e == cudaSuccess; ++l) e = cudaEventCreateWithFlags(&c->upd_ready[l], cudaEventDisableTiming);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&c->upd_done, cudaEventDisableTiming);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&c->dgrad_done, cudaEventDisableTiming);
    if (e != cudaSuccess) s2 = cuda_fail(c, e, "update stream");
    if (s2 == HS_OK) s2 = dalloc(c, &c->d_shadow_next, sizeof(__nv_bfloat16) * (size_t)c->Ps);
  }
  if (s2 == HS_OK) s2 = apply_partition(c, sizes, cpn, nullptr, 0);
  if (s2 == HS_OK) {
    e = cudaDeviceSynchronize();
    if (e != cudaSuccess) s2 = cuda_fail(c, e, "initial partition");
  }
  if (s2 != HS_OK) {
    g_init_error = c->err;
    free_all(c);
    delete c;
    return s2;
  }
  *out = c;
  return HS_OK;
}

hs_status hs_partition(hs_ctx* c, const double* measured_throughputs, int32_t* counts_out, int32_t* index_map_out,
                       void* stream, hs_partition_t* out) {
  if (!c) return HS_ERR_INVALID_ARG;
  c->err.clear();
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (measured_throughputs) {
    for (int m = 0; m < c->M; ++m)
      if (!std::isfinite(measured_throughputs[m]) || !(measured_throughputs[m] > 0.0))
        return fail(c, HS_ERR_INVALID_ARG, "measured_throughputs: compute power must be finite and > 0");
    // the estimate handed to Algorithm 1: the last measurement, or a history of them (Section 4.1)
    std::vector<double> est(measured_throughputs, measured_throughputs + c->M);
    if (c->cp_hist_mode == 1) {
      const double a = c->cp_hist_param;
      if (c->cp_ema.empty()) {
        c->cp_ema = est;
      } else {
        for (int m = 0; m < c->M; ++m) c->cp_ema[m] = a * est[m] + (1.0 - a) * c->cp_ema[m];
      }
      est = c->cp_ema;
    } else if (c->cp_hist_mode == 2) {
      c->cp_window.push_back(est);
      if ((int)c->cp_window.size() > (int)c->cp_hist_param) c->cp_window.erase(c->cp_window.begin());
      for (int m = 0; m < c->M; ++m) {
        double acc = 0.0;
        for (const auto& row : c->cp_window) acc = acc + row[m];
        est[m] = acc / (double)c->cp_window.size();
      }
    }
    std::vector<int32_t> sizes(c->M);
    std::vector<double> cpn(c->M);
    const char* why = nullptr;
    hs_status st = hs::partition_sizes_impl(c->M, c->N, est.data(), sizes.data(), cpn.data(), &why);
    if (st != HS_OK) return fail(c, st, std::string("measured_throughputs: ") + why);
    st = apply_partition(c, sizes, cpn, index_map_out, s);
    if (st != HS_OK) return st;
  } else if (index_map_out) {
    hs::launch_partition_scatter(c->d_offsets, c->M, c->N, c->d_index_map, c->d_scale, index_map_out, s);
    HS_CUDA(c, cudaGetLastError());
  }
  if (counts_out) std::memcpy(counts_out, c->counts.data(), sizeof(int32_t) * c->M);
  fill_partition_view(c, out);
  return HS_OK;
}

hs_status hs_sync_params(hs_ctx* c, const float* params, void* stream) {
  if (!c || !params) return c ? fail(c, HS_ERR_INVALID_ARG, "params is NULL") : HS_ERR_INVALID_ARG;
  c->err.clear();
  if (c->precision != HS_BF16) return HS_OK;
  hs::launch_cast_f32_bf16(params, c->d_shadow, c->P, reinterpret_cast<cudaStream_t>(stream));
  HS_CUDA(c, cudaGetLastError());
  c->shadow_src = params;
  c->shadow_valid = true;
  c->cnn_wcopy_src = nullptr;   // the CNN's permuted copies are re-derived by the next step
  return HS_OK;
}

hs_status hs_step(hs_ctx* c, float* params, const void* x, const int32_t* y, const hs_partition_t* part, float lr,
                  void* stream, float* loss_out) {
  if (!c) return HS_ERR_INVALID_ARG;
  c->err.clear();
  if (!params || !x || !y) return fail(c, HS_ERR_INVALID_ARG, "params, x and y must be non-NULL");
  if ((reinterpret_cast<uintptr_t>(params) & 15u) != 0) return fail(c, HS_ERR_INVALID_ARG, "params must be 16-byte aligned");
  if (!std::isfinite(lr)) return fail(c, HS_ERR_INVALID_ARG, "lr must be finite");
  if (part && (part->version != c->version || part->M != c->M || part->N != c->N))
    return fail(c, HS_ERR_INVALID_ARG, "partition does not match the context's current partition");
  if (!is_device_ptr(params)) return fail(c, HS_ERR_INVALID_ARG, "params must be a device pointer");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const size_t in_feat = (size_t)c->in_features;
  const float* xd = reinterpret_cast<const float*>(x);
  const int32_t* yd = y;
  int slot = -1;   // inputs from hs_stage_inputs: wait for their copy, mark the slot read afterwards
  for (int k = 0; k < 2; ++k)
    if (c->d_xslot[k] && x == c->d_xslot[k]) slot = k;
  if (slot >= 0) {
    if (y != c->d_yslot[slot] || !c->slot_pending[slot])
      return fail(c, HS_ERR_INVALID_ARG, "staged x and y must come from the same, not yet used hs_stage_inputs call");
    HS_CUDA(c, cudaStreamWaitEvent(s, c->slot_staged[slot], 0));
  } else if (!is_device_ptr(x)) {
    if (!c->d_xstage) {
      hs_status r = dalloc(c, &c->d_xstage, sizeof(float) * c->N * in_feat);
      if (r != HS_OK) return r;
    }
    HS_CUDA(c, cudaMemcpyAsync(c->d_xstage, x, sizeof(float) * c->N * in_feat, cudaMemcpyHostToDevice, s));
    xd = reinterpret_cast<const float*>(c->d_xstage);
  }
  if (!is_device_ptr(y)) {
    if (!c->d_ystage) {
      hs_status r = dalloc(c, &c->d_ystage, sizeof(int32_t) * c->N);
      if (r != HS_OK) return r;
    }
    HS_CUDA(c, cudaMemcpyAsync(c->d_ystage, y, sizeof(int32_t) * c->N, cudaMemcpyHostToDevice, s));
    yd = c->d_ystage;
  }
  if (c->precision == HS_BF16 && (!c->shadow_valid || c->shadow_src != params)) {
    PhaseScope ph(c, HS_PHASE_CAST, s);
    hs::launch_cast_f32_bf16(params, c->d_shadow, c->P, s);
    ph.launched();
  }
  if (c->debug && !c->d_gdebug) {
    hs_status r = dalloc(c, &c->d_gdebug, sizeof(float) * c->Ps);
    if (r != HS_OK) return r;
  }
  if (c->arch == HS_CNN && c->precision == HS_BF16 && c->cnn_wcopy_src != params) {
    hs_status r = hs::cnn_refresh_weights(c, params, s);
    if (r != HS_OK) return r;
  }
  // A caller capturing its own graph gets the step's kernels enqueued as they are.
  cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
  const bool caller_capture = cudaStreamIsCapturing(s, &cap) != cudaSuccess || cap != cudaStreamCaptureStatusNone;
  if (caller_capture) cudaGetLastError();
  hs_status st = (c->graph_on && !caller_capture) ? step_via_graph(c, params, xd, yd, lr, s)
                                                  : step_body(c, params, xd, yd, lr, nullptr, s);
  if (st != HS_OK) return st;
  if (slot >= 0) {
    HS_CUDA(c, cudaEventRecord(c->slot_consumed[slot], s));
    c->slot_pending[slot] = false;
    c->slot_used[slot] = true;
  }
  HS_CUDA(c, cudaGetLastError());
  c->shadow_src = params;
  c->shadow_valid = (c->precision == HS_BF16);
  c->cnn_wcopy_src = hs::cnn_fused_update(c) ? params : nullptr;   // the fused update wrote the copies
  c->gdebug_valid = c->debug;
  if (c->opt_recipe) c->mom_valid = true;
  if (loss_out) {
    HS_CUDA(c, cudaMemcpyAsync(c->h_status, c->d_status, sizeof(DevStatus), cudaMemcpyDeviceToHost, s));
    HS_CUDA(c, cudaStreamSynchronize(s));
    *loss_out = c->h_status->loss;
    if (c->h_status->err != hs::kDevOk) {
      const int code = c->h_status->err, info = c->h_status->err_info;
      cudaMemsetAsync(c->d_status, 0, sizeof(DevStatus), s);
      cudaStreamSynchronize(s);
      char buf[160];
      std::snprintf(buf, sizeof(buf), "device check failed: code %d (%s), detail %d", code,
                    code == hs::kDevWaitTimeout ? "bounded wait expired" : "label out of range", info);
      return fail(c, HS_ERR_DEVICE_CHECK, buf);
    }
  }
  return HS_OK;
}

hs_status hs_stage_inputs(hs_ctx* c, const float* x_host, const int32_t* y_host, void* stream, const float** x_dev,
                          const int32_t** y_dev) {
  if (!c) return HS_ERR_INVALID_ARG;
  c->err.clear();
  if (!x_host || !y_host || !x_dev || !y_dev) return fail(c, HS_ERR_INVALID_ARG, "x, y and the outputs must be non-NULL");
  const int k = c->next_slot;
  if (c->slot_pending[k])
    return fail(c, HS_ERR_INVALID_ARG, "both staging slots hold inputs no hs_step has read yet");
  const size_t xbytes = sizeof(float) * (size_t)c->N * (size_t)c->in_features;
  if (!c->d_xslot[k]) {
    hs_status r = dalloc(c, &c->d_xslot[k], xbytes);
    if (r == HS_OK) r = dalloc(c, &c->d_yslot[k], sizeof(int32_t) * (size_t)c->N);
    if (r != HS_OK) return r;
    HS_CUDA(c, cudaEventCreateWithFlags(&c->slot_staged[k], cudaEventDisableTiming));
    HS_CUDA(c, cudaEventCreateWithFlags(&c->slot_consumed[k], cudaEventDisableTiming));
  }
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (c->slot_used[k]) HS_CUDA(c, cudaStreamWaitEvent(s, c->slot_consumed[k], 0));   // the last reader is done
  HS_CUDA(c, cudaMemcpyAsync(c->d_xslot[k], x_host, xbytes, cudaMemcpyHostToDevice, s));
  HS_CUDA(c, cudaMemcpyAsync(c->d_yslot[k], y_host, sizeof(int32_t) * (size_t)c->N, cudaMemcpyHostToDevice, s));
  HS_CUDA(c, cudaEventRecord(c->slot_staged[k], s));
  c->slot_pending[k] = true;
  c->next_slot = k ^ 1;
  *x_dev = c->d_xslot[k];
  *y_dev = c->d_yslot[k];
  return HS_OK;
}

hs_status hs_set_profiling(hs_ctx* c, int32_t enable) {
  if (!c) return HS_ERR_INVALID_ARG;
  c->profiling = enable != 0;
  return HS_OK;
}

hs_status hs_read_profile(hs_ctx* c, double* ms_out, int64_t* launches_out) {
  if (!c) return HS_ERR_INVALID_ARG;
  c->err.clear();
  double ms[HS_PHASE_COUNT] = {0};
  cudaError_t first = cudaSuccess;
  for (auto& r : c->pending) {
    cudaError_t e = cudaEventSynchronize(r.b);
    float t = 0.f;
    if (e == cudaSuccess) e = cudaEventElapsedTime(&t, r.a, r.b);
    if (e != cudaSuccess && first == cudaSuccess) first = e;
    ms[r.phase] += t;
    c->event_pool.push_back(r.a);
    c->event_pool.push_back(r.b);
  }
  c->pending.clear();
  if (ms_out)
    for (int i = 0; i < HS_PHASE_COUNT; ++i) ms_out[i] = ms[i];
  if (launches_out)
    for (int i = 0; i < HS_PHASE_COUNT; ++i) launches_out[i] = c->launches[i];
  for (int i = 0; i < HS_PHASE_COUNT; ++i) c->launches[i] = 0;
  if (first != cudaSuccess) return cuda_fail(c, first, "reading profile events");
  return HS_OK;
}

hs_status hs_set_fused_sync(hs_ctx* c, int32_t enable) {
  if (!c) return HS_ERR_INVALID_ARG;
  c->err.clear();
  if (c->arch != HS_MLP) return fail(c, HS_ERR_UNSUPPORTED, "the slab-free formulation is built for the MLP only");
  if (c->fused_sync != (enable != 0)) invalidate_step_graphs(c);
  c->fused_sync = enable != 0;
  return HS_OK;
}

hs_status hs_set_cp_history(hs_ctx* c, int32_t mode, double param) {
  if (!c) return HS_ERR_INVALID_ARG;
  c->err.clear();
  if (mode == HS_CP_EMA && !(param > 0.0 && param <= 1.0))
    return fail(c, HS_ERR_INVALID_ARG, "EMA weight must be in (0, 1]");
  if (mode == HS_CP_WINDOW && !(param >= 1.0 && param <= 1024.0 && param == (double)(int)param))
    return fail(c, HS_ERR_INVALID_ARG, "window length must be an integer in [1, 1024]");
  if (mode != HS_CP_LAST && mode != HS_CP_EMA && mode != HS_CP_WINDOW)
    return fail(c, HS_ERR_INVALID_ARG, "unknown compute-power history mode");
  c->cp_hist_mode = mode;
  c->cp_hist_param = param;
  c->cp_ema.clear();
  c->cp_window.clear();
  return HS_OK;
}

hs_status hs_set_optimizer(hs_ctx* c, float momentum, float weight_decay) {
  if (!c) return HS_ERR_INVALID_ARG;
  c->err.clear();
  if (!std::isfinite(momentum) || !std::isfinite(weight_decay) || momentum < 0.f || momentum >= 1.f ||
      weight_decay < 0.f)
    return fail(c, HS_ERR_INVALID_ARG, "momentum must be in [0, 1) and weight_decay >= 0");
  invalidate_step_graphs(c);
  if (momentum == 0.f && weight_decay == 0.f) {
    c->opt_recipe = false;
    return HS_OK;
  }
  if (!c->d_mom) {
    hs_status r = dalloc(c, &c->d_mom, sizeof(float) * (size_t)c->Ps);
    if (r != HS_OK) return r;
  }
  c->opt_recipe = true;
  c->opt_momentum = momentum;
  c->opt_weight_decay = weight_decay;
  c->mom_valid = false;
  return HS_OK;
}

hs_status hs_optimizer_state(hs_ctx* c, float* buf_dev, int32_t save, void* stream) {
  if (!c || !buf_dev) return c ? fail(c, HS_ERR_INVALID_ARG, "buf_dev is NULL") : HS_ERR_INVALID_ARG;
  c->err.clear();
  if (!c->opt_recipe || !c->d_mom) return fail(c, HS_ERR_INVALID_ARG, "no optimizer state: call hs_set_optimizer first");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (save) {
    if (!c->mom_valid) return fail(c, HS_ERR_INVALID_ARG, "the momentum buffer has not been started yet");
    HS_CUDA(c, cudaMemcpyAsync(buf_dev, c->d_mom, sizeof(float) * c->P, cudaMemcpyDeviceToDevice, s));
  } else {
    HS_CUDA(c, cudaMemcpyAsync(c->d_mom, buf_dev, sizeof(float) * c->P, cudaMemcpyDeviceToDevice, s));
    c->mom_valid = true;
  }
  return HS_OK;
}

double hs_cosine_lr(double eta0, double eta_min, int64_t t, int64_t T) {
  if (T <= 0) return eta0;
  if (t > T) t = T;
  return eta_min + (eta0 - eta_min) * (1.0 + std::cos(M_PI * (double)t / (double)T)) / 2.0;
}

hs_status hs_set_debug(hs_ctx* c, int32_t enable) {
  if (!c) return HS_ERR_INVALID_ARG;
  if (c->debug != (enable != 0)) invalidate_step_graphs(c);
  c->debug = enable != 0;
  return HS_OK;
}

hs_status hs_debug_grads(hs_ctx* c, float* g_out, float* slabs_out, void* stream) {
  if (!c) return HS_ERR_INVALID_ARG;
  c->err.clear();
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (g_out) {
    if (!c->gdebug_valid || !c->d_gdebug)
      return fail(c, HS_ERR_INVALID_ARG, "no synchronised gradient kept: call hs_set_debug(ctx, 1) before hs_step");
    HS_CUDA(c, cudaMemcpyAsync(g_out, c->d_gdebug, sizeof(float) * c->P, cudaMemcpyDeviceToDevice, s));
  }
  if (slabs_out) {
    if (c->fused_sync) return fail(c, HS_ERR_INVALID_ARG, "the slab-free formulation keeps no per-worker slabs");
    if (c->tile_step)
      return fail(c, HS_ERR_INVALID_ARG,
                  "the last step kept the per-worker weight gradients in tensor memory: call hs_set_debug(ctx, 1) "
                  "before hs_step for slabs");
    HS_CUDA(c, cudaMemcpy2DAsync(slabs_out, sizeof(float) * c->P, c->d_slabs, sizeof(float) * c->Ps,
                                 sizeof(float) * c->P, c->M, cudaMemcpyDeviceToDevice, s));
  }
  return HS_OK;
}

hs_status hs_worker_losses(hs_ctx* c, float* losses_out) {
  if (!c || !losses_out) return HS_ERR_INVALID_ARG;
  c->err.clear();
  HS_CUDA(c, cudaDeviceSynchronize());
  HS_CUDA(c, cudaMemcpy(losses_out, c->d_lm, sizeof(float) * c->M, cudaMemcpyDeviceToHost));
  return HS_OK;
}

void hs_destroy(hs_ctx* c) {
  if (!c) return;
  cudaDeviceSynchronize();
  invalidate_step_graphs(c);
  free_all(c);
  delete c;
}

hs_status hs_debug_gemm_bf16(int32_t mode, int32_t M, int32_t N, int32_t K, const void* A, int64_t lda, const void* B,
                             int64_t ldb, void* D, int64_t ldd, const float* bias, const void* Z, int64_t ldz,
                             const int32_t* k_offsets_host, int32_t groups, int64_t d_gstride, void* stream) {
  g_init_error.clear();
  const bool stall = (mode & HS_GEMM_TEST_STALL) != 0;
  mode &= ~HS_GEMM_TEST_STALL;
  const int form = mode >> 8;
  mode &= 0xFF;
  if (form < 0 || form > 2) return fail(nullptr, HS_ERR_INVALID_ARG, "unknown kernel form");
  if (M < 1 || N < 1 || K < 0 || !A || !B || !D) return fail(nullptr, HS_ERR_INVALID_ARG, "bad GEMM arguments");
  const bool bf16_out = (mode == HS_GEMM_FWD_RELU || mode == HS_GEMM_DGRAD);
  if (lda % 8 || ldb % 8 || (bf16_out ? ldd % 8 : ldd % 4) || (mode == HS_GEMM_DGRAD && (ldz % 8 || !Z)) ||
      d_gstride % 4)
    return fail(nullptr, HS_ERR_INVALID_ARG, "leading dimensions must be multiples of 8 elements");
  auto a16 = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; };
  if (!a16(D) || (bias && !a16(bias)) || (Z && !a16(Z)))
    return fail(nullptr, HS_ERR_INVALID_ARG, "D, bias and Z must be 16-byte aligned");
  if (mode < HS_GEMM_FWD_RELU || mode > HS_GEMM_WGRAD) return fail(nullptr, HS_ERR_INVALID_ARG, "unknown mode");
  if ((mode == HS_GEMM_FWD_RELU || mode == HS_GEMM_FWD_LOGITS) && !bias)
    return fail(nullptr, HS_ERR_INVALID_ARG, "bias required");
  const char* why = nullptr;
  if (!hs::tc_init_driver(&why)) return fail(nullptr, HS_ERR_CUDA, why);
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  std::vector<hs::TcGemmParams> plans;
  const auto* pa = reinterpret_cast<const __nv_bfloat16*>(A);
  const auto* pb = reinterpret_cast<const __nv_bfloat16*>(B);
  if (mode == HS_GEMM_WGRAD) {
    if (!k_offsets_host || groups < 1) return fail(nullptr, HS_ERR_INVALID_ARG, "k_offsets and groups required");
    for (int g0 = 0; g0 < groups; g0 += hs::kTcMaxGroups) {
      const int ng = std::min(hs::kTcMaxGroups, groups - g0);
      plans.emplace_back();
      hs::TcGemmParams& p = plans.back();
      std::memset(&p, 0, sizeof(p));
      for (int g = 0; g < ng; ++g) {
        const int64_t k0 = k_offsets_host[g0 + g], kn = k_offsets_host[g0 + g + 1] - k0;
        if (kn < 1) return fail(nullptr, HS_ERR_INVALID_ARG, "every group needs K >= 1");
        if (!hs::tc_make_mnmajor_map(&p.tmA[g], hs::TcOperand{pa + k0 * lda, kn, M, lda}, &why) ||
            !hs::tc_make_mnmajor_map(&p.tmB[g], hs::TcOperand{pb + k0 * ldb, kn, N, ldb}, &why) ||
            !hs::tc_make_store_map(&p.tmD[g], reinterpret_cast<float*>(D) + (int64_t)(g0 + g) * d_gstride, true, M,
                                   N, ldd, &why))
          return fail(nullptr, HS_ERR_INVALID_ARG, why);
        p.num_kb[g] = (int)((kn + hs::kTcBK - 1) / hs::kTcBK);
        p.last_ksteps[g] = last_ksteps(kn);
      }
      p.groups = ng;
      p.epi = hs::kTcEpiStoreF32;
      p.a_mn = 1;
      p.b_mn = 1;
      p.D = reinterpret_cast<float*>(D) + (int64_t)g0 * d_gstride;
      p.d_gstride = d_gstride;
    }
  } else {
    if (K < 1) return fail(nullptr, HS_ERR_INVALID_ARG, "K must be >= 1");
    plans.emplace_back();
    hs::TcGemmParams& p = plans.back();
    std::memset(&p, 0, sizeof(p));
    bool ok = hs::tc_make_kmajor_map(&p.tmA[0], hs::TcOperand{pa, M, K, lda}, hs::kTcBoxA, &why);
    if (mode == HS_GEMM_DGRAD) ok = ok && hs::tc_make_mnmajor_map(&p.tmB[0], hs::TcOperand{pb, K, N, ldb}, &why);
    else ok = ok && hs::tc_make_kmajor_map(&p.tmB[0], hs::TcOperand{pb, N, K, ldb}, hs::kTcBoxB, &why);
    if (!ok) return fail(nullptr, HS_ERR_INVALID_ARG, why);
    p.num_kb[0] = (K + hs::kTcBK - 1) / hs::kTcBK;
    p.groups = 1;
    p.epi = mode == HS_GEMM_FWD_RELU ? hs::kTcEpiBiasReluBf16
          : mode == HS_GEMM_FWD_LOGITS ? hs::kTcEpiBiasF32 : hs::kTcEpiMaskBf16;
    p.b_mn = (mode == HS_GEMM_DGRAD);
    p.D = D;
    p.bias = bias;
    p.Z = reinterpret_cast<const __nv_bfloat16*>(Z);
    p.ldz = ldz;
    if (!hs::tc_make_store_map(&p.tmD[0], D, mode == HS_GEMM_FWD_LOGITS, M, N, ldd, &why))
      return fail(nullptr, HS_ERR_INVALID_ARG, why);
  }
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  DevStatus* dst = nullptr;   // the kernel's status word for this call
  cudaError_t ea = cudaMalloc(reinterpret_cast<void**>(&dst), sizeof(DevStatus));
  if (ea != cudaSuccess) return cuda_fail(nullptr, ea, "status word");
  ea = cudaMemsetAsync(dst, 0, sizeof(DevStatus), s);
  if (ea != cudaSuccess) {
    cudaFree(dst);
    return cuda_fail(nullptr, ea, "status word");
  }
  for (hs::TcGemmParams& p : plans) {
    p.Mdim = M;
    p.Ndim = N;
    p.n_store = N;
    p.tiles_m = (M + hs::kTcBM - 1) / hs::kTcBM;
    p.tiles_n = (N + hs::kTcBN - 1) / hs::kTcBN;
    p.ldd = ldd;
    p.st = dst;
    p.test_stall = stall ? 1 : 0;
    cudaError_t e = hs::launch_tc_gemm_form(p, sms, s, form ? form : hs::tc_get_form());
    if (e != cudaSuccess) {
      cudaFree(dst);
      return cuda_fail(nullptr, e, "GEMM launch");
    }
  }
  cudaError_t e = cudaStreamSynchronize(s);
  DevStatus hst{};
  if (e == cudaSuccess) e = cudaMemcpy(&hst, dst, sizeof(DevStatus), cudaMemcpyDeviceToHost);
  cudaFree(dst);
  if (e != cudaSuccess) return cuda_fail(nullptr, e, "GEMM run");
  if (hst.err != hs::kDevOk) {
    char buf[128];
    std::snprintf(buf, sizeof(buf), "device check failed in the GEMM: code %d, detail %d", hst.err, hst.err_info);
    return fail(nullptr, HS_ERR_DEVICE_CHECK, buf);
  }
  return HS_OK;
}

hs_status hs_debug_wgrad_avg(int32_t M, int32_t N, const void* A, int64_t lda, const void* B, int64_t ldb,
                             const int32_t* k_offsets_host, int32_t groups, const float* wavg, float lr,
                             float* theta, int64_t ld_theta, void* shadow, int64_t ld_shadow, int32_t test_stall,
                             void* stream) {
  g_init_error.clear();
  if (M < 1 || N < 1 || !A || !B || !k_offsets_host || !wavg || !theta || !shadow || groups < 1 ||
      groups > hs::kTcMaxGroups)
    return fail(nullptr, HS_ERR_INVALID_ARG, "bad arguments (groups must be 1..32)");
  if (lda % 8 || ldb % 8 || ld_theta % 8 || ld_shadow % 8 || lda < M || ldb < N || ld_theta < N || ld_shadow < N)
    return fail(nullptr, HS_ERR_INVALID_ARG, "leading dimensions must be multiples of 8 elements");
  auto a16 = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; };
  if (!a16(A) || !a16(B) || !a16(theta) || !a16(shadow))
    return fail(nullptr, HS_ERR_INVALID_ARG, "pointers must be 16-byte aligned");
  const char* why = nullptr;
  if (!hs::tc_init_driver(&why)) return fail(nullptr, HS_ERR_CUDA, why);
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  hs::TcGemmParams p;
  std::memset(&p, 0, sizeof(p));
  const auto* pa = reinterpret_cast<const __nv_bfloat16*>(A);
  const auto* pb = reinterpret_cast<const __nv_bfloat16*>(B);
  for (int g = 0; g < groups; ++g) {
    const int64_t k0 = k_offsets_host[g], kn = k_offsets_host[g + 1] - k0;
    if (kn < 1) return fail(nullptr, HS_ERR_INVALID_ARG, "every group needs at least one row");
    if (!hs::tc_make_mnmajor_map(&p.tmA[g], hs::TcOperand{pa + k0 * lda, kn, M, lda}, &why) ||
        !hs::tc_make_mnmajor_map(&p.tmB[g], hs::TcOperand{pb + k0 * ldb, kn, N, ldb}, &why))
      return fail(nullptr, HS_ERR_INVALID_ARG, why);
    p.num_kb[g] = (int32_t)((kn + hs::kTcBK - 1) / hs::kTcBK);
    p.last_ksteps[g] = last_ksteps(kn);
  }
  if (!hs::tc_make_store_map(&p.tmT, theta, true, M, N, ld_theta, &why) ||
      !hs::tc_make_store_map_bf16_32(&p.tmS, shadow, M, N, ld_shadow, &why))
    return fail(nullptr, HS_ERR_INVALID_ARG, why);
  p.groups = groups;
  p.Mdim = M;
  p.Ndim = N;
  p.n_store = N;
  p.epi = hs::kTcEpiAvgUpdate;
  p.a_mn = 1;
  p.b_mn = 1;
  p.wavg = wavg;
  p.lr = lr;
  p.test_stall = test_stall ? 1 : 0;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  DevStatus* dst = nullptr;
  cudaError_t e = cudaMalloc(reinterpret_cast<void**>(&dst), sizeof(DevStatus));
  if (e != cudaSuccess) return cuda_fail(nullptr, e, "status word");
  e = cudaMemsetAsync(dst, 0, sizeof(DevStatus), s);
  p.st = dst;
  if (e == cudaSuccess) e = hs::launch_tc_wgrad_avg(p, sms, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  DevStatus hst{};
  if (e == cudaSuccess) e = cudaMemcpy(&hst, dst, sizeof(DevStatus), cudaMemcpyDeviceToHost);
  cudaFree(dst);
  if (e != cudaSuccess) return cuda_fail(nullptr, e, "weight-gradient average launch");
  if (hst.err != hs::kDevOk) {
    char buf[128];
    std::snprintf(buf, sizeof(buf), "device check failed in the weight-gradient average: code %d, detail %d", hst.err,
                  hst.err_info);
    return fail(nullptr, HS_ERR_DEVICE_CHECK, buf);
  }
  return HS_OK;
}

}  // extern "C"
