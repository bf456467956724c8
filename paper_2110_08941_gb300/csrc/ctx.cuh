// Internal: the context behind hs_ctx* and helpers shared by the step implementations.
#pragma once

#include <string>
#include <vector>

#include "../../include/hs.h"
#include "common.cuh"
#include "gemm_tc.cuh"

namespace hs {

struct Layer {
  int in, out;
  int64_t w_off, b_off;
};

// One 3x3 convolution (padding 1) of the CNN workload, as a product over im2col rows.
struct ConvLayer {
  int cin, cout, hin, win, hout, wout, stride;
  int K, Kp;          // Cin*9 and its row stride in the bf16 patch buffer (multiple of 8)
  int64_t w_off, b_off;
  int64_t rows;       // N * hout * wout
  bool implicit;      // bf16: the products read the patch rows straight from the input (no col buffer)
  bool subpixel;      // bf16: the input gradient is the grouped sub-pixel product (no patch-space buffer)
  bool comb;          // ... as one product whose columns are the four classes' blocks (d_wsub holds
                      // the combined weights [4 shifts x Cout][4 classes x Cin]; else [9 x Cout][Cin]
                      // class matrices)
};

inline int64_t round_up(int64_t v, int64_t m) { return (v + m - 1) / m * m; }

// The first convolution in one kernel (csrc/conv_first.cu): patch rows from the NCHW fp32 input in
// shared memory (and written out for the weight gradient), the product with the resident bf16
// weights, bias + ReLU into the NHWC bf16 activations.
struct ConvFirstParams {
  CUtensorMap tmW;            // bf16 weights [Cout][Kp], K-major, one box of 64 x npad
  CUtensorMap tmX;            // the NCHW fp32 input in boxes of box_w x box_h x C (tc_make_nchw_box_map)
  const float* x;             // NCHW fp32 input (the one tmX maps)
  const float* bias;          // fp32 [Cout] (theta's bias of the layer, per launch)
  __nv_bfloat16* col;         // patch rows out [rows][Kp] (tap-major, ones column at 9 * C)
  __nv_bfloat16* out;         // activations [rows][Cout]
  int64_t rows;               // N * Ho * Wo
  int C, H, W, Ho, Wo, stride, Cout, Kp;
  int npad, acc_cols;         // MMA width (Cout rounded up to 16), tensor-memory columns per accumulator
  uint64_t* bits;             // non-null: ReLU' of the stored activations as bits, word [c / 64][row]
  int64_t bits_ld;            // (rows); Cout a multiple of 64
  int R, tpi, tiles;          // output rows per tile (whole rows of one image), tiles per image, tiles
  int box_w, box_h;           // input box: columns from -4, rows from stride * ho0 - 1
  DevStatus* st;
};

// Per-layer bias-gradient chunk tables (worker, row begin, row end) for a given rows-per-sample.
struct ChunkTable {
  int4* d_chunks = nullptr;
  int32_t* d_begin = nullptr;
  int n = 0;
  int rows_per_sample = 1;
};

// Split-K weight-gradient plan of one CNN layer (groups = workers, each split into k-block parts).
struct CnnWgrad {
  std::vector<TcGemmParams> plans;
  int rows_out = 0, K = 0, ldp = 0;
  float* d_partial = nullptr;        // [workers x parts][rows_out][ldp]
  int64_t partial_capacity = 0;      // floats
  int32_t* d_chunk_begin = nullptr;  // [M + 1]: worker m's parts are [begin[m], begin[m + 1])
};

}  // namespace hs

struct hs_ctx {
  int device = 0;
  int num_sms = 0;
  int arch = HS_MLP, precision = HS_BF16, sync = HS_SYNC_MEAN;
  std::vector<int32_t> dims;
  std::vector<hs::Layer> layers;
  int L = 0;
  int M = 0, N = 0;
  int64_t P = 0, Ps = 0;
  int C = 0, Cp = 0, maxw = 0;

  // partition state (host mirror + device copies)
  std::vector<int32_t> counts, offsets;
  std::vector<double> weights, cp_norm;
  uint64_t version = 0;
  int32_t* d_offsets = nullptr;
  int32_t* d_index_map = nullptr;
  float* d_scale = nullptr;
  float* d_w = nullptr;
  int4* d_bg_chunks = nullptr;       // bias-gradient row chunks (worker, begin, end, 0)
  int32_t* d_bg_chunk_begin = nullptr;
  int n_bg_chunks = 0;
  float* d_bg_partial = nullptr;     // [max chunks, maxw] partial column sums

  // workspace
  std::vector<void*> d_act;        // H_0 .. H_{L-1}
  std::vector<uint64_t*> d_relu_bits;   // bf16: ReLU' of H_1 .. H_{L-1} as bits, [width / 64][N] words
  float* d_logits = nullptr;       // [N, Cp]
  void* d_delta[2] = {nullptr, nullptr};
  float* d_ce = nullptr;
  float* d_lm = nullptr;
  unsigned int* d_ticket = nullptr;   // completion counter of the per-worker loss reduction (zero between steps)
  hs::DevStatus* d_status = nullptr;
  hs::DevStatus* h_status = nullptr;   // pinned
  float* d_slabs = nullptr;        // [M, Ps]
  __nv_bfloat16* d_shadow = nullptr;
  // overlapped updates: layers 2..L write their new bf16 weights here while the same step's
  // input-gradient products still read d_shadow; copied over d_shadow before the step ends
  __nv_bfloat16* d_shadow_next = nullptr;
  float* d_gdebug = nullptr;
  void* d_xstage = nullptr;
  int32_t* d_ystage = nullptr;
  // double-buffered input staging (hs_stage_inputs): slot k holds one step's x and y
  float* d_xslot[2] = {nullptr, nullptr};
  int32_t* d_yslot[2] = {nullptr, nullptr};
  cudaEvent_t slot_staged[2] = {nullptr, nullptr};     // copy into slot k done (on the staging stream)
  cudaEvent_t slot_consumed[2] = {nullptr, nullptr};   // the step that read slot k done (on its stream)
  bool slot_pending[2] = {false, false};               // staged, not yet read by a step
  bool slot_used[2] = {false, false};                  // slot_consumed[k] has been recorded
  int next_slot = 0;
  const float* shadow_src = nullptr;
  bool shadow_valid = false;
  bool debug = false;
  bool gdebug_valid = false;
  std::string err;

  // profiling: per-phase event pairs recorded on the step's stream, summed on read
  bool profiling = false;
  struct Rec { int phase; cudaEvent_t a, b; };
  std::vector<Rec> pending;
  std::vector<cudaEvent_t> event_pool;
  int64_t launches[HS_PHASE_COUNT] = {0};

  // The step's kernels as a CUDA graph: captured once per key (parameters, inputs, momentum state,
  // profiling), replayed by later steps with the learning rate written to d_lr first.  The launch
  // overhead of a step's 20-40 kernels is then paid once; the kernels and their order are the
  // eager path's.  Invalidated by every call that changes what a step enqueues; HS_STEP_GRAPH=0
  // keeps every step eager.
  struct StepGraph {
    const float* params = nullptr;
    const float* x = nullptr;
    const int32_t* y = nullptr;
    bool mom_valid = false, profiling = false;
    cudaGraph_t graph = nullptr;
    cudaGraphExec_t exec = nullptr;
    struct PhaseNodes { int phase; cudaGraphNode_t a, b; };   // the profile's event-record nodes
    std::vector<PhaseNodes> phase_nodes;
    int64_t launches[HS_PHASE_COUNT] = {0};                   // kernel launches of one step, by phase
    uint64_t last_use = 0;
  };
  bool graph_on = true;
  bool graph_force = false;       // HS_STEP_GRAPH=1: also for the largest steps
  bool graph_warm = false;        // a step ran eagerly since the last invalidation (kernels loaded)
  bool capturing = false;         // the step's work is being captured (phase events become nodes)
  uint64_t graph_clock = 0;
  std::vector<StepGraph> graphs;  // at most kMaxStepGraphs, least recently used replaced
  float* d_lr = nullptr;
  cudaStream_t cap_stream = nullptr;

  cudaEvent_t take_event() {
    if (!event_pool.empty()) {
      cudaEvent_t e = event_pool.back();
      event_pool.pop_back();
      return e;
    }
    cudaEvent_t e = nullptr;
    if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
    return e;
  }

  // slab-free formulation (opt-in): worker weights folded into the per-sample loss-gradient scale,
  // one weight-gradient product over all rows into slab 0, and the update with a single "worker"
  bool fused_sync = false;
  float* d_scale_fused = nullptr;      // [N] w_{m(i)} / n_{m(i)}
  int32_t* d_all_off = nullptr;        // {0, N}
  float* d_w_one = nullptr;            // {1.0f}
  hs::ChunkTable all_rows;             // bias-gradient chunks over all rows, one worker
  std::vector<hs::TcGemmParams> tc_wgrad_fused;   // per layer, one group spanning all rows

  // compute-power history (Section 4.1): 0 = last measurement, 1 = EMA, 2 = window mean
  int cp_hist_mode = 0;
  double cp_hist_param = 0.0;
  std::vector<double> cp_ema;
  std::vector<std::vector<double>> cp_window;

  // training recipe of the paper's experiments (Section 5): momentum + weight decay in the update
  bool opt_recipe = false;
  float opt_momentum = 0.f, opt_weight_decay = 0.f;
  float* d_mom = nullptr;      // momentum buffer [Ps]
  bool mom_valid = false;      // false: the next step starts the buffer (b = d)

  // per-layer updates overlapped with the rest of the backward pass (bf16 MLP): a side stream that
  // waits for each layer's backward, and the event the caller's stream waits for at the end
  bool overlap_update = false;
  cudaStream_t upd_stream = nullptr;
  std::vector<cudaEvent_t> upd_ready;
  cudaEvent_t upd_done = nullptr;
  cudaEvent_t dgrad_done = nullptr;   // the step's last input-gradient product has read d_shadow

  // CNN workload: convs[0..2], then the fully connected layer (index 3 in per-layer arrays)
  int64_t in_features = 0;
  std::vector<hs::ConvLayer> convs;
  int64_t fc_w_off = 0, fc_b_off = 0;
  void* d_col[3] = {nullptr, nullptr, nullptr};
  void* d_cact[3] = {nullptr, nullptr, nullptr};
  void* d_pooled = nullptr;
  float* d_dpooled = nullptr;
  void* d_dA[3] = {nullptr, nullptr, nullptr};
  float* d_dcol = nullptr;
  __nv_bfloat16* d_wperm[3] = {nullptr, nullptr, nullptr};   // bf16 [Cout][Kp], tap-major columns
  __nv_bfloat16* d_ones = nullptr;                           // bf16 [64][64], column 0 ones (implicit convs)
  __nv_bfloat16* d_wsub[3] = {nullptr, nullptr, nullptr};    // bf16 sub-pixel class weights, 9 x Cout x Cin
  int32_t* d_row_off[4] = {nullptr, nullptr, nullptr, nullptr};
  hs::ChunkTable cnn_chunks[4];
  hs::CnnWgrad cnn_wgrad[4];
  bool cnn_fuse_update = true;        // HS_CNN_FUSED_UPDATE=0: split-K reductions, slab update and permutations apart
  bool conv_first_on = false;         // bf16: the first convolution's forward in one kernel (conv_first_plan)
  bool subpixel_comb = true;          // sub-pixel input gradients as one product over all four classes
  bool cnn_fc_pool = true;            // bf16 CNN: the fc layer's forward and input gradient inside the pooling kernels
                                      // (HS_SUBPIXEL=classes: one group per class); per layer where its
                                      // input has a multiple of 64 channels (ConvLayer::comb)
  hs::ConvFirstParams conv_first{};
  const float* cnn_wcopy_src = nullptr;   // the params the bf16 weight copies (wperm, wsub) were last written from

  // tensor-core launch parameters (bf16 precision)
  // per-worker weight gradients averaged in tensor memory and applied in the same kernel
  // (launch_tc_wgrad_avg): per layer, valid where avg_ok[l]; tmT points at avg_theta's weights
  bool tile_avg = false;
  bool tile_avg_all = false;   // also layers with fewer weight tiles than SM pairs
  std::vector<hs::TcGemmParams> tc_wgrad_avg;
  std::vector<char> avg_ok;
  const float* avg_theta = nullptr;
  bool avg_recipe = false;     // the maps are bound for the momentum recipe's update
  bool tile_step = false;   // the last step used it for some layer (its slabs lack those weight ranges)
  std::vector<hs::TcGemmParams> tc_fwd;                // per layer
  std::vector<hs::TcGemmParams> tc_dgrad;              // per layer (index 0 unused)
  std::vector<std::vector<hs::TcGemmParams>> tc_wgrad; // per layer, per chunk of <= 32 workers

  size_t act_elem() const { return precision == HS_BF16 ? 2 : 4; }
  int delta_ld(int l) const { return l == L - 1 ? Cp : layers[l].out; }     // l: 0-based layer
  void* delta_buf(int l) const { return d_delta[(L - 1 - l) & 1]; }
};

namespace hs {

class PhaseScope {
 public:
  PhaseScope(hs_ctx* c, int phase, cudaStream_t s) : c_(c), phase_(phase), s_(s) {
    if (c_->profiling) {
      a_ = c_->take_event();
      if (a_) record(a_);
    }
  }
  ~PhaseScope() {
    if (c_->profiling && a_) {
      cudaEvent_t b = c_->take_event();
      if (b) {
        record(b);
        c_->pending.push_back({phase_, a_, b});
      }
    }
  }
  void launched(int n = 1) { c_->launches[phase_] += n; }

 private:
  // under capture the record becomes an event-record node of the step's graph
  void record(cudaEvent_t e) {
    if (c_->capturing) cudaEventRecordWithFlags(e, s_, cudaEventRecordExternal);
    else cudaEventRecord(e, s_);
  }
  hs_ctx* c_;
  int phase_;
  cudaStream_t s_;
  cudaEvent_t a_ = nullptr;
};

inline hs_status fail(hs_ctx* c, hs_status s, const std::string& msg) {
  if (c) c->err = msg; else set_init_error(msg.c_str());
  return s;
}

inline hs_status cuda_fail(hs_ctx* c, cudaError_t e, const char* what) {
  return fail(c, e == cudaErrorMemoryAllocation ? HS_ERR_OOM : HS_ERR_CUDA,
              std::string(what) + ": " + cudaGetErrorString(e));
}

#define HS_CUDA(ctx, call)                                   \
  do {                                                       \
    cudaError_t e_ = (call);                                 \
    if (e_ != cudaSuccess) return cuda_fail(ctx, e_, #call); \
  } while (0)

template <typename T>
inline hs_status dalloc(hs_ctx* c, T** p, size_t bytes) {
  *p = nullptr;
  if (bytes == 0) bytes = 16;
  cudaError_t e = cudaMalloc(reinterpret_cast<void**>(p), bytes);
  if (e != cudaSuccess) return cuda_fail(c, e, "cudaMalloc");
  return HS_OK;
}

// CNN workload (csrc/cnn.cu)
hs_status cnn_build_static(hs_ctx* c);
hs_status cnn_build_partition_plans(hs_ctx* c);
hs_status cnn_step(hs_ctx* c, float* params, const float* x, const int32_t* y, cudaStream_t s);
// bf16 CNN without debug read-back: one kernel sums the split-K parts per worker, synchronises,
// updates theta and writes the bf16 copies the next step reads (cnn_update_kernel)
bool cnn_fused_update(const hs_ctx* c);
hs_status cnn_refresh_weights(hs_ctx* c, const float* params, cudaStream_t s);
hs_status launch_cnn_update(hs_ctx* c, float* params, float lr, const float* lr_dev, cudaStream_t s);
// The first convolution's forward in one kernel where its shape allows (HS_CONV_FIRST=0: never)
bool conv_first_ok(const ConvLayer& L);
hs_status conv_first_plan(hs_ctx* c, ConvFirstParams* p);
// Points the input map at x (re-encoded only when x changes); false: x is not addressable by TMA
// (the generic path runs instead)
bool conv_first_bind_input(hs_ctx* c, const float* x);
cudaError_t launch_conv_first(const ConvFirstParams& p, int num_sms, cudaStream_t s);

}  // namespace hs
