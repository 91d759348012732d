// C ABI of the Oscars hot path: context, schedule, round orchestration.
//
// One context simulates the parameter server and its W workers on one GPU
// (Introduction: parameter-server architecture; Problem Formulation and
// Algorithm 1: the load-balanced barrier; Eq. 4: local steps and merge).
//
// Device memory of a context (MLP mode):
//   slab    (W+1) slots x P_pad fp32   slots 0..W-1 worker replicas (the
//                                      pushed models), slot W the global model
//   shadow  (W+1) x P_pad bf16         bf16 copy of every slot (GEMM operand;
//                                      read MN-major by the input-gradient GEMM)
//   per-worker activations, gradients, labels, loss partials, cursors.
// Inside a slot every W_l and b_l starts on a 64-element boundary; the
// padding stays zero.
#include <algorithm>
#include <limits>
#include <cstdio>
#include <cstring>
#include <new>
#include <string>
#include <vector>

#include "../../include/oscars.h"
#include "common.cuh"
#include "internal.h"

using namespace oscars;

namespace {

int64_t round_up(int64_t x, int64_t m) { return (x + m - 1) / m * m; }

constexpr int kMaxBranches = 16;
// blocks of the per-layer round's staging when it reads host-resident shards
// (16 KB of rows in flight per block; 48 to 76 blocks measured within 2% of
// one another on the 3072-1024-1024-10 MLP with 32 workers, 128 and the full
// grid up to 25% slower per round)
constexpr int kHostStageBlocks = 64;

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

// 3-D bf16 tensor map: element (x, y, z) at base + z*stride_z + y*stride_y +
// 2x bytes; boxes of 64 (x) by box_y rows, 128-byte swizzle, zero fill
// outside the extents.
bool make_map(CUtensorMap* m, const void* base, uint64_t dx, uint64_t dy, uint64_t dz, uint64_t stride_y,
              uint64_t stride_z, uint32_t box_y) {
  EncodeTiledFn f = encode_fn();
  if (!f) return false;
  cuuint64_t dims[3] = {dx, dy, dz};
  cuuint64_t strides[2] = {stride_y, stride_z};
  cuuint32_t box[3] = {64, box_y, 1};
  cuuint32_t es[3] = {1, 1, 1};
  return f(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, es,
           CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
           CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// 4-D bf16 tensor map, boxes of 64 x box_y x 1 x 1, 128-byte swizzle
bool make_map4(CUtensorMap* m, const void* base, uint64_t d0, uint64_t d1, uint64_t d2, uint64_t d3, uint64_t s1,
               uint64_t s2, uint64_t s3, uint32_t box_y) {
  EncodeTiledFn f = encode_fn();
  if (!f) return false;
  cuuint64_t dims[4] = {d0, d1, d2, d3};
  cuuint64_t strides[3] = {s1, s2, s3};
  cuuint32_t box[4] = {64, box_y, 1, 1};
  cuuint32_t es[4] = {1, 1, 1, 1};
  return f(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box, es,
           CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
           CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// 4-D bf16 tensor map with an explicit box, 128-byte swizzle, zero fill
bool make_map_box4(CUtensorMap* m, const void* base, const uint64_t (&d)[4], const uint64_t (&st)[3],
                   const uint32_t (&box)[4]) {
  EncodeTiledFn f = encode_fn();
  if (!f) return false;
  cuuint64_t dims[4] = {d[0], d[1], d[2], d[3]};
  cuuint64_t strides[3] = {st[0], st[1], st[2]};
  cuuint32_t bx[4] = {box[0], box[1], box[2], box[3]};
  cuuint32_t es[4] = {1, 1, 1, 1};
  return f(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, bx, es,
           CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
           CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// 3-D fp32 tensor map, boxes of 32 x box_y x 1 (128-byte rows), 128-byte swizzle
bool make_map_f32(CUtensorMap* m, const void* base, uint64_t dx, uint64_t dy, uint64_t dz, uint64_t stride_y,
                  uint64_t stride_z, uint32_t box_y, uint32_t box_x = 32,
                  CUtensorMapSwizzle swz = CU_TENSOR_MAP_SWIZZLE_128B) {
  EncodeTiledFn f = encode_fn();
  if (!f) return false;
  cuuint64_t dims[3] = {dx, dy, dz};
  cuuint64_t strides[2] = {stride_y, stride_z};
  cuuint32_t box[3] = {box_x, box_y, 1};
  cuuint32_t es[3] = {1, 1, 1};
  return f(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, const_cast<void*>(base), dims, strides, box, es,
           CU_TENSOR_MAP_INTERLEAVE_NONE, swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
           CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

struct Layer {
  int in, out;
  int64_t offW, offB;
};

}  // namespace

struct oscars_ctx {
  // configuration
  int W = 0, model = 0, L = 0, B = 0, C = 0;
  std::vector<int> dims;
  float lr = 0.f, server_lr = 1.f;
  int rule = 0, bf16 = 0, flags = 0;
  int64_t P = 0, P_pad = 0;
  std::vector<Layer> layers;
  // schedule (Eq. 1-3, Algorithm 1)
  std::vector<int64_t> t_iter, clock, idle;
  std::vector<int32_t> tau;
  int64_t T_star = 0, max_wait = 0, M = 0, barrier = 0;
  int search_mode = 0, max_tau = 0;
  std::vector<int> n_active;  // per local step
  // data (borrowed)
  std::vector<const float*> shard_x;
  std::vector<const int32_t*> shard_y;
  std::vector<int64_t> shard_n;
  // device memory
  std::vector<void*> allocs;
  float* slab = nullptr;
  __nv_bfloat16* shadow = nullptr;
  std::vector<__nv_bfloat16*> A, AT, G, GT;  // per layer
  std::vector<float*> gb;
  int32_t* labels = nullptr;
  float* dlog = nullptr;
  float* loss_part = nullptr;
  float* loss_dev = nullptr;
  int64_t* cursor = nullptr;
  int32_t* tau_dev = nullptr;
  int32_t* order_dev = nullptr;         // workers of the round kernel, cluster by cluster (longest first)
  int32_t* cl_first_dev = nullptr;      // [n_clusters + 1] first entry of each cluster in order_dev
  int n_clusters = 0;                   // clusters of the round kernel
  int fused_max_clusters = 0;           // clusters of the round kernel that fit on the device at once
  int* act_wid = nullptr;  // [max_tau][W]
  int32_t* stage_slots = nullptr;   // [sum tau] active staging slots s * W + w, step-major
  int n_stage_slots = 0;
  int* act_src = nullptr;
  int* lane_ids = nullptr;   // [W] 0..W-1
  int* global_src = nullptr; // [W] all = W
  const float** dx_tab = nullptr;
  const int32_t** dy_tab = nullptr;
  int64_t* dn_tab = nullptr;
  int* err = nullptr;
  // eval scratch
  const float** ex_tab = nullptr;
  const int32_t** ey_tab = nullptr;
  int64_t* en_tab = nullptr;
  int64_t* estart = nullptr;
  int64_t estart_cap = 0;
  float* eval_part = nullptr;
  int64_t eval_part_cap = 0;
  // tensor maps per layer
  std::vector<CUtensorMap> mShadow, mShadowMN, mA, mG, mGT, mAT;
  // G^T [lane][out][B] in boxes of 64 x 64: the MN-major B operand of the input
  // gradient.  With it (g_rows false: B a multiple of 64 and the tensor-core
  // head) the row-major output gradients G are neither kept nor written.
  std::vector<CUtensorMap> mGTmn;
  bool g_rows = true;
  // fp32 W_l of every slot: boxes {32, 128} (loads) and {32, 32} (stores), and
  // the bf16 copy with boxes {64, 32} (stores): the persistent weight gradient
  std::vector<CUtensorMap> mMaster, mMasterSt, mShadowSt;
  // the last layer's input [lane][B][H] (box {64, 128}) and weights of every slot (box {64, 16})
  CUtensorMap mHeadIn, mHeadW;
  // per-step input buffers of layer 0 (a round's mini-batches are staged at once)
  int stage_cap = 0;
  __nv_bfloat16* A0all = nullptr;
  __nv_bfloat16* A0Tall = nullptr;
  int32_t* labels_all = nullptr;
  std::vector<CUtensorMap> mA0s, mAT0s;
  bool fused = false;                   // whole-round kernel (2-layer MLP)
  bool ahead_mlp = false;               // per-layer bf16 MLP round that stages the next round beside it
  bool shards_host = false;             // some shard's samples live in host memory
  int cur_buf = 0;                      // ahead_mlp: the input buffer the round being enqueued reads
  std::vector<CUtensorMap> mA0p[2], mAT0p[2];   // ahead_mlp: per-step maps of each input buffer
  // the one-launch round (and ahead_mlp) stages the next round while the
  // current one runs: two input buffers, used alternately (index `parity`
  // holds the next round)
  __nv_bfloat16* A0b[2] = {};
  __nv_bfloat16* A0Tb[2] = {};
  int32_t* labb[2] = {};
  CUtensorMap mX4b[2], mXT4b[2];
  CUtensorMap mW0f;                     // the global slot's fp32 W0 for the round kernel
  CUtensorMap mRep32, mRep16;           // every replica slot's W0 (the round kernel's last-step stores)
  int parity = 0;
  bool staged = false;                  // A0b[parity] holds the mini-batches of the next round
  cudaGraphExec_t ahead_exec[2] = {};   // round graphs, one per parity
  unsigned long long* phase_ts = nullptr;   // flag bit 4: phase stamps of the fused round
  // convolutional worker (OSCARS_MODEL_CNN)
  int cnn_blocks = 0, cnn_chunks = 0;
  std::vector<int64_t> cnn_offW, cnn_offB;   // conv layers: stem, then (a, b) of every block
  int64_t cnn_offWf = 0, cnn_offBf = 0;
  int64_t cnn_wt_slot = 0;                   // elements per slot of the transposed copies
  bool cnn_im2col = false;                   // stem over the im2col input (9 Cin <= 64): weights [64 out][64 k]
  __nv_bfloat16* cnn_wt = nullptr;           // [slot][2 * blocks][9][64 in][64 out]
  std::vector<__nv_bfloat16*> cnn_buf;       // x, s, (u_k, v_k) per block, dz0, dz1, dz2: [W][B][1024][64]
  std::vector<CUtensorMap> cnn_m6, cnn_m4, cnn_m2;   // per buffer: boxes of 6, 4 and 2 image rows
  int sms = 0;                               // multiprocessors of the device
  std::vector<CUtensorMap> cnn_mw, cnn_mwt;  // weights per conv layer: forward layout, transposed (blocks)
  float* cnn_g = nullptr;                    // [W][B][64] pooled features
  float* cnn_dg = nullptr;                   // [W][B][64] their gradient
  float* cnn_wpart = nullptr;                // [layer][W][chunks][9][64][64]
  float* cnn_bpart = nullptr;                // [layer][W][B * 8][64]
  // streams / graph
  cudaStream_t stream = nullptr;
  cudaStream_t cap = nullptr;
  // concurrent branches of a round: workers are independent between merges,
  // so each branch runs the local steps of its own workers on its own stream
  int n_br = 1;
  std::vector<cudaStream_t> br_streams;
  std::vector<cudaEvent_t> br_join;
  cudaEvent_t br_fork = nullptr;
  // one-launch rounds: the next round's staging runs beside the round on a
  // side stream, at the lowest launch priority (the round at the highest)
  cudaStream_t side = nullptr;
  cudaEvent_t side_fork = nullptr, side_join = nullptr;
  int prio_least = 0, prio_greatest = 0;
  std::vector<int> br_max_tau;          // [n_br]
  std::vector<int> br_na;               // [n_br][max_tau] active workers per step
  int* br_wid = nullptr;                // [n_br][max_tau][W]
  int* br_src = nullptr;
  cudaGraphExec_t round_exec = nullptr;
  bool pending = false;
  int64_t rounds_run = 0;               // oscars_local_steps calls that launched a round
  std::string last_error;
  // per-kernel-class CUDA-event profile (flag bit 1, direct launches only)
  struct ProfEntry {
    const char* name;
    cudaEvent_t a, b;
    bool graph_owned;   // recorded by an event node of a captured graph: never recycled
  };
  std::vector<ProfEntry> prof_pending;
  std::vector<ProfEntry> prof_round_graph, prof_merge_graph;   // event nodes of the captured graphs
  std::vector<ProfEntry> prof_ahead_graph[2];                   // event nodes of the two parity round graphs
  std::vector<ProfEntry>* prof_sink = nullptr;                  // where ProfScope files entries
  cudaGraphExec_t merge_exec = nullptr;                         // replica-mode merge + shadow refresh
  std::vector<cudaEvent_t> prof_pool;
  std::vector<std::string> prof_names;
  std::vector<double> prof_ms;
  std::vector<int> prof_count;
  bool profiling = false;
  // oscars_train without evaluation: two pinned host slots for the per-worker
  // losses and one event per slot (rounds pipelined one deep)
  float* train_loss_host = nullptr;
  cudaEvent_t train_done[2] = {nullptr, nullptr};
};

namespace {

oscars_status fail(oscars_ctx* c, oscars_status s, const std::string& msg) {
  if (c) c->last_error = msg;
  return s;
}

oscars_status cuda_fail(oscars_ctx* c, cudaError_t e, const char* where) {
  return fail(c, OSCARS_ECUDA, std::string(where) + ": " + cudaGetErrorString(e));
}

// ---- profiler: events around each launch on the launching stream
cudaEvent_t prof_event(oscars_ctx* c) {
  if (!c->prof_pool.empty()) {
    cudaEvent_t e = c->prof_pool.back();
    c->prof_pool.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  cudaEventCreate(&e);
  return e;
}

// Events around one launch.  Recorded with cudaEventRecordExternal, so that
// inside a stream capture they become event nodes of the graph and time the
// kernel on the device timeline (no host launch gaps).
struct ProfScope {
  oscars_ctx* c;
  const char* name;
  cudaStream_t s;
  cudaEvent_t a = nullptr;
  // an event record is an event node of the graph while a round is captured
  // (prof_sink set), a plain record otherwise
  unsigned flags() const { return c->prof_sink ? cudaEventRecordExternal : cudaEventRecordDefault; }
  ProfScope(oscars_ctx* c_, const char* n, cudaStream_t s_) : c(c_), name(n), s(s_) {
    if (c->profiling) {
      a = prof_event(c);
      cudaEventRecordWithFlags(a, s, flags());
    }
  }
  ~ProfScope() {
    if (a) {
      cudaEvent_t b = prof_event(c);
      cudaEventRecordWithFlags(b, s, flags());
      if (c->prof_sink)
        c->prof_sink->push_back({name, a, b, true});
      else
        c->prof_pending.push_back({name, a, b, false});
    }
  }
};

// fold finished event pairs into per-name totals (synchronises)
void prof_collect(oscars_ctx* c) {
  if (c->prof_pending.empty()) return;
  cudaEventSynchronize(c->prof_pending.back().b);
  for (auto& p : c->prof_pending) {
    float ms = 0.f;
    cudaEventElapsedTime(&ms, p.a, p.b);
    size_t i = 0;
    while (i < c->prof_names.size() && c->prof_names[i] != p.name) ++i;
    if (i == c->prof_names.size()) {
      c->prof_names.push_back(p.name);
      c->prof_ms.push_back(0.0);
      c->prof_count.push_back(0);
    }
    c->prof_ms[i] += ms;
    c->prof_count[i] += 1;
    if (!p.graph_owned) {
      c->prof_pool.push_back(p.a);
      c->prof_pool.push_back(p.b);
    }
  }
  c->prof_pending.clear();
}

// after a replay of a profiled graph: queue its event nodes for collection
void prof_after_replay(oscars_ctx* c, const std::vector<oscars_ctx::ProfEntry>& g) {
  if (g.empty()) return;
  for (const auto& e : g) c->prof_pending.push_back(e);
  prof_collect(c);   // read now: the next replay records the same events again
}

// guard words after the model slab and after its bf16 copy: a byte pattern
// written at creation that no kernel writes (oscars_check_padding reads it)
constexpr size_t kGuardWords = 256;
constexpr int kGuardByte = 0xA5;

template <typename T>
bool dev_alloc(oscars_ctx* c, T** p, size_t count) {
  void* q = nullptr;
  if (count == 0) count = 1;
  if (cudaMalloc(&q, count * sizeof(T)) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  c->allocs.push_back(q);
  *p = static_cast<T*>(q);
  return true;
}

void free_all(oscars_ctx* c) {
  for (auto& p : c->prof_pending)
    if (!p.graph_owned) {
      cudaEventDestroy(p.a);
      cudaEventDestroy(p.b);
    }
  c->prof_pending.clear();
  for (auto* v : {&c->prof_round_graph, &c->prof_merge_graph, &c->prof_ahead_graph[0], &c->prof_ahead_graph[1]}) {
    for (auto& p : *v) {
      cudaEventDestroy(p.a);
      cudaEventDestroy(p.b);
    }
    v->clear();
  }
  if (c->merge_exec) cudaGraphExecDestroy(c->merge_exec);
  c->merge_exec = nullptr;
  for (cudaEvent_t e : c->prof_pool) cudaEventDestroy(e);
  c->prof_pool.clear();
  for (auto& e : c->train_done) {
    if (e) cudaEventDestroy(e);
    e = nullptr;
  }
  if (c->train_loss_host) cudaFreeHost(c->train_loss_host);
  c->train_loss_host = nullptr;
  if (c->round_exec) cudaGraphExecDestroy(c->round_exec);
  c->round_exec = nullptr;
  for (auto& g : c->ahead_exec) {
    if (g) cudaGraphExecDestroy(g);
    g = nullptr;
  }
  for (void* p : c->allocs) cudaFree(p);
  c->allocs.clear();
  if (c->cap) cudaStreamDestroy(c->cap);
  c->cap = nullptr;
  for (cudaStream_t b : c->br_streams) cudaStreamDestroy(b);
  c->br_streams.clear();
  for (cudaEvent_t e : c->br_join) cudaEventDestroy(e);
  c->br_join.clear();
  if (c->br_fork) cudaEventDestroy(c->br_fork);
  c->br_fork = nullptr;
  if (c->side) cudaStreamDestroy(c->side);
  c->side = nullptr;
  for (auto* e : {&c->side_fork, &c->side_join}) {
    if (*e) cudaEventDestroy(*e);
    *e = nullptr;
  }
}

// Simulated barrier and idle time per worker for the current tau (Eq. 1).
void update_barrier(oscars_ctx* c, bool from_search) {
  if (from_search) {
    c->barrier = c->T_star;
  } else {
    int64_t b = 0;
    for (int i = 0; i < c->W; ++i) b = std::max(b, static_cast<int64_t>(c->tau[i]) * c->t_iter[i]);
    c->barrier = b;
  }
}

// Layer-0 inputs and labels for every local step of a round ([max_tau][W][...])
// and one pair of tensor maps per step.  Grows when tau grows.
oscars_status ensure_stage_buffers(oscars_ctx* c) {
  if (!(c->bf16 && c->L >= 2) || c->stage_cap >= c->max_tau) return OSCARS_OK;
  const int W = c->W, B = c->B, D = c->dims[0];
  const size_t per = static_cast<size_t>(W) * B * D;
  const int cap = c->max_tau;
  if (!dev_alloc(c, &c->A0all, per * cap) || !dev_alloc(c, &c->A0Tall, per * cap) ||
      !dev_alloc(c, &c->labels_all, static_cast<size_t>(W) * B * cap))
    return fail(c, OSCARS_ENOMEM, "device allocation failed (per-step inputs)");
  c->mA0s.resize(cap);
  c->mAT0s.resize(cap);
  for (int s = 0; s < cap; ++s) {
    if (!make_map(&c->mA0s[s], c->A0all + per * s, D, B, W, D * 2ull, static_cast<uint64_t>(B) * D * 2ull, B) ||
        !make_map(&c->mAT0s[s], c->A0Tall + per * s, B, D, W, B * 2ull, static_cast<uint64_t>(B) * D * 2ull, 128))
      return fail(c, OSCARS_ECUDA, "cuTensorMapEncodeTiled failed (per-step inputs)");
  }
  if (c->fused && (c->flags & 16) &&
      !dev_alloc(c, &c->phase_ts, static_cast<size_t>(cap) * 4))   // stamps of every step (flag bit 4)
    return fail(c, OSCARS_ENOMEM, "device allocation failed (phase stamps)");
  if (c->fused || c->ahead_mlp) {
    c->A0b[0] = c->A0all;
    c->A0Tb[0] = c->A0Tall;
    c->labb[0] = c->labels_all;
    if (!dev_alloc(c, &c->A0b[1], per * cap) || !dev_alloc(c, &c->A0Tb[1], per * cap) ||
        !dev_alloc(c, &c->labb[1], static_cast<size_t>(W) * B * cap))
      return fail(c, OSCARS_ENOMEM, "device allocation failed (second input buffer)");
  }
  if (c->ahead_mlp) {   // the per-step maps of both input buffers
    for (int b = 0; b < 2; ++b) {
      c->mA0p[b].resize(cap);
      c->mAT0p[b].resize(cap);
      for (int s = 0; s < cap; ++s)
        if (!make_map(&c->mA0p[b][s], c->A0b[b] + per * s, D, B, W, D * 2ull, static_cast<uint64_t>(B) * D * 2ull, B) ||
            !make_map(&c->mAT0p[b][s], c->A0Tb[b] + per * s, B, D, W, B * 2ull, static_cast<uint64_t>(B) * D * 2ull,
                      128))
          return fail(c, OSCARS_ECUDA, "cuTensorMapEncodeTiled failed (per-step inputs)");
    }
  }
  if (c->fused) {
    const uint64_t per_b = static_cast<uint64_t>(per) * 2;
    for (int i = 0; i < 2; ++i)
      if (!make_map4(&c->mX4b[i], c->A0b[i], D, B, W, cap, D * 2ull, static_cast<uint64_t>(B) * D * 2ull, per_b, B) ||
          !make_map4(&c->mXT4b[i], c->A0Tb[i], B, D, W, cap, B * 2ull, static_cast<uint64_t>(B) * D * 2ull, per_b,
                     fused_round_xt_rows(B)))
        return fail(c, OSCARS_ECUDA, "cuTensorMapEncodeTiled failed (fused round inputs)");
    // the global slot's W0: fp32 tiles of 128 rows x 32 columns
    const int64_t gw0 = static_cast<int64_t>(W) * c->P_pad + c->layers[0].offW;
    const uint64_t H = static_cast<uint64_t>(c->dims[1]);
    // every replica slot's W0, for the last step's stores: boxes of 32 rows
    // x 32 (swizzled) and x 16 columns
    const int64_t rw0 = c->layers[0].offW;
    const uint64_t slots = static_cast<uint64_t>(W);
    if (!make_map_f32(&c->mW0f, c->slab + gw0, D, H, 1, D * 4ull, D * H * 4ull, 128) ||
        !make_map_f32(&c->mRep32, c->slab + rw0, D, H, slots, D * 4ull, static_cast<uint64_t>(c->P_pad) * 4ull, 32) ||
        !make_map_f32(&c->mRep16, c->slab + rw0, D, H, slots, D * 4ull, static_cast<uint64_t>(c->P_pad) * 4ull, 32, 16,
                      CU_TENSOR_MAP_SWIZZLE_NONE))
      return fail(c, OSCARS_ECUDA, "cuTensorMapEncodeTiled failed (fused round model)");
  }
  // step 0 doubles as the single-step buffers (evaluation)
  c->A[0] = c->A0all;
  c->AT[0] = c->A0Tall;
  c->labels = c->labels_all;
  c->mA[0] = c->mA0s[0];
  c->mAT[0] = c->mAT0s[0];
  c->stage_cap = cap;
  return OSCARS_OK;
}

oscars_status build_tables(oscars_ctx* c) {
  c->max_tau = 0;
  for (int i = 0; i < c->W; ++i) c->max_tau = std::max(c->max_tau, static_cast<int>(c->tau[i]));
  c->n_active.assign(c->max_tau, 0);
  std::vector<int> wid(static_cast<size_t>(c->max_tau) * c->W, 0), src(wid.size(), 0);
  for (int s = 0; s < c->max_tau; ++s) {
    int n = 0;
    for (int i = 0; i < c->W; ++i)
      if (c->tau[i] > s) {
        wid[static_cast<size_t>(s) * c->W + n] = i;
        src[static_cast<size_t>(s) * c->W + n] = s == 0 ? c->W : i;  // first step reads the global model
        ++n;
      }
    c->n_active[s] = n;
  }
  // branches: workers sorted by tau (descending), dealt round-robin
  std::vector<int> order(c->W);
  for (int i = 0; i < c->W; ++i) order[i] = i;
  std::stable_sort(order.begin(), order.end(), [&](int x, int y) { return c->tau[x] > c->tau[y]; });
  std::vector<std::vector<int>> members(c->n_br);
  for (int j = 0; j < c->W; ++j) members[j % c->n_br].push_back(order[j]);
  c->br_max_tau.assign(c->n_br, 0);
  c->br_na.assign(static_cast<size_t>(c->n_br) * c->max_tau, 0);
  std::vector<int> bw(static_cast<size_t>(c->n_br) * c->max_tau * c->W, 0), bs(bw.size(), 0);
  for (int g = 0; g < c->n_br; ++g) {
    std::sort(members[g].begin(), members[g].end());
    for (int s = 0; s < c->max_tau; ++s) {
      int n = 0;
      for (int i : members[g])
        if (c->tau[i] > s) {
          const size_t at = (static_cast<size_t>(g) * c->max_tau + s) * c->W + n;
          bw[at] = i;
          bs[at] = s == 0 ? c->W : i;
          ++n;
        }
      c->br_na[static_cast<size_t>(g) * c->max_tau + s] = n;
      if (n > 0) c->br_max_tau[g] = s + 1;
    }
  }
  if (!dev_alloc(c, &c->br_wid, bw.size()) || !dev_alloc(c, &c->br_src, bs.size()))
    return fail(c, OSCARS_ENOMEM, "device allocation failed (branch tables)");
  {
    cudaError_t e = cudaMemcpy(c->br_wid, bw.data(), bw.size() * sizeof(int), cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMemcpy(c->br_src, bs.data(), bs.size() * sizeof(int), cudaMemcpyHostToDevice);
    if (e != cudaSuccess) return cuda_fail(c, e, "branch table upload");
  }
  std::vector<int32_t> slots;
  for (int st = 0; st < c->max_tau; ++st)
    for (int i = 0; i < c->W; ++i)
      if (c->tau[i] > st) slots.push_back(st * c->W + i);
  c->n_stage_slots = static_cast<int>(slots.size());
  if (!dev_alloc(c, &c->stage_slots, slots.size()))
    return fail(c, OSCARS_ENOMEM, "device allocation failed (staging slots)");
  {
    const cudaError_t e = cudaMemcpy(c->stage_slots, slots.data(), slots.size() * sizeof(int32_t), cudaMemcpyHostToDevice);
    if (e != cudaSuccess) return cuda_fail(c, e, "staging slot upload");
  }
  if (!dev_alloc(c, &c->act_wid, wid.size()) || !dev_alloc(c, &c->act_src, src.size()) ||
      !dev_alloc(c, &c->loss_part, static_cast<size_t>(c->W) * c->max_tau * std::max(1, c->B / kRowsPerLossChunk)))
    return fail(c, OSCARS_ENOMEM, "device allocation failed (schedule tables)");
  cudaError_t e = cudaMemcpy(c->act_wid, wid.data(), wid.size() * sizeof(int), cudaMemcpyHostToDevice);
  if (e == cudaSuccess) e = cudaMemcpy(c->act_src, src.data(), src.size() * sizeof(int), cudaMemcpyHostToDevice);
  if (e == cudaSuccess) e = cudaMemcpy(c->tau_dev, c->tau.data(), c->W * sizeof(int32_t), cudaMemcpyHostToDevice);
  if (e == cudaSuccess) {
    // Round-kernel clusters: one per worker when they all fit on the device,
    // else as many as fit, each running its workers one after the other
    // (longest processing time first: oscars_round_clusters)
    std::vector<int32_t> flat(c->W), first(static_cast<size_t>(c->W) + 1);
    int32_t ncl = 0;
    if (oscars_round_clusters(c->tau.data(), c->W, c->fused_max_clusters, flat.data(), first.data(), &ncl) !=
        OSCARS_OK)
      return fail(c, OSCARS_EINVAL, "round cluster plan");
    first.resize(static_cast<size_t>(ncl) + 1);
    c->n_clusters = ncl;
    if (!c->order_dev && !dev_alloc(c, &c->order_dev, c->W))
      return fail(c, OSCARS_ENOMEM, "device allocation failed (worker order)");
    if (!c->cl_first_dev && !dev_alloc(c, &c->cl_first_dev, c->W + 1))
      return fail(c, OSCARS_ENOMEM, "device allocation failed (cluster table)");
    e = cudaMemcpy(c->order_dev, flat.data(), c->W * sizeof(int32_t), cudaMemcpyHostToDevice);
    if (e == cudaSuccess)
      e = cudaMemcpy(c->cl_first_dev, first.data(), first.size() * sizeof(int32_t), cudaMemcpyHostToDevice);
  }
  if (e != cudaSuccess) return cuda_fail(c, e, "schedule upload");
  if (c->round_exec) {
    cudaGraphExecDestroy(c->round_exec);
    c->round_exec = nullptr;
  }
  for (int i = 0; i < 2; ++i) {
    if (c->ahead_exec[i]) cudaGraphExecDestroy(c->ahead_exec[i]);
    c->ahead_exec[i] = nullptr;
    for (auto& p : c->prof_ahead_graph[i]) {   // the graph's event nodes go with it
      cudaEventDestroy(p.a);
      cudaEventDestroy(p.b);
    }
    c->prof_ahead_graph[i].clear();
  }
  c->staged = false;   // the staged next round used the previous tau
  if (c->merge_exec) {
    cudaGraphExecDestroy(c->merge_exec);
    c->merge_exec = nullptr;
  }
  return ensure_stage_buffers(c);
}

// bf16 copies of the global slot after it changed; `plain_done`: the merge
// already wrote the (non-transposed) shadow
cudaError_t refresh_global_shadows(oscars_ctx* c, cudaStream_t s, bool plain_done = false) {
  if (!c->shadow) return cudaSuccess;
  const int64_t g = static_cast<int64_t>(c->W) * c->P_pad;
  cudaError_t e = plain_done ? cudaSuccess : launch_shadow_refresh(c->slab + g, c->shadow + g, c->P_pad, s);
  if (e != cudaSuccess) return e;
  for (size_t l = 1; l < c->cnn_offW.size(); ++l) {   // CNN: transposed copies of the block convolutions
    e = launch_conv_refresh_wt(c->slab + g, c->cnn_wt + static_cast<int64_t>(c->W) * c->cnn_wt_slot +
                                                static_cast<int64_t>(l - 1) * 9 * 64 * 64,
                               c->cnn_offW[l], s);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

// Eq. 4, first branch, over the workers' replica slots: x_g += eta sum_k
// w_k (x^k - x_g) with the weights w, the bf16 copy of x_g in the same pass
// (and, for the CNN, its transposed copies)
cudaError_t enqueue_replica_merge(oscars_ctx* c, const float* w, cudaStream_t st) {
  MergeArgs a;
  std::memset(&a, 0, sizeof(a));
  a.W = c->W;
  for (int k = 0; k < c->W; ++k) {
    a.w[k] = w[k];
    a.src[k] = c->slab + static_cast<int64_t>(k) * c->P_pad;
  }
  const int64_t g = static_cast<int64_t>(c->W) * c->P_pad;
  cudaError_t r;
  {
    ProfScope ps(c, "merge", st);
    r = launch_merge(a, c->slab + g, c->P_pad, c->server_lr, true, st, c->shadow ? c->shadow + g : nullptr);
  }
  if (r != cudaSuccess) return r;
  if (c->model != OSCARS_MODEL_CNN) return cudaSuccess;   // no transposed copies to refresh
  ProfScope ps(c, "shadow_refresh", st);
  return refresh_global_shadows(c, st, true);
}

GemmArgs gemm_base(oscars_ctx* c, const int* wid, const int* src) {
  GemmArgs g;
  std::memset(&g, 0, sizeof(g));
  g.wid = wid;
  g.src = src;
  g.err = c->err;
  g.master = c->slab;
  g.master_w = c->slab;
  g.shadow = c->shadow;
  g.slot_stride = c->P_pad;
  g.lr = c->lr;
  return g;
}

HeadArgs head_base(oscars_ctx* c) {
  HeadArgs h;
  std::memset(&h, 0, sizeof(h));
  const Layer& ly = c->layers.back();
  h.H = ly.in;
  h.C = ly.out;
  h.B = c->B;
  h.Ain = c->A[c->L - 1];
  h.labels = c->labels;
  h.shadow = c->shadow;
  h.master = c->slab;
  h.master_w = c->slab;
  h.shadow_w = c->shadow;
  h.slot_stride = c->P_pad;
  h.offW = ly.offW;
  h.offB = ly.offB;
  h.lr = c->lr;
  h.dlog = c->dlog;
  h.err = c->err;
  if (c->L >= 2) {
    h.G = c->g_rows ? c->G[c->L - 2] : nullptr;
    h.GT = c->GT[c->L - 2];
    h.gb = c->gb[c->L - 2];
  }
  return h;
}

// the staged layer-0 inputs of local step `step` (and their labels): the
// input buffer of the round being enqueued when rounds stage ahead
const CUtensorMap& step_inputs(oscars_ctx* c, int step) {
  return c->ahead_mlp ? c->mA0p[c->cur_buf][step] : c->mA0s[step];
}
const CUtensorMap& step_inputs_t(oscars_ctx* c, int step) {
  return c->ahead_mlp ? c->mAT0p[c->cur_buf][step] : c->mAT0s[step];
}
const int32_t* step_labels(oscars_ctx* c) { return c->ahead_mlp ? c->labb[c->cur_buf] : c->labels_all; }

// forward layers 0..L-2 for `na` lanes (training step or evaluation)
cudaError_t enqueue_forward(oscars_ctx* c, const int* wid, const int* src, int na, cudaStream_t st, int step = 0) {
  for (int l = 0; l + 1 < c->L; ++l) {
    const Layer& ly = c->layers[l];
    GemmArgs g = gemm_base(c, wid, src);
    g.M = ly.out;
    g.N = c->B;
    g.K = ly.in;
    g.a_z_src = 1;
    g.b_z_src = 0;
    g.offW = ly.offW;
    g.offB = ly.offB;
    g.out = c->A[l + 1];
    g.outT = c->AT[l + 1];
    g.pdl = c->profiling ? 0 : 1;   // overlaps its prologue with the previous kernel's tail
    ProfScope ps(c, "gemm_fwd", st);
    cudaError_t e = launch_gemm(kEpiFwd, c->mShadow[l], l == 0 ? step_inputs(c, step) : c->mA[l], g, na, st);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

// One local step of the active workers `wid` (parameters from slots `src`):
// forward, last layer, and backward of the hidden layers (Eq. 4, "otherwise").
cudaError_t enqueue_step(oscars_ctx* c, int s, int na, const int* wid, const int* src, cudaStream_t st) {
  cudaError_t e;
  if ((e = enqueue_forward(c, wid, src, na, st, s)) != cudaSuccess) return e;
  HeadArgs h = head_base(c);
  h.wid = wid;
  h.src = src;
  h.labels = step_labels(c) + static_cast<size_t>(s) * c->W * c->B;
  h.loss_part = c->loss_part;
  h.part_mul = c->max_tau;
  h.part_add = s;
  if (head_tc_supported(h.H, h.B, h.C)) {
    h.pdl = c->profiling ? 0 : 1;
    ProfScope ps(c, "head_fused", st);
    if ((e = launch_head_tc(c->mHeadIn, c->mHeadW, h, na, st)) != cudaSuccess) return e;
  } else if (head_fused_supported(h.H, h.B, h.C)) {
    ProfScope ps(c, "head_fused", st);
    if ((e = launch_head_fused(h, na, st)) != cudaSuccess) return e;
  } else {
    {
      ProfScope ps(c, "head_fwd", st);
      if ((e = launch_head_fwd(h, na, st)) != cudaSuccess) return e;
    }
    ProfScope ps(c, "head_bwd", st);
    if ((e = launch_head_bwd(h, na, st)) != cudaSuccess) return e;
  }
  for (int l = c->L - 2; l >= 0; --l) {
    const Layer& ly = c->layers[l];
    if (l >= 1) {  // input gradient of layer l -> gradient of layer l-1's output
      GemmArgs g = gemm_base(c, wid, src);
      g.M = ly.in;
      g.N = c->B;
      g.K = ly.out;
      g.a_z_src = 1;
      g.b_z_src = 0;
      g.hmask = c->A[l];
      g.out = c->g_rows ? c->G[l - 1] : nullptr;
      g.b_mn = c->g_rows ? 0 : 1;
      g.pdl = c->profiling ? 0 : 1;
      g.outT = c->GT[l - 1];
      g.gb_out = c->gb[l - 1];
      ProfScope ps(c, "gemm_dh", st);
      if ((e = launch_gemm(kEpiDh, c->mShadowMN[l], c->g_rows ? c->mG[l] : c->mGTmn[l], g, na, st)) != cudaSuccess)
        return e;
    }
    const CUtensorMap& mX = l == 0 ? step_inputs_t(c, s) : c->mAT[l];
    if (gemm_dw_supported(ly.out, ly.in, c->B)) {
      DwArgs d{};
      d.wid = wid;
      d.src = src;
      d.n_active = na;
      d.M = ly.out;
      d.N = ly.in;
      d.K = c->B;
      d.lr = c->lr;
      d.master = c->slab;
      d.master_w = c->slab;
      d.slot_stride = c->P_pad;
      d.offB = ly.offB;
      d.gb = c->gb[l];
      d.err = c->err;
      d.pdl = c->profiling ? 0 : 1;
      ProfScope ps(c, "gemm_dw_sgd", st);
      if ((e = launch_gemm_dw(c->mGT[l], mX, c->mMaster[l], c->mMasterSt[l], c->mShadowSt[l], d, c->sms, st)) !=
          cudaSuccess)
        return e;
      continue;
    }
    GemmArgs g = gemm_base(c, wid, src);
    g.M = ly.out;
    g.N = ly.in;
    g.K = c->B;
    g.a_z_src = 0;
    g.b_z_src = 0;
    g.offW = ly.offW;
    g.offB = ly.offB;
    g.gb_in = c->gb[l];
    ProfScope ps(c, "gemm_dw_sgd", st);
    if ((e = launch_gemm(kEpiDw, c->mGT[l], mX, g, na, st)) != cudaSuccess) return e;
  }
  return cudaSuccess;
}

FusedRoundArgs fused_args(oscars_ctx* c) {
  FusedRoundArgs f{};
  f.tau = c->tau_dev;
  f.order = c->order_dev;
  f.cl_first = c->cl_first_dev;
  f.n_clusters = c->n_clusters;
  f.W = c->W;
  f.D = c->dims[0];
  f.H = c->dims[1];
  f.B = c->B;
  f.global_slot = c->W;
  f.lr = c->lr;
  f.master = c->slab;
  f.master_w = c->slab;
  f.slot_stride = c->P_pad;
  f.offW0 = c->layers[0].offW;
  f.offB0 = c->layers[0].offB;
  f.offW1 = c->layers[1].offW;
  f.offB1 = c->layers[1].offB;
  f.labels = c->labels_all;
  f.max_tau = c->max_tau;
  f.err = c->err;
  f.phase_ts = (c->flags & 16) ? c->phase_ts : nullptr;
  f.loss_out = c->loss_dev;
  f.cursor = c->cursor;
  f.shard_n = c->dn_tab;
  return f;
}

StageArgs stage_args(oscars_ctx* c, int buf, const int32_t* ahead) {
  StageArgs sa{};
  sa.x = c->dx_tab;
  sa.y = c->dy_tab;
  sa.n = c->dn_tab;
  sa.start = c->cursor;
  sa.row_add = 0;
  sa.wid = nullptr;
  sa.D = c->dims[0];
  sa.B = c->B;
  sa.A0 = c->A0b[buf];
  sa.A0T = c->A0Tb[buf];
  sa.labels = c->labb[buf];
  sa.slots = c->stage_slots;
  sa.n_slots = c->n_stage_slots;
  sa.ahead = ahead;
  return sa;
}

// one-launch round from input buffer `buf` (staged earlier) and, beside it,
// the staging of the next round into the other buffer followed by the cursor
// advance.  The staging forks onto the side stream at the lowest launch
// priority and the round kernel launches at the highest, so the staging
// reads its rows (from host memory, for host-resident shards) on the SMs
// the round's clusters leave free from the round's start, and a cluster
// still waiting to start takes an SM before any staging block does.  While
// profiling, everything runs in sequence on `st` so that the event pairs
// bracket whole kernels.
cudaError_t enqueue_round_fused_ahead(oscars_ctx* c, int buf, cudaStream_t st) {
  cudaError_t e;
  FusedRoundArgs f = fused_args(c);
  f.labels = c->labb[buf];
  f.cursor = nullptr;   // advanced below, after the next round's rows were read
  const StageArgs sa = stage_args(c, buf ^ 1, c->tau_dev);
  if (c->profiling) {
    {
      ProfScope ps(c, "fused_round", st);
      if ((e = launch_fused_round(c->mX4b[buf], c->mXT4b[buf], c->mW0f, c->mRep32, c->mRep16, f, st)) != cudaSuccess) return e;
    }
    {
      ProfScope ps(c, "stage", st);
      if ((e = launch_stage_round(sa, c->tau_dev, c->W, c->max_tau, st)) != cudaSuccess) return e;
    }
    ProfScope ps(c, "round_bookkeeping", st);
    return launch_cursor_advance(c->cursor, c->tau_dev, c->dn_tab, c->B, c->W, st);
  }
  if ((e = cudaEventRecord(c->side_fork, st)) != cudaSuccess) return e;
  if ((e = cudaStreamWaitEvent(c->side, c->side_fork, 0)) != cudaSuccess) return e;
  f.priority = c->prio_greatest;
  if ((e = launch_fused_round(c->mX4b[buf], c->mXT4b[buf], c->mW0f, c->mRep32, c->mRep16, f, st)) != cudaSuccess) return e;
  if ((e = launch_stage_round_priority(sa, c->tau_dev, c->W, c->max_tau, c->prio_least, c->side)) != cudaSuccess)
    return e;
  if ((e = launch_cursor_advance(c->cursor, c->tau_dev, c->dn_tab, c->B, c->W, c->side)) != cudaSuccess) return e;
  if ((e = cudaEventRecord(c->side_join, c->side)) != cudaSuccess) return e;
  return cudaStreamWaitEvent(st, c->side_join, 0);
}

cudaError_t enqueue_round_mlp(oscars_ctx* c, cudaStream_t st) {
  cudaError_t e;
  {
    StageArgs sa{};
    sa.x = c->dx_tab;
    sa.y = c->dy_tab;
    sa.n = c->dn_tab;
    sa.start = c->cursor;
    sa.row_add = 0;
    sa.wid = nullptr;
    sa.D = c->dims[0];
    sa.B = c->B;
    sa.A0 = c->A0all;
    sa.A0T = c->A0Tall;
    sa.labels = c->labels_all;
    sa.slots = c->stage_slots;
    sa.n_slots = c->n_stage_slots;
    ProfScope ps(c, "stage", st);
    if ((e = launch_stage_round(sa, c->tau_dev, c->W, c->max_tau, st)) != cudaSuccess) return e;
  }
  {
    if (c->n_br > 1) {
      cudaError_t e2 = cudaEventRecord(c->br_fork, st);
      if (e2 != cudaSuccess) return e2;
    }
    for (int g = 0; g < c->n_br; ++g) {
      cudaStream_t sg = c->n_br > 1 ? c->br_streams[g] : st;
      if (c->n_br > 1 && (e = cudaStreamWaitEvent(sg, c->br_fork, 0)) != cudaSuccess) return e;
      for (int s = 0; s < c->br_max_tau[g]; ++s) {
        const size_t at = (static_cast<size_t>(g) * c->max_tau + s);
        const int na = c->br_na[at];
        if ((e = enqueue_step(c, s, na, c->br_wid + at * c->W, c->br_src + at * c->W, sg)) != cudaSuccess) return e;
      }
      if (c->n_br > 1) {
        if ((e = cudaEventRecord(c->br_join[g], sg)) != cudaSuccess) return e;
        if ((e = cudaStreamWaitEvent(st, c->br_join[g], 0)) != cudaSuccess) return e;
      }
    }
  }
  const int nc = c->B / kRowsPerLossChunk;
  ProfScope ps(c, "round_bookkeeping", st);
  if ((e = launch_loss_finalize(c->loss_part, c->tau_dev, c->W, c->max_tau, nc, c->B, c->loss_dev, st)) != cudaSuccess)
    return e;
  return launch_cursor_advance(c->cursor, c->tau_dev, c->dn_tab, c->B, c->W, st);
}

// per-layer round from input buffer `buf` (staged earlier) and, beside it
// on the side stream at the lowest launch priority, the staging of the next
// round into the other buffer followed by the cursor advance (as the
// one-launch round does): with shards in host memory the next round's rows
// cross the host link while this round computes.  While profiling,
// everything runs in sequence on `st`.
cudaError_t enqueue_round_mlp_ahead(oscars_ctx* c, int buf, cudaStream_t st) {
  cudaError_t e;
  c->cur_buf = buf;
  const StageArgs sa = stage_args(c, buf ^ 1, c->tau_dev);
  auto steps = [&](cudaStream_t s0) -> cudaError_t {
    for (int s = 0; s < c->br_max_tau[0]; ++s) {
      cudaError_t r = enqueue_step(c, s, c->br_na[s], c->br_wid + static_cast<size_t>(s) * c->W,
                                   c->br_src + static_cast<size_t>(s) * c->W, s0);
      if (r != cudaSuccess) return r;
    }
    return cudaSuccess;
  };
  // from host memory every load waits a round trip over the host link: a
  // grid of kHostStageBlocks blocks striding over the tiles keeps enough rows
  // in flight and leaves the SMs to the round's GEMMs (the full grid of one
  // block per tile fills every SM between GEMM waves); from device memory the
  // full grid is done soonest
  auto stage_next = [&](cudaStream_t s0) {
    return c->shards_host
               ? launch_stage_round_strided(sa, c->tau_dev, c->W, c->max_tau, kHostStageBlocks, c->prio_least, s0)
               : launch_stage_round_priority(sa, c->tau_dev, c->W, c->max_tau, c->prio_least, s0);
  };
  const int nc = c->B / kRowsPerLossChunk;
  if (c->profiling) {
    if ((e = steps(st)) != cudaSuccess) return e;
    {
      ProfScope ps(c, "stage", st);
      if ((e = stage_next(st)) != cudaSuccess) return e;
    }
    ProfScope ps(c, "round_bookkeeping", st);
    if ((e = launch_loss_finalize(c->loss_part, c->tau_dev, c->W, c->max_tau, nc, c->B, c->loss_dev, st)) != cudaSuccess)
      return e;
    return launch_cursor_advance(c->cursor, c->tau_dev, c->dn_tab, c->B, c->W, st);
  }
  if ((e = cudaEventRecord(c->side_fork, st)) != cudaSuccess) return e;
  if ((e = cudaStreamWaitEvent(c->side, c->side_fork, 0)) != cudaSuccess) return e;
  if ((e = stage_next(c->side)) != cudaSuccess) return e;
  if ((e = launch_cursor_advance(c->cursor, c->tau_dev, c->dn_tab, c->B, c->W, c->side)) != cudaSuccess) return e;
  if ((e = cudaEventRecord(c->side_join, c->side)) != cudaSuccess) return e;
  if ((e = steps(st)) != cudaSuccess) return e;
  if ((e = launch_loss_finalize(c->loss_part, c->tau_dev, c->W, c->max_tau, nc, c->B, c->loss_dev, st)) != cudaSuccess)
    return e;
  return cudaStreamWaitEvent(st, c->side_join, 0);
}

cudaError_t enqueue_round_softreg(oscars_ctx* c, cudaStream_t st) {
  SoftregArgs a;
  a.master = c->slab;
  a.master_out = c->slab;
  a.slot_stride = c->P_pad;
  a.global_slot = c->W;
  a.offW = c->layers[0].offW;
  a.offB = c->layers[0].offB;
  a.D = c->dims[0];
  a.C = c->dims[1];
  a.B = c->B;
  a.lr = c->lr;
  a.tau = c->tau_dev;
  a.shard_x = c->dx_tab;
  a.shard_y = c->dy_tab;
  a.shard_n = c->dn_tab;
  a.cursor = c->cursor;
  a.loss_part = c->loss_part;
  a.max_tau = c->max_tau;
  a.loss_out = c->loss_dev;   // the round's bookkeeping in the same launch
  a.cursor_next = c->cursor;
  ProfScope ps(c, "softreg_round", st);
  return softreg_cluster_supported(a.D, a.C, a.B) ? launch_softreg_cluster_round(a, c->W, st)
                                                  : launch_softreg_round(a, c->W, st);
}

// one local step of the convolutional worker for the `na` active workers
cudaError_t enqueue_step_cnn(oscars_ctx* c, int s, int na, const int* wid, const int* src, cudaStream_t st) {
  cudaError_t e;
  const int B = c->B, nb = c->cnn_blocks, layers = 1 + 2 * nb;
  const int tiles = B * cnn_tiles_per_image();
  const int X = 0, S = 1, dzbase = 2 + 2 * nb;
  auto U = [&](int k) { return 2 + 2 * k; };
  auto V = [&](int k) { return 3 + 2 * k; };
  const int ipc = conv_wgrad_images_per_chunk(B, na, c->sms);
  const int chunks = (B + ipc - 1) / ipc;
  const size_t wpl = static_cast<size_t>(c->W) * chunks * 9 * 64 * 64;          // weight partials per layer
  const size_t bpl = static_cast<size_t>(c->W) * tiles * 64;                    // bias partials per layer
  {
    CnnStageArgs a{};
    a.x = c->dx_tab;
    a.y = c->dy_tab;
    a.n = c->dn_tab;
    a.start = c->cursor;
    a.wid = wid;
    a.step = s;
    a.B = B;
    a.Cin = c->dims[2];
    a.im2col = c->cnn_im2col ? 1 : 0;
    a.out = c->cnn_buf[X];
    a.labels = c->labels;
    ProfScope ps(c, "cnn_stage", st);
    if ((e = launch_cnn_stage(a, na, st)) != cudaSuccess) return e;
  }
  auto conv = [&](int mode, int layer, int in, int add, int mask, int out, float* bpart) -> cudaError_t {
    ConvArgs a;
    std::memset(&a, 0, sizeof(a));
    a.wid = wid;
    a.src = src;
    a.B = B;
    a.bias = c->slab;
    a.slot_stride = c->P_pad;
    a.off_bias = c->cnn_offB[layer];
    a.add = add >= 0 ? c->cnn_buf[add] : nullptr;
    a.mask = mask >= 0 ? c->cnn_buf[mask] : nullptr;
    a.out = c->cnn_buf[out];
    a.bias_part = bpart;
    a.err = c->err;
    a.im2col = layer == 0 && c->cnn_im2col ? 1 : 0;
    ProfScope ps(c, mode == 0 ? "conv_fwd" : "conv_dgrad", st);
    return launch_conv_igemm(mode, a.im2col ? c->cnn_m4[in] : c->cnn_m6[in],
                             mode == 0 ? c->cnn_mw[layer] : c->cnn_mwt[layer - 1], a, na,
                             conv_ctas_per_worker(B, na, c->sms), st);
  };
  auto wgrad = [&](int layer, int in, int dz) -> cudaError_t {
    WgradArgs a;
    a.wid = wid;
    a.B = B;
    a.n_chunks = chunks;
    a.img_per_chunk = ipc;
    a.part = c->cnn_wpart + layer * wpl;
    a.err = c->err;
    a.im2col = layer == 0 && c->cnn_im2col ? 1 : 0;
    ProfScope ps(c, "conv_wgrad", st);
    return launch_conv_wgrad(a.im2col ? c->cnn_m2[in] : c->cnn_m4[in], c->cnn_m2[dz], a, na, st);
  };
  // forward
  if ((e = conv(0, 0, X, -1, -1, S, nullptr)) != cudaSuccess) return e;
  for (int k = 0; k < nb; ++k) {
    const int h = k == 0 ? S : V(k - 1);
    if ((e = conv(0, 1 + 2 * k, h, -1, -1, U(k), nullptr)) != cudaSuccess) return e;
    if ((e = conv(0, 2 + 2 * k, U(k), h, -1, V(k), nullptr)) != cudaSuccess) return e;
  }
  // head: pooling, FC, softmax cross-entropy, its backward and SGD
  {
    ProfScope ps(c, "cnn_head", st);
    if ((e = launch_cnn_pool(c->cnn_buf[V(nb - 1)], wid, B, c->cnn_g, na, st)) != cudaSuccess) return e;
    CnnHeadArgs h;
    h.wid = wid;
    h.src = src;
    h.B = B;
    h.K = c->C;
    h.step = s;
    h.max_tau = c->max_tau;
    h.n_loss_chunks = B / kRowsPerLossChunk;
    h.g = c->cnn_g;
    h.labels = c->labels;
    h.dg = c->cnn_dg;
    h.loss_part = c->loss_part;
    h.master = c->slab;
    h.master_w = c->slab;
    h.shadow = c->shadow;
    h.slot_stride = c->P_pad;
    h.offWf = c->cnn_offWf;
    h.offBf = c->cnn_offBf;
    h.lr = c->lr;
    if ((e = launch_cnn_head(h, na, st)) != cudaSuccess) return e;
  }
  // backward through the blocks; dz buffers rotate: cur = output gradient of block k
  int cur = dzbase, nxt = dzbase + 1, nx2 = dzbase + 2;
  {
    ProfScope ps(c, "cnn_dzb", st);
    if ((e = launch_cnn_dzb(c->cnn_buf[V(nb - 1)], c->cnn_dg, wid, B, c->cnn_buf[cur],
                            c->cnn_bpart + (2 + 2 * (nb - 1)) * bpl, na, st)) != cudaSuccess)
      return e;
  }
  for (int k = nb - 1; k >= 0; --k) {
    const int la = 1 + 2 * k, lb = 2 + 2 * k;
    const int h = k == 0 ? S : V(k - 1);
    const int lprev = k == 0 ? 0 : 2 + 2 * (k - 1);   // the layer whose output h is
    if ((e = wgrad(lb, U(k), cur)) != cudaSuccess) return e;
    if ((e = conv(1, lb, cur, -1, U(k), nxt, c->cnn_bpart + la * bpl)) != cudaSuccess) return e;
    if ((e = wgrad(la, h, nxt)) != cudaSuccess) return e;
    if ((e = conv(1, la, nxt, cur, h, nx2, c->cnn_bpart + lprev * bpl)) != cudaSuccess) return e;
    const int t0 = cur;
    cur = nx2;
    nx2 = t0;
  }
  if ((e = wgrad(0, X, cur)) != cudaSuccess) return e;
  // SGD of every convolution layer (after all input gradients used the old weights)
  ProfScope ps(c, "conv_sgd", st);
  ConvSgdArgs a;
  std::memset(&a, 0, sizeof(a));
  a.wid = wid;
  a.src = src;
  a.n_chunks = chunks;
  a.layers = layers;
  const int cpw = conv_ctas_per_worker(B, na, c->sms);
  for (int l = 0; l < layers; ++l) {
    // the last block's b_b sums come from the output-gradient kernel (one per
    // tile), all others from an input-gradient launch (one per CTA)
    a.n_tiles[l] = l == layers - 1 ? tiles : cpw;
    a.part[l] = c->cnn_wpart + l * wpl;
    a.bias_part[l] = c->cnn_bpart + l * bpl;
    a.wt[l] = l >= 1 ? c->cnn_wt + static_cast<int64_t>(l - 1) * 9 * 64 * 64 : nullptr;
    a.offW[l] = c->cnn_offW[l];
    a.offB[l] = c->cnn_offB[l];
    a.im2col[l] = l == 0 && c->cnn_im2col ? 1 : 0;
  }
  a.master = c->slab;
  a.master_w = c->slab;
  a.shadow = c->shadow;
  a.slot_stride = c->P_pad;
  a.wt_slot_stride = c->cnn_wt_slot;
  a.lr = c->lr;
  return launch_conv_sgd(a, na, st);
}

cudaError_t enqueue_round_cnn(oscars_ctx* c, cudaStream_t st) {
  cudaError_t e;
  for (int s = 0; s < c->max_tau; ++s) {
    const int na = c->n_active[s];
    if ((e = enqueue_step_cnn(c, s, na, c->act_wid + static_cast<size_t>(s) * c->W,
                              c->act_src + static_cast<size_t>(s) * c->W, st)) != cudaSuccess)
      return e;
  }
  const int nc = c->B / kRowsPerLossChunk;
  ProfScope ps(c, "round_bookkeeping", st);
  if ((e = launch_loss_finalize(c->loss_part, c->tau_dev, c->W, c->max_tau, nc, c->B, c->loss_dev, st)) != cudaSuccess)
    return e;
  return launch_cursor_advance(c->cursor, c->tau_dev, c->dn_tab, c->B, c->W, st);
}

cudaError_t enqueue_round(oscars_ctx* c, cudaStream_t st) {
  if (c->model == OSCARS_MODEL_CNN) return enqueue_round_cnn(c, st);
  return c->L == 1 && !c->bf16 ? enqueue_round_softreg(c, st) : enqueue_round_mlp(c, st);
}

oscars_status check_err_word(oscars_ctx* c) {
  if (!c->err) return OSCARS_OK;
  int h = 0;
  cudaError_t e = cudaMemcpy(&h, c->err, sizeof(int), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(c, e, "reading the kernel error word");
  if (h != 0) {
    cudaMemset(c->err, 0, sizeof(int));
    return fail(c, OSCARS_ETIMEOUT, "a kernel's bounded wait ran out (code " + std::to_string(h) + ")");
  }
  return OSCARS_OK;
}

bool slotted(const oscars_ctx* c) { return c->model == OSCARS_MODEL_MLP || c->model == OSCARS_MODEL_CNN; }

// convolutional worker: checks and the slot layout (every tensor on a
// 64-element boundary; the stem's input channels padded to 64)
oscars_status layout_cnn(oscars_ctx* c, const oscars_config* cfg) {
  c->cnn_blocks = cfg->num_layers;
  c->dims.assign(cfg->dims, cfg->dims + 5);
  const int H = c->dims[0], Wd = c->dims[1], Cin = c->dims[2], C = c->dims[3], K = c->dims[4];
  c->B = cfg->batch;
  c->C = K;
  c->L = 0;
  if (H < 1 || Wd < 1 || Cin < 1 || C < 1 || K < 1 || c->B < 1) return fail(c, OSCARS_EINVAL, "CNN: dims and batch must be >= 1");
  if (!(c->lr == c->lr)) return fail(c, OSCARS_EINVAL, "lr is NaN");
  if (c->cnn_blocks < 1 || c->cnn_blocks > 4) return fail(c, OSCARS_ENOTSUP, "CNN: 1 to 4 residual blocks");
  if (H != 32 || Wd != 32 || C != 64) return fail(c, OSCARS_ENOTSUP, "CNN: 32 x 32 images and 64 channels");
  if (Cin > 64) return fail(c, OSCARS_ENOTSUP, "CNN: at most 64 input channels");
  if (K < 2 || K > kMaxClasses) return fail(c, OSCARS_ENOTSUP, "classes must be in [2, 32]");
  if (!c->bf16) return fail(c, OSCARS_ENOTSUP, "CNN: bf16 GEMMs only");
  if (c->B % kRowsPerLossChunk != 0 || c->B > 256) return fail(c, OSCARS_ENOTSUP, "CNN: batch must be a multiple of 16, <= 256");
  if (c->W > kMaxWorkersMLP) return fail(c, OSCARS_ENOTSUP, "CNN mode supports at most 64 workers");
  const int layers = 1 + 2 * c->cnn_blocks;
  int64_t off = 0;
  for (int l = 0; l < layers; ++l) {
    c->cnn_offW.push_back(off);
    off += 64 * 9 * 64;
    c->cnn_offB.push_back(off);
    off += 64;
  }
  c->cnn_offWf = off;
  off += round_up(static_cast<int64_t>(K) * C, 64);
  c->cnn_offBf = off;
  off += round_up(K, 64);
  c->P_pad = round_up(off, 64);
  c->P = static_cast<int64_t>(C) * 9 * Cin + C + static_cast<int64_t>(c->cnn_blocks) * 2 * (C * 9 * C + C) +
         static_cast<int64_t>(K) * C + K;
  c->cnn_wt_slot = static_cast<int64_t>(2 * c->cnn_blocks) * 9 * 64 * 64;
  c->cnn_im2col = 9 * Cin <= 64;   // layer 0 then uses the first 64 x 64 of its 64 x 9 x 64 block
  c->cnn_chunks = c->B;   // capacity: at most one image per chunk
  return OSCARS_OK;
}

oscars_status validate_and_layout(oscars_ctx* c, const oscars_config* cfg) {
  c->W = cfg->num_workers;
  c->model = cfg->model;
  if (c->W < 1 || c->W > kMaxMergeWorkers) return fail(c, OSCARS_EINVAL, "num_workers must be in [1, 256]");
  if (!cfg->dims) return fail(c, OSCARS_EINVAL, "dims is NULL");
  c->lr = cfg->lr;
  c->server_lr = cfg->server_lr;
  c->rule = cfg->weight_rule;
  c->bf16 = cfg->bf16_gemm;
  if (c->rule < OSCARS_W_UNIFORM || c->rule > OSCARS_W_EXPLICIT) return fail(c, OSCARS_EINVAL, "bad weight rule");
  if (!(c->server_lr == c->server_lr)) return fail(c, OSCARS_EINVAL, "server_lr is NaN");
  if (c->model == OSCARS_MODEL_FLAT) {
    if (cfg->dims[0] < 1) return fail(c, OSCARS_EINVAL, "FLAT: dims[0] = P must be >= 1");
    c->L = 0;
    c->P = cfg->dims[0];
    c->P_pad = round_up(c->P, 64);
    return OSCARS_OK;
  }
  if (c->model == OSCARS_MODEL_CNN) return layout_cnn(c, cfg);
  if (c->model != OSCARS_MODEL_MLP) return fail(c, OSCARS_EINVAL, "unknown model");
  c->L = cfg->num_layers;
  if (c->L < 1 || c->L > 16) return fail(c, OSCARS_EINVAL, "num_layers must be in [1, 16]");
  c->dims.assign(cfg->dims, cfg->dims + c->L + 1);
  for (int d : c->dims)
    if (d < 1) return fail(c, OSCARS_EINVAL, "dims must be >= 1");
  c->B = cfg->batch;
  c->C = c->dims[c->L];
  if (c->B < 1) return fail(c, OSCARS_EINVAL, "batch must be >= 1");
  if (c->C < 2 || c->C > kMaxClasses) return fail(c, OSCARS_ENOTSUP, "classes must be in [2, 32]");
  if (!(c->lr == c->lr)) return fail(c, OSCARS_EINVAL, "lr is NaN");
  if (c->L == 1 && !c->bf16) {
    if (c->B > kSoftregMaxBatch) return fail(c, OSCARS_ENOTSUP, "softmax regression: batch must be <= 512");
    if (softreg_smem_bytes(c->dims[0], c->C, c->B) > 220 * 1024)
      return fail(c, OSCARS_ENOTSUP, "softmax regression: weights plus one batch must fit in shared memory");
  } else if (c->bf16 && c->L >= 2) {
    if (c->W > kMaxWorkersMLP) return fail(c, OSCARS_ENOTSUP, "MLP mode supports at most 64 workers");
    if (c->B % 32 != 0 || c->B > 256) return fail(c, OSCARS_ENOTSUP, "bf16 MLP: batch must be a multiple of 32, <= 256");
    if (c->dims[0] % 8 != 0) return fail(c, OSCARS_ENOTSUP, "bf16 MLP: input dim must be a multiple of 8");
    for (int l = 1; l < c->L; ++l)
      if (c->dims[l] % 128 != 0) return fail(c, OSCARS_ENOTSUP, "bf16 MLP: hidden dims must be multiples of 128");
    if (c->dims[c->L - 1] > 2048) return fail(c, OSCARS_ENOTSUP, "bf16 MLP: the last hidden dim must be <= 2048");
  } else {
    return fail(c, OSCARS_ENOTSUP, "supported: fp32 softmax regression (L=1) or bf16 MLP (L>=2)");
  }
  int64_t off = 0;
  c->P = 0;
  for (int l = 0; l < c->L; ++l) {
    Layer ly;
    ly.in = c->dims[l];
    ly.out = c->dims[l + 1];
    ly.offW = off;
    off += round_up(static_cast<int64_t>(ly.in) * ly.out, 64);
    ly.offB = off;
    off += round_up(ly.out, 64);
    c->P += static_cast<int64_t>(ly.in) * ly.out + ly.out;
    c->layers.push_back(ly);
  }
  c->P_pad = round_up(off, 64);
  return OSCARS_OK;
}

// the slab of W + 1 slots and the per-worker tables (MLP and CNN)
oscars_status allocate_common(oscars_ctx* c) {
  {
    int dev = 0;
    cudaGetDevice(&dev);
    if (cudaDeviceGetAttribute(&c->sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || c->sms < 1) c->sms = 1;
  }
  const int W = c->W;
  const size_t slots = static_cast<size_t>(W) + 1;
  if (!dev_alloc(c, &c->slab, slots * c->P_pad + kGuardWords))
    return fail(c, OSCARS_ENOMEM, "device allocation failed (model slab)");
  cudaMemset(c->slab, 0, slots * c->P_pad * sizeof(float));
  cudaMemset(c->slab + slots * c->P_pad, kGuardByte, kGuardWords * sizeof(float));
  if (!dev_alloc(c, &c->cursor, W) || !dev_alloc(c, &c->tau_dev, W) || !dev_alloc(c, &c->loss_dev, std::max(W, 1)) ||
      !dev_alloc(c, &c->dx_tab, W) || !dev_alloc(c, &c->dy_tab, W) || !dev_alloc(c, &c->dn_tab, W) ||
      !dev_alloc(c, &c->err, 1) || !dev_alloc(c, &c->lane_ids, W) || !dev_alloc(c, &c->global_src, W) ||
      !dev_alloc(c, &c->ex_tab, W) || !dev_alloc(c, &c->ey_tab, W) || !dev_alloc(c, &c->en_tab, W))
    return fail(c, OSCARS_ENOMEM, "device allocation failed (tables)");
  cudaMemset(c->cursor, 0, W * sizeof(int64_t));
  cudaMemset(c->err, 0, sizeof(int));
  std::vector<int> ids(W), gs(W, W);
  for (int i = 0; i < W; ++i) ids[i] = i;
  cudaMemcpy(c->lane_ids, ids.data(), W * sizeof(int), cudaMemcpyHostToDevice);
  cudaMemcpy(c->global_src, gs.data(), W * sizeof(int), cudaMemcpyHostToDevice);
  cudaMemcpy(c->dx_tab, c->shard_x.data(), W * sizeof(float*), cudaMemcpyHostToDevice);
  cudaMemcpy(c->dy_tab, c->shard_y.data(), W * sizeof(int32_t*), cudaMemcpyHostToDevice);
  cudaError_t e = cudaMemcpy(c->dn_tab, c->shard_n.data(), W * sizeof(int64_t), cudaMemcpyHostToDevice);
  if (e != cudaSuccess) return cuda_fail(c, e, "table upload");
  return OSCARS_OK;
}

oscars_status allocate_cnn(oscars_ctx* c) {
  oscars_status st = allocate_common(c);
  if (st != OSCARS_OK) return st;
  const int W = c->W, B = c->B;
  const size_t slots = static_cast<size_t>(W) + 1;
  const int layers = 1 + 2 * c->cnn_blocks;
  if (!dev_alloc(c, &c->shadow, slots * c->P_pad + kGuardWords) || !dev_alloc(c, &c->cnn_wt, slots * c->cnn_wt_slot))
    return fail(c, OSCARS_ENOMEM, "device allocation failed (bf16 weights)");
  cudaMemset(c->shadow, 0, slots * c->P_pad * sizeof(__nv_bfloat16));
  cudaMemset(c->shadow + slots * c->P_pad, kGuardByte, kGuardWords * sizeof(__nv_bfloat16));
  cudaMemset(c->cnn_wt, 0, slots * c->cnn_wt_slot * sizeof(__nv_bfloat16));
  const size_t act = static_cast<size_t>(W) * B * 1024 * 64;
  const int nbuf = 2 + 2 * c->cnn_blocks + 3;
  c->cnn_buf.assign(nbuf, nullptr);
  for (int i = 0; i < nbuf; ++i)
    if (!dev_alloc(c, &c->cnn_buf[i], act)) return fail(c, OSCARS_ENOMEM, "device allocation failed (activations)");
  // the input buffer's channels past the image's stay zero: the staging kernel writes only the input channels
  if (cudaMemset(c->cnn_buf[0], 0, act * sizeof(__nv_bfloat16)) != cudaSuccess)
    return fail(c, OSCARS_ECUDA, "clearing the input buffer failed");
  const size_t tiles = static_cast<size_t>(B) * cnn_tiles_per_image();
  if (!dev_alloc(c, &c->cnn_g, static_cast<size_t>(W) * B * 64) ||
      !dev_alloc(c, &c->cnn_dg, static_cast<size_t>(W) * B * 64) ||
      !dev_alloc(c, &c->labels, static_cast<size_t>(W) * B) ||
      !dev_alloc(c, &c->cnn_wpart, static_cast<size_t>(layers) * W * c->cnn_chunks * 9 * 64 * 64) ||
      !dev_alloc(c, &c->cnn_bpart, static_cast<size_t>(layers) * W * tiles * 64))
    return fail(c, OSCARS_ENOMEM, "device allocation failed (gradients)");
  // tensor maps: activations {64 ch, 32 x, 32 y, images}; weights per slot
  c->cnn_m6.resize(nbuf);
  c->cnn_m4.resize(nbuf);
  c->cnn_m2.resize(nbuf);
  const uint64_t imgs = static_cast<uint64_t>(W) * B;
  bool ok = true;
  for (int i = 0; i < nbuf; ++i) {
    const uint64_t d[4] = {64, 32, 32, imgs};
    const uint64_t stv[3] = {64 * 2, 32 * 64 * 2, 1024 * 64 * 2};
    ok &= make_map_box4(&c->cnn_m6[i], c->cnn_buf[i], d, stv, {64, 32, 6, 1});
    ok &= make_map_box4(&c->cnn_m4[i], c->cnn_buf[i], d, stv, {64, 32, 4, 1});
    ok &= make_map_box4(&c->cnn_m2[i], c->cnn_buf[i], d, stv, {64, 32, 2, 1});
  }
  c->cnn_mw.resize(layers);
  c->cnn_mwt.resize(layers > 1 ? layers - 1 : 1);
  for (int l = 0; l < layers; ++l) {
    // forward layout [out][tap][in] of every slot: dims {in, tap, out, slot};
    // the im2col stem [out][k]: one tap
    const uint64_t ntap = l == 0 && c->cnn_im2col ? 1 : 9;
    const uint64_t d[4] = {64, ntap, 64, slots};
    const uint64_t stv[3] = {64 * 2, ntap * 64 * 2, static_cast<uint64_t>(c->P_pad) * 2};
    ok &= make_map_box4(&c->cnn_mw[l], c->shadow + c->cnn_offW[l], d, stv, {64, 1, 64, 1});
    if (l >= 1) {
      // transposed [tap][in][out]: dims {out, in, tap, slot}
      const uint64_t dt[4] = {64, 64, 9, slots};
      const uint64_t stt[3] = {64 * 2, 64 * 64 * 2, static_cast<uint64_t>(c->cnn_wt_slot) * 2};
      ok &= make_map_box4(&c->cnn_mwt[l - 1], c->cnn_wt + static_cast<int64_t>(l - 1) * 9 * 64 * 64, dt, stt,
                          {64, 64, 1, 1});
    }
  }
  if (!ok) return fail(c, OSCARS_ECUDA, "cuTensorMapEncodeTiled failed (CNN)");
  return OSCARS_OK;
}

oscars_status allocate_mlp(oscars_ctx* c) {
  oscars_status st0 = allocate_common(c);
  if (st0 != OSCARS_OK) return st0;
  const int W = c->W, B = c->B, L = c->L;
  const size_t slots = static_cast<size_t>(W) + 1;
  if (L == 1 && !c->bf16) return OSCARS_OK;

  if (!dev_alloc(c, &c->shadow, slots * c->P_pad + kGuardWords))
    return fail(c, OSCARS_ENOMEM, "device allocation failed (bf16 shadow)");
  cudaMemset(c->shadow, 0, slots * c->P_pad * sizeof(__nv_bfloat16));
  cudaMemset(c->shadow + slots * c->P_pad, kGuardByte, kGuardWords * sizeof(__nv_bfloat16));
  c->A.assign(L, nullptr);
  c->AT.assign(L, nullptr);
  c->G.assign(L, nullptr);
  {
    const Layer& hl = c->layers.back();
    c->g_rows = !(B % 64 == 0 && head_tc_supported(hl.in, B, hl.out));
  }
  c->GT.assign(L, nullptr);
  c->gb.assign(L, nullptr);
  for (int l = 0; l < L; ++l) {
    const size_t act = static_cast<size_t>(W) * B * c->dims[l];
    if (l > 0 && (!dev_alloc(c, &c->A[l], act) || !dev_alloc(c, &c->AT[l], act)))
      return fail(c, OSCARS_ENOMEM, "device allocation failed (activations)");
    if (l + 1 < L) {
      const size_t gsz = static_cast<size_t>(W) * B * c->dims[l + 1];
      if ((c->g_rows && !dev_alloc(c, &c->G[l], gsz)) || !dev_alloc(c, &c->GT[l], gsz) ||
          !dev_alloc(c, &c->gb[l], static_cast<size_t>(W) * c->dims[l + 1]))
        return fail(c, OSCARS_ENOMEM, "device allocation failed (gradients)");
    }
  }
  if (!dev_alloc(c, &c->dlog, static_cast<size_t>(W) * B * c->C))
    return fail(c, OSCARS_ENOMEM, "device allocation failed (head)");

  // tensor maps
  c->mShadow.resize(L);
  c->mMaster.resize(L);
  c->mMasterSt.resize(L);
  c->mShadowSt.resize(L);
  c->mShadowMN.resize(L);
  c->mA.resize(L);
  c->mG.resize(L);
  c->mGTmn.resize(L);
  c->mGT.resize(L);
  c->mAT.resize(L);
  const uint64_t slots64 = slots;
  for (int l = 0; l + 1 < L; ++l) {
    const Layer& ly = c->layers[l];
    bool ok = true;
    // W_l [out][in] of every slot: A operand of the forward GEMM
    ok &= make_map(&c->mShadow[l], c->shadow + ly.offW, ly.in, ly.out, slots64, ly.in * 2ull, c->P_pad * 2ull, 128);
    // the fp32 master of W_l in every slot: read and written by the weight-gradient kernel
    ok &= make_map_f32(&c->mMaster[l], c->slab + ly.offW, ly.in, ly.out, slots64, ly.in * 4ull, c->P_pad * 4ull, 128);
    ok &= make_map_f32(&c->mMasterSt[l], c->slab + ly.offW, ly.in, ly.out, slots64, ly.in * 4ull, c->P_pad * 4ull, 32);
    ok &= make_map(&c->mShadowSt[l], c->shadow + ly.offW, ly.in, ly.out, slots64, ly.in * 2ull, c->P_pad * 2ull, 32);
    // layer input [lane][B][in]: B operand of the forward GEMM (layer 0: per step)
    if (l > 0) ok &= make_map(&c->mA[l], c->A[l], ly.in, B, W, ly.in * 2ull, static_cast<uint64_t>(B) * ly.in * 2ull, B);
    // output gradient^T [lane][out][B]: A operand of the weight-gradient GEMM
    ok &= make_map(&c->mGT[l], c->GT[l], B, ly.out, W, B * 2ull, static_cast<uint64_t>(B) * ly.out * 2ull, 128);
    // layer input^T [lane][in][B]: B operand of the weight-gradient GEMM (layer 0: per step)
    if (l > 0) ok &= make_map(&c->mAT[l], c->AT[l], B, ly.in, W, B * 2ull, static_cast<uint64_t>(B) * ly.in * 2ull, 128);
    if (l >= 1) {
      // W_l [out][in] of every slot, boxes of 64 inputs x 64 outputs: the
      // MN-major A operand (M = in, K = out) of the input-gradient GEMM
      ok &= make_map(&c->mShadowMN[l], c->shadow + ly.offW, ly.in, ly.out, slots64, ly.in * 2ull, c->P_pad * 2ull, 64);
      // output gradient [lane][B][out]: B operand of the input-gradient GEMM
      if (c->g_rows)
        ok &= make_map(&c->mG[l], c->G[l], ly.out, B, W, ly.out * 2ull, static_cast<uint64_t>(B) * ly.out * 2ull, B);
      else   // output gradient^T [lane][out][B], boxes of 64 samples x 64 outputs: the MN-major B operand
        ok &= make_map(&c->mGTmn[l], c->GT[l], B, ly.out, W, B * 2ull, static_cast<uint64_t>(B) * ly.out * 2ull, 64);
    }
    if (!ok) return fail(c, OSCARS_ECUDA, "cuTensorMapEncodeTiled failed (or the driver entry point is missing)");
  }
  {
    const Layer& hl = c->layers.back();
    if (!make_map(&c->mHeadIn, c->A[L - 1], hl.in, B, W, hl.in * 2ull, static_cast<uint64_t>(B) * hl.in * 2ull, 128) ||
        !make_map(&c->mHeadW, c->shadow + hl.offW, hl.in, hl.out, slots64, hl.in * 2ull, c->P_pad * 2ull, 16))
      return fail(c, OSCARS_ECUDA, "cuTensorMapEncodeTiled failed (head)");
  }
  return OSCARS_OK;
}

// copy a canonical-layout vector into the padded slot layout (or back)
cudaError_t copy_canonical(oscars_ctx* c, float* padded, const float* canon, bool to_padded, cudaStream_t s) {
  if (c->model == OSCARS_MODEL_CNN) {
    const int Cin = c->dims[2], K = c->dims[4];
    float* dst = const_cast<float*>(canon);
    int64_t co = 0;
    // stem [64][9][Cin] <-> [64][9][64], or <-> [64][64] with im2col (k = tap * Cin + i);
    // the padding stays zero
    const size_t wrow = (c->cnn_im2col ? 9 * Cin : Cin) * sizeof(float);
    const size_t nrow = c->cnn_im2col ? 64 : 64 * 9;
    cudaError_t e = to_padded ? cudaMemcpy2DAsync(padded + c->cnn_offW[0], 64 * sizeof(float), canon, wrow, wrow, nrow,
                                                  cudaMemcpyDefault, s)
                              : cudaMemcpy2DAsync(dst, wrow, padded + c->cnn_offW[0], 64 * sizeof(float), wrow, nrow,
                                                  cudaMemcpyDefault, s);
    co = static_cast<int64_t>(64) * 9 * Cin;
    auto seg = [&](int64_t off, int64_t n) -> cudaError_t {
      cudaError_t r = to_padded ? cudaMemcpyAsync(padded + off, canon + co, n * sizeof(float), cudaMemcpyDefault, s)
                                : cudaMemcpyAsync(dst + co, padded + off, n * sizeof(float), cudaMemcpyDefault, s);
      co += n;
      return r;
    };
    if (e == cudaSuccess) e = seg(c->cnn_offB[0], 64);
    for (size_t l = 1; e == cudaSuccess && l < c->cnn_offW.size(); ++l) {
      e = seg(c->cnn_offW[l], 64 * 9 * 64);
      if (e == cudaSuccess) e = seg(c->cnn_offB[l], 64);
    }
    if (e == cudaSuccess) e = seg(c->cnn_offWf, static_cast<int64_t>(K) * 64);
    if (e == cudaSuccess) e = seg(c->cnn_offBf, K);
    return e;
  }
  if (c->model == OSCARS_MODEL_FLAT) {
    return to_padded ? cudaMemcpyAsync(padded, canon, c->P * sizeof(float), cudaMemcpyDefault, s)
                     : cudaMemcpyAsync(const_cast<float*>(canon), padded, c->P * sizeof(float), cudaMemcpyDefault, s);
  }
  int64_t co = 0;
  for (const Layer& ly : c->layers) {
    const int64_t nw = static_cast<int64_t>(ly.in) * ly.out;
    cudaError_t e;
    if (to_padded) {
      e = cudaMemcpyAsync(padded + ly.offW, canon + co, nw * sizeof(float), cudaMemcpyDefault, s);
      if (e == cudaSuccess) e = cudaMemcpyAsync(padded + ly.offB, canon + co + nw, ly.out * sizeof(float), cudaMemcpyDefault, s);
    } else {
      float* dst = const_cast<float*>(canon);
      e = cudaMemcpyAsync(dst + co, padded + ly.offW, nw * sizeof(float), cudaMemcpyDefault, s);
      if (e == cudaSuccess) e = cudaMemcpyAsync(dst + co + nw, padded + ly.offB, ly.out * sizeof(float), cudaMemcpyDefault, s);
    }
    if (e != cudaSuccess) return e;
    co += nw + ly.out;
  }
  return cudaSuccess;
}

// the round from input buffer b (staged by the round before) with, beside
// it, the staging of the next round into the other buffer
cudaError_t enqueue_ahead(oscars_ctx* c, int b, cudaStream_t s0) {
  return c->fused ? enqueue_round_fused_ahead(c, b, s0) : enqueue_round_mlp_ahead(c, b, s0);
}

// the first staged-ahead round (or the first after tau changed or an
// evaluation) stages its own mini-batches into buffer b first
cudaError_t stage_own_round(oscars_ctx* c, int b) {
  c->profiling = (c->flags & 2) != 0;
  cudaError_t e;
  {
    ProfScope ps(c, "stage", c->stream);
    e = launch_stage_round(stage_args(c, b, nullptr), c->tau_dev, c->W, c->max_tau, c->stream);
  }
  c->profiling = false;
  return e;
}

// the simulated clocks after an enqueued round: every worker reaches the
// barrier T*, idle for T* minus its busy time
void advance_clocks(oscars_ctx* c) {
  for (int i = 0; i < c->W; ++i) {
    const int64_t busy = static_cast<int64_t>(c->tau[i]) * c->t_iter[i];
    c->clock[i] += c->barrier;
    c->idle[i] += c->barrier - busy;
  }
  ++c->rounds_run;
}

bool is_host_ptr(const void* p) {
  cudaPointerAttributes at;
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    cudaGetLastError();
    return true;
  }
  return at.type == cudaMemoryTypeHost || at.type == cudaMemoryTypeUnregistered;
}

}  // namespace

extern "C" {

oscars_status oscars_create(const oscars_config* cfg, oscars_ctx** out) {
  if (!cfg || !out) return OSCARS_EINVAL;
  oscars_ctx* c = new (std::nothrow) oscars_ctx();
  if (!c) return OSCARS_ENOMEM;
  oscars_status st = OSCARS_OK;
  try {
    st = validate_and_layout(c, cfg);
    c->flags = cfg->flags;
    if (st == OSCARS_OK) {
      c->stream = static_cast<cudaStream_t>(cfg->cuda_stream);
      c->M = cfg->M;
      c->search_mode = cfg->search_mode;
      c->t_iter.assign(c->W, 0);
      c->tau.assign(c->W, 1);
      const char* why = "";
      int r = OSCARS_OK;
      if (cfg->t_ticks) {
        for (int i = 0; i < c->W; ++i) c->t_iter[i] = cfg->t_ticks[i];
      } else if (cfg->speed) {
        r = iteration_ticks(cfg->speed, c->W, cfg->ticks_per_unit, c->t_iter.data(), &why);
      } else {
        for (int i = 0; i < c->W; ++i) c->t_iter[i] = 1;  // homogeneous
      }
      if (r == OSCARS_OK)
        r = schedule_solve(c->t_iter.data(), c->W, c->M, c->search_mode, &c->T_star, &c->max_wait, c->tau.data(), &why);
      if (r != OSCARS_OK) st = fail(c, static_cast<oscars_status>(r), why);
    }
    if (st == OSCARS_OK) {
      update_barrier(c, true);
      c->clock.assign(c->W, 0);
      c->idle.assign(c->W, 0);
      if (slotted(c)) {
        if (!cfg->shard_x || !cfg->shard_y || !cfg->shard_n) st = fail(c, OSCARS_EINVAL, "MLP: shard pointers are NULL");
        for (int i = 0; st == OSCARS_OK && i < c->W; ++i) {
          if (!cfg->shard_x[i] || !cfg->shard_y[i] || cfg->shard_n[i] < 1)
            st = fail(c, OSCARS_EINVAL, "MLP: shard " + std::to_string(i) + " is NULL or empty");
          else if (c->model == OSCARS_MODEL_MLP && c->bf16 && (reinterpret_cast<uintptr_t>(cfg->shard_x[i]) & 15))
            st = fail(c, OSCARS_EINVAL, "bf16 MLP: shard " + std::to_string(i) + " samples must be 16-byte aligned");
          else {
            c->shard_x.push_back(cfg->shard_x[i]);
            if (is_host_ptr(cfg->shard_x[i])) c->shards_host = true;
            c->shard_y.push_back(cfg->shard_y[i]);
            c->shard_n.push_back(cfg->shard_n[i]);
          }
        }
        if (st == OSCARS_OK && !cfg->init_params) st = fail(c, OSCARS_EINVAL, "MLP: init_params is NULL");
        // a 2-layer bf16 MLP runs each round as one fused launch (flag bit 3: per-layer kernels)
        c->fused = c->model == OSCARS_MODEL_MLP && c->bf16 && !(cfg->flags & 8) && !(cfg->flags & 4) &&
                   fused_round_supported(c->L, c->dims[0], c->L >= 2 ? c->dims[1] : 0, c->C, c->B);
        if (c->fused) c->fused_max_clusters = fused_round_max_clusters(c->dims[0], c->dims[1], c->B);
        // flag bit 2: bf16 MLP rounds fork into up to 16 concurrent worker branches
        c->n_br = (c->model == OSCARS_MODEL_MLP && c->bf16 && c->L >= 2 && (cfg->flags & 4)) ? std::min(c->W, kMaxBranches) : 1;
        // the per-layer round stages the next round beside the current one
        // (not with concurrent worker branches)
        c->ahead_mlp = c->model == OSCARS_MODEL_MLP && c->bf16 && c->L >= 2 && !c->fused && c->n_br == 1;
        if (st == OSCARS_OK) st = c->model == OSCARS_MODEL_CNN ? allocate_cnn(c) : allocate_mlp(c);
        if (st == OSCARS_OK) st = build_tables(c);
        if (st == OSCARS_OK) {
          cudaError_t e = copy_canonical(c, c->slab + static_cast<int64_t>(c->W) * c->P_pad, cfg->init_params, true, c->stream);
          if (e == cudaSuccess) e = refresh_global_shadows(c, c->stream);
          if (e == cudaSuccess) e = cudaStreamSynchronize(c->stream);
          if (e != cudaSuccess) st = cuda_fail(c, e, "initial model upload");
        }
        if (st == OSCARS_OK && cudaStreamCreateWithFlags(&c->cap, cudaStreamNonBlocking) != cudaSuccess)
          st = fail(c, OSCARS_ECUDA, "stream creation failed");
        c->flags = cfg->flags;
        for (int g = 1; st == OSCARS_OK && c->n_br > 1 && g <= c->n_br; ++g) {
          cudaStream_t bs;
          cudaEvent_t ev;
          if (cudaStreamCreateWithFlags(&bs, cudaStreamNonBlocking) != cudaSuccess ||
              cudaEventCreateWithFlags(&ev, cudaEventDisableTiming) != cudaSuccess) {
            st = fail(c, OSCARS_ECUDA, "stream creation failed");
            break;
          }
          c->br_streams.push_back(bs);
          c->br_join.push_back(ev);
        }
        if (st == OSCARS_OK && c->n_br > 1 && cudaEventCreateWithFlags(&c->br_fork, cudaEventDisableTiming) != cudaSuccess)
          st = fail(c, OSCARS_ECUDA, "event creation failed");
        if (st == OSCARS_OK && (c->fused || c->ahead_mlp) &&
            (cudaDeviceGetStreamPriorityRange(&c->prio_least, &c->prio_greatest) != cudaSuccess ||
             cudaStreamCreateWithFlags(&c->side, cudaStreamNonBlocking) != cudaSuccess ||
             cudaEventCreateWithFlags(&c->side_fork, cudaEventDisableTiming) != cudaSuccess ||
             cudaEventCreateWithFlags(&c->side_join, cudaEventDisableTiming) != cudaSuccess))
          st = fail(c, OSCARS_ECUDA, "stream creation failed");
      } else {
        c->flags = cfg->flags;
        if (!dev_alloc(c, &c->slab, c->P_pad)) st = fail(c, OSCARS_ENOMEM, "device allocation failed (global model)");
        if (st == OSCARS_OK) {
          cudaError_t e = cudaMemsetAsync(c->slab, 0, c->P_pad * sizeof(float), c->stream);
          if (e == cudaSuccess && cfg->init_params) e = copy_canonical(c, c->slab, cfg->init_params, true, c->stream);
          if (e == cudaSuccess) e = cudaStreamSynchronize(c->stream);
          if (e != cudaSuccess) st = cuda_fail(c, e, "initial model upload");
        }
      }
    }
  } catch (const std::bad_alloc&) {
    st = OSCARS_ENOMEM;
  } catch (...) {
    st = OSCARS_EINVAL;
  }
  if (st != OSCARS_OK) {
    free_all(c);
    delete c;
    return st;
  }
  *out = c;
  return OSCARS_OK;
}

oscars_status oscars_destroy(oscars_ctx* c) {
  if (!c) return OSCARS_OK;
  cudaStreamSynchronize(c->stream);
  free_all(c);
  delete c;
  return OSCARS_OK;
}

oscars_status oscars_local_steps(oscars_ctx* c, int32_t* tau_out, float* loss_out) {
  if (!c) return OSCARS_EINVAL;
  if (!slotted(c)) return fail(c, OSCARS_ESTATE, "local steps need an MLP or CNN context");
  if (c->pending) return fail(c, OSCARS_ESTATE, "the previous round has not been merged");
  try {
    cudaError_t e = cudaSuccess;
    if (c->fused || c->ahead_mlp) {
      // the one-launch round (or the per-layer round): every round stages
      // the next one
      const int buf = c->parity;
      if (!c->staged && (e = stage_own_round(c, buf)) != cudaSuccess) return cuda_fail(c, e, "local steps launch");
      if (c->flags & 1) {
        c->profiling = (c->flags & 2) != 0;
        e = enqueue_ahead(c, buf, c->stream);
        c->profiling = false;
      } else {
        if (!c->ahead_exec[buf]) {
          cudaGraph_t g = nullptr;
          c->profiling = (c->flags & 2) != 0;
          c->prof_sink = &c->prof_ahead_graph[buf];   // empty: this parity's graph does not exist yet
          e = cudaStreamBeginCapture(c->cap, cudaStreamCaptureModeThreadLocal);
          if (e == cudaSuccess) {
            cudaError_t e2 = enqueue_ahead(c, buf, c->cap);
            e = cudaStreamEndCapture(c->cap, &g);
            if (e2 != cudaSuccess) e = e2;
          }
          c->profiling = false;
          c->prof_sink = nullptr;
          if (e == cudaSuccess) e = cudaGraphInstantiateWithFlags(&c->ahead_exec[buf], g, 0);
          if (g) cudaGraphDestroy(g);
        }
        if (e == cudaSuccess) e = cudaGraphLaunch(c->ahead_exec[buf], c->stream);
        if (e == cudaSuccess) prof_after_replay(c, c->prof_ahead_graph[buf]);
      }
      if (e == cudaSuccess) {
        c->staged = true;
        c->parity = buf ^ 1;
      }
    } else if (c->flags & 1) {
      c->profiling = (c->flags & 2) != 0;
      e = enqueue_round(c, c->stream);
      c->profiling = false;
    } else {
      if (!c->round_exec) {
        cudaGraph_t g = nullptr;
        for (auto& p : c->prof_round_graph) {
          cudaEventDestroy(p.a);
          cudaEventDestroy(p.b);
        }
        c->prof_round_graph.clear();
        c->profiling = (c->flags & 2) != 0;
        c->prof_sink = &c->prof_round_graph;
        e = cudaStreamBeginCapture(c->cap, cudaStreamCaptureModeThreadLocal);
        if (e == cudaSuccess) {
          cudaError_t e2 = enqueue_round(c, c->cap);
          e = cudaStreamEndCapture(c->cap, &g);
          if (e2 != cudaSuccess) e = e2;
        }
        c->profiling = false;
        c->prof_sink = nullptr;
        if (e == cudaSuccess) e = cudaGraphInstantiateWithFlags(&c->round_exec, g, 0);
        if (g) cudaGraphDestroy(g);
      }
      if (e == cudaSuccess) e = cudaGraphLaunch(c->round_exec, c->stream);
      if (e == cudaSuccess) prof_after_replay(c, c->prof_round_graph);
    }
    if (e != cudaSuccess) return cuda_fail(c, e, "local steps launch");
    advance_clocks(c);
    c->pending = true;
    if (tau_out) std::memcpy(tau_out, c->tau.data(), c->W * sizeof(int32_t));
    if (loss_out) {
      e = cudaStreamSynchronize(c->stream);
      if (e == cudaSuccess) e = cudaMemcpy(loss_out, c->loss_dev, c->W * sizeof(float), cudaMemcpyDeviceToHost);
      if (e != cudaSuccess) return cuda_fail(c, e, "local steps");
      return check_err_word(c);
    }
    return OSCARS_OK;
  } catch (const std::bad_alloc&) {
    return fail(c, OSCARS_ENOMEM, "host allocation failed");
  }
}

oscars_status oscars_losses_async(oscars_ctx* c, float* dst) {
  if (!c || !dst) return OSCARS_EINVAL;
  if (!slotted(c) || c->rounds_run == 0) return fail(c, OSCARS_ESTATE, "no local steps to report");
  const cudaError_t e = cudaMemcpyAsync(dst, c->loss_dev, c->W * sizeof(float), cudaMemcpyDefault, c->stream);
  return e == cudaSuccess ? OSCARS_OK : cuda_fail(c, e, "loss copy");
}

oscars_status oscars_push_merge(oscars_ctx* c, const float* const* deltas, const float* weights) {
  if (!c) return OSCARS_EINVAL;
  if (c->rule == OSCARS_W_EXPLICIT && !weights) return fail(c, OSCARS_EINVAL, "explicit weight rule needs weights");
  MergeArgs a;
  std::memset(&a, 0, sizeof(a));
  a.W = c->W;
  if (c->rule == OSCARS_W_EXPLICIT) {
    for (int k = 0; k < c->W; ++k) a.w[k] = weights[k];
  } else {
    merge_weights(c->rule, c->tau.data(), c->W, a.w);
  }
  const float eta = c->server_lr;
  c->profiling = (c->flags & 2) != 0;
  struct ProfOff {
    oscars_ctx* c;
    ~ProfOff() { c->profiling = false; }
  } prof_off{c};
  float* xg = c->slab + (slotted(c) ? static_cast<int64_t>(c->W) * c->P_pad : 0);
  cudaError_t e = cudaSuccess;
  if (!deltas) {
    if (!slotted(c) || !c->pending)
      return fail(c, OSCARS_ESTATE, "push_merge without deltas needs pending local steps");
    auto enqueue = [&](cudaStream_t st) { return enqueue_replica_merge(c, a.w, st); };
    if (c->flags & 1) {
      e = enqueue(c->stream);
    } else {
      // the buffers of a replica-mode merge never change and its weights only
      // with the schedule, which drops the graph: one graph
      if (!c->merge_exec || c->rule == OSCARS_W_EXPLICIT) {
        if (c->merge_exec) cudaGraphExecDestroy(c->merge_exec);
        c->merge_exec = nullptr;
        for (auto& p : c->prof_merge_graph) {
          cudaEventDestroy(p.a);
          cudaEventDestroy(p.b);
        }
        c->prof_merge_graph.clear();
        c->prof_sink = &c->prof_merge_graph;
        cudaGraph_t g = nullptr;
        e = cudaStreamBeginCapture(c->cap, cudaStreamCaptureModeThreadLocal);
        if (e == cudaSuccess) {
          cudaError_t e2 = enqueue(c->cap);
          e = cudaStreamEndCapture(c->cap, &g);
          if (e2 != cudaSuccess) e = e2;
        }
        c->prof_sink = nullptr;
        if (e == cudaSuccess) e = cudaGraphInstantiateWithFlags(&c->merge_exec, g, 0);
        if (g) cudaGraphDestroy(g);
      }
      if (e == cudaSuccess) e = cudaGraphLaunch(c->merge_exec, c->stream);
      if (e == cudaSuccess) prof_after_replay(c, c->prof_merge_graph);
    }
    if (e != cudaSuccess) return cuda_fail(c, e, "merge launch");
    c->pending = false;
    return OSCARS_OK;
  } else {
    for (int k = 0; k < c->W; ++k)
      if (!deltas[k]) return fail(c, OSCARS_EINVAL, "NULL delta pointer");
    if (c->model == OSCARS_MODEL_CNN) return fail(c, OSCARS_ENOTSUP, "CNN: merge the workers' replicas (deltas == NULL)");
    if (c->model == OSCARS_MODEL_FLAT) {
      for (int k = 0; k < c->W; ++k) a.src[k] = deltas[k];
      ProfScope ps(c, "merge", c->stream);
      e = launch_merge(a, xg, c->P, eta, false, c->stream);
    } else {
      int64_t co = 0;
      for (const Layer& ly : c->layers) {
        const int64_t nw = static_cast<int64_t>(ly.in) * ly.out;
        for (int k = 0; k < c->W; ++k) a.src[k] = deltas[k] + co;
        e = launch_merge(a, xg + ly.offW, nw, eta, false, c->stream);
        if (e != cudaSuccess) break;
        for (int k = 0; k < c->W; ++k) a.src[k] = deltas[k] + co + nw;
        e = launch_merge(a, xg + ly.offB, ly.out, eta, false, c->stream);
        if (e != cudaSuccess) break;
        co += nw + ly.out;
      }
    }
  }
  if (e == cudaSuccess && c->model == OSCARS_MODEL_MLP) {
    ProfScope ps(c, "shadow_refresh", c->stream);
    e = refresh_global_shadows(c, c->stream);
  }
  if (e != cudaSuccess) return cuda_fail(c, e, "merge launch");
  c->pending = false;
  return OSCARS_OK;
}

oscars_status oscars_pull(oscars_ctx* c, float* dst) {
  if (!c) return OSCARS_EINVAL;
  cudaError_t e = cudaSuccess;
  const int64_t g = slotted(c) ? static_cast<int64_t>(c->W) * c->P_pad : 0;
  if (dst) {
    e = copy_canonical(c, c->slab + g, dst, false, c->stream);
    if (e == cudaSuccess && is_host_ptr(dst)) e = cudaStreamSynchronize(c->stream);
  } else if (slotted(c)) {
    e = launch_broadcast(c->slab + g, c->slab, c->P_pad, c->W, c->P_pad, c->stream);
    for (int k = 0; e == cudaSuccess && k < c->W && c->shadow; ++k)
      e = cudaMemcpyAsync(c->shadow + static_cast<int64_t>(k) * c->P_pad, c->shadow + g,
                          c->P_pad * sizeof(__nv_bfloat16), cudaMemcpyDeviceToDevice, c->stream);
  }
  if (e != cudaSuccess) return cuda_fail(c, e, "pull");
  return OSCARS_OK;
}

oscars_status oscars_get_schedule(const oscars_ctx* c, int64_t* T_star, int64_t* max_wait, int64_t* t_iter,
                                  int32_t* tau, int64_t* wait, int64_t* clock, int64_t* idle) {
  if (!c) return OSCARS_EINVAL;
  if (T_star) *T_star = c->barrier;
  if (max_wait) {
    int64_t m = 0;
    for (int i = 0; i < c->W; ++i) m = std::max(m, c->barrier - static_cast<int64_t>(c->tau[i]) * c->t_iter[i]);
    *max_wait = m;
  }
  for (int i = 0; i < c->W; ++i) {
    if (t_iter) t_iter[i] = c->t_iter[i];
    if (tau) tau[i] = c->tau[i];
    if (wait) wait[i] = c->barrier - static_cast<int64_t>(c->tau[i]) * c->t_iter[i];
    if (clock) clock[i] = c->clock[i];
    if (idle) idle[i] = c->idle[i];
  }
  return OSCARS_OK;
}

oscars_status oscars_set_local_steps(oscars_ctx* c, const int32_t* tau) {
  if (!c || !tau) return OSCARS_EINVAL;
  if (c->pending) return fail(c, OSCARS_ESTATE, "cannot change tau while a round is pending");
  for (int i = 0; i < c->W; ++i)
    if (tau[i] < 1) return fail(c, OSCARS_EINVAL, "tau must be >= 1");
  for (int i = 0; i < c->W; ++i) c->tau[i] = tau[i];
  update_barrier(c, false);
  if (slotted(c)) {
    cudaStreamSynchronize(c->stream);
    return build_tables(c);
  }
  return OSCARS_OK;
}

oscars_status oscars_set_iteration_ticks(oscars_ctx* c, const int64_t* t_iter) {
  if (!c || !t_iter) return OSCARS_EINVAL;
  if (c->pending) return fail(c, OSCARS_ESTATE, "cannot re-schedule while a round is pending");
  std::vector<int64_t> t(t_iter, t_iter + c->W);
  std::vector<int32_t> tau(c->W, 1);
  int64_t T = 0, mw = 0;
  const char* why = "";
  const int r = schedule_solve(t.data(), c->W, c->M, c->search_mode, &T, &mw, tau.data(), &why);
  if (r != OSCARS_OK) return fail(c, static_cast<oscars_status>(r), why);
  c->t_iter = t;
  c->tau = tau;
  c->T_star = T;
  c->max_wait = mw;
  update_barrier(c, true);
  if (slotted(c)) {
    cudaStreamSynchronize(c->stream);
    return build_tables(c);
  }
  return OSCARS_OK;
}

oscars_status oscars_eval_loss(oscars_ctx* c, const float* x, const int32_t* y, int64_t n, float* loss) {
  if (!c || !x || !y || !loss || n < 1) return OSCARS_EINVAL;
  if (!slotted(c)) return fail(c, OSCARS_ESTATE, "eval needs an MLP or CNN context");
  cudaError_t e = cudaSuccess;
  const int64_t g = static_cast<int64_t>(c->W) * c->P_pad;
  if (c->model == OSCARS_MODEL_CNN) {
    // chunks of up to B images through lane 0 with the global model's weights
    const int64_t chunks = (n + c->B - 1) / c->B;
    if (c->eval_part_cap < chunks) {
      if (!dev_alloc(c, &c->eval_part, chunks)) return fail(c, OSCARS_ENOMEM, "eval scratch");
      c->eval_part_cap = chunks;
    }
    if (c->estart_cap < 1) {
      if (!dev_alloc(c, &c->estart, 1)) return fail(c, OSCARS_ENOMEM, "eval scratch");
      c->estart_cap = 1;
    }
    const int64_t zero = 0;
    const int64_t img = static_cast<int64_t>(c->dims[0]) * c->dims[1] * c->dims[2];
    e = cudaMemcpyAsync(c->estart, &zero, sizeof(int64_t), cudaMemcpyHostToDevice, c->stream);
    for (int64_t ch = 0; e == cudaSuccess && ch < chunks; ++ch) {
      const int Bc = static_cast<int>(std::min<int64_t>(c->B, n - ch * c->B));
      const float* xc = x + ch * c->B * img;
      const int32_t* yc = y + ch * c->B;
      const int64_t nc = Bc;
      e = cudaMemcpyAsync(c->ex_tab, &xc, sizeof(float*), cudaMemcpyHostToDevice, c->stream);
      if (e == cudaSuccess) e = cudaMemcpyAsync(c->ey_tab, &yc, sizeof(int32_t*), cudaMemcpyHostToDevice, c->stream);
      if (e == cudaSuccess) e = cudaMemcpyAsync(c->en_tab, &nc, sizeof(int64_t), cudaMemcpyHostToDevice, c->stream);
      if (e == cudaSuccess) e = cudaStreamSynchronize(c->stream);   // the host values above must not go out of scope early
      if (e != cudaSuccess) break;
      CnnStageArgs a{};
      a.x = c->ex_tab;
      a.y = c->ey_tab;
      a.n = c->en_tab;
      a.start = c->estart;
      a.wid = c->lane_ids;
      a.step = 0;
      a.B = Bc;
      a.Cin = c->dims[2];
      a.im2col = c->cnn_im2col ? 1 : 0;
      a.out = c->cnn_buf[0];
      a.labels = c->labels;
      e = launch_cnn_stage(a, 1, c->stream);
      auto conv = [&](int layer, int in, int add, int out) -> cudaError_t {
        ConvArgs ca;
        std::memset(&ca, 0, sizeof(ca));
        ca.wid = c->lane_ids;
        ca.src = c->global_src;
        ca.B = Bc;
        ca.bias = c->slab;
        ca.slot_stride = c->P_pad;
        ca.off_bias = c->cnn_offB[layer];
        ca.add = add >= 0 ? c->cnn_buf[add] : nullptr;
        ca.out = c->cnn_buf[out];
        ca.err = c->err;
        ca.im2col = layer == 0 && c->cnn_im2col ? 1 : 0;
        return launch_conv_igemm(0, ca.im2col ? c->cnn_m4[in] : c->cnn_m6[in], c->cnn_mw[layer], ca, 1,
                                 conv_ctas_per_worker(Bc, 1, c->sms), c->stream);
      };
      if (e == cudaSuccess) e = conv(0, 0, -1, 1);
      for (int k = 0; e == cudaSuccess && k < c->cnn_blocks; ++k) {
        const int h = k == 0 ? 1 : 3 + 2 * (k - 1);
        e = conv(1 + 2 * k, h, -1, 2 + 2 * k);
        if (e == cudaSuccess) e = conv(2 + 2 * k, 2 + 2 * k, h, 3 + 2 * k);
      }
      if (e == cudaSuccess)
        e = launch_cnn_pool(c->cnn_buf[3 + 2 * (c->cnn_blocks - 1)], c->lane_ids, Bc, c->cnn_g, 1, c->stream);
      if (e == cudaSuccess)
        e = launch_cnn_head_loss(c->cnn_g, c->labels, Bc, c->C, c->slab + g, c->cnn_offWf, c->cnn_offBf,
                                 c->eval_part + ch, c->stream);
    }
    if (e == cudaSuccess) e = launch_sum_scaled(c->eval_part, chunks, 1.0 / static_cast<double>(n), c->loss_dev, c->stream);
  } else if (c->L == 1 && !c->bf16) {
    const int blocks = static_cast<int>(std::min<int64_t>(1024, (n + 7) / 8));
    if (c->eval_part_cap < blocks) {
      if (!dev_alloc(c, &c->eval_part, blocks)) return fail(c, OSCARS_ENOMEM, "eval scratch");
      c->eval_part_cap = blocks;
    }
    SoftregEvalArgs a;
    a.master = c->slab + g;
    a.offW = c->layers[0].offW;
    a.offB = c->layers[0].offB;
    a.D = c->dims[0];
    a.C = c->C;
    a.x = x;
    a.y = y;
    a.n = n;
    a.loss_sum = c->eval_part;
    e = launch_softreg_eval(a, blocks, c->stream);
    if (e == cudaSuccess) e = launch_sum_scaled(c->eval_part, blocks, 1.0 / static_cast<double>(n), c->loss_dev, c->stream);
  } else {
    if (n % c->B != 0) return fail(c, OSCARS_ENOTSUP, "MLP eval: n must be a multiple of the batch size");
    const int64_t chunks = n / c->B;
    const int nc = c->B / kRowsPerLossChunk;
    if (c->estart_cap < chunks) {
      if (!dev_alloc(c, &c->estart, chunks)) return fail(c, OSCARS_ENOMEM, "eval scratch");
      c->estart_cap = chunks;
    }
    if (c->eval_part_cap < chunks * nc) {
      if (!dev_alloc(c, &c->eval_part, chunks * nc)) return fail(c, OSCARS_ENOMEM, "eval scratch");
      c->eval_part_cap = chunks * nc;
    }
    std::vector<int64_t> starts(chunks), ns(c->W, n);
    for (int64_t i = 0; i < chunks; ++i) starts[i] = i * c->B;
    std::vector<const float*> xs(c->W, x);
    std::vector<const int32_t*> ys(c->W, y);
    e = cudaStreamSynchronize(c->stream);
    if (e == cudaSuccess) e = cudaMemcpy(c->estart, starts.data(), chunks * sizeof(int64_t), cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMemcpy(c->ex_tab, xs.data(), c->W * sizeof(float*), cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMemcpy(c->ey_tab, ys.data(), c->W * sizeof(int32_t*), cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMemcpy(c->en_tab, ns.data(), c->W * sizeof(int64_t), cudaMemcpyHostToDevice);
    for (int64_t base = 0; e == cudaSuccess && base < chunks; base += c->W) {
      const int na = static_cast<int>(std::min<int64_t>(c->W, chunks - base));
      StageArgs sa{};
      sa.x = c->ex_tab;
      sa.y = c->ey_tab;
      sa.n = c->en_tab;
      sa.start = c->estart + base;
      sa.row_add = 0;
      sa.wid = c->lane_ids;
      sa.D = c->dims[0];
      sa.B = c->B;
      sa.A0 = c->A[0];
      sa.A0T = c->AT[0];
      sa.labels = c->labels;
      e = launch_stage(sa, na, c->stream);
      c->cur_buf = 0;   // the evaluation stages its rows into the first input buffer
      if (e == cudaSuccess) e = enqueue_forward(c, c->lane_ids, c->global_src, na, c->stream);
      if (e == cudaSuccess) {
        HeadArgs h = head_base(c);
        h.wid = c->lane_ids;
        h.src = c->global_src;
        h.loss_part = c->eval_part;
        h.part_mul = 1;
        h.part_add = static_cast<int>(base);
        e = launch_head_fwd(h, na, c->stream);
      }
    }
    if (e == cudaSuccess)
      e = launch_sum_scaled(c->eval_part, chunks * nc, 1.0 / static_cast<double>(n), c->loss_dev, c->stream);
  }
  if (c->model == OSCARS_MODEL_MLP && c->L >= 2) c->staged = false;   // eval used the first input buffer
  if (e == cudaSuccess) e = cudaStreamSynchronize(c->stream);
  if (e == cudaSuccess) e = cudaMemcpy(loss, c->loss_dev, sizeof(float), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(c, e, "eval");
  return check_err_word(c);
}

oscars_status oscars_debug_slab(const oscars_ctx* c, float** slab, int64_t* slot_stride) {
  if (!c || !slab || !slot_stride) return OSCARS_EINVAL;
  *slab = c->slab;
  *slot_stride = c->P_pad;
  return OSCARS_OK;
}

oscars_status oscars_check_padding(oscars_ctx* c, int64_t* bad) {
  if (!c || !bad) return OSCARS_EINVAL;
  if (!slotted(c)) return fail(c, OSCARS_ESTATE, "the padding check needs an MLP or CNN context");
  try {
    const size_t slots = static_cast<size_t>(c->W) + 1, n = slots * c->P_pad;
    std::vector<uint32_t> f(n + kGuardWords);
    cudaError_t e = cudaStreamSynchronize(c->stream);
    if (e == cudaSuccess) e = cudaMemcpy(f.data(), c->slab, f.size() * sizeof(uint32_t), cudaMemcpyDeviceToHost);
    std::vector<uint16_t> h;
    if (e == cudaSuccess && c->shadow) {
      h.resize(n + kGuardWords);
      e = cudaMemcpy(h.data(), c->shadow, h.size() * sizeof(uint16_t), cudaMemcpyDeviceToHost);
    }
    if (e != cudaSuccess) return cuda_fail(c, e, "padding check");
    int64_t count = 0;
    const uint32_t g32 = 0x01010101u * kGuardByte;
    const uint16_t g16 = static_cast<uint16_t>(0x0101u * kGuardByte);
    for (size_t i = n; i < f.size(); ++i) count += f[i] != g32;
    for (size_t i = n; i < h.size(); ++i) count += h[i] != g16;
    if (c->model == OSCARS_MODEL_MLP) {
      // the gaps between a slot's tensors and its tail (the layout pads each
      // W_l and b_l to 64 elements); the value bits of -0.0 count as set
      for (size_t k = 0; k < slots; ++k) {
        const size_t base = k * c->P_pad;
        for (size_t l = 0; l < c->layers.size(); ++l) {
          const Layer& ly = c->layers[l];
          const int64_t end = l + 1 < c->layers.size() ? c->layers[l + 1].offW : c->P_pad;
          const int64_t gaps[2][2] = {{ly.offW + static_cast<int64_t>(ly.in) * ly.out, ly.offB},
                                      {ly.offB + ly.out, end}};
          for (const auto& g : gaps)
            for (int64_t i = g[0]; i < g[1]; ++i) {
              count += f[base + i] != 0u;
              if (!h.empty()) count += h[base + i] != 0u;
            }
        }
      }
    }
    *bad = count;
    return OSCARS_OK;
  } catch (const std::bad_alloc&) {
    return fail(c, OSCARS_ENOMEM, "host allocation failed");
  }
}

oscars_status oscars_check_wait_timeout(oscars_ctx* c, int32_t polls) {
  if (!c || polls < 1 || polls > (1 << 20)) return OSCARS_EINVAL;
  if (!c->err) return fail(c, OSCARS_ESTATE, "the context has no kernel error word (FLAT mode)");
  cudaError_t e = launch_wait_selfcheck(c->err, static_cast<uint32_t>(polls), c->stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(c->stream);
  if (e != cudaSuccess) return cuda_fail(c, e, "wait self-check");
  return check_err_word(c);
}

oscars_status oscars_read_replica(oscars_ctx* c, int32_t k, float* dst) {
  if (!c || !dst) return OSCARS_EINVAL;
  if (!slotted(c)) return fail(c, OSCARS_ESTATE, "replicas exist in MLP and CNN mode only");
  if (k < 0 || k >= c->W) return fail(c, OSCARS_EINVAL, "worker index out of range");
  cudaError_t e = copy_canonical(c, c->slab + static_cast<int64_t>(k) * c->P_pad, dst, false, c->stream);
  if (e == cudaSuccess && is_host_ptr(dst)) e = cudaStreamSynchronize(c->stream);
  if (e != cudaSuccess) return cuda_fail(c, e, "read replica");
  return OSCARS_OK;
}

oscars_status oscars_gemm_bf16_nt(const void* A, const void* B, float* C, int32_t M, int32_t N, int32_t K,
                                  void* stream) {
  if (!A || !B || !C || M < 128 || M % 128 != 0 || N < 1 || K < 8 || K % 8 != 0) return OSCARS_EINVAL;
  if ((reinterpret_cast<uintptr_t>(A) | reinterpret_cast<uintptr_t>(B)) & 15) return OSCARS_EINVAL;
  CUtensorMap mA, mB;
  if (!make_map(&mA, A, K, M, 1, K * 2ull, static_cast<uint64_t>(M) * K * 2ull, 128) ||
      !make_map(&mB, B, K, N, 1, K * 2ull, static_cast<uint64_t>(N) * K * 2ull, 128))
    return OSCARS_ECUDA;
  GemmArgs g;
  std::memset(&g, 0, sizeof(g));
  g.M = M;
  g.N = N;
  g.K = K;
  g.c_out = C;
  return launch_gemm(kEpiStore, mA, mB, g, 1, static_cast<cudaStream_t>(stream)) == cudaSuccess ? OSCARS_OK
                                                                                               : OSCARS_ECUDA;
}

int32_t oscars_phase_times(oscars_ctx* c, int32_t cap, double* us) {
  if (!c || !us || cap < 1) return -1;
  if (!c->phase_ts || !c->fused) return 0;
  std::vector<unsigned long long> h(static_cast<size_t>(c->max_tau) * 4);
  if (cudaStreamSynchronize(c->stream) != cudaSuccess ||
      cudaMemcpy(h.data(), c->phase_ts, h.size() * sizeof(unsigned long long), cudaMemcpyDeviceToHost) != cudaSuccess)
    return -1;
  const int steps = c->tau[0];
  int n = 0;
  for (int s = 0; s < steps && n + 3 <= cap; ++s)
    for (int p = 0; p < 3; ++p) us[n++] = (h[s * 4 + p + 1] - h[s * 4 + p]) * 1e-3;
  return n;
}

int32_t oscars_profile_read(oscars_ctx* c, int32_t cap, const char** names, double* ms_total, int32_t* launches) {
  if (!c) return -1;
  prof_collect(c);
  const int n = static_cast<int>(c->prof_names.size());
  for (int i = 0; i < n && i < cap; ++i) {
    if (names) names[i] = c->prof_names[i].c_str();
    if (ms_total) ms_total[i] = c->prof_ms[i];
    if (launches) launches[i] = c->prof_count[i];
  }
  return n;
}

oscars_status oscars_profile_reset(oscars_ctx* c) {
  if (!c) return OSCARS_EINVAL;
  prof_collect(c);
  c->prof_names.clear();
  c->prof_ms.clear();
  c->prof_count.clear();
  return OSCARS_OK;
}

namespace {

// oscars_train without evaluation: round r (local steps, the asynchronous copy
// of its W losses into a pinned host slot, push + merge) is enqueued before
// the host waits for round r - 1 and reads that round's losses, so the host
// work of one round overlaps the device work of the next.
oscars_status train_pipelined(oscars_ctx* c, int32_t rounds, oscars_round_log* log, int32_t* rounds_done) {
  if (!c->train_loss_host) {
    cudaError_t e = cudaHostAlloc(&c->train_loss_host, 2 * sizeof(float) * c->W, cudaHostAllocDefault);
    if (e != cudaSuccess) {
      c->train_loss_host = nullptr;
      return cuda_fail(c, e, "train loss buffer");
    }
    for (auto& ev : c->train_done)
      if ((e = cudaEventCreateWithFlags(&ev, cudaEventDisableTiming)) != cudaSuccess) return cuda_fail(c, e, "train event");
  }
  auto finish = [&](int32_t r) -> oscars_status {
    const cudaError_t e = cudaEventSynchronize(c->train_done[r & 1]);
    if (e != cudaSuccess) return cuda_fail(c, e, "train round");
    if (log) {
      const float* l = c->train_loss_host + (r & 1) * c->W;
      double m = 0.0;
      for (int i = 0; i < c->W; ++i) m += l[i];
      log[r].worker_loss = static_cast<float>(m / c->W);
    }
    if (rounds_done) *rounds_done = r + 1;
    return OSCARS_OK;
  };
  for (int32_t r = 0; r < rounds; ++r) {
    oscars_status st = oscars_local_steps(c, nullptr, nullptr);
    if (st == OSCARS_OK) st = oscars_losses_async(c, c->train_loss_host + (r & 1) * c->W);
    if (st == OSCARS_OK) st = oscars_push_merge(c, nullptr, nullptr);
    if (st != OSCARS_OK) return st;
    if (log) {
      log[r].ticks = *std::max_element(c->clock.begin(), c->clock.end());
      log[r].barrier = c->barrier;
      log[r].eval_loss = std::numeric_limits<float>::quiet_NaN();
    }
    const cudaError_t e = cudaEventRecord(c->train_done[r & 1], c->stream);
    if (e != cudaSuccess) return cuda_fail(c, e, "train event");
    if (r >= 1 && (st = finish(r - 1)) != OSCARS_OK) return st;
  }
  const oscars_status st = finish(rounds - 1);
  // the kernels' error word is sticky: one read after the last round reports
  // a bounded wait that ran out in any of them
  return st == OSCARS_OK ? check_err_word(c) : st;
}

}  // namespace

oscars_status oscars_train(oscars_ctx* c, int32_t rounds, const float* eval_x, const int32_t* eval_y,
                           int64_t eval_n, float target_loss, oscars_round_log* log, int32_t* rounds_done) {
  if (rounds_done) *rounds_done = 0;
  if (!c || rounds < 1) return OSCARS_EINVAL;
  if (eval_x && (!eval_y || eval_n < 1)) return OSCARS_EINVAL;
  if (c->rule == OSCARS_W_EXPLICIT) return fail(c, OSCARS_EINVAL, "train merges with the context's rule; explicit weights need push_merge");
  try {
    if (!eval_x) return train_pipelined(c, rounds, log, rounds_done);
    std::vector<float> wl(c->W);
    for (int32_t r = 0; r < rounds; ++r) {
      oscars_status st = oscars_local_steps(c, nullptr, wl.data());
      if (st != OSCARS_OK) return st;
      st = oscars_push_merge(c, nullptr, nullptr);
      if (st != OSCARS_OK) return st;
      float ev = std::numeric_limits<float>::quiet_NaN();
      if (eval_x) {
        st = oscars_eval_loss(c, eval_x, eval_y, eval_n, &ev);
        if (st != OSCARS_OK) return st;
      }
      if (log) {
        double m = 0.0;
        for (int i = 0; i < c->W; ++i) m += wl[i];
        log[r].ticks = *std::max_element(c->clock.begin(), c->clock.end());
        log[r].barrier = c->barrier;
        log[r].eval_loss = ev;
        log[r].worker_loss = static_cast<float>(m / c->W);
      }
      if (rounds_done) *rounds_done = r + 1;
      if (eval_x && target_loss > 0.f && ev <= target_loss) break;
    }
    return OSCARS_OK;
  } catch (const std::bad_alloc&) {
    return fail(c, OSCARS_ENOMEM, "host allocation failed");
  }
}

oscars_status oscars_num_params(const oscars_ctx* c, int64_t* P) {
  if (!c || !P) return OSCARS_EINVAL;
  *P = c->P;
  return OSCARS_OK;
}

const char* oscars_last_error(const oscars_ctx* c) { return c ? c->last_error.c_str() : ""; }

oscars_status oscars_merge(float* x_g, const float* const* deltas, const float* w, int32_t W, int64_t P,
                           float server_lr, void* stream) {
  if (!x_g || !deltas || !w || W < 1 || W > kMaxMergeWorkers || P < 0) return OSCARS_EINVAL;
  MergeArgs a;
  std::memset(&a, 0, sizeof(a));
  a.W = W;
  for (int k = 0; k < W; ++k) {
    if (!deltas[k]) return OSCARS_EINVAL;
    a.src[k] = deltas[k];
    a.w[k] = w[k];
  }
  return launch_merge(a, x_g, P, server_lr, false, static_cast<cudaStream_t>(stream)) == cudaSuccess ? OSCARS_OK
                                                                                                   : OSCARS_ECUDA;
}

}  // extern "C"
