// Internal declarations shared by the translation units of liboscars.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace oscars {

constexpr int kMaxMergeWorkers = 256;   // pointer table of the merge kernel
constexpr int kMaxWorkersMLP = 64;
constexpr int kMaxClasses = 32;
constexpr int kRowsPerLossChunk = 16;   // rows per loss partial in the head kernel

// ---------------------------------------------------------------- merge
struct MergeArgs {
  const float* src[kMaxMergeWorkers];  // delta_k, or replica x^k
  float w[kMaxMergeWorkers];
  int W;
};

// x_g <- x_g + eta * sum_k w_k * (replica ? src_k - x_g : src_k), p < P;
// shadow (optional): shadow[p] = bf16(new x_g[p]) in the same pass.
cudaError_t launch_merge(const MergeArgs& a, float* x_g, int64_t P, float eta, bool replica,
                         cudaStream_t s, __nv_bfloat16* shadow = nullptr);

// one thread waits `polls` polls on an mbarrier nothing completes, then
// records its timeout code in *err (the bounded-wait failure path)
cudaError_t launch_wait_selfcheck(int* err, uint32_t polls, cudaStream_t s);

// ---------------------------------------------------------------- scheduler (host)
int iteration_ticks(const double* speed, int n, int64_t Q, int64_t* t, const char** why);
int schedule_solve(const int64_t* t, int n, int64_t M, int mode, int64_t* T_star,
                   int64_t* max_wait, int32_t* tau, const char** why);
void merge_weights(int rule, const int32_t* tau, int n, float* w);

// ---------------------------------------------------------------- softmax regression (fp32)
struct SoftregArgs {
  const float* master;          // slab base (slots of P_pad floats)
  float* master_out;
  int64_t slot_stride;          // P_pad
  int global_slot;              // W
  int64_t offW, offB;           // element offsets inside a slot
  int D, C, B;
  float lr;
  const int32_t* tau;           // [W]
  const float* const* shard_x;  // [W] device pointers
  const int32_t* const* shard_y;
  const int64_t* shard_n;       // [W]
  const int64_t* cursor;        // [W]
  float* loss_part;             // [W][max_tau]  (sum of per-sample losses of one step)
  int max_tau;
  // round bookkeeping in the same launch (null: not done): the worker's mean
  // loss over its steps, and its cursor advanced by tau * B (mod the shard)
  float* loss_out = nullptr;    // [W]
  int64_t* cursor_next = nullptr;   // [W], may be `cursor` itself
};
cudaError_t launch_softreg_round(const SoftregArgs& a, int W, cudaStream_t s);
size_t softreg_smem_bytes(int D, int C, int B);
// the round kernel gives each mini-batch row one thread for its row offset,
// label and softmax: B must not exceed its block size
constexpr int kSoftregMaxBatch = 512;
// the same round with each worker on a cluster of 8 CTAs splitting the input
// columns (B <= 256 and a column slice plus one batch slice in shared memory)
bool softreg_cluster_supported(int D, int C, int B);
int softreg_cluster_cols(int D);
size_t softreg_cluster_smem_bytes(int D, int C, int B);
cudaError_t launch_softreg_cluster_round(const SoftregArgs& a, int W, cudaStream_t s);

struct SoftregEvalArgs {
  const float* master;  // global slot
  int64_t offW, offB;
  int D, C;
  const float* x;
  const int32_t* y;
  int64_t n;
  float* loss_sum;      // [blocks] partial sums
};
cudaError_t launch_softreg_eval(const SoftregEvalArgs& a, int blocks, cudaStream_t s);

// ---------------------------------------------------------------- MLP (bf16 GEMMs)
// Rows of one step's work: active lane i uses activation buffers of lane
// `wid[i]` and reads parameters from slot `src[i]` (the global slot on the
// first local step: the fused pull), writing them to slot `wid[i]`.
struct StageArgs {
  const float* const* x;   // [lanes] sample matrix per lane (device pointers)
  const int32_t* const* y;
  const int64_t* n;        // [lanes] rows available
  const int64_t* start;    // [lanes] first row (cursor)
  int64_t row_add;         // added to start (step * B)
  const int* wid;          // [n_active]
  int D, B;
  __nv_bfloat16* A0;       // [lanes][B][D]
  __nv_bfloat16* A0T;      // [lanes][D][B]
  int32_t* labels;         // [lanes][B]
  const int32_t* ahead;    // stage_round: null, or tau (the next round: rows from start + tau * B)
  const int32_t* slots;    // stage_round: the n_slots active slots s * W + w (s < tau[w]), or null (all)
  int n_slots;
};
cudaError_t launch_stage(const StageArgs& a, int n_active, cudaStream_t s);
// all mini-batches of a round: step s of worker w (s < tau[w]) at slot s * W + w
// (grid z over a.slots when given, else over all max_tau * W slots)
cudaError_t launch_stage_round(const StageArgs& a, const int32_t* tau, int W, int max_tau, cudaStream_t s);
// the same with a launch priority (cudaLaunchAttributePriority)
// the same staging from `blocks` blocks striding over the tiles (bounded footprint beside other kernels)
cudaError_t launch_stage_round_strided(const StageArgs& a, const int32_t* tau, int W, int max_tau, int blocks,
                                       int priority, cudaStream_t s);
cudaError_t launch_stage_round_priority(const StageArgs& a, const int32_t* tau, int W, int max_tau, int priority,
                                        cudaStream_t s);

enum GemmEpi { kEpiFwd = 0, kEpiDh = 1, kEpiDw = 2, kEpiStore = 3 };

struct GemmArgs {
  const int* wid;     // [n_active]
  const int* src;     // [n_active]
  int M, N, K;
  int a_z_src, b_z_src;  // TMA z coordinate of A / B: 1 = src slot, 0 = lane id
  int b_mn;              // kEpiDh: B read MN-major (G^T [lane][K][N] in boxes of 64 N x 64 K; N % 64 == 0)
  int pdl;               // launch as a programmatic dependent of the previous kernel on the stream
  int* err;
  // kEpiFwd: out = relu(acc + bias[m]) -> H [lane][N][M], HT [lane][M][N]
  // kEpiDh : out = acc * (Hmask[lane][n][m] > 0) -> G (if out), GT, gb[lane][m]
  // kEpiDw : W[dst] = W[src] - lr * acc (rows m, cols n < N), shadows, bias
  const float* master;      // fp32 slab base
  float* master_w;          // same slab (written)
  __nv_bfloat16* shadow;    // bf16 slab (same layout as master)
  int64_t slot_stride;      // P_pad
  int64_t offW, offB;       // element offsets of W_l, b_l in a slot
  float lr;
  const float* gb_in;       // [lanes][M] bias gradient (kEpiDw)
  const __nv_bfloat16* hmask;  // [lanes][N][M] (kEpiDh)
  __nv_bfloat16* out;       // [lanes][N][M]
  __nv_bfloat16* outT;      // [lanes][M][N]
  float* gb_out;            // [lanes][M] (kEpiDh)
  float* c_out;             // kEpiStore: C [M][N] fp32 row-major (lane 0 only)
};
cudaError_t launch_gemm(int epi, const CUtensorMap& mapA, const CUtensorMap& mapB,
                        const GemmArgs& a, int n_active, cudaStream_t s);

// Weight gradient + SGD of one layer, persistent (csrc/gemm_dw.cu):
// W[wid] = W[src] - lr * G^T X over the batch, its bf16 copy, and the bias
// b[wid] = b[src] - lr * gb[wid] (outputs m < M, inputs n < N, batch K).
struct DwArgs {
  const int* wid;           // [n_active] destination slots (device), or null = lane id
  const int* src;           // [n_active] source slots (device), or null = lane id
  int n_active;
  int M, N, K;
  float lr;
  const float* master;      // fp32 slab (bias read)
  float* master_w;          // fp32 slab (bias written)
  int64_t slot_stride;      // P_pad
  int64_t offB;             // element offset of b_l in a slot
  const float* gb;          // [W][M] bias gradient
  int* err;
  int pdl;                  // launch as a programmatic dependent of the previous kernel on the stream
};
bool gemm_dw_supported(int M, int N, int K);
// mA: G^T [lane][M][K] bf16, box {64, 128}; mB: X^T [lane][N][K] bf16, box
// {64, 128}; mMaster: W_l fp32 [slot][M][N], box {32, 128} (loads);
// mMasterSt: the same with box {32, 32} (stores); mShadowSt: W_l bf16
// [slot][M][N], box {64, 32} (stores); all with 128-byte swizzle.  `sms`:
// the device's multiprocessors (one CTA each at most).
cudaError_t launch_gemm_dw(const CUtensorMap& mA, const CUtensorMap& mB, const CUtensorMap& mMaster,
                           const CUtensorMap& mMasterSt, const CUtensorMap& mShadowSt, const DwArgs& a, int sms,
                           cudaStream_t s);
int gemm_bn_for(int epi, int N);

struct HeadArgs {
  const int* wid;
  const int* src;
  int H, C, B;
  const __nv_bfloat16* Ain;   // [lanes][B][H] input of the last layer
  const int32_t* labels;      // [lanes][B]
  const __nv_bfloat16* shadow;
  const float* master;
  float* master_w;
  __nv_bfloat16* shadow_w;
  int64_t slot_stride;
  int64_t offW, offB;
  float lr;
  float* dlog;                // [lanes][B][C]
  float* loss_part;           // rows of (B/16) partial sums
  int part_mul, part_add;     // row = wid * part_mul + part_add
  __nv_bfloat16* G;           // [lanes][B][H] (head_bwd)
  __nv_bfloat16* GT;          // [lanes][H][B]
  float* gb;                  // [lanes][H]
  int* err;                   // device error word (bounded waits of the tensor-core head)
  int pdl;                    // tensor-core head: launch as a programmatic dependent
};
cudaError_t launch_head_fwd(const HeadArgs& a, int n_active, cudaStream_t s);
// forward + backward of the last layer on the tensor cores (csrc/head_tc.cu):
// one cluster of H/128 CTAs per active lane; C = 10, 32 <= B <= 128.  mH: the
// layer input [lane][B][H] bf16, box {64, 128}; mW2: the head weights of every
// slot [slot][C][H] bf16, box {64, 16}; both with 128-byte swizzle.
bool head_tc_supported(int H, int B, int C);
cudaError_t launch_head_tc(const CUtensorMap& mH, const CUtensorMap& mW2, const HeadArgs& a, int n_active,
                           cudaStream_t s);
// forward + backward of the last layer in one launch: one cluster of H/128
// CTAs per active lane (H <= 1024); false if the shape needs the two-kernel path
bool head_fused_supported(int H, int B, int C);
cudaError_t launch_head_fused(const HeadArgs& a, int n_active, cudaStream_t s);
cudaError_t launch_head_bwd(const HeadArgs& a, int n_active, cudaStream_t s);

// ---------------------------------------------------------------- fused round (2-layer MLP)
struct FusedRoundArgs {
  const int32_t* tau;
  const int32_t* order;           // [W] workers, cluster by cluster (longest first)
  const int32_t* cl_first;        // [n_clusters + 1] cluster k runs order[cl_first[k] .. cl_first[k + 1])
  int W, n_clusters, D, H, B;
  int global_slot;
  float lr;
  const float* master;
  float* master_w;
  int64_t slot_stride;
  int64_t offW0, offB0, offW1, offB1;
  const int32_t* labels;
  int max_tau;
  int* err;
  unsigned long long* phase_ts;   // [max_tau][4] phase stamps of worker 0, or null
  float* loss_out;                // [W] mean mini-batch loss of the round (written at the end)
  int64_t* cursor;                // [W] advanced by tau * B modulo n at the end, or null
  const int64_t* shard_n;         // [W]
  int priority;                   // launch priority (cudaLaunchAttributePriority); 0: the stream's
};
// whole-round kernel for input -> H ReLU -> 10 classes (one cluster per
// worker, the worker's model resident on chip for the round)
bool fused_round_supported(int L, int D, int H, int C, int B);
int fused_round_xt_rows(int B);   // rows of the X^T box the kernel loads
// clusters of the round kernel that fit on the device at once (0 if unknown)
int fused_round_max_clusters(int D, int H, int B);
// mX: staged inputs {D, B, W, steps} box {64, B}; mXT: staged transposed
// inputs {B, D, W, steps} box {64, fused_round_xt_rows(B)}; both bf16,
// 128-byte swizzle.  mW0f: the global slot's W0 {D, H, 1} fp32, box
// {32, 128}, 128-byte swizzle (the kernel rounds its own bf16 operand).
// mRep32 / mRep16: W0 of every replica slot {D, H, slots} fp32, box
// {32, 32} with 128-byte swizzle / {16, 32} without (the last step's stores)
cudaError_t launch_fused_round(const CUtensorMap& mX, const CUtensorMap& mXT, const CUtensorMap& mW0f,
                               const CUtensorMap& mRep32, const CUtensorMap& mRep16, const FusedRoundArgs& a,
                               cudaStream_t s);

// loss[w] = sum_{s < tau[w]} sum_c part[(w*max_tau + s)*nc + c] / (B * tau[w])
cudaError_t launch_loss_finalize(const float* part, const int32_t* tau, int W, int max_tau,
                                 int nc, int B, float* loss, cudaStream_t s);
// out[0] = sum_i part[i] / n (fixed order)
cudaError_t launch_sum_scaled(const float* part, int64_t count, double scale, float* out,
                              cudaStream_t s);
// cursor[w] = (cursor[w] + tau[w] * B) % n[w]
cudaError_t launch_cursor_advance(int64_t* cursor, const int32_t* tau, const int64_t* n, int B,
                                  int W, cudaStream_t s);
// shadow[p] = bf16(master[p]) for one slot; shadowT for layers with a transposed copy
cudaError_t launch_shadow_refresh(const float* master, __nv_bfloat16* shadow, int64_t count,
                                  cudaStream_t s);
cudaError_t launch_transpose_bf16(const __nv_bfloat16* src, __nv_bfloat16* dst, int rows,
                                  int cols, cudaStream_t s);
// replicas[k] = x_g for k < W (fp32 and bf16 shadows)
cudaError_t launch_broadcast(const float* xg, float* slab, int64_t stride, int W, int64_t count,
                             cudaStream_t s);

// ---------------------------------------------------------------- convolutional worker
// 32 x 32 images, 64 channels, 3x3 convolutions (csrc/cnn.cu)

struct ConvArgs {
  const int* wid;              // [n_active] lane of each active entry
  const int* src;              // [n_active] slot whose weights the step reads
  int B;                       // images per lane
  const float* bias;           // forward: fp32 slab; bias of slot s at bias + s * slot_stride + off_bias
  int64_t slot_stride, off_bias;
  const __nv_bfloat16* add;    // [lane][B][1024][64] added before the activation / mask, or null
  const __nv_bfloat16* mask;   // input gradient: stored activation of the layer input (> 0 keeps)
  __nv_bfloat16* out;          // [lane][B][1024][64]
  float* bias_part;            // input gradient: [lane][cpw][64] per-CTA channel sums, or null
  int* err;
  int im2col;                  // forward only: 1 = the stem as one 64 x 64 product over the im2col input
};
struct WgradArgs {
  const int* wid;
  int B, n_chunks, img_per_chunk;
  float* part;                 // [lane][n_chunks][9][64 in][64 out]
  int* err;
  int im2col;                  // 1 = the stem over the im2col input: tap 0 of `part` only
};
constexpr int kMaxConvLayers = 9;
struct ConvSgdArgs {
  const int* wid;
  const int* src;
  int n_chunks, layers;
  int n_tiles[kMaxConvLayers];             // per layer: bias partials per lane
  const float* part[kMaxConvLayers];       // per layer, as WgradArgs::part
  const float* bias_part[kMaxConvLayers];  // per layer: [lane][n_tiles][64]
  __nv_bfloat16* wt[kMaxConvLayers];       // per layer: transposed bf16 copy in slot 0, or null
  int im2col[kMaxConvLayers];              // per layer: 1 = weights [64 out][64 k] (one tap)
  int64_t offW[kMaxConvLayers], offB[kMaxConvLayers];
  const float* master;
  float* master_w;
  __nv_bfloat16* shadow;
  int64_t slot_stride, wt_slot_stride;
  float lr;
};
struct CnnStageArgs {
  const float* const* x;       // [W] fp32 NHWC shards
  const int32_t* const* y;
  const int64_t* n;
  const int64_t* start;        // [W] cursors
  const int* wid;
  int step, B, Cin;
  int im2col;                  // 1: channel k = tap * Cin + i holds x[y + dy - 1][x + dx - 1][i], tap = 3 dy + dx
  __nv_bfloat16* out;          // [lane][B][1024][64]
  int32_t* labels;             // [lane][B] or null
};
struct CnnHeadArgs {
  const int* wid;
  const int* src;
  int B, K, step, max_tau, n_loss_chunks;
  const float* g;              // [lane][B][64]
  const int32_t* labels;       // [lane][B]
  float* dg;                   // [lane][B][64]
  float* loss_part;            // [(lane * max_tau + step) * n_loss_chunks + chunk]
  const float* master;
  float* master_w;
  __nv_bfloat16* shadow;
  int64_t slot_stride, offWf, offBf;
  float lr;
};
int cnn_tiles_per_image();
// images per split-K chunk of the weight gradient (one wave of CTAs over the active workers)
int conv_wgrad_images_per_chunk(int B, int n_active, int sms);
// CTAs per worker of the implicit-GEMM kernel (one per SM over the active workers)
int conv_ctas_per_worker(int B, int n_active, int sms);
cudaError_t launch_conv_igemm(int mode, const CUtensorMap& mIn, const CUtensorMap& mW, const ConvArgs& a, int n_active,
                              int cpw, cudaStream_t s);
cudaError_t launch_conv_wgrad(const CUtensorMap& mIn, const CUtensorMap& mDz, const WgradArgs& a, int n_active,
                              cudaStream_t s);
cudaError_t launch_conv_sgd(const ConvSgdArgs& a, int n_active, cudaStream_t s);
cudaError_t launch_conv_refresh_wt(const float* master, __nv_bfloat16* wt, int64_t offW, cudaStream_t s);
cudaError_t launch_cnn_stage(const CnnStageArgs& a, int n_active, cudaStream_t s);
cudaError_t launch_cnn_pool(const __nv_bfloat16* v, const int* wid, int B, float* g, int n_active, cudaStream_t s);
size_t cnn_head_smem(int B, int K);
cudaError_t launch_cnn_head(const CnnHeadArgs& a, int n_active, cudaStream_t s);
cudaError_t launch_cnn_head_loss(const float* g, const int32_t* labels, int B, int K, const float* master,
                                 int64_t offWf, int64_t offBf, float* out, cudaStream_t s);
cudaError_t launch_cnn_dzb(const __nv_bfloat16* v, const float* dg, const int* wid, int B, __nv_bfloat16* dz,
                           float* bias_part, int n_active, cudaStream_t s);

}  // namespace oscars
