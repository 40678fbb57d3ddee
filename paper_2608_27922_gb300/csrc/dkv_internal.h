// Internal (non-ABI) declarations shared by the host API and the kernel files.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "dkv_device.cuh"

namespace dkv {

// Caller-owned bank buffers plus their dimensions.
struct Bank {
  void* k;
  void* v;
  float* rho;
  float* base;
  float* knorm;
  int64_t* prov_step;
  int32_t* prov_src;
  int32_t* occ;
  int H, d, M_max, n_max;
  int bf16;   // 1: bf16 keys/values, 0: fp32
};

// Device workspace, carved from the caller's workspace buffer (dkv_api.cu).
struct Ws {
  DevLayer* L;          // [H / layer_heads] per-layer state; L[0] also holds the error word
  DevHead* hd;          // [H]
  int32_t* budgets;     // [H]
  float* cnorm;         // [H][n_max]     ||k_x||^2 of the candidates (source order)
  float* score;         // [H][n_max]     Eq. 6 scores
  int32_t* perm;        // [H][n_max]     stable ascending order of the scores (pi)
  void* kperm;          // [H][n_max][d]  candidate keys in pi order
  float* kperm_norm;    // [H][n_max]
  int32_t* cross;       // [H][M_max]     first prefix length with g >= tau (INT32_MAX: none)
  int32_t* hist;        // [H][hist_stride] histogram of cross over 0..rmax+1
  uint32_t* feas;       // [H][feas_words] bit r set: prefix r feasible in head h
  float* snap;          // [H][M_max][snap_stride] running prefix sums every SNAP columns
  float* rho_t;         // [H][M_max]     projected density rho~(r_h) (Eq. C.2)
  int32_t* evict_list;  // [H][n_max]     evicted slots, ascending
  int32_t* surv_list;   // [H][M_max]     surviving slots, ascending
  void* kevict;         // [H][n_max][d]  keys of evicted states (written by commit, read by the
                        //   survivor pass); during admit with temporal re-zeroing it holds
                        //   the re-zeroed candidate keys, [H][N][d] like the caller's K_c
  float* kevict_norm;   // [H][n_max]
  void* ksurv;          // [H][M_max][d]  keys of surviving states
  float* ksurv_norm;    // [H][M_max]
  int32_t* slot_new;    // [H][n_max]     bank slot of the j-th admitted candidate
  // extension rows of the tensor-core passes, bf16 [..][32]: row form | column form
  void* cext;           // [H][n_max][32] candidates, source order
  void* kperm_ext;      // [H][n_max][32] candidates, pi order
  void* bext;           // [H][M_max][32] bank (derived from the bank keys, kept in step)
  void* ksurv_ext;      // [H][M_max][32]
  void* kevict_ext;     // [H][n_max][32]
  // values beside the key copies, [K; V] descriptor only (nullptr otherwise)
  void* vperm;          // [H][n_max][d]  candidate values in pi order
  void* vsurv;          // [H][M_max][d]  values of surviving states
  void* vevict;         // [H][n_max][d]  values of evicted states
  unsigned long long* sortbuf;   // [H][sort_stride] sorted runs of 256 sort keys
  float* invb;          // [H][invb_stride] 1 / b of the bank states (derived from the
                        //   baselines, kept in step; 256 floats of padding at the end)
  float* part;          // [2][H][part_stride] per-row partial sums of column-split passes
  int32_t* cnt;         // [H][cnt_stride] arrival counters of column-split row tiles (kept 0)
  int32_t* tile_head;   // [n_mtiles] head of each 128-row tile of the heads' budgets, head-major
  int32_t* tile_first;  // [H] index of each head's first such tile
  int n_mtiles;         // sum over heads of ceil(M_h / 128)
  int32_t* pair_head;   // [n_mpairs] head of each pair of those tiles (tiles 2k, 2k + 1 of a
                        //   head): the units of the two-row-tile crossing pass
  int32_t* pair_first;  // [H] index of each head's first pair
  int n_mpairs;         // sum over heads of ceil(ceil(M_h / 128) / 2)
  int32_t* head_order;  // [H] heads by decreasing budget, ties by index (the order of the
                        //   persistent score pass's units: largest first)
  int32_t* loop_list;   // [3][loop_stride] row tiles with work of the persistent projection,
                        //   survivor and new-baseline passes (each its own: the last two run
                        //   side by side), appended by the pass's classification kernel
  int32_t* loop_ctr;    // [3][2] their count, and the next one to take
  int64_t loop_stride;  // H * max(ceil(M_max / 128), ceil(n_max / 128))
  int hist_stride, snap_stride, feas_words, part_stride, cnt_stride, invb_stride, sort_stride;
  int layer_heads;      // heads per layer (the handle's heads form H / layer_heads layers)
};

// Temporal rotary re-zeroing of the offered keys (App. A), device arrays of the caller.
struct RopeArgs {
  const float* theta;    // [d/2] angular frequency of rotation pair j (0: pair not rotated)
  const int32_t* tpos;   // [N] temporal coordinate of each candidate (all heads)
  int layout;            // 0: pair j = elements (2j, 2j + 1); 1: (j, j + d/2)
};

// Per-layer state of head h.
__host__ __device__ inline DevLayer* layer_of(const Ws& w, int h) { return w.L + h / w.layer_heads; }

// Computes the sub-buffer offsets of the workspace; returns the total bytes.
size_t ws_layout(int H, int d, int M_max, int n_max, int bf16, int kv, Ws* out, char* base);

// Kernel timing hook (dkv_api.cu): brackets a launch with events when enabled.
struct Timer;
void timer_begin(Timer* t, const char* name, cudaStream_t s);
void timer_end(Timer* t, cudaStream_t s);

// ---- launches (each returns cudaGetLastError() of its launch) ----
// update front half (admit)
// candidates' norms and extension rows, zeroed crossing histogram, update snapshot
// (rope != nullptr: the keys re-zeroed into w.kevict first, norms of the stored keys;
// [K; V] descriptor: the norms and extension rows are those of [k; v], Vc read too)
cudaError_t launch_cand_norms(const Bank& b, const Ws& w, const void* Kc, const void* Vc, int N, int64_t step,
                              const KParams& kp, const RopeArgs* rope, cudaStream_t s, Timer* t);
// (Vc: the candidates' values, read with the [K; V] descriptor)
cudaError_t launch_score_fp32(const Bank& b, const Ws& w, const void* Kc, const void* Vc, int N, const KParams& kp,
                              cudaStream_t s, Timer* t);
cudaError_t launch_sort(const Bank& b, const Ws& w, const void* Kc, const void* Vc, int identity, cudaStream_t s,
                        Timer* t);
cudaError_t launch_cross_fp32(const Bank& b, const Ws& w, const KParams& kp, cudaStream_t s, Timer* t);
cudaError_t launch_rstar(const Bank& b, const Ws& w, const KParams& kp, cudaStream_t s, Timer* t);
// update back half (compress)
cudaError_t launch_project_fp32(const Bank& b, const Ws& w, const KParams& kp, cudaStream_t s, Timer* t);
cudaError_t launch_select(const Bank& b, const Ws& w, int eviction, cudaStream_t s, Timer* t);
cudaError_t launch_commit(const Bank& b, const Ws& w, const void* Vc, int N, const int32_t* src_map, cudaStream_t s,
                          Timer* t);
// sequential admission: the block in pi order (keys, values, source indices) into scratch
cudaError_t launch_seq_gather(const Bank& b, const Ws& w, const void* Kc, const void* Vc, int N, void* Kseq,
                              void* Vseq, int32_t* srcseq, cudaStream_t s);
cudaError_t launch_subtract_fp32(const Bank& b, const Ws& w, const KParams& kp, cudaStream_t s, Timer* t);
cudaError_t launch_newbase_fp32(const Bank& b, const Ws& w, const KParams& kp, cudaStream_t s, Timer* t);
// tensor-core (tcgen05) versions of the pair passes, bf16 and d = 128 only
cudaError_t launch_score_tc(const Bank& b, const Ws& w, const void* Kc, const void* Vc, int N, const KParams& kp,
                            cudaStream_t s, Timer* t);
cudaError_t launch_cross_tc(const Bank& b, const Ws& w, const KParams& kp, cudaStream_t s, Timer* t);
cudaError_t launch_project_tc(const Bank& b, const Ws& w, const KParams& kp, cudaStream_t s, Timer* t);
cudaError_t launch_subtract_tc(const Bank& b, const Ws& w, const KParams& kp, cudaStream_t s, Timer* t);
cudaError_t launch_newbase_tc(const Bank& b, const Ws& w, const KParams& kp, cudaStream_t s, Timer* t);
// bank maintenance
cudaError_t launch_bank_norms(const Bank& b, const Ws& w, const KParams& kp, cudaStream_t s, Timer* t);
cudaError_t launch_inv_base(const Bank& b, const Ws& w, cudaStream_t s);
cudaError_t launch_set_occupancy(const Bank& b, const int32_t* occ_dev_src, int value, cudaStream_t s);
// attention
cudaError_t launch_attend_fp32(const Bank& b, const void* Q, int Nq, const void* Kw, const void* Vw, int W,
                               void* O, cudaStream_t s, Timer* t);
cudaError_t launch_attend_tc(const Bank& b, DevLayer* L, const void* Q, int Nq, const void* Kw, const void* Vw,
                             int W, void* O, cudaStream_t s, Timer* t);
bool tc_supported(int d, int bf16);
int sm_count();   // multiprocessors of the current device (0 if unknown)
cudaError_t simt_set_smem_limits();
cudaError_t update_set_smem_limits();
cudaError_t tc_set_smem_limits();

}  // namespace dkv
