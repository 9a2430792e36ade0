// Library-internal declarations shared by the planner (plan.cpp) and the device code (*.cu).
#pragma once

#include <cstdint>
#include <string>
#include <vector>

#include "bandggnn.h"

struct bg_plan {
  // shape
  int32_t K = 0, S = 0, P = 0, W32 = 0;  // W32 = S / 32 mask words per tile row
  int32_t n_graphs = 0, n_packed = 0, n_real = 0;
  int64_t n_edges_in = 0, n_unique = 0, n_kept = 0, n_dropped = 0;
  int64_t bw_before_max = 0, bw_after_max = 0;
  // per input graph
  std::vector<int32_t> n_nodes;
  std::vector<int64_t> node_base;  // prefix sums of n_nodes
  std::vector<int32_t> perm;       // concatenated perm[new] = old
  std::vector<int32_t> offset;     // -1 if not packed
  std::vector<int64_t> bw_before, bw_after;
  // per packed position / graph
  std::vector<int32_t> gather;          // [n_real] row of the concatenated input
  std::vector<int32_t> seg_off, seg_cnt;  // packed graphs
  // band tiles as bit rows: [K][3][P][S][W32] words, bit c of word c/32 (LSB first)
  std::vector<uint32_t> masks;   // row = target r in block k, bits = source c in block k+d-1
  std::vector<uint32_t> masksT;  // row = source c in block j, bits = target i in block j+e-1
  // supernodes: count per input graph (its first positions); kept edges with a supernode end,
  // (target, source, type) in positions, sorted
  int32_t n_super = 0;
  std::vector<int32_t> nsup;
  std::vector<int32_t> sup_edges;  // [n_super_edges][3]
  // device copies of the supernode edges (super.cu): in-edges by target row, out-edges by source
  // row, the (source row, type) pairs of the out-edges and those pairs grouped by type
  int32_t sup_rows_in = 0, sup_rows_out = 0, sup_pairs = 0;
  int32_t* d_sup = nullptr;        // one allocation holding the arrays below
  int32_t* d_sin_rows = nullptr;   // [rows_in] target positions
  int32_t* d_sin_off = nullptr;    // [rows_in + 1]
  int32_t* d_sin_src = nullptr;    // [n_super_edges] sorted by (type, source) within a row
  int32_t* d_sin_type = nullptr;
  int32_t* d_sin_slot = nullptr;   // [n_pad] row index of a target position, or -1
  int32_t* d_sout_rows = nullptr;  // [rows_out] source positions
  int32_t* d_sout_poff = nullptr;  // [rows_out + 1] pair ranges of each row
  int32_t* d_pair_type = nullptr;  // [pairs]
  int32_t* d_pair_off = nullptr;   // [pairs + 1] edge ranges of each pair
  int32_t* d_pair_row = nullptr;   // [pairs] index into rows_out
  int32_t* d_sout_dst = nullptr;   // [n_super_edges] sorted by (type, target) within a row
  int32_t* d_type_off = nullptr;   // [P + 1] ranges of d_type_pairs per type
  int32_t* d_type_pairs = nullptr; // [pairs] pair ids grouped by type, ascending row
  int64_t n_super_edges() const { return (int64_t)sup_edges.size() / 3; }
  // device copies (valid once uploaded)
  int device = -1;
  uint32_t* d_masks = nullptr;
  uint32_t* d_masksT = nullptr;
  int32_t* d_gather = nullptr;
  int32_t* d_seg_off = nullptr;
  int32_t* d_seg_cnt = nullptr;
  int32_t* d_row_graph = nullptr;  // [n_pad] packed graph of each position, -1 for padding
  // tensor-core path: bit-interleaved window chunks [n_pad / 128][P][C1][128][4] (C1 128-column
  // chunks per 128-row tile, band_tc.cu) in both orientations and per-row in-degree counts
  // [n_pad][64] (type p at columns p and 32 + p), bf16 while max_deg <= 256, else fp16
  uint32_t* d_maskI = nullptr;
  uint32_t* d_maskTI = nullptr;
  uint16_t* d_deg2 = nullptr;
  int32_t max_deg = 0;
  int32_t n_pad() const { return K * S; }
};

// error plumbing (api.cu)
int bg_fail(int code, const std::string& msg);
void bg_clear_error();
// The device status word of device `dev` that bounded waits write and bg_check_device reads, or
// NULL when it has not been created yet (api.cu; bg_plan_upload creates it).  Never allocates.
int* bg_status_word_if_created(int dev);
// Device-side set-up of the allocation-free entry point for the current device (noalloc.cu):
// resolves its static scratch array's address and loads the forward kernels of this plan's block
// size.  Called by bg_plan_upload, which allocates anyway.
int bg_noalloc_prepare(const bg_plan* p);

// block-row partition (plan.cpp)
int bg_plan_partition_build(const bg_plan* full, int32_t n_parts, int32_t part, bg_plan** out,
                            bg_part_info* info);

// planner entry (plan.cpp)
int bg_plan_build(const bg_graph* graphs, int32_t n_graphs, int32_t P, int32_t S, int32_t cap,
                  uint32_t flags, int32_t super_min_degree, int32_t max_super, bg_plan** out);
