// Internal interface of the slice-dataflow engine (mds_flow.cu) to the C ABI
// (mds_api.cu).  Not installed; not part of the public ABI.
//
// The engine splits every row the walk visits into slices of T tokens.  A
// persistent grid takes slice tasks from a ring in global memory; each task
// reduces its slice of the rows of one pass of one sequence to a record; the
// CTA that completes a pass's last slice runs that sequence's decision for the
// pass and publishes its next pass (or finishes the sequence).
#pragma once
#include <cstdint>
#include <cuda_runtime.h>

#include "mds_internal.h"

namespace mds {
namespace flow {

constexpr int kBufBytes = 32 * 1024;   // one slice buffer (every streamed row of one slice)
constexpr int kListRowsMax = 4;        // candidate lists: target + at most 3 draft models
constexpr int kMaxSlicesList = 32;     // slices per row with candidate lists
constexpr int kMaxSlices = 256;        // slices per row otherwise
constexpr int kSliceQuantum = 256;     // T is a multiple of this many tokens

// Control words (ctl[]): task head and tail, finished sequences, abort flag,
// CTAs that left the kernel.  All zero between launches.
enum { kCtlHead = 0, kCtlTail = 1, kCtlDone = 2, kCtlAbort = 3, kCtlExit = 4, kCtlDecHead = 5, kCtlDecTail = 6,
       kCtlWords = 16 };

struct Params {
  const char* target;                  // [B][K][L+1][V]
  const char* drafts[MDS_MAX_K];       // K x [B][L][V]
  const int32_t* tokens;               // [B][K][L]
  const float* temps;                  // [B][1+K]
  int32_t* out_tokens;                 // [B][L+1]
  int32_t* out_accept;                 // [B]
  float* out_diag;                     // [B][L+1][4] or null
  unsigned* status;                    // status word
  unsigned* ctl;                       // control words
  unsigned long long* ring_tag;        // [ring_cap] published task tags
  unsigned long long* ring_rtag;       // [ring_cap] tags of tasks taken
  unsigned* ring_pay;                  // [ring_cap] (sequence << 16) | slice
  unsigned long long* dec_tag;         // [dec_cap] published decision requests
  unsigned long long* dec_rtag;        // [dec_cap] tags of requests taken
  unsigned* dec_pay;                   // [dec_cap] the requests
  unsigned* cnt;                       // [B] slices of the current pass completed
  char* seq;                           // [B] per-sequence pass and walk state
  float* rec;                          // [B][ns][rec_floats] slice records
  float* dbg_rows;                     // [B][L+1][MDS_DEBUG_ROWS][4] row statistics, or null
  unsigned long long seed;
  unsigned epoch;                      // launch number (tags of the ring)
  int B, K, L, V;
  int scheme, dtype, esize;
  int wis_s, omega0, acc_prob;
  int T;                               // tokens per slice (multiple of kSliceQuantum)
  int ns;                              // slices per row
  int ln;                              // candidate list length of a sequence (0: no candidate lists)
  int lns;                             // candidate list length of one slice (<= ln)
  int rec_floats;                      // record stride per slice
  int hdr_floats;                      // start of a record's list entries
  int ring_cap;
  int dec_cap;
  int dec_sms;                         // SMs (ids 0..dec_sms-1) whose CTAs run the decisions
  int bulk;                            // rows are fetched with bulk copies (device memory, 16-byte aligned rows)
  int aligned;                         // rows start 16-byte aligned and V * esize is a multiple of 16
  int n_models;
  int8_t model_of[MDS_MAX_K];
};

// Geometry of one call: fills T, ns, ln, rec_floats, hdr_floats.  Returns
// false if the configuration is outside what this engine serves (the caller
// then uses the per-sequence engine).
bool plan_geometry(Params& p, int grid);

// Bytes of per-sequence state, for the workspace.
size_t seq_bytes();

// Workspace of one launch geometry (p after plan_geometry) for up to nseq
// sequences and a grid of `grid` CTAs: its size in bytes, and the carving of
// a buffer of that size into p's control words, ring, counters, per-sequence
// state and records.  The control words and counters must be zero before the
// first launch on a buffer; the kernel leaves them zero.  clear_bytes() is the
// length of that prefix (control words, then the ring, then the counters).
size_t workspace_bytes(const Params& p, int nseq, int grid);
void carve_workspace(Params& p, char* base, int nseq, int grid);
size_t clear_bytes(const Params& p, int nseq, int grid);

// Persistent grid size for this device (CTAs); 0 on error.
int grid_size(int device);

// One-time kernel attribute set-up for a logit type.
cudaError_t configure(int dtype);

// Phase timers of the instrumented build (-DMDS_PHASE_TIMERS): synchronises
// the device, copies up to n counters to out, clears them; returns the number
// of counters, -2 if the build has none, -1 on a CUDA error.
int read_phase_timers(unsigned long long* out, int n);

// Launch on `stream` with `grid` CTAs.
cudaError_t launch(const Params& p, int grid, cudaStream_t stream);

// Every token's probability of one row under given statistics (test export).
cudaError_t launch_probs(const void* row, int dtype, int V, float M, float invZ, float c, float* out,
                         cudaStream_t stream);

}  // namespace flow
}  // namespace mds
